"""The C-ABI library loads and exports every entry point include/dtp.h declares;
host-side argument validation rejects bad calls before any launch (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dtp.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_13846_gb300 import build, dtp
    build.build()
    return dtp.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dtp_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("dtp_affinity_accumulate", "dtp_search_layout", "dtp_search_layout_batched",
                     "dtp_affinity_workspace_size", "dtp_search_workspace_size", "dtp_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} not exported by libdtp.so"


def test_no_symbol_outside_header_is_extern_c(lib):
    """The library has no extra dtp_* C symbols beyond the header's."""
    import subprocess
    from paper_2609_13846_gb300 import dtp
    out = subprocess.run(["nm", "-D", "--defined-only", dtp.LIB_PATH], capture_output=True, text=True).stdout
    exported = sorted({m for m in re.findall(r"\bT (dtp_[a-z0-9_]+)\b", out)})
    assert exported == declared_functions()


def test_version_and_status_strings(lib):
    from paper_2609_13846_gb300 import dtp
    assert lib.dtp_version() >= 100
    assert dtp.status_string(0) == "ok"
    assert "argument" in dtp.status_string(-1)
    assert dtp.status_string(12345) == "unknown status"


def test_workspace_size_queries(lib):
    from paper_2609_13846_gb300 import dtp
    n = dtp.affinity_workspace_size(16384, 1024, 8, 3072, dtp.DTP_BF16)
    assert n >= 256 + 128 * 24 * 8 * 128 * 4  # one G x 128 partial per (token chunk, neuron tile)
    assert dtp.affinity_workspace_size(256, 64, 2, 128, dtp.DTP_F32) > 256
    assert dtp.search_workspace_size(28, 8, 3072, 4) >= 256
    # a layer that does not fit in shared memory gets a global buffer
    assert dtp.search_workspace_size(1, 8, 14336, 8) > 14336 * 8 * 8


@pytest.mark.parametrize("args", [
    (-1, 64, 2, 128, 0), (16, 12, 2, 128, 0), (16, 64, 0, 128, 0), (16, 64, 17, 128, 0),
    (16, 64, 2, 0, 0), (16, 64, 2, 128, 7)])
def test_affinity_size_query_rejects_bad_sizes(lib, args):
    n = ctypes.c_size_t(0)
    assert lib.dtp_affinity_workspace_size(*args, ctypes.byref(n)) == -1


def test_affinity_rejects_null_and_misaligned_before_launch(lib):
    vp = ctypes.c_void_p
    ok = vp(1 << 20)
    bad = vp((1 << 20) + 2)
    # null input
    assert lib.dtp_affinity_accumulate(None, ok, ok, ok, 16, 64, 2, 128, 0, ok, ok, 1 << 30, None) == -1
    # misaligned weight
    assert lib.dtp_affinity_accumulate(ok, ok, bad, ok, 16, 64, 2, 128, 0, ok, ok, 1 << 30, None) == -1
    # workspace too small
    assert lib.dtp_affinity_accumulate(ok, ok, ok, ok, 16, 64, 2, 128, 0, ok, ok, 8, None) == -5
    # d not a multiple of 8
    assert lib.dtp_affinity_accumulate(ok, ok, ok, ok, 16, 60, 2, 128, 0, ok, ok, 1 << 30, None) == -1


@pytest.mark.parametrize("layers,H,N,D,iters", [
    (1, 8, 3072, 3, 10), (1, 8, 3071, 2, 10), (1, 8, 3072, 16, 10), (1, 8, 3072, 1, 10),
    (0, 8, 3072, 2, 10), (1, 8, 3072, 2, 0), (1, 32, 64, 2, 1), (1, 8, 1 << 19, 2, 1)])
def test_search_rejects_bad_sizes(lib, layers, H, N, D, iters):
    vp = ctypes.c_void_p
    ok = vp(1 << 20)
    st = lib.dtp_search_layout_batched(ok, layers, H, N, D, iters, ok, ok, ok, ok, ok, ok, 1 << 30, None)
    assert st == -1


def test_search_rejects_missing_workspace(lib):
    vp = ctypes.c_void_p
    ok = vp(1 << 20)
    assert lib.dtp_search_layout(ok, 8, 64, 2, 3, ok, ok, ok, ok, ok, None, 0, None) == -5


@pytest.mark.parametrize("args,ok", [
    ((16384, 1024, 16, 2, 3072, 0), True), ((16, 64, 32, 4, 128, 0), True), ((16, 64, 128, 16, 128, 1), True),
    ((16, 64, 34, 2, 128, 0), False),        # 17 KV groups
    ((16, 64, 16, 3, 128, 0), False),        # q_per_group does not divide H_q
    ((16, 64, 136, 8, 128, 0), False),       # more than 128 query heads
    ((16, 64, 16, 0, 128, 0), False), ((16, 12, 16, 2, 128, 0), False)])
def test_grouped_size_queries(lib, args, ok):
    n = ctypes.c_size_t(0)
    st = lib.dtp_affinity_grouped_workspace_size(*args, ctypes.byref(n))
    assert (st == 0) == ok
    T, d, Hq, q, N, dtype = args
    st2 = lib.dtp_affinity_add_grouped_workspace_size(T, d, Hq, q, N, ctypes.byref(n))
    assert (st2 == 0) == ok


def test_grouped_workspace_covers_one_launch_of_whole_groups(lib):
    from paper_2609_13846_gb300 import dtp
    # 32 query heads at 4 per group run as two launches of 16 heads: the workspace of one 16-head launch
    assert dtp.affinity_grouped_workspace_size(4096, 1024, 32, 4, 3072, dtp.DTP_BF16) == \
        dtp.affinity_workspace_size(4096, 1024, 16, 3072, dtp.DTP_BF16)
    # 6 heads at 3 per group: one launch of all 6
    assert dtp.affinity_grouped_workspace_size(300, 64, 6, 3, 130, dtp.DTP_F32) == \
        dtp.affinity_workspace_size(300, 64, 6, 130, dtp.DTP_F32)


def test_chain_score_and_ablation_reject_before_launch(lib):
    buf = ctypes.create_string_buffer(1 << 16)
    p = ctypes.cast(buf, ctypes.c_void_p)
    # bad sizes (D does not divide N)
    assert lib.dtp_chain_score(p, p, 2, 8, 30, 4, p, p, None, p, p, p, ctypes.c_size_t(1 << 16), None) == -1
    # missing outputs
    assert lib.dtp_search_chain_ex(p, p, 2, 8, 32, 4, 5, None, None, 1, None, p, p, p, p, p,
                                   ctypes.c_size_t(1 << 16), None) == -1
    # too small a workspace
    assert lib.dtp_chain_score(p, p, 2, 8, 32, 4, p, p, None, p, p, p, ctypes.c_size_t(16), None) == -5


def test_affinity_opts_reject_bad_options(lib):
    from paper_2609_13846_gb300 import dtp
    buf = ctypes.create_string_buffer(1 << 12)
    p = ctypes.cast(buf, ctypes.c_void_p)
    bad = dtp.AffinityOpts(max_ctas=-1)
    assert lib.dtp_affinity_accumulate_opts(p, p, p, p, None, 16, 64, 2, 128, 0, p, None, ctypes.byref(bad), p,
                                            ctypes.c_size_t(1 << 12), None) == -1
    res = dtp.AffinityOpts(max_ctas=4)
    res.reserved[3] = 1
    assert lib.dtp_affinity_accumulate_opts(p, p, p, p, None, 16, 64, 2, 128, 0, p, None, ctypes.byref(res), p,
                                            ctypes.c_size_t(1 << 12), None) == -1
    assert lib.dtp_affinity_accumulate_opts(p, p, p, p, None, 16, 64, 2, 128, 0, p, None, None, p,
                                            ctypes.c_size_t(1 << 12), None) == -1


def test_global_search_size_rules(lib):
    n = ctypes.c_size_t(0)
    assert lib.dtp_search_global_workspace_size(28, 8, 3072, 4, ctypes.byref(n)) == 0
    assert n.value >= 256 + 28 * 105 * 8
    assert lib.dtp_search_global_workspace_size(1, 16, 64, 2, ctypes.byref(n)) == 0      # 6435 partitions
    assert lib.dtp_search_global_workspace_size(1, 16, 64, 4, ctypes.byref(n)) == -1     # 2.6M partitions
    assert lib.dtp_search_global_workspace_size(1, 8, 30, 4, ctypes.byref(n)) == -1      # D does not divide N


def test_affinity_defer_and_reduce_argument_checks(lib):
    from paper_2609_13846_gb300 import dtp
    buf = ctypes.create_string_buffer(1 << 12)
    p = ctypes.cast(buf, ctypes.c_void_p)
    bad = dtp.AffinityOpts(max_ctas=0, flags=2)                  # unknown flag
    assert lib.dtp_affinity_accumulate_opts(p, p, p, p, None, 16, 64, 2, 128, 0, p, None, ctypes.byref(bad), p,
                                            ctypes.c_size_t(1 << 12), None) == -1
    f32 = dtp.AffinityOpts(max_ctas=0, flags=dtp.DTP_AFFINITY_DEFER_REDUCE)   # bf16 only
    assert lib.dtp_affinity_accumulate_opts(p, p, p, p, None, 16, 64, 2, 128, 1, p, None, ctypes.byref(f32), p,
                                            ctypes.c_size_t(1 << 12), None) == -4
    assert lib.dtp_affinity_reduce(p, ctypes.c_size_t(16), 16, 64, 2, 128, p, None, 0, 0, None) == -5   # small ws
    assert lib.dtp_affinity_reduce(p, ctypes.c_size_t(1 << 12), 16, 12, 2, 128, p, None, 0, 0, None) == -1  # d % 8
    assert lib.dtp_affinity_reduce(p, ctypes.c_size_t(1 << 12), 16, 64, 2, 128, p, None, -1, 0, None) == -1


def test_apply_layout_argument_checks(lib):
    buf = ctypes.create_string_buffer(1 << 12)
    p = ctypes.cast(buf, ctypes.c_void_p)
    ptrs = (ctypes.c_void_p * 7)(*([p.value + 16 * i for i in range(7)]))
    outs = (ctypes.c_void_p * 7)(*([p.value + 1024 + 16 * i for i in range(7)]))
    same = (ctypes.c_void_p * 7)(*([p.value + 16 * i for i in range(7)]))
    ws = ctypes.c_size_t(1 << 12)
    # D does not divide the heads; a source used as its own destination; a null pointer array; no workspace
    assert lib.dtp_apply_layout(p, p, 2, 8, 64, 3, 2, 16, 64, 2, ptrs, outs, p, p, p, ws, None) == -1
    assert lib.dtp_apply_layout(p, p, 2, 8, 64, 4, 2, 16, 64, 2, ptrs, same, p, p, p, ws, None) == -1
    assert lib.dtp_apply_layout(p, p, 2, 8, 64, 4, 2, 16, 64, 2, None, outs, p, p, p, ws, None) == -1
    assert lib.dtp_apply_layout(p, p, 2, 8, 64, 4, 2, 16, 64, 2, ptrs, outs, p, p, None, ws, None) == -5


def test_selftest_bounded_wait_rejects_bad_arguments(lib):
    """The bounded-wait self-test validates its arguments on the host, before any CUDA call."""
    import ctypes as ct
    from paper_2609_13846_gb300 import dtp
    el = (ct.c_uint64 * 2)()
    dummy = ct.c_void_p(256)   # never dereferenced: every call below fails validation first
    assert lib.dtp_selftest_bounded_wait(10 ** 6, 0, None, 256, el, None) == dtp.DTP_ERR_ARG
    assert lib.dtp_selftest_bounded_wait(10 ** 6, 0, dummy, 64, el, None) == dtp.DTP_ERR_ARG
    assert lib.dtp_selftest_bounded_wait(10 ** 6, 0, dummy, 256, None, None) == dtp.DTP_ERR_ARG
    assert lib.dtp_selftest_bounded_wait(10, 0, dummy, 256, el, None) == dtp.DTP_ERR_ARG
    assert lib.dtp_selftest_bounded_wait(2 * 10 ** 9, 0, dummy, 256, el, None) == dtp.DTP_ERR_ARG
    assert lib.dtp_selftest_bounded_wait(10 ** 6, 2, dummy, 256, el, None) == dtp.DTP_ERR_ARG
