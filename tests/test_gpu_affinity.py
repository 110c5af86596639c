"""GPU parity of the first-order affinity (Sec. 3 "Affinity scores") against the fp64 oracle.

Tolerances (relative Frobenius error of A): 5e-3 for bf16 operands (tcgen05
path), 1e-5 for the fp32 mode.  The inputs are the same bf16/fp32 values on
both sides, so the error budget is fp32 accumulation and the fp32 epilogue.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu

BF16_TOL = 5e-3
F32_TOL = 1e-5
DEV = "cuda:0"


def _rel_fro(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _oracle(L, rows=None):
    X, C, Wg, Wu = (L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up"))
    if rows is not None:
        Wg, Wu = Wg[rows], Wu[rows]
    return oracle.affinity_fo(X, C, Wg, Wu)


def _sample_columns(N, n_random, seed):
    """Neuron columns for a full-size check: one whole 128-neuron tile in the middle of the grid, the
    last tile (in chunk-major unit order its units are the left-over ones that may be split by heads),
    the first column and a few random ones."""
    mid = (N // 128) // 2 * 128
    rng = np.random.default_rng(seed)
    cols = [np.arange(mid, min(mid + 128, N)), np.arange(max(N - 128, 0), N), [0],
            rng.choice(N, size=n_random, replace=False)]
    return np.unique(np.concatenate(cols))


def _check_columns(got, ref):
    """Relative Frobenius error over the sampled columns, and every entry within the elementwise
    bound of the ragged-shape tests."""
    assert _rel_fro(got, ref) <= BF16_TOL
    assert np.all(np.abs(got - ref) <= 2e-2 * np.abs(ref) + 1e-6 * np.abs(ref).max())


def _gpu(L, A=None):
    g = {k: v.to(DEV) for k, v in L.items()}
    out = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"], A=A)
    torch.cuda.synchronize()
    return out


def test_tiny_workload_fp32_mode():
    """The tiny calibration workload (d=64, G=2, N=128, T=256) in fp32 mode: <= 1e-5."""
    L = synth.make_workload_layer(synth.WORKLOADS["tiny"])
    A = _gpu(L).cpu().numpy()
    assert _rel_fro(A, _oracle(L)) <= F32_TOL


def test_tiny_workload_bf16_mode():
    L = synth.make_workload_layer(synth.WORKLOADS["tiny"])
    Lb = {k: v.to(torch.bfloat16) for k, v in L.items()}
    A = _gpu(Lb).cpu().numpy()
    assert _rel_fro(A, _oracle(Lb)) <= BF16_TOL


@pytest.mark.parametrize("d,G,N,T", [
    (328, 3, 300, 333),     # ragged in every dimension, several tiles of each
    (1024, 8, 384, 384),    # Qwen-like d and G, 3 neuron tiles x 3 token chunks
    (64, 1, 1, 1),          # single head, neuron and token
    (8, 2, 130, 129),       # smallest d (one 16-byte row), ragged tiles
    (136, 16, 200, 77),     # the largest supported head count
])
def test_bf16_parity_ragged(d, G, N, T):
    L = synth.make_layer(d, G, N, T, seed=d + G + N + T, dtype="bf16", outliers=d >= 64)
    A = _gpu(L).cpu().numpy()
    err = _rel_fro(A, _oracle(L))
    assert err <= BF16_TOL, err
    # elementwise: every entry within a loose relative bound of the fp64 value
    ref = _oracle(L)
    assert np.all(np.abs(A - ref) <= 2e-2 * np.abs(ref) + 1e-6 * np.abs(ref).max())


@pytest.mark.parametrize("d,G,N,T", [
    (64, 8, 1280, 2048),    # 160 units on up to 152 SMs: the 8 left-over units are split by heads
    (72, 3, 1300, 1900),    # 165 units, 3 heads: left-over units split into single heads
])
def test_bf16_parity_left_over_units_split_by_heads(d, G, N, T):
    L = synth.make_layer(d, G, N, T, seed=G + N, dtype="bf16", outliers=True)
    A = _gpu(L).cpu().numpy()
    assert _rel_fro(A, _oracle(L)) <= BF16_TOL


@pytest.mark.parametrize("d,G,N,T", [(328, 3, 300, 333), (64, 2, 65, 70)])
def test_fp32_parity_ragged(d, G, N, T):
    L = synth.make_layer(d, G, N, T, seed=3, dtype="f32", outliers=True)
    A = _gpu(L).cpu().numpy()
    assert _rel_fro(A, _oracle(L)) <= F32_TOL


def test_zero_tokens_is_a_noop():
    L = synth.make_layer(64, 2, 32, 8, seed=1, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    A = torch.full((2, 32), 3.0, device=DEV)
    dtp.affinity_accumulate(g["X"][:0].contiguous(), g["C"][:, :0].contiguous(), g["W_gate"], g["W_up"], A=A)
    torch.cuda.synchronize()
    assert torch.all(A == 3.0)


def test_accumulates_over_token_chunks():
    """A is accumulated, so streaming token chunks equals one call on all tokens (Sec. 3: E_t over tokens)."""
    L = synth.make_layer(256, 4, 256, 600, seed=9, dtype="bf16")
    full = _gpu(L)
    A = torch.zeros_like(full)
    for lo, hi in ((0, 128), (128, 333), (333, 600)):
        part = {"X": L["X"][lo:hi].contiguous(), "C": L["C"][:, lo:hi].contiguous(),
                "W_gate": L["W_gate"], "W_up": L["W_up"]}
        _gpu(part, A=A)
    assert torch.allclose(A, full, rtol=1e-5, atol=0)


def test_deterministic():
    L = synth.make_layer(512, 8, 384, 1024, seed=4, dtype="bf16")
    a = _gpu(L)
    b = _gpu(L)
    assert torch.equal(a, b)


def test_workspace_status_ok_and_explicit_workspace():
    L = synth.make_layer(128, 2, 128, 256, seed=2, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    ws = dtp.affinity_workspace(256, 128, 2, 128, dtp.DTP_BF16, DEV)
    A = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"], workspace=ws)
    assert dtp.workspace_status(ws) == dtp.DTP_OK
    assert _rel_fro(A.cpu().numpy(), _oracle(L)) <= BF16_TOL


def test_finalize_and_down_norm():
    """S^{up,fo} = E_t[Delta^2] ||w^d_k||^2 (Sec. 3)."""
    L = synth.make_layer(128, 2, 96, 200, seed=5, dtype="bf16", with_down=True)
    A = _gpu({k: L[k] for k in ("X", "C", "W_gate", "W_up")})
    wd = dtp.down_sqnorm(L["W_down"].to(DEV))
    ref_wd = (L["W_down"].double() ** 2).sum(0).numpy()
    assert np.allclose(wd.cpu().numpy(), ref_wd, rtol=1e-5)
    dtp.affinity_finalize(A, 200, wd)
    torch.cuda.synchronize()
    ref = oracle.finalize(_oracle(L), 200, ref_wd)
    assert _rel_fro(A.cpu().numpy(), ref) <= BF16_TOL


@pytest.mark.parametrize("name", ["qwen3_0.6b_layer", "llama3.1_8b_layer"])
def test_full_size_sampled_neurons(name):
    """Full-size layer in the launch configuration the benchmark times; the oracle
    computes a sample of neuron columns over all T tokens (column k of A depends
    only on row k of the weights)."""
    w = synth.WORKLOADS[name]
    L = synth.make_workload_layer(w, device=DEV)
    A = dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"])
    # the benchmark's step caps the grid at one CTA below the SM count (the search runs beside it)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    A_capped = dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"], max_ctas=sms - 1)
    torch.cuda.synchronize()
    assert torch.equal(A, A_capped)
    cols = _sample_columns(w.N, 6, seed=0)
    assert len(cols) >= 136
    Lh = {k: v.cpu() for k, v in L.items()}
    ref = _oracle(Lh, rows=cols)
    got = A_capped[:, torch.as_tensor(cols, device=DEV)].double().cpu().numpy()
    _check_columns(got, ref)
    assert torch.isfinite(A).all() and (A >= 0).all()


@pytest.mark.parametrize("T", [1, 129, 257, 640])
def test_odd_and_even_token_chunk_counts(T):
    """Chunk counts 1, 2, 3 and 5: with CTA pairs the odd CTA of a last, half-empty pair reloads
    the last chunk and its sums go to a spare slot that must not reach A."""
    d, G, N = 256, 4, 200
    L = synth.make_layer(d, G, N, T, seed=40 + T, dtype="bf16")
    A = _gpu(L).cpu().numpy()
    assert _rel_fro(A, _oracle(L)) <= BF16_TOL


@pytest.mark.parametrize("T,max_ctas", [(300, 0), (300, 5), (1000, 151)])
def test_weights_beyond_half_of_l2(T, max_ctas):
    """W_gate + W_up of 128 MiB (d = 4096, N = 8192) exceed half of L2, so the kernel runs as
    single CTAs with chunk grouping; sampled neuron columns against the oracle, and the grid cap
    leaves A bitwise unchanged."""
    d, G, N = 4096, 2, 8192
    L = synth.make_layer(d, G, N, T, seed=60, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    A = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"], max_ctas=max_ctas)
    A_full = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    torch.cuda.synchronize()
    assert torch.equal(A, A_full)
    cols = np.unique(np.concatenate([np.random.default_rng(2).choice(N, size=5, replace=False), [0, 127, 128, N - 1]]))
    ref = _oracle(L, rows=cols)
    got = A[:, torch.as_tensor(cols, device=DEV)].double().cpu().numpy()
    assert _rel_fro(got, ref) <= BF16_TOL


@pytest.mark.parametrize("max_ctas", [1, 7, 151])
def test_grid_cap_does_not_change_the_result(max_ctas):
    """The persistent grid may be capped (SMs left to a concurrent search); A is bitwise the same."""
    L = synth.make_layer(1024, 8, 3072, 2048, seed=12, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    full = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    capped = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"], max_ctas=max_ctas)
    torch.cuda.synchronize()
    assert torch.equal(full, capped)


@pytest.mark.parametrize("name", ["qwen3_0.6b_model", "danube3_500m_model"])
def test_full_model_layer_sampled_neurons_with_down_term(name):
    """Layer 0 of the full-model workloads (T = 65536 tokens) through the call the whole-model
    benchmark makes (affinity pass with the down-edge activation term); the oracle computes
    sampled neuron columns of A and entries of act2 over all tokens."""
    w = synth.WORKLOADS[name]
    L = synth.make_workload_layer(w, 0, device=DEV)
    Dn = synth.make_down_inputs(w.d, w.G, w.qkv_rows, w.N, w.T, seed=w.seed + 1000, device=DEV)
    A, act2 = dtp.affinity_accumulate_down(L["X"], L["C"], L["W_gate"], L["W_up"], Dn["rms"])
    torch.cuda.synchronize()
    cols = _sample_columns(w.N, 3, seed=1)
    assert len(cols) >= 136
    Lh = {k: v.cpu() for k, v in L.items()}
    ref = _oracle(Lh, rows=cols)
    got = A[:, torch.as_tensor(cols, device=DEV)].double().cpu().numpy()
    _check_columns(got, ref)
    ref_act = oracle.down_activation(Lh["X"].double().numpy(), Lh["W_gate"][cols].double().numpy(),
                                     Lh["W_up"][cols].double().numpy(), Dn["rms"].double().cpu().numpy())
    _check_columns(act2[torch.as_tensor(cols, device=DEV)].double().cpu().numpy(), ref_act)


@pytest.mark.parametrize("with_act", [False, True])
def test_deferred_reduce_on_another_stream_is_bitwise_the_same(with_act):
    """The main kernel alone (partials left in the workspace), then the reduce on a second
    stream ordered by an event: A (and act2) equal the one-call result bit for bit."""
    d, G, N, T = 512, 8, 640, 1000
    L = synth.make_layer(d, G, N, T, seed=33, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    rms = (0.5 + torch.rand(T, generator=torch.Generator().manual_seed(2))).to(DEV)
    ws = dtp.affinity_workspace(T, d, G, N, dtp.DTP_BF16, DEV)
    if with_act:
        ref, ref_act = dtp.affinity_accumulate_down(g["X"], g["C"], g["W_gate"], g["W_up"], rms)
    else:
        ref = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    A = torch.zeros((G, N), dtype=torch.float32, device=DEV)
    act2 = torch.zeros(N, dtype=torch.float32, device=DEV) if with_act else None
    opts = dtp.AffinityOpts(max_ctas=100, flags=dtp.DTP_AFFINITY_DEFER_REDUCE)
    st = dtp.lib().dtp_affinity_accumulate_opts(dtp._ptr(g["X"]), dtp._ptr(g["C"]), dtp._ptr(g["W_gate"]),
                                                dtp._ptr(g["W_up"]), dtp._ptr(rms) if with_act else None, T, d, G,
                                                N, dtp.DTP_BF16, dtp._ptr(A), dtp._ptr(act2), ctypes.byref(opts),
                                                dtp._ptr(ws), ws.numel(), dtp._stream(None))
    assert st == dtp.DTP_OK
    assert not A.any()                                  # nothing reduced yet
    ev = torch.cuda.Event()
    ev.record()
    side = torch.cuda.Stream()
    side.wait_event(ev)
    dtp.affinity_reduce(ws, T, d, G, N, A, act2, stream=side)
    torch.cuda.synchronize()
    assert torch.equal(A, ref)
    if with_act:
        assert torch.equal(act2, ref_act)
    # the same partials reduced by one 1024-thread block, overwriting stale values
    A.fill_(7.0)
    if with_act:
        act2.fill_(7.0)
    dtp.affinity_reduce(ws, T, d, G, N, A, act2, max_blocks=1, overwrite=True)
    torch.cuda.synchronize()
    assert torch.equal(A, ref)
    if with_act:
        assert torch.equal(act2, ref_act)


def test_top_group_share_matches_oracle():
    mats = [synth.make_affinity_matrix(8, 3072, seed=s).numpy() for s in range(3)]
    mats.append(np.ones((8, 3072), np.float32))
    z = np.zeros((8, 3072), np.float32)
    z[:, ::3] = synth.make_affinity_matrix(8, 1024, seed=9).numpy()
    mats.append(z)                                      # two thirds of the columns empty
    A = torch.as_tensor(np.stack(mats), device=DEV)
    got = dtp.top_group_share(A).cpu().numpy()
    for i, m in enumerate(mats):
        assert got[i] == pytest.approx(oracle.top_group_share(m), rel=1e-12)
    w = synth.WORKLOADS["qwen3_0.6b_layer"]
    L = synth.make_workload_layer(w, T=2048, device=DEV)
    Aw = dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"])
    assert float(dtp.top_group_share(Aw)) == pytest.approx(oracle.top_group_share(Aw.cpu().numpy()), rel=1e-12)


def test_binding_rejects_mismatched_shapes_before_any_launch():
    """A C with fewer tokens than X, or weights of another width, would let the kernels read past a
    buffer: the affinity, ADD and down-edge entry points of the binding refuse them on the host."""
    X = torch.zeros((64, 32), dtype=torch.bfloat16, device=DEV)
    C_short = torch.zeros((2, 48, 32), dtype=torch.bfloat16, device=DEV)
    W = torch.zeros((16, 32), dtype=torch.bfloat16, device=DEV)
    W_wide = torch.zeros((16, 40), dtype=torch.bfloat16, device=DEV)
    rms = torch.ones(64, device=DEV)
    A = torch.zeros((2, 16), device=DEV)
    for C, Wg in ((C_short, W), (torch.zeros((2, 64, 32), dtype=torch.bfloat16, device=DEV), W_wide)):
        with pytest.raises(ValueError):
            dtp.affinity_accumulate(X, C, Wg, W)
        with pytest.raises(ValueError):
            dtp.affinity_accumulate_down(X, C, Wg, W, rms)
        with pytest.raises(ValueError):
            dtp.affinity_accumulate_grouped(X, C, Wg, W, 2)
        with pytest.raises(ValueError):
            dtp.affinity_accumulate_noalloc(X, C, Wg, W, A)
    with pytest.raises(TypeError):
        dtp.affinity_accumulate_noalloc(X.float(), torch.zeros((2, 64, 32), device=DEV), W.float(), W.float(), A)
    C = torch.zeros((2, 64, 32), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(ValueError):
        dtp.affinity_add_accumulate(C, W_wide, W)
    with pytest.raises(ValueError):
        dtp.affinity_add_accumulate_grouped(C, W, W_wide, 2)
    Wqkv = torch.zeros((2, 24, 32), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(ValueError):
        dtp.down_weight_sqnorm(Wqkv, torch.ones(40, dtype=torch.bfloat16, device=DEV),
                               torch.zeros((32, 16), dtype=torch.bfloat16, device=DEV))
    with pytest.raises(ValueError):
        dtp.down_weight_sqnorm(Wqkv, torch.ones(32, dtype=torch.bfloat16, device=DEV),
                               torch.zeros((40, 16), dtype=torch.bfloat16, device=DEV))
    with pytest.raises(ValueError):
        dtp.down_finalize(torch.zeros(15, device=DEV), torch.zeros((2, 16), device=DEV), 64)
