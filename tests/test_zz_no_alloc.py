"""The allocation-free affinity entry point (dtp_affinity_accumulate_noalloc).

It serves callers that cannot allocate device memory or hand the library a
workspace (e.g. a plugin whose host owns every device allocation); its scratch
is a fixed array inside the library.  It runs the same kernels in the same
launch shape as dtp_affinity_accumulate, so on consecutive calls that reuse the
shared array with different shapes it must give A bit for bit equal to that
entry point's, and its status reader must report DTP_OK after each call.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
BF16_TOL = 5e-3  # the relative Frobenius tolerance of the bf16 affinity tests


def _rel_fro(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def _both(L):
    A_ref = dtp.affinity_accumulate(L["X"], L["C"], L["W_gate"], L["W_up"])
    A_new = torch.zeros_like(A_ref)
    dtp.affinity_accumulate_noalloc(L["X"], L["C"], L["W_gate"], L["W_up"], A_new)
    assert dtp.affinity_noalloc_status() == dtp.DTP_OK
    return A_new, A_ref


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    # the larger call first, so stale partial sums of the first would show in the second
    for d, G, N, T, seed in ((1024, 8, 384, 1000, 11), (328, 3, 300, 333, 12)):
        L = synth.make_layer(d, G, N, T, seed, dtype="bf16", device=DEV)
        A_new, A_ref = _both(L)
        assert torch.isfinite(A_new).all()
        assert torch.equal(A_new, A_ref)


def test_noalloc_matches_the_oracle_on_a_ragged_shape():
    d, G, N, T = 328, 3, 300, 333  # ragged in every dimension, several tiles of each
    L = synth.make_layer(d, G, N, T, seed=13, dtype="bf16", outliers=True)
    g = {k: v.to(DEV) for k, v in L.items()}
    A = torch.zeros((G, N), dtype=torch.float32, device=DEV)
    dtp.affinity_accumulate_noalloc(g["X"], g["C"], g["W_gate"], g["W_up"], A)
    assert dtp.affinity_noalloc_status() == dtp.DTP_OK
    ref = oracle.affinity_fo(*(L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up")))
    got = A.cpu().numpy()
    assert _rel_fro(got, ref) <= BF16_TOL
    assert np.all(np.abs(got - ref) <= 2e-2 * np.abs(ref) + 1e-6 * np.abs(ref).max())


def test_noalloc_rejects_calls_beyond_its_scratch():
    # 129 chunks, rounded up to 130: 130 * ceil(N/128) * H_kv = 130 * 16 * 16 > 32768, the documented limit
    G, N, T, d = 16, 2048, 129 * 128, 8
    X = torch.zeros((T, d), dtype=torch.bfloat16, device=DEV)
    C = torch.zeros((G, T, d), dtype=torch.bfloat16, device=DEV)
    W = torch.zeros((N, d), dtype=torch.bfloat16, device=DEV)
    A = torch.zeros((G, N), dtype=torch.float32, device=DEV)
    with pytest.raises(dtp.DTPError) as e:
        dtp.affinity_accumulate_noalloc(X, C, W, W, A)
    assert e.value.status == dtp.DTP_ERR_WORKSPACE


def test_noalloc_at_its_limit_uses_every_slot():
    # exactly at the limit (128 chunks * 16 tiles * 16 heads = 32768): every slot of the array is
    # written and read, on seeded non-zero inputs
    L = synth.make_layer(64, 16, 2048, 128 * 128, seed=14, dtype="bf16", device=DEV)
    A_new, A_ref = _both(L)
    assert (A_ref > 0).all()
    assert torch.equal(A_new, A_ref)
