"""GPU parity of the down-edge score and the ADD score (Sec. 3) against the oracle.

Tolerance: relative Frobenius error <= 5e-3 for bf16 operands, <= 1e-5 for the
fp32 mode.  ||b_gk||^2 rounds gamma' . w^d_k to bf16 once before the tensor
cores; the error that adds stays well inside 5e-3.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
BF16_TOL = 5e-3
F32_TOL = 1e-5


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


@pytest.mark.parametrize("dtype,d,G,N,T", [
    ("bf16", 328, 3, 300, 333), ("bf16", 1024, 8, 384, 400), ("bf16", 64, 8, 1280, 2048),
    ("f32", 328, 3, 300, 333), ("f32", 64, 2, 65, 70)])
def test_down_activation_fused_in_affinity_pass(dtype, d, G, N, T):
    """act2[k] = sum_t (silu(g) u)^2 / r'^2 from the X pass; A is bitwise unchanged."""
    L = synth.make_layer(d, G, N, T, seed=N + T, dtype=dtype, outliers=True)
    D = synth.make_down_inputs(d, G, 64, N, T, seed=5, dtype=dtype)
    g = {k: v.to(DEV) for k, v in L.items()}
    A_plain = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    A, act2 = dtp.affinity_accumulate_down(g["X"], g["C"], g["W_gate"], g["W_up"], D["rms"].to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(A, A_plain)
    ref = oracle.down_activation(L["X"].double().numpy(), L["W_gate"].double().numpy(),
                                 L["W_up"].double().numpy(), D["rms"].double().numpy())
    assert _rel(act2.cpu().numpy(), ref) <= (BF16_TOL if dtype == "bf16" else F32_TOL)


@pytest.mark.parametrize("G,R,d,N", [(4, 200, 256, 300), (8, 512, 1024, 640), (2, 96, 64, 1000)])
def test_down_weight_sqnorm(G, R, d, N):
    D = synth.make_down_inputs(d, G, R, N, 8, seed=G + R, dtype="bf16")
    bn = dtp.down_weight_sqnorm(D["Wqkv"].to(DEV), D["gamma"].to(DEV), D["W_down"].to(DEV))
    torch.cuda.synchronize()
    ref = oracle.down_weight_sqnorm(D["Wqkv"].double().numpy(), D["gamma"].double().numpy(),
                                    D["W_down"].double().numpy())
    assert _rel(bn.cpu().numpy(), ref) <= BF16_TOL
    assert (bn >= 0).all()


def test_down_score_end_to_end():
    d, G, N, T, R = 256, 4, 384, 500, 128
    L = synth.make_layer(d, G, N, T, seed=2, dtype="bf16")
    D = synth.make_down_inputs(d, G, R, N, T, seed=3, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    _, act2 = dtp.affinity_accumulate_down(g["X"], g["C"], g["W_gate"], g["W_up"], D["rms"].to(DEV))
    bn = dtp.down_weight_sqnorm(D["Wqkv"].to(DEV), D["gamma"].to(DEV), D["W_down"].to(DEV))
    S = dtp.down_finalize(act2, bn, T)
    torch.cuda.synchronize()
    a_ref = oracle.down_activation(L["X"].double().numpy(), L["W_gate"].double().numpy(),
                                   L["W_up"].double().numpy(), D["rms"].double().numpy())
    b_ref = oracle.down_weight_sqnorm(D["Wqkv"].double().numpy(), D["gamma"].double().numpy(),
                                      D["W_down"].double().numpy())
    assert _rel(S.cpu().numpy(), oracle.down_score(a_ref, b_ref, T)) <= BF16_TOL


@pytest.mark.parametrize("d,G,N,T", [(328, 3, 300, 333), (1024, 8, 384, 256), (64, 1, 1, 1), (8, 2, 130, 129)])
def test_add_score(d, G, N, T):
    L = synth.make_layer(d, G, N, T, seed=d + N, dtype="bf16", outliers=True)
    g = {k: v.to(DEV) for k, v in L.items()}
    A = dtp.affinity_add_accumulate(g["C"], g["W_gate"], g["W_up"])
    torch.cuda.synchronize()
    ref = oracle.affinity_add(L["C"].double().numpy(), L["W_gate"].double().numpy(), L["W_up"].double().numpy())
    assert _rel(A.cpu().numpy(), ref) <= BF16_TOL


def test_add_score_accumulates_and_is_deterministic():
    L = synth.make_layer(256, 4, 256, 600, seed=9, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    full = dtp.affinity_add_accumulate(g["C"], g["W_gate"], g["W_up"])
    again = dtp.affinity_add_accumulate(g["C"], g["W_gate"], g["W_up"])
    A = torch.zeros_like(full)
    for lo, hi in ((0, 200), (200, 600)):
        dtp.affinity_add_accumulate(g["C"][:, lo:hi].contiguous(), g["W_gate"], g["W_up"], A_add=A)
    torch.cuda.synchronize()
    assert torch.equal(full, again)
    assert torch.allclose(A, full, rtol=1e-5, atol=0)


def _tile_columns(N, tile, n_random, seed):
    """A whole tile of columns in the middle of the grid, the last tile (left-over units), the first
    column and a few random ones."""
    mid = (N // tile) // 2 * tile
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([np.arange(mid, mid + tile), np.arange(N - tile, N), [0],
                                     rng.choice(N, size=n_random, replace=False)]))


def _elementwise_ok(got, ref):
    return bool(np.all(np.abs(got - ref) <= 2e-2 * np.abs(ref) + 1e-6 * np.abs(ref).max()))


def test_add_score_weights_beyond_half_of_l2():
    """W_gate + W_up of 128 MiB (d = 4096, N = 8192): the sum-of-squares kernel runs as single CTAs;
    two whole neuron tiles and sampled columns against the oracle (column k depends only on row k of
    the weights)."""
    d, G, N, T = 4096, 2, 8192, 300
    L = synth.make_layer(d, G, N, T, seed=70, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    A = dtp.affinity_add_accumulate(g["C"], g["W_gate"], g["W_up"])
    torch.cuda.synchronize()
    cols = np.unique(np.concatenate([_tile_columns(N, 128, 5, 3), [127, 128]]))
    ref = oracle.affinity_add(L["C"].double().numpy(), L["W_gate"][cols].double().numpy(),
                              L["W_up"][cols].double().numpy())
    got = A[:, torch.as_tensor(cols, device=DEV)].cpu().numpy()
    assert _rel(got, ref) <= BF16_TOL and _elementwise_ok(got, ref)


def test_down_weight_sqnorm_beyond_half_of_l2():
    """gamma' . W_down^T of 128 MiB (d = 4096, N = 16384): single CTAs; two whole column tiles and
    sampled columns (column k of ||b_gk||^2 depends only on column k of W_down)."""
    G, R, d, N = 2, 200, 4096, 16384
    D = synth.make_down_inputs(d, G, R, N, 8, seed=71, dtype="bf16")
    bn = dtp.down_weight_sqnorm(D["Wqkv"].to(DEV), D["gamma"].to(DEV), D["W_down"].to(DEV))
    torch.cuda.synchronize()
    cols = np.unique(np.concatenate([_tile_columns(N, 256, 5, 4), [255, 256]]))
    ref = oracle.down_weight_sqnorm(D["Wqkv"].double().numpy(), D["gamma"].double().numpy(),
                                    D["W_down"][:, cols].double().numpy())
    got = bn[:, torch.as_tensor(cols, device=DEV)].cpu().numpy()
    assert _rel(got, ref) <= BF16_TOL and _elementwise_ok(got, ref)
