"""GPU parity of the per-query-head scores (Sec. 3: E[Delta^2] per query head,
summed over each KV group's query heads) against the fp64 oracle.

Tolerances as for the per-group scores: relative Frobenius error <= 5e-3 with
bf16 operands, <= 1e-5 in the fp32 mode.  With one query head per group the
grouped entry points must reproduce the plain ones bit for bit.
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


def _np(L):
    return (L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up"))


@pytest.mark.parametrize("dtype,d,Hq,q,N,T", [
    ("bf16", 256, 16, 2, 384, 300),      # 16 query heads in 8 KV groups (Qwen3-0.6B, Danube3-500M ratio)
    ("bf16", 128, 32, 4, 300, 257),      # 32 query heads in 8 groups (Llama-3.1-8B ratio): two launches
    ("bf16", 64, 6, 3, 130, 129),        # ragged neuron and token tails
    ("bf16", 1024, 16, 2, 640, 512),
    ("f32", 128, 16, 2, 200, 150),
    ("f32", 64, 24, 4, 65, 70)])
def test_grouped_fo_matches_oracle(dtype, d, Hq, q, N, T):
    L = synth.make_layer(d, Hq, N, T, seed=Hq + N + T, dtype=dtype, outliers=True)
    g = {k: v.to(DEV) for k, v in L.items()}
    A = dtp.affinity_accumulate_grouped(g["X"], g["C"], g["W_gate"], g["W_up"], q)
    torch.cuda.synchronize()
    assert A.shape == (Hq // q, N)
    X, C, Wg, Wu = _np(L)
    ref = oracle.affinity_fo_qheads(X, C, Wg, Wu, q)
    assert _rel(A.cpu().numpy(), ref) <= (BF16_TOL if dtype == "bf16" else F32_TOL)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_grouped_with_one_head_per_group_is_the_plain_pass(dtype):
    L = synth.make_layer(256, 8, 384, 333, seed=5, dtype=dtype)
    g = {k: v.to(DEV) for k, v in L.items()}
    plain = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    grouped = dtp.affinity_accumulate_grouped(g["X"], g["C"], g["W_gate"], g["W_up"], 1)
    torch.cuda.synchronize()
    assert torch.equal(plain, grouped)


def test_grouped_down_term_and_determinism():
    d, Hq, q, N, T = 256, 16, 2, 384, 300
    L = synth.make_layer(d, Hq, N, T, seed=8, dtype="bf16")
    Dn = synth.make_down_inputs(d, Hq // q, 64, N, T, seed=9)
    g = {k: v.to(DEV) for k, v in L.items()}
    rms = Dn["rms"].to(DEV)
    A1, act2 = dtp.affinity_accumulate_grouped(g["X"], g["C"], g["W_gate"], g["W_up"], q, rms_next=rms)
    A2 = dtp.affinity_accumulate_grouped(g["X"], g["C"], g["W_gate"], g["W_up"], q)
    torch.cuda.synchronize()
    assert torch.equal(A1, A2)
    ref = oracle.down_activation(L["X"].double().numpy(), L["W_gate"].double().numpy(),
                                 L["W_up"].double().numpy(), Dn["rms"].double().numpy())
    assert _rel(act2.cpu().numpy(), ref) <= BF16_TOL


def test_grouped_two_launches_add_the_term_once():
    """32 query heads at 4 per group run as two 16-head launches; act2 must be added once."""
    d, Hq, q, N, T = 128, 32, 4, 256, 200
    L = synth.make_layer(d, Hq, N, T, seed=10, dtype="bf16")
    Dn = synth.make_down_inputs(d, Hq // q, 64, N, T, seed=11)
    g = {k: v.to(DEV) for k, v in L.items()}
    _, act2 = dtp.affinity_accumulate_grouped(g["X"], g["C"], g["W_gate"], g["W_up"], q, rms_next=Dn["rms"].to(DEV))
    _, act2_plain = dtp.affinity_accumulate_down(g["X"], g["C"][:8].contiguous(), g["W_gate"], g["W_up"],
                                                 Dn["rms"].to(DEV))
    torch.cuda.synchronize()
    assert torch.allclose(act2, act2_plain, rtol=1e-6, atol=0)


@pytest.mark.parametrize("d,Hq,q,N,T", [(256, 16, 2, 384, 300), (128, 32, 4, 300, 257), (64, 6, 3, 130, 129)])
def test_grouped_add_matches_oracle(d, Hq, q, N, T):
    L = synth.make_layer(d, Hq, N, T, seed=d + Hq, dtype="bf16", outliers=True)
    g = {k: v.to(DEV) for k, v in L.items()}
    A = dtp.affinity_add_accumulate_grouped(g["C"], g["W_gate"], g["W_up"], q)
    torch.cuda.synchronize()
    ref = oracle.affinity_add_qheads(L["C"].double().numpy(), L["W_gate"].double().numpy(),
                                     L["W_up"].double().numpy(), q)
    assert _rel(A.cpu().numpy(), ref) <= BF16_TOL


def test_grouped_add_one_head_per_group_is_plain():
    L = synth.make_layer(256, 8, 384, 333, seed=6, dtype="bf16")
    g = {k: v.to(DEV) for k, v in L.items()}
    plain = dtp.affinity_add_accumulate(g["C"], g["W_gate"], g["W_up"])
    grouped = dtp.affinity_add_accumulate_grouped(g["C"], g["W_gate"], g["W_up"], 1)
    torch.cuda.synchronize()
    assert torch.equal(plain, grouped)


def test_grouped_sampled_neurons_at_qwen_size():
    """The Qwen3-0.6B layer with its 16 query heads (2 per KV group) at 16384 tokens; two whole
    128-neuron tiles (the middle one and the last) and 24 sampled neurons checked against the oracle,
    by relative Frobenius error and every entry within 2%."""
    w = synth.WORKLOADS["qwen3_0.6b_layer"]
    L = synth.make_layer(w.d, 16, w.N, w.T, seed=w.seed, dtype="bf16", outliers=True, device=DEV)
    A = dtp.affinity_accumulate_grouped(L["X"], L["C"], L["W_gate"], L["W_up"], 2)
    torch.cuda.synchronize()
    mid = (w.N // 128) // 2 * 128
    rows = np.unique(np.concatenate([np.arange(mid, mid + 128), np.arange(w.N - 128, w.N),
                                     np.random.default_rng(0).choice(w.N, 24, replace=False)]))
    sub = {k: L[k].cpu() for k in ("X", "C")}
    ref = oracle.affinity_fo_qheads(sub["X"].double().numpy(), sub["C"].double().numpy(),
                                    L["W_gate"][rows].cpu().double().numpy(), L["W_up"][rows].cpu().double().numpy(), 2)
    got = A[:, rows].cpu().numpy()
    assert _rel(got, ref) <= BF16_TOL
    assert np.all(np.abs(got - ref) <= 2e-2 * np.abs(ref) + 1e-6 * np.abs(ref).max())


def test_grouped_rejects_bad_group_sizes():
    L = synth.make_layer(64, 6, 64, 16, seed=1, dtype="bf16", device=DEV)
    with pytest.raises(ValueError):
        dtp.affinity_accumulate_grouped(L["X"], L["C"], L["W_gate"], L["W_up"], 4)
    with pytest.raises(dtp.DTPError):
        dtp.affinity_grouped_workspace_size(16, 64, 34, 2, 64, dtp.DTP_BF16)   # 17 KV groups
