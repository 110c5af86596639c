"""GPU parity of the whole-model optimiser (Sec. 3, Eq. objective with both edges) against the oracle.

Both sides get the same fp32 S_up and S_down; the contract is bit-exact on
every layer's head partition and neuron assignment, on J in units of 2^-43
and on the iteration count.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_13846_gb300 import dtp, synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _model(L, G, N, seed, kind="lognormal"):
    Su = np.stack([synth.make_affinity_matrix(G, N, seed=seed + i, kind=kind).numpy() for i in range(L)])
    Sd = np.stack([synth.make_affinity_matrix(G, N, seed=seed + 500 + i, kind=kind).numpy()
                   for i in range(max(L - 1, 1))])[: L - 1]
    return Su.astype(np.float32), Sd.astype(np.float32)


def _compare(Su, Sd, D, iters):
    gSu = torch.as_tensor(Su, device=DEV).contiguous()
    gSd = torch.as_tensor(Sd, device=DEV).contiguous() if Su.shape[0] > 1 else None
    res = dtp.search_chain(gSu, gSd, D, iters)
    ref = oracle.chain_search(Su, Sd if Su.shape[0] > 1 else None, D, iters)
    np.testing.assert_array_equal(res["h"].cpu().numpy(), ref["h"])
    np.testing.assert_array_equal(res["nu"].cpu().numpy(), ref["nu"])
    assert int(res["J_q"]) == ref["J_q"]
    assert int(res["iters_done"]) == ref["iters_done"]
    assert float(res["J"]) == ref["J"]
    return ref


@pytest.mark.parametrize("L,G,N,D", [(1, 8, 256, 2), (2, 8, 256, 2), (4, 8, 512, 4), (3, 2, 4, 2),
                                     (5, 6, 96, 3), (3, 8, 64, 8), (6, 8, 3072, 2)])
@pytest.mark.parametrize("kind", ["lognormal", "integer"])
def test_chain_matches_oracle(L, G, N, D, kind):
    Su, Sd = _model(L, G, N, seed=L * 100 + N + D, kind=kind)
    _compare(Su, Sd, D, 10)


@pytest.mark.parametrize("iters", [1, 2])
def test_chain_iteration_cap(iters):
    Su, Sd = _model(4, 8, 256, seed=9)
    _compare(Su, Sd, 4, iters)


def test_chain_qwen_shaped_28_layers_d4():
    """The 28-layer Qwen3-0.6B shape (G=8, N=3072) at D=4, synthetic affinities."""
    Su, Sd = _model(28, 8, 3072, seed=100)
    ref = _compare(Su, Sd, 4, 10)
    assert ref["J"] > 55 / 4    # beats a random layout's expectation (2L-1)/D


def test_chain_from_gpu_affinities():
    """Three Qwen-shaped layers end to end: up edges from the affinity pass, down edges from
    the fused activation term, ||b_gk||^2 and finalize; then both searches on the same matrices."""
    w = synth.WORKLOADS["qwen3_0.6b_model"]
    T, R = 512, 512
    ups, downs = [], []
    for i in range(3):
        Lr = synth.make_workload_layer(w, i, T=T, device=DEV)
        Dn = synth.make_down_inputs(w.d, w.G, R, w.N, T, seed=w.seed + 50 + i, device=DEV)
        A, act2 = dtp.affinity_accumulate_down(Lr["X"], Lr["C"], Lr["W_gate"], Lr["W_up"], Dn["rms"])
        dtp.affinity_finalize(A, T)
        ups.append(A)
        if i < 2:
            bn = dtp.down_weight_sqnorm(Dn["Wqkv"], Dn["gamma"], Dn["W_down"])
            downs.append(dtp.down_finalize(act2, bn, T))
    Su = torch.stack(ups).contiguous().cpu().numpy()
    Sd = torch.stack(downs).contiguous().cpu().numpy()
    for D in (2, 4):
        _compare(Su, Sd, D, 10)


def test_chain_invalid_entry_reported():
    Su, Sd = _model(3, 8, 64, seed=4)
    Sd[1, 2, 3] = -1.0
    with pytest.raises(dtp.DTPError) as e:
        dtp.search_chain(torch.as_tensor(Su, device=DEV), torch.as_tensor(Sd, device=DEV), 2, 10)
    assert e.value.status == dtp.DTP_ERR_ARG
