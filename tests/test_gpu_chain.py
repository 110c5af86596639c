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


# ------------------------------------------------------------- ablations ----

from paper_2609_13846_gb300 import ablation  # noqa: E402


def _compare_ablation(Su, Sd, D, iters, kind):
    Lyr = Su.shape[0]
    mh, mn, mini = ablation.ablation_masks(Lyr, kind)
    gSu = torch.as_tensor(Su, device=DEV).contiguous()
    gSd = torch.as_tensor(Sd, device=DEV).contiguous() if Lyr > 1 else None
    res = dtp.search_chain(gSu, gSd, D, iters, move_heads=mh, move_neurons=mn, minimize=mini)
    ref = oracle.chain_search(Su, Sd if Lyr > 1 else None, D, iters, move_heads=mh, move_neurons=mn, minimize=mini)
    np.testing.assert_array_equal(res["h"].cpu().numpy(), ref["h"])
    np.testing.assert_array_equal(res["nu"].cpu().numpy(), ref["nu"])
    assert int(res["J_q"]) == ref["J_q"]
    assert int(res["iters_done"]) == ref["iters_done"]
    assert float(res["J"]) == ref["J"]
    return ref


@pytest.mark.parametrize("kind", ["anti", "heads_only", "neurons_only", "layers2", "layers3"])
@pytest.mark.parametrize("L,G,N,D", [(6, 8, 256, 2), (6, 8, 512, 4), (3, 6, 96, 3), (4, 8, 64, 8), (1, 8, 128, 4)])
def test_chain_ablations_match_oracle(kind, L, G, N, D):
    if kind.startswith("layers") and int(kind[6:]) > L:
        pytest.skip("subset larger than the model")
    Su, Sd = _model(L, G, N, seed=7 * L + N + D)
    _compare_ablation(Su, Sd, D, 10, kind)


@pytest.mark.parametrize("kind", ["anti", "neurons_only", "layers4"])
def test_chain_ablations_qwen_shaped(kind):
    """28 layers x (G=8, N=3072) at D=4: the Table 4 ablations, bit-exact."""
    Su, Sd = _model(28, 8, 3072, seed=100)
    _compare_ablation(Su, Sd, 4, 10, kind)


def test_chain_anti_on_integer_ties():
    """Integer-valued affinities leave many equal gains; minimising must pick the same canonical layout."""
    Su, Sd = _model(5, 8, 256, seed=3, kind="integer")
    for D in (2, 4):
        _compare_ablation(Su, Sd, D, 10, "anti")


@pytest.mark.parametrize("L,G,N,D", [(1, 8, 256, 2), (5, 8, 384, 4), (28, 8, 3072, 4), (3, 6, 96, 3)])
def test_chain_score_matches_oracle(L, G, N, D):
    Su, Sd = _model(L, G, N, seed=L + N)
    gSu = torch.as_tensor(Su, device=DEV).contiguous()
    gSd = torch.as_tensor(Sd, device=DEV).contiguous() if L > 1 else None
    for seed in (1000, 1001, 1002):
        h, nu = ablation.random_layout(L, G, N, D, seed)
        r = dtp.chain_score(gSu, gSd, torch.as_tensor(h, device=DEV), torch.as_tensor(nu, device=DEV), D)
        ref_e = oracle.chain_edge_scores(Su, Sd if L > 1 else None, h, nu)
        np.testing.assert_array_equal(r["edge_q"].cpu().numpy(), ref_e)
        assert int(r["J_q"]) == int(ref_e.sum()) == oracle.chain_score(Su, Sd if L > 1 else None, h, nu)
    # the optimiser's own layout scores its own J
    res = dtp.search_chain(gSu, gSd, D, 10)
    r = dtp.chain_score(gSu, gSd, res["h"], res["nu"], D)
    assert int(r["J_q"]) == int(res["J_q"])


def test_chain_score_rejects_out_of_range_layout():
    Su, Sd = _model(3, 8, 64, seed=5)
    h, nu = ablation.random_layout(3, 8, 64, 4, 1000)
    nu[1, 7] = 4
    with pytest.raises(dtp.DTPError) as e:
        dtp.chain_score(torch.as_tensor(Su, device=DEV), torch.as_tensor(Sd, device=DEV),
                        torch.as_tensor(h, device=DEV), torch.as_tensor(nu, device=DEV), 4)
    assert e.value.status == dtp.DTP_ERR_ARG


@pytest.mark.parametrize("D", [2, 4])
def test_random_layouts_score_one_over_D_per_edge(D):
    """A uniform random balanced layout co-locates 1/D of each edge's mass in expectation (Sec. 3: a
    random layout scores (2L-1)/D): the mean over 256 seeded layouts, each scored on the GPU, lies
    within five standard errors of 1/D on every edge and of (2L-1)/D in total."""
    L, G, N = 4, 8, 3072
    Su, Sd = _model(L, G, N, seed=77)
    gSu = torch.as_tensor(Su, device=DEV).contiguous()
    gSd = torch.as_tensor(Sd, device=DEV).contiguous()
    n = 256
    edges = []
    for seed in range(2000, 2000 + n):
        h, nu = ablation.random_layout(L, G, N, D, seed)
        r = dtp.chain_score(gSu, gSd, torch.as_tensor(h, device=DEV), torch.as_tensor(nu, device=DEV), D)
        edges.append(r["edge_q"].double().cpu() / 2.0 ** 43)
    E = torch.stack(edges)                       # [n, 2L-1] co-located fraction of each edge
    se = E.std(0) / n ** 0.5
    assert torch.all((E.mean(0) - 1.0 / D).abs() <= 5 * se + 1e-4), (E.mean(0), se)
    J = E.sum(1)
    assert abs(float(J.mean()) - (2 * L - 1) / D) <= 5 * float(J.std()) / n ** 0.5 + 1e-4
