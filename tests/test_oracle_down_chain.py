"""Pins of the oracle's down-edge score and whole-model objective (Sec. 3).

Down edge: neuron k of layer i writes alpha_k w^d_k into the residual; through
the next layer's pre-norm (gain gamma', rms r') it reaches KV group g's q/k/v
projections as (alpha_k / r') W^qkv_g (gamma' . w^d_k), so the score is
S_down[g,k] = E_t[alpha_k^2 / r'^2] ||b_gk||^2.  The first test simulates that
removal through the residual stream and the next layer's projections.

Whole model: Eq. objective sums the co-located unit-mass up-edge and down-edge
affinities over all layers; the optimiser alternates exact neuron and head
steps.  Pins: brute force over every layout of tiny models, block-step
exactness, monotonicity, and the paper's random-layout expectation (2L-1)/L.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
from paper_2609_13846_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_printed.json")


def _silu(z):
    return z / (1.0 + np.exp(-z))


def _down_setup(seed=0, T=40, d=12, N=6, G=3, R=5):
    rng = np.random.default_rng(seed)
    return dict(X=rng.standard_normal((T, d)), Wg=rng.standard_normal((N, d)) * 0.4,
                Wu=rng.standard_normal((N, d)) * 0.4, Wd=rng.standard_normal((d, N)) * 0.3,
                base=rng.standard_normal((T, d)), gamma=1.0 + 0.3 * rng.standard_normal(d),
                rms=0.5 + rng.random(T), Wqkv=rng.standard_normal((G, R, d)) * 0.2)


def _oracle_down(s):
    act2 = oracle.down_activation(s["X"], s["Wg"], s["Wu"], s["rms"])
    bn = oracle.down_weight_sqnorm(s["Wqkv"], s["gamma"], s["Wd"])
    return oracle.down_score(act2, bn, s["X"].shape[0])


def test_down_edge_is_the_removed_write_seen_by_the_next_layer():
    """Simulate the residual write of every neuron, the next layer's pre-norm with its rms held
    fixed, and each KV group's q/k/v rows; removing neuron k changes group g's projections by
    exactly its share, whose mean squared norm is S_down[g,k]."""
    s = _down_setup()
    T, N, G = s["X"].shape[0], s["Wg"].shape[0], s["Wqkv"].shape[0]
    alpha = _silu(s["X"] @ s["Wg"].T) * (s["X"] @ s["Wu"].T)          # [T, N] neuron activations
    resid = s["base"] + alpha @ s["Wd"].T                                  # residual after the FFN
    def qkv(x):                                                            # next layer, rms held fixed
        y = s["gamma"] * x / s["rms"][:, None]
        return np.einsum("grd,td->tgr", s["Wqkv"], y)
    full = qkv(resid)
    expect = np.zeros((G, N))
    for k in range(N):
        without = qkv(resid - np.outer(alpha[:, k], s["Wd"][:, k]))
        expect[:, k] = ((full - without) ** 2).sum(axis=2).mean(axis=0)
    np.testing.assert_allclose(_oracle_down(s), expect, rtol=1e-10)


def test_down_edge_scalings():
    s = _down_setup(seed=1)
    S = _oracle_down(s)
    s2 = dict(s, gamma=2.0 * s["gamma"])
    np.testing.assert_allclose(_oracle_down(s2), 4.0 * S, rtol=1e-12)
    s3 = dict(s, rms=3.0 * s["rms"])
    np.testing.assert_allclose(_oracle_down(s3), S / 9.0, rtol=1e-12)
    Wd = s["Wd"].copy()
    Wd[:, 2] = 0.0
    assert np.all(_oracle_down(dict(s, Wd=Wd))[:, 2] == 0.0)


def test_down_weight_norm_invariant_to_row_rotation_and_equivariant_in_neurons():
    s = _down_setup(seed=2)
    bn = oracle.down_weight_sqnorm(s["Wqkv"], s["gamma"], s["Wd"])
    Q, _ = np.linalg.qr(np.random.default_rng(3).standard_normal((5, 5)))
    rot = np.einsum("ij,gjd->gid", Q, s["Wqkv"])
    np.testing.assert_allclose(oracle.down_weight_sqnorm(rot, s["gamma"], s["Wd"]), bn, rtol=1e-10)
    perm = np.array([3, 0, 5, 1, 4, 2])
    np.testing.assert_array_equal(oracle.down_weight_sqnorm(s["Wqkv"], s["gamma"], s["Wd"][:, perm]), bn[:, perm])
    act2 = oracle.down_activation(s["X"], s["Wg"], s["Wu"], s["rms"])
    np.testing.assert_array_equal(oracle.down_activation(s["X"], s["Wg"][perm], s["Wu"][perm], s["rms"]), act2[perm])


# --------------------------------------------------------- normalisation ----

def test_unit_mass_normalisation():
    S = synth.make_affinity_matrix(4, 50, seed=3).numpy()
    n = oracle.normalize_unit_mass(S)
    total = int(n.sum())
    assert total <= 2 ** 43 and total >= 2 ** 43 - 2 * S.size
    ratio = n / 2.0 ** 43
    np.testing.assert_allclose(ratio, S / S.sum(), rtol=1e-6, atol=2.0 ** -36)   # 40-bit pre-quantisation
    for k in (-5, 7):
        np.testing.assert_array_equal(oracle.normalize_unit_mass(S * np.float32(2.0 ** k)), n)
    assert not oracle.normalize_unit_mass(np.zeros((2, 3), np.float32)).any()
    with pytest.raises(ValueError):
        oracle.normalize_unit_mass(np.array([[1.0, -1.0]], np.float32))


# ---------------------------------------------------------- whole model -----

def _balanced(n, D):
    cap = n // D
    for a in itertools.product(range(D), repeat=n):
        if all(a.count(l) == cap for l in range(D)):
            yield np.array(a, dtype=np.int32)


def _random_model(L, G, N, seed, kind="lognormal"):
    Su = np.stack([synth.make_affinity_matrix(G, N, seed=seed + i, kind=kind).numpy() for i in range(L)])
    Sd = np.stack([synth.make_affinity_matrix(G, N, seed=seed + 100 + i, kind=kind).numpy() for i in range(L - 1)]) \
        if L > 1 else np.zeros((0, G, N), np.float32)
    return Su, Sd


@pytest.mark.parametrize("L,seed", [(2, 0), (2, 1), (3, 2)])
def test_chain_ascent_against_brute_force(L, seed):
    """Every layout of a tiny model (G=2, N=4, D=2): the ascent's J is the J of its layout and
    does not exceed the global optimum; the first iteration's two block steps are exact."""
    G, N, D = 2, 4, 2
    Su, Sd = _random_model(L, G, N, seed)
    hs, nus = list(_balanced(G, D)), list(_balanced(N, D))
    best = max(oracle.chain_score(Su, Sd, np.stack(h), np.stack(nu))
               for h in itertools.product(hs, repeat=L) for nu in itertools.product(nus, repeat=L))
    res = oracle.chain_search(Su, Sd, D, 10)
    assert res["J_q"] == oracle.chain_score(Su, Sd, res["h"], res["nu"])
    assert res["J_q"] <= best
    one = oracle.chain_search(Su, Sd, D, 1)
    h0 = np.stack([np.array([(g * D) // G for g in range(G)], np.int32)] * L)
    best_nu = max(oracle.chain_score(Su, Sd, h0, np.stack(nu)) for nu in itertools.product(nus, repeat=L))
    assert oracle.chain_score(Su, Sd, h0, one["nu"]) == best_nu
    best_h = max(oracle.chain_score(Su, Sd, np.stack(h), one["nu"]) for h in itertools.product(hs, repeat=L))
    assert one["J_q"] == best_h


def test_chain_ascent_monotone_and_stops():
    Su, Sd = _random_model(4, 8, 64, seed=11)
    trace = [oracle.chain_search(Su, Sd, 4, i)["J_q"] for i in range(1, 6)]
    assert all(b >= a for a, b in zip(trace, trace[1:]))
    res = oracle.chain_search(Su, Sd, 4, 10)
    assert res["J_q"] == trace[-1] or res["iters_done"] < 5
    assert 0.0 < res["J"] <= 2 * 4 - 1


def test_chain_single_layer_is_up_edge_only():
    Su, _ = _random_model(1, 8, 48, seed=5)
    res = oracle.chain_search(Su, None, 2, 10)
    assert 0.5 <= res["J"] <= 1.0


def test_random_layout_expectation_matches_paper():
    """E[J] of a uniform random balanced layout is (2L-1)/L devices: 13.75 for the 28-layer
    Qwen3-0.6B and 7.75 for the 16-layer Danube3-500M at L=4 (Table 4 caption)."""
    gold = json.load(open(GOLDEN))
    for key, layers in (("random_layout_expected_J_qwen", 28), ("random_layout_expected_J_danube", 16)):
        Su, Sd = _random_model(layers, 8, 64, seed=7)
        rng = np.random.default_rng(1)
        vals = []
        for _ in range(60):
            h = np.stack([rng.permutation(np.repeat(np.arange(4), 2)) for _ in range(layers)]).astype(np.int32)
            nu = np.stack([rng.permutation(np.repeat(np.arange(4), 16)) for _ in range(layers)]).astype(np.int32)
            vals.append(oracle.chain_score(Su, Sd, h, nu) / 2.0 ** 43)
        mean, sem = float(np.mean(vals)), float(np.std(vals) / np.sqrt(len(vals)))
        assert abs(mean - gold[key]["value"]) < 4 * sem + 0.05


# ------------------------------------------------------------- ablations ----
# Sec. 3 "Optimiser": restricting which layers move, freezing heads or
# neurons, or minimising J gives the ablation layouts of Table 4.

from paper_2609_13846_gb300 import ablation  # noqa: E402


def _contiguous(L, G, N, D):
    h = np.stack([np.array([(g * D) // G for g in range(G)], np.int32)] * L)
    nu = np.stack([np.array([(k * D) // N for k in range(N)], np.int32)] * L)
    return h, nu


@pytest.mark.parametrize("L,seed", [(2, 3), (3, 4)])
def test_neurons_only_is_the_exact_optimum_over_neurons(L, seed):
    """Heads frozen contiguous: the neuron steps of different layers are independent given h, so
    one sweep reaches the global optimum over every nu; brute force over all of them."""
    G, N, D = 2, 4, 2
    Su, Sd = _random_model(L, G, N, seed)
    h0, nu0 = _contiguous(L, G, N, D)
    nus = list(_balanced(N, D))
    best = max(oracle.chain_score(Su, Sd, h0, np.stack(nu)) for nu in itertools.product(nus, repeat=L))
    res = oracle.chain_search(Su, Sd, D, 10, move_heads=np.zeros(L), move_neurons=np.ones(L))
    np.testing.assert_array_equal(res["h"], h0)
    assert res["J_q"] == best == oracle.chain_score(Su, Sd, res["h"], res["nu"])
    worst = min(oracle.chain_score(Su, Sd, h0, np.stack(nu)) for nu in itertools.product(nus, repeat=L))
    anti = oracle.chain_search(Su, Sd, D, 10, move_heads=np.zeros(L), minimize=True)
    assert anti["J_q"] == worst == oracle.chain_score(Su, Sd, anti["h"], anti["nu"])


@pytest.mark.parametrize("L,seed", [(2, 5), (3, 6)])
def test_heads_only_is_the_exact_optimum_over_heads(L, seed):
    G, N, D = 4, 4, 2
    Su, Sd = _random_model(L, G, N, seed)
    h0, nu0 = _contiguous(L, G, N, D)
    hs = list(_balanced(G, D))
    best = max(oracle.chain_score(Su, Sd, np.stack(h), nu0) for h in itertools.product(hs, repeat=L))
    res = oracle.chain_search(Su, Sd, D, 10, move_heads=np.ones(L), move_neurons=np.zeros(L))
    np.testing.assert_array_equal(res["nu"], nu0)
    assert res["J_q"] == best
    worst = min(oracle.chain_score(Su, Sd, np.stack(h), nu0) for h in itertools.product(hs, repeat=L))
    anti = oracle.chain_search(Su, Sd, D, 10, move_neurons=np.zeros(L), minimize=True)
    assert anti["J_q"] == worst


@pytest.mark.parametrize("L,seed", [(2, 7), (3, 8)])
def test_anti_optimised_against_brute_force(L, seed):
    """Minimising J: the result's J is its layout's J, at or above the global minimum, and the
    first sweep's neuron and head steps are exact minimisers."""
    G, N, D = 2, 4, 2
    Su, Sd = _random_model(L, G, N, seed)
    hs, nus = list(_balanced(G, D)), list(_balanced(N, D))
    worst = min(oracle.chain_score(Su, Sd, np.stack(h), np.stack(nu))
                for h in itertools.product(hs, repeat=L) for nu in itertools.product(nus, repeat=L))
    res = oracle.chain_search(Su, Sd, D, 10, minimize=True)
    assert res["J_q"] == oracle.chain_score(Su, Sd, res["h"], res["nu"]) >= worst
    one = oracle.chain_search(Su, Sd, D, 1, minimize=True)
    h0, _ = _contiguous(L, G, N, D)
    assert oracle.chain_score(Su, Sd, h0, one["nu"]) == min(
        oracle.chain_score(Su, Sd, h0, np.stack(nu)) for nu in itertools.product(nus, repeat=L))
    assert one["J_q"] == min(oracle.chain_score(Su, Sd, np.stack(h), one["nu"]) for h in itertools.product(hs, repeat=L))


def test_layer_subset_keeps_other_layers_contiguous():
    L, G, N, D = 6, 8, 64, 4
    Su, Sd = _random_model(L, G, N, seed=12)
    h0, nu0 = _contiguous(L, G, N, D)
    mh, mn, mini = ablation.ablation_masks(L, "layers2")
    assert list(np.flatnonzero(mh)) == [0, 3] and not mini
    res = oracle.chain_search(Su, Sd, D, 10, move_heads=mh, move_neurons=mn)
    for i in range(L):
        if not mh[i]:
            np.testing.assert_array_equal(res["h"][i], h0[i])
            np.testing.assert_array_equal(res["nu"][i], nu0[i])
    assert res["J_q"] == oracle.chain_score(Su, Sd, res["h"], res["nu"])
    assert res["J_q"] >= oracle.chain_score(Su, Sd, h0, nu0)
    frozen = oracle.chain_search(Su, Sd, D, 10, move_heads=np.zeros(L), move_neurons=np.zeros(L))
    assert frozen["J_q"] == oracle.chain_score(Su, Sd, h0, nu0) and frozen["iters_done"] == 2


def test_ablation_ordering_invariants():
    """anti <= contiguous <= neurons-only <= optimised (the full ascent's first neuron sweep is
    the neurons-only layout, and every later step can only raise J); anti < random mean < optimised."""
    L, G, N, D = 8, 8, 128, 4
    Su, Sd = _random_model(L, G, N, seed=21)
    h0, nu0 = _contiguous(L, G, N, D)
    J = {k: oracle.chain_search(Su, Sd, D, 10, *[None if m is None else m for m in ablation.ablation_masks(L, k)[:2]],
                                minimize=ablation.ablation_masks(L, k)[2])["J_q"]
         for k in ("optimised", "anti", "heads_only", "neurons_only", "layers4")}
    Jc = oracle.chain_score(Su, Sd, h0, nu0)
    assert J["anti"] <= Jc <= J["neurons_only"] <= J["optimised"]
    assert Jc <= J["heads_only"] and Jc <= J["layers4"]
    rnd = np.mean([oracle.chain_score(Su, Sd, *ablation.random_layout(L, G, N, D, 1000 + s)) for s in range(8)])
    assert J["anti"] < rnd < J["optimised"]


def test_edge_scores_sum_to_the_objective_and_give_fractions():
    L, G, N, D = 5, 8, 96, 4
    Su, Sd = _random_model(L, G, N, seed=30)
    h, nu = ablation.random_layout(L, G, N, D, 1001)
    e = oracle.chain_edge_scores(Su, Sd, h, nu)
    assert e.shape == (2 * L - 1,) and int(e.sum()) == oracle.chain_score(Su, Sd, h, nu)
    # every layer on one device: each edge keeps all of its unit mass (up to the floor per entry)
    h1, nu1 = np.zeros((L, G), np.int32), np.zeros((L, N), np.int32)
    e1 = oracle.chain_edge_scores(Su, Sd, h1, nu1)
    assert np.all(e1 <= 2 ** 43) and np.all(e1 >= 2 ** 43 - G * N)
    # a layer whose heads and neurons sit on disjoint devices keeps none of its up edge
    h2 = h1.copy(); h2[2] = 1
    assert oracle.chain_edge_scores(Su, Sd, h2, nu1)[4] == 0


def test_evenly_spaced_layers():
    assert ablation.evenly_spaced_layers(28, 4) == [0, 7, 14, 21]
    for L, n in ((28, 8), (28, 12), (16, 4), (16, 12), (5, 5)):
        ls = ablation.evenly_spaced_layers(L, n)
        assert ls[0] == 0 and len(set(ls)) == n and ls == sorted(ls) and ls[-1] < L
    with pytest.raises(ValueError):
        ablation.evenly_spaced_layers(4, 5)
    h, nu = ablation.random_layout(3, 8, 64, 4, 1000)
    assert all(np.bincount(r, minlength=4).tolist() == [2] * 4 for r in h)
    assert all(np.bincount(r, minlength=4).tolist() == [16] * 4 for r in nu)
