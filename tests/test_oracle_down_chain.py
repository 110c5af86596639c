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
