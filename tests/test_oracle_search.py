"""Pins of the layout-search oracle (Sec. 3 "Objective" and "Optimiser").

The oracle's neuron step (exact balanced assignment, lexicographically
smallest optimum), head step (exhaustive labelled partitions) and coordinate
ascent are checked against brute force over every layout on tiny inputs, the
textbook Hungarian method, the counts the paper prints, and Monte-Carlo
expectations of random balanced layouts.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2609_13846_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_printed.json")


def _balanced_assignments(N, D):
    """Every balanced assignment of N items to D labels, in lexicographic order."""
    cap = N // D
    for nu in itertools.product(range(D), repeat=N):
        if all(nu.count(l) == cap for l in range(D)):
            yield nu


def _brute_neuron_step(q, h, D):
    G, N = q.shape
    best, arg, count = None, None, 0
    for nu in _balanced_assignments(N, D):
        s = sum(int(q[g, k]) for g in range(G) for k in range(N) if h[g] == nu[k])
        if best is None or s > best:
            best, arg, count = s, nu, 1
        elif s == best:
            count += 1
    return np.array(arg, dtype=np.int32), best, count == 1


def _brute_head_step(q, nu, D):
    G, N = q.shape
    best, arg = None, None
    for h in _balanced_assignments(G, D):
        s = sum(int(q[g, k]) for g in range(G) for k in range(N) if h[g] == nu[k])
        if best is None or s > best:
            best, arg = s, h
    return np.array(arg, dtype=np.int32), best


def _rand_q(G, N, seed, kind="lognormal"):
    A = synth.make_affinity_matrix(G, N, seed, kind=kind).numpy()
    q, _ = oracle.quantize(A)
    return A, q


# ---------------------------------------------------------------- counts ----

def test_partition_count_printed_in_paper():
    gold = json.load(open(GOLDEN))["partitions_G8_L4"]
    assert oracle.count_partitions(8, 4) == gold["value"]


@pytest.mark.parametrize("G,D", [(2, 2), (4, 2), (6, 3), (8, 2), (8, 4), (8, 8), (6, 2), (9, 3)])
def test_partition_count_formula(G, D):
    """The walked count equals G!/((G/L)!)^L (Sec. 3 'Optimiser')."""
    assert oracle.count_partitions(G, D) == math.factorial(G) // math.factorial(G // D) ** D


# ---------------------------------------------------------- quantisation ----

def test_quantize_definition():
    A = np.array([[0.75, 0.1], [0.0, 3.0e-3]], dtype=np.float32)
    q, e = oracle.quantize(A)
    assert e == 0  # 0.75 = 0.75 * 2^0
    assert q[0, 0] == int(0.75 * 2 ** 40)
    assert q[1, 0] == 0
    assert q[0, 1] == math.floor(float(np.float32(0.1)) * 2 ** 40)
    assert q.max() < 2 ** 40 and q.max() >= 2 ** 39


def test_quantize_power_of_two_scale_invariance():
    """Unit-mass normalisation is scale-free; so is the fixed-point form under 2^k scalings."""
    A, q = _rand_q(4, 64, 0)
    for k in (-7, 3, 20):
        q2, _ = oracle.quantize(A * np.float32(2.0 ** k))
        np.testing.assert_array_equal(q2, q)


def test_quantize_rejects_negative_and_nan():
    for bad in (-1.0, float("nan"), float("inf")):
        with pytest.raises(ValueError):
            oracle.quantize(np.array([[1.0, bad]], dtype=np.float32))


def test_quantize_zero_matrix():
    q, e = oracle.quantize(np.zeros((2, 4), dtype=np.float32))
    assert e == 0 and not q.any()


# ---------------------------------------------------------- neuron step -----

@pytest.mark.parametrize("G,N,D", [(2, 12, 2), (4, 12, 2), (3, 9, 3), (4, 8, 4), (6, 9, 3), (2, 8, 4)])
@pytest.mark.parametrize("kind", ["lognormal", "integer"])
def test_neuron_step_brute_force(G, N, D, kind):
    """Exact optimum and lexicographically smallest tie-break against all balanced assignments."""
    if G % D:
        h = np.array([g % D for g in range(G)], dtype=np.int32)
    else:
        h = np.array([(g * D) // G for g in range(G)], dtype=np.int32)
    for seed in range(3):
        _, q = _rand_q(G, N, 100 * seed + N + D, kind)
        nu_bf, best, uniq_bf = _brute_neuron_step(q, h, D)
        for general in (False, True):
            nu, uniq = oracle.neuron_step(q, h, D, general=general)
            assert oracle.assignment_gain(q, h, nu, D) == best
            np.testing.assert_array_equal(nu, nu_bf)
            assert uniq == uniq_bf


def test_neuron_step_all_ties_gives_contiguous():
    q = np.zeros((4, 12), dtype=np.int64)
    h = np.array([0, 1, 2, 0], dtype=np.int32)
    nu, uniq = oracle.neuron_step(q, h, 3)
    np.testing.assert_array_equal(nu, [0] * 4 + [1] * 4 + [2] * 4)
    assert not uniq


@pytest.mark.parametrize("N,D", [(60, 3), (64, 4), (48, 8), (40, 2)])
def test_neuron_step_matches_hungarian(N, D):
    """Slot-expanded matrix (N/D slots per device) solved by the textbook Hungarian method
    (Sec. 3: the best balanced nu_i is a linear assignment on I/L replicated slots)."""
    G = 8
    h = np.array([(g * D) // G for g in range(G)], dtype=np.int32)
    for seed in range(2):
        for kind in ("lognormal", "integer"):
            _, q = _rand_q(G, N, seed * 7 + N, kind)
            M = np.zeros((N, D), dtype=np.int64)
            for g in range(G):
                M[:, h[g]] += q[g]
            cap = N // D
            W = np.repeat(M, cap, axis=1)  # column s is a slot of device s // cap
            total, r2c = oracle.hungarian_max(W)
            nu, _ = oracle.neuron_step(q, h, D)
            assert oracle.assignment_gain(q, h, nu, D) == total
            assert sorted(r2c.tolist()) == list(range(N))


def _lex_smallest_by_fixing(q, h, D):
    """The lexicographically smallest optimal balanced assignment, straight from its definition:
    for k = 0, 1, ... give neuron k the smallest device with which the optimum total is still
    reachable, each test a textbook Hungarian solve of the slot-expanded matrix in which the rows of
    the neurons fixed so far keep only their device's slots.  The optimum is unique exactly when
    every step finds a single such device (a second optimum differs from the lexicographically
    smallest one first at some neuron k, and agrees with it before k)."""
    G, N = q.shape
    M = np.zeros((N, D), dtype=np.int64)
    for g in range(G):
        M[:, h[g]] += q[g]
    cap = N // D
    W = np.repeat(M, cap, axis=1)
    best, _ = oracle.hungarian_max(W)
    penalty = -(1 << 50)                 # far below any total the scores can reach (< 2^47 here)
    nu = np.zeros(N, dtype=np.int32)
    unique = True
    for k in range(N):
        keep = []
        for l in range(D):
            trial = W.copy()
            trial[k, :] = penalty
            trial[k, l * cap:(l + 1) * cap] = W[k, l * cap:(l + 1) * cap]
            if oracle.hungarian_max(trial)[0] == best:
                keep.append((l, trial))
        assert keep, "no device keeps the optimum"
        unique &= len(keep) == 1
        nu[k], W = keep[0]
    return nu, best, unique


@pytest.mark.parametrize("G,N,D", [(8, 48, 4), (8, 96, 3), (6, 60, 3), (8, 64, 8), (4, 40, 2), (8, 72, 4)])
def test_neuron_step_tie_break_by_fixing(G, N, D):
    """The oracle's lexicographic tie-break (successive shortest paths, then LP duality and Hall's
    condition) and its uniqueness flag against the plain definition of the lexicographically smallest
    optimum, on tie-heavy integer scores far beyond brute-force sizes (Sec. 3 "Optimiser"; ties to
    the lowest index), and on continuous scores with a unique optimum."""
    h = np.array([(g * D) // G for g in range(G)] if G % D == 0 else [g % D for g in range(G)], dtype=np.int32)
    for seed, kind in ((0, "integer"), (1, "integer"), (2, "lognormal")):
        _, q = _rand_q(G, N, 500 + 10 * seed + N + D, kind)
        ref, best, ref_unique = _lex_smallest_by_fixing(q, h, D)
        for general in (False, True):
            nu, uniq = oracle.neuron_step(q, h, D, general=general)
            assert oracle.assignment_gain(q, h, nu, D) == best
            np.testing.assert_array_equal(nu, ref)
            assert uniq == ref_unique


def _qwen_layer_q(layer, T=64):
    """Exact scores of a Qwen3-0.6B-shaped layer (G = 8, N = 3072) from the oracle's affinity on a
    token slice of that layer's synthetic activations."""
    L = synth.make_workload_layer(synth.WORKLOADS["qwen3_0.6b_model"], layer, T=T)
    A = oracle.affinity_fo(*(L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up")))
    q, _ = oracle.quantize(A.astype(np.float32))
    return q


@pytest.mark.slow
@pytest.mark.parametrize("case", ["qwen_layer0", "qwen_layer1", "integer"])
def test_neuron_step_matches_hungarian_at_qwen_size(case):
    """Qwen-sized cross-check of the exact balanced assignment (Sec. 3 "Optimiser": a linear
    assignment on I/L replicated slots): N = 3072 neurons, D = 4, the 3072 x 3072 slot-expanded
    matrix solved by the textbook Hungarian method (O(n^3), about 20 s each) must reach the same
    optimum as the oracle's successive-shortest-path solver, for two layers of continuous scores
    (unique optimum certified) and one tie-heavy integer layer."""
    N, D = 3072, 4
    if case == "integer":
        _, q = _rand_q(8, N, 31, "integer")
        h = np.array([0, 0, 1, 1, 2, 2, 3, 3], dtype=np.int32)
    else:
        layer = int(case[-1])
        q = _qwen_layer_q(layer)
        h = np.array([0, 0, 1, 1, 2, 2, 3, 3] if layer == 0 else [0, 1, 2, 3, 3, 2, 1, 0], dtype=np.int32)
    M = np.zeros((N, D), dtype=np.int64)
    for g in range(q.shape[0]):
        M[:, h[g]] += q[g]
    cap = N // D
    total, r2c = oracle.hungarian_max(np.repeat(M, cap, axis=1))
    assert sorted(r2c.tolist()) == list(range(N))
    assert int(M[np.arange(N), r2c // cap].sum()) == total  # the Hungarian's own assignment
    nu, uniq = oracle.neuron_step(q, h, D)
    assert np.bincount(nu, minlength=D).tolist() == [cap] * D
    assert oracle.assignment_gain(q, h, nu, D) == total
    if case == "integer":
        assert not uniq  # integer scores in a small range: many optima, the tie-break decides
    else:
        assert uniq
        np.testing.assert_array_equal(nu, r2c // cap)  # a unique optimum: the same assignment


def test_neuron_step_d2_is_a_sort():
    """D = 2 reduces to sorting M_k0 - M_k1 (textbook): device 0 takes the top half."""
    _, q = _rand_q(4, 200, 5)
    h = np.array([0, 0, 1, 1], dtype=np.int32)
    nu, uniq = oracle.neuron_step(q, h, 2)
    diff = q[0] + q[1] - q[2] - q[3]
    order = sorted(range(200), key=lambda k: (-int(diff[k]), k))
    expect = np.ones(200, dtype=np.int32)
    expect[order[:100]] = 0
    np.testing.assert_array_equal(nu, expect)
    assert uniq


def test_neuron_step_general_matches_sort_for_d2_large():
    _, q = _rand_q(8, 3072, 9)
    h = np.array([0, 0, 0, 0, 1, 1, 1, 1], dtype=np.int32)
    a, _ = oracle.neuron_step(q, h, 2)
    b, _ = oracle.neuron_step(q, h, 2, general=True)
    np.testing.assert_array_equal(a, b)


# ------------------------------------------------------------ head step -----

@pytest.mark.parametrize("G,D", [(4, 2), (6, 3), (8, 4), (6, 2), (8, 2)])
@pytest.mark.parametrize("kind", ["lognormal", "integer"])
def test_head_step_brute_force(G, D, kind):
    N = 24
    for seed in range(2):
        _, q = _rand_q(G, N, seed + 31 * G + D, kind)
        nu = np.array(np.random.default_rng(seed).permutation(np.repeat(np.arange(D), N // D)),
                      dtype=np.int32)
        h_bf, best = _brute_head_step(q, nu, D)
        h, score = oracle.head_step(q, nu, D)
        assert score == best
        np.testing.assert_array_equal(h, h_bf)
        assert oracle.layout_score(q, h, nu) == best


# ---------------------------------------------------- coordinate ascent -----

def _search_trace(A, D, iters):
    """Scores after 1..iters iterations (each run restarts from the contiguous layout)."""
    return [oracle.search_layout(A, D, i)["score_q"] for i in range(1, iters + 1)]


@pytest.mark.parametrize("seed", range(4))
def test_ascent_below_global_optimum_and_monotone(seed):
    """Joint brute force over (h, nu) for G=4, N=8, D=2 bounds the ascent (Sec. 3 'Optimiser')."""
    A = synth.make_affinity_matrix(4, 8, seed).numpy()
    q, _ = oracle.quantize(A)
    glob = max(oracle.layout_score(q, np.array(h, dtype=np.int32), np.array(nu, dtype=np.int32))
               for h in _balanced_assignments(4, 2) for nu in _balanced_assignments(8, 2))
    res = oracle.search_layout(A, 2, 10)
    assert res["score_q"] <= glob
    trace = _search_trace(A, 2, 6)
    assert all(b >= a for a, b in zip(trace, trace[1:]))
    assert res["score_q"] == oracle.layout_score(q, res["h"], res["nu"])
    # the neuron step from the final h cannot improve the final layout
    nu2, _ = oracle.neuron_step(q, res["h"], 2)
    assert oracle.layout_score(q, res["h"], nu2) == res["score_q"]


def test_ascent_stops_without_strict_increase():
    A = synth.make_affinity_matrix(8, 96, 3).numpy()
    res = oracle.search_layout(A, 4, 10)
    assert 1 <= res["iters_done"] <= 10
    if res["iters_done"] < 10:
        longer = oracle.search_layout(A, 4, res["iters_done"] + 1)
        assert longer["score_q"] == res["score_q"]


def test_ascent_zero_matrix_returns_start_layout():
    A = np.zeros((8, 32), dtype=np.float32)
    res = oracle.search_layout(A, 4, 10)
    np.testing.assert_array_equal(res["h"], [0, 0, 1, 1, 2, 2, 3, 3])
    np.testing.assert_array_equal(res["nu"], np.repeat(np.arange(4), 8))
    assert res["score_q"] == 0 and res["score"] == 0.0 and res["iters_done"] == 2


def test_ascent_beats_contiguous_and_random():
    A = synth.make_affinity_matrix(8, 256, 11).numpy()
    q, _ = oracle.quantize(A)
    res = oracle.search_layout(A, 4, 10)
    contiguous = oracle.layout_score(q, np.repeat(np.arange(4), 2), np.repeat(np.arange(4), 64))
    assert res["score_q"] >= contiguous
    assert res["score"] > 0.25


def test_random_layout_expectation_is_one_over_L():
    """A uniform random balanced layout co-locates 1/L of an edge's mass in expectation
    (Sec. 3 'Objective'); with 2N-1 unit-mass edges this is the paper's (2N-1)/L, printed as
    13.75 (Qwen3-0.6B) and 7.75 (Danube3-500M) in the Table 4 caption."""
    gold = json.load(open(GOLDEN))
    A = synth.make_affinity_matrix(8, 512, 21).numpy()
    q, _ = oracle.quantize(A)
    total = int(q.sum())
    rng = np.random.default_rng(0)
    L = 4
    fr = []
    for _ in range(400):
        h = rng.permutation(np.repeat(np.arange(L), 2)).astype(np.int32)
        nu = rng.permutation(np.repeat(np.arange(L), 128)).astype(np.int32)
        fr.append(oracle.layout_score(q, h, nu) / total)
    mean, sem = float(np.mean(fr)), float(np.std(fr) / np.sqrt(len(fr)))
    assert abs(mean - 1 / L) < 4 * sem + 1e-3
    for key in ("random_layout_expected_J_qwen", "random_layout_expected_J_danube"):
        g = gold[key]
        assert g["edges"] == 2 * g["layers"] - 1
        assert abs(g["edges"] * mean - g["value"]) < g["edges"] * (4 * sem + 1e-3)


def test_search_d8_single_partition_is_global():
    """D = G = 8: every head partition is a relabelling, so one neuron step is globally optimal
    and the ascent stops after the second iteration."""
    A = synth.make_affinity_matrix(8, 64, 2).numpy()
    q, _ = oracle.quantize(A)
    res = oracle.search_layout(A, 8, 10)
    best = max(oracle.assignment_gain(q, np.arange(8, dtype=np.int32), nu, 8)
               for nu in [oracle.neuron_step(q, np.arange(8, dtype=np.int32), 8)[0]])
    assert res["score_q"] == best
    assert res["iters_done"] == 2


# ------------------------------------------------- global optimum (Sec. 3 "Objective") ----

import itertools as _it  # noqa: E402
import math as _math  # noqa: E402


def _balanced_labelings(n, D):
    cap = n // D
    for a in _it.product(range(D), repeat=n):
        if all(a.count(l) == cap for l in range(D)):
            yield np.array(a, dtype=np.int32)


@pytest.mark.parametrize("G,N,D,seed", [(4, 8, 2, 0), (4, 8, 2, 1), (6, 6, 3, 2), (4, 8, 4, 3), (2, 10, 2, 4)])
def test_global_layout_against_brute_force(G, N, D, seed):
    """The maximum over every labelled head partition and every balanced assignment equals the
    best exact neuron step over the unlabelled partitions; the ascent never exceeds it."""
    A = synth.make_affinity_matrix(G, N, seed=seed).numpy()
    q, _ = oracle.quantize(A)
    best = max(oracle.layout_score(q, h, nu) for h in _balanced_labelings(G, D) for nu in _balanced_labelings(N, D))
    g = oracle.global_layout(A, D)
    assert g["score_q"] == best == oracle.layout_score(q, g["h"], g["nu"])
    assert oracle.search_layout(A, D, 10)["score_q"] <= best


@pytest.mark.parametrize("G,D", [(8, 2), (8, 4), (8, 8), (6, 3), (6, 2), (4, 2), (12, 3), (12, 4), (16, 2)])
def test_global_layout_visits_every_unlabelled_partition_once(G, D):
    A = synth.make_affinity_matrix(G, 2 * D, seed=G + D).numpy()
    g = oracle.global_layout(A, D)
    cap = G // D
    assert g["parts"] == _math.factorial(G) // (_math.factorial(cap) ** D * _math.factorial(D))
    # canonical labelling: balanced, and each label first appears after every smaller one
    h = g["h"].tolist()
    assert all(h.count(l) == cap for l in range(D))
    firsts = [h.index(l) for l in range(D)]
    assert firsts == sorted(firsts) and firsts[0] == 0


def test_global_layout_ties_take_the_first_canonical_partition():
    """Tie-heavy integer affinities: the winner is the first canonical partition (in lexicographic
    order) reaching the maximum, with its lexicographically smallest optimal assignment."""
    G, N, D = 4, 8, 2
    for seed in range(6):
        A = synth.make_affinity_matrix(G, N, seed=50 + seed, kind="integer").numpy()
        q, _ = oracle.quantize(A)
        canon = [h for h in _balanced_labelings(G, D) if list(h).index(1) > 0 and h[0] == 0]
        best, first = -1, None
        for h in sorted(canon, key=tuple):
            nu, _ = oracle.neuron_step(q, h, D)
            v = oracle.layout_score(q, h, nu)
            if v > best:
                best, first = v, (h, nu)
        g = oracle.global_layout(A, D)
        assert g["score_q"] == best
        np.testing.assert_array_equal(g["h"], first[0])
        np.testing.assert_array_equal(g["nu"], first[1])


def test_global_layout_with_one_head_per_device_is_one_neuron_step():
    A = synth.make_affinity_matrix(8, 64, seed=9).numpy()
    g = oracle.global_layout(A, 8)
    assert g["parts"] == 1
    one = oracle.search_layout(A, 8, 1)
    assert g["score_q"] == one["score_q"]
