"""Planted mistakes: each copy of the oracle source with one plausible mistake (a sign, a derivative,
an operand, a tie-break, a stop rule, a scale, an order) must fail at least one pin, and the
unmodified source must pass them all.  The copies are compiled into a git-ignored folder.
"""
import itertools
import os
import subprocess

import numpy as np
import pytest

import oracle
from paper_2609_13846_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "dtp_oracle.c")
OUT = os.path.join(ROOT, "_build", "oracle_mutants")


def _silu(z):
    return z / (1.0 + np.exp(-z))


# ------------------------------------------------------------------ pin checks --

def check_first_order():
    """Central difference of removing eps * p_h matches Delta (Sec. 3)."""
    rng = np.random.default_rng(0)
    X, C = rng.standard_normal((24, 12)), rng.standard_normal((2, 24, 12)) * 0.5
    Wg, Wu = rng.standard_normal((5, 12)) * 0.3, rng.standard_normal((5, 12)) * 0.3
    A = oracle.affinity_fo(X, C, Wg, Wu)
    g, u, eps = X @ Wg.T, X @ Wu.T, 1e-4
    for h in range(2):
        pg, pu = C[h] @ Wg.T, C[h] @ Wu.T
        d = (_silu(g + eps * pg) * (u + eps * pu) - _silu(g - eps * pg) * (u - eps * pu)) / (2 * eps)
        if not np.allclose(A[h], (d ** 2).sum(axis=0), rtol=1e-6):
            return False
    return True


def check_add():
    rng = np.random.default_rng(1)
    C = rng.standard_normal((2, 16, 8))
    Wg, Wu = rng.standard_normal((4, 8)), rng.standard_normal((4, 8))
    ref = np.stack([((C[h] @ Wg.T) ** 2 + (C[h] @ Wu.T) ** 2).sum(axis=0) for h in range(2)])
    return np.allclose(oracle.affinity_add(C, Wg, Wu), ref, rtol=1e-12)


def check_quantize():
    A = synth.make_affinity_matrix(4, 32, seed=2).numpy()
    q, e = oracle.quantize(A)
    return int(q.max()) >= 2 ** 39 and int(q.max()) < 2 ** 40


def _balanced(n, D):
    for a in itertools.product(range(D), repeat=n):
        if all(a.count(l) == n // D for l in range(D)):
            yield np.array(a, np.int32)


def check_neuron_ties():
    """D = 2 on tie-heavy integer scores: the lexicographically smallest optimal assignment."""
    for seed in range(4):
        A = synth.make_affinity_matrix(2, 8, seed=10 + seed, kind="integer").numpy()
        q, _ = oracle.quantize(A)
        h = np.array([0, 1], np.int32)
        best, first = -1, None
        for nu in sorted(_balanced(8, 2), key=tuple):
            v = oracle.layout_score(q, h, nu)
            if v > best:
                best, first = v, nu
        nu, _ = oracle.neuron_step(q, h, 2)
        if not np.array_equal(nu, first):
            return False
    return True


def check_head_ties():
    """Head step on tie-heavy scores: the lexicographically smallest best labelled partition."""
    mats = [synth.make_affinity_matrix(4, 8, seed=20 + seed, kind="integer").numpy() for seed in range(4)]
    mats.append(np.ones((4, 8), np.float32))             # every partition ties
    for A in mats:
        q, _ = oracle.quantize(A)
        nu = np.array([0, 1] * 4, np.int32)
        best, first = -1, None
        for h in sorted(_balanced(4, 2), key=tuple):
            v = oracle.layout_score(q, h, nu)
            if v > best:
                best, first = v, h
        h, _ = oracle.head_step(q, nu, 2)
        if not np.array_equal(h, first):
            return False
    return True


def check_layer_stop():
    """The ascent stops after the first iteration without a strict increase."""
    for seed in range(3):
        A = synth.make_affinity_matrix(8, 48, seed=30 + seed).numpy()
        q, _ = oracle.quantize(A)
        h, prev, done = np.array([(g * 4) // 8 for g in range(8)], np.int32), -1, 0
        for it in range(10):
            nu, _ = oracle.neuron_step(q, h, 4)
            h, J = oracle.head_step(q, nu, 4)
            done = it + 1
            if J <= prev:
                break
            prev = J
        if oracle.search_layout(A, 4, 10)["iters_done"] != done:
            return False
    return True


def check_chain_stop():
    Su = np.stack([synth.make_affinity_matrix(8, 32, seed=40 + i).numpy() for i in range(4)])
    Sd = np.stack([synth.make_affinity_matrix(8, 32, seed=50 + i).numpy() for i in range(3)])
    Js = [oracle.chain_search(Su, Sd, 4, i)["J_q"] for i in range(1, 11)]
    expect = next((i + 1 for i in range(1, 10) if Js[i] <= Js[i - 1]), 10)
    return oracle.chain_search(Su, Sd, 4, 10)["iters_done"] == expect


def check_unit_mass():
    S = synth.make_affinity_matrix(4, 50, seed=3).numpy()
    n = oracle.normalize_unit_mass(S)
    return 2 ** 43 - 2 * S.size <= int(n.sum()) <= 2 ** 43


def check_head_writes():
    rng = np.random.default_rng(4)
    attn, Wo = rng.standard_normal((10, 12)), rng.standard_normal((8, 12)) * 0.3
    gamma, rms = 1 + 0.2 * rng.standard_normal(8), 0.5 + rng.random(10)
    C = oracle.head_writes(attn, Wo, gamma, rms, 4)
    ref = np.stack([gamma * (attn[:, 4 * h:4 * h + 4] @ Wo[:, 4 * h:4 * h + 4].T) / rms[:, None] for h in range(3)])
    return np.allclose(C, ref, rtol=1e-12, atol=1e-14)


def check_layout_order():
    lab = np.array([1, 0, 2, 1, 0, 2], np.int32)
    return oracle.layout_order(lab, 3).tolist() == [1, 4, 0, 3, 2, 5]


def check_minimise():
    """Minimising J (Table 4's anti-optimised layout) reaches the exact minimum over neurons when heads
    are frozen (brute force over every nu)."""
    Su = np.stack([synth.make_affinity_matrix(2, 4, seed=60 + i).numpy() for i in range(2)])
    Sd = np.stack([synth.make_affinity_matrix(2, 4, seed=70).numpy()])
    h0 = np.array([[0, 1], [0, 1]], np.int32)
    worst = min(oracle.chain_score(Su, Sd, h0, np.stack(nu)) for nu in itertools.product(list(_balanced(4, 2)), repeat=2))
    return oracle.chain_search(Su, Sd, 2, 10, move_heads=np.zeros(2), minimize=True)["J_q"] == worst


def check_global_optimum():
    """Best exact neuron step over the 35 unlabelled partitions equals brute force over all layouts."""
    A = synth.make_affinity_matrix(4, 8, seed=80).numpy()
    q, _ = oracle.quantize(A)
    best = max(oracle.layout_score(q, h, nu) for h in _balanced(4, 2) for nu in _balanced(8, 2))
    g = oracle.global_layout(A, 2)
    g8 = oracle.global_layout(synth.make_affinity_matrix(8, 16, seed=81).numpy(), 2)
    return g["score_q"] == best and g["parts"] == 3 and g8["parts"] == 35


CHECKS = [check_first_order, check_add, check_quantize, check_neuron_ties, check_head_ties, check_layer_stop,
          check_chain_stop, check_unit_mass, check_head_writes, check_layout_order, check_minimise,
          check_global_optimum]

# (name, text in dtp_oracle.c, replacement, occurrence to replace: 1 = first)
MUTANTS = [
    ("sign_of_beta_term", "double delta = dsilu * u * pg + silu * pu;", "double delta = dsilu * u * pg - silu * pu;", 1),
    ("silu_derivative", "double dsilu = sigma * (1.0 + g * (1.0 - sigma));", "double dsilu = sigma * (1.0 + g * sigma);", 1),
    ("gate_for_up_in_first_order", "double pu = dot(p, wu, d);", "double pu = dot(p, wg, d);", 1),
    ("gate_for_up_in_add", "double pu = dot(p, wu, d);", "double pu = dot(p, wg, d);", 2),
    ("fixed_point_exponent", "OR_FIXED_POINT_BITS - e));", "OR_FIXED_POINT_BITS - e + 1));", 1),
    ("neuron_tie_break", "return a->k < b->k ? -1 : (a->k > b->k ? 1 : 0);",
     "return a->k > b->k ? -1 : (a->k < b->k ? 1 : 0);", 1),
    ("head_strict_ties", "partial > s->best_score", "partial >= s->best_score", 1),
    ("layer_stop_rule", "if (J <= prev) break;", "if (J < prev) break;", 1),
    ("chain_stop_rule", "if (it > 0 && total <= prev) break;", "if (it > 0 && total < prev) break;", 1),
    ("unit_mass_scale", "<< OR_NORM_BITS) / total);", "<< (OR_NORM_BITS - 1)) / total);", 1),
    ("rms_multiplied", "gamma[i] * s / rms[t];", "gamma[i] * s * rms[t];", 1),
    ("device_order", "if (labels[k] == l) order[pos++] = k;", "if (labels[k] == D - 1 - l) order[pos++] = k;", 1),
    ("minimise_sign", "const int64_t sign = minimize ? -1 : 1;", "const int64_t sign = minimize ? 1 : 1;", 1),
    ("labelled_partitions_in_global", "for (int l = 0; l <= used && l < c->D; ++l)", "for (int l = 0; l < c->D; ++l)",
     1),
]


def _build(name, text):
    os.makedirs(OUT, exist_ok=True)
    src = os.path.join(OUT, f"{name}.c")
    lib = os.path.join(OUT, f"{name}.so")
    with open(src, "w") as f:
        f.write(text)
    subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", lib, src, "-lm"], check=True)
    return lib


def _replace_nth(text, old, new, n):
    at = -1
    for _ in range(n):
        at = text.index(old, at + 1)
    return text[:at] + new + text[at + len(old):]


def test_unmodified_oracle_passes_every_check():
    for check in CHECKS:
        assert check(), check.__name__


@pytest.mark.parametrize("name,old,new,n", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(name, old, new, n):
    text = open(SRC).read()
    assert text.count(old) >= n, f"mutation site of {name} not found"
    lib = _build(name, _replace_nth(text, old, new, n))
    with oracle.use_library(lib):
        failed = []
        for check in CHECKS:
            try:
                ok = check()
            except Exception:
                ok = False
            if not ok:
                failed.append(check.__name__)
    assert failed, f"no pin catches the planted mistake {name}"
