"""Pins of the affinity oracle against facts fixed by the paper and by mathematics.

Sec. 3 "Affinity scores" defines Delta_hk as the first-order change of neuron
k's output silu(g_k) u_k when head h's piece p_h of the normalised FFN input
is removed, and S^{up,fo} as E_t[Delta^2] ||w^d_k||^2.  Each test below checks
the oracle against something other than its own formula: a finite difference
of the removal, a symbolic derivative, invariances and equivariances, closed
special cases.
"""
import math

import numpy as np
import pytest
import sympy as sp
import torch

import oracle
from paper_2609_13846_gb300 import synth


def _tiny(seed=0, T=64, d=16, G=3, N=10, scale=1.0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((T, d)) * scale
    C = rng.standard_normal((G, T, d)) * 0.5 * scale
    Wg = rng.standard_normal((N, d)) * 0.3
    Wu = rng.standard_normal((N, d)) * 0.3
    return X, C, Wg, Wu


def _silu(z):
    return z / (1.0 + np.exp(-z))


def test_finite_difference_of_head_removal():
    """Central difference of removing eps * p_h from the operating point matches Delta.

    f(eps) = silu(g - eps*pg) * (u - eps*pu); (f(-eps) - f(eps)) / (2 eps) = Delta + O(eps^2).
    """
    X, C, Wg, Wu = _tiny()
    A = oracle.affinity_fo(X, C, Wg, Wu)
    g = X @ Wg.T
    u = X @ Wu.T
    eps = 1e-4
    for h in range(C.shape[0]):
        pg = C[h] @ Wg.T
        pu = C[h] @ Wu.T
        f_minus = _silu(g + eps * pg) * (u + eps * pu)
        f_plus = _silu(g - eps * pg) * (u - eps * pu)
        delta_fd = (f_minus - f_plus) / (2 * eps)
        A_fd = (delta_fd ** 2).sum(axis=0)
        np.testing.assert_allclose(A[h], A_fd, rtol=1e-6)


def test_finite_difference_on_tiny_workload():
    """Same pin on the tiny calibration workload (d=64, G=2, N=128, T=256, fp32 inputs)."""
    w = synth.WORKLOADS["tiny"]
    L = synth.make_workload_layer(w)
    X, C, Wg, Wu = (L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up"))
    A = oracle.affinity_fo(X, C, Wg, Wu)
    g, u = X @ Wg.T, X @ Wu.T
    eps = 1e-4
    for h in range(w.G):
        pg, pu = C[h] @ Wg.T, C[h] @ Wu.T
        d_fd = (_silu(g + eps * pg) * (u + eps * pu) - _silu(g - eps * pg) * (u - eps * pu)) / (2 * eps)
        np.testing.assert_allclose(A[h], (d_fd ** 2).sum(0), rtol=1e-6)


def test_single_token_symbolic_derivative():
    """T=1, d=1, N=1: A equals the square of a derivative that sympy takes symbolically."""
    x, wg, wu, c = 0.5, 2.0, -1.5, 0.3
    eps = sp.Symbol("eps")
    xs, cs, wgs, wus = sp.Rational(1, 2), sp.Rational(3, 10), sp.Integer(2), sp.Rational(-3, 2)
    gs = (xs - eps * cs) * wgs   # gate pre-activation with eps * p_h removed
    us = (xs - eps * cs) * wus   # up pre-activation with eps * p_h removed
    f = gs / (1 + sp.exp(-gs)) * us
    delta = -sp.diff(f, eps).subs(eps, 0)
    expected = float(sp.N(delta ** 2, 30))
    A = oracle.affinity_fo(np.array([[x]]), np.array([[[c]]]), np.array([[wg]]), np.array([[wu]]))
    assert A.shape == (1, 1)
    assert math.isclose(A[0, 0], expected, rel_tol=1e-13)


def test_head_equal_to_input_is_directional_derivative():
    """C_h = X: removing the whole input along the ray s -> s*x gives
    Delta = d/ds [silu(s g) s u] at s = 1, taken by sympy."""
    X, _, Wg, Wu = _tiny(seed=3, G=1)
    A = oracle.affinity_fo(X, X[None], Wg, Wu)
    s, gg, uu = sp.symbols("s g u")
    dfun = sp.lambdify((gg, uu), sp.diff(s * gg / (1 + sp.exp(-s * gg)) * s * uu, s).subs(s, 1), "numpy")
    g, u = X @ Wg.T, X @ Wu.T
    np.testing.assert_allclose(A[0], (dfun(g, u) ** 2).sum(0), rtol=1e-12)


def test_zero_up_projection_gives_zero():
    X, C, Wg, Wu = _tiny(seed=4)
    A = oracle.affinity_fo(X, C, Wg, np.zeros_like(Wu))
    assert np.all(A == 0.0)


def test_zero_head_gives_zero_row():
    X, C, Wg, Wu = _tiny(seed=5)
    C[1] = 0.0
    A = oracle.affinity_fo(X, C, Wg, Wu)
    assert np.all(A[1] == 0.0) and np.all(A[0] > 0)


def test_neuron_permutation_equivariance():
    """Permuting the gate/up rows jointly permutes the columns of A (Sec. 3 'The layout as a free variable')."""
    X, C, Wg, Wu = _tiny(seed=6)
    perm = np.random.default_rng(0).permutation(Wg.shape[0])
    A = oracle.affinity_fo(X, C, Wg, Wu)
    Ap = oracle.affinity_fo(X, C, Wg[perm], Wu[perm])
    np.testing.assert_array_equal(Ap, A[:, perm])


def test_head_permutation_equivariance():
    X, C, Wg, Wu = _tiny(seed=7)
    perm = np.array([2, 0, 1])
    A = oracle.affinity_fo(X, C, Wg, Wu)
    Ap = oracle.affinity_fo(X, C[perm], Wg, Wu)
    np.testing.assert_array_equal(Ap, A[perm])


def test_gate_up_swap_is_not_symmetric():
    """Swapping the roles of W_gate and W_up changes A (catches a transposed operand)."""
    X, C, Wg, Wu = _tiny(seed=8)
    A = oracle.affinity_fo(X, C, Wg, Wu)
    B = oracle.affinity_fo(X, C, Wu, Wg)
    assert np.max(np.abs(A - B)) > 1e-3 * np.max(A)


def test_orthogonal_rotation_invariance():
    """Rotating the d channels of X, C and both weight matrices leaves every dot product, hence A, unchanged."""
    X, C, Wg, Wu = _tiny(seed=9)
    Q, _ = np.linalg.qr(np.random.default_rng(1).standard_normal((X.shape[1], X.shape[1])))
    A = oracle.affinity_fo(X, C, Wg, Wu)
    Ar = oracle.affinity_fo(X @ Q, C @ Q, Wg @ Q, Wu @ Q)
    np.testing.assert_allclose(Ar, A, rtol=1e-10)


def test_token_additivity():
    X, C, Wg, Wu = _tiny(seed=10, T=50)
    A = oracle.affinity_fo(X, C, Wg, Wu)
    A1 = oracle.affinity_fo(X[:17], C[:, :17], Wg, Wu)
    A2 = oracle.affinity_fo(X[17:], C[:, 17:], Wg, Wu)
    np.testing.assert_allclose(A1 + A2, A, rtol=1e-12)


def test_head_scaling_is_quadratic():
    X, C, Wg, Wu = _tiny(seed=11)
    A = oracle.affinity_fo(X, C, Wg, Wu)
    C2 = C.copy()
    C2[0] *= 3.0
    A2 = oracle.affinity_fo(X, C2, Wg, Wu)
    np.testing.assert_allclose(A2[0], 9.0 * A[0], rtol=1e-12)
    np.testing.assert_array_equal(A2[1:], A[1:])


def test_linear_in_head_piece_before_squaring():
    """Delta is linear in p_h: A(C_a + C_b) + A(C_a - C_b) = 2 A(C_a) + 2 A(C_b) (parallelogram law)."""
    X, C, Wg, Wu = _tiny(seed=12, G=2)
    Ca, Cb = C[0:1], C[1:2]
    lhs = oracle.affinity_fo(X, Ca + Cb, Wg, Wu) + oracle.affinity_fo(X, Ca - Cb, Wg, Wu)
    rhs = 2 * oracle.affinity_fo(X, Ca, Wg, Wu) + 2 * oracle.affinity_fo(X, Cb, Wg, Wu)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-10)


def test_repeat_is_bitwise_identical():
    """Each entry is summed in token order by one thread: bitwise identical across runs."""
    X, C, Wg, Wu = _tiny(seed=13, N=37)
    A1 = oracle.affinity_fo(X, C, Wg, Wu)
    A2 = oracle.affinity_fo(X, C, Wg, Wu)
    np.testing.assert_array_equal(A1, A2)


def test_bf16_inputs_are_upcast_exactly():
    L = synth.make_layer(32, 2, 16, 8, seed=5, dtype="bf16", outliers=True)
    A1 = oracle.affinity_fo(*(L[k].float().numpy() for k in ("X", "C", "W_gate", "W_up")))
    A2 = oracle.affinity_fo(*(L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up")))
    np.testing.assert_array_equal(A1, A2)


def test_finalize_mean_and_down_norm():
    """finalize multiplies by ||w^d_k||^2 / T_total (Sec. 3 S^{up,fo} = E_t[Delta^2] ||w^d_k||^2)."""
    rng = np.random.default_rng(3)
    A = rng.random((3, 5))
    Wd = rng.standard_normal((7, 5))
    wd = (Wd ** 2).sum(0)
    out = oracle.finalize(A, 40, wd)
    for h in range(3):
        for k in range(5):
            assert math.isclose(out[h, k], A[h, k] / 40 * float(np.dot(Wd[:, k], Wd[:, k])), rel_tol=1e-14)
    np.testing.assert_allclose(oracle.finalize(A, 4, None), A / 4, rtol=1e-15)


def test_synthetic_recipe_shapes_and_scales():
    """The model-shaped recipe: 4 outlier channels at 20x and per-head norms in [0.1, 1] x ||X||."""
    L = synth.make_layer(256, 4, 32, 512, seed=1, dtype="f32", outliers=True)
    X, C = L["X"], L["C"]
    col = X.pow(2).mean(0).sqrt()
    assert int((col > 10).sum()) == 4
    ratio = torch.linalg.vector_norm(C.reshape(4, -1), dim=1) / torch.linalg.vector_norm(X)
    assert torch.all(ratio >= 0.1 - 1e-5) and torch.all(ratio <= 1.0 + 1e-5)
    assert abs(float(L["W_gate"].std()) - 0.02) < 2e-3


def test_add_score_is_the_removed_pre_activation_change():
    """ADD (Sec. 3): removing head h's piece changes neuron k's gate and up pre-activations by
    exactly p_h . w (they are linear); the score is the summed square of both changes."""
    X, C, Wg, Wu = _tiny(seed=14)
    A = oracle.affinity_add(C, Wg, Wu)
    for h in range(C.shape[0]):
        dg = X @ Wg.T - (X - C[h]) @ Wg.T
        du = X @ Wu.T - (X - C[h]) @ Wu.T
        np.testing.assert_allclose(A[h], (dg ** 2 + du ** 2).sum(0), rtol=1e-10)


def test_add_score_ignores_the_operating_point_and_fo_does_not():
    """ADD does not depend on X; FO does (Sec. 3: ADD ignores the operating point of the nonlinearity)."""
    X, C, Wg, Wu = _tiny(seed=15)
    A1 = oracle.affinity_add(C, Wg, Wu)
    assert np.array_equal(A1, oracle.affinity_add(C, Wg, Wu))
    F1 = oracle.affinity_fo(X, C, Wg, Wu)
    F2 = oracle.affinity_fo(2.0 * X, C, Wg, Wu)
    assert np.max(np.abs(F1 - F2)) > 1e-3 * np.max(F1)


# ------------------------------------------------ per-query-head scores ----
# Sec. 3: the damage is taken per query head from that head's own write, and a
# KV group's score is the sum over its query heads of E[Delta^2].

def test_query_head_sum_with_one_head_per_group_is_plain_fo():
    X, C, Wg, Wu = _tiny(seed=40, G=4)
    np.testing.assert_array_equal(oracle.affinity_fo_qheads(X, C, Wg, Wu, 1), oracle.affinity_fo(X, C, Wg, Wu))
    np.testing.assert_array_equal(oracle.affinity_add_qheads(C, Wg, Wu, 1), oracle.affinity_add(C, Wg, Wu))


def test_query_head_sum_is_a_sum_of_squares_not_the_square_of_the_sum():
    """Duplicated query heads (each group's heads all equal to c): Delta is linear in the write,
    so the group's combined write q*c scores q^2 E[Delta_c^2] while the per-query-head sum is
    q E[Delta_c^2]; the groups are consecutive heads."""
    X, c, Wg, Wu = _tiny(seed=41, G=3)
    for q in (2, 4):
        Cq = np.repeat(c, q, axis=0)                      # heads g*q .. g*q+q-1 all equal c[g]
        per_q = oracle.affinity_fo_qheads(X, Cq, Wg, Wu, q)
        combined = oracle.affinity_fo(X, q * c, Wg, Wu)
        np.testing.assert_allclose(per_q, combined / q, rtol=1e-12)
        np.testing.assert_allclose(per_q, q * oracle.affinity_fo(X, c, Wg, Wu), rtol=1e-12)
        np.testing.assert_allclose(oracle.affinity_add_qheads(Cq, Wg, Wu, q),
                                   oracle.affinity_add(q * c, Wg, Wu) / q, rtol=1e-12)


def test_query_head_sum_with_silent_heads_equals_group_write():
    """A group whose other query heads write nothing: both readings agree."""
    X, c, Wg, Wu = _tiny(seed=42, G=2)
    Cq = np.zeros((6, *c.shape[1:]))
    Cq[0], Cq[3] = c[0], c[1]                              # q = 3: one live head per group
    np.testing.assert_allclose(oracle.affinity_fo_qheads(X, Cq, Wg, Wu, 3), oracle.affinity_fo(X, c, Wg, Wu),
                               rtol=1e-13)


def test_query_head_sum_against_finite_differences():
    X, C, Wg, Wu = _tiny(seed=43, G=4, T=48)
    g, u = X @ Wg.T, X @ Wu.T
    eps = 1e-4
    expect = np.zeros((2, Wg.shape[0]))
    for h in range(4):
        pg, pu = C[h] @ Wg.T, C[h] @ Wu.T
        d = (_silu(g + eps * pg) * (u + eps * pu) - _silu(g - eps * pg) * (u - eps * pu)) / (2 * eps)
        expect[h // 2] += (d ** 2).sum(axis=0)
    np.testing.assert_allclose(oracle.affinity_fo_qheads(X, C, Wg, Wu, 2), expect, rtol=1e-6)
    with pytest.raises(ValueError):
        oracle.affinity_fo_qheads(X, C, Wg, Wu, 3)


def test_more_than_sixteen_heads_equal_split_calls():
    """32 query heads (Llama-3.1-8B: 4 per KV group) in one call equal two 16-head calls."""
    X, C, Wg, Wu = _tiny(seed=44, G=32, T=24)
    A = oracle.affinity_fo(X, C, Wg, Wu)
    np.testing.assert_array_equal(A, np.concatenate([oracle.affinity_fo(X, C[:16], Wg, Wu),
                                                     oracle.affinity_fo(X, C[16:], Wg, Wu)]))
    assert oracle.affinity_fo_qheads(X, C, Wg, Wu, 4).shape == (8, Wg.shape[0])


def test_top_group_share_pins():
    """Sec. 5: the largest KV group's share of a neuron's affinity, averaged over neurons."""
    G, N = 8, 40
    assert oracle.top_group_share(np.ones((G, N), np.float32)) == pytest.approx(1 / G, rel=1e-12)
    one_hot = np.zeros((G, N), np.float32)
    one_hot[np.arange(N) % G, np.arange(N)] = 3.0
    assert oracle.top_group_share(one_hot) == pytest.approx(1.0, rel=1e-12)
    A = np.zeros((2, 3), np.float32)
    A[:, 0] = [1.0, 3.0]                        # 3/4
    A[:, 2] = [2.0, 2.0]                        # 1/2; column 1 is empty and skipped
    assert oracle.top_group_share(A) == pytest.approx((0.75 + 0.5) / 2, rel=1e-12)
    assert oracle.top_group_share(np.zeros((2, 3), np.float32)) == 0.0
    B = synth.make_affinity_matrix(G, N, seed=4).numpy()
    assert oracle.top_group_share(B * np.float32(8.0)) == pytest.approx(oracle.top_group_share(B), rel=1e-12)
    assert oracle.top_group_share(B[::-1].copy()) == pytest.approx(oracle.top_group_share(B), rel=1e-12)
