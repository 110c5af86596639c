"""Reference oracle for the affinity-aware sharding hot path -- TEST INFRASTRUCTURE.

A plain fp64 / exact-integer CPU statement of what the path computes, written
from "Affinity-Aware Sharding for Delayed Tensor Parallelism" (arXiv
2609.13846), Sec. 3 ("Affinity scores", "Objective", "Optimiser").  The C
source is ``dtp_oracle.c``; this module compiles it with gcc and wraps it with
ctypes and numpy.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this package.  It shares no code with the CUDA library and
imports nothing from it.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(finite differences, closed forms, invariances, brute force, the Hungarian
method, and the counts the paper prints).  Values the paper prints for its own
models (the J values of Table 4) need the paper's weights and data and are
unpinned.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dtp_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None

_i64p = ctypes.POINTER(ctypes.c_int64)
_i32p = ctypes.POINTER(ctypes.c_int)
_f64p = ctypes.POINTER(ctypes.c_double)
_f32p = ctypes.POINTER(ctypes.c_float)


def build(force: bool = False) -> str:
    """Compile ``dtp_oracle.c`` into ``liboracle.so`` (plain gcc, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", _LIB, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
    return _LIB


def _load():
    global _lib
    if _lib is not None:
        return _lib
    _lib = _declare(ctypes.CDLL(build()))
    return _lib


class use_library:
    """Context manager: route every oracle call through another build of ``dtp_oracle.c`` (the
    tests that plant a mistake in a copy of the source and check that a pin catches it)."""

    def __init__(self, path: str):
        self.path = path
        self.saved = None

    def __enter__(self):
        global _lib
        self.saved = _load()
        _lib = _declare(ctypes.CDLL(self.path))
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self.saved


def _declare(lib):
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_affinity_fo.argtypes = [_f64p, _f64p, _f64p, _f64p, ctypes.c_int64, ctypes.c_int,
                                       ctypes.c_int, ctypes.c_int, _f64p]
    lib.oracle_affinity_fo.restype = None
    lib.oracle_finalize.argtypes = [_f64p, ctypes.c_int, ctypes.c_int, ctypes.c_int64, _f64p]
    lib.oracle_finalize.restype = None
    lib.oracle_quantize.argtypes = [_f32p, ctypes.c_int, ctypes.c_int, _i64p, _i32p]
    lib.oracle_quantize.restype = ctypes.c_int
    lib.oracle_layout_score.argtypes = [_i64p, ctypes.c_int, ctypes.c_int, _i32p, _i32p]
    lib.oracle_layout_score.restype = ctypes.c_int64
    lib.oracle_neuron_step_ex.argtypes = [_i64p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p,
                                          _i32p, _i32p, ctypes.c_int]
    lib.oracle_neuron_step_ex.restype = ctypes.c_int
    lib.oracle_assignment_gain.argtypes = [_i64p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p, _i32p]
    lib.oracle_assignment_gain.restype = ctypes.c_int64
    lib.oracle_count_partitions.argtypes = [ctypes.c_int, ctypes.c_int]
    lib.oracle_count_partitions.restype = ctypes.c_int64
    lib.oracle_head_step.argtypes = [_i64p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p, _i32p, _i64p]
    lib.oracle_head_step.restype = ctypes.c_int
    lib.oracle_search_layout.argtypes = [_f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                         _i32p, _i32p, _i64p, _f64p, _i32p, _i32p]
    lib.oracle_search_layout.restype = ctypes.c_int
    lib.oracle_global_layout.argtypes = [_f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p, _i32p, _i64p,
                                         _f64p, _i32p]
    lib.oracle_global_layout.restype = ctypes.c_int
    lib.oracle_top_group_share.argtypes = [_f32p, ctypes.c_int, ctypes.c_int]
    lib.oracle_top_group_share.restype = ctypes.c_double
    lib.oracle_head_writes.argtypes = [_f64p, _f64p, _f64p, _f64p, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                                       ctypes.c_int, ctypes.c_int, _f64p]
    lib.oracle_head_writes.restype = None
    lib.oracle_layout_order.argtypes = [_i32p, ctypes.c_int, ctypes.c_int, _i32p]
    lib.oracle_layout_order.restype = ctypes.c_int
    lib.oracle_hungarian_max.argtypes = [_i64p, ctypes.c_int, _i32p]
    lib.oracle_hungarian_max.restype = ctypes.c_int64
    lib.oracle_affinity_add.argtypes = [_f64p, _f64p, _f64p, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, _f64p]
    lib.oracle_affinity_add.restype = None
    lib.oracle_down_activation.argtypes = [_f64p, _f64p, _f64p, _f64p, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
                                           _f64p]
    lib.oracle_down_activation.restype = None
    lib.oracle_down_weight_sqnorm.argtypes = [_f64p, _f64p, _f64p, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                              ctypes.c_int, _f64p]
    lib.oracle_down_weight_sqnorm.restype = None
    lib.oracle_down_score.argtypes = [_f64p, _f64p, ctypes.c_int, ctypes.c_int, ctypes.c_int64, _f64p]
    lib.oracle_down_score.restype = None
    lib.oracle_normalize_unit_mass.argtypes = [_f32p, ctypes.c_int64, _i64p]
    lib.oracle_normalize_unit_mass.restype = ctypes.c_int
    lib.oracle_chain_search.argtypes = [_f32p, _f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, _i32p, _i32p, _i64p, _f64p, _i32p, _i32p]
    lib.oracle_chain_search.restype = ctypes.c_int
    lib.oracle_chain_search_ex.argtypes = [_f32p, _f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, ctypes.c_char_p, ctypes.c_char_p, ctypes.c_int, _i32p, _i32p,
                                           _i64p, _f64p, _i32p, _i32p]
    lib.oracle_chain_search_ex.restype = ctypes.c_int
    lib.oracle_chain_score.argtypes = [_f32p, _f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p, _i32p]
    lib.oracle_chain_score.restype = ctypes.c_int64
    lib.oracle_chain_edge_scores.argtypes = [_f32p, _f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _i32p, _i32p,
                                             _i64p]
    lib.oracle_chain_edge_scores.restype = ctypes.c_int
    return lib


def _p(a: np.ndarray, ptype):
    return a.ctypes.data_as(ptype)


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def num_threads() -> int:
    """OpenMP threads the affinity oracle uses."""
    return int(_load().oracle_num_threads())


def affinity_fo(X, C, W_gate, W_up) -> np.ndarray:
    """A[h,k] = sum_t Delta_{t,h,k}^2 in fp64 (Sec. 3, equation for Delta).

    X [T,d], C [G,T,d], W_gate/W_up [N,d]; any real dtype, upcast exactly to fp64.
    """
    X = _c(X, np.float64)
    C = _c(C, np.float64)
    Wg = _c(W_gate, np.float64)
    Wu = _c(W_up, np.float64)
    T, d = X.shape
    G = C.shape[0]
    N = Wg.shape[0]
    assert C.shape == (G, T, d) and Wg.shape == (N, d) and Wu.shape == (N, d)
    A = np.zeros((G, N), dtype=np.float64)
    _load().oracle_affinity_fo(_p(X, _f64p), _p(C, _f64p), _p(Wg, _f64p), _p(Wu, _f64p),
                               T, d, G, N, _p(A, _f64p))
    return A


def affinity_fo_qheads(X, C_q, W_gate, W_up, q_per_group: int) -> np.ndarray:
    """The first-order score per query head, summed over each KV group's query heads (Sec. 3).

    C_q [H_q, T, d] holds each query head's own write p_h; row g of the result
    is sum over h = g*q_per_group .. (g+1)*q_per_group - 1 of sum_t Delta_{t,h,k}^2
    (a sum of per-head squares).  [H_q / q_per_group, N] fp64.
    """
    A = affinity_fo(X, C_q, W_gate, W_up)
    H = A.shape[0]
    if q_per_group < 1 or H % q_per_group:
        raise ValueError("q_per_group must divide the number of query heads")
    return A.reshape(H // q_per_group, q_per_group, -1).sum(axis=1)


def affinity_add_qheads(C_q, W_gate, W_up, q_per_group: int) -> np.ndarray:
    """The ADD score per query head, summed over each KV group's query heads (Sec. 3)."""
    A = affinity_add(C_q, W_gate, W_up)
    H = A.shape[0]
    if q_per_group < 1 or H % q_per_group:
        raise ValueError("q_per_group must divide the number of query heads")
    return A.reshape(H // q_per_group, q_per_group, -1).sum(axis=1)


def affinity_add(C, W_gate, W_up) -> np.ndarray:
    """ADD score before the mean: sum_t (p_h . w^g_k)^2 + (p_h . w^u_k)^2 (Sec. 3), fp64."""
    C = _c(C, np.float64)
    Wg = _c(W_gate, np.float64)
    Wu = _c(W_up, np.float64)
    G, T, d = C.shape
    N = Wg.shape[0]
    A = np.zeros((G, N), dtype=np.float64)
    _load().oracle_affinity_add(_p(C, _f64p), _p(Wg, _f64p), _p(Wu, _f64p), T, d, G, N, _p(A, _f64p))
    return A


def finalize(A, T_total: int, wd_sqnorm=None) -> np.ndarray:
    """A * ||w^d_k||^2 / T_total (Sec. 3: the E_t mean and the down-projection factor)."""
    A = _c(A, np.float64).copy()
    G, N = A.shape
    wd = None if wd_sqnorm is None else _c(wd_sqnorm, np.float64)
    _load().oracle_finalize(_p(A, _f64p), G, N, T_total, None if wd is None else _p(wd, _f64p))
    return A


def quantize(A):
    """Exact fixed-point form of a layer's affinity: (q int64 [G,N], e)."""
    A = _c(A, np.float32)
    G, N = A.shape
    q = np.zeros((G, N), dtype=np.int64)
    e = ctypes.c_int(0)
    st = _load().oracle_quantize(_p(A, _f32p), G, N, _p(q, _i64p), ctypes.byref(e))
    if st != 0:
        raise ValueError(f"oracle_quantize: status {st}")
    return q, e.value


def layout_score(q, h, nu) -> int:
    """Integer up-edge co-located mass of a layout (Eq. objective, one layer)."""
    q = _c(q, np.int64)
    G, N = q.shape
    return int(_load().oracle_layout_score(_p(q, _i64p), G, N, _p(_c(h, np.int32), _i32p),
                                           _p(_c(nu, np.int32), _i32p)))


def neuron_step(q, h, D: int, general: bool = False):
    """Lexicographically smallest optimal balanced neuron assignment: (nu, unique)."""
    q = _c(q, np.int64)
    G, N = q.shape
    nu = np.zeros(N, dtype=np.int32)
    uniq = ctypes.c_int(0)
    st = _load().oracle_neuron_step_ex(_p(q, _i64p), G, N, D, _p(_c(h, np.int32), _i32p),
                                       _p(nu, _i32p), ctypes.byref(uniq), int(general))
    if st != 0:
        raise ValueError(f"oracle_neuron_step: status {st}")
    return nu, bool(uniq.value)


def assignment_gain(q, h, nu, D: int) -> int:
    q = _c(q, np.int64)
    G, N = q.shape
    return int(_load().oracle_assignment_gain(_p(q, _i64p), G, N, D, _p(_c(h, np.int32), _i32p),
                                              _p(_c(nu, np.int32), _i32p)))


def count_partitions(G: int, D: int) -> int:
    return int(_load().oracle_count_partitions(G, D))


def head_step(q, nu, D: int):
    """Best labelled balanced head partition given nu: (h, score)."""
    q = _c(q, np.int64)
    G, N = q.shape
    h = np.zeros(G, dtype=np.int32)
    s = ctypes.c_int64(0)
    st = _load().oracle_head_step(_p(q, _i64p), G, N, D, _p(_c(nu, np.int32), _i32p), _p(h, _i32p),
                                  ctypes.byref(s))
    if st != 0:
        raise ValueError(f"oracle_head_step: status {st}")
    return h, int(s.value)


def search_layout(A, D: int, iters: int):
    """Coordinate ascent on one layer: dict(h, nu, score_q, score, iters_done, unique)."""
    A = _c(A, np.float32)
    G, N = A.shape
    h = np.zeros(G, dtype=np.int32)
    nu = np.zeros(N, dtype=np.int32)
    sq = ctypes.c_int64(0)
    sc = ctypes.c_double(0.0)
    it = ctypes.c_int(0)
    uq = ctypes.c_int(0)
    st = _load().oracle_search_layout(_p(A, _f32p), G, N, D, iters, _p(h, _i32p), _p(nu, _i32p),
                                      ctypes.byref(sq), ctypes.byref(sc), ctypes.byref(it),
                                      ctypes.byref(uq))
    if st != 0:
        raise ValueError(f"oracle_search_layout: status {st}")
    return dict(h=h, nu=nu, score_q=int(sq.value), score=float(sc.value), iters_done=int(it.value),
                unique=bool(uq.value))


def global_layout(A, D: int):
    """The exact maximum of one layer's up-edge J over every balanced layout (Sec. 3 'Objective'):
    the best exact neuron step over the unlabelled head partitions, each in its canonical labelling,
    the first (lexicographic) best one kept.  dict(h, nu, score_q, score, parts)."""
    A = _c(A, np.float32)
    G, N = A.shape
    h = np.zeros(G, dtype=np.int32)
    nu = np.zeros(N, dtype=np.int32)
    sq = ctypes.c_int64(0)
    sc = ctypes.c_double(0.0)
    npart = ctypes.c_int(0)
    st = _load().oracle_global_layout(_p(A, _f32p), G, N, D, _p(h, _i32p), _p(nu, _i32p), ctypes.byref(sq),
                                      ctypes.byref(sc), ctypes.byref(npart))
    if st != 0:
        raise ValueError(f"oracle_global_layout: status {st}")
    return dict(h=h, nu=nu, score_q=sq.value, score=sc.value, parts=npart.value)


def hungarian_max(W):
    """Textbook Hungarian method: (max total, row_to_col) of a square int64 matrix."""
    W = _c(W, np.int64)
    n = W.shape[0]
    r2c = np.zeros(n, dtype=np.int32)
    total = _load().oracle_hungarian_max(_p(W, _i64p), n, _p(r2c, _i32p))
    return int(total), r2c


# --------------------------------------------------------------- down edge ---

def down_activation(X, W_gate, W_up, rms_next):
    """act2[k] = sum_t (silu(g_k) u_k)^2 / r'_t^2 (Sec. 3, down edge), fp64."""
    X = _c(X, np.float64)
    Wg = _c(W_gate, np.float64)
    Wu = _c(W_up, np.float64)
    r = _c(rms_next, np.float64)
    T, d = X.shape
    N = Wg.shape[0]
    assert Wg.shape == (N, d) and Wu.shape == (N, d) and r.shape == (T,)
    out = np.zeros(N, dtype=np.float64)
    _load().oracle_down_activation(_p(X, _f64p), _p(Wg, _f64p), _p(Wu, _f64p), _p(r, _f64p), T, d, N,
                                   _p(out, _f64p))
    return out


def down_weight_sqnorm(Wqkv, gamma_next, W_down):
    """bn[g,k] = ||W^qkv_g (gamma' * w^d_k)||^2 for Wqkv [G,R,d], gamma' [d], W_down [d,N]."""
    Wq = _c(Wqkv, np.float64)
    gm = _c(gamma_next, np.float64)
    Wd = _c(W_down, np.float64)
    G, R, d = Wq.shape
    N = Wd.shape[1]
    assert gm.shape == (d,) and Wd.shape == (d, N)
    out = np.zeros((G, N), dtype=np.float64)
    _load().oracle_down_weight_sqnorm(_p(Wq, _f64p), _p(gm, _f64p), _p(Wd, _f64p), G, R, d, N, _p(out, _f64p))
    return out


def down_score(act2, bn, T_total: int):
    """S_down[g,k] = act2[k] / T_total * bn[g,k] ([G,N], transpose of the paper's I x G)."""
    a = _c(act2, np.float64)
    b = _c(bn, np.float64)
    G, N = b.shape
    out = np.zeros((G, N), dtype=np.float64)
    _load().oracle_down_score(_p(a, _f64p), _p(b, _f64p), G, N, T_total, _p(out, _f64p))
    return out


def normalize_unit_mass(S):
    """Exact integer unit-mass form of one affinity matrix (units of 2^-43)."""
    S = _c(S, np.float32)
    n = np.zeros(S.shape, dtype=np.int64)
    st = _load().oracle_normalize_unit_mass(_p(S, _f32p), S.size, _p(n, _i64p))
    if st != 0:
        raise ValueError(f"oracle_normalize_unit_mass: status {st}")
    return n


def chain_search(S_up, S_down, D: int, iters: int, move_heads=None, move_neurons=None, minimize=False):
    """Coordinate ascent on the whole-model objective (both edges): dict(h, nu, J_q, J, iters_done, unique).

    move_heads / move_neurons: per-layer 0/1 (None = every layer moves); minimize: the
    anti-optimised layout (Sec. 3 'Optimiser', Table 4 ablations).
    """
    Su = _c(S_up, np.float32)
    L, G, N = Su.shape
    Sd = _c(S_down if L > 1 else np.zeros((1, G, N)), np.float32)
    assert Sd.shape[1:] == (G, N) and (L == 1 or Sd.shape[0] == L - 1)
    h = np.zeros((L, G), dtype=np.int32)
    nu = np.zeros((L, N), dtype=np.int32)
    jq = ctypes.c_int64(0)
    j = ctypes.c_double(0.0)
    it = ctypes.c_int(0)
    uq = ctypes.c_int(0)
    mh = None if move_heads is None else bytes(np.asarray(move_heads, dtype=np.uint8).tolist())
    mn = None if move_neurons is None else bytes(np.asarray(move_neurons, dtype=np.uint8).tolist())
    st = _load().oracle_chain_search_ex(_p(Su, _f32p), _p(Sd, _f32p), L, G, N, D, iters, mh, mn, int(minimize),
                                        _p(h, _i32p), _p(nu, _i32p), ctypes.byref(jq), ctypes.byref(j),
                                        ctypes.byref(it), ctypes.byref(uq))
    if st != 0:
        raise ValueError(f"oracle_chain_search: status {st}")
    return dict(h=h, nu=nu, J_q=int(jq.value), J=float(j.value), iters_done=int(it.value), unique=bool(uq.value))


def chain_score(S_up, S_down, h, nu) -> int:
    """J of a layout over all layers (Eq. objective), in units of 2^-43."""
    Su = _c(S_up, np.float32)
    L, G, N = Su.shape
    Sd = _c(S_down if L > 1 else np.zeros((1, G, N)), np.float32)
    return int(_load().oracle_chain_score(_p(Su, _f32p), _p(Sd, _f32p), L, G, N, _p(_c(h, np.int32), _i32p),
                                          _p(_c(nu, np.int32), _i32p)))


def chain_edge_scores(S_up, S_down, h, nu) -> np.ndarray:
    """Co-located mass per edge [2L-1] (up_0, down_0, up_1, ..., up_{L-1}), units of 2^-43 of each edge."""
    Su = _c(S_up, np.float32)
    L, G, N = Su.shape
    Sd = _c(S_down if L > 1 else np.zeros((1, G, N)), np.float32)
    out = np.zeros(2 * L - 1, np.int64)
    bad = _load().oracle_chain_edge_scores(_p(Su, _f32p), _p(Sd, _f32p), L, G, N, _p(_c(h, np.int32), _i32p),
                                           _p(_c(nu, np.int32), _i32p), _p(out, _i64p))
    if bad:
        raise ValueError("negative or non-finite affinity entry")
    return out


def head_writes(attn, W_o, gamma, rms, head_dim: int, q_per_row: int = 1) -> np.ndarray:
    """p_h = gamma . (a_h W_o^(h)T) / r per head (Sec. 3), rows summed over q_per_row consecutive heads.

    attn [T, Hq*hd], W_o [d, Hq*hd], gamma [d], rms [T]; returns C [Hq/q_per_row, T, d] fp64.
    """
    A = _c(attn, np.float64)
    W = _c(W_o, np.float64)
    g = _c(gamma, np.float64)
    r = _c(rms, np.float64)
    T, K = A.shape
    d = W.shape[0]
    if K % head_dim or W.shape != (d, K) or g.shape != (d,) or r.shape != (T,):
        raise ValueError("shapes must be attn [T, Hq*hd], W_o [d, Hq*hd], gamma [d], rms [T]")
    Hq = K // head_dim
    if q_per_row < 1 or Hq % q_per_row:
        raise ValueError("q_per_row must divide the number of heads")
    C = np.zeros((Hq // q_per_row, T, d), np.float64)
    _load().oracle_head_writes(_p(A, _f64p), _p(W, _f64p), _p(g, _f64p), _p(r, _f64p), T, d, Hq, head_dim,
                               q_per_row, _p(C, _f64p))
    return C


def layout_order(labels, D: int) -> np.ndarray:
    """Items listed device by device (each device's in increasing index): the permutation that
    makes every device's items one contiguous shard."""
    lab = _c(labels, np.int32)
    out = np.zeros(lab.shape[0], np.int32)
    if _load().oracle_layout_order(_p(lab, _i32p), lab.shape[0], D, _p(out, _i32p)) != 0:
        raise ValueError("label outside [0, D)")
    return out


def top_group_share(A) -> float:
    """Mean over neurons of max_g A[g,k] / sum_g A[g,k] (Sec. 5; neurons with a zero column skipped)."""
    A = _c(A, np.float32)
    G, N = A.shape
    return float(_load().oracle_top_group_share(_p(A, _f32p), G, N))
