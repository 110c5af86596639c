"""Pins of the producer (head writes into the FFN input) and of the layout application (Sec. 3).

Head writes: p_h = gamma . (a_h W_o^(h)T) / r is head h's share of the FFN
input with the rms held fixed; the first test removes each head from a
simulated residual stream.  Layout application: permuting KV groups (with their
query heads) and neurons leaves a dense GQA Transformer block unchanged, and
the contiguous shards of the permuted block are exactly the devices of the
layout, their partial outputs summing to the dense output.
"""
import itertools

import numpy as np
import pytest

import oracle
from oracle import dense_block
from paper_2609_13846_gb300 import ablation


def _attn_setup(seed=0, T=20, d=24, Hq=6, hd=4):
    rng = np.random.default_rng(seed)
    return dict(attn=rng.standard_normal((T, Hq * hd)), Wo=rng.standard_normal((d, Hq * hd)) * 0.3,
                gamma=1 + 0.2 * rng.standard_normal(d), rms=0.5 + rng.random(T), base=rng.standard_normal((T, d)),
                hd=hd, Hq=Hq)


def test_head_write_is_the_removed_share_of_the_ffn_input():
    s = _attn_setup()
    T, hd, Hq = s["attn"].shape[0], s["hd"], s["Hq"]
    resid = s["base"] + s["attn"] @ s["Wo"].T
    ffn_in = lambda r: s["gamma"] * r / s["rms"][:, None]          # the FFN pre-norm, rms held fixed
    C = oracle.head_writes(s["attn"], s["Wo"], s["gamma"], s["rms"], hd)
    assert C.shape == (Hq, T, s["Wo"].shape[0])
    for h in range(Hq):
        cols = slice(h * hd, (h + 1) * hd)
        without = resid - s["attn"][:, cols] @ s["Wo"][:, cols].T
        np.testing.assert_allclose(C[h], ffn_in(resid) - ffn_in(without), rtol=1e-11, atol=1e-12)
    # all heads together: the whole attention write
    np.testing.assert_allclose(C.sum(axis=0), ffn_in(s["attn"] @ s["Wo"].T), rtol=1e-11, atol=1e-12)


def test_group_rows_sum_consecutive_query_heads():
    s = _attn_setup(seed=1, Hq=6)
    per_head = oracle.head_writes(s["attn"], s["Wo"], s["gamma"], s["rms"], s["hd"], 1)
    for q in (2, 3):
        grouped = oracle.head_writes(s["attn"], s["Wo"], s["gamma"], s["rms"], s["hd"], q)
        np.testing.assert_allclose(grouped, per_head.reshape(6 // q, q, *per_head.shape[1:]).sum(axis=1),
                                   rtol=1e-12, atol=1e-13)
    z = dict(s)
    z["attn"] = s["attn"].copy()
    z["attn"][:, 2 * s["hd"]:3 * s["hd"]] = 0.0                       # head 2 silent
    assert not oracle.head_writes(z["attn"], s["Wo"], s["gamma"], s["rms"], s["hd"])[2].any()
    with pytest.raises(ValueError):
        oracle.head_writes(s["attn"], s["Wo"], s["gamma"], s["rms"], s["hd"], 4)


def test_layout_order_groups_devices_contiguously():
    for n, D in ((8, 2), (12, 4), (9, 3)):
        for labels in itertools.islice(itertools.permutations(np.repeat(np.arange(D), n // D)), 0, 200, 7):
            labels = np.array(labels, np.int32)
            o = oracle.layout_order(labels, D)
            assert sorted(o.tolist()) == list(range(n))
            assert [labels[k] for k in o] == [(p * D) // n for p in range(n)]
            for l in range(D):
                blk = o[l * n // D:(l + 1) * n // D]
                assert list(blk) == sorted(blk)
    with pytest.raises(ValueError):
        oracle.layout_order(np.array([0, 2, 1, 0], np.int32), 2)


@pytest.mark.parametrize("G,qpg,hd,N,D", [(4, 2, 8, 16, 2), (8, 2, 4, 32, 4), (6, 3, 4, 24, 3), (4, 1, 8, 12, 4)])
def test_layout_application_keeps_the_dense_function_and_shards_by_device(G, qpg, hd, N, D):
    d, T = 32, 12
    W = dense_block.random_layer(d, G * qpg, G, hd, N, seed=G + N)
    x = np.random.default_rng(5).standard_normal((T, d))
    h, nu = ablation.random_layout(1, G, N, D, seed=1000 + D)
    h, nu = h[0], nu[0]
    Wp, ho, no = dense_block.apply_layout(W, h, nu, D, G, hd)
    y = dense_block.block(x, W, G, hd)
    np.testing.assert_allclose(dense_block.block(x, Wp, G, hd), y, rtol=1e-12, atol=1e-12)
    # contiguous shards of the permuted block = the layout's devices; partials sum to the dense output
    shards = ([np.arange(l * G // D, (l + 1) * G // D) for l in range(D)],
              [np.arange(l * N // D, (l + 1) * N // D) for l in range(D)])
    yp, attn_p, ffn_p = dense_block.block(x, Wp, G, hd, parts=shards)
    for l in range(D):
        assert set(ho[shards[0][l]].tolist()) == set(np.flatnonzero(h == l).tolist())
        assert set(no[shards[1][l]].tolist()) == set(np.flatnonzero(nu == l).tolist())
    heads = dense_block.attention_heads(x, Wp, G, hd).reshape(T, -1)
    np.testing.assert_allclose(sum(attn_p), heads @ Wp["o"].T, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(x + sum(attn_p) + sum(ffn_p), yp, rtol=1e-12, atol=1e-12)


def test_a_wrong_permutation_changes_the_function():
    """Moving query heads without their KV group (or gate rows without down columns) breaks it."""
    G, qpg, hd, N, d, T = 4, 2, 8, 16, 32, 10
    W = dense_block.random_layer(d, G * qpg, G, hd, N, seed=3)
    x = np.random.default_rng(6).standard_normal((T, d))
    y = dense_block.block(x, W, G, hd)
    bad = dict(W)
    bad["gate"] = W["gate"][::-1].copy()
    bad["up"] = W["up"][::-1].copy()
    assert np.abs(dense_block.block(x, bad, G, hd) - y).max() > 1e-3
    bad = dense_block.permute_layer(W, [1, 0, 2, 3], np.arange(N), G, hd)
    bad["k"], bad["v"] = W["k"], W["v"]
    assert np.abs(dense_block.block(x, bad, G, hd) - y).max() > 1e-3
