"""Plain fp64 dense Transformer block and layout application -- TEST INFRASTRUCTURE.

Checks the layout application of Sec. 3: a layout (h, nu) is applied by
permuting the dense model's KV groups (with their query heads) and FFN neurons
so that every device's heads and neurons form one contiguous shard.  A
permutation of heads and neurons leaves the dense function unchanged; the
contiguous shards then split it into per-device partial outputs whose sum is
the dense output (the tensor-parallel decomposition the delayed form starts
from).

Weights follow nn.Linear's [out, in]: q [Hq*hd, d], k and v [G*hd, d],
o [d, Hq*hd], gate and up [N, d], down [d, N]; norms attn_norm / ffn_norm [d]
and the per-head q_norm / k_norm [hd].  Query heads g*qpg .. g*qpg+qpg-1 share
KV group g.  Only tests may import this module.
"""
from __future__ import annotations

import numpy as np

from . import layout_order


def _rms(x, w, eps=1e-6):
    return w * x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps)


def _rope(x, base=10000.0):
    """Rotary position embedding on [T, heads, hd] (pairs (i, i + hd/2))."""
    T, _, hd = x.shape
    half = hd // 2
    inv = base ** (-np.arange(half) / half)
    ang = np.arange(T)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def _silu(z):
    return z / (1.0 + np.exp(-z))


def attention_heads(x, W, G: int, hd: int):
    """Per-query-head attention outputs [T, Hq, hd] of the block's attention (causal, GQA)."""
    T = x.shape[0]
    a = _rms(x, W["attn_norm"])
    q = (a @ W["q"].T).reshape(T, -1, hd)
    k = (a @ W["k"].T).reshape(T, G, hd)
    v = (a @ W["v"].T).reshape(T, G, hd)
    if "q_norm" in W:
        q, k = _rms(q, W["q_norm"]), _rms(k, W["k_norm"])
    q, k = _rope(q), _rope(k)
    Hq = q.shape[1]
    qpg = Hq // G
    mask = np.triu(np.full((T, T), -np.inf), 1)
    out = np.empty_like(q)
    for h in range(Hq):
        s = q[:, h] @ k[:, h // qpg].T / np.sqrt(hd) + mask
        p = np.exp(s - s.max(axis=1, keepdims=True))
        out[:, h] = (p / p.sum(axis=1, keepdims=True)) @ v[:, h // qpg]
    return out


def block(x, W, G: int, hd: int, parts=None):
    """The dense block x -> x + attn + ffn in fp64.  With ``parts`` = (head_sets, neuron_sets) it
    also returns each device's partial attention and FFN outputs (its heads' and neurons' terms)."""
    T = x.shape[0]
    heads = attention_heads(x, W, G, hd)
    o = heads.reshape(T, -1) @ W["o"].T
    h2 = x + o
    f = _rms(h2, W["ffn_norm"])
    act = _silu(f @ W["gate"].T) * (f @ W["up"].T)
    y = h2 + act @ W["down"].T
    if parts is None:
        return y
    Hq = heads.shape[1]
    qpg = Hq // G
    attn_p, ffn_p = [], []
    for groups, neurons in zip(*parts):
        cols = np.concatenate([np.arange(g * qpg * hd, (g + 1) * qpg * hd) for g in groups]) if len(groups) else \
            np.zeros(0, int)
        attn_p.append(heads.reshape(T, -1)[:, cols] @ W["o"][:, cols].T)
        ffn_p.append(act[:, neurons] @ W["down"][:, neurons].T)
    return y, attn_p, ffn_p


def permute_layer(W, head_order, neuron_order, G: int, hd: int):
    """Weights with KV group p = head_order[p] and neuron p = neuron_order[p] of the input."""
    Hq = W["q"].shape[0] // hd
    qpg = Hq // G
    qrows = np.concatenate([np.arange(g * qpg * hd, (g + 1) * qpg * hd) for g in head_order])
    kvrows = np.concatenate([np.arange(g * hd, (g + 1) * hd) for g in head_order])
    out = dict(W)
    out["q"] = W["q"][qrows]
    out["k"] = W["k"][kvrows]
    out["v"] = W["v"][kvrows]
    out["o"] = W["o"][:, qrows]
    out["gate"] = W["gate"][neuron_order]
    out["up"] = W["up"][neuron_order]
    out["down"] = W["down"][:, neuron_order]
    return out


def apply_layout(W, h, nu, D: int, G: int, hd: int):
    """Permute one layer for layout (h [G], nu [N]): device l's groups and neurons become the
    contiguous shard l (groups l*G/D .., neurons l*N/D ..).  Returns (weights, head_order, neuron_order)."""
    ho, no = layout_order(h, D), layout_order(nu, D)
    return permute_layer(W, ho, no, G, hd), ho, no


def random_layer(d: int, Hq: int, G: int, hd: int, N: int, seed: int, qk_norm: bool = True):
    rng = np.random.default_rng(seed)
    W = dict(q=rng.standard_normal((Hq * hd, d)) / np.sqrt(d), k=rng.standard_normal((G * hd, d)) / np.sqrt(d),
             v=rng.standard_normal((G * hd, d)) / np.sqrt(d), o=rng.standard_normal((d, Hq * hd)) / np.sqrt(Hq * hd),
             gate=rng.standard_normal((N, d)) / np.sqrt(d), up=rng.standard_normal((N, d)) / np.sqrt(d),
             down=rng.standard_normal((d, N)) / np.sqrt(N), attn_norm=1 + 0.1 * rng.standard_normal(d),
             ffn_norm=1 + 0.1 * rng.standard_normal(d))
    if qk_norm:
        W["q_norm"] = 1 + 0.1 * rng.standard_normal(hd)
        W["k_norm"] = 1 + 0.1 * rng.standard_normal(hd)
    return W
