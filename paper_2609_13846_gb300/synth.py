"""Seeded synthetic inputs for the affinity pass and the layout search.

This module holds only random-number recipes; none of the method's arithmetic.
It is the one piece shared by the CUDA path's callers and by the oracle's
tests.

The paper calibrates on 64 x 1024 FineWeb-Edu tokens through Qwen3-0.6B and
Danube3-500M (Sec. 3 "Affinity scores", Sec. 4 "Models and sharding"); neither
the data nor the weights are available, so seeded Gaussian stand-ins with the
paper's shapes are used:

* ``X`` [T, d]: the FFN input after RMSNorm.  N(0,1); in the model-shaped
  workloads 4 distinct channels (drawn by the generator) are scaled by 20 to
  mimic massive-activation outlier channels (Sec. 5.6 "Where the affinity
  concentrates").  The tiny workload draws N(0,1)/sqrt(d) without outliers.
* ``C`` [G, T, d]: each KV group's piece of the normalised FFN input
  (p_h = gamma * (a_h W_o^(h)) / r, Sec. 3).  Z_h ~ N(0,1) rescaled so that
  ||C_h||_F = s_h ||X||_F with s_h log-uniform in [0.1, 1] (tiny workload:
  N(0,1)/sqrt(d)).
* ``W_gate``, ``W_up`` [N, d] and ``W_down`` [d, N]: N(0, 0.02^2).

Draw order for one layer: X, outlier indices, head scales, Z_0..Z_{G-1},
W_gate, W_up, W_down.  Everything is drawn in fp32 from a ``torch.Generator``
on ``device`` and, in bf16 mode, rounded to bf16 once; the CUDA path and the
oracle then read the same rounded values.  The same seed gives different
draws on a CPU and a CUDA generator.
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    """One calibration-layer shape: d, KV groups G, FFN neurons N, tokens T, devices D."""

    name: str
    d: int
    G: int
    N: int
    T: int
    D: tuple
    dtype: str  # "bf16" or "f32"
    layers: int = 1
    seed: int = 0
    outliers: bool = True
    iters: int = 10
    qkv_rows: int = 512   # next layer's q/k/v rows per KV group: (query heads per group + 2) * head_dim
    head_dim: int = 128
    q_per_group: int = 2  # query heads per KV group

    def layer_seed(self, layer: int) -> int:
        """Seed of layer ``layer``: the workload seed plus the layer index."""
        return self.seed + layer


# The five calibration workloads.  FLOP per token of the affinity pass is
# 2*d*2N*(G+1).
WORKLOADS = {
    "tiny": Workload("tiny", d=64, G=2, N=128, T=256, D=(2,), dtype="f32", seed=0, outliers=False, qkv_rows=64,
                     head_dim=16),
    "qwen3_0.6b_layer": Workload("qwen3_0.6b_layer", d=1024, G=8, N=3072, T=16384, D=(2,),
                                 dtype="bf16", seed=1),
    "qwen3_0.6b_model": Workload("qwen3_0.6b_model", d=1024, G=8, N=3072, T=65536, D=(2, 4),
                                 dtype="bf16", layers=28, seed=100),
    "danube3_500m_model": Workload("danube3_500m_model", d=1536, G=8, N=4096, T=65536, D=(4,),
                                   dtype="bf16", layers=16, seed=200, qkv_rows=384, head_dim=96),
    "llama3.1_8b_layer": Workload("llama3.1_8b_layer", d=4096, G=8, N=14336, T=32768, D=(4, 8),
                                  dtype="bf16", seed=3, qkv_rows=768, q_per_group=4),
}


def _randn(gen, shape, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32)


def make_layer(d: int, G: int, N: int, T: int, seed: int, *, dtype: str = "bf16",
               outliers: bool = True, device="cpu", with_down: bool = False):
    """Draw one layer's calibration inputs.  Returns a dict of tensors on ``device``.

    Keys: X [T,d], C [G,T,d], W_gate [N,d], W_up [N,d] (and W_down [d,N] when
    ``with_down``), all bf16 or fp32 per ``dtype``.
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    if outliers:
        X = _randn(gen, (T, d), device)
        idx = torch.randperm(d, generator=gen, device=device)[:4]
        X[:, idx] *= 20.0
        u = torch.rand((G,), generator=gen, device=device, dtype=torch.float32)
        scales = torch.exp(math.log(0.1) * (1.0 - u))  # log-uniform in [0.1, 1]
        xnorm = torch.linalg.vector_norm(X)
        C = torch.empty((G, T, d), device=device, dtype=torch.float32)
        for h in range(G):
            Z = _randn(gen, (T, d), device)
            C[h] = Z * (scales[h] * xnorm / torch.linalg.vector_norm(Z))
    else:
        X = _randn(gen, (T, d), device) / math.sqrt(d)
        C = _randn(gen, (G, T, d), device) / math.sqrt(d)
    W_gate = _randn(gen, (N, d), device) * 0.02
    W_up = _randn(gen, (N, d), device) * 0.02
    out = dict(X=X, C=C, W_gate=W_gate, W_up=W_up)
    if with_down:
        out["W_down"] = _randn(gen, (d, N), device) * 0.02
    if dtype == "bf16":
        out = {k: v.to(torch.bfloat16) for k, v in out.items()}
    elif dtype != "f32":
        raise ValueError(f"dtype must be 'bf16' or 'f32', got {dtype!r}")
    return out


def make_workload_layer(w: Workload, layer: int = 0, *, T: int | None = None, device="cpu",
                        with_down: bool = False):
    """Inputs of ``layer`` of workload ``w``; ``T`` overrides the token count (a slice)."""
    return make_layer(w.d, w.G, w.N, w.T if T is None else T, w.layer_seed(layer), dtype=w.dtype,
                      outliers=w.outliers, device=device, with_down=with_down)


def make_affinity_matrix(G: int, N: int, seed: int, *, kind: str = "lognormal", device="cpu"):
    """A synthetic nonnegative affinity matrix [G, N] fp32 for search-only tests.

    ``lognormal``: continuous positive values with a spread like a real layer's
    (per-head scale times per-entry noise).  ``integer``: small integers 0..3,
    which make ties common.  ``zeros``: all zero.
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    if kind == "lognormal":
        head = torch.exp(torch.randn((G, 1), generator=gen, device=device))
        return (head * torch.exp(2.0 * torch.randn((G, N), generator=gen, device=device))).float()
    if kind == "integer":
        return torch.randint(0, 4, (G, N), generator=gen, device=device).float()
    if kind == "zeros":
        return torch.zeros((G, N), device=device, dtype=torch.float32)
    raise ValueError(kind)


def make_down_inputs(d: int, G: int, R: int, N: int, T: int, seed: int, *, dtype: str = "bf16", device="cpu"):
    """Seeded stand-ins for the next layer's side of the down edge (Sec. 3).

    Wqkv [G, R, d]: the next layer's q/k/v rows of each KV group, N(0, 0.02^2);
    gamma [d]: its pre-norm gain, 1 + N(0, 0.1^2); W_down [d, N]: this layer's
    down projection, N(0, 0.02^2); rms [T] fp32: the rms of the residual entering
    the next pre-norm, uniform in [0.5, 1.5].  Draw order as listed.
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    out = dict(Wqkv=_randn(gen, (G, R, d), device) * 0.02,
               gamma=1.0 + 0.1 * _randn(gen, (d,), device),
               W_down=_randn(gen, (d, N), device) * 0.02)
    rms = 0.5 + torch.rand((T,), generator=gen, device=device, dtype=torch.float32)
    if dtype == "bf16":
        out = {k: v.to(torch.bfloat16) for k, v in out.items()}
    out["rms"] = rms
    return out


def make_attention_inputs(T: int, d: int, Hq: int, head_dim: int, seed: int, *, device="cpu"):
    """Seeded stand-ins for the producer of C (Sec. 3: p_h = gamma . (a_h W_o^(h)T) / r).

    attn [T, Hq*head_dim] bf16: the heads' outputs before o_proj, N(0,1) with
    head h scaled by s_h log-uniform in [0.1, 1]; W_o [d, Hq*head_dim] bf16:
    N(0, 0.02^2); gamma [d] fp32: 1 + N(0, 0.1^2); rms [T] fp32: uniform in
    [0.5, 1.5].  Draw order as listed (the head scales first).
    """
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    u = torch.rand((Hq,), generator=gen, device=device, dtype=torch.float32)
    scales = torch.exp(math.log(0.1) * (1.0 - u)).repeat_interleave(head_dim)
    attn = (_randn(gen, (T, Hq * head_dim), device) * scales).to(torch.bfloat16)
    W_o = (_randn(gen, (d, Hq * head_dim), device) * 0.02).to(torch.bfloat16)
    gamma = 1.0 + 0.1 * _randn(gen, (d,), device)
    rms = 0.5 + torch.rand((T,), generator=gen, device=device, dtype=torch.float32)
    return dict(attn=attn, W_o=W_o, gamma=gamma, rms=rms)


def make_dense_weights(layers: int, d: int, Hq: int, G: int, head_dim: int, N: int, seed: int, *, device="cpu"):
    """Stacked bf16 stand-ins for a model's permuted weights [layers, ...]: q [Hq*hd, d], k and v
    [G*hd, d], o [d, Hq*hd], gate and up [N, d], down [d, N], all N(0, 0.02^2), drawn in that order."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    shapes = dict(q=(Hq * head_dim, d), k=(G * head_dim, d), v=(G * head_dim, d), o=(d, Hq * head_dim),
                  gate=(N, d), up=(N, d), down=(d, N))
    return {k: (_randn(gen, (layers, *sh), device) * 0.02).to(torch.bfloat16) for k, sh in shapes.items()}
