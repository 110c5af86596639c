"""Ablation layouts of Sec. 3 ("Optimiser") and Table 4: which layers move, and random layouts.

Host-side configuration only.  The masks feed ``dtp.search_chain`` (and the
oracle) as ``move_heads`` / ``move_neurons``; the random layouts feed
``dtp.chain_score``.
"""
from __future__ import annotations

import numpy as np


def evenly_spaced_layers(L: int, n: int) -> list[int]:
    """n of L layers, evenly spaced and always including layer 0: floor(j L / n), j < n.

    The layer-subset ablation optimises 4, 8 or 12 such layers and keeps the
    rest contiguous; 28 layers and n = 4 give 0, 7, 14, 21.
    """
    if not 1 <= n <= L:
        raise ValueError(f"need 1 <= n <= L, got n={n}, L={L}")
    return [(j * L) // n for j in range(n)]


def layer_mask(L: int, layers) -> np.ndarray:
    """uint8 [L], 1 on the listed layers."""
    m = np.zeros(L, np.uint8)
    m[list(layers)] = 1
    return m


def ablation_masks(L: int, kind: str) -> tuple[np.ndarray | None, np.ndarray | None, bool]:
    """(move_heads, move_neurons, minimize) of a named ablation layout.

    'optimised' (everything), 'anti' (everything, J minimised), 'heads_only'
    (neurons contiguous), 'neurons_only' (KV groups contiguous), 'layers<n>'
    (n evenly spaced layers, the rest contiguous).
    """
    ones, zeros = np.ones(L, np.uint8), np.zeros(L, np.uint8)
    if kind == "optimised":
        return None, None, False
    if kind == "anti":
        return None, None, True
    if kind == "heads_only":
        return ones, zeros, False
    if kind == "neurons_only":
        return zeros, ones, False
    if kind.startswith("layers"):
        m = layer_mask(L, evenly_spaced_layers(L, int(kind[len("layers"):])))
        return m, m.copy(), False
    raise ValueError(f"unknown ablation {kind!r}")


def random_layout(L: int, G: int, N: int, D: int, seed: int) -> tuple[np.ndarray, np.ndarray]:
    """A uniformly random balanced layout: h [L, G] and nu [L, N] int32, G/D heads and N/D neurons per device."""
    if G % D or N % D:
        raise ValueError("D must divide G and N")
    rng = np.random.default_rng(seed)
    h = np.stack([rng.permutation(np.repeat(np.arange(D), G // D)) for _ in range(L)]).astype(np.int32)
    nu = np.stack([rng.permutation(np.repeat(np.arange(D), N // D)) for _ in range(L)]).astype(np.int32)
    return h, nu
