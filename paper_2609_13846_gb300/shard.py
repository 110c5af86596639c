"""Layer sharding across ranks for the affinity pass and the layout search.

The up-edge objective (Sec. 3, Eq. objective, first sum) decouples across
layers, and a layer's affinity depends only on that layer's calibration
inputs, so a model's layers are split across ranks (one process per GPU) with
no exchange on the data path.  Results are gathered once at the end.

The whole-model objective (both sums) couples neighbouring layers, but its
inputs do not: each rank scores the up edge of its layers and the down edge
leaving each of them (which needs only the next layer's weights and the rms of
its input), then one all-gather gives every rank the full set of matrices and
the optimiser runs on them (milliseconds on one GPU).
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def layers_for_rank(n_layers: int, rank: int, world: int) -> list[int]:
    """Contiguous block of layers owned by ``rank``; blocks differ in size by at most one."""
    if world < 1 or not 0 <= rank < world or n_layers < 0:
        raise ValueError("need world >= 1, 0 <= rank < world, n_layers >= 0")
    base, extra = divmod(n_layers, world)
    start = rank * base + min(rank, extra)
    count = base + (1 if rank < extra else 0)
    return list(range(start, start + count))


def max_over_ranks(value: float, device=None) -> float:
    """The maximum of a per-rank scalar (e.g. elapsed time) over all ranks."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def gather_layer_results(local: dict, n_layers: int, device=None) -> dict:
    """Assemble per-layer results from every rank, in layer order, on every rank.

    ``local`` maps names to tensors whose first dimension indexes this rank's
    layers (``layers_for_rank``); trailing shapes and dtypes agree across ranks.
    Returns the same names with a first dimension of ``n_layers``.
    """
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return {k: v.clone() for k, v in local.items()}
    world, rank = dist.get_world_size(), dist.get_rank()
    counts = [len(layers_for_rank(n_layers, r, world)) for r in range(world)]
    width = max(counts)
    out = {}
    for name in sorted(local):
        t = local[name].to(device) if device is not None else local[name]
        if t.shape[0] != counts[rank]:
            raise ValueError(f"{name}: rank {rank} holds {t.shape[0]} layers, expected {counts[rank]}")
        pad = torch.zeros((width,) + tuple(t.shape[1:]), dtype=t.dtype, device=t.device)
        pad[: t.shape[0]] = t
        parts = [torch.empty_like(pad) for _ in range(world)]
        dist.all_gather(parts, pad)
        out[name] = torch.cat([parts[r][: counts[r]] for r in range(world)], dim=0)
    return out


def gather_model_affinities(S_up_local: torch.Tensor, S_down_local: torch.Tensor, n_layers: int,
                            device=None) -> tuple[torch.Tensor, torch.Tensor]:
    """All-gather a layer-sharded model's affinity matrices for the whole-model search.

    S_up_local [n_mine, G, N]: the up edges of this rank's layers
    (``layers_for_rank``); S_down_local [n_mine, G, N]: the down edge leaving
    each of them (any values for the model's last layer, which has none).
    Returns S_up [n_layers, G, N] and S_down [n_layers - 1, G, N] on every rank.
    """
    full = gather_layer_results({"up": S_up_local, "down": S_down_local}, n_layers, device=device)
    return full["up"], full["down"][: max(n_layers - 1, 0)]
