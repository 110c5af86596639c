"""Multi-rank host logic of the layer-sharded path, run as world_size-2 gloo ranks on CPU.

The GPU kernels are not involved: each rank produces stand-in per-layer
results on the CPU, and the tests check the sharding, the gather in layer
order and the max-over-ranks timing reduction that bench.py uses under
torchrun.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_13846_gb300 import shard


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, n_layers, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = shard.layers_for_rank(n_layers, rank, world)
        # stand-in per-layer results that encode their layer index
        h = torch.tensor([[layer, layer + 1] for layer in mine], dtype=torch.int32).reshape(len(mine), 2)
        score = torch.tensor([0.5 + layer for layer in mine], dtype=torch.float64)
        full = shard.gather_layer_results({"h": h, "score": score}, n_layers)
        t = shard.max_over_ranks(1.0 + rank)
        q.put((rank, mine, full["h"].tolist(), full["score"].tolist(), t))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("n_layers", [28, 5, 1])
def test_two_rank_shard_gather_and_max(n_layers):
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, n_layers, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    owned = sorted(layer for _, mine, _, _, _ in results for layer in mine)
    assert owned == list(range(n_layers))
    for rank, mine, h, score, t in results:
        assert h == [[i, i + 1] for i in range(n_layers)]
        assert score == [0.5 + i for i in range(n_layers)]
        assert t == 2.0


@pytest.mark.parametrize("n,world", [(28, 1), (28, 2), (28, 3), (16, 4), (3, 8), (0, 2)])
def test_layers_for_rank_partitions_exactly(n, world):
    seen = []
    sizes = []
    for r in range(world):
        block = shard.layers_for_rank(n, r, world)
        assert block == list(range(block[0], block[0] + len(block))) if block else True
        seen += block
        sizes.append(len(block))
    assert seen == list(range(n))
    assert max(sizes) - min(sizes) <= 1


def test_single_process_fallbacks():
    h = torch.arange(6).reshape(3, 2)
    assert torch.equal(shard.gather_layer_results({"h": h}, 3)["h"], h)
    assert shard.max_over_ranks(3.5) == 3.5
    with pytest.raises(ValueError):
        shard.layers_for_rank(4, 2, 2)


def _model_worker(rank, world, port, n_layers, q):
    """Each rank scores only its own layers (seeded stand-ins); after the all-gather the oracle's
    whole-model search must see the same matrices as a single process."""
    import numpy as np

    import oracle
    from paper_2609_13846_gb300 import synth
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = shard.layers_for_rank(n_layers, rank, world)
        up = torch.stack([synth.make_affinity_matrix(8, 64, seed=300 + i) for i in mine]) if mine else \
            torch.zeros((0, 8, 64))
        down = torch.stack([synth.make_affinity_matrix(8, 64, seed=400 + i) if i + 1 < n_layers
                            else torch.zeros(8, 64) for i in mine]) if mine else torch.zeros((0, 8, 64))
        S_up, S_down = shard.gather_model_affinities(up, down, n_layers)
        res = oracle.chain_search(S_up.numpy(), S_down.numpy() if n_layers > 1 else None, 4, 10)
        q.put((rank, S_up.shape[0], S_down.shape[0], int(res["J_q"]), res["h"].tolist()))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("n_layers,world", [(6, 2), (5, 2), (3, 3)])
def test_whole_model_search_after_gather(n_layers, world):
    import numpy as np

    import oracle
    from paper_2609_13846_gb300 import synth
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_model_worker, args=(r, world, port, n_layers, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=180) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    S_up = np.stack([synth.make_affinity_matrix(8, 64, seed=300 + i).numpy() for i in range(n_layers)])
    S_down = np.stack([synth.make_affinity_matrix(8, 64, seed=400 + i).numpy() for i in range(n_layers - 1)])
    ref = oracle.chain_search(S_up, S_down, 4, 10)
    for rank, nu_, nd_, jq, h in results:
        assert nu_ == n_layers and nd_ == n_layers - 1
        assert jq == ref["J_q"] and h == ref["h"].tolist()
