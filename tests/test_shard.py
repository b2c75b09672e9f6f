"""Multi-rank path on CPU: two gloo ranks each score their own block of
requests (no data-path collective); the union equals scoring the whole batch
in one process, and timing reduces to the max over ranks."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import shard
from paper_2607_28940_gb300 import workload as W

PER_RANK = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_req=3, L=("uniform", 5, 40), M=("uniform", 0, 9), dL=2)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        gwl = shard.global_workload(PER_RANK, world)
        reqs = shard.shard_requests(PER_RANK.n_req, rank, world)
        b = W.batch(gwl, requests=reqs)
        model = O.Model.from_arrays(W.weights(gwl), gwl)
        caches = O.append_caches(model, O.build_caches(model, b.beh, b.beh_off), b.app, b.app_off)
        lg, _ = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off)
        np.save(os.path.join(out_dir, f"lg{rank}.npy"), lg)
        np.save(os.path.join(out_dir, f"req{rank}.npy"), np.asarray(reqs))
        t = shard.reduce_max(10.0 + rank)
        np.save(os.path.join(out_dir, f"t{rank}.npy"), np.asarray([t]))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_partition_requests(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    reqs = [np.load(tmp_path / f"req{r}.npy") for r in range(world)]
    assert sorted(np.concatenate(reqs).tolist()) == list(range(world * PER_RANK.n_req))
    assert not set(reqs[0]) & set(reqs[1])
    assert all(float(np.load(tmp_path / f"t{r}.npy")[0]) == 11.0 for r in range(world))
    gwl = shard.global_workload(PER_RANK, world)
    b = W.batch(gwl)
    model = O.Model.from_arrays(W.weights(gwl), gwl)
    caches = O.append_caches(model, O.build_caches(model, b.beh, b.beh_off), b.app, b.app_off)
    whole, _ = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off)
    parts = np.concatenate([np.load(tmp_path / f"lg{r}.npy") for r in range(world)])
    np.testing.assert_allclose(parts, whole, rtol=0, atol=1e-12)


def test_shard_bounds():
    assert shard.shard_requests(4, 1, 3) == [4, 5, 6, 7]
    import pytest
    with pytest.raises(ValueError):
        shard.shard_requests(4, 3, 3)
    assert shard.reduce_max(3.5) == 3.5
