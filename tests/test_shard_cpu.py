"""Multi-rank host logic on CPU (gloo, world size 2): sharding of the train
examples and the merge of per-rank top-k candidates into the global top-k."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_38767_gb300 import shard


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _cpu_select(cand_val, k):
    # descending, earlier candidate position first among equal scores (the device top-k's rule)
    v = cand_val.numpy()
    pos = np.argsort(-v, axis=1, kind="stable")[:, :k]
    return torch.from_numpy(pos.astype(np.int32)), torch.from_numpy(np.take_along_axis(v, pos, 1))


def _worker(rank, world, port, S, k, out_dir):
    import oracle

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        n_local = S.shape[1] // world
        off = shard.shard_offset(rank, n_local)
        idx, val = oracle.topk(S[:, off:off + n_local], k)
        gidx, gval = shard.merge_topk(torch.from_numpy(idx), torch.from_numpy(val.astype(np.float32)), off, k, dist,
                                      world, _cpu_select)
        np.save(os.path.join(out_dir, f"r{rank}.npy"), gidx.numpy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("ties", [False, True])
def test_merge_topk_equals_global_topk_two_ranks(tmp_path, orc, ties):
    rng = np.random.default_rng(5)
    nq, n_local, k, world = 4, 50, 12, 2
    S = rng.standard_normal((nq, world * n_local)).astype(np.float32)
    if ties:
        S = np.round(S, 1)  # many equal scores across the two shards
    mp.start_processes(_worker, args=(world, _free_port(), S, k, str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    want, _ = orc.topk(S.astype(np.float64), k)
    for r in range(world):
        np.testing.assert_array_equal(np.load(tmp_path / f"r{r}.npy"), want)


def test_shards_are_disjoint_and_cover_the_job():
    n_local, world = 37, 4
    ranges = [range(shard.shard_offset(r, n_local), shard.shard_offset(r, n_local) + n_local) for r in range(world)]
    flat = [i for rg in ranges for i in rg]
    assert flat == list(range(world * n_local))
