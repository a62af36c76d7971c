"""Multi-rank host logic on CPU (gloo, world size 2): sharding of the train
examples, the merge of per-rank top-k candidates into the global top-k, and the
all-reduce that fits the curvature over all shards."""
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


def _curv_worker(rank, world, port, phis, D, out_dir):
    import oracle

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # a two-layer fp32 precondition state laid out as tda.h documents: 64-byte header, M, then
        # the diagonal-block inverses; this rank's sums Phi_r^T Phi_r in M, its own marks elsewhere
        nl, nblk = 2, (D + 31) // 32
        per = (64 + (D * D + nblk * 1024) * 4 + 255) // 256 * 256
        st = torch.zeros(nl * per, dtype=torch.uint8)
        for l in range(nl):
            P = phis[rank][:, l * D:(l + 1) * D].astype(np.float64)
            st[l * per + 64:l * per + 64 + D * D * 4].view(torch.float32)[:] = torch.from_numpy(
                (P.T @ P).astype(np.float32).reshape(-1))
            st[l * per:l * per + 64].view(torch.float64)[:] = float(rank + 1)
            st[l * per + 64 + D * D * 4:(l + 1) * per].view(torch.float32)[:] = float(10 + rank)
        shard.allreduce_fisher(st, nl, D, per, 4, dist, world)
        np.save(os.path.join(out_dir, f"f{rank}.npy"), st.numpy())
        # K-FAC state (fp64): every double marked with the rank; only the documented sums add up
        ka, kg = 3, 5
        tot = 8 + 2 * ka * ka + 2 * kg * kg + ka + kg + ka * kg
        kper = (tot * 8 + 255) // 256 * 256
        ks = torch.zeros(2 * kper, dtype=torch.uint8)
        for l in range(2):
            ks[l * kper:(l + 1) * kper].view(torch.float64)[:] = torch.arange(kper // 8, dtype=torch.float64) + rank
        shard.allreduce_kfac(ks, 2, ka, kg, kper, dist, world)
        np.save(os.path.join(out_dir, f"k{rank}.npy"), ks.numpy())
        shard.allreduce_kfac(ks, 2, ka, kg, kper, dist, world, eigenvalue_sums=True)
        np.save(os.path.join(out_dir, f"e{rank}.npy"), ks.numpy())
    finally:
        dist.destroy_process_group()


def test_curvature_sums_add_over_ranks(tmp_path, orc):
    # the fit over all shards: per-rank sums all-reduced equal the sums over the whole training set;
    # header, inverses and the non-sum parts of a K-FAC state stay as each rank had them
    rng = np.random.default_rng(9)
    world, D, n = 2, 40, 30
    phis = [rng.standard_normal((n, 2 * D)).astype(np.float32) for _ in range(world)]
    mp.start_processes(_curv_worker, args=(world, _free_port(), phis, D, str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    nblk = (D + 31) // 32
    per = (64 + (D * D + nblk * 1024) * 4 + 255) // 256 * 256
    allphi = np.concatenate(phis).astype(np.float64)
    for r in range(world):
        st = np.load(tmp_path / f"f{r}.npy")
        for l in range(2):
            M = st[l * per + 64:l * per + 64 + D * D * 4].view(np.float32).reshape(D, D)
            want = orc.fisher(allphi[:, l * D:(l + 1) * D]) * (world * n)  # F = M / n_total
            np.testing.assert_allclose(M, want, rtol=1e-5, atol=1e-4)
            assert (st[l * per:l * per + 64].view(np.float64) == r + 1).all()
            assert (st[l * per + 64 + D * D * 4:(l + 1) * per].view(np.float32) == 10 + r).all()
    ka, kg = 3, 5
    factor, ekfac = shard.kfac_sum_ranges(ka, kg)
    tot = 8 + 2 * ka * ka + 2 * kg * kg + ka + kg + ka * kg
    kper = (tot * 8 + 255) // 256 * 256
    base = np.arange(kper // 8, dtype=np.float64)
    for r in range(world):
        for name, summed in (("k", factor), ("e", factor + ekfac)):
            ks = np.load(tmp_path / f"{name}{r}.npy")
            for l in range(2):
                v = ks[l * kper:(l + 1) * kper].view(np.float64)
                want = base + r
                for a, b in summed:
                    want[a:b] = 2 * base[a:b] + 1  # (base + 0) + (base + 1)
                np.testing.assert_array_equal(v, want)
