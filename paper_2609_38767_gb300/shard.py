"""Sharding the train examples over ranks (one process per GPU).

Train examples are independent in every step of the path, so a job splits them
into contiguous shards, one per rank: rank r owns global examples
[r * n_local, (r + 1) * n_local). The queries (and, once solved, the
preconditioned queries) are replicated. Scores and top-k are computed per shard.
Two steps exchange data: the curvature fit over the training set (each rank's
sums are all-reduced before the factorisation, so every rank preconditions with
the same global curvature), and the merge of the per-rank top-k candidates into
the global top-k: an all-gather of n_q x k (index, score) pairs per rank, then a
top-k over the n_q x (world * k) candidates.

Ties: candidates are laid out rank-major and, within a rank, in the local
top-k order (score descending, index ascending); a top-k that prefers the
earlier position among equal scores therefore prefers the smaller global index,
which is the single-device rule.
"""
from __future__ import annotations

import torch


def shard_offset(rank: int, n_local: int) -> int:
    """First global train index owned by `rank` when every rank holds n_local examples."""
    return rank * n_local


def gather_candidates(idx: torch.Tensor, val: torch.Tensor, offset: int, dist, world: int):
    """All-gather the local top-k of every rank.

    idx (n_q, k) int32 local train indices, val (n_q, k) fp32 scores; returns
    (cand_idx int64 global indices, cand_val fp32), each (n_q, world * k),
    rank-major along the candidate axis."""
    gidx = idx.to(torch.int64) + offset
    if world == 1:
        return gidx, val
    idx_all = [torch.empty_like(gidx) for _ in range(world)]
    val_all = [torch.empty_like(val) for _ in range(world)]
    dist.all_gather(idx_all, gidx)
    dist.all_gather(val_all, val)
    return torch.cat(idx_all, dim=1), torch.cat(val_all, dim=1)


def merge_topk(idx, val, offset, k, dist, world, select):
    """Global top-k from the per-rank top-k.

    select(cand_val, k) -> (pos int tensor (n_q, k), top values): the positions
    of the k best candidates per row, earlier position first among equal
    scores (tda_topk on the device)."""
    cand_idx, cand_val = gather_candidates(idx, val, offset, dist, world)
    pos, top = select(cand_val.contiguous(), k)
    return cand_idx.gather(1, pos.to(torch.int64)), top


def device_select(tda):
    """select() for merge_topk through the library's top-k kernel."""
    def select(cand_val, k):
        n_q, n_c = cand_val.shape
        pos = torch.empty((n_q, k), dtype=torch.int32, device=cand_val.device)
        top = torch.empty((n_q, k), dtype=torch.float32, device=cand_val.device)
        tda.tda_topk(cand_val, n_q, n_c, n_c, k, pos, top)
        return pos, top
    return select


# ---------------------------------------------------------------- curvature fit over all shards
# The fit over the training set is the path's other exchange step: every rank
# accumulates its shard's sums, an all-reduce adds them, and every rank then
# factorises the same global curvature (the layouts are those tda.h documents).

def allreduce_fisher(state, n_layers: int, D: int, state_bytes: int, itemsize: int, dist, world: int) -> None:
    """Add the Fisher sums M of every layer over the ranks (between FIT_ACCUM and FACTOR).
    state: uint8 tensor of n_layers * state_bytes; itemsize 4 (F32 state) or 8 (F64)."""
    if world == 1:
        return
    dt = {4: torch.float32, 8: torch.float64}[itemsize]
    for l in range(n_layers):
        m = state[l * state_bytes + 64:l * state_bytes + 64 + D * D * itemsize].view(dt)
        dist.all_reduce(m)


def kfac_sum_ranges(k_in: int, k_out: int):
    """Double-index ranges of one layer's K-FAC state that hold sums: (factor sums, EK-FAC sums)."""
    ka, kg = k_in, k_out
    le = 8 + 2 * ka * ka + 2 * kg * kg + ka + kg
    return [(0, 1), (8, 8 + ka * ka + kg * kg)], [(1, 2), (le, le + ka * kg)]


def allreduce_kfac(states, n_layers: int, k_in: int, k_out: int, state_bytes: int, dist, world: int,
                   eigenvalue_sums: bool = False) -> None:
    """Add the K-FAC factor sums (before tda_kfac_eigen) or, with eigenvalue_sums, the EK-FAC
    eigenvalue sums (before tda_kfac_apply) of every layer over the ranks."""
    if world == 1:
        return
    factor, ekfac = kfac_sum_ranges(k_in, k_out)
    for l in range(n_layers):
        st = states[l * state_bytes:(l + 1) * state_bytes].view(torch.float64)
        for a, b in (ekfac if eigenvalue_sums else factor):
            dist.all_reduce(st[a:b])
