"""Halo exchange and gradient reduction for a supergraph split into block-row ranges across ranks
(bg_plan_partition; Eq. 3: block-row k couples only to block-rows k - 1 and k + 1).

Each rank holds its local rows [0, n_local): halo rows from rank - 1, its own rows
[own_begin, own_end), halo rows from rank + 1.  Before a forward propagation the halo rows of E,
before a backward one those of dY, are filled from the neighbours' own rows; after the backward
the weight gradients are summed over the ranks.  Point-to-point over torch.distributed: NCCL for
device tensors, gloo for host tensors.  Argument marshalling only; no arithmetic of the method.
"""
from __future__ import annotations


def halo_plan(infos: list) -> list:
    """For every rank r the copies that fill its halo rows, as (src_rank, src_row0, dst_row0,
    rows) in local row numbers: rank r - 1's last halo_lo own rows into [0, halo_lo), rank
    r + 1's first halo_hi own rows into [own_end, n_local)."""
    out = []
    for r, inf in enumerate(infos):
        cp = []
        if inf["halo_lo"]:
            nb = infos[r - 1]
            cp.append((r - 1, nb["own_end"] - inf["halo_lo"], 0, inf["halo_lo"]))
        if inf["halo_hi"]:
            nb = infos[r + 1]
            cp.append((r + 1, nb["own_begin"], inf["own_end"], inf["halo_hi"]))
        out.append(cp)
    return out


def exchange(local, info: dict, rank: int, world: int, group=None):
    """Fills the halo rows of this rank's `local` tensor ([n_local, ...]) from the neighbouring
    ranks' own rows (one send and one receive per neighbour)."""
    import torch.distributed as dist
    ops = []
    lo, hi = info["halo_lo"], info["halo_hi"]
    ob, oe = info["own_begin"], info["own_end"]
    # the neighbours' halos have the same size as ours on the shared boundary
    if rank > 0:
        ops.append(dist.P2POp(dist.isend, local[ob:ob + lo].contiguous(), rank - 1, group))
        ops.append(dist.P2POp(dist.irecv, local[0:lo], rank - 1, group))
    if rank + 1 < world:
        ops.append(dist.P2POp(dist.isend, local[oe - hi:oe].contiguous(), rank + 1, group))
        ops.append(dist.P2POp(dist.irecv, local[oe:oe + hi], rank + 1, group))
    if ops:
        for req in dist.batch_isend_irecv(ops):
            req.wait()


def allreduce_sum(tensors, group=None):
    """Sums each tensor over the ranks in place (the weight gradients of a split supergraph)."""
    import torch.distributed as dist
    for t in tensors:
        dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
