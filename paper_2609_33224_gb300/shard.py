"""Column-block scoring: one instance pool split over several scheduler contexts.

Algorithm 1 (Section 6) evaluates every (request, instance) pair and then reduces each request's row
twice: W_min over the capacity-eligible set A (the reference point of Eq. 8's recompute filter),
then the smallest packing key over C.  Both reductions are minima, so when a pool's instances are
split into column blocks (one context each, e.g. one per GPU) a window is scored in two exchanges:

1. each block computes W_min over its own A (``ps_shard_wmin``); a MIN over blocks gives the pool's;
2. each block classifies its pairs under the pool's W_min and takes its smallest (key, tie)
   (``ps_shard_pick``); a MIN of the keys over blocks, then a MIN of the tie words among the blocks
   holding that key, gives the pool's pick.

The exchanges are plain all-reduce MINs of 64-bit integers (``allreduce_min``): over
``torch.distributed`` (NCCL between GPUs, gloo on CPU) or between threads of one process
(``LocalGroup``).  The greedy assignment does not split this way: each decision needs the state left
by the previous one, so it runs on one context holding the whole pool.
"""
from __future__ import annotations

import threading

import numpy as np

NO_KEY = (1 << 64) - 1       # a block with no candidate in C
NO_W = (1 << 32) - 1         # W_min bits of an empty A
TIE_INST_MASK_HCQ = 0xFFF    # under H-C-Q the tie word is qr << 12 | instance id


def _torch():
    import torch
    return torch


def _as_i64(x, bits: int):
    """Unsigned words (numpy uint32/uint64 or a torch int32/int64 tensor of raw bits) as a torch
    int64 tensor with the same order: u32 zero-extended, u64 with the top bit flipped."""
    torch = _torch()
    if isinstance(x, np.ndarray):
        if bits == 32:
            return torch.from_numpy(x.astype(np.uint32).astype(np.int64))
        return torch.from_numpy((x.astype(np.uint64) ^ np.uint64(1 << 63)).view(np.int64).copy())
    if bits == 32:
        return x.to(torch.int64) & 0xFFFFFFFF
    return x.to(torch.int64) ^ torch.iinfo(torch.int64).min


def dist_allreduce_min(group=None):
    """An ``allreduce_min`` over torch.distributed (in place on an int64 tensor, returned)."""
    import torch.distributed as dist

    def f(t):
        dist.all_reduce(t, op=dist.ReduceOp.MIN, group=group)
        return t
    return f


class LocalGroup:
    """Ranks that are threads of one process (e.g. one thread per GPU, each driving its own
    context): ``allreduce_min(rank)`` returns a function that blocks until every rank has
    contributed, then gives each rank the element-wise minimum."""

    def __init__(self, world: int):
        self.world = world
        self._bar = threading.Barrier(world)
        self._parts = [None] * world
        self._result = None

    def abort(self):
        """Release every rank waiting in an exchange (they raise threading.BrokenBarrierError):
        for a rank that failed and will not contribute."""
        self._bar.abort()

    def allreduce_min(self, rank: int):
        torch = _torch()

        def f(t):
            self._parts[rank] = t.detach().to("cpu")
            if self._bar.wait() == 0:
                self._result = torch.stack(self._parts).min(dim=0).values
            self._bar.wait()
            out = self._result.to(t.device)
            self._bar.wait()  # every rank has its copy before the next exchange overwrites it
            t.copy_(out)
            return t
        return f


def pool_wmin(local_wmin_ord, allreduce_min):
    """First exchange: the pool's W_min bits per request (int64 tensor) from this block's."""
    return allreduce_min(_as_i64(local_wmin_ord, 32).clone())


def merge_picks(key, tie, wmin_pool, allreduce_min, hcq: bool = False) -> dict:
    """Second exchange: the pool's pick per request from this block's (key, tie).

    Returns numpy ``best`` (int32 pool instance id, -1 = Reject) and ``path`` (uint8: 0 packed,
    1 fallback, 2 reject), identical on every rank."""
    torch = _torch()
    k = _as_i64(key, 64).clone()
    kmin = allreduce_min(k.clone())
    t = _as_i64(tie, 32)
    t = torch.where(k == kmin, t, torch.full_like(t, NO_W)).clone()
    tmin = allreduce_min(t)
    kmin_u = (kmin ^ torch.iinfo(torch.int64).min).cpu().numpy().view(np.uint64)
    tmin = tmin.cpu().numpy().astype(np.int64)
    wmin = wmin_pool.cpu().numpy() if hasattr(wmin_pool, "cpu") else np.asarray(wmin_pool)
    pick = (kmin_u != np.uint64(NO_KEY)) & (wmin != NO_W)
    inst = (tmin & TIE_INST_MASK_HCQ) if hcq else tmin
    best = np.where(pick, inst, -1).astype(np.int32)
    path = np.where(pick, (kmin_u >> np.uint64(62)).astype(np.int64), 2).astype(np.uint8)
    return {"best": best, "path": path}


def score_window_sharded(sched, window, id_base: int, allreduce_min, scores=(),
                         device_outputs: bool = False) -> dict:
    """Score ``window`` on one column block (``sched`` holds pool instances id_base ..
    id_base + sched.I - 1) and merge with the other blocks through ``allreduce_min``.

    Returns {"best", "path"} of the whole pool (as ps_score_window on one context holding every
    instance), "wmin" (the pool's W_min bits) and, with ``scores``, this block's columns of the
    per-pair outputs under the pool's W_min."""
    local = sched.shard_wmin(window, device_outputs=device_outputs)
    wpool = pool_wmin(local, allreduce_min)
    if device_outputs:
        torch = _torch()
        w_in = torch.where(wpool >= (1 << 31), wpool - (1 << 32), wpool).to(device=local.device, dtype=torch.int32)
    else:
        w_in = wpool.cpu().numpy().astype(np.uint32)
    part = sched.shard_pick(w_in, id_base, scores=scores, device_outputs=device_outputs)
    res = merge_picks(part["key"], part["tie"], wpool, allreduce_min, hcq=sched.selector == 5)
    res["wmin"] = wpool.cpu().numpy().astype(np.uint32)
    if scores:
        res["scores"] = part["scores"]
    return res
