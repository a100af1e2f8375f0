"""Layer-wise ownership across data-parallel ranks (section 6, "layer-wise distributed optimizer").

Every weight matrix is stepped by exactly one rank (libsoap's soap_layerwise_assign: the paper's
size-sorted round-robin, or longest-processing-time first on the step's FLOPs); after its local
step each rank shares the matrices it updated with all others, one broadcast per owning rank
of its updated matrices packed end to end (a variable-size all-gather). The optimizer state
of a matrix lives only on its owner.

As in the paper's overlapped parameter all-gather, the exchange can be split into buckets of
consecutive matrices in the caller's (execution) order, each bucket's all-gather issued
asynchronously: ``step(..., overlap=True)`` returns a ``PendingExchange`` whose ``wait(b)``
completes bucket b alone, so the next forward pass can start on the first bucket's weights
while the later buckets are still in flight.

This module only plans and moves data: the step itself runs in the library's kernels (through
the optimizer object the caller's factory builds for the owned matrices), the exchange through
torch.distributed (NCCL on GPUs, gloo on the host).
"""
from __future__ import annotations

import torch
import torch.distributed as dist

from .soap import layerwise_assign


def plan_buckets(shapes, bucket_bytes=None, elem_bytes: int = 4):
    """Consecutive matrices (in the given order) grouped into buckets of at most ``bucket_bytes``
    bytes of weights each; a matrix larger than the bound gets a bucket of its own. ``None``:
    one bucket holding every matrix."""
    if bucket_bytes is None:
        return [list(range(len(shapes)))] if shapes else []
    if bucket_bytes <= 0:
        raise ValueError("bucket_bytes must be positive")
    buckets, cur, used = [], [], 0
    for i, s in enumerate(shapes):
        b = int(s[0]) * int(s[1]) * elem_bytes
        if cur and used + b > bucket_bytes:
            buckets.append(cur)
            cur, used = [], 0
        cur.append(i)
        used += b
    if cur:
        buckets.append(cur)
    return buckets


class PendingExchange:
    """The all-gather of one step's updated weights, in flight bucket by bucket. ``wait(b)``
    finishes bucket b's broadcasts and writes the matrices that other ranks own into ``params``;
    until then those matrices hold their previous values."""

    def __init__(self, params, pieces):
        self.params = params
        self.pieces = pieces          # per bucket: [(work, buf, indices, received)]
        self.done = [False] * len(pieces)

    def wait(self, b: int):
        if self.done[b]:
            return
        for work, buf, idx, received in self.pieces[b]:
            work.wait()
            if received:
                off = 0
                for i in idx:
                    k = self.params[i].numel()
                    self.params[i].copy_(buf[off:off + k].view_as(self.params[i]))
                    off += k
        self.pieces[b] = []
        self.done[b] = True

    def wait_all(self):
        for b in range(len(self.pieces)):
            self.wait(b)


class LayerwiseOptimizer:
    """Steps this rank's share of the matrices, then all-gathers the updated weights.

    ``shapes``: (rows, cols[, precond_left, precond_right]) per matrix, the same on every rank.
    ``make_optimizer(owned_shapes)``: builds the local optimizer for the owned matrices (an object
    with ``step(params, grads)``), e.g. ``lambda sh: SoapOptimizer(sh, hparams)``; it is not
    called on a rank that owns nothing.
    ``bucket_bytes``: the exchange's bucket bound (``plan_buckets``); ``None`` is one bucket.
    """

    def __init__(self, shapes, make_optimizer, group=None, policy: int = 0, bucket_bytes=None):
        self.group = group
        self.rank = dist.get_rank(group)
        self.world = dist.get_world_size(group)
        self.shapes = [tuple(s) for s in shapes]
        self.owner, self.load = layerwise_assign(self.shapes, self.world, policy)
        self.mine = [i for i, o in enumerate(self.owner) if o == self.rank]
        self.buckets = plan_buckets(self.shapes, bucket_bytes)
        # per bucket, per rank: the bucket's matrices that rank owns (its all-gather piece)
        self.pieces = [[[i for i in bkt if self.owner[i] == r] for r in range(self.world)] for bkt in self.buckets]
        self.opt = make_optimizer([self.shapes[i] for i in self.mine]) if self.mine else None

    def step(self, params, grads, overlap: bool = False):
        """One step: local step of the owned matrices, then the all-gather of updated weights.
        ``params`` (updated in place on every rank) and ``grads`` hold every matrix. With
        ``overlap`` the all-gather is left in flight and its ``PendingExchange`` returned."""
        if self.opt is not None:
            self.opt.step([params[i] for i in self.mine], [grads[i] for i in self.mine])
        if overlap:
            return self.start_exchange(params)
        self.exchange(params)
        return None

    def start_exchange(self, params) -> PendingExchange:
        """Issues every bucket's all-gather asynchronously, in bucket order: within a bucket each
        owning rank broadcasts its matrices packed end to end."""
        pending = []
        for per_rank in self.pieces:
            works = []
            for r, idx in enumerate(per_rank):
                if not idx:
                    continue
                if r == self.rank:
                    buf = torch.cat([params[i].reshape(-1) for i in idx])
                else:
                    n = sum(params[i].numel() for i in idx)
                    buf = torch.empty(n, dtype=params[idx[0]].dtype, device=params[idx[0]].device)
                src = dist.get_global_rank(self.group, r) if self.group is not None else r
                work = dist.broadcast(buf, src=src, group=self.group, async_op=True)
                works.append((work, buf, idx, r != self.rank))
            pending.append(works)
        return PendingExchange(params, pending)

    def exchange(self, params):
        """The whole all-gather, waited for: every rank holds every updated matrix afterwards."""
        self.start_exchange(params).wait_all()

    # the local optimizer's status and profiling, for a caller that treats this like one handle
    def status(self) -> int:
        return self.opt.status() if self.opt is not None else 0

    def last_error(self) -> str:
        return self.opt.last_error() if self.opt is not None else ""

    def profile_begin(self, max_launches: int = 1 << 16):
        if self.opt is not None:
            self.opt.profile_begin(max_launches)

    def profile_end(self) -> dict:
        if self.opt is not None:
            return self.opt.profile_end()
        from .soap import KERNEL_FAMILIES
        res = {k: dict(launches=0, ms=0.0, flops=0.0, bytes=0.0) for k in KERNEL_FAMILIES}
        res["overflow"] = False
        return res

    def destroy(self):
        if self.opt is not None:
            self.opt.destroy()
            self.opt = None
