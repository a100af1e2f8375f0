"""Layer-wise ownership across data-parallel ranks (section 6, "layer-wise distributed optimizer").

Every weight matrix is stepped by exactly one rank (libsoap's soap_layerwise_assign: the paper's
size-sorted round-robin, or longest-processing-time first on the step's FLOPs); after its local
step each rank shares the matrices it updated with all others, one broadcast per owning rank
of its updated matrices packed end to end (a variable-size all-gather). The optimizer state
of a matrix lives only on its owner.

This module only plans and moves data: the step itself runs in the library's kernels (through
the optimizer object the caller's factory builds for the owned matrices), the exchange through
torch.distributed (NCCL on GPUs, gloo on the host).
"""
from __future__ import annotations

import torch
import torch.distributed as dist

from .soap import layerwise_assign


class LayerwiseOptimizer:
    """Steps this rank's share of the matrices, then all-gathers the updated weights.

    ``shapes``: (rows, cols[, precond_left, precond_right]) per matrix, the same on every rank.
    ``make_optimizer(owned_shapes)``: builds the local optimizer for the owned matrices (an object
    with ``step(params, grads)``), e.g. ``lambda sh: SoapOptimizer(sh, hparams)``; it is not
    called on a rank that owns nothing.
    """

    def __init__(self, shapes, make_optimizer, group=None, policy: int = 0):
        self.group = group
        self.rank = dist.get_rank(group)
        self.world = dist.get_world_size(group)
        self.shapes = [tuple(s) for s in shapes]
        self.owner, self.load = layerwise_assign(self.shapes, self.world, policy)
        self.mine = [i for i, o in enumerate(self.owner) if o == self.rank]
        self.of_rank = [[i for i, o in enumerate(self.owner) if o == r] for r in range(self.world)]
        self.opt = make_optimizer([self.shapes[i] for i in self.mine]) if self.mine else None

    def step(self, params, grads):
        """One step: local step of the owned matrices, then the all-gather of updated weights.
        ``params`` (updated in place on every rank) and ``grads`` hold every matrix."""
        if self.opt is not None:
            self.opt.step([params[i] for i in self.mine], [grads[i] for i in self.mine])
        self.exchange(params)

    def exchange(self, params):
        """Each owning rank broadcasts its matrices, packed end to end; the others unpack."""
        for r, idx in enumerate(self.of_rank):
            if not idx:
                continue
            if r == self.rank:
                buf = torch.cat([params[i].reshape(-1) for i in idx])
            else:
                n = sum(params[i].numel() for i in idx)
                buf = torch.empty(n, dtype=params[idx[0]].dtype, device=params[idx[0]].device)
            dist.broadcast(buf, src=dist.get_global_rank(self.group, r) if self.group is not None else r,
                           group=self.group)
            if r != self.rank:
                off = 0
                for i in idx:
                    k = params[i].numel()
                    params[i].copy_(buf[off:off + k].view_as(params[i]))
                    off += k

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
