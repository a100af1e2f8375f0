"""Seeded synthetic workloads for the SOAP step: shapes, weights and gradients.

This module only draws inputs; it holds none of the optimizer's arithmetic, and both
the CUDA path's tests/bench and the oracle consume what it produces.

Shapes follow the paper's models (section 5: a dense transformer block with hidden
2048 and SwiGLU FFN 8192; the Qwen3-30B-A3B-like fine-grained MoE with hidden 2048 and
expert width 768; an 8192-wide dense layer). The gradient of every matrix is
rank-structured plus noise:

    G_t = c * (A + 0.3 * N_t),   A = U diag(s) V^T,  s_i = i^-1.5 / ||(i^-1.5)||_2,

with U (rows x k), V (cols x k) random orthonormal (QR of a Gaussian), k = min(rows, cols),
N_t i.i.d. N(0, 1/cols) drawn afresh every step, W_0 ~ N(0, 0.02^2), and c = 1 except for MoE
experts, whose c is drawn once per expert, log-uniform in [1e-2, 1], to mimic uneven token
routing.

All tensors are float32 and drawn on the stream's device (U and V by a QR of a Gaussian there);
the oracle gets host copies of exactly the same values. A shape group of more than
SHARED_BASES matrices (the 24-layer stack has thousands of experts of one shape) draws
SHARED_BASES Haar-random bases per side and gives each matrix one of them with its columns
permuted and their signs flipped at random (still exactly orthonormal, with the same
power-law spectrum); such a group keeps no A and forms it chunk by chunk when drawing G.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch


@dataclass(frozen=True)
class MatrixSpec:
    """One weight matrix: rows x cols, and which sides carry a preconditioner."""
    rows: int
    cols: int
    left: bool = True
    right: bool = True


def _block(h=2048, ffn=8192):
    return ([MatrixSpec(h, h)] * 4 + [MatrixSpec(h, ffn)] * 2 + [MatrixSpec(ffn, h)])


def _moe(h=2048, e=768, experts=64, router=True):
    s = [MatrixSpec(h, e)] * (2 * experts) + [MatrixSpec(e, h)] * experts
    if router:
        s.append(MatrixSpec(h, experts))
    return s


# name -> (matrix list, steps, expert-scale groups)
WORKLOADS = {
    # one 256x512 weight, both sides preconditioned, 20 steps
    "single_256x512": ([MatrixSpec(256, 512)], 20),
    # one dense transformer block: Wq/Wk/Wv/Wo 2048^2, W_gate/W_up 2048x8192, W_down 8192x2048
    "dense_block_h2048_ffn8192": (_block(), 20),
    # one fine-grained MoE layer: 64 experts (2048x768 gate/up, 768x2048 down) + router 2048x64
    "moe_layer_64x768_h2048": (_moe(), 20),
    # large dense layer; the 28672 side is not preconditioned
    "dense_8192_ffn28672": ([MatrixSpec(8192, 8192)] * 2 + [MatrixSpec(8192, 28672, True, False)] * 2
                            + [MatrixSpec(28672, 8192, False, True)], 10),
    # 24-layer MoE stack + embedding and LM head (32768 side not preconditioned)
    "moe_stack_24x_h2048": ([m for _ in range(24) for m in ([MatrixSpec(2048, 2048)] * 4 + _moe(router=False))]
                            + [MatrixSpec(2048, 32768, True, False)] * 2, 10),
}


def expert_scales(specs, name: str, seed: int):
    """Per-matrix gradient scale c: log-uniform [1e-2, 1] per MoE expert, 1 otherwise."""
    c = [1.0] * len(specs)
    if name not in ("moe_layer_64x768_h2048", "moe_stack_24x_h2048"):
        return c
    g = torch.Generator().manual_seed(seed * 7919 + 17)
    per_layer = 192 if name == "moe_stack_24x_h2048" else None
    if per_layer is None:
        u = torch.rand(64, generator=g, dtype=torch.float64)
        ce = torch.exp(math.log(1e-2) + u * (0.0 - math.log(1e-2)))
        for j in range(64):  # gate, up and down of expert j share its scale
            c[j] = c[64 + j] = c[128 + j] = float(ce[j])
        return c
    stride = 4 + 192
    for layer in range(24):
        u = torch.rand(64, generator=g, dtype=torch.float64)
        ce = torch.exp(math.log(1e-2) + u * (0.0 - math.log(1e-2)))
        base = layer * stride + 4
        for j in range(64):
            c[base + j] = c[base + 64 + j] = c[base + 128 + j] = float(ce[j])
    return c


def _seed(*parts: int) -> int:
    h = 0x9E3779B97F4A7C15
    for p in parts:
        h = (h ^ (p + 0x632BE59BD9B4E019 + (h << 6) + (h >> 2))) & 0xFFFFFFFFFFFFFFFF
    return h & 0x7FFFFFFFFFFFFFFF


SHARED_BASES = 64
_CHUNK_ELEMS = 1 << 27  # matrices per chunk: about this many elements (512 MB) at a time


class GradientStream:
    """Draws W_0 and G_t for a list of matrices, grouped into same-shape batches.

    ``groups`` is a list of (spec, [matrix indices]); tensors are [batch, rows, cols].
    """

    def __init__(self, specs, seed: int = 0, scales=None, device="cpu", name: str = ""):
        self.specs = list(specs)
        self.seed = seed
        self.device = torch.device(device)
        self.scales = list(scales) if scales is not None else [1.0] * len(self.specs)
        order = {}
        for j, s in enumerate(self.specs):
            order.setdefault((s.rows, s.cols), []).append(j)
        self.groups = [(self.specs[idx[0]], idx) for idx in order.values()]
        self._A = []      # per group: A [B, rows, cols], or None if formed per chunk
        self._bases = []  # per group (chunked only): U, V bases and each matrix's pick
        self._c = []
        for gi, (s, idx) in enumerate(self.groups):
            k = min(s.rows, s.cols)
            B = len(idx)
            g = torch.Generator(device=self.device).manual_seed(_seed(seed, gi, 1))
            nb = min(B, SHARED_BASES)
            U = torch.linalg.qr(torch.randn(nb, s.rows, k, generator=g, device=self.device))[0]
            V = torch.linalg.qr(torch.randn(nb, s.cols, k, generator=g, device=self.device))[0]
            i = torch.arange(1, k + 1, dtype=torch.float64)
            sv = i.pow(-1.5)
            sv = (sv / sv.norm()).to(torch.float32).to(self.device)
            self._c.append(torch.tensor([self.scales[j] for j in idx], dtype=torch.float32,
                                        device=self.device).view(B, 1, 1))
            if nb == B:
                self._A.append(torch.matmul(U * sv, V.transpose(1, 2)).contiguous())
                self._bases.append(None)
                continue
            # each matrix: one of the nb bases per side, columns permuted, signs flipped
            pick = torch.randint(0, nb, (B,), generator=g, device=self.device)
            perm_u = torch.argsort(torch.rand(B, k, generator=g, device=self.device), dim=1)
            perm_v = torch.argsort(torch.rand(B, k, generator=g, device=self.device), dim=1)
            sgn_u = torch.randint(0, 2, (B, k), generator=g, device=self.device).float().mul_(2).sub_(1)
            sgn_v = torch.randint(0, 2, (B, k), generator=g, device=self.device).float().mul_(2).sub_(1)
            self._A.append(None)
            self._bases.append((U, V, sv, pick, perm_u, perm_v, sgn_u, sgn_v))

    def _A_chunk(self, gi, b0, b1):
        A = self._A[gi]
        if A is not None:
            return A[b0:b1]
        U, V, sv, pick, pu, pv, su, sv_sign = self._bases[gi]
        Uc = torch.gather(U[pick[b0:b1]], 2, pu[b0:b1, None, :].expand(-1, U.shape[1], -1)) * su[b0:b1, None, :]
        Vc = torch.gather(V[pick[b0:b1]], 2, pv[b0:b1, None, :].expand(-1, V.shape[1], -1)) * sv_sign[b0:b1, None, :]
        return torch.matmul(Uc * sv, Vc.transpose(1, 2))

    def weights(self):
        """W_0 ~ N(0, 0.02^2), one [batch, rows, cols] tensor per group."""
        out = []
        for gi, (s, idx) in enumerate(self.groups):
            g = torch.Generator(device=self.device).manual_seed(_seed(self.seed, gi, 2))
            out.append(torch.randn(len(idx), s.rows, s.cols, generator=g, device=self.device).mul_(0.02))
        return out

    def grads(self, step: int, out=None):
        """G_t for step ``step`` (1-based), one [batch, rows, cols] tensor per group (written into
        ``out``, a list of such tensors, if given)."""
        res = []
        for gi, (s, idx) in enumerate(self.groups):
            B = len(idx)
            dst = out[gi] if out is not None else torch.empty(B, s.rows, s.cols, device=self.device)
            if self._A[gi] is not None and B * s.rows * s.cols <= _CHUNK_ELEMS:
                g = torch.Generator(device=self.device).manual_seed(_seed(self.seed, gi, 3, step))
                torch.randn(B, s.rows, s.cols, generator=g, device=self.device, out=dst)
                dst.mul_(0.3 / math.sqrt(s.cols)).add_(self._A[gi]).mul_(self._c[gi])
            else:
                per = max(1, _CHUNK_ELEMS // (s.rows * s.cols))
                for ci, b0 in enumerate(range(0, B, per)):
                    b1 = min(B, b0 + per)
                    g = torch.Generator(device=self.device).manual_seed(_seed(self.seed, gi, 3, step, ci))
                    d = dst[b0:b1]
                    torch.randn(b1 - b0, s.rows, s.cols, generator=g, device=self.device, out=d)
                    d.mul_(0.3 / math.sqrt(s.cols)).add_(self._A_chunk(gi, b0, b1)).mul_(self._c[gi][b0:b1])
            res.append(dst)
        return res


def make_stream(name: str, seed: int = 0, device="cpu", specs=None):
    """GradientStream for a named workload (optionally restricted to ``specs``)."""
    all_specs, _ = WORKLOADS[name]
    scales = expert_scales(all_specs, name, seed)
    if specs is not None:
        keep = [j for j in specs]
        return GradientStream([all_specs[j] for j in keep], seed, [scales[j] for j in keep],
                              device, name)
    return GradientStream(all_specs, seed, scales, device, name)
