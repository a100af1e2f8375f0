"""Seeded synthetic workloads for the SOAP step: shapes, weights and gradients.

This module only draws inputs; it holds none of the optimizer's arithmetic, and both
the CUDA path's tests/bench and the oracle consume what it produces.

Shapes follow the paper's models (section 5: a dense transformer block with hidden
2048 and SwiGLU FFN 8192; the Qwen3-30B-A3B-like fine-grained MoE with hidden 2048 and
expert width 768; an 8192-wide dense layer). The gradient of every matrix is
rank-structured plus noise:

    G_t = c * (A + 0.3 * N_t),   A = U diag(s) V^T,  s_i = i^-1.5 / ||(i^-1.5)||_2,

with U (rows x k), V (cols x k) random orthonormal (QR of a Gaussian), k = min(rows,
cols, 1024) (the spectrum beyond i = 1024 lies far below the noise: s_1024 / s_1 = 3e-5, so
the cap only keeps the host QR of the 28672-wide matrices cheap), N_t i.i.d. N(0, 1/cols) drawn afresh every step, W_0 ~ N(0, 0.02^2), and c = 1
except for MoE experts, whose c is drawn once per expert, log-uniform in [1e-2, 1],
to mimic uneven token routing.

All tensors are float32. U, V (and so A) are drawn on the host; W_0 and the per-step
noise are drawn with torch on the requested device; the oracle gets host copies of
exactly the same values.
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
        self._A = []
        self._c = []
        for gi, (s, idx) in enumerate(self.groups):
            # U, V and A are drawn on the host (the same values whatever the device), then moved
            k = min(s.rows, s.cols, 1024)
            g = torch.Generator().manual_seed(_seed(seed, gi, 1))
            B = len(idx)
            U = torch.linalg.qr(torch.randn(B, s.rows, k, generator=g))[0]
            V = torch.linalg.qr(torch.randn(B, s.cols, k, generator=g))[0]
            i = torch.arange(1, k + 1, dtype=torch.float64)
            sv = i.pow(-1.5)
            sv = (sv / sv.norm()).to(torch.float32)
            A = torch.matmul(U * sv, V.transpose(1, 2))
            self._A.append(A.contiguous().to(self.device))
            self._c.append(torch.tensor([self.scales[j] for j in idx], dtype=torch.float32,
                                        device=self.device).view(B, 1, 1))

    def weights(self):
        """W_0 ~ N(0, 0.02^2), one [batch, rows, cols] tensor per group."""
        out = []
        for gi, (s, idx) in enumerate(self.groups):
            g = torch.Generator(device=self.device).manual_seed(_seed(self.seed, gi, 2))
            out.append(0.02 * torch.randn(len(idx), s.rows, s.cols, generator=g, device=self.device))
        return out

    def grads(self, step: int):
        """G_t for step ``step`` (1-based), one [batch, rows, cols] tensor per group."""
        out = []
        for gi, (s, idx) in enumerate(self.groups):
            g = torch.Generator(device=self.device).manual_seed(_seed(self.seed, gi, 3, step))
            N = torch.randn(len(idx), s.rows, s.cols, generator=g, device=self.device)
            N.mul_(0.3 / math.sqrt(s.cols)).add_(self._A[gi]).mul_(self._c[gi])
            out.append(N)
        return out


def make_stream(name: str, seed: int = 0, device="cpu", specs=None):
    """GradientStream for a named workload (optionally restricted to ``specs``)."""
    all_specs, _ = WORKLOADS[name]
    scales = expert_scales(all_specs, name, seed)
    if specs is not None:
        keep = [j for j in specs]
        return GradientStream([all_specs[j] for j in keep], seed, [scales[j] for j in keep],
                              device, name)
    return GradientStream(all_specs, seed, scales, device, name)
