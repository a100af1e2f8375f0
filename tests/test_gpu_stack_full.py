"""The 24-layer MoE stack at full size, in the configuration bench.py times: all 4706 matrices
(200 GB of optimizer state, the fp32 parameters and one set of gradients resident) stepped by one
handle whose workspace is cut into pipelined waves. Matrices from the first, a middle and the last
waves, of every shape class, are teacher-forced against the oracle on the first two steps (the
matrices are independent, so checking a sample loses nothing for the ones checked)."""
import gc

import pytest
import torch

from paper_2607_20548_gb300 import soap as S
from paper_2607_20548_gb300.workloads import make_stream

from tests.parity_tools import TeacherForcedCheck, oracle_hparams

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

PER_LAYER = 4 + 192  # Wq, Wk, Wv, Wo, then 64 gate, 64 up, 64 down experts
SAMPLE = [
    0,                                  # layer 0 Wq (2048 x 2048)
    4,                                  # layer 0 gate of expert 0 (2048 x 768)
    4 + 128,                            # layer 0 down of expert 0 (768 x 2048)
    12 * PER_LAYER + 4 + 63,            # layer 12 gate of expert 63
    23 * PER_LAYER + 3,                 # layer 23 Wo
    23 * PER_LAYER + 4 + 64 + 31,       # layer 23 up of expert 31
    24 * PER_LAYER,                     # embedding (2048 x 32768, left side only)
    24 * PER_LAYER + 1,                 # LM head
]


def _flat(stream, tensors):
    out = [None] * len(stream.specs)
    for (spec, idx), t in zip(stream.groups, tensors):
        for b, j in enumerate(idx):
            out[j] = t[b]
    return out


def test_moe_stack_full_size(cuda):
    gc.collect()
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    assert free >= 275e9, f"the full stack needs about 270 GB of free device memory, {free / 1e9:.0f} GB free"
    hp = S.default_hparams()
    stream = make_stream("moe_stack_24x_h2048", seed=0, device=cuda)
    assert len(stream.specs) == 4706
    shapes = [(s.rows, s.cols, s.left, s.right) for s in stream.specs]
    Wg = [w.contiguous() for w in stream.weights()]
    Gg = stream.grads(1)
    W, G = _flat(stream, Wg), _flat(stream, Gg)
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    opt = S.SoapOptimizer(shapes, hp)
    info = opt.plan_info()
    print(f"\nplan: {info}")
    assert info["waves"] > 1 and info["pipelined"]
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    for t in (1, 2):
        if t > 1:
            stream.grads(t, out=Gg)  # step t's gradients, into the same buffers
        for i in SAMPLE:
            chk.before(i, W[i], G[i])
        opt.step(W, G)
        torch.cuda.synchronize()
        assert opt.status() == 0, opt.last_error()
        for i in SAMPLE:
            chk.after(i, W[i])
    print("\n" + chk.report())
    chk.assert_ok()
    opt.destroy()
