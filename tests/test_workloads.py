"""The seeded synthetic workloads: shapes of the paper's layers and the gradient recipe."""
import math

import numpy as np
import torch

from paper_2607_20548_gb300.workloads import WORKLOADS, expert_scales, make_stream


def test_workload_shapes():
    counts = {name: len(specs) for name, (specs, _) in WORKLOADS.items()}
    assert counts == {"single_256x512": 1, "dense_block_h2048_ffn8192": 7, "moe_layer_64x768_h2048": 193,
                      "dense_8192_ffn28672": 5, "moe_stack_24x_h2048": 4706}
    big = WORKLOADS["dense_8192_ffn28672"][0]
    assert [(s.rows, s.cols, s.left, s.right) for s in big[2:]] == [
        (8192, 28672, True, False), (8192, 28672, True, False), (28672, 8192, False, True)]
    head = WORKLOADS["moe_stack_24x_h2048"][0][-1]
    assert (head.rows, head.cols, head.left, head.right) == (2048, 32768, True, False)


def test_generator_recipe_and_determinism():
    s = make_stream("single_256x512", seed=0)
    A = s._A[0][0].double()
    assert abs(A.norm().item() - 1.0) < 1e-5                    # ||A||_F = ||s||_2 = 1
    sv = torch.linalg.svdvals(A)
    i = torch.arange(1, 257, dtype=torch.float64)
    want = i.pow(-1.5) / i.pow(-1.5).norm()
    assert torch.allclose(sv, want, atol=1e-5)                  # power-law spectrum i^-1.5
    G1, G1b = s.grads(1)[0][0], make_stream("single_256x512", seed=0).grads(1)[0][0]
    assert torch.equal(G1, G1b)
    noise = (G1.double() - A) / 0.3
    assert abs(noise.var().item() - 1 / 512) < 1e-4             # N(0, 1/cols)
    assert not torch.equal(G1, s.grads(2)[0][0])
    W = s.weights()[0][0]
    assert abs(W.std().item() - 0.02) < 1e-3


def test_expert_scales_log_uniform():
    specs, _ = WORKLOADS["moe_layer_64x768_h2048"]
    c = expert_scales(specs, "moe_layer_64x768_h2048", 0)
    assert c[192] == 1.0                                        # router unscaled
    ce = np.array(c[:64])
    assert (ce >= 1e-2).all() and (ce <= 1).all()
    assert c[5] == c[64 + 5] == c[128 + 5]                      # gate, up and down share the expert's scale
    assert abs(np.mean(np.log(ce)) - 0.5 * math.log(1e-2)) < 0.8
