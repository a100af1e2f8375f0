"""Layer-wise ownership (section 6): the planner (C ABI, host-only) and the all-gather of the
updated weights across ranks, with world_size 2 on gloo (CPU; no GPU involved)."""
import ctypes
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_20548_gb300 import soap as S
from paper_2607_20548_gb300.layerwise import LayerwiseOptimizer, plan_buckets
from paper_2607_20548_gb300.workloads import WORKLOADS

BLOCK = [(s.rows, s.cols, int(s.left), int(s.right)) for s in WORKLOADS["dense_block_h2048_ffn8192"][0]]


def test_paper_assignment_is_size_sorted_round_robin():
    """Policy 0: sorted by rows * cols (largest first, ties by index) and dealt round-robin."""
    shapes = [(4, 4), (8, 8), (2, 2), (8, 8), (6, 6)]
    owner, _ = S.layerwise_assign(shapes, 2, 0)
    # order: (8,8)#1, (8,8)#3, (6,6)#4, (4,4)#0, (2,2)#2 -> ranks 0, 1, 0, 1, 0
    assert owner == [1, 0, 0, 1, 0]
    owner3, _ = S.layerwise_assign(shapes, 3, 0)
    assert owner3 == [0, 0, 1, 1, 2]


def test_lpt_assignment_balances_cost_and_covers_every_matrix():
    """Policy 1 gives every matrix one owner and no rank more than the largest single matrix's
    cost above the lightest rank (the LPT bound); the loads add up to the whole step."""
    for world in (1, 2, 3, 4, 8):
        owner, load = S.layerwise_assign(BLOCK, world, 1)
        assert len(owner) == len(BLOCK) and all(0 <= o < world for o in owner)
        _, total = S.layerwise_assign(BLOCK, 1, 1)
        assert abs(sum(load) - total[0]) <= 1e-9 * total[0]
        _, single = zip(*[S.layerwise_assign([s], 1, 1) for s in BLOCK])
        assert max(load) - min(load) <= max(x[0] for x in single) * (1 + 1e-12)


def test_planner_rejects_bad_arguments():
    lib = S.load_library()
    arr = (S.soap_shape * 1)(S.soap_shape(4, 4, 1, 1))
    own = (ctypes.c_int32 * 1)()
    assert lib.soap_layerwise_assign(arr, 1, 0, 0, own, None) == 1
    assert lib.soap_layerwise_assign(arr, 1, 2, 5, own, None) == 1
    bad = (S.soap_shape * 1)(S.soap_shape(0, 4, 1, 1))
    assert lib.soap_layerwise_assign(bad, 1, 2, 0, own, None) == 1


def test_buckets_are_consecutive_and_bounded():
    shapes = [(4, 4), (4, 4), (8, 8), (2, 2), (16, 16), (2, 2), (2, 2)]   # 64, 64, 256, 16, 1024, 16, 16 B
    assert plan_buckets(shapes) == [list(range(7))]
    assert plan_buckets([]) == []
    b = plan_buckets(shapes, bucket_bytes=256)
    # in order, nothing skipped or repeated; a bucket only exceeds the bound when it holds one matrix
    assert [i for bkt in b for i in bkt] == list(range(7))
    assert b == [[0, 1], [2], [3], [4], [5, 6]]
    for bkt in b:
        assert len(bkt) == 1 or sum(shapes[i][0] * shapes[i][1] * 4 for i in bkt) <= 256
    assert plan_buckets(shapes, bucket_bytes=1) == [[i] for i in range(7)]


class _Descent:
    """A stand-in local optimizer for the exchange test: W <- W - 0.5 G on the owned matrices."""

    def __init__(self, shapes):
        self.shapes = shapes

    def step(self, params, grads):
        for p, g in zip(params, grads):
            p.sub_(0.5 * g)


def _worker(rank, world, port, shapes, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        g = torch.Generator().manual_seed(0)
        W = [torch.randn(r, c, generator=g) for r, c in shapes]
        W0 = [w.clone() for w in W]
        G = [torch.randn(r, c, generator=g) for r, c in shapes]
        opt = LayerwiseOptimizer(shapes, _Descent)
        opt.step(W, G)
        for w, w0, gg in zip(W, W0, G):
            # every matrix was stepped exactly once, by its owner, and every rank holds the result
            assert torch.equal(w, w0 - 0.5 * gg)
        out[rank] = opt.mine
    finally:
        dist.destroy_process_group()


def test_exchange_world_size_2_gloo():
    shapes = [(12, 20), (20, 12), (8, 8), (16, 4), (4, 16), (12, 20)]
    with socket.socket() as sock:
        sock.bind(("127.0.0.1", 0))
        port = sock.getsockname()[1]
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(2, port, shapes, out), nprocs=2, join=True)
    owned = sorted(out[0] + out[1])
    assert owned == list(range(len(shapes)))


def _overlap_worker(rank, world, port, shapes, policy, bucket_bytes, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        g = torch.Generator().manual_seed(1)
        W = [torch.randn(r, c, generator=g) for r, c in shapes]
        W0 = [w.clone() for w in W]
        G = [torch.randn(r, c, generator=g) for r, c in shapes]
        opt = LayerwiseOptimizer(shapes, _Descent, policy=policy, bucket_bytes=bucket_bytes)
        assert len(opt.buckets) > 1
        pending = opt.step(W, G, overlap=True)
        for b, bkt in enumerate(opt.buckets):
            for i in bkt:
                # a matrix another rank owns keeps its old value until its bucket is waited for
                want_before = W0[i] - 0.5 * G[i] if opt.owner[i] == rank else W0[i]
                assert torch.equal(W[i], want_before)
            pending.wait(b)
            for i in bkt:
                assert torch.equal(W[i], W0[i] - 0.5 * G[i])
        pending.wait_all()
        # a second step through the blocking path agrees with the same rule
        W1 = [w.clone() for w in W]
        opt.step(W, G)
        for w, w1, gg in zip(W, W1, G):
            assert torch.equal(w, w1 - 0.5 * gg)
        out[rank] = opt.mine
    finally:
        dist.destroy_process_group()


def test_bucketed_overlapped_exchange_world_size_2_gloo():
    shapes = [(12, 20), (20, 12), (8, 8), (16, 4), (4, 16), (12, 20), (30, 2), (2, 30)]
    for policy in (0, 1):
        with socket.socket() as sock:
            sock.bind(("127.0.0.1", 0))
            port = sock.getsockname()[1]
        mgr = mp.Manager()
        out = mgr.dict()
        mp.spawn(_overlap_worker, args=(2, port, shapes, policy, 1000, out), nprocs=2, join=True)
        assert sorted(out[0] + out[1]) == list(range(len(shapes)))


def _departing_worker(rank, world, port, shapes, out):
    """Rank 1 leaves between steps (no collective of its own in flight); rank 0's next exchange
    must end with an error from the process group, not wait forever."""
    import datetime
    import time
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=10))
    g = torch.Generator().manual_seed(2)
    W = [torch.randn(r, c, generator=g) for r, c in shapes]
    G = [torch.randn(r, c, generator=g) for r, c in shapes]
    opt = LayerwiseOptimizer(shapes, _Descent)
    opt.step(W, G)                       # one good step on both ranks
    if rank == 1:
        out[rank] = "left"
        os._exit(0)                      # gone without a goodbye
    t0 = time.monotonic()
    try:
        opt.step(W, G)
        out[rank] = "no error"
    except Exception as e:  # noqa: BLE001 - any process-group error is the expected outcome
        out[rank] = f"raised after {time.monotonic() - t0:.1f} s: {type(e).__name__}"
    os._exit(0)


def test_exchange_with_a_departed_rank_raises_instead_of_hanging():
    shapes = [(12, 20), (20, 12), (8, 8), (16, 4)]
    with socket.socket() as sock:
        sock.bind(("127.0.0.1", 0))
        port = sock.getsockname()[1]
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=_departing_worker, args=(r, 2, port, shapes, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()                         # only the processes this test started
        p.join()
    assert not alive, "a rank hung in the exchange"
    assert out.get(1) == "left"
    assert str(out.get(0, "")).startswith("raised after"), out.get(0)


def test_lpt_cost_model_is_the_step_flop_model():
    """Policy 1 balances the literal Alg. 1 FLOP count (the bench's model) plus 10 FLOP per
    weight element for the elementwise work; identity sides cost nothing of their own."""
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    for shape in [(2048, 2048, 1, 1), (2048, 8192, 1, 1), (8192, 28672, 1, 0), (28672, 8192, 0, 1), (768, 2048, 1, 1)]:
        _, load = S.layerwise_assign([shape], 1, 1)
        want = bench.model_flops(*shape) + 10.0 * shape[0] * shape[1]
        assert abs(load[0] - want) <= 1e-9 * want, (shape, load[0], want)
