"""Multi-rank path on the CPU: two gloo ranks refine disjoint row shards and
gather the result, which must equal the single-process refinement (rows are
independent, Sec. 3.3).  The oracle stands in for the per-rank GPU call."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_38599_gb300.shard import row_range


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import Options, prepare_hessian, refine_layer
        from paper_2609_38599_gb300.shard import gather_rows
        from synth import small_layer
        lay = small_layer(128, 37, 64, 3, seed=31)
        a, b = row_range(lay.dout, rank, world)
        prep = prepare_hessian(lay.H, lay.g)
        res = refine_layer(prep, lay.W[a:b], lay.S0[a:b], lay.Q0[a:b], lay.Z[a:b], 3,
                           Options(max_iters=3))
        S = gather_rows(torch.as_tensor(res.S), lay.dout)
        Q = gather_rows(torch.as_tensor(res.Q), lay.dout)
        t = torch.tensor([float(rank + 1)])
        dist.all_reduce(t, op=dist.ReduceOp.MAX)      # max-over-ranks timing reduction
        if rank == 0:
            q.put((S.numpy(), Q.numpy(), float(t.item())))
    finally:
        dist.destroy_process_group()


def test_row_range_partitions_rows():
    for dout in (1, 7, 37, 4096, 14336):
        for world in (1, 2, 3, 8):
            spans = [row_range(dout, r, world) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == dout
            assert all(spans[r][1] == spans[r + 1][0] for r in range(world - 1))
            sizes = [b - a for a, b in spans]
            assert max(sizes) - min(sizes) <= 1


def test_two_gloo_ranks_match_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    S, Q, tmax = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    from oracle import Options, prepare_hessian, refine_layer
    from synth import small_layer
    lay = small_layer(128, 37, 64, 3, seed=31)
    ref = refine_layer(prepare_hessian(lay.H, lay.g), lay.W, lay.S0, lay.Q0, lay.Z, 3,
                       Options(max_iters=3))
    assert np.array_equal(Q, ref.Q)
    np.testing.assert_allclose(S, ref.S, rtol=0, atol=0)
    assert tmax == 2.0


def _hessian_worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import accumulate_hessian
        from paper_2609_38599_gb300.shard import allreduce_hessian, token_range
        from synth import integer_activations_np
        X = integer_activations_np(1001, 24, amax=8, seed=5)
        a, b = token_range(X.shape[0], rank, world)
        H = torch.as_tensor(accumulate_hessian(X[a:b]))   # this rank's partial X^T X
        allreduce_hessian(H)
        if rank == 0:
            q.put(H.numpy())
    finally:
        dist.destroy_process_group()


def test_token_sharded_hessian_equals_single_process():
    """Three gloo ranks accumulate disjoint token ranges and sum the partial
    Hessians with one all-reduce; on integer activations the sum is exact,
    so it must equal the single-process product bit for bit.  The oracle
    stands in for each rank's GPU call."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_hessian_worker, args=(r, 3, port, q)) for r in range(3)]
    for p in procs:
        p.start()
    H = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    from oracle import accumulate_hessian
    from synth import integer_activations_np
    X = integer_activations_np(1001, 24, amax=8, seed=5)
    np.testing.assert_array_equal(H, accumulate_hessian(X))


def test_rank_layer_instances():
    """Under torchrun each rank refines its own instance of the named layer
    (independent problems, weak scaling): offset 0 is the named layer itself,
    another offset draws different data of the same shape."""
    from synth import config_layer
    a = config_layer("tiny_256x256_g64_w3", device="cpu")
    b = config_layer("tiny_256x256_g64_w3", device="cpu", seed_offset=0)
    c = config_layer("tiny_256x256_g64_w3", device="cpu", seed_offset=1)
    assert torch.equal(a.W, b.W) and torch.equal(a.H, b.H) and torch.equal(a.Q0, b.Q0)
    assert a.W.shape == c.W.shape and a.H.shape == c.H.shape
    assert not torch.equal(a.W, c.W) and not torch.equal(a.H, c.H)
