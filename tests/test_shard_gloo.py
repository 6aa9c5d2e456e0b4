"""Data-parallel sharding of the BGPO path over sequences, on CPU ranks (gloo).

Every (sequence, MC sample) unit is independent once A and l_old are given
(Linearity, Sec. 3), so the path shards by sequences with no collective in the
data path; the dW sum over ranks belongs to the optimiser step. Two gloo ranks
each run the fp64 oracle on their half of a batch (b_offset = first global
sequence index), sum dW with the bench's data-parallel exchange
(paper_2510_11683_gb300.dp.allreduce_dw) and gather dX and l; rank 0 compares
with the single-process run of the whole batch. The bench's rank aggregation (slowest
rank's time, tokens of all ranks) is checked on the same ranks.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import bgpo_oracle as O
from paper_2510_11683_gb300.dp import allreduce_dw
from synth import CONFIGS, make_inputs
from tests.harness import oracle_advantages, to64

WORLD = 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _workload():
    return CONFIGS["tiny"].with_(B=4, G=2, R=20, n_t=3, H=64, V=96)


def _rank_main(rank, port, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        import bench
        wl = _workload()
        inp = make_inputs(wl)                      # the whole batch (same seed on every rank)
        nb = wl.B // WORLD
        b0 = rank * nb
        X, W, Y = to64(inp["X"])[b0:b0 + nb], to64(inp["W"]), to64(inp["Y"])[b0:b0 + nb]
        A = oracle_advantages(wl, inp)[b0:b0 + nb]
        eps = to64(inp["eps"])[b0:b0 + nb]
        ts, masks = O.sample_masks(wl.seed, nb, wl.R, wl.n_t, wl.t_mode, b_offset=b0)
        ell_old = O.elbo_all(X, W, Y, wl.P, ts, masks) + eps
        out = O.bgpo_step(X, W, Y, wl.P, A, ell_old, ts, masks, 1.0 / wl.G)
        dW = torch.from_numpy(out["dW"])
        allreduce_dw(dW)                           # the optimiser step's gradient sum
        dX = [torch.zeros_like(torch.from_numpy(out["dX"])) for _ in range(WORLD)]
        dist.all_gather(dX, torch.from_numpy(out["dX"]))
        ell = [torch.zeros_like(torch.from_numpy(out["ell"])) for _ in range(WORLD)]
        dist.all_gather(ell, torch.from_numpy(out["ell"]))
        ms, tokens = bench.aggregate_ranks(10.0 + rank, 100 * (rank + 1))
        if rank == 0:
            np.savez(os.path.join(out_dir, "shard.npz"), dW=dW.numpy(),
                     dX=torch.cat(dX).numpy(), ell=torch.cat(ell).numpy(),
                     masks=masks, ms=ms, tokens=tokens)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_shards_reproduce_the_full_batch(tmp_path):
    mp.spawn(_rank_main, args=(_free_port(), str(tmp_path)), nprocs=WORLD, join=True)
    got = np.load(os.path.join(str(tmp_path), "shard.npz"))
    wl = _workload()
    inp = make_inputs(wl)
    X, W, Y = to64(inp["X"]), to64(inp["W"]), to64(inp["Y"])
    A = oracle_advantages(wl, inp)
    ts, masks = O.sample_masks(wl.seed, wl.B, wl.R, wl.n_t, wl.t_mode)
    ell_old = O.elbo_all(X, W, Y, wl.P, ts, masks) + to64(inp["eps"])
    ref = O.bgpo_step(X, W, Y, wl.P, A, ell_old, ts, masks, 1.0 / wl.G)
    # draws of rank 0's shard equal the whole batch's draws for those sequences
    assert np.array_equal(got["masks"], masks[:, : wl.B // WORLD])
    assert np.allclose(got["ell"], ref["ell"], rtol=1e-13, atol=0)
    assert np.allclose(got["dX"], ref["dX"], rtol=1e-12, atol=1e-15)
    assert np.allclose(got["dW"], ref["dW"], rtol=1e-12, atol=1e-14)
    # bench aggregation: the slowest rank's time, the tokens of every rank
    assert float(got["ms"]) == 11.0 and int(got["tokens"]) == 300


def test_shard_of_assigns_disjoint_global_sequences():
    import bench
    wl = CONFIGS["llada8b_r512_onpolicy"]
    offsets = [bench.shard_of(wl, r, 8)[1] for r in range(8)]
    assert offsets == [r * wl.B for r in range(8)]
    assert bench.shard_of(wl, 0, 1) == (wl, 0)
    seeds = {bench.shard_of(wl, r, 8)[0].seed for r in range(8)}
    assert len(seeds) == 8


def _lost_rank_main(rank, port, out_dir):
    # rank 1 leaves after its shard's work and before the dW sum; rank 0 must
    # learn of it from the failed collective (or the group's short timeout)
    # instead of hanging, and stop between steps with nothing in flight
    import datetime
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD,
                            timeout=datetime.timedelta(seconds=20))
    wl = _workload()
    inp = make_inputs(wl)
    nb = wl.B // WORLD
    b0 = rank * nb
    X, W, Y = to64(inp["X"])[b0:b0 + nb], to64(inp["W"]), to64(inp["Y"])[b0:b0 + nb]
    ts, masks = O.sample_masks(wl.seed, nb, wl.R, wl.n_t, wl.t_mode, b_offset=b0)
    ell = O.elbo_all(X, W, Y, wl.P, ts, masks)
    out = O.bgpo_step(X, W, Y, wl.P, oracle_advantages(wl, inp)[b0:b0 + nb], ell, ts, masks,
                      1.0 / wl.G)
    if rank == 1:
        return                                     # leaves without joining the sum
    dW = torch.from_numpy(out["dW"])
    try:
        allreduce_dw(dW)
        result = "completed"
    except Exception as e:                         # noqa: BLE001 - any collective failure
        result = "detected: " + type(e).__name__
    with open(os.path.join(out_dir, "rank0.txt"), "w") as f:
        f.write(result)


def test_lost_rank_is_detected_by_the_survivor(tmp_path):
    import time
    t0 = time.time()
    mp.spawn(_lost_rank_main, args=(_free_port(), str(tmp_path)), nprocs=WORLD, join=True)
    with open(os.path.join(str(tmp_path), "rank0.txt")) as f:
        result = f.read()
    assert result.startswith("detected"), result
    assert time.time() - t0 < 120


def test_single_process_exchange_is_the_identity():
    # without an initialised process group there is nothing to sum over
    dW = torch.arange(12, dtype=torch.float32).reshape(3, 4)
    ref = dW.clone()
    assert allreduce_dw(dW) is dW and torch.equal(dW, ref)
