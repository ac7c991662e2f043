"""The benchmark's multi-GPU logic on CPU: two gloo ranks on 127.0.0.1.

Requests are independent, so each rank verifies its own batch (weak scaling)
and nothing crosses ranks on the data path; the only collectives are the
timing barrier and the max over ranks. These tests run that host logic with
world_size 2 and check the per-rank workloads, the max-reduction and the job
throughput, plus the oracle on each rank's own batch (distinct requests).
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, result_dir):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from oracle import oracle
    from paper_2608_03447_gb300 import inputs
    # each rank's own batch: a small block seeded by the rank's config family
    blk = inputs.gen_block(4, 8, 512, torch.float32, inputs.seed_for(bench.rank_config(rank), 0, 0), "cpu")
    res = oracle.verify(blk.logits, blk.draft.numpy(), np.array([[8.0, 0.0]] * 4, np.float32), 1.0, 2)
    local_ms = 10.0 * (rank + 1)                       # rank 1 is the slow one
    dist.barrier()
    job_ms = bench.max_over_ranks(local_ms, "cpu", world)
    value = bench.job_rows_per_s(world, 288, 100, job_ms / 1e3)
    np.savez(os.path.join(result_dir, f"rank{rank}.npz"), job_ms=job_ms, value=value,
             argmax=res["row_argmax"], draft=blk.draft.numpy())
    dist.destroy_process_group()


def test_two_gloo_ranks_weak_scaling(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    r0 = np.load(tmp_path / "rank0.npz")
    r1 = np.load(tmp_path / "rank1.npz")
    assert float(r0["job_ms"]) == float(r1["job_ms"]) == 20.0       # the slowest rank's time
    assert float(r0["value"]) == pytest.approx(2 * 288 * 100 / 0.020)  # all ranks' rows / that time
    assert not np.array_equal(r0["draft"], r1["draft"])              # disjoint batches per rank
    assert not np.array_equal(r0["argmax"], r1["argmax"])


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, "cpu", 1) == 3.5
    assert bench.job_rows_per_s(1, 288, 10, 0.5) == pytest.approx(5760.0)


def _np_partials(z_shard, draft, v_offset):
    """One shard's asd_partial rows (int32 [R, 6]) restated in numpy: the test's own key encoding."""
    B, K1, Vs = z_shard.shape
    K = K1 - 1
    rows = z_shard.reshape(B * K1, Vs).astype(np.float32)
    out = np.zeros((B * K1, 6), np.int32)
    for r in range(B * K1):
        loc = int(np.argmax(rows[r]))                    # first maximum
        top = rows[r, loc]
        u = np.array([top], np.float32).view(np.uint32)[0]
        if (u << np.uint32(1)) == 0:
            u = np.uint32(0)
        o = (~u) if (u & 0x80000000) else (u | np.uint32(0x80000000))
        key = (int(o) << 32) | (0xFFFFFFFF - (loc + v_offset))
        out[r, 0:2] = np.array([key], np.uint64).view(np.int32)
        out[r, 2] = np.array([top], np.float32).view(np.int32)[0]
        b, j = divmod(r, K1)
        zx = -np.inf
        if j < K and v_offset <= draft[b, j] < v_offset + Vs:
            zx = rows[r, draft[b, j] - v_offset]
        out[r, 3] = np.array([zx], np.float32).view(np.int32)[0]
    return out


def _shard_rank(rank, world, port, result_dir):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2608_03447_gb300 import asd, inputs
    blk = inputs.gen_block(3, 4, 999, torch.float32, 4242, "cpu")   # every rank generates the same block
    V = blk.logits.shape[-1]
    bounds = [0, 517, V]                                            # rank r holds vocabulary [bounds[r], bounds[r+1])
    z = blk.logits.numpy()[:, :, bounds[rank]:bounds[rank + 1]]
    part = torch.from_numpy(_np_partials(z, blk.draft.numpy(), bounds[rank]))
    gathered = asd.allgather_partials(part)                        # the exchange step
    np.save(os.path.join(result_dir, f"gathered{rank}.npy"), gathered.numpy())
    dist.destroy_process_group()


def test_two_gloo_ranks_exchange_vocab_partials(tmp_path):
    from oracle import oracle
    from paper_2608_03447_gb300 import inputs
    world = 2
    mp.spawn(_shard_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    g0 = np.load(tmp_path / "gathered0.npy")
    g1 = np.load(tmp_path / "gathered1.npy")
    assert np.array_equal(g0, g1) and g0.shape[0] == 2              # every rank holds both shards' partials
    keys = np.ascontiguousarray(g0[:, :, 0:2]).view(np.uint64)[..., 0]   # [S, R]
    win = np.argmax(keys, axis=0)                                   # combine: the largest key
    gidx = 0xFFFFFFFF - (keys[win, np.arange(keys.shape[1])] & 0xFFFFFFFF)
    zx = np.where(g0[0, :, 3].view(np.float32) != -np.inf, g0[0, :, 3].view(np.float32), g0[1, :, 3].view(np.float32))
    blk = inputs.gen_block(3, 4, 999, torch.float32, 4242, "cpu")
    o = oracle.verify(blk.logits, blk.draft.numpy(), None, strict=True)
    assert np.array_equal(gidx.reshape(3, 5), o["row_argmax"])
    top = g0[win, np.arange(keys.shape[1]), 2].view(np.float32).reshape(3, 5)
    r = (top[:, :4] - zx.reshape(3, 5)[:, :4]).astype(np.float32)
    assert np.array_equal(r.view(np.uint32), o["row_regret"].view(np.uint32))
