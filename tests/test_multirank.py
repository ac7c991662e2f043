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
