"""bench.py's multi-GPU mode runs independent replicas (sequences are
independent, no collective on the data path); the only cross-rank step is the
timing reduction.  Checked here with world_size 2 over gloo on the CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import synth
    # rank 0: 90 tokens in 10 ms; rank 1: 60 tokens in 20 ms -> 150 tokens per 20 ms
    committed, ms = [(90.0, 10.0), (60.0, 20.0)][rank]
    value, step_ms = bench.replica_throughput(committed, ms, world)
    sched = synth.forced_schedule(synth.QWEN3_8B, 8, seed=synth.SEED_SCHEDULE + rank)
    out[rank] = (value, step_ms, sched.tolist())
    dist.barrier()
    dist.destroy_process_group()


def test_two_replicas_over_gloo():
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(2, port, out), nprocs=2, join=True, start_method="spawn")
        res = dict(out)
    for r in (0, 1):
        value, step_ms, _ = res[r]
        assert step_ms == pytest.approx(20.0)
        assert value == pytest.approx(150.0 / 0.020)
    assert res[0][2] != res[1][2]  # each replica draws its own acceptance schedule


def test_single_replica_needs_no_process_group():
    import bench
    value, ms = bench.replica_throughput(90.0, 10.0, 1)
    assert value == pytest.approx(9000.0) and ms == 10.0
