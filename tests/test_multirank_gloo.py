"""The multi-GPU host logic of bench.py on CPU: two gloo ranks, each planning
its own shard of traces (weak scaling, no data-path collective), with the
max-over-ranks time and the summed unit counts the bench reports."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    import oracle
    import tracegen as tg

    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, _ = bench.dist_env()
    assert (r, w) == (rank, world)
    # --gpus must match the ranks torchrun started: each rank refuses a mismatch
    assert bench.resolve_launch(world) == "run"
    assert bench.resolve_launch(world + 2) == "mismatch" and bench.resolve_launch(1) == "mismatch"
    n_traces = 6
    ts = tg.random_batch(bench.shard_seed0(r, n_traces), n_traces, 40, 64)
    off, pk, st = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    t_max = bench.max_over_ranks(float(rank + 1), dist)
    total = bench.sum_over_ranks(float(ts.n_tensors), dist)
    np.savez(os.path.join(out_dir, f"rank{rank}.npz"), off=off, pk=pk, st=st, t_max=t_max, total=total)
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_rank_sharding_matches_single_process(tmp_path):
    world, port = 2, _free_port()
    mp.spawn(_worker, args=(world, port, str(tmp_path)), nprocs=world, join=True)
    import oracle
    import tracegen as tg

    whole = tg.random_batch(0, 12, 40, 64)
    off, pk, st = oracle.plan_greedy_by_size(whole, oracle.FIT_FIRST)
    parts = [np.load(tmp_path / f"rank{r}.npz") for r in range(world)]
    assert np.array_equal(np.concatenate([p["off"] for p in parts]), off)
    assert np.array_equal(np.concatenate([p["pk"] for p in parts]), pk)
    assert all((p["st"] == 0).all() for p in parts)
    assert all(float(p["t_max"]) == 2.0 for p in parts)
    assert all(float(p["total"]) == whole.n_tensors for p in parts)


def test_gpus_argument_without_torchrun():
    """Outside torchrun, --gpus 1 runs in this process and --gpus N > 1 re-launches
    the command with N ranks; a bad count is refused."""
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    assert bench.resolve_launch(1, {}) == "run"
    assert bench.resolve_launch(4, {}) == "spawn"
    assert bench.resolve_launch(0, {}) == "mismatch"
    assert bench.resolve_launch(2, {"WORLD_SIZE": "2"}) == "run"
    assert bench.resolve_launch(8, {"WORLD_SIZE": "2"}) == "mismatch"
