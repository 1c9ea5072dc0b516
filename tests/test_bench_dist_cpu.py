"""The multi-rank reduction of bench.py on CPU: two gloo ranks, the job's numbers come from the
slowest rank and count every rank's grid (replicas, weak scaling)."""

import os
import socket

import pytest

torch = pytest.importorskip("torch")


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = 10.0 * (rank + 1)                     # rank 1 is the slow one
    slowest = bench.allreduce_max(dist, ms)
    q.put((rank, slowest, bench.aggregate(slowest, 4, world)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_reduction_takes_the_slowest_rank():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    import bench
    for rank, slowest, (ms_step, iters, pairs) in out:
        assert slowest == 20.0
        assert ms_step == pytest.approx(5.0)
        assert iters == pytest.approx(2 * 200.0)
        assert pairs == pytest.approx(2 * 200.0 * bench.PAIRS)


def test_grid_option_scales_the_work_with_the_cells():
    """bench.py --grid RxC (small-case kernel captures) re-derives every per-iteration work
    figure from the cell count: evaluation and training FLOP and the backward's algorithmic
    bytes are per-cell sums, so a 6x6 torus has a quarter of the 12x12 figures."""
    import importlib.util
    import pathlib
    path = pathlib.Path(__file__).resolve().parents[1] / "bench.py"
    spec = importlib.util.spec_from_file_location("bench_grid_probe", path)
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    full = (b.CELLS, b.PAIRS, b.EVAL_G_FLOP, b.EVAL_D_FLOP, b.TRAIN_FWD_FLOP, b.TRAIN_BWD_FLOP,
            b.MIX_FLOP, b.TRAIN_BWD_BYTES)
    assert full[0] == 144 and full[1] == 3600
    b.ROWS, b.COLS = 6, 6
    b._derive()
    small = (b.CELLS, b.PAIRS, b.EVAL_G_FLOP, b.EVAL_D_FLOP, b.TRAIN_FWD_FLOP, b.TRAIN_BWD_FLOP,
             b.MIX_FLOP, b.TRAIN_BWD_BYTES)
    for f, s in zip(full, small):
        assert s * 4 == f
    # the evaluation's FLOP: 2 B rows x (z h + h h + h x) per generator slot, 2 x 6B rows x
    # (x h + h h + h) per discriminator slot, 5 slots of each per cell
    assert b.EVAL_G_FLOP == 2 * 36 * 5 * 100 * (64 * 256 + 256 * 256 + 256 * 784)
    assert b.EVAL_D_FLOP == 2 * 36 * 30 * 100 * (784 * 256 + 256 * 256 + 256)
