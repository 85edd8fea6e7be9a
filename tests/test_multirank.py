"""The multi-rank path of bench.py on CPU: two gloo ranks, each timing its
own batch. The job time is the slowest rank's (MAX all-reduce, the only
collective), and the throughput counts every rank's tokens."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    local_ms = [30.0, 50.0][rank]          # rank 1 is slower
    ms_per_step, value = bench.weak_scaling(local_ms, steps=10, query_tokens_per_step=4096 * 32, ws=ws)
    out[rank] = (ms_per_step, value)
    bench.barrier(ws)
    dist.destroy_process_group()


def test_weak_scaling_uses_slowest_rank_and_all_tokens():
    ws = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, ws, port, out)) for r in range(ws)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for r in range(ws):
        ms, val = out[r]
        assert ms == pytest.approx(5.0)                       # max(30, 50) / 10 steps
        assert val == pytest.approx(4096 * 32 * ws / 5e-3)


def test_single_rank_needs_no_process_group():
    import bench
    ms, val = bench.weak_scaling(20.0, 4, 100, 1)
    assert ms == 5.0 and val == pytest.approx(100 / 5e-3)
