"""Host logic of bench.py's multi-GPU line on CPU: world_size 2 over gloo.

Rows are independent, so N GPUs run N replicas of the step with no collective
on the data path; the only cross-rank steps are the barrier and the
max-over-ranks of the timed region, tested here without a GPU."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    ms = bench.max_over_ranks(10.0 * (rank + 1), ws, torch.device("cpu"))
    out[rank] = (ms, bench.replica_value(ws, 32, 100, ms))
    # the reference arm: only rank 0 works (and prints); the others return at once
    os.environ["RANK"] = str(rank)
    if rank != 0:
        assert bench.run_reference(None) is None
    dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ws = 2
    port = _free_port()
    with mp.Manager() as man:
        out = man.dict()
        mp.spawn(_worker, args=(ws, port, out), nprocs=ws, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 20.0
    # 2 ranks x 32 rows x 100 steps in 20 ms
    assert abs(res[0][1] - 2 * 32 * 100 / 0.020) < 1e-6


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(12.5, 1, None) == 12.5
    assert bench.replica_value(1, 32, 200, 40.0) == 32 * 200 / 0.040
