"""Host-side multi-rank logic of bench.py on CPU: two gloo ranks (the layer
shards into independent replicas, so the only cross-rank step is the timing
reduction: the job's time is the slowest rank's)."""
import os
import socket
import sys
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parent.parent


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist
    sys.path.insert(0, str(ROOT))
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed = 1.0 + rank                       # rank 1 is the slow one
        m = bench.max_over_ranks(elapsed, dist)
        rate = bench.whole_job_rate(21, 10, m, world)
        dist.barrier()
        (Path(out_dir) / f"rank{rank}.txt").write_text(f"{m} {rate}")
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time(tmp_path):
    import torch.multiprocessing as mp
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    for r in range(2):
        m, rate = map(float, (tmp_path / f"rank{r}.txt").read_text().split())
        assert m == 2.0
        assert rate == pytest.approx(2 * 21 * 10 / 2.0)


def test_single_process_is_identity():
    sys.path.insert(0, str(ROOT))
    import bench
    assert bench.max_over_ranks(3.5, None) == 3.5
    assert bench.whole_job_rate(21, 100, 0.5, 1) == pytest.approx(4200.0)
