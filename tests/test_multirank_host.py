"""The multi-GPU path is replicas only: every rank decodes its own batch and the job's
throughput is all ranks' rows over the slowest rank's time.  The host side of that
(max over ranks, aggregation, which ranks print) runs here on CPU with gloo, world size 2."""
import os
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, times, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    t = bench.job_time_max(times[rank], world)
    out[rank] = (t, bench.job_rows_per_s(256, 100, world, t))
    dist.barrier()
    dist.destroy_process_group()


def test_job_time_is_the_slowest_rank():
    world, port = 2, 29511
    times = [0.020, 0.025]
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_worker, args=(world, port, times, out), nprocs=world, start_method="spawn")
        res = dict(out)
    for rank in range(world):
        t, v = res[rank]
        assert t == max(times)
        assert v == pytest.approx(world * 256 * 100 / max(times))


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "3",
                        "--warmup", "3"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""
