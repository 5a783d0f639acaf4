"""Host-side pieces of bench.py that need no GPU."""
import json
import shutil
from pathlib import Path

import bench

ROOT = Path(bench.ROOT)
WORKLOAD = "llada8b_d4096_V126464_B1_L128"


def _copy_tree(tmp_path):
    (tmp_path / "profiles").mkdir()
    shutil.copy(ROOT / "profiles" / "score_kernel_traffic.txt", tmp_path / "profiles")
    src = ROOT / "paper_2605_16941_gb300" / "csrc"
    dst = tmp_path / "paper_2605_16941_gb300" / "csrc"
    dst.mkdir(parents=True)
    for f in src.iterdir():
        if f.is_file():
            shutil.copy(f, dst)
    return dst


def test_ncu_traffic_is_tied_to_the_kernel_sources(tmp_path, monkeypatch):
    rec = json.loads((ROOT / "profiles" / "score_kernel_traffic.txt").read_text())
    want = float(rec["dram_bytes_read"]) + float(rec["dram_bytes_write"])
    assert bench.ncu_traffic(WORKLOAD) == want
    assert bench.ncu_traffic("some_other_workload") is None
    csrc = _copy_tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.ncu_traffic(WORKLOAD) == want
    for name in rec["score_kernel_sources"]:  # a change to any source the kernel is built from voids it
        f = csrc / name
        old = f.read_bytes()
        f.write_bytes(old + b"\n// edited\n")
        assert bench.ncu_traffic(WORKLOAD) is None, name
        f.write_bytes(old)
    assert bench.ncu_traffic(WORKLOAD) == want


def test_job_rows_per_s_counts_every_rank():
    assert bench.job_rows_per_s(256, 10, 4, 2.0) == 256 * 10 * 4 / 2.0
