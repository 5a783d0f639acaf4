"""Host-side pieces of bench.py that need no GPU."""
import json
import shutil
from pathlib import Path

import bench

ROOT = Path(bench.ROOT)


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


def _sha(csrc, names):
    import hashlib
    h = hashlib.sha256()
    for name in names:
        h.update((csrc / name).read_bytes())
    return h.hexdigest()[:16]


def test_ncu_traffic_is_tied_to_the_kernel_sources(tmp_path, monkeypatch):
    """A traffic record counts only for its workload and LM-head layout, and only while every source file the score
    kernel is built from is unchanged."""
    rec = json.loads((ROOT / "profiles" / "score_kernel_traffic.txt").read_text())
    want = float(rec["dram_bytes_read"]) + float(rec["dram_bytes_write"])
    fresh = rec["sources_sha256_prefix"] == _sha(ROOT / "paper_2605_16941_gb300" / "csrc", rec["score_kernel_sources"])
    assert bench.ncu_traffic(rec["workload"]) == (want if fresh else None)
    assert bench.ncu_traffic("some_other_workload") is None
    csrc = _copy_tree(tmp_path)
    rec["sources_sha256_prefix"] = _sha(csrc, rec["score_kernel_sources"])  # a record taken on these sources
    (tmp_path / "profiles" / "score_kernel_traffic.txt").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.ncu_traffic(rec["workload"]) == want
    other = "rows" if rec.get("w_layout", "rows") == "panels" else "panels"
    assert bench.ncu_traffic(rec["workload"], other) is None  # taken with the other LM-head layout
    for name in rec["score_kernel_sources"]:  # a change to any source the kernel is built from voids it
        f = csrc / name
        old = f.read_bytes()
        f.write_bytes(old + b"\n// edited\n")
        assert bench.ncu_traffic(rec["workload"]) is None, name
        f.write_bytes(old)
    assert bench.ncu_traffic(rec["workload"]) == want


def test_job_rows_per_s_counts_every_rank():
    assert bench.job_rows_per_s(256, 10, 4, 2.0) == 256 * 10 * 4 / 2.0
