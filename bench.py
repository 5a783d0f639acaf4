#!/usr/bin/env python3
"""Throughput of one WINO step (fused LM head + vocabulary softmax + Eq. 4 revoke) on GB300.

Workload (default): the unified text+image vocabulary step, the largest of the
single-GPU configurations: d=4096, V=134400, 4 sequences of a 256-position block
plus its 256 shadow rows (N=2048 scored rows), seeded synthetic inputs
(wino_synth).  A step is one wino_step call through the C ABI: the fused score
kernel (LM-head GEMM + online vocabulary softmax on 2-SM tensor-core tiles) and
the finish kernel (cross-tile merge + Eq. 4 update).

Prints one JSON line (rank 0).  `value` is scored rows/s over the K timed
steps with inputs resident in HBM (W is 1.1 GB, larger than L2, so no L2
flush is needed); `e2e` is the same metric with each step's hidden states
and token state copied in from pinned host memory and the tokens and counts
copied back, through the same C ABI; `roofline` rates the dominant kernel
(the fused score kernel, timed by CUDA events the library records around
each launch on the launch stream, in a second region of K steps) against the
measured peak of its bound; `configs` repeats the step and kernel timing, at
the same K, on the three LLaDA-8B-shaped configurations (one sequence, N=256;
eight sequences, N=2048; the 16-sequence decode step, N=1024); `cpu_baseline`
times the fp64 CPU oracle on a bounded sample of the workload's rows on this
host's cores, and `parity` compares one whole GPU step with the oracle's whole
step (every row scored in fp64).

--impl reference times the oracle itself as the reference arm (CPU, fp64).
Multi-GPU (torchrun): every rank decodes its own replica (weak scaling); no
collective on the data path.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "scored rows/s for fused LM-head+softmax+WINO revoke; % of GEMM/HBM roofline"
UNIT = "rows/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured (MEASURED_PEAKS.json)"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


W_LAYOUTS = {"panels": "the LM head as 64-column panels (wino_lm_head_panels, made once before timing; "
                      "WINO_OPT_W_PANELS)",
             "rows": "the LM head row-major [V, d]"}


def lm_head(wino, Wd, layout: str):
    """The W argument of the steps for the chosen layout (the panel copy is made here, outside any timing)."""
    return wino.wino_lm_head_panels(Wd) if layout == "panels" else Wd


def config_dict(w):
    return {"workload": w.name, "N": w.N, "d": w.d, "V": w.V, "n_seq": w.n_seq, "blk_len": w.blk_len,
            "tau1": w.tau1, "tau2": w.tau2, "seed": w.seed,
            "l2": ("inputs larger than L2: W_lm is %.3f GB, read once per step" % (w.V * w.d * 2 / 1e9)
                   if w.V * w.d * 2 > 129e6 else
                   "L2-resident: W_lm is %.1f MB (a latency-bound case; L2 not flushed)" % (w.V * w.d * 2 / 1e6)),
            "parallelism": "replicas (one independent decode per GPU)"}


class ClockSampler:
    """nvidia-smi sampling of SM clock, power and throttle reasons while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw.instant,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.samples = []
        self.proc = None
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50"]
        if gpu_id:
            cmd += ["-i", gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def wait_first(self, timeout_s: float = 10.0):
        """Return once nvidia-smi has printed a sample (its start-up is then over), or after the timeout."""
        t0 = time.time()
        while self.proc and not self.samples and time.time() - t0 < timeout_s and self.proc.poll() is None:
            time.sleep(0.05)

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0, t1):
        if not self.samples:
            return None
        inside = [s for t, s in self.samples if t0 <= t <= t1 + 0.06]
        used = inside or [min(self.samples, key=lambda ts: min(abs(ts[0] - t0), abs(ts[0] - t1)))[1]]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, pw, reasons = [], [], [], set()
        for s in used:
            try:
                sm.append(float(s[0]))
                mx.append(float(s[1]))
                pw.append(float(s[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, s[3:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(mx), "power_w_max": max(pw), "reasons": sorted(reasons),
                "samples": len(sm), "samples_in_timed_region": len(inside)}


def ncu_traffic(workload_name: str, layout: str = "panels"):
    """DRAM bytes per score launch from the committed ncu capture, if it was taken on this workload with this
    LM-head layout and none of the score kernel's source files has changed since (else None)."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "score_kernel_traffic.txt")) as f:
            rec = json.load(f)
        h = hashlib.sha256()
        for name in rec["score_kernel_sources"]:
            with open(os.path.join(ROOT, "paper_2605_16941_gb300", "csrc", name), "rb") as f:
                h.update(f.read())
    except (OSError, ValueError, KeyError, TypeError):
        return None
    if rec.get("workload") != workload_name or rec.get("sources_sha256_prefix") != h.hexdigest()[:16] or \
            rec.get("w_layout", "rows") != layout:
        return None
    return float(rec["dram_bytes_read"]) + float(rec["dram_bytes_write"])


def job_time_max(seconds_local: float, world: int, device=None) -> float:
    """The slowest rank's time (max over ranks); the job's throughput divides all ranks' work by it."""
    import torch
    t = torch.tensor([seconds_local], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rows_per_s(rows_per_rank_step: int, steps: int, world: int, t_max_s: float) -> float:
    """Whole-job scored rows/s: every rank decodes its own replica (weak scaling)."""
    return world * rows_per_rank_step * steps / t_max_s


def gpu_uuid(dev):
    import torch
    try:
        u = torch.cuda.get_device_properties(dev).uuid
        s = str(u)
        return s if s.startswith("GPU-") else "GPU-" + s
    except Exception:
        return None


def roofline_terms(w, rows_scored, peaks):
    """Algorithmic work of one score launch (2 N d V flops; W and H read once, 12 B of results per row) and
    the time each would take at the measured peaks."""
    flops = 2.0 * rows_scored * w.d * w.V
    w_bytes = w.V * w.d * 2.0
    alg_bytes = w_bytes + rows_scored * w.d * 2.0 + 12.0 * rows_scored
    t_flop = flops / (peaks["bf16_tflops"] * 1e12)
    t_hbm = alg_bytes / (peaks["hbm_gbs"] * 1e9)
    return flops, w_bytes, alg_bytes, t_flop, t_hbm, ("hbm" if t_hbm >= t_flop else "tensor")


def kernel_roofline(w, rows_scored, peaks, score_avg_s):
    """The score kernel's achieved rate against the measured peak of its bound."""
    flops, w_bytes, alg_bytes, t_flop, t_hbm, bound = roofline_terms(w, rows_scored, peaks)
    if bound == "hbm":
        achieved, peak, unit = alg_bytes / score_avg_s / 1e9, peaks["hbm_gbs"], "GB/s"
    else:
        achieved, peak, unit = flops / score_avg_s / 1e12, peaks["bf16_tflops"], "TFLOP/s"
    tflops = flops / score_avg_s / 1e12
    return {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit, "frac": achieved / peak,
            "algorithmic_per_launch": {"bytes": alg_bytes, "flops": flops}, "avg_launch_us": score_avg_s * 1e6,
            "tensor_tflops": tflops, "tensor_frac": tflops / peaks["bf16_tflops"],
            "tensor_frac_sustained": tflops / peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])}


def time_steps(step, steps, stream, dev):
    """K calls of step(i) back to back between two CUDA events on the launch stream (ms)."""
    import torch
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    ev0.record(stream)
    for i in range(steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    return ev0.elapsed_time(ev1)


def time_score_kernel(wino, step, steps, dev):
    """Average duration (s) of the score kernel over K more steps, from the CUDA events the library records
    around each of its launches on the launch stream (this serialises the launches)."""
    import torch
    torch.cuda.synchronize(dev)
    wino.wino_profile_begin(steps)
    for i in range(steps):
        step(i)
    score_ms, score_n = wino.wino_profile_end()
    torch.cuda.synchronize(dev)
    return (score_ms / max(1, score_n)) / 1e3, score_n


def measure_configs(names, args, wino, ws, dev, sid, peaks, to_dev):
    """Step and score-kernel timing of other configurations at the same step count (resident inputs)."""
    import torch
    out, w_cache = {}, {}
    for name in names:
        w = ws.WORKLOADS[name]
        key = (w.d, w.V, w.seed)
        if key not in w_cache:
            w_cache.clear()  # one extra LM head resident at a time
            W = ws.weights(w)
            w_cache[key] = (W, lm_head(wino, to_dev(W), args.w_layout))
        W, Wd = w_cache[key]
        st = ws.initial_state(w)
        Hd = [to_dev(ws.hidden_states(w, W, st, step=k)) for k in range(2)]
        tok = to_dev(st.tokens)
        counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device=dev)
        wsp = wino.workspace(w.N, w.d, w.V, device=dev)
        p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len,
                             w_panels=args.w_layout == "panels")

        def step(i):
            wino.wino_step(Hd[i % 2], Wd, tok, p, counts, wsp, stream=sid)

        for i in range(args.warmup):
            step(i)
        ms = time_steps(step, args.steps, torch.cuda.current_stream(dev), dev)
        score_avg_s, _ = time_score_kernel(wino, step, args.steps, dev)
        if wino.wino_read_device_status(wsp, stream=sid) != wino.WINO_OK:
            raise RuntimeError(f"device status not OK on {name}")
        flops, w_bytes, _, t_flop, _, _ = roofline_terms(w, w.N, peaks)
        step_s = ms / 1e3 / args.steps
        out[name] = {"workload": w.name, "N": w.N, "d": w.d, "V": w.V, "steps": args.steps,
                     "ms_per_step": ms / args.steps, "rows_per_s": w.N / step_s,
                     "tflops_per_step": flops / step_s / 1e12,
                     "step_roofline_frac": max(t_flop, w_bytes / (peaks["hbm_gbs"] * 1e9)) / step_s,
                     "kernel_roofline": kernel_roofline(w, w.N, peaks, score_avg_s),
                     "w_layout": W_LAYOUTS[args.w_layout]}
        del Hd, tok, wsp
    return out


def oracle_baseline_and_parity(w, W, H, st, gpu_stats, tok_gpu, cnt_gpu, budget_s: float = 15.0):
    """The fp64 oracle on every row of one step of the workload.  A first chunk of rows (about budget_s of
    CPU work) is the timed CPU baseline; all rows then give the oracle's whole step, compared with one GPU
    step from the same state: per-row probabilities within 1e-3, argmax and token state exact outside the
    counted near-tie and near-threshold positions (the tolerances of the parity tests)."""
    import numpy as np

    import oracle
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    from gpu_helpers import PROB_TOL, TIE_TOL, flagged_positions
    nt = oracle.num_threads()
    t = oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id)
    n1 = min(nt, w.N)
    t0 = time.perf_counter()
    first = oracle.score_rows(H[:n1], W, t[:n1])
    t_first = time.perf_counter() - t0
    chunk = int(min(w.N - n1, max(nt, nt * round(budget_s / t_first))))
    parts = [first]
    t_chunk = t_rest = 0.0
    if chunk > 0:
        t0 = time.perf_counter()
        parts.append(oracle.score_rows(H[n1:n1 + chunk], W, t[n1:n1 + chunk]))
        t_chunk = time.perf_counter() - t0
    timed_rows, timed_s = (chunk, t_chunk) if chunk > 0 else (n1, t_first)
    cpu = {"value": timed_rows / timed_s, "unit": UNIT, "cores": nt, "kind": "oracle",
           "sample": f"{timed_rows} of the {w.N} rows of one step of {w.name}, each scored over the full vocabulary "
                     f"in fp64 ({timed_s:.1f} s); the Eq. 4 update (microseconds) is not included",
           "seconds": timed_s}
    if n1 + chunk < w.N:
        t0 = time.perf_counter()
        parts.append(oracle.score_rows(H[n1 + chunk:], W, t[n1 + chunk:]))
        t_rest = time.perf_counter() - t0
    o = type(first)(*(np.concatenate([getattr(x, f) for x in parts]) for f in first.__dataclass_fields__))
    tok, cnt, fl = oracle.draft_verify(st.tokens, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2, o.argmax,
                                       o.pmax, o.ptarget)
    ostep = oracle.StepResult(tok, cnt, fl, o.argmax, o.pmax, o.ptarget, o.gap)
    flag = flagged_positions(st.tokens, ostep, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2)
    b0, L = st.blk_start, w.blk_len
    g_blk, o_blk = tok_gpu[:, b0:b0 + L], tok[:, b0:b0 + L]
    outside = np.ones(st.tokens.shape[1], bool)
    outside[b0:b0 + L] = False
    near = o.gap < TIE_TOL
    clean = ~flag.any(1)
    parity = {
        "rows": int(w.N), "oracle": "fp64 CPU oracle, every row over the full vocabulary, then Eq. 4",
        "tolerance": f"per-row probabilities within {PROB_TOL} absolute; argmax and token state exact except at "
                     f"positions whose top-2 logits differ by < {TIE_TOL} or whose decision probability lies within "
                     f"{PROB_TOL} of its threshold (flagged, counted)",
        "max_abs_dpmax": float(np.abs(gpu_stats.pmax.astype(np.float64) - o.pmax).max()),
        "max_abs_dptarget": float(np.abs(gpu_stats.ptarget.astype(np.float64) - o.ptarget).max()),
        "argmax_mismatch_outside_near_ties": int(((gpu_stats.argmax != o.argmax) & ~near).sum()),
        "argmax_near_ties": int(near.sum()),
        "token_mismatch_outside_flagged": int(((g_blk != o_blk) & ~flag).sum()),
        "flagged_positions": int(flag.sum()),
        "flagged_mismatch": int(((g_blk != o_blk) & flag).sum()),
        "positions_outside_block_changed": int((tok_gpu[:, outside] != st.tokens[:, outside]).sum()),
        "counts_mismatch_unflagged_sequences": int((cnt_gpu[clean] != cnt[clean]).any(1).sum()),
        "oracle_branches": {"threshold_drafts": int((fl == oracle.FLAG_DRAFT).sum()),
                            "fallback_drafts": int((fl == oracle.FLAG_DRAFT_FALLBACK).sum()),
                            "remasked": int((fl == oracle.FLAG_REMASK).sum())},
        "oracle_seconds": t_first + t_chunk + t_rest,
    }
    parity["ok"] = (parity["max_abs_dpmax"] <= PROB_TOL and parity["max_abs_dptarget"] <= PROB_TOL and
                    parity["argmax_mismatch_outside_near_ties"] == 0 and parity["token_mismatch_outside_flagged"] == 0
                    and parity["positions_outside_block_changed"] == 0
                    and parity["counts_mismatch_unflagged_sequences"] == 0)
    return cpu, parity


def oracle_cpu_baseline(w, W, H, targets, budget_s: float = 12.0, max_rows: int = 256):
    """Time the oracle scoring rows of this step in batches of one row per thread until the budget is spent."""
    import numpy as np

    import oracle
    nt = oracle.num_threads()
    rows, t_total, i = 0, 0.0, 0
    while rows < max_rows and (t_total < budget_s or rows == 0):
        idx = np.arange(i, i + nt) % w.N
        t0 = time.perf_counter()
        oracle.score_rows(H[idx], W, targets[idx])
        t_total += time.perf_counter() - t0
        rows += nt
        i += nt
    return {"value": rows / t_total, "unit": UNIT, "cores": nt, "kind": "oracle",
            "sample": f"{rows} of the {w.N} rows of one step of {w.name}, each scored over the full vocabulary "
                      f"in fp64 ({t_total:.1f} s); the Eq. 4 update (microseconds) is not included",
            "seconds": t_total}


def run_reference(args):
    """Reference arm: the fp64 oracle as it stands, on this host's cores, same workload and metric."""
    import numpy as np

    import oracle
    import wino_synth as ws
    w = ws.WORKLOADS[args.workload]
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    t = oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id)
    nt = oracle.num_threads()
    # calibrate: one batch of nt rows over a vocabulary slice
    slice_v = min(w.V, 4096)
    t0 = time.perf_counter()
    oracle.score_rows(H[:nt], W[:slice_v], t[:nt])
    per_logit = (time.perf_counter() - t0) / (nt * slice_v)
    per_step = max(0.005, args.ref_budget_s / (args.steps + args.warmup))
    # rows x vocabulary-slice sample per step sized to the per-step budget (at least one row-slice per thread)
    sv = int(min(w.V, max(256, per_step / (per_logit * nt))))
    sample_logits = nt * sv
    times = []
    for i in range(args.warmup + args.steps):
        idx = (np.arange(nt) + i * nt) % w.N
        v0 = (i * 7919) % max(1, w.V - sv + 1)
        t0 = time.perf_counter()
        oracle.score_rows(H[idx], W[v0:v0 + sv], None)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.append(dt)
    tot = sum(times)
    rows_equiv = args.steps * sample_logits / w.V
    value = rows_equiv / tot
    sample = (f"per step {nt} rows x a {sv}-entry vocabulary slice ({sample_logits / w.V:.4f} full-vocabulary rows) "
              f"of {w.name}, fp64 oracle; value counts full-vocabulary-row equivalents")
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(w), "impl": "reference",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": nt, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


def run_wino(args, rank, world, local_rank):
    import numpy as np
    import torch
    import torch.distributed as dist

    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)

    from paper_2605_16941_gb300 import build as pkg_build
    if rank == 0:
        pkg_build.build()
    if world > 1:
        dist.barrier()
    import paper_2605_16941_gb300 as wino
    import wino_synth as ws

    w = ws.WORKLOADS[args.workload]
    if args.no_shadow:  # WINO+ inference: block rows only
        import dataclasses
        w = dataclasses.replace(w, shadow=False)
    score_only = args.score_rows or args.entropy
    t_gen = time.time()
    W = ws.weights(w)
    st = ws.initial_state(w)
    n_h = 4
    Hs = [ws.hidden_states(w, W, st, step=k) for k in range(n_h)]
    log(f"[rank {rank}] inputs generated in {time.time() - t_gen:.1f} s")

    def to_dev(a):
        a = np.ascontiguousarray(a)
        return torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).to(dev)

    W_rows = to_dev(W)  # row-major: wino_score_rows reads this layout
    layout = "rows" if score_only else args.w_layout
    Wd = lm_head(wino, W_rows, layout)
    Hd = [to_dev(h) for h in Hs]
    tok = to_dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device=dev)
    wsp = wino.workspace(w.N, w.d, w.V, device=dev)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len,
                         compact=args.compact, no_shadow=args.no_shadow, draft_m=args.draft_m,
                         w_panels=layout == "panels")
    if args.compact:  # row compaction needs room for the gathered rows
        wsp = wino.step_workspace(p, w.d, w.V, device=dev)
    stream = torch.cuda.current_stream(dev)
    sid = stream.cuda_stream
    am = torch.empty(w.N, dtype=torch.int32, device=dev)
    pm = torch.empty(w.N, dtype=torch.float32, device=dev)
    pt = torch.empty(w.N, dtype=torch.float32, device=dev)
    ent = torch.empty(w.N, dtype=torch.float32, device=dev) if args.entropy else None

    def step(i):
        if score_only:  # wino_score_rows alone (statistics of every row, optionally with H(p))
            wino.wino_score_rows(Hd[i % n_h], W_rows, None, am, pm, pt, wsp, stream=sid, entropy=ent)
        else:
            wino.wino_step(Hd[i % n_h], Wd, tok, p, counts, wsp, stream=sid)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize(dev)
    if wino.wino_read_device_status(wsp, stream=sid) != wino.WINO_OK:
        raise RuntimeError("device status not OK after warm-up")
    run_steps = None
    if args.graph:  # capture `graph` consecutive steps once; the timed region replays the graph
        if args.steps % args.graph:
            raise SystemExit("--steps must be a multiple of --graph")
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for i in range(args.graph):
                if score_only:
                    wino.wino_score_rows(Hd[i % n_h], W_rows, None, am, pm, pt, wsp, entropy=ent)
                else:
                    wino.wino_step(Hd[i % n_h], Wd, tok, p, counts, wsp)
        torch.cuda.synchronize(dev)

        def run_steps(k):
            for _ in range(k // args.graph):
                graph.replay()
        run_steps(args.graph)  # one untimed replay
        torch.cuda.synchronize(dev)

    clocks = ClockSampler(gpu_uuid(dev)) if rank == 0 else None
    if clocks:
        clocks.wait_first()  # nvidia-smi's start-up must not overlap the timed region
        time.sleep(0.2)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    # Timed region: K steps back to back, nothing between the kernels (consecutive steps overlap
    # through programmatic dependent launch).
    tw0 = time.time()
    ev0.record(stream)
    if run_steps is not None:
        run_steps(args.steps)
    else:
        for i in range(args.steps):
            step(i)
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    tw1 = time.time()
    if world > 1:
        dist.barrier()
    elapsed_ms = ev0.elapsed_time(ev1)
    # Second region, K more steps: the library brackets every score-kernel launch with CUDA events
    # on the launch stream (this serialises the launches), giving the kernel's own average duration.
    torch.cuda.synchronize(dev)
    wino.wino_profile_begin(args.steps)
    for i in range(args.steps):
        step(i)
    score_ms, score_n = wino.wino_profile_end()
    torch.cuda.synchronize(dev)
    if clocks:
        time.sleep(0.1)
        clocks.stop()
    if wino.wino_read_device_status(wsp, stream=sid) != wino.WINO_OK:
        raise RuntimeError("device status not OK after the timed region")
    t_max = 1e3 * job_time_max(elapsed_ms / 1e3, world, device=dev)

    # ---- end to end through the C ABI with host buffers (pinned): every step uploads its hidden states and
    # token state, and the host reads that step's result (token state and counts) back.  Two buffer sets
    # and three streams (upload, compute, download) let step i+1's upload and step i-1's download run
    # under step i's kernels; the host reads a step's result before its buffers are reused.
    Hh = [torch.from_numpy(np.ascontiguousarray(h).view(np.int16)).pin_memory() for h in Hs]
    tok_h = torch.from_numpy(st.tokens).pin_memory()
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    Hbuf = [torch.empty_like(Hd[0]) for _ in range(2)]
    tokb = [torch.empty_like(tok) for _ in range(2)]
    cntb = [torch.zeros_like(counts) for _ in range(2)]
    tok_out = [torch.empty_like(tok_h).pin_memory() for _ in range(2)]
    cnt_out = [torch.empty((w.n_seq, 3), dtype=torch.int32).pin_memory() for _ in range(2)]
    ev_up = [torch.cuda.Event() for _ in range(2)]
    ev_step = [torch.cuda.Event() for _ in range(2)]
    ev_down = [torch.cuda.Event() for _ in range(2)]
    pending = [False, False]
    e2e_bad = [0]
    e2e_steps = args.steps

    def consume(j):  # the host reads a finished step's result
        ev_down[j].synchronize()
        if int(cnt_out[j].min()) < 0 or int(tok_out[j][0, 0]) < 0:
            e2e_bad[0] += 1
        pending[j] = False

    def e2e_step(i):
        j = i % 2
        if pending[j]:
            consume(j)
        with torch.cuda.stream(up):
            up.wait_event(ev_step[j])  # step i-2 is done with these buffers
            Hbuf[j].copy_(Hh[i % n_h], non_blocking=True)
            tokb[j].copy_(tok_h, non_blocking=True)
            ev_up[j].record(up)
        stream.wait_event(ev_up[j])
        wino.wino_step(Hbuf[j], Wd, tokb[j], p, cntb[j], wsp, stream=sid)
        ev_step[j].record(stream)
        with torch.cuda.stream(down):
            down.wait_event(ev_step[j])
            tok_out[j].copy_(tokb[j], non_blocking=True)
            cnt_out[j].copy_(cntb[j], non_blocking=True)
            ev_down[j].record(down)
        pending[j] = True

    def e2e_drain():
        for j in range(2):
            if pending[j]:
                consume(j)

    if score_only:
        e2e_steps = 0
    for i in range(max(3, args.warmup) if e2e_steps else 0):
        e2e_step(i)
    e2e_drain()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    te0 = time.perf_counter()
    for i in range(e2e_steps):
        e2e_step(i)
    e2e_drain()
    torch.cuda.synchronize(dev)
    te = time.perf_counter() - te0
    te = job_time_max(te, world, device=dev) if e2e_steps else 0.0
    if e2e_bad[0]:
        raise RuntimeError(f"{e2e_bad[0]} end-to-end steps returned an error status")
    h2d = Hh[0].numel() * 2 + tok_h.numel() * 4
    d2h = tok_out[0].numel() * 4 + cnt_out[0].numel() * 4

    if rank != 0:
        if world > 1:
            dist.barrier()
            dist.destroy_process_group()
        return

    peaks, peak_src = load_peaks()
    rows_scored = w.N // 2 if args.compact else w.N  # rows the score kernel actually multiplies
    flops, w_bytes, alg_bytes, t_flop, t_hbm, bound = roofline_terms(w, rows_scored, peaks)
    score_avg_s = (score_ms / max(1, score_n)) / 1e3
    roof = kernel_roofline(w, rows_scored, peaks, score_avg_s)
    step_s = t_max / 1e3 / args.steps
    value = job_rows_per_s(w.N, args.steps, world, t_max / 1e3)
    clock_info = clocks.summary(tw0, tw1) if clocks else None

    # The other LLaDA-shaped configurations at the same step count (rank 0 only).
    configs = None
    plain = not (args.no_shadow or score_only or args.compact or args.draft_m or args.graph)
    if plain and not args.no_configs:
        names = [n for n in ("llada_b1", "llada_b8", "loop_b16") if n != args.workload]
        configs = measure_configs(names, args, wino, ws, dev, sid, peaks, to_dev)

    cpu, parity = None, None
    if world == 1 and not args.no_cpu_baseline:
        import oracle
        if plain:
            # one GPU step and the GPU's statistics of every row, from the initial state; then the oracle
            tok1 = to_dev(st.tokens)
            cnt1 = torch.zeros_like(counts)
            ws1 = wino.workspace(w.N, w.d, w.V, device=dev)
            wino.wino_step(Hd[0], Wd, tok1, p, cnt1, ws1, stream=sid)
            t_rows = to_dev(oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id))
            wino.wino_score_rows(Hd[0], W_rows, t_rows, am, pm, pt, ws1, stream=sid)
            torch.cuda.synchronize(dev)
            if wino.wino_read_device_status(ws1, stream=sid) != wino.WINO_OK:
                raise RuntimeError("device status not OK in the parity step")
            from types import SimpleNamespace
            g = SimpleNamespace(argmax=am.cpu().numpy(), pmax=pm.cpu().numpy(), ptarget=pt.cpu().numpy())
            cpu, parity = oracle_baseline_and_parity(w, W, Hs[0], st, g, tok1.cpu().numpy(), cnt1.cpu().numpy(),
                                                     budget_s=args.cpu_budget_s)
        else:
            t = np.full(w.N, -1, np.int32) if (args.no_shadow or score_only) else \
                oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id)
            cpu = oracle_cpu_baseline(w, W, Hs[0], t, budget_s=args.cpu_budget_s)

    cfg = config_dict(w)
    if args.no_shadow:
        cfg["no_shadow"] = "WINO+ inference (WINO_OPT_NO_SHADOW): block rows only"
    if args.draft_m:
        cfg["draft_m"] = args.draft_m
    if score_only:
        cfg["mode"] = "wino_score_rows alone" + (" with the entropy output" if args.entropy else "")
    if args.graph:
        cfg["launch"] = "CUDA graph of %d consecutive steps, replayed %d times" % (args.graph, args.steps // args.graph)
    if args.compact:
        cfg["compact"] = "rows scored per step: %d of %d (WINO_OPT_COMPACT); value counts all %d" % (
            w.N // 2, w.N, w.N)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_max / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": cfg,
        "roofline": {**{k: roof[k] for k in ("bound", "achieved", "peak", "unit", "frac")},
                     "traffic": ncu_traffic(w.name, layout), "kernel": "score_kernel (fused LM-head GEMM + online vocab softmax)",
                     **{k: v for k, v in roof.items() if k not in ("bound", "achieved", "peak", "unit", "frac")},
                     "launches_timed": score_n, "peak_source": peak_src,
                     "timing": "per-launch CUDA events around the score kernel over a second region of K steps"},
        "step_roofline_frac": max(t_flop, w_bytes / (peaks["hbm_gbs"] * 1e9)) / step_s,
        "tflops_per_step": flops / step_s / 1e12,
        "e2e": None if not e2e_steps else {
            "value": job_rows_per_s(w.N, e2e_steps, world, te), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": 1e3 * te / e2e_steps},
        "gpu_launches": (3 if args.compact and not score_only else 2) * args.steps,  # (gather +) score + finish
        "clocks": clock_info,
        "w_layout": W_LAYOUTS[layout],
        "cpu_baseline": cpu,
        "parity": parity,
        "configs": configs,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def run_loop(args):
    """The whole semi-autoregressive decode of a workload (config 5: B = 16, gen 256 in 8 blocks of 32),
    until no MASK remains, through the loop driver: every step is one wino_step plus the host read of
    the counts that decides whether the block is done.  The hidden states of each global step (the
    model's forward is outside this library) are drawn once, in an untimed first pass, and kept in
    device memory; the timed pass replays the same decode from the same initial state."""
    import numpy as np
    import torch

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    from paper_2605_16941_gb300 import build as pkg_build
    pkg_build.build()
    import paper_2605_16941_gb300 as wino
    import paper_2605_16941_gb300.loop as loop
    import wino_synth as ws

    w = ws.WORKLOADS[args.workload]
    if args.no_shadow:  # WINO+ inference: block rows only
        import dataclasses
        w = dataclasses.replace(w, shadow=False)
    W = ws.weights(w)
    st = ws.initial_state(w)

    def to_dev(a):
        a = np.ascontiguousarray(a)
        return torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).to(dev)

    Wd = lm_head(wino, to_dev(W), args.w_layout)
    cache = {}

    def hidden(k, b0):
        if k not in cache:
            st.blk_start = b0
            cache[k] = to_dev(ws.hidden_states(w, W, st, step=k))
        return cache[k]

    driver = loop.decode if args.python_loop else loop.decode_native

    def run():
        tok = to_dev(st.tokens)
        stats = driver(Wd, tok, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks,
                       tau1=w.tau1, tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, max_steps=4096,
                       compact=args.compact, no_shadow=args.no_shadow, draft_m=args.draft_m,
                       skip_finished=args.skip_finished, w_panels=args.w_layout == "panels")
        return stats, tok

    t_gen = time.time()
    first, tok1 = run()  # draws and caches every step's hidden states
    log(f"[loop] first pass: {first.total_steps} steps, {time.time() - t_gen:.1f} s with input generation")
    runs = []
    for _ in range(max(1, args.loop_repeats)):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        stats, tok = run()
        torch.cuda.synchronize(dev)
        runs.append(time.perf_counter() - t0)
        assert stats.total_steps == first.total_steps and torch.equal(tok, tok1), "the replay diverged"
    t = sorted(runs)[len(runs) // 2]
    final = tok.cpu().numpy()
    assert not (final[:, w.prompt_len:] == w.mask_id).any()
    rows = w.N * stats.total_steps  # rows of H the decode scored (2 per position per step)
    line = {
        "metric": METRIC, "mode": "decode_loop", "value": rows / t, "unit": UNIT, "n_gpus": 1,
        "steps": stats.total_steps, "ms_per_step": 1e3 * t / stats.total_steps, "seconds": t,
        "higher_is_better": True, "dtype": "bf16", "data": "synthetic", "config": config_dict(w),
        "w_layout": W_LAYOUTS[args.w_layout], "loop": {"reading": "bias U[0, 4 + 0.5 k] with k the global step index; a sequence whose block has no "
                            "MASK is frozen until the batch's block is done",
                 "steps_per_block": [b.steps for b in stats.blocks],
                 "drafted_per_block": [b.drafted for b in stats.blocks],
                 "remasked_per_block": [b.remasked for b in stats.blocks],
                 "fallback_drafts_per_block": [b.fallback for b in stats.blocks],
                 "total_steps": stats.total_steps, "repeats": len(runs),
                 "rows_scored": stats.rows_scored, "rows_all_sequences": rows,
                 "timing": "wall clock around the whole decode (median of the repeats); hidden states resident "
                           "in device memory; includes the per-step counts read-back the loop needs",
                 "driver": "Python loop (loop.decode)" if args.python_loop else "library loop (wino_decode)"},
    }
    if args.compact:
        line["config"]["compact"] = "rows scored per step: %d of %d (WINO_OPT_COMPACT); value counts all %d" % (
            w.N // 2, w.N, w.N)
    if args.no_shadow:
        line["config"]["no_shadow"] = "WINO+ inference (WINO_OPT_NO_SHADOW): block rows only"
    if args.draft_m:
        line["config"]["draft_m"] = args.draft_m
    if args.skip_finished:
        line["config"]["skip_finished"] = ("only sequences whose block still has a MASK are scored (%d of %d rows); "
                                           "value counts all sequences' rows" % (stats.rows_scored, rows))
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["wino", "reference"], default="wino")
    ap.add_argument("--workload", default="unified_b4")
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="skip the oracle legs (CPU baseline and whole-step parity)")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the timing of the other LLaDA-shaped configurations")
    ap.add_argument("--compact", action="store_true",
                    help="row compaction: score only the row each position's update reads (not the headline: "
                         "the metric counts all 2*n_seq*blk_len rows)")
    ap.add_argument("--no-shadow", action="store_true", help="WINO+ inference step: block rows only")
    ap.add_argument("--draft-m", type=int, default=0, help="fixed-M drafting (naive parallel sampling)")
    ap.add_argument("--score-rows", action="store_true", help="time wino_score_rows alone instead of the step")
    ap.add_argument("--entropy", action="store_true", help="time wino_score_rows with the entropy output")
    ap.add_argument("--graph", type=int, default=0,
                    help="capture this many consecutive steps in a CUDA graph and time its replays")
    ap.add_argument("--loop", action="store_true",
                    help="time the workload's whole decode loop (until no MASK is left) instead of K steps")
    ap.add_argument("--loop-repeats", type=int, default=3)
    ap.add_argument("--skip-finished", action="store_true",
                    help="with --loop: score only the sequences whose block still has a MASK")
    ap.add_argument("--python-loop", action="store_true",
                    help="with --loop: step from the Python driver (loop.decode) instead of the library's loop")
    ap.add_argument("--w-layout", choices=sorted(W_LAYOUTS), default="panels",
                    help="LM head layout the steps read (wino_score_rows always reads row-major W)")
    ap.add_argument("--cpu-budget-s", type=float, default=15.0)
    ap.add_argument("--ref-budget-s", type=float, default=90.0)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args)
        return
    if args.loop:
        if world > 1:
            ap.error("--loop runs on one GPU")
        run_loop(args)
        return
    run_wino(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
