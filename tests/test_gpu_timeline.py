"""Timeline of the score kernel (per-CTA %globaltimer stamps, off by default), on steps run back to
back: the spread of the CTA pairs' finish times against their tile counts, the time before the first
tile's copies are issued, and the drain after the last MMA, at the single-sequence LLaDA shape (N = 256,
bandwidth-bound) and at N = 2048 (tensor-bound).  Also checks the work split: one CTA per SM, every
(row block, vocabulary tile) computed exactly once, tile counts within one of each other in a group.

With WINO_TIMELINE_RECORD=<path> the per-launch summaries are appended to that file as JSON lines.
"""
import json
import os

import numpy as np
import pytest
import torch

import wino_synth as ws

pytestmark = pytest.mark.gpu

SLOTS = 256  # CTA slots per launch in the buffer (the grid is at most one CTA per SM)


def _run(name, launches=8):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev
    w = ws.WORKLOADS[name]
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = dev(W)
    Hd = [dev(ws.hidden_states(w, W, st, step=k)) for k in range(2)]
    tok = dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    wsp = wino.workspace(w.N, w.d, w.V)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
    for i in range(3):  # warm-up outside the timeline
        wino.wino_step(Hd[i % 2], Wd, tok, p, counts, wsp)
    buf = torch.zeros(launches * SLOTS * wino.TIMELINE_WORDS, dtype=torch.int64, device="cuda")
    torch.cuda.synchronize()
    wino.wino_timeline_begin(buf, launches, SLOTS)
    try:
        for i in range(launches):
            wino.wino_step(Hd[i % 2], Wd, tok, p, counts, wsp)
        torch.cuda.synchronize()
    finally:
        n = wino.wino_timeline_end()
    assert n == launches
    assert wino.wino_read_device_status(wsp) == wino.WINO_OK
    plan = wino.wino_score_plan(w.N, w.d, w.V)
    T = buf.view(launches, SLOTS, wino.TIMELINE_WORDS).cpu().numpy().view(np.uint64)
    return w, plan, T


def _summaries(w, plan, T):
    ctas = plan["ctas"]
    out = []
    prev_exit = None
    for l in range(T.shape[0]):
        t = T[l, :ctas].astype(np.int64)
        assert np.all(T[l, ctas:] == 0), "a CTA slot past the grid was written"
        entry, setup, first, dep, last, done, exit_ = (t[:, i] for i in range(7))
        # stamps taken by the same thread (thread 0: entry, set-up, first copy, all done, exit) are ordered;
        # stamps of other warps are compared with them only in the summaries
        assert np.all(entry > 0) and np.all(entry <= setup) and np.all(setup <= first) and np.all(setup <= done)
        assert np.all(done <= exit_) and np.all(last > 0) and np.all(dep > 0)
        sm = (T[l, :ctas, 7] >> np.uint64(32)).astype(np.int64)
        assert len(np.unique(sm[0::2])) == ctas // 2, "two pairs on one SM"
        tiles = (T[l, 0:ctas:2, 7] & np.uint64(0xFFFFFFFF)).astype(np.int64)  # per pair (leader CTAs)
        assert tiles.sum() == plan["n_mb"] * plan["n_vt"], (tiles.sum(), plan)
        groups = plan["n_groups"]
        for g in range(groups):  # pairs of group g: c % groups == g
            tg = tiles[g::groups]
            assert tg.max() - tg.min() <= plan["n_mb"] // groups + 1
        t0, t1 = entry.min(), exit_.max()
        pair_last = last[0::2]
        busiest = tiles == tiles.max()
        rec = {"workload": w.name, "launch": l, "plan": plan, "duration_us": (t1 - t0) / 1e3,
               "entry_spread_us": (entry.max() - t0) / 1e3,
               "first_copy_after_entry_us_median": float(np.median(first - entry)) / 1e3,
               "first_copy_latest_us": (first.max() - t0) / 1e3,
               "last_mma_spread_us": (pair_last.max() - pair_last.min()) / 1e3,
               "last_mma_busiest_pairs_mean_us": float((pair_last[busiest] - t0).mean()) / 1e3,
               "last_mma_other_pairs_mean_us": float((pair_last[~busiest] - t0).mean()) / 1e3 if (~busiest).any()
               else None,
               "drain_after_last_mma_us": (t1 - pair_last.max()) / 1e3,
               "tiles_per_pair": [int(tiles.min()), int(tiles.max())],
               "pairs_with_most_tiles": int(busiest.sum()),
               "idle_cta_share": float(((entry - t0) + (t1 - exit_)).sum() / (ctas * (t1 - t0))),
               "gap_after_previous_launch_us": None if prev_exit is None else (t0 - prev_exit) / 1e3}
        prev_exit = t1
        out.append(rec)
    return out


@pytest.mark.parametrize("name", ["tiny", "llada_b1", "llada_b8"])
def test_score_kernel_timeline(name):
    w, plan, T = _run(name)
    path = os.environ.get("WINO_TIMELINE_RECORD")
    if path:
        np.save(f"{path}.{name}.npy", T)
    recs = _summaries(w, plan, T)
    for r in recs:
        print(json.dumps(r))
        if path:
            with open(path, "a") as f:
                f.write(json.dumps(r) + "\n")


def test_device_plan_matches_host_plan():
    """wino_score_plan on this GPU equals the host-side split for its SM count and resident pairs (all 76
    pairs are used at these shapes, so the device's pair count is what the plan shows)."""
    import paper_2605_16941_gb300 as wino
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for N, V in ((256, 126464), (2048, 134400), (1024, 126464)):
        dev = wino.wino_score_plan(N, 4096, V)
        pairs = dev["ctas"] // 2
        host = wino.wino_score_plan_host(N, 4096, V, sms, pairs)
        assert {k: host[k] for k in dev} == dev, (dev, host)
