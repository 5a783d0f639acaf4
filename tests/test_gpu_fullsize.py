"""Whole-step parity at the full benchmark sizes, every row against the fp64 oracle.

* LLaDA head shape, 8 sequences (N = 2048, d = 4096, V = 126464), tau1 in {0.5, 0.7, 0.9};
* unified text+image vocabulary, 4 sequences of 256 + 256 rows (N = 2048, V = 134400);
* the 16-sequence decode loop (N = 1024 per step): the first step of every one of its 8 blocks.

Each workload is run as specified and, for the single-step ones, as its coverage variant (doubled
biases, half of the pre-decoded positions holding their planted token), where threshold drafts
(Eq. 2), verified keeps and re-masks (Eq. 3) all occur and tau1 changes the draft set.  The oracle
scores every row once per workload; its statistics do not depend on the thresholds, so Eq. 4 is then
applied by the oracle for each tau1.  Tolerances are those of ``gpu_helpers``: per-row probabilities
within 1e-3 absolute, argmax and token state bit-exact outside the counted near-tie positions.

With WINO_PARITY_RECORD=<path> every comparison appends one JSON line (workload, tau1, rows, largest
probability differences, near-tie and flagged-position counts, branch counts) to that file.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
import wino_synth as ws

pytestmark = pytest.mark.gpu


def _record(**kw):
    path = os.environ.get("WINO_PARITY_RECORD")
    print(json.dumps(kw))
    if path:
        with open(path, "a") as f:
            f.write(json.dumps(kw) + "\n")


def _step_result(st, w, o, tau1, **kw):
    """The oracle's Eq. 4 from its own fp64 statistics: oracle.step without re-scoring the rows."""
    tok, cnt, fl = oracle.draft_verify(st.tokens, st.blk_start, w.blk_len, w.mask_id, tau1, w.tau2, o.argmax,
                                       o.pmax, o.ptarget, **kw)
    return oracle.StepResult(tok, cnt, fl, o.argmax, o.pmax, o.ptarget, o.gap)


def _gpu_stats_and_steps(w, Wd, st, H, taus):
    """The GPU's statistics of every row (wino_score_rows with the step's targets) and, per tau1, the
    whole wino_step and wino_draft_verify on those statistics."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, gpu_score, host
    t = oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id)
    Hd = dev(H)
    g = gpu_score(Hd, Wd, t)
    wsp = wino.workspace(w.N, w.d, w.V)
    out = {}
    for tau1 in taus:
        p = wino.make_params(tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
        res = []
        for path in ("step", "decomposed"):
            tok_d = dev(st.tokens)
            counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
            flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
            if path == "step":
                wino.wino_step(Hd, Wd, tok_d, p, counts, wsp, flags=flags)
            else:
                wino.wino_draft_verify(tok_d, dev(g.argmax), dev(g.pmax), dev(g.ptarget), p, counts, flags)
            torch.cuda.synchronize()
            res.append((host(tok_d), host(counts), host(flags)))
        assert wino.wino_read_device_status(wsp) == wino.WINO_OK
        out[tau1] = res
    return t, g, out


def _whole_step(name, variant, taus):
    from gpu_helpers import compare_rows, compare_step, dev, f32
    w = ws.WORKLOADS[name]
    w = ws.coverage_variant(w) if variant == "coverage" else w
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    t, g, gpu = _gpu_stats_and_steps(w, Wd, st, H, taus)
    o = oracle.score_rows(H, W, t)  # every row, fp64
    rows = compare_rows(o, g)
    drafts = {}
    for tau1 in taus:
        (tok, cnt, fl), (tok2, cnt2, fl2) = gpu[tau1]
        # one launch or two: the same state; and exactly the oracle's Eq. 4 on the GPU's own statistics
        assert np.array_equal(tok, tok2) and np.array_equal(cnt, cnt2) and np.array_equal(fl, fl2)
        ref = oracle.draft_verify(st.tokens, st.blk_start, w.blk_len, w.mask_id, f32(tau1), f32(w.tau2),
                                  g.argmax, g.pmax.astype(np.float64), g.ptarget.astype(np.float64))
        assert np.array_equal(tok, ref[0]) and np.array_equal(cnt, ref[1]) and np.array_equal(fl, ref[2])
        # the whole step against the oracle's whole step (its own fp64 statistics)
        ostep = _step_result(st, w, o, tau1)
        rep = compare_step(st.tokens, tok, cnt, ostep, st.blk_start, w.blk_len, w.mask_id, tau1, w.tau2)
        _record(test="whole_step", workload=w.name, tau1=tau1, tau2=w.tau2, **rows, **rep)
        drafts[tau1] = ostep.flags == oracle.FLAG_DRAFT
        if variant == "coverage":
            assert rep["threshold_drafts"] > 0 and rep["kept_decoded"] > 0 and rep["remasked"] > 0, rep
    if variant == "coverage" and len(taus) > 1:
        for a in taus:
            for b in taus:
                if a < b:  # a lower threshold drafts a strict superset here
                    assert drafts[b].sum() < drafts[a].sum() and not (drafts[b] & ~drafts[a]).any()


@pytest.mark.parametrize("variant", ["base", "coverage"])
def test_llada_b8_whole_step(variant):
    """N = 2048 rows on the LLaDA head shape, tau1 swept over {0.5, 0.7, 0.9}."""
    _whole_step("llada_b8", variant, (0.5, 0.7, 0.9))


@pytest.mark.parametrize("variant", ["base", "coverage"])
def test_unified_b4_whole_step(variant):
    """N = 2048 rows over the unified vocabulary (V = 134400), the bimodal bias law, tau1 = 0.6
    (and 0.5 / 0.9 on the coverage variant)."""
    _whole_step("unified_b4", variant, (0.6,) if variant == "base" else (0.5, 0.6, 0.9))


def test_decode_loop_b16_block_starts():
    """The 16-sequence decode (gen 256 in 8 blocks of 32, bias U[0, 4 + 0.5 k] at global step k) run to
    the end; invariants on every step; the whole oracle step (all 1024 rows, fp64) on the first step of
    every block; the oracle's Eq. 4 on the GPU's own statistics on a few more steps."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import compare_rows, compare_step, dev, f32, gpu_score, host
    w = ws.WORKLOADS["loop_b16"]
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    rec = {"b0": None}
    eq4_only = {1, 2, 3, 40, 200}
    checked = []

    def hidden(k, b0):
        rec["first"] = b0 != rec["b0"]
        rec["b0"] = b0
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        rec["pre"] = host(tok_d).copy()
        rec["H"] = H
        rec["Hd"] = dev(H)
        return rec["Hd"]

    def on_step(k, b0, counts, flags):
        pre, post = rec["pre"], host(tok_d)
        L = w.blk_len
        outside = np.ones(w.seq_len, bool)
        outside[b0:b0 + L] = False
        assert np.array_equal(post[:, outside], pre[:, outside])
        a, b = pre[:, b0:b0 + L], post[:, b0:b0 + L]
        fl = host(flags)
        assert np.all((b == a) | (a == w.mask_id) | (b == w.mask_id))
        had_mask = (a == w.mask_id).any(1)
        assert np.all((counts[:, 0] >= 1) | ~had_mask | (fl == 4).any(1))
        assert np.array_equal(counts[:, 2], (b == w.mask_id).sum(1))
        if rec["first"]:
            o = oracle.step(rec["H"], W, pre, b0, L, w.mask_id, w.tau1, w.tau2, freeze_finished=True)
            t = oracle.row_targets(pre, b0, L, w.mask_id)
            rows = compare_rows(o, gpu_score(rec["Hd"], Wd, t))
            rep = compare_step(pre, post, counts, o, b0, L, w.mask_id, w.tau1, w.tau2)
            _record(test="loop_block_start", workload=w.name, step=k, blk_start=b0, tau1=w.tau1, tau2=w.tau2,
                    **rows, **rep)
            checked.append(k)
        elif k in eq4_only:
            t = oracle.row_targets(pre, b0, L, w.mask_id)
            g = gpu_score(rec["Hd"], Wd, t)
            ref = oracle.draft_verify(pre, b0, L, w.mask_id, f32(w.tau1), f32(w.tau2), g.argmax,
                                      g.pmax.astype(np.float64), g.ptarget.astype(np.float64), freeze_finished=True)
            assert np.array_equal(post, ref[0]) and np.array_equal(counts, ref[1])

    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=4096)
    final = host(tok_d)
    assert not np.any(final[:, w.prompt_len:] == w.mask_id)
    assert len(checked) == w.n_blocks
    _record(test="loop_summary", workload=w.name, steps_per_block=[b.steps for b in stats.blocks],
            total_steps=stats.total_steps, drafted_per_block=[b.drafted for b in stats.blocks],
            remasked_per_block=[b.remasked for b in stats.blocks], oracle_checked_steps=checked)
