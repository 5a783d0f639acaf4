"""GPU parity of wino_draft_verify / wino_step / the decode loop against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
import wino_synth as ws

pytestmark = pytest.mark.gpu


def _random_case(rng, n_seq, L, S, b0, M):
    tokens = rng.integers(0, M + 1, size=(n_seq, S)).astype(np.int32)
    tokens[rng.random((n_seq, S)) < 0.4] = M
    N = n_seq * 2 * L
    am = rng.integers(0, M + 1, size=N).astype(np.int32)  # includes MASK itself now and then
    pm = rng.random(N).astype(np.float32)
    pt = rng.random(N).astype(np.float32)
    pm[rng.random(N) < 0.05] = np.float32(0.5)  # exact threshold hits
    pt[rng.random(N) < 0.05] = np.float32(0.75)
    return tokens, am, pm, pt


CASES = [(1, 1, 3, 1), (1, 32, 40, 4), (5, 31, 70, 2), (17, 33, 100, 50), (3, 128, 300, 100), (4, 256, 600, 0),
         (2, 1024, 1030, 3)]


@pytest.mark.parametrize("n_seq,L,S,b0", CASES, ids=[f"B{c[0]}_L{c[1]}" for c in CASES])
@pytest.mark.parametrize("taus", [(0.5, 0.75), (0.7, 0.9), (1.0, 0.0), (0.0, 1.0)], ids=str)
@pytest.mark.parametrize("freeze", [False, True], ids=["eq4", "freeze"])
def test_draft_verify_bit_exact(n_seq, L, S, b0, taus, freeze):
    """Given the same fp32 statistics, the kernel's Eq. 4 equals the oracle's bit for bit."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, f32, host
    M = 997
    rng = np.random.default_rng(n_seq * 1000 + L)
    tokens, am, pm, pt = _random_case(rng, n_seq, L, S, b0, M)
    if freeze and n_seq > 1:
        tokens[0, b0:b0 + L] = rng.integers(0, M, size=L)  # a finished block
    t1, t2 = taus
    last0 = rng.integers(0, 5, size=(n_seq, S)).astype(np.int32)
    ref_last = last0.copy()
    ref_tok, ref_cnt, ref_fl = oracle.draft_verify(tokens, b0, L, M, f32(t1), f32(t2), am, pm.astype(np.float64),
                                                   pt.astype(np.float64), freeze_finished=freeze, step_index=7,
                                                   last_change=ref_last)
    tok_d = dev(tokens)
    last_d = dev(last0)
    counts = torch.full((n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((n_seq, L), -9, dtype=torch.int8, device="cuda")
    p = wino.make_params(t1, t2, M, n_seq, S, b0, L, freeze_finished=freeze, step_index=7, last_change=last_d)
    wino.wino_draft_verify(tok_d, dev(am), dev(pm), dev(pt), p, counts, flags)
    torch.cuda.synchronize()
    assert np.array_equal(host(tok_d), ref_tok)
    assert np.array_equal(host(counts), ref_cnt)
    assert np.array_equal(host(flags), ref_fl)
    assert np.array_equal(host(last_d), ref_last)


def _gpu_step(w, Wd, tokens, H, blk_start, tau1=None):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    tau1 = w.tau1 if tau1 is None else tau1
    tok_d = dev(tokens)
    counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    ws_ = wino.workspace(w.N, w.d, w.V)
    p = wino.make_params(tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, blk_start, w.blk_len)
    wino.wino_step(dev(H), Wd, tok_d, p, counts, ws_, flags=flags)
    torch.cuda.synchronize()
    return host(tok_d), host(counts), host(flags)


def _gpu_decomposed(w, Wd, tokens, H, blk_start, tau1):
    """score_rows (targets from the oracle's gather) + draft_verify: the GPU's own statistics."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, gpu_score, host
    t = oracle.row_targets(tokens, blk_start, w.blk_len, w.mask_id)
    g = gpu_score(dev(H), Wd, t)
    tok_d = dev(tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    flags = torch.zeros((w.n_seq, w.blk_len), dtype=torch.int8, device="cuda")
    p = wino.make_params(tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, blk_start, w.blk_len)
    wino.wino_draft_verify(tok_d, dev(g.argmax), dev(g.pmax), dev(g.ptarget), p, counts, flags)
    torch.cuda.synchronize()
    return g, t, host(tok_d), host(counts), host(flags)


def _check_full(w, W, Wd, tau1=None, step=0):
    from gpu_helpers import compare_rows, compare_step
    tau1 = w.tau1 if tau1 is None else tau1
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=step)
    tok, cnt, fl = _gpu_step(w, Wd, st.tokens, H, st.blk_start, tau1)
    o = oracle.step(H, W, st.tokens, st.blk_start, w.blk_len, w.mask_id, tau1, w.tau2)
    rows = compare_rows(o, _gpu_decomposed(w, Wd, st.tokens, H, st.blk_start, tau1)[0])
    rep = compare_step(st.tokens, tok, cnt, o, st.blk_start, w.blk_len, w.mask_id, tau1, w.tau2)
    return rows, rep


@pytest.mark.parametrize("variant", ["base", "coverage"])
def test_step_tiny(variant):
    from gpu_helpers import dev
    w = ws.WORKLOADS["tiny"]
    w = ws.coverage_variant(w) if variant == "coverage" else w
    W = ws.weights(w)
    Wd = dev(W)
    for step in range(4):
        rows, rep = _check_full(w, W, Wd, step=step)
        print(f"tiny/{variant} step {step}: {rows} {rep}")


@pytest.fixture(scope="module")
def llada():
    from gpu_helpers import dev
    w = ws.WORKLOADS["llada_b1"]
    W = ws.weights(w)
    return W, dev(W)


@pytest.mark.parametrize("variant", ["base", "coverage"])
def test_step_llada_b1_full_oracle(llada, variant):
    """N=256, d=4096, V=126464: the whole step against the whole oracle step."""
    W, Wd = llada
    w = ws.WORKLOADS["llada_b1"]
    w = ws.coverage_variant(w) if variant == "coverage" else w
    rows, rep = _check_full(w, W, Wd)
    print(f"llada_b1/{variant}: {rows} {rep}")
    if variant == "coverage":
        assert rep["threshold_drafts"] > 0 and rep["kept_decoded"] > 0 and rep["remasked"] > 0


def test_decode_loop_tiny_lockstep():
    """The tiny workload decoded to the end through the package's loop driver; every step is
    re-run by the oracle from the same pre-step state and compared."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import compare_step, dev, host
    w = ws.Workload("tiny_loop", d=64, V=1000, n_seq=2, blk_len=32, bias=((1.0, 0.0, 6.0),), n_blocks=3,
                    bias_step=0.5, tau1=0.7, tau2=0.9)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    last_d = torch.zeros_like(tok_d)
    record = {}
    traj = [st.tokens.copy()]

    def hidden(k, b0):
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        record["pre"] = host(tok_d).copy()
        record["last_pre"] = host(last_d).copy()
        record["H"] = H
        return dev(H)

    reports = []

    def on_step(k, b0, counts, flags):
        last_ref = record["last_pre"]
        o = oracle.step(record["H"], W, record["pre"], b0, w.blk_len, w.mask_id, w.tau1, w.tau2,
                        freeze_finished=True, step_index=k + 1, last_change=last_ref)
        rep = compare_step(record["pre"], host(tok_d), counts, o, b0, w.blk_len, w.mask_id, w.tau1, w.tau2)
        if rep["flagged_positions"] == 0:  # same decisions: the finalization bookkeeping must agree exactly
            assert np.array_equal(host(last_d), last_ref)
        reports.append(rep)
        traj.append(host(tok_d).copy())

    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=500,
                        last_change=last_d)
    final = host(tok_d)
    assert not np.any(final[:, w.prompt_len:] == w.mask_id)
    assert np.array_equal(final[:, :w.prompt_len], st.tokens[:, :w.prompt_len])
    from oracle_pins import finalization_steps_from_trajectory
    assert np.array_equal(host(last_d), finalization_steps_from_trajectory(traj))  # t_l of Sec. 5.1
    print("tiny loop steps/block", [b.steps for b in stats.blocks], "flagged",
          sum(r["flagged_positions"] for r in reports))


@pytest.mark.parametrize("n_seq,L,S,b0", CASES[:5], ids=[f"B{c[0]}_L{c[1]}" for c in CASES[:5]])
def test_draft_verify_no_shadow_bit_exact(n_seq, L, S, b0):
    """WINO+ inference rule (block rows only, single threshold, no re-mask), ptarget not passed."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, f32, host
    M = 997
    rng = np.random.default_rng(n_seq * 77 + L)
    tokens, _, _, _ = _random_case(rng, n_seq, L, S, b0, M)
    N = n_seq * L
    am = rng.integers(0, M + 1, size=N).astype(np.int32)
    pm = rng.random(N).astype(np.float32)
    pm[rng.random(N) < 0.05] = np.float32(0.75)
    for tau in (0.5, 0.75, 1.0):
        ref_tok, ref_cnt, ref_fl = oracle.draft_verify(tokens, b0, L, M, f32(tau), f32(0.9), am,
                                                       pm.astype(np.float64), None, no_shadow=True)
        tok_d = dev(tokens)
        counts = torch.full((n_seq, 3), -9, dtype=torch.int32, device="cuda")
        flags = torch.full((n_seq, L), -9, dtype=torch.int8, device="cuda")
        p = wino.make_params(tau, 0.9, M, n_seq, S, b0, L, no_shadow=True)
        wino.wino_draft_verify(tok_d, dev(am), dev(pm), None, p, counts, flags)
        torch.cuda.synchronize()
        assert np.array_equal(host(tok_d), ref_tok)
        assert np.array_equal(host(counts), ref_cnt) and np.array_equal(host(flags), ref_fl)
        assert np.all(ref_cnt[:, 1] == 0)


def test_decode_loop_wino_plus_lockstep():
    """WINO+ inference decode (no shadow block, one threshold) through the loop driver, every step
    re-run by the oracle from the same state; finalization steps tracked as well."""
    import dataclasses
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import compare_step, dev, host
    w = ws.Workload("wino_plus_loop", d=128, V=3000, n_seq=3, blk_len=32, bias=((1.0, 0.0, 8.0),), n_blocks=2,
                    bias_step=0.4, tau1=0.8, tau2=0.9, shadow=False)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    last_d = torch.zeros_like(tok_d)
    rec = {}

    def hidden(k, b0):
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        assert H.shape[0] == w.n_seq * w.blk_len
        rec["pre"], rec["H"], rec["last"] = host(tok_d).copy(), H, host(last_d).copy()
        return dev(H)

    reports = []

    def on_step(k, b0, counts, flags):
        o = oracle.step(rec["H"], W, rec["pre"], b0, w.blk_len, w.mask_id, w.tau1, w.tau2, freeze_finished=True,
                        step_index=k + 1, last_change=rec["last"], no_shadow=True)
        ow = dataclasses.replace(o)  # compare_step reads the [s][kind][l] layout: give it block rows twice
        ow.pmax = np.repeat(o.pmax.reshape(w.n_seq, 1, w.blk_len), 2, axis=1).reshape(-1)
        ow.gap = np.repeat(o.gap.reshape(w.n_seq, 1, w.blk_len), 2, axis=1).reshape(-1)
        ow.ptarget = np.ones(2 * w.N)  # never below tau2: no verification decision to flag
        rep = compare_step(rec["pre"], host(tok_d), counts, ow, b0, w.blk_len, w.mask_id, w.tau1, w.tau2)
        assert rep["remasked"] == 0
        if rep["flagged_positions"] == 0:
            assert np.array_equal(host(last_d), rec["last"])
        reports.append(rep)

    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=500,
                        last_change=last_d, no_shadow=True)
    final = host(tok_d)
    assert not np.any(final[:, w.prompt_len:] == w.mask_id)
    assert all(b.remasked == 0 for b in stats.blocks)
    print("WINO+ loop steps/block", [b.steps for b in stats.blocks])


@pytest.mark.parametrize("gen", [256, 512])
def test_decode_loop_full_diffusion_lockstep(gen):
    """Full diffusion decoding (Sec. 6.3.2): one block spanning the whole generation (256 and 512 tokens),
    every step re-run by the oracle from the same state."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import compare_step, dev, host
    # Both ends of the bias law grow: with independent per-step biases a long block only settles once
    # every position clears verification in the same step.
    w = ws.Workload(f"full_diffusion_{gen}", d=128, V=2000, n_seq=2, blk_len=gen, bias=((1.0, 0.0, 8.0),),
                    n_blocks=1, bias_step=0.3, bias_floor_step=0.1, tau1=0.6, tau2=0.9)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    rec = {}

    def hidden(k, b0):
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        rec["pre"], rec["H"] = host(tok_d).copy(), H
        return dev(H)

    reps = []

    def on_step(k, b0, counts, flags):
        o = oracle.step(rec["H"], W, rec["pre"], b0, w.blk_len, w.mask_id, w.tau1, w.tau2, freeze_finished=True)
        reps.append(compare_step(rec["pre"], host(tok_d), counts, o, b0, w.blk_len, w.mask_id, w.tau1, w.tau2))

    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=1, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=400)
    final = host(tok_d)
    assert not np.any(final[:, w.prompt_len:] == w.mask_id)
    print(f"full diffusion gen {gen}: {stats.total_steps} steps, remasked {stats.blocks[0].remasked}, "
          f"flagged {sum(r['flagged_positions'] for r in reps)}")


def _gpu_step_opts(w, Wd, tokens, H, blk_start, compact):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    tok_d = dev(tokens)
    counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, blk_start, w.blk_len, compact=compact)
    wsp = wino.step_workspace(p, w.d, w.V)
    wino.wino_step(dev(H), Wd, tok_d, p, counts, wsp, flags=flags)
    torch.cuda.synchronize()
    assert wino.wino_read_device_status(wsp) == wino.WINO_OK
    return host(tok_d), host(counts), host(flags)


@pytest.mark.parametrize("name", ["tiny_cov", "mid_cov", "llada_b1_cov"])
def test_step_compact_matches_full_step_and_oracle(name):
    """Row compaction scores only the row each position's update reads; the step's result is the same."""
    from gpu_helpers import compare_step, dev
    base = {"tiny_cov": ws.WORKLOADS["tiny"],
            "mid_cov": ws.Workload("mid", d=256, V=5000, n_seq=4, blk_len=64, bias=((1.0, 0.0, 10.0),),
                                   predecoded=0.5),
            "llada_b1_cov": ws.WORKLOADS["llada_b1"]}[name]
    w = ws.coverage_variant(base)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    for step in range(2 if name != "llada_b1_cov" else 1):
        H = ws.hidden_states(w, W, st, step=step)
        tf, cf, ff = _gpu_step_opts(w, Wd, st.tokens, H, st.blk_start, compact=False)
        tc, cc, fc = _gpu_step_opts(w, Wd, st.tokens, H, st.blk_start, compact=True)
        o = oracle.step(H, W, st.tokens, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2)
        rep = compare_step(st.tokens, tc, cc, o, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2)
        if rep["flagged_positions"] == 0:
            assert np.array_equal(tc, tf) and np.array_equal(cc, cf) and np.array_equal(fc, ff)
        print(f"compact {name} step {step}: {rep}")


def test_decode_loop_compact_lockstep():
    """A decode loop with row compaction, every step re-run by the (full) oracle step."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import compare_step, dev, host
    w = ws.Workload("compact_loop", d=64, V=1000, n_seq=2, blk_len=32, bias=((1.0, 0.0, 6.0),), n_blocks=3,
                    bias_step=0.5, tau1=0.7, tau2=0.9)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    rec = {}

    def hidden(k, b0):
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        rec["pre"], rec["H"] = host(tok_d).copy(), H
        return dev(H)

    def on_step(k, b0, counts, flags):
        o = oracle.step(rec["H"], W, rec["pre"], b0, w.blk_len, w.mask_id, w.tau1, w.tau2, freeze_finished=True)
        compare_step(rec["pre"], host(tok_d), counts, o, b0, w.blk_len, w.mask_id, w.tau1, w.tau2)

    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=500, compact=True)
    assert not np.any(host(tok_d)[:, w.prompt_len:] == w.mask_id)
    assert stats.rows_scored == stats.total_steps * w.n_seq * w.blk_len


@pytest.mark.parametrize("n_seq,L,S,b0", CASES, ids=[f"B{c[0]}_L{c[1]}" for c in CASES])
@pytest.mark.parametrize("m", [1, 2, 5, 2000])
@pytest.mark.parametrize("shadow", [True, False], ids=["verify", "no_shadow"])
def test_draft_verify_fixed_m_bit_exact(n_seq, L, S, b0, m, shadow):
    """Fixed-M drafting (naive parallel sampling, Sec. 3) on the same fp32 statistics equals the oracle bit
    for bit, exact ties on a coarse confidence grid included (smallest position first)."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, f32, host
    M = 997
    rng = np.random.default_rng(n_seq * 31 + L + m)
    tokens, am, pm, pt = _random_case(rng, n_seq, L, S, b0, M)
    pm = (np.round(pm * 16) / 16).astype(np.float32)
    if not shadow:  # block rows only
        am = am.reshape(n_seq, 2, L)[:, 0].reshape(-1).copy()
        pm = pm.reshape(n_seq, 2, L)[:, 0].reshape(-1).copy()
        pt = None
    last0 = np.zeros((n_seq, S), np.int32)
    ref_last = last0.copy()
    ref_tok, ref_cnt, ref_fl = oracle.draft_verify(tokens, b0, L, M, f32(0.7), f32(0.9), am, pm.astype(np.float64),
                                                   None if pt is None else pt.astype(np.float64), step_index=3,
                                                   last_change=ref_last, no_shadow=not shadow, draft_m=m)
    tok_d, last_d = dev(tokens), dev(last0)
    counts = torch.full((n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((n_seq, L), -9, dtype=torch.int8, device="cuda")
    p = wino.make_params(0.7, 0.9, M, n_seq, S, b0, L, step_index=3, last_change=last_d, no_shadow=not shadow,
                         draft_m=m)
    wino.wino_draft_verify(tok_d, dev(am), dev(pm), None if pt is None else dev(pt), p, counts, flags)
    torch.cuda.synchronize()
    assert np.array_equal(host(tok_d), ref_tok)
    assert np.array_equal(host(counts), ref_cnt) and np.array_equal(host(flags), ref_fl)
    assert np.array_equal(host(last_d), ref_last)
    masked = (tokens[:, b0:b0 + L] == M).sum(1)
    assert np.array_equal(((ref_fl == 5) | (ref_fl == 4)).sum(1), np.minimum(masked, m))


def test_decode_loop_fixed_m_lockstep():
    """Naive parallel sampling at 2 tokens per step (no shadow block) through the loop driver with the
    whole trajectory recorded: every step re-run by the oracle from the GPU's state, ceil(L_b / 2) steps
    per block, and the finalization steps read off the trajectory equal the in-kernel bookkeeping."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import PROB_TOL, TIE_TOL, dev, host
    from oracle_pins import finalization_steps_from_trajectory
    m = 2
    w = ws.Workload("fixed_m_loop", d=128, V=3000, n_seq=3, blk_len=32, bias=((1.0, 0.0, 8.0),), n_blocks=2,
                    tau1=0.8, tau2=0.9, shadow=False)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    tok_d = dev(st.tokens)
    last_d = torch.zeros_like(tok_d)
    rec = {}
    flagged = [0]
    mask_drafts = [0]

    def hidden(k, b0):
        st.blk_start = b0
        H = ws.hidden_states(w, W, st, step=k)
        rec["pre"], rec["H"] = host(tok_d).copy(), H
        return dev(H)

    def on_step(k, b0, counts, flags):
        o = oracle.step(rec["H"], W, rec["pre"], b0, w.blk_len, w.mask_id, w.tau1, w.tau2, freeze_finished=True,
                        no_shadow=True, draft_m=m)
        got = host(tok_d)
        L = w.blk_len
        for s in range(w.n_seq):
            y = rec["pre"][s, b0:b0 + L]
            masked = y == w.mask_id
            conf = o.pmax.reshape(w.n_seq, L)[s]
            gap = o.gap.reshape(w.n_seq, L)[s]
            c = np.sort(np.where(masked, conf, -np.inf))[::-1]
            boundary_tie = masked.sum() > m and c[m - 1] - c[m] < PROB_TOL
            diff = got[s, b0:b0 + L] != o.tokens[s, b0:b0 + L]
            near = (masked & (gap < TIE_TOL)) | (boundary_tie & masked & (np.abs(conf - c[m - 1]) < PROB_TOL))
            assert not (diff & ~near).any(), (k, s, np.flatnonzero(diff & ~near))
            flagged[0] += int(near.sum())
        mask_drafts[0] += int((host(flags) == 4).sum())

    traj = []
    stats = loop.decode(Wd, tok_d, prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1,
                        tau2=w.tau2, mask_id=w.mask_id, hidden=hidden, on_step=on_step, max_steps=200,
                        last_change=last_d, no_shadow=True, draft_m=m, trajectory=traj)
    final = host(tok_d)
    assert not np.any(final[:, w.prompt_len:] == w.mask_id)
    assert len(traj) == stats.total_steps + 1 and np.array_equal(traj[-1], final)
    assert np.array_equal(traj[0], st.tokens)  # Y^(0): the state before the first step
    assert np.array_equal(finalization_steps_from_trajectory(traj), host(last_d))
    if mask_drafts[0] == 0:
        assert [b.steps for b in stats.blocks] == [-(-w.blk_len // m)] * w.n_blocks
    print("fixed-M loop steps/block", [b.steps for b in stats.blocks], "flagged", flagged[0],
          "drafts whose argmax is MASK", mask_drafts[0])


def test_decode_loop_checkpoint_resume():
    """A decode interrupted after a step and resumed from its checkpoint (token state, finalization
    bookkeeping, resume point) ends in the same state as the uninterrupted decode, with the same steps,
    whether the interruption falls inside a block or at a block's last step."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    w = ws.Workload("resume", d=64, V=1000, n_seq=3, blk_len=8, bias=((1.0, 2.0, 6.0),), n_blocks=3,
                    bias_step=0.5, tau1=0.7, tau2=0.9)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)

    def hidden(k, b0):
        st.blk_start = b0
        return dev(ws.hidden_states(w, W, st, step=k))

    kw = dict(prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1, tau2=w.tau2,
              mask_id=w.mask_id, hidden=hidden, max_steps=400)
    tok_a, last_a = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    ends = []  # per step: did it finish its block?
    full = loop.decode(Wd, tok_a, last_change=last_a,
                       on_step=lambda k, b0, c, f: ends.append(bool((c[:, 2] == 0).all())), **kw)
    block_ends = [k for k, e in enumerate(ends) if e]
    assert len(block_ends) == w.n_blocks and full.next_step == full.total_steps
    for stop_at in sorted({3, block_ends[0], block_ends[1] - 1}):

        class Stop(Exception):
            pass

        saved = {}

        def on_step(k, b0, counts, flags):
            if k == stop_at:
                saved["tok"], saved["last"] = host(tok_b).copy(), host(last_b).copy()
                saved["at"] = loop.resume_point(k, b0, counts, prompt_len=w.prompt_len, blk_len=w.blk_len)
                raise Stop

        tok_b, last_b = dev(st.tokens), torch.zeros_like(dev(st.tokens))
        with pytest.raises(Stop):
            loop.decode(Wd, tok_b, last_change=last_b, on_step=on_step, **kw)
        start_block, start_step = saved["at"]
        tok_c, last_c = dev(saved["tok"]), dev(saved["last"])
        rest = loop.decode(Wd, tok_c, last_change=last_c, start_block=start_block, start_step=start_step, **kw)
        assert np.array_equal(host(tok_c), host(tok_a)) and np.array_equal(host(last_c), host(last_a)), stop_at
        assert start_step + rest.total_steps == full.total_steps and rest.next_step == full.next_step


@pytest.mark.parametrize("name,mode", [("llada_b8", "compact"), ("unified_b4", "compact"), ("llada_b1", "no_shadow"),
                                       ("llada_b8", "no_shadow"), ("llada_b8", "fixed_m4"),
                                       ("unified_b4", "fixed_m4_verify")])
def test_step_modes_full_size(name, mode):
    """The step's other modes at the benchmark configurations' full sizes: row compaction gives the full
    step's result; WINO+ and fixed-M steps equal the oracle's Eq. 4 on the GPU's own statistics, whose
    sampled rows match the oracle's."""
    import dataclasses

    import paper_2605_16941_gb300 as wino
    from gpu_helpers import compare_rows, dev, f32, gpu_score, host
    w = ws.WORKLOADS[name]
    no_shadow = mode in ("no_shadow", "fixed_m4")
    draft_m = 4 if mode.startswith("fixed_m4") else 0
    if no_shadow:
        w = dataclasses.replace(w, shadow=False)
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)

    def step(**opts):
        tok_d = dev(st.tokens)
        counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
        flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
        p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, **opts)
        wsp = wino.step_workspace(p, w.d, w.V)
        wino.wino_step(dev(H), Wd, tok_d, p, counts, wsp, flags=flags)
        torch.cuda.synchronize()
        assert wino.wino_read_device_status(wsp) == wino.WINO_OK
        return host(tok_d), host(counts), host(flags)

    if mode == "compact":
        full = step()
        comp = step(compact=True)
        assert all(np.array_equal(a, b) for a, b in zip(full, comp))
        print(f"{name} compact: drafted {int(comp[1][:, 0].sum())} remasked {int(comp[1][:, 1].sum())}")
        return
    tok, cnt, fl = step(no_shadow=no_shadow, draft_m=draft_m)
    t = None if no_shadow else oracle.row_targets(st.tokens, st.blk_start, w.blk_len, w.mask_id)
    g = gpu_score(dev(H), Wd, t)
    ref = oracle.draft_verify(st.tokens, st.blk_start, w.blk_len, w.mask_id, f32(w.tau1), f32(w.tau2), g.argmax,
                              g.pmax.astype(np.float64), None if no_shadow else g.ptarget.astype(np.float64),
                              no_shadow=no_shadow, draft_m=draft_m)
    assert np.array_equal(tok, ref[0]) and np.array_equal(cnt, ref[1]) and np.array_equal(fl, ref[2])
    rows = np.random.default_rng(5).choice(w.N, 16, replace=False)
    rep = compare_rows(oracle.score_rows(H[rows], W, None if t is None else t[rows]), g, rows)
    if draft_m:
        masked = (st.tokens[:, st.blk_start:st.blk_start + w.blk_len] == w.mask_id).sum(1)
        assert np.array_equal(((fl == 5) | (fl == 4)).sum(1), np.minimum(masked, draft_m))
    print(f"{name} {mode}: {rep} drafted {int(cnt[:, 0].sum())} remasked {int(cnt[:, 1].sum())}")
