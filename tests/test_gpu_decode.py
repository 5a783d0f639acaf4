"""The library's decode loop (wino_decode) against the Python loop driver: the same steps, states,
finalization steps and per-block statistics, in every decoding mode; resume and error paths."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
import wino_synth as ws

pytestmark = pytest.mark.gpu

W_LOOP = ws.Workload("native_loop", d=64, V=1000, n_seq=3, blk_len=8, bias=((1.0, 2.0, 6.0),), n_blocks=3,
                     bias_step=0.5, tau1=0.7, tau2=0.9)


def _setup(w):
    from gpu_helpers import dev
    W = ws.weights(w)
    st = ws.initial_state(w)
    cache = {}

    def hidden(k, b0):
        if (k, b0) not in cache:
            st.blk_start = b0
            cache[(k, b0)] = dev(ws.hidden_states(w, W, st, step=k))
        return cache[(k, b0)]
    return dev(W), st, hidden


def _kw(w, **extra):
    return dict(prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1, tau2=w.tau2,
                mask_id=w.mask_id, max_steps=400, **extra)


@pytest.mark.parametrize("mode", ["wino", "wino_plus", "fixed_m2", "compact"])
def test_native_loop_matches_python_loop(mode):
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    extra = {"wino": {}, "wino_plus": {"no_shadow": True}, "fixed_m2": {"no_shadow": True, "draft_m": 2},
             "compact": {"compact": True}}[mode]
    w = W_LOOP if not extra.get("no_shadow") else dataclasses.replace(W_LOOP, shadow=False)
    Wd, st, hidden = _setup(w)
    tok_py, last_py = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    ref = loop.decode(Wd, tok_py, hidden=hidden, last_change=last_py, **_kw(w, **extra))
    tok_c, last_c = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    got = loop.decode_native(Wd, tok_c, hidden=hidden, last_change=last_c, **_kw(w, **extra))
    assert np.array_equal(host(tok_c), host(tok_py)) and np.array_equal(host(last_c), host(last_py))
    assert [(b.steps, b.drafted, b.remasked, b.fallback) for b in got.blocks] == \
        [(b.steps, b.drafted, b.remasked, b.fallback) for b in ref.blocks]
    assert got.total_steps == ref.total_steps == got.next_step and got.rows_scored == ref.rows_scored
    assert not np.any(host(tok_c)[:, w.prompt_len:] == w.mask_id)
    print(mode, [b.steps for b in got.blocks], "at-least-one drafts", [b.fallback for b in got.blocks])


def test_native_loop_resumes_a_python_checkpoint():
    """Interrupt the Python loop inside block 1, resume the rest with the library's loop: same end state."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    w = W_LOOP
    Wd, st, hidden = _setup(w)
    tok_a, last_a = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    full = loop.decode(Wd, tok_a, hidden=hidden, last_change=last_a, **_kw(w))
    stop_at = full.blocks[0].steps + min(1, full.blocks[1].steps - 1)  # inside block 1

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
        loop.decode(Wd, tok_b, hidden=hidden, last_change=last_b, on_step=on_step, **_kw(w))
    b, k = saved["at"]
    tok_c, last_c = dev(saved["tok"]), dev(saved["last"])
    rest = loop.decode_native(Wd, tok_c, hidden=hidden, last_change=last_c, start_block=b, start_step=k, **_kw(w))
    assert np.array_equal(host(tok_c), host(tok_a)) and np.array_equal(host(last_c), host(last_a))
    assert rest.next_step == full.next_step


def test_native_loop_errors():
    import paper_2605_16941_gb300 as wino
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    w = W_LOOP
    Wd, st, hidden = _setup(w)
    # the callback has no hidden states for step 2: the loop stops before it
    tok = dev(st.tokens)
    with pytest.raises(wino.WinoError) as e:
        loop.decode_native(Wd, tok, hidden=lambda k, b0: hidden(k, b0) if k < 2 else None, **_kw(w))
    assert e.value.status == wino.WINO_ERR_ARG
    # an exception raised by the callback comes back as itself
    with pytest.raises(ZeroDivisionError):
        loop.decode_native(Wd, dev(st.tokens), hidden=lambda k, b0: 1 // 0, **_kw(w))
    # a block budget of one step runs out at the first block that needs more
    with pytest.raises(wino.WinoError) as e:
        loop.decode_native(Wd, dev(st.tokens), hidden=hidden, **{**_kw(w), "max_steps": 1})
    assert e.value.status == wino.WINO_ERR_MAX_STEPS
    # the state after the stop equals one Python step from the start
    ref = dev(st.tokens)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, w.prompt_len, w.blk_len,
                         freeze_finished=True, step_index=1)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    wino.wino_step(hidden(0, w.prompt_len), Wd, ref, p, counts, wino.step_workspace(p, w.d, w.V))
    tok1 = dev(st.tokens)
    with pytest.raises(wino.WinoError):
        loop.decode_native(Wd, tok1, hidden=hidden, **{**_kw(w), "max_steps": 1})
    torch.cuda.synchronize()
    assert (host(ref)[:, w.prompt_len:w.prompt_len + w.blk_len] == w.mask_id).any(), "block 0 needs two steps"
    assert np.array_equal(host(tok1), host(ref))


@pytest.mark.parametrize("mode", ["wino", "compact", "wino_plus"])
def test_step_with_an_active_list(mode):
    """A step over a list of sequences (unordered) scores and updates those alone: their results match the
    oracle's step on just those sequences; every other sequence's tokens, counts and flags stay as they were."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import compare_step, dev, host
    base = ws.Workload("active", d=256, V=5000, n_seq=6, blk_len=32, bias=((1.0, 0.0, 10.0),), predecoded=0.5)
    w = ws.coverage_variant(base)
    if mode == "wino_plus":
        w = dataclasses.replace(w, shadow=False)
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=1)
    listed = [4, 1, 3]
    act = dev(np.array(listed, np.int32))
    opts = {"wino": {}, "compact": {"compact": True}, "wino_plus": {"no_shadow": True}}[mode]
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, active_seq=act,
                         **opts)
    tok_d = dev(st.tokens)
    counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    wsp = wino.step_workspace(p, w.d, w.V)
    wino.wino_step(dev(H), dev(W), tok_d, p, counts, wsp, flags=flags)
    torch.cuda.synchronize()
    assert wino.wino_read_device_status(wsp) == wino.WINO_OK
    tok, cnt, fl = host(tok_d), host(counts), host(flags)
    others = [s for s in range(w.n_seq) if s not in listed]
    assert np.array_equal(tok[others], st.tokens[others])
    assert np.all(cnt[others] == -9) and np.all(fl[others] == -9)
    # the oracle's step on the listed sequences alone (rows of each listed sequence, in list order)
    rows_per_seq = w.kinds * w.blk_len
    H_sub = np.concatenate([H[s * rows_per_seq:(s + 1) * rows_per_seq] for s in listed])
    o = oracle.step(H_sub, W, st.tokens[listed], st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2,
                    no_shadow=(mode == "wino_plus"))
    if mode == "wino_plus":  # compare_step reads the [s][kind][l] layout: give it block rows twice
        o = dataclasses.replace(o)
        o.pmax = np.repeat(o.pmax.reshape(len(listed), 1, w.blk_len), 2, axis=1).reshape(-1)
        o.gap = np.repeat(o.gap.reshape(len(listed), 1, w.blk_len), 2, axis=1).reshape(-1)
        o.ptarget = np.ones(2 * len(listed) * w.blk_len)
    rep = compare_step(st.tokens[listed], tok[listed], cnt[listed], o, st.blk_start, w.blk_len, w.mask_id, w.tau1,
                       w.tau2)
    print(mode, rep)


def test_step_active_list_with_a_bad_entry():
    """An out-of-range entry of the list is caught by the kernels' own checks: nothing is read or written for
    it, the valid entries are stepped, and the device status reports WINO_ERR_ARG."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    w = ws.coverage_variant(ws.WORKLOADS["tiny"])
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    act7 = dev(np.array([7], np.int32))  # n_seq is 1: entry 7 is out of range
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, active_seq=act7)
    tok_d = dev(st.tokens)
    counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    wsp = wino.step_workspace(p, w.d, w.V)
    wino.wino_step(dev(H), dev(W), tok_d, p, counts, wsp)
    torch.cuda.synchronize()
    assert wino.wino_read_device_status(wsp) == wino.WINO_ERR_ARG
    assert np.array_equal(host(tok_d), st.tokens) and np.all(host(counts) == -9)


@pytest.mark.parametrize("native", [False, True], ids=["python", "library"])
def test_decode_skipping_finished_sequences(native):
    """Skipping the sequences whose block is done reaches the same states, finalization steps and per-block
    counts as stepping every sequence (frozen), while scoring fewer rows."""
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    w = ws.Workload("skip_loop", d=64, V=1000, n_seq=6, blk_len=8, bias=((1.0, 1.0, 6.0),), n_blocks=3,
                    bias_step=0.4, tau1=0.7, tau2=0.9)
    Wd, st, hidden = _setup(w)
    tok_a, last_a = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    ref = loop.decode(Wd, tok_a, hidden=hidden, last_change=last_a, **_kw(w))
    drive = loop.decode_native if native else loop.decode
    tok_b, last_b = dev(st.tokens), torch.zeros_like(dev(st.tokens))
    got = drive(Wd, tok_b, hidden=hidden, last_change=last_b, skip_finished=True, **_kw(w))
    assert np.array_equal(host(tok_b), host(tok_a)) and np.array_equal(host(last_b), host(last_a))
    assert [(b.steps, b.drafted, b.remasked, b.fallback) for b in got.blocks] == \
        [(b.steps, b.drafted, b.remasked, b.fallback) for b in ref.blocks]
    assert got.rows_scored < ref.rows_scored
    print("rows scored", got.rows_scored, "of", ref.rows_scored)
