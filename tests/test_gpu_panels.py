"""The LM head's panel copy (wino_lm_head_panels, WINO_OPT_W_PANELS).

The copy must be the stated permutation of W, bit for bit, and a step that reads W through it must give the same
bytes as the step over row-major W: the score kernel then multiplies the same operands in the same order, so the
token state, the counts, the flags and the whole workspace (partial softmax records, per-row statistics, status
words) are compared for equality, in single-tile launches (one 256-row block), passes (N = 2048) and
with ragged vocabulary and row tails.  The row-major step itself is compared with the oracle elsewhere."""
import dataclasses

import numpy as np
import pytest
import torch

import wino_synth as ws

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("V,d", [(1000, 64), (300, 128), (129, 192), (126464, 4096)])
def test_panel_copy_is_the_permutation(V, d):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev
    W = dev(ws.random_bf16(V, d, 1.0 / d, seed=11))
    Wp = wino.wino_lm_head_panels(W)
    torch.cuda.synchronize()
    assert Wp.shape == (d // 64, V, 64)
    ref = W.view(V, d // 64, 64).permute(1, 0, 2).contiguous()
    assert torch.equal(Wp.view(torch.int16), ref.view(torch.int16))


def _step_pair(w, H, W, Wp, st, **opts):
    """One step from the same state with row-major W and with the panel copy: (tokens, counts, flags, ws)."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev
    out = []
    for panels, Wx in ((False, W), (True, Wp)):
        p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len,
                             w_panels=panels, **opts)
        tok = dev(st.tokens)
        counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
        flags = torch.zeros((w.n_seq, w.blk_len), dtype=torch.int8, device="cuda")
        wsp = wino.step_workspace(p, w.d, w.V)
        wino.wino_step(H, Wx, tok, p, counts, wsp, flags=flags)
        torch.cuda.synchronize()
        assert wino.wino_read_device_status(wsp) == wino.WINO_OK
        out.append((tok, counts, flags, wsp))
    return out


def _assert_same(a, b):
    for x, y, what in zip(a, b, ("tokens", "counts", "flags", "workspace")):
        assert torch.equal(x, y), f"{what} differ between row-major W and its panel copy"


# tiny (N = 64), a ragged shape (V % 240 and N % 256 both non-zero, three row blocks: tile-pair passes with a
# single-tile remainder), the LLaDA single step (N = 256, bn = 240) and its coverage variant, and the
# unified-vocabulary step (N = 2048, V = 134400, row-pair passes)
RAGGED = ws.Workload("panels_ragged", d=128, V=5003, n_seq=5, blk_len=56, bias=((1.0, 0.0, 9.0),), predecoded=0.4,
                     hold=0.5, tau1=0.6, tau2=0.8)


@pytest.mark.parametrize("name", ["tiny", "ragged", "llada_b1", "llada_b1_cov", "unified_b4"])
def test_step_with_panels_is_bit_identical(name):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev
    w = {"ragged": RAGGED, "llada_b1_cov": ws.coverage_variant(ws.WORKLOADS["llada_b1"])}.get(name) or \
        ws.WORKLOADS[name]
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = dev(W)
    Wp = wino.wino_lm_head_panels(Wd)
    H = dev(ws.hidden_states(w, W, st))
    a, b = _step_pair(w, H, Wd, Wp, st)
    _assert_same(a, b)
    c, e = _step_pair(w, H, Wd, Wp, st, compact=True)  # gathered rows: a different H, the same W path
    _assert_same(c, e)
    print(name, "N", w.N, "plan", wino.wino_score_plan(w.N, w.d, w.V))


def test_static_scratch_and_library_loop_with_panels():
    import paper_2605_16941_gb300 as wino
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev, host
    w = ws.Workload("panels_loop", d=64, V=1000, n_seq=3, blk_len=8, bias=((1.0, 2.0, 6.0),), n_blocks=3,
                    bias_step=0.5, tau1=0.7, tau2=0.9)
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = dev(W)
    Wp = wino.wino_lm_head_panels(Wd)
    H = dev(ws.hidden_states(w, W, st))
    toks = []
    for panels, Wx in ((False, Wd), (True, Wp)):
        p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len,
                             w_panels=panels)
        tok = dev(st.tokens)
        counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
        wino.wino_step_static_scratch(H, Wx, tok, p, counts)
        torch.cuda.synchronize()
        toks.append((host(tok), host(counts)))
    assert np.array_equal(toks[0][0], toks[1][0]) and np.array_equal(toks[0][1], toks[1][1])

    cache = {}

    def hidden(k, b0):
        if (k, b0) not in cache:
            s = ws.initial_state(w)
            s.blk_start = b0
            cache[(k, b0)] = dev(ws.hidden_states(w, W, s, step=k))
        return cache[(k, b0)]
    kw = dict(prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks, tau1=w.tau1, tau2=w.tau2,
              mask_id=w.mask_id, max_steps=400, hidden=hidden)
    tok_a, tok_b = dev(st.tokens), dev(st.tokens)
    ref = loop.decode_native(Wd, tok_a, **kw)
    got = loop.decode_native(Wp, tok_b, w_panels=True, **kw)
    assert np.array_equal(host(tok_a), host(tok_b))
    assert [b.steps for b in got.blocks] == [b.steps for b in ref.blocks]
    got_py = loop.decode(Wp, dev(st.tokens), w_panels=True, **kw)
    assert got_py.total_steps == ref.total_steps


def test_panel_argument_errors():
    """Refused before any launch (every buffer here is a real device allocation)."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev
    W = dev(ws.random_bf16(1000, 128, 1.0 / 128, seed=3))
    with pytest.raises(wino.WinoError) as e:  # in place
        wino.wino_lm_head_panels(W, Wp=W.view(2, 1000, 64))
    assert e.value.status == wino.WINO_ERR_ARG
    buf = torch.empty(1000 * 128 + 8, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wino.WinoError) as e:  # misaligned destination
        wino.wino_lm_head_panels(W, Wp=buf[1:1 + 1000 * 128].view(2, 1000, 64))
    assert e.value.status == wino.WINO_ERR_ARG
    W72 = dev(ws.random_bf16(1000, 72, 1.0 / 72, seed=3))
    with pytest.raises(wino.WinoError) as e:  # d not a multiple of 64
        wino.wino_lm_head_panels(W72, Wp=torch.empty((2, 1000, 64), dtype=torch.bfloat16, device="cuda"))
    assert e.value.status == wino.WINO_ERR_SHAPE
    # a step over a panel copy needs d % 64 == 0 as well
    w = dataclasses.replace(ws.WORKLOADS["tiny"], d=72)
    st = ws.initial_state(w)
    H = dev(ws.random_bf16(w.N, 72, 1.0, seed=4))
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, w_panels=True)
    tok = dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    wsp = wino.step_workspace(p, 72, w.V)
    with pytest.raises(wino.WinoError) as e:
        wino.wino_step(H, W72, tok, p, counts, wsp, d=72, V=1000)
    assert e.value.status == wino.WINO_ERR_SHAPE
