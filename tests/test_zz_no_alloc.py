"""wino_step_static_scratch: the step for callers that cannot allocate device memory (an
inference-server plugin that only receives its input and output buffers, a process whose memory
pool owns all device memory, a decode loop that must not call cudaMalloc or cudaFree while it
runs).  It must give exactly what wino_step gives with a caller workspace, call after call, up to
the size the fixed array holds (wino_workspace_size_step <= WINO_STATIC_SCRATCH_BYTES), refuse
anything larger before launching, and leave the device's free memory unchanged.  This file sorts
last so that a run stopping at the first failure has already run every other test; it also passes
alone in a fresh process."""
import ctypes as C

import numpy as np
import pytest
import torch

import wino_synth as ws

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wino():
    from paper_2605_16941_gb300 import build
    build.build()
    import paper_2605_16941_gb300 as w
    return w


def _dev(a):
    a = np.ascontiguousarray(a)
    return torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).cuda()


def _params(wino, w, st, **opts):
    return wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, **opts)


def _same_as_wino_step(wino, w, calls=2, **opts):
    """Run `calls` consecutive steps through wino_step (caller workspace) and through the fixed array,
    each from its own copy of the state, and require identical tokens, counts and flags after each."""
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = _dev(W)
    tok_ref, tok_new = _dev(st.tokens), _dev(st.tokens)
    cnt_ref = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    cnt_new = cnt_ref.clone()
    fl_ref = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    fl_new = fl_ref.clone()
    p = _params(wino, w, st, **opts)
    assert wino.wino_workspace_size_step(p, w.d, w.V) <= wino.WINO_STATIC_SCRATCH_BYTES
    wsp = wino.step_workspace(p, w.d, w.V)
    for k in range(calls):  # the fixed scratch keeps the previous call's contents
        Hd = _dev(ws.hidden_states(w, W, st, step=k))
        wino.wino_step(Hd, Wd, tok_ref, p, cnt_ref, wsp, flags=fl_ref)
        wino.wino_step_static_scratch(Hd, Wd, tok_new, p, cnt_new, flags=fl_new)
        torch.cuda.synchronize()
        assert torch.equal(tok_new, tok_ref), f"token state differs after call {k}"
        assert torch.equal(cnt_new, cnt_ref), f"counts differ after call {k}"
        assert torch.equal(fl_new, fl_ref), f"flags differ after call {k}"
        assert int((cnt_ref >= 0).all()) == 1
    return int(cnt_ref[:, 0].sum()), int(cnt_ref[:, 1].sum())


@pytest.mark.parametrize("name", ["tiny", "llada_b1"])
@pytest.mark.parametrize("mode", ["plain", "compact", "no_shadow"])
def test_static_scratch_step_matches_wino_step(wino, name, mode):
    w = ws.coverage_variant(ws.WORKLOADS[name])
    if mode == "no_shadow":
        import dataclasses
        w = dataclasses.replace(w, shadow=False)
    _same_as_wino_step(wino, w, compact=(mode == "compact"), no_shadow=(mode == "no_shadow"))


# The largest problems the 16 MiB array holds at V = 126464: 4080 scored rows plain (63 sequences of
# 32 + 32 rows = 4032), 1363 scored rows with compaction at d = 4096 (42 sequences of 32 = 1344).
LIMIT_PLAIN = ws.Workload("limit_plain_d256_V126464_B63_L32", d=256, V=126464, n_seq=63, blk_len=32,
                          bias=((1.0, 0.0, 20.0),), predecoded=0.5, hold=0.5)
LIMIT_COMPACT = ws.Workload("limit_compact_d4096_V126464_B42_L32", d=4096, V=126464, n_seq=42, blk_len=32,
                            bias=((1.0, 0.0, 20.0),), predecoded=0.5, hold=0.5)


@pytest.mark.parametrize("w,compact", [(LIMIT_PLAIN, False), (LIMIT_COMPACT, True)], ids=["plain", "compact"])
def test_static_scratch_at_its_limit(wino, w, compact):
    """The largest accepted sequence count (at 32 positions per block) runs and matches wino_step; one
    sequence more is refused."""
    import dataclasses
    drafted, remasked = _same_as_wino_step(wino, w, compact=compact)
    assert drafted > 0 and remasked > 0
    bigger = dataclasses.replace(w, n_seq=w.n_seq + 1)
    st = ws.initial_state(bigger)
    p = _params(wino, bigger, st, compact=compact)
    assert wino.wino_workspace_size_step(p, w.d, w.V) > wino.WINO_STATIC_SCRATCH_BYTES
    H = torch.zeros((bigger.N, w.d), dtype=torch.int16, device="cuda")
    W = torch.zeros((w.V, w.d), dtype=torch.int16, device="cuda")
    tok = _dev(st.tokens)
    counts = torch.full((bigger.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    rc = wino.lib().wino_step_static_scratch(H.data_ptr(), W.data_ptr(), w.d, w.V, tok.data_ptr(), C.byref(p),
                                             counts.data_ptr(), None, None)
    torch.cuda.synchronize()
    assert rc == wino.WINO_ERR_WORKSPACE
    assert torch.equal(tok, _dev(st.tokens)) and int((counts == -9).all()) == 1  # nothing ran


def test_static_scratch_allocates_nothing(wino):
    """After a first call (which loads the module and looks up the array), further calls leave the
    device's free memory exactly as it was."""
    w = ws.WORKLOADS["llada_b1"]
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = _dev(W)
    Hd = _dev(ws.hidden_states(w, W, st))
    tok = _dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    p = _params(wino, w, st)
    wino.wino_step_static_scratch(Hd, Wd, tok, p, counts)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        wino.wino_step_static_scratch(Hd, Wd, tok, p, counts)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, (free0, free1)
