"""wino_step_static_scratch: the step for callers that cannot allocate device memory
(an inference-server plugin that only receives its input and output buffers, a process
whose memory pool owns all device memory, a decode loop that must not call cudaMalloc or
cudaFree while it runs).  It must give exactly what wino_step gives with a caller
workspace, call after call.  This file sorts last so that a run stopping at the first
failure has already run every other test; it also passes alone in a fresh process."""
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


@pytest.mark.parametrize("name", ["tiny", "llada_b1"])
def test_static_scratch_step_matches_wino_step(wino, name):
    w = ws.coverage_variant(ws.WORKLOADS[name])
    W = ws.weights(w)
    st = ws.initial_state(w)
    Wd = _dev(W)
    tok_ref, tok_new = _dev(st.tokens), _dev(st.tokens)
    cnt_ref = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    cnt_new = cnt_ref.clone()
    fl_ref = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    fl_new = fl_ref.clone()
    wsp = wino.workspace(w.N, w.d, w.V)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
    for k in range(2):  # two calls in a row: the fixed scratch keeps the previous call's contents
        Hd = _dev(ws.hidden_states(w, W, st, step=k))
        wino.wino_step(Hd, Wd, tok_ref, p, cnt_ref, wsp, flags=fl_ref)
        wino.wino_step_static_scratch(Hd, Wd, tok_new, p, cnt_new, flags=fl_new)
        torch.cuda.synchronize()
        assert torch.equal(tok_new, tok_ref), f"token state differs after call {k}"
        assert torch.equal(cnt_new, cnt_ref), f"counts differ after call {k}"
        assert torch.equal(fl_new, fl_ref), f"flags differ after call {k}"
        assert int((cnt_ref >= 0).all()) == 1


def test_static_scratch_rejects_problems_larger_than_the_array(wino):
    """A problem whose workspace would exceed the fixed array is refused before any launch."""
    V, d, blk_len = 126464, 4096, 1024
    n_seq = 3  # N = 6144 rows > 4080
    assert wino.wino_workspace_size(2 * n_seq * blk_len, d, V) > wino.WINO_STATIC_SCRATCH_BYTES
    p = wino.make_params(0.7, 0.9, V - 1, n_seq, blk_len + 32, 32, blk_len)
    fake = 0x10000  # never dereferenced: the size check comes first
    rc = wino.lib().wino_step_static_scratch(fake, fake, d, V, fake, C.byref(p), fake, None, None)
    assert rc == wino.WINO_ERR_WORKSPACE
