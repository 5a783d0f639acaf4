"""Failure detection on the GPU without faulting or hanging it: a bounded device wait that
nothing satisfies gives up, reports WINO_ERR_DEVICE_TIMEOUT, and the context stays usable."""
import time

import numpy as np
import pytest
import torch

import wino_synth as ws

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives():
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    status = torch.full((1,), 12345, dtype=torch.int32, device="cuda")
    t0 = time.time()
    wino.wino_selftest_wait_timeout(status, 20_000_000)  # 20 ms
    torch.cuda.synchronize()
    dt = time.time() - t0
    assert int(status.item()) == wino.WINO_ERR_DEVICE_TIMEOUT
    assert 0.015 < dt < 5.0, dt
    # the context still works: a normal step runs and reports OK
    w = ws.WORKLOADS["tiny"]
    W = ws.weights(w)
    st = ws.initial_state(w)
    tok = dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    wsp = wino.workspace(w.N, w.d, w.V)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
    wino.wino_step(dev(ws.hidden_states(w, W, st)), dev(W), tok, p, counts, wsp)
    torch.cuda.synchronize()
    assert wino.wino_read_device_status(wsp) == wino.WINO_OK
    assert np.all(host(counts) >= 0)


def test_loop_driver_reports_a_device_failure(monkeypatch):
    """A step whose bounded device wait expired reports WINO_ERR_DEVICE_TIMEOUT in every counts entry; the
    decode loop stops there and raises it.  The failing step is a host-side fake (no GPU fault)."""
    import paper_2605_16941_gb300 as wino
    import paper_2605_16941_gb300.loop as loop
    from gpu_helpers import dev
    w = ws.WORKLOADS["tiny"]
    W = ws.weights(w)
    st = ws.initial_state(w)
    real_step = loop.wino_step
    calls = []

    def flaky_step(H, Wt, tokens, p, counts, wsp, flags=None, stream=None):
        calls.append(p.step_index)
        if len(calls) < 3:
            return real_step(H, Wt, tokens, p, counts, wsp, flags=flags, stream=stream)
        counts.fill_(wino.WINO_ERR_DEVICE_TIMEOUT)  # what the finish kernel writes after a timeout

    monkeypatch.setattr(loop, "wino_step", flaky_step)
    with pytest.raises(wino.WinoError) as e:
        loop.decode(dev(W), dev(st.tokens), prompt_len=w.prompt_len, blk_len=w.blk_len, n_blocks=w.n_blocks,
                     tau1=w.tau1, tau2=w.tau2, mask_id=w.mask_id,
                     hidden=lambda k, b0: dev(ws.hidden_states(w, W, st, step=k)))
    assert e.value.status == wino.WINO_ERR_DEVICE_TIMEOUT and calls == [1, 2, 3]


def test_failure_status_reaches_the_host_once_and_is_cleared():
    """The status words at the start of a workspace: an error recorded for a call (planted here on the
    host, as a score-kernel CTA would record a timeout) makes that call's finish kernel leave the token
    state alone, write the status into every counts entry and publish it for wino_read_device_status;
    the next call starts clean and runs normally."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    w = ws.WORKLOADS["tiny"]
    W = ws.weights(w)
    st = ws.initial_state(w)
    Hd, Wd = dev(ws.hidden_states(w, W, st)), dev(W)
    wsp = wino.workspace(w.N, w.d, w.V)
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
    tok = dev(st.tokens)
    counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
    wsp[:4].view(torch.int32).fill_(wino.WINO_ERR_DEVICE_TIMEOUT)  # the word errors of the call in flight go to
    wino.wino_step(Hd, Wd, tok, p, counts, wsp)
    assert wino.wino_read_device_status(wsp) == wino.WINO_ERR_DEVICE_TIMEOUT
    assert np.all(host(counts) == wino.WINO_ERR_DEVICE_TIMEOUT)
    assert np.array_equal(host(tok), st.tokens)
    wino.wino_step(Hd, Wd, tok, p, counts, wsp)
    assert wino.wino_read_device_status(wsp) == wino.WINO_OK
    assert np.all(host(counts) >= 0) and not np.array_equal(host(tok), st.tokens)
