"""A WINO step captured in a CUDA graph replays to the same state as the eagerly launched steps."""
import numpy as np
import pytest
import torch

import wino_synth as ws

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("compact", [False, True], ids=["full", "compact"])
def test_steps_replay_in_a_cuda_graph(compact):
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    w = ws.coverage_variant(ws.WORKLOADS["tiny"])
    W = ws.weights(w)
    Wd = dev(W)
    st = ws.initial_state(w)
    Hs = [dev(ws.hidden_states(w, W, st, step=k)) for k in range(3)]
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len, compact=compact)

    def buffers():
        return (dev(st.tokens), torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda"),
                torch.zeros((w.n_seq, w.blk_len), dtype=torch.int8, device="cuda"), wino.step_workspace(p, w.d, w.V))

    tok_e, cnt_e, fl_e, ws_e = buffers()
    states = []
    for k in range(3):
        wino.wino_step(Hs[k], Wd, tok_e, p, cnt_e, ws_e, flags=fl_e)
        states.append(host(tok_e).copy())
    torch.cuda.synchronize()

    tok_g, cnt_g, fl_g, ws_g = buffers()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for k in range(3):
            wino.wino_step(Hs[k], Wd, tok_g, p, cnt_g, ws_g, flags=fl_g)
    torch.cuda.synchronize()
    assert np.array_equal(host(tok_g), st.tokens), "capturing must not run the steps"
    for _ in range(2):  # replay twice from the initial state
        tok_g.copy_(dev(st.tokens))
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(host(tok_g), states[-1])
        assert np.array_equal(host(cnt_g), host(cnt_e)) and np.array_equal(host(fl_g), host(fl_e))
        assert wino.wino_read_device_status(ws_g) == wino.WINO_OK
    assert not np.array_equal(states[0], st.tokens), "the steps should change the state"
