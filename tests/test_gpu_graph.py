"""CUDA graph capture of WINO steps, and steps issued from several host threads on their own streams."""
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


def test_steps_from_two_host_threads_on_two_streams():
    """Two host threads, each stepping its own batch on its own stream with its own workspace, end in the
    states that the same steps reach when run one after the other."""
    import threading

    import paper_2605_16941_gb300 as wino
    from gpu_helpers import dev, host
    ws_a, ws_b = ws.coverage_variant(ws.WORKLOADS["tiny"]), ws.Workload(
        "thread_b", d=128, V=1537, n_seq=3, blk_len=16, bias=((1.0, 0.0, 16.0),), predecoded=0.5, hold=0.5)
    jobs = []
    for w in (ws_a, ws_b):
        W = ws.weights(w)
        st = ws.initial_state(w)
        Hs = [dev(ws.hidden_states(w, W, st, step=k)) for k in range(6)]
        p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
        jobs.append((w, dev(W), st, Hs, p))

    def run(job, stream, out):
        w, Wd, st, Hs, p = job
        tok = dev(st.tokens)
        counts = torch.zeros((w.n_seq, 3), dtype=torch.int32, device="cuda")
        wsp = wino.step_workspace(p, w.d, w.V)
        torch.cuda.synchronize()
        for H in Hs:
            wino.wino_step(H, Wd, tok, p, counts, wsp, stream=stream)
        stream.synchronize()
        out.append((host(tok).copy(), host(counts).copy(), wino.wino_read_device_status(wsp, stream=stream)))

    serial = []
    for job in jobs:
        out = []
        run(job, torch.cuda.current_stream(), out)
        serial.append(out[0])
    outs = [[], []]
    threads = [threading.Thread(target=run, args=(job, torch.cuda.Stream(), outs[i])) for i, job in enumerate(jobs)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    for (t_s, c_s, st_s), o in zip(serial, outs):
        t_p, c_p, st_p = o[0]
        assert st_s == st_p == wino.WINO_OK
        assert np.array_equal(t_s, t_p) and np.array_equal(c_s, c_p)
