"""GPU parity at the edges of the supported shapes: the largest N, d and V wino_score_rows accepts, and a
step over thousands of sequences.  Rows the oracle cannot score in seconds are sampled (first, last and
random rows); properties that hold for every row are checked on all of them."""
import numpy as np
import pytest
import torch

import oracle
import wino_synth as ws

pytestmark = pytest.mark.gpu


def _every_row(g, V):
    """Range checks on every row of a GPU result."""
    assert np.all((g.argmax >= 0) & (g.argmax < V))
    assert np.all(np.isfinite(g.pmax)) and np.all(np.isfinite(g.ptarget))
    assert np.all((g.pmax >= np.float32(1.0 / V) * np.float32(0.999)) & (g.pmax <= 1.0 + 1e-6))
    assert np.all((g.ptarget >= 0) & (g.ptarget <= g.pmax * (1 + 1e-5) + 1e-12))


def _sample(n, k, seed):
    rows = np.random.default_rng(seed).choice(n, k, replace=False)
    return np.unique(np.concatenate([rows, np.arange(256), np.arange(n - 256, n)]))


def test_score_rows_max_rows():
    """N = 2^24 (the largest N): 65 536 row blocks spread over every SM pair."""
    from gpu_helpers import compare_rows, dev, gpu_score
    N, d, V = 1 << 24, 8, 24
    H = ws.random_bf16(N, d, 1.0, seed=11)
    W = ws.random_bf16(V, d, 1.0, seed=12)
    t = (np.arange(N, dtype=np.int64) * 7 % (V + 1) - 1).astype(np.int32)  # -1 and every id in turn
    g = gpu_score(dev(H), dev(W), t)
    _every_row(g, V)
    rows = _sample(N, 2048, 13)
    rep = compare_rows(oracle.score_rows(H[rows], W, t[rows]), g, rows)
    print(f"N=2^24: {rep}")


def test_score_rows_max_vocabulary():
    """V = 2^27 (the largest vocabulary): 524 288 tiles of 256 columns per row, W = 2 GiB."""
    from gpu_helpers import compare_rows, dev, gpu_score
    N, d, V = 40, 8, 1 << 27
    H = ws.random_bf16(N, d, 1.0, seed=21)
    W = ws.random_bf16(V, d, 2.0, seed=22)  # logits ~ N(0, 32): the maximum stands out over 2^27 entries
    t = np.random.default_rng(23).integers(0, V, size=N).astype(np.int32)
    t[:3] = [0, V - 1, -1]
    g = gpu_score(dev(H), dev(W), t)
    _every_row(g, V)
    rows = np.array([0, 1, 2, 17, 38, 39])
    rows = np.unique(np.concatenate([rows, np.random.default_rng(24).choice(N, 6, replace=False)]))
    # the oracle keeps one fp64 row of V logits per thread (1 GiB each): a few threads only
    o = oracle.score_rows(H[rows], W, t[rows], nthreads=4)
    o_am = o.argmax.copy()
    rep = compare_rows(o, g, rows)
    assert np.all(o.pmax > 1e-3), "the test wants probabilities well above the tolerance"
    print(f"V=2^27: {rep}, pmax {np.round(o.pmax, 4).tolist()}, argmax {o_am.tolist()}")


def test_score_rows_max_dimension():
    """d = 65 536 (the largest hidden size): 1024 K slices per tile, fp32 accumulation over all of them."""
    from gpu_helpers import compare_rows, dev, gpu_score
    N, d, V = 300, 65536, 700
    H = ws.random_bf16(N, d, 1.0, seed=31)
    W = ws.random_bf16(V, d, 2.0 / np.sqrt(d), seed=32)
    t = np.random.default_rng(33).integers(-1, V, size=N).astype(np.int32)
    g = gpu_score(dev(H), dev(W), t, entropy=True)
    rep = compare_rows(oracle.score_rows(H, W, t), g)
    print(f"d=65536: {rep}")


def test_step_many_sequences():
    """One step over 4096 sequences with blocks of 4 (N = 32 768 rows, 4096 Eq. 4 tickets) against the
    whole oracle step."""
    import paper_2605_16941_gb300 as wino
    from gpu_helpers import compare_step, dev, host
    w = ws.Workload("many_seq", d=64, V=1000, n_seq=4096, blk_len=4, bias=((1.0, 0.0, 16.0),), predecoded=0.5,
                    hold=0.5, tau1=0.7, tau2=0.9, prompt_len=3)
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    o = oracle.step(H, W, st.tokens, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2)
    tok_d = dev(st.tokens)
    counts = torch.full((w.n_seq, 3), -9, dtype=torch.int32, device="cuda")
    flags = torch.full((w.n_seq, w.blk_len), -9, dtype=torch.int8, device="cuda")
    p = wino.make_params(w.tau1, w.tau2, w.mask_id, w.n_seq, w.seq_len, st.blk_start, w.blk_len)
    wino.wino_step(dev(H), dev(W), tok_d, p, counts, wino.workspace(w.N, w.d, w.V), flags=flags)
    torch.cuda.synchronize()
    rep = compare_step(st.tokens, host(tok_d), host(counts), o, st.blk_start, w.blk_len, w.mask_id, w.tau1, w.tau2)
    assert rep["drafted"] > 0 and rep["remasked"] > 0 and rep["kept_decoded"] > 0, rep
    print(f"4096 sequences: {rep}")
