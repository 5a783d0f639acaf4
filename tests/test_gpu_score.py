"""GPU parity of wino_score_rows (fused LM head + vocabulary softmax) against the fp64 oracle."""
import numpy as np
import pytest

import oracle
import wino_synth as ws

pytestmark = pytest.mark.gpu

# (N, d, V): tiny; ragged rows, K and vocabulary tails; several tiles each way; minimal; long K
SHAPES = [
    (64, 64, 1000),
    (129, 72, 1001),
    (300, 256, 3000),
    (1, 8, 2),
    (257, 128, 513),
    (128, 4096, 2048),
    (384, 520, 777),
    (100, 64, 19400),   # last pair: one 256-wide tile with 200 valid columns
    (256, 128, 50000),  # several 256-wide tiles per pair and a 128-wide tail tile
    # passes (two or more 256-row blocks), tile-pair sweeps (one row block per group):
    (512, 64, 40000),   # one K slice: the second accumulator's MMAs deferred over a one-stage window
    (520, 8, 300),      # d = 8 (K slice mostly zero fill), ragged last row block
    (2048, 64, 129),    # a vocabulary narrower than one tile: every pass holds a single tile
    (1024, 192, 70000),  # many passes per pair, odd tile counts (a single-tile last pass), ragged vocabulary
    # row-pair sweeps (groups owning two or more row blocks; the third stage slot holds an H box):
    (2400, 64, 5000),   # 5 groups x 2 blocks, bn = 176; the ragged last block is a partner whose second
                        # CTA's rows all lie past N
    (2000, 64, 20000),  # 4 groups x 2 blocks, ragged partner block with rows in both CTAs
    (1300, 64, 20000),  # 2 groups x 3 blocks: a row-pair sweep, then the ragged third block alone
    (3100, 64, 20000),  # 2 groups x 7 / 6 blocks: several row-pair sweeps per pair (records of each sweep)
]


@pytest.mark.parametrize("N,d,V", SHAPES, ids=[f"N{n}_d{d}_V{v}" for n, d, v in SHAPES])
def test_score_rows_matches_oracle(N, d, V):
    from gpu_helpers import compare_rows, dev, gpu_score
    H = ws.random_bf16(N, d, 1.0, seed=N * 7 + d)
    W = ws.random_bf16(V, d, 1.0 / np.sqrt(d), seed=V * 3 + d)
    rng = np.random.default_rng(N + d + V)
    target = rng.integers(-1, V, size=N).astype(np.int32)
    o = oracle.score_rows(H, W, target)
    g = gpu_score(dev(H), dev(W), target)
    rep = compare_rows(o, g)
    ge = gpu_score(dev(H), dev(W), target, entropy=True)  # the entropy variant of the kernel
    compare_rows(o, ge)
    assert np.array_equal(ge.argmax, g.argmax)
    print(f"N={N} d={d} V={V}: {rep}")


def test_score_rows_planted_and_edge_targets():
    """Planted winners, targets at vocabulary index 0 and V-1, no target, targets out of range."""
    from gpu_helpers import compare_rows, dev, gpu_score
    w = ws.Workload("planted", d=128, V=1537, n_seq=3, blk_len=40, bias=((1.0, 0.0, 16.0),), predecoded=0.0)
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=3)
    t = ws.row_targets_planted(w, st)
    t[0], t[1], t[2], t[3], t[4] = 0, w.V - 1, -1, w.V, -5
    o = oracle.score_rows(H, W, np.where((t >= 0) & (t < w.V), t, -1))
    g = gpu_score(dev(H), dev(W), t)
    compare_rows(o, g)
    assert g.ptarget[2] == 0 and g.ptarget[3] == 0 and g.ptarget[4] == 0


def test_score_rows_exact_ties_pick_lowest_index():
    """Duplicate LM-head rows give exactly equal logits; the smaller vocabulary id must win,
    also when the duplicates sit in different vocabulary tiles."""
    from gpu_helpers import dev, gpu_score
    d, V, N = 64, 1200, 16
    W = ws.random_bf16(V, d, 0.05, seed=5)
    H = ws.random_bf16(N, d, 1.0, seed=6)
    top = 700
    # integer-valued row 0 and winner rows: every partial sum is exact in fp32, in any order
    H[0] = ws.f32_to_bf16_bits(np.random.default_rng(9).integers(-4, 5, size=d).astype(np.float32))
    W[top] = H[0]  # a clear winner for row 0 (logit = |h|^2)
    W[3] = W[top]  # same logit at index 3 (tile 0) ...
    W[1100] = W[top]  # ... and 1100 (tile 4)
    H[1] = 0  # every logit 0: argmax must be 0
    o = oracle.score_rows(H, W, None)
    g = gpu_score(dev(H), dev(W), None)
    assert o.argmax[0] == 3 and g.argmax[0] == 3
    assert o.argmax[1] == 0 and g.argmax[1] == 0
    assert abs(g.pmax[1] - 1.0 / V) < 1e-6


def test_score_rows_deterministic():
    from gpu_helpers import dev, gpu_score
    H = ws.random_bf16(300, 256, 1.0, seed=1)
    W = ws.random_bf16(5000, 256, 1 / 16, seed=2)
    t = np.arange(300, dtype=np.int32) * 13 % 5000
    Hd, Wd = dev(H), dev(W)
    a = gpu_score(Hd, Wd, t)
    b = gpu_score(Hd, Wd, t)
    assert np.array_equal(a.argmax, b.argmax)
    assert np.array_equal(a.pmax.view(np.int32), b.pmax.view(np.int32))
    assert np.array_equal(a.ptarget.view(np.int32), b.ptarget.view(np.int32))


@pytest.fixture(scope="module")
def llada_head():
    from gpu_helpers import dev
    w = ws.WORKLOADS["llada_b1"]
    W = ws.weights(w)
    return w, W, dev(W)


def test_score_rows_llada_shape_sampled(llada_head):
    """LLaDA-8B head (d=4096, V=126464) at the bench's N=256 launch; 24 sampled rows against the oracle."""
    from gpu_helpers import compare_rows, dev, gpu_score
    w, W, Wd = llada_head
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    t = ws.row_targets_planted(w, st)
    g = gpu_score(dev(H), Wd, t, entropy=True)
    rows = np.random.default_rng(0).choice(w.N, 24, replace=False)
    rows[:2] = [0, w.N - 1]
    o = oracle.score_rows(H[rows], W, t[rows])
    rep = compare_rows(o, g, rows)
    print(f"llada N=256 sampled: {rep}")
    # properties that hold on every row: probabilities in range, ptarget <= pmax
    assert np.all((g.pmax >= 1.0 / w.V * 0.999) & (g.pmax <= 1.0 + 1e-6))
    assert np.all(g.ptarget <= g.pmax * (1 + 1e-5) + 1e-12)
    assert np.all((g.argmax >= 0) & (g.argmax < w.V))
