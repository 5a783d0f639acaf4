"""Pins that tie the fp64 oracle to facts fixed outside it.

Each pin takes an ``oracle.Oracle`` and raises ``AssertionError`` when the
oracle disagrees with what the paper or plain mathematics fixes:

* closed forms (bf16 widening; all-zero hidden state gives the uniform
  distribution over V; one-hot LM-head rows make the logits equal to the
  hidden-state entries, so the statistics equal a library softmax of them);
* exact brute force (logits as exact rationals, softmax in 60-digit mpmath);
* an independent fp64 library path (numpy matmul + scipy logsumexp) on a
  rectangular case, so a transposed operand cannot pass;
* Eq. 4's branches on hand-built states with exactly representable
  probabilities, including the strict comparisons at equality;
* the tau2 = 0 "only draft" ablation (Sec. 6.3.4): verification never fires;
* the tau1 >= 1, tau2 = 0 corner, where Eq. 4 plus the at-least-one rule is
  exactly high-confidence greedy decoding (Eq. 1);
* an exhaustive enumeration of small states checked against the properties
  Eq. 2-4 state (drafts only on MASK, re-masks only on decoded positions,
  each draft/re-mask justified by its threshold, completeness, positions
  outside the block untouched, counts consistent);
* naive parallel sampling (a fixed number M of tokens per step, Sec. 3):
  M = 1 is Eq. 1, the drafted set is the unique size-min(M, #MASK) subset
  that beats every left-out masked position (brute force over all subsets),
  and a block of L_b positions takes ceil(L_b / M) steps (the 256 / 128 / 64
  steps of Sec. 6.3.3 for 1 / 2 / 4 tokens per step).

``tests/test_oracle_pins.py`` runs them on the oracle;
``tests/test_oracle_mutants.py`` checks that planted mistakes fail them.
"""
from __future__ import annotations

import itertools
from fractions import Fraction
from pathlib import Path

import numpy as np

import wino_synth as ws

try:  # mpmath ships with sympy
    import mpmath
except ImportError:  # pragma: no cover
    mpmath = None

MASK_FLAG = {"none": 0, "draft": 1, "fallback": 2, "remask": 3, "draft_is_mask": 4, "draft_top_m": 5}


# ----------------------------------------------------------------------------- scoring

def pin_bf16_widening(O):
    cases = {0x3F80: 1.0, 0xBF80: -1.0, 0x4049: 3.140625, 0x0000: 0.0, 0x0001: 2.0 ** -133,
             0x7F7F: (2 - 2.0 ** -7) * 2.0 ** 127, 0x3C00: 2.0 ** -7, 0xC2F7: -123.5}
    for bits, val in cases.items():
        got = O.bf16_to_double(bits)
        assert got == val, (hex(bits), got, val)


def pin_zero_hidden_is_uniform(O):
    for V, d in ((1000, 64), (7, 8), (1, 16)):
        W = ws.random_bf16(V, d, 1.0, seed=3)
        H = np.zeros((3, d), np.uint16)
        tgt = np.array([V - 1, 0, -1], np.int32)
        r = O.score_rows(H, W, tgt)
        assert np.all(r.argmax == 0), r.argmax
        assert np.all(r.pmax == 1.0 / V), (r.pmax, 1.0 / V)
        assert r.ptarget[0] == 1.0 / V and r.ptarget[1] == 1.0 / V and r.ptarget[2] == 0.0, r.ptarget
        assert np.all(r.maxlogit == 0.0)
        assert np.allclose(r.logz, np.log(V), rtol=0, atol=1e-15)
        assert np.allclose(r.entropy, np.log(V), rtol=1e-13, atol=1e-15)  # the uniform distribution
        if V > 1:
            assert np.all(r.gap == 0.0)


def pin_one_hot_weights(O):
    from scipy.special import softmax
    d, V = 48, 40
    W = np.zeros((V, d), np.uint16)
    W[np.arange(V), np.arange(V)] = 0x3F80  # bf16 1.0
    H = ws.random_bf16(5, d, 2.0, seed=11)
    h = ws.bf16_bits_to_f32(H).astype(np.float64)
    for n in range(H.shape[0]):
        assert np.array_equal(O.logits_row(H[n], W), h[n, :V])
    tgt = np.array([3, 39, 0, -1, 17], np.int32)
    r = O.score_rows(H, W, tgt)
    p = softmax(h[:, :V], axis=1)
    assert np.array_equal(r.argmax, np.argmax(h[:, :V], axis=1).astype(np.int32))
    assert np.allclose(r.pmax, p.max(axis=1), rtol=1e-14, atol=0)
    want_t = np.array([p[n, t] if t >= 0 else 0.0 for n, t in enumerate(tgt)])
    assert np.allclose(r.ptarget, want_t, rtol=1e-14, atol=0)
    from scipy.stats import entropy
    assert np.allclose(r.entropy, entropy(p, axis=1), rtol=1e-12, atol=0)


def _exact_stats(H, W, tgt):
    """Exact rationals for the logits; 60-digit mpmath for the softmax."""
    mpmath.mp.dps = 60
    Hf = [[Fraction(float(x)) for x in row] for row in ws.bf16_bits_to_f32(H).astype(np.float64)]
    Wf = [[Fraction(float(x)) for x in row] for row in ws.bf16_bits_to_f32(W).astype(np.float64)]
    out = []
    for n, hrow in enumerate(Hf):
        logit = [sum((a * b for a, b in zip(hrow, wrow)), Fraction(0)) for wrow in Wf]
        m = max(logit)
        a = logit.index(m)  # first occurrence = smallest index
        rest = [x for i, x in enumerate(logit) if i != a]
        gap = (m - max(rest)) if rest else None
        Z = mpmath.fsum(mpmath.exp(mpmath.mpf(x.numerator) / x.denominator - mpmath.mpf(m.numerator) / m.denominator)
                        for x in logit)
        t = int(tgt[n])
        pt = (mpmath.exp(mpmath.mpf((logit[t] - m).numerator) / (logit[t] - m).denominator) / Z) if 0 <= t < len(
            logit) else mpmath.mpf(0)
        ps = [mpmath.exp(mpmath.mpf((x - m).numerator) / (x - m).denominator) / Z for x in logit]
        ent = -mpmath.fsum(q * mpmath.log(q) for q in ps if q > 0)
        out.append((a, float(1 / Z), float(pt), gap, m, float(ent)))
    return out


def pin_exact_brute_force(O):
    assert mpmath is not None, "mpmath (from sympy) is required for the exact pin"
    rng = np.random.default_rng(7)
    for (N, d, V) in ((6, 5, 7), (4, 9, 13), (3, 16, 3)):
        H = ws.random_bf16(N, d, 1.5, seed=int(rng.integers(1 << 30)))
        W = ws.random_bf16(V, d, 1.0, seed=int(rng.integers(1 << 30)))
        W[V - 1] = W[0]  # an exact tie between vocab 0 and V-1: argmax must pick 0 when they lead
        H[0] = 0  # an all-zero row: every logit ties
        tgt = rng.integers(-1, V, size=N).astype(np.int32)
        r = O.score_rows(H, W, tgt)
        ex = _exact_stats(H, W, tgt)
        for n, (a, pm, pt, gap, m, ent) in enumerate(ex):
            assert abs(r.entropy[n] - ent) <= 1e-12 * max(1.0, ent), (n, r.entropy[n], ent)
            assert r.argmax[n] == a, (n, r.argmax[n], a)
            assert abs(r.pmax[n] - pm) <= 1e-13 * pm, (n, r.pmax[n], pm)
            assert abs(r.ptarget[n] - pt) <= 1e-13 * max(pt, 1e-300), (n, r.ptarget[n], pt)
            assert r.maxlogit[n] == float(m), (n, r.maxlogit[n], float(m))
            if gap is not None:
                assert abs(r.gap[n] - float(gap)) <= 1e-12, (n, r.gap[n], float(gap))


def pin_library_path_rectangular(O):
    from scipy.special import logsumexp
    N, d, V = 37, 96, 1001
    H = ws.random_bf16(N, d, 1.0, seed=21)
    W = ws.random_bf16(V, d, 1.0 / np.sqrt(d), seed=22)
    tgt = np.random.default_rng(5).integers(-1, V, size=N).astype(np.int32)
    r = O.score_rows(H, W, tgt)
    Lg = ws.bf16_bits_to_f32(H).astype(np.float64) @ ws.bf16_bits_to_f32(W).astype(np.float64).T  # [N, V]
    lse = logsumexp(Lg, axis=1)
    assert np.array_equal(r.argmax, Lg.argmax(axis=1).astype(np.int32))
    assert np.allclose(r.pmax, np.exp(Lg.max(axis=1) - lse), rtol=1e-12, atol=0)
    want_t = np.where(tgt >= 0, np.exp(Lg[np.arange(N), np.maximum(tgt, 0)] - lse), 0.0)
    assert np.allclose(r.ptarget, want_t, rtol=1e-12, atol=1e-300)
    assert np.allclose(r.logz, lse, rtol=1e-13, atol=0)
    P = np.exp(Lg - lse[:, None])
    assert np.allclose(r.entropy, -(P * np.log(P)).sum(axis=1), rtol=1e-11, atol=0)
    srt = np.sort(Lg, axis=1)
    assert np.allclose(r.gap, srt[:, -1] - srt[:, -2], rtol=0, atol=1e-12)


def pin_planted_bias_dominates(O):
    w = ws.Workload("pin", d=64, V=1000, n_seq=2, blk_len=8, bias=((1.0, 60.0, 60.0),), predecoded=0.0)
    W = ws.weights(w)
    st = ws.initial_state(w)
    H = ws.hidden_states(w, W, st, step=0)
    t = ws.row_targets_planted(w, st)
    r = O.score_rows(H, W, t)
    assert np.array_equal(r.argmax, t)
    assert np.all(r.pmax > 1 - 1e-6) and np.array_equal(r.ptarget, r.pmax)


def pin_row_targets(O):
    mask = 9
    tokens = np.array([[1, 2, mask, 4, 5, mask, 7],
                       [mask, 3, 3, mask, mask, 0, 8]], np.int32)
    t = O.row_targets(tokens, blk_start=2, blk_len=3, mask_id=mask)
    want = np.array([-1, -1, -1, -1, 4, 5,      # seq 0: block rows, then shadow rows of [mask, 4, 5]
                     -1, -1, -1, 3, -1, -1], np.int32)  # seq 1: [3, mask, mask]
    assert np.array_equal(t, want), t


SCORING_PINS = [pin_bf16_widening, pin_zero_hidden_is_uniform, pin_one_hot_weights, pin_exact_brute_force,
                pin_library_path_rectangular, pin_planted_bias_dominates, pin_row_targets]


# ----------------------------------------------------------------------------- Eq. 4

def _rows(n_seq, L, blk, shd):
    """Assemble [s][kind][l] row arrays from per-sequence block / shadow values."""
    blk = np.asarray(blk).reshape(n_seq, L)
    shd = np.asarray(shd).reshape(n_seq, L)
    return np.stack([blk, shd], axis=1).reshape(-1)


def pin_eq4_hand_cases(O):
    M = 99
    # prompt [5], block of 4, right [M]
    tokens = np.array([[5, M, M, 7, 8, M]], np.int32)
    am = _rows(1, 4, [11, 12, 13, 14], [0, 0, 0, 0])
    pm = _rows(1, 4, [0.75, 0.5, 0.0, 0.0], [0.0, 0.0, 0.0, 0.0])
    pt = _rows(1, 4, [0.0, 0.0, 0.0, 0.0], [0.0, 0.0, 0.875, 0.25])
    tok, cnt, fl = O.draft_verify(tokens, 1, 4, M, 0.5, 0.875, am, pm, pt)
    # l0: 0.75 > 0.5 drafted; l1: 0.5 is not > 0.5; l2: 0.875 is not < 0.875 kept; l3: 0.25 < 0.875 re-masked
    assert tok.tolist() == [[5, 11, M, 7, M, M]], tok
    assert cnt.tolist() == [[1, 1, 2]], cnt
    assert fl.tolist() == [[1, 0, 0, 3]], fl

    # nothing clears tau1 -> the most confident masked position is drafted; ties -> lowest position
    tokens = np.array([[M, 3, M, M, 3]], np.int32)
    am = _rows(1, 5, [20, 21, 22, 23, 24], [0] * 5)
    pm = _rows(1, 5, [0.25, 0.9, 0.5, 0.5, 0.75], [1.0] * 5)  # l1/l4 decoded: their pmax is irrelevant
    pt = _rows(1, 5, [0.0] * 5, [1.0] * 5)
    tok, cnt, fl = O.draft_verify(tokens, 0, 5, M, 0.5, 0.9, am, pm, pt)
    assert tok.tolist() == [[M, 3, 22, M, 3]], tok
    assert cnt.tolist() == [[1, 0, 2]] and fl.tolist() == [[0, 0, 2, 0, 0]], (cnt, fl)

    # a fully decoded block: no draft, no fallback; verification still runs
    tokens = np.array([[1, 2, 3]], np.int32)
    am = _rows(1, 3, [7, 7, 7], [0] * 3)
    pm = _rows(1, 3, [1.0] * 3, [0.0] * 3)
    pt = _rows(1, 3, [0.0] * 3, [0.5, 0.95, 0.0])
    tok, cnt, fl = O.draft_verify(tokens, 0, 3, M, 0.1, 0.9, am, pm, pt)
    assert tok.tolist() == [[M, 2, M]] and cnt.tolist() == [[0, 2, 2]] and fl.tolist() == [[3, 0, 3]]

    # the argmax of a drafted row is MASK itself: the position stays MASK and is not counted
    tokens = np.array([[M, M]], np.int32)
    am = _rows(1, 2, [M, 4], [0, 0])
    pm = _rows(1, 2, [0.95, 0.6], [0.0, 0.0])
    pt = _rows(1, 2, [0.0, 0.0], [0.0, 0.0])
    tok, cnt, fl = O.draft_verify(tokens, 0, 2, M, 0.7, 0.9, am, pm, pt)
    assert tok.tolist() == [[M, M]] and cnt.tolist() == [[0, 0, 2]] and fl.tolist() == [[4, 0]], (tok, cnt, fl)

    # two sequences are independent and rows are [s][kind][l]
    tokens = np.array([[M, 6], [6, M]], np.int32)
    am = _rows(2, 2, [[30, 31], [32, 33]], [[0, 0], [0, 0]])
    pm = _rows(2, 2, [[0.8, 0.0], [0.0, 0.1]], [[0.0, 0.0], [0.0, 0.0]])
    pt = _rows(2, 2, [[0.0, 0.0], [0.0, 0.0]], [[0.0, 0.95], [0.5, 0.0]])
    tok, cnt, fl = O.draft_verify(tokens, 0, 2, M, 0.7, 0.9, am, pm, pt)
    assert tok.tolist() == [[30, 6], [M, 33]], tok
    assert cnt.tolist() == [[1, 0, 0], [1, 1, 1]], cnt


def pin_only_draft_never_remasks(O):
    rng = np.random.default_rng(3)
    n_seq, L, M = 64, 16, 50
    tokens = rng.integers(0, M + 1, size=(n_seq, L + 4)).astype(np.int32)
    N = n_seq * 2 * L
    am = rng.integers(0, M, size=N).astype(np.int32)
    pm = rng.random(N)
    pt = rng.random(N)
    pt[::7] = 0.0
    tok, cnt, fl = O.draft_verify(tokens, 2, L, M, 0.6, 0.0, am, pm, pt)
    assert np.all(cnt[:, 1] == 0) and not np.any(fl == 3)
    blk_old, blk_new = tokens[:, 2:2 + L], tok[:, 2:2 + L]
    assert np.all(blk_new[blk_old != M] == blk_old[blk_old != M])


def pin_greedy_reduction(O):
    """tau1 = 1 (no probability exceeds it) and tau2 = 0: every step is Eq. 1."""
    rng = np.random.default_rng(17)
    n_seq, L, M, P = 5, 12, 1000, 3
    tokens = np.full((n_seq, P + L), M, np.int32)
    tokens[:, :P] = 1
    ref = tokens.copy()
    for k in range(L):
        N = n_seq * 2 * L
        am = rng.integers(0, M, size=N).astype(np.int32)
        pm = np.round(rng.random(N) * 8) / 8  # coarse grid: plenty of exact ties
        pt = rng.random(N)
        tokens, cnt, _ = O.draft_verify(tokens, P, L, M, 1.0, 0.0, am, pm, pt)
        # Eq. 1 written with numpy primitives: most confident masked position, first on ties
        conf = pm.reshape(n_seq, 2, L)[:, 0, :]
        tok_am = am.reshape(n_seq, 2, L)[:, 0, :]
        for s in range(n_seq):
            masked = ref[s, P:] == M
            lstar = int(np.argmax(np.where(masked, conf[s], -np.inf)))
            ref[s, P + lstar] = tok_am[s, lstar]
        assert np.array_equal(tokens, ref), (k, tokens, ref)
        assert np.all(cnt[:, 0] == 1) and np.all(cnt[:, 2] == L - 1 - k)
    assert not np.any(tokens == M)


def pin_eq4_exhaustive_properties(O):
    """Every state of a 3-position block over tokens {0, 1, MASK}, every pair of
    probabilities on a grid that hits the thresholds exactly."""
    L, M, P = 3, 2, 1
    grid = np.array([0.0, 0.25, 0.5, 0.75, 1.0])
    states = np.array(list(itertools.product([0, 1, M], repeat=L)), np.int32)  # 27
    combos = np.array(list(itertools.product(range(len(grid)), repeat=2 * L)))  # pmax blk x3, ptarget shd x3
    n_seq = len(combos)
    for tau1, tau2 in ((0.5, 0.75), (0.25, 0.5), (0.0, 1.0), (0.75, 0.25), (1.0, 0.0)):
        for st in states:
            tokens = np.empty((n_seq, P + L + 1), np.int32)
            tokens[:, 0] = 1
            tokens[:, P:P + L] = st
            tokens[:, -1] = M
            pm_b = grid[combos[:, :L]]
            pt_s = grid[combos[:, L:]]
            am_b = (np.arange(n_seq)[:, None] + np.arange(L)[None, :]) % 2  # alternate 0/1 tokens
            am_b[::5, 1] = M  # some drafted argmaxes are MASK itself
            am = np.stack([am_b, np.zeros_like(am_b)], 1).reshape(-1).astype(np.int32)
            pm = np.stack([pm_b, np.full_like(pm_b, 0.5)], 1).reshape(-1)
            pt = np.stack([np.full_like(pt_s, 0.5), pt_s], 1).reshape(-1)
            tok, cnt, fl = O.draft_verify(tokens, P, L, M, tau1, tau2, am, pm, pt)
            old, new = tokens[:, P:P + L], tok[:, P:P + L]
            assert np.array_equal(tok[:, :P], tokens[:, :P]) and np.array_equal(tok[:, -1], tokens[:, -1])
            is_m = old == M
            clear = is_m & (pm_b > tau1)
            none_clear = ~clear.any(1) & is_m.any(1)
            fb = np.where(is_m, pm_b, -np.inf).argmax(1)
            drafted = clear.copy()
            drafted[none_clear, fb[none_clear]] = True
            remask = ~is_m & (pt_s < tau2)
            want = np.where(drafted, am_b, np.where(remask, M, old))
            assert np.array_equal(new, want), (tau1, tau2, st)
            assert np.array_equal(cnt[:, 0], (drafted & (am_b != M)).sum(1))
            assert np.array_equal(cnt[:, 1], remask.sum(1))
            assert np.array_equal(cnt[:, 2], (new == M).sum(1))
            assert np.all((fl == 3) == remask) and np.all((fl == 4) == (drafted & (am_b == M)))
            assert np.all(((fl == 1) | (fl == 2)) == (drafted & (am_b != M)))
            # at least one draft whenever the block had a MASK (Sec. 4.2.3 loop progress)
            assert np.all(drafted.any(1) == is_m.any(1))


def pin_loop_terminates(O):
    """The tiny workload decoded to the end: every step drafts at least one token
    while a MASK is left, nothing outside the current block changes, and each
    block ends with no MASK (Sec. 4.2.3)."""
    w = ws.Workload("pin_loop", d=64, V=1000, n_seq=3, blk_len=8, bias=((1.0, 2.0, 6.0),), n_blocks=3,
                    bias_step=0.5, tau1=0.7, tau2=0.9)
    W = ws.weights(w)
    st = ws.initial_state(w)
    tokens = st.tokens.copy()
    k = 0
    for blk in range(w.n_blocks):
        b0 = w.block_start(blk)
        st.blk_start = b0
        for _ in range(400):
            H = ws.hidden_states(w, W, st, step=k)
            r = O.step(H, W, tokens, b0, w.blk_len, w.mask_id, w.tau1, w.tau2)
            had_mask = (tokens[:, b0:b0 + w.blk_len] == w.mask_id).any(1)
            outside = np.ones(w.seq_len, bool)
            outside[b0:b0 + w.blk_len] = False
            assert np.array_equal(r.tokens[:, outside], tokens[:, outside])
            assert np.all((r.counts[:, 0] >= 1) | ~had_mask | (r.flags == 4).any(1))
            tokens = r.tokens
            k += 1
            if np.all(r.counts[:, 2] == 0):
                break
        else:
            raise AssertionError(f"block {blk} did not finish")
    assert not np.any(tokens[:, w.prompt_len:] == w.mask_id)


def pin_freeze_finished(O):
    """A sequence whose block has no MASK has finished its loop (Sec. 4.2.3): with the
    freeze option it is not stepped; without it Eq. 4 still verifies it."""
    M = 9
    tokens = np.array([[1, 2, 3, 4], [1, M, 3, 4]], np.int32)
    am = _rows(2, 3, [[5, 5, 5], [6, 6, 6]], [[0] * 3, [0] * 3])
    pm = _rows(2, 3, [[0.9] * 3, [0.9] * 3], [[0.0] * 3, [0.0] * 3])
    pt = _rows(2, 3, [[0.0] * 3, [0.0] * 3], [[0.1, 0.1, 0.95], [0.1, 0.1, 0.1]])
    tok, cnt, fl = O.draft_verify(tokens, 1, 3, M, 0.5, 0.9, am, pm, pt, freeze_finished=True)
    assert tok.tolist() == [[1, 2, 3, 4], [1, 6, M, M]], tok
    assert cnt.tolist() == [[0, 0, 0], [1, 2, 2]] and fl.tolist() == [[0, 0, 0], [1, 3, 3]], (cnt, fl)
    tok, cnt, fl = O.draft_verify(tokens, 1, 3, M, 0.5, 0.9, am, pm, pt, freeze_finished=False)
    assert tok.tolist() == [[1, M, M, 4], [1, 6, M, M]] and cnt.tolist() == [[0, 2, 2], [1, 2, 2]], (tok, cnt)


def finalization_steps_from_trajectory(traj):
    """t_l = min{t : y_l^(j) = y_l^(K) for all j >= t} over a trajectory Y^(0..K) (Sec. 5.1)."""
    Y = np.stack(traj)  # [K + 1, n_seq, S]
    final = Y[-1]
    differs = Y != final[None]
    K = Y.shape[0] - 1
    # the last index j at which the state still differs from the final one, plus one; 0 if never
    any_diff = differs.any(0)
    last_diff = K - np.argmax(differs[::-1], axis=0)
    return np.where(any_diff, last_diff + 1, 0).astype(np.int32)


def pin_finalization_steps(O):
    """The step bookkeeping equals the paper's finalization step computed from the whole trajectory,
    including positions that were drafted, re-masked and drafted again."""
    w = ws.Workload("pin_final", d=64, V=500, n_seq=3, blk_len=8, bias=((1.0, 0.0, 5.0),), n_blocks=2,
                    bias_step=0.4, tau1=0.6, tau2=0.9)
    W = ws.weights(w)
    st = ws.initial_state(w)
    tokens = st.tokens.copy()
    last = np.zeros_like(tokens)
    traj = [tokens.copy()]
    k = 0
    remasked = 0
    for blk in range(w.n_blocks):
        b0 = w.block_start(blk)
        st.blk_start = b0
        for _ in range(400):
            H = ws.hidden_states(w, W, st, step=k)
            k += 1
            r = O.step(H, W, tokens, b0, w.blk_len, w.mask_id, w.tau1, w.tau2, freeze_finished=True, step_index=k,
                       last_change=last)
            tokens = r.tokens
            traj.append(tokens.copy())
            remasked += int(r.counts[:, 1].sum())
            if np.all(r.counts[:, 2] == 0):
                break
    assert remasked > 0, "the trajectory should revoke some tokens"
    want = finalization_steps_from_trajectory(traj)
    assert np.array_equal(last, want), (last, want)
    assert np.all(last[:, :w.prompt_len] == 0) and np.all(last[:, w.prompt_len:] >= 1)


def pin_no_shadow_is_threshold_decoding(O):
    """WINO+ inference (no shadow block): on the block rows it is exactly Eq. 4 with verification off
    (tau2 = 0, the "only draft" ablation of Sec. 6.3.4), whatever the shadow rows would have said."""
    rng = np.random.default_rng(23)
    n_seq, L, M, P = 40, 12, 70, 5
    for tau1 in (0.25, 0.5, 1.0):
        tokens = rng.integers(0, M + 1, size=(n_seq, P + L + 3)).astype(np.int32)
        tokens[rng.random(tokens.shape) < 0.5] = M
        am_b = rng.integers(0, M + 1, size=(n_seq, L)).astype(np.int32)
        pm_b = np.round(rng.random((n_seq, L)) * 8) / 8
        # WINO+ rows: [s][l]
        t1, c1, f1 = O.draft_verify(tokens, P, L, M, tau1, 0.9, am_b.reshape(-1), pm_b.reshape(-1), None,
                                    no_shadow=True)
        # the same block rows inside the [s][kind][l] layout, shadow rows random, tau2 = 0
        am = np.stack([am_b, rng.integers(0, M, size=(n_seq, L))], 1).reshape(-1).astype(np.int32)
        pm = np.stack([pm_b, rng.random((n_seq, L))], 1).reshape(-1)
        pt = rng.random(2 * n_seq * L)
        t2, c2, f2 = O.draft_verify(tokens, P, L, M, tau1, 0.0, am, pm, pt)
        assert np.array_equal(t1, t2) and np.array_equal(c1, c2) and np.array_equal(f1, f2)
        assert np.all(c1[:, 1] == 0)


def pin_fixed_m_hand_case(O):
    """M = 2 picks the two most confident masked positions, the lower position first on ties; decoded
    positions are verified as usual (or left alone without the shadow block)."""
    M = 50
    tokens = np.array([[1, M, 7, M, M, M, 8]], np.int32)  # block = positions 1..5
    am = _rows(1, 5, [11, 12, 13, 14, 15], [0] * 5)
    pm = _rows(1, 5, [0.25, 0.99, 0.5, 0.75, 0.5], [0.0] * 5)  # l1 is decoded: its pmax is irrelevant
    pt = _rows(1, 5, [0.0] * 5, [0.0, 0.1, 0.0, 0.0, 0.0])
    tok, cnt, fl = O.draft_verify(tokens, 1, 5, M, 0.0, 0.9, am, pm, pt, draft_m=2)
    # masked l0 (0.25), l2 (0.5), l3 (0.75), l4 (0.5): l3 first, then l2 (ties with l4, lower position)
    assert tok.tolist() == [[1, M, M, 13, 14, M, 8]], tok  # l1 re-masked: 0.1 < 0.9
    assert cnt.tolist() == [[2, 1, 3]] and fl.tolist() == [[0, 3, 5, 5, 0]], (cnt, fl)
    tok, cnt, fl = O.draft_verify(tokens, 1, 5, M, 0.0, 0.9, am.reshape(1, 2, 5)[:, 0].reshape(-1),
                                  pm.reshape(1, 2, 5)[:, 0].reshape(-1), None, no_shadow=True, draft_m=2)
    assert tok.tolist() == [[1, M, 7, 13, 14, M, 8]] and cnt.tolist() == [[2, 0, 2]], (tok, cnt)
    # M at least the number of masks: every masked position is drafted, whatever tau1 says
    tok, cnt, fl = O.draft_verify(tokens, 1, 5, M, 1.0, 0.0, am, pm, pt, draft_m=9)
    assert tok.tolist() == [[1, 11, 7, 13, 14, 15, 8]] and cnt.tolist() == [[4, 0, 0]], (tok, cnt)


def _top_m_by_sort(masked, conf, m):
    """The drafted set of naive parallel sampling via numpy's stable sort: by confidence, then position."""
    L = len(conf)
    order = np.lexsort((np.arange(L), -np.where(masked, conf, -np.inf)))
    sel = np.zeros(L, bool)
    sel[order[:min(m, int(masked.sum()))]] = True
    return sel & masked


def pin_fixed_m_one_is_greedy(O):
    """M = 1 equals the tau1 = 1 reduction (Eq. 1) step for step, and every M equals a stable sort."""
    rng = np.random.default_rng(29)
    n_seq, L, V, P = 24, 10, 300, 2
    for m in (1, 2, 3, 5, 10, 12):
        tokens = rng.integers(0, V, size=(n_seq, P + L + 2)).astype(np.int32)
        tokens[:, P:P + L][rng.random((n_seq, L)) < 0.6] = V
        am_b = rng.integers(0, V, size=(n_seq, L)).astype(np.int32)
        pm_b = np.round(rng.random((n_seq, L)) * 6) / 6  # coarse grid: many exact ties
        t1, c1, f1 = O.draft_verify(tokens, P, L, V, 0.5, 0.0, am_b.reshape(-1), pm_b.reshape(-1), None,
                                    no_shadow=True, draft_m=m)
        for s in range(n_seq):
            masked = tokens[s, P:P + L] == V
            sel = _top_m_by_sort(masked, pm_b[s], m)
            want = np.where(sel, am_b[s], tokens[s, P:P + L])
            assert np.array_equal(t1[s, P:P + L], want), (m, s)
            assert np.array_equal(f1[s] == 5, sel) and c1[s, 0] == sel.sum() and c1[s, 1] == 0
        if m == 1:
            t2, c2, _ = O.draft_verify(tokens, P, L, V, 1.0, 0.0, am_b.reshape(-1), pm_b.reshape(-1), None,
                                       no_shadow=True)
            assert np.array_equal(t1, t2) and np.array_equal(c1, c2)


def pin_fixed_m_subsets(O):
    """Brute force over all subsets: the drafted set is the only one of size min(M, #MASK) in which every
    member beats every masked position left out (higher confidence, or equal and a lower position)."""
    L, V = 5, 7
    grid = np.array([0.0, 0.5, 1.0])
    confs = np.array(list(itertools.product(range(len(grid)), repeat=L)))  # 243 confidence patterns
    for mask_bits in range(1 << L):
        masked = np.array([(mask_bits >> l) & 1 for l in range(L)], bool)
        n_seq = len(confs)
        tokens = np.zeros((n_seq, L), np.int32)
        tokens[:, masked] = V
        pm_b = grid[confs]
        am_b = np.tile(np.arange(L, dtype=np.int32), (n_seq, 1))
        for m in (1, 2, 4):
            tok, cnt, fl = O.draft_verify(tokens, 0, L, V, 0.5, 0.0, am_b.reshape(-1), pm_b.reshape(-1), None,
                                          no_shadow=True, draft_m=m)
            k = min(m, int(masked.sum()))
            idx = np.flatnonzero(masked)
            for s in range(0, n_seq, 7):
                got = set(np.flatnonzero(fl[s] == 5).tolist())
                valid = []
                for sub in itertools.combinations(idx.tolist(), k):
                    out = [l for l in idx if l not in sub]
                    if all(pm_b[s, a] > pm_b[s, b] or (pm_b[s, a] == pm_b[s, b] and a < b) for a in sub for b in out):
                        valid.append(set(sub))
                assert len(valid) == 1 and got == valid[0], (mask_bits, m, s, got, valid)
                assert np.array_equal(tok[s][masked & (fl[s] == 0)], np.full(int((masked & (fl[s] == 0)).sum()), V))


GOLDEN = Path(__file__).resolve().parent / "golden"


def naive_parallel_steps():
    """(gen_len, blk_len, tokens_per_step, steps) rows printed in Sec. 6.3.3 (tests/golden)."""
    rows = []
    for line in (GOLDEN / "naive_parallel_steps.txt").read_text().splitlines():
        if line.strip() and not line.startswith("#"):
            rows.append(tuple(int(x) for x in line.split()))
    return rows


def pin_fixed_m_step_count(O):
    """The paper's step counts for a fixed number of tokens per step (Sec. 6.3.3: a generation of 256 in
    blocks of 128 takes 256, 128 and 64 steps at 1, 2 and 4 tokens per step), and ceil(L_b / M) per block
    for other splits (8 blocks of 32, M = 3: 8 x 11 steps)."""
    rng = np.random.default_rng(31)
    cases = [(gen // blk, blk, m, steps) for gen, blk, m, steps in naive_parallel_steps()]
    assert len(cases) == 3
    cases.append((8, 32, 3, 8 * 11))
    for n_blk, L, m, want_total in cases:
        n_seq, V, P = 3, 1000, 4
        tokens = np.full((n_seq, P + L * n_blk), V, np.int32)
        tokens[:, :P] = 1
        total = 0
        for b in range(n_blk):
            b0 = P + b * L
            steps = 0
            while (tokens[:, b0:b0 + L] == V).any():
                am = rng.integers(0, V, size=n_seq * L).astype(np.int32)  # never MASK (= V)
                pm = rng.random(n_seq * L)
                tokens, cnt, _ = O.draft_verify(tokens, b0, L, V, 0.9, 0.9, am, pm, None, freeze_finished=True,
                                                no_shadow=True, draft_m=m)
                steps += 1
                assert steps <= L
            assert steps == -(-L // m), (m, b, steps)
            total += steps
        assert total == want_total, (m, total)
        assert not (tokens == V).any()


EQ4_PINS = [pin_eq4_hand_cases, pin_freeze_finished, pin_finalization_steps, pin_no_shadow_is_threshold_decoding,
            pin_fixed_m_hand_case, pin_fixed_m_one_is_greedy, pin_fixed_m_subsets, pin_fixed_m_step_count,
            pin_only_draft_never_remasks, pin_greedy_reduction, pin_eq4_exhaustive_properties, pin_loop_terminates]

ALL_PINS = SCORING_PINS + EQ4_PINS
