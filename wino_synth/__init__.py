"""Seeded synthetic workloads for the WINO scoring-and-revoke step.

This module draws the INPUTS of one WINO decoding step and nothing else: LM-head
weights W[V, d], hidden states H[N, d] for the block rows and the verification
(shadow-block) rows, planted target tokens, and the int32 token/mask state.
It holds none of the method's arithmetic (no logits, softmax, thresholds or
re-masking); both the CPU oracle and the CUDA path consume the bytes it makes.

Value conventions
-----------------
* bf16 tensors are returned as ``uint16`` bit patterns (the top half of an IEEE
  binary32), rounded to nearest-even from float32.
* ``MASK`` is the last vocabulary id, ``V - 1``; planted targets and
  pre-decoded tokens are never ``MASK``.
* Sequence layout: ``prompt_len`` prompt tokens, then ``n_blocks`` generation
  blocks of ``blk_len`` positions (semi-autoregressive blocks, Sec. 3).  A
  single-step workload decodes block 0 with one all-MASK block to its right, so
  the state has positions on both sides of the current block (Sec. 4.2.1).
* Hidden-state rows are ordered ``[s][kind][l]``: for sequence ``s``, the
  ``blk_len`` rows of the current block Y_cur (kind 0, drafting, Eq. 2) and then
  the ``blk_len`` rows of the shadow block Y_shad (kind 1, verification, Eq. 3).

Planting: row (s, kind, l) gets hidden state ``z + b * w_t / |w_t|^2`` with
``z ~ N(0, I_d)``, ``t`` the planted target of position l (shared by both
kinds), ``w_t`` the bf16 row of W for ``t`` and ``b`` drawn from the
workload's bias mixture independently per row.  This raises the logit of
``t`` by about ``b`` over a N(0, 1) background (W ~ N(0, 1/d)).

Random streams are numpy ``PCG64`` generators keyed by ``[seed, tag, ...]``,
so each tensor is a pure function of (workload, seed, step).
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

_TAG_W, _TAG_STATE, _TAG_H, _TAG_BIAS, _TAG_RAND = 1, 2, 3, 4, 5
_CHUNK_ROWS = 2048


def _threads() -> int:
    return max(1, min(16, os.cpu_count() or 1))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest-even) and return the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).copy()
    u += ((u >> 16) & 1) + np.uint32(0x7FFF)
    return (u >> 16).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal_rows_bf16(rows: int, d: int, scale: float, key: list[int]) -> np.ndarray:
    """rows x d matrix of N(0, scale^2) values rounded to bf16, drawn in row
    chunks (one PCG64 stream per chunk, keyed by ``key + [chunk]``) so that the
    fill can run on several threads and stay deterministic."""
    out = np.empty((rows, d), dtype=np.uint16)
    n_chunks = (rows + _CHUNK_ROWS - 1) // _CHUNK_ROWS
    sc = np.float32(scale)

    def work(c: int) -> None:
        r0, r1 = c * _CHUNK_ROWS, min(rows, (c + 1) * _CHUNK_ROWS)
        x = np.random.default_rng(key + [c]).standard_normal((r1 - r0, d), dtype=np.float32)
        if scale != 1.0:
            x *= sc
        u = x.view(np.uint32)
        r = (u >> 16) & 1
        r += np.uint32(0x7FFF)
        u += r
        u >>= 16
        out[r0:r1] = u

    if n_chunks == 1:
        work(0)
    else:
        with ThreadPoolExecutor(_threads()) as ex:
            list(ex.map(work, range(n_chunks)))
    return out


def random_bf16(rows: int, d: int, scale: float = 1.0, seed: int = 0, tag: int = _TAG_RAND) -> np.ndarray:
    """Generic seeded N(0, scale^2) bf16 matrix (uint16 bits), for shape sweeps."""
    return _normal_rows_bf16(rows, d, scale, [seed, tag])


@dataclass(frozen=True)
class Workload:
    """One synthetic WINO decoding workload (shapes, bias law, thresholds)."""

    name: str
    d: int
    V: int
    n_seq: int
    blk_len: int
    # bias mixture: tuple of (weight, lo, hi); each row draws b ~ U[lo, hi + bias_step * step]
    bias: tuple = ((1.0, 0.0, 8.0),)
    predecoded: float = 0.0  # fraction of block positions pre-decoded with random tokens
    tau1: float = 0.7
    tau2: float = 0.9
    prompt_len: int = 32
    n_blocks: int = 2
    seed: int = 0
    hold: float = 0.0  # fraction of pre-decoded positions that hold their planted target
    bias_step: float = 0.0  # growth of every component's upper bound per global step
    bias_floor_step: float = 0.0  # growth of every component's lower bound per global step
    shadow: bool = True  # False: WINO+ inference, block rows only (no verification rows)

    @property
    def mask_id(self) -> int:
        return self.V - 1

    @property
    def gen_len(self) -> int:
        return self.n_blocks * self.blk_len

    @property
    def seq_len(self) -> int:
        return self.prompt_len + self.gen_len

    @property
    def kinds(self) -> int:
        return 2 if self.shadow else 1

    @property
    def N(self) -> int:
        return self.n_seq * self.kinds * self.blk_len

    def block_start(self, block: int = 0) -> int:
        return self.prompt_len + block * self.blk_len


# The five workloads: the paper's decoding setup (LLaDA-8B head shape d=4096,
# V=126464; MMaDA's unified text+image vocabulary V=134400; gen length 256)
# with synthetic hidden states standing in for the model's.
WORKLOADS: dict[str, Workload] = {
    "tiny": Workload("tiny_d64_V1000_B1_L32", d=64, V=1000, n_seq=1, blk_len=32,
                     bias=((1.0, 0.0, 8.0),), predecoded=0.5, tau1=0.7, tau2=0.9),
    "llada_b1": Workload("llada8b_d4096_V126464_B1_L128", d=4096, V=126464, n_seq=1, blk_len=128,
                         bias=((1.0, 0.0, 10.0),), predecoded=0.4, tau1=0.7, tau2=0.9),
    "llada_b8": Workload("llada8b_d4096_V126464_B8_L128", d=4096, V=126464, n_seq=8, blk_len=128,
                         bias=((1.0, 0.0, 10.0),), predecoded=0.4, tau1=0.7, tau2=0.9),
    "unified_b4": Workload("unified_d4096_V134400_B4_L256", d=4096, V=134400, n_seq=4, blk_len=256,
                           bias=((0.7, 0.0, 3.0), (0.3, 6.0, 12.0)), predecoded=0.25, tau1=0.6, tau2=0.9),
    "loop_b16": Workload("loop_d4096_V126464_B16_gen256_L32", d=4096, V=126464, n_seq=16, blk_len=32,
                         bias=((1.0, 0.0, 4.0),), predecoded=0.0, tau1=0.7, tau2=0.9,
                         n_blocks=8, bias_step=0.5),
}


def coverage_variant(w: Workload) -> Workload:
    """Same shapes with doubled biases and half of the pre-decoded positions
    holding their planted token, so that every branch of the step (threshold
    draft, verify keep, verify re-mask) is exercised."""
    bias = tuple((wt, 2.0 * lo, 2.0 * hi) for (wt, lo, hi) in w.bias)
    return replace(w, name=w.name + "_coverage", bias=bias, hold=0.5,
                   predecoded=w.predecoded if w.predecoded > 0 else 0.5)


def weights(w: Workload) -> np.ndarray:
    """LM-head weights W[V, d] ~ N(0, 1/d), bf16 bits.  Depends only on (d, V, seed)."""
    return _normal_rows_bf16(w.V, w.d, 1.0 / np.sqrt(w.d), [w.seed, _TAG_W, w.d, w.V])


@dataclass
class State:
    tokens: np.ndarray  # int32 [n_seq, seq_len]
    targets: np.ndarray  # int32 [n_seq, gen_len], planted target per generation position
    blk_start: int


def initial_state(w: Workload, block: int = 0) -> State:
    """Prompt tokens (random non-MASK), planted targets, and the current block's
    pre-decoded subset; every other generation position is MASK."""
    rng = np.random.default_rng([w.seed, _TAG_STATE])
    mask = w.mask_id
    tokens = np.full((w.n_seq, w.seq_len), mask, dtype=np.int32)
    tokens[:, : w.prompt_len] = rng.integers(0, w.V - 1, size=(w.n_seq, w.prompt_len), dtype=np.int32)
    targets = rng.integers(0, w.V - 1, size=(w.n_seq, w.gen_len), dtype=np.int32)
    b0 = w.block_start(block)
    n_pre = int(round(w.predecoded * w.blk_len))
    n_hold = int(round(w.hold * n_pre))
    for s in range(w.n_seq):
        pos = rng.permutation(w.blk_len)[:n_pre]
        vals = rng.integers(0, w.V - 1, size=n_pre, dtype=np.int32)
        gen0 = b0 - w.prompt_len
        vals[:n_hold] = targets[s, gen0 + pos[:n_hold]]
        tokens[s, b0 + pos] = vals
    return State(tokens=tokens, targets=targets, blk_start=b0)


def row_biases(w: Workload, step: int = 0) -> np.ndarray:
    """Planted logit bias per hidden-state row (float32 [N])."""
    rng = np.random.default_rng([w.seed, _TAG_BIAS, step])
    wts = np.array([c[0] for c in w.bias], dtype=np.float64)
    cum = np.cumsum(wts / wts.sum())
    u = rng.random(w.N)
    comp = np.minimum(np.searchsorted(cum, u, side="right"), len(w.bias) - 1)
    lo = np.array([c[1] for c in w.bias])[comp] + w.bias_floor_step * step
    hi = np.maximum(np.array([c[2] for c in w.bias])[comp] + w.bias_step * step, lo)
    return (lo + (hi - lo) * rng.random(w.N)).astype(np.float32)


def hidden_states(w: Workload, W: np.ndarray, state: State, step: int = 0) -> np.ndarray:
    """H[N, d] bf16 bits for the current block of ``state`` at global step ``step``.

    Rows are ``[s][kind][l]`` (``[s][l]`` without the shadow block); every row of
    position l plants target ``state.targets[s, blk_start - prompt_len + l]`` with
    independent noise and bias."""
    z = _normal_rows_bf16(w.N, w.d, 1.0, [w.seed, _TAG_H, step])  # noise (bf16-exact values)
    h = bf16_bits_to_f32(z).reshape(w.N, w.d)
    b = row_biases(w, step)
    gen0 = state.blk_start - w.prompt_len
    L = w.blk_len
    t = state.targets[:, gen0: gen0 + L]  # [n_seq, L]
    t_rows = np.repeat(t[:, None, :], w.kinds, axis=1).reshape(-1)  # [s][kind][l]
    wt = bf16_bits_to_f32(W[t_rows])  # [N, d]
    nrm2 = np.einsum("nd,nd->n", wt.astype(np.float64), wt.astype(np.float64)).astype(np.float32)
    h += (b / nrm2)[:, None] * wt
    return f32_to_bf16_bits(h)


def row_targets_planted(w: Workload, state: State) -> np.ndarray:
    """Planted target token of every hidden-state row (int32 [N]); for reporting."""
    gen0 = state.blk_start - w.prompt_len
    t = state.targets[:, gen0: gen0 + w.blk_len]
    return np.repeat(t[:, None, :], w.kinds, axis=1).reshape(-1).astype(np.int32)
