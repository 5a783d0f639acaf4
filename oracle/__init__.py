"""Plain fp64 CPU oracle of the WINO scoring-and-revoke step -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference leg may import this package.  It shares no code with the CUDA path;
the only common input is the seeded workload module ``wino_synth``.

The arithmetic lives in ``wino_oracle.c`` (see its header for what each
function computes and which equation of the paper it follows); this module
only compiles it on first use and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import numpy as np

from .build import build as _build

FLAG_NONE, FLAG_DRAFT, FLAG_DRAFT_FALLBACK, FLAG_REMASK, FLAG_DRAFT_IS_MASK, FLAG_DRAFT_TOP_M = 0, 1, 2, 3, 4, 5


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _lc(last_change, tokens):
    """Validate an in-place int32 [n_seq, seq_len] last-change array (or None)."""
    if last_change is None:
        return None
    assert last_change.dtype == np.int32 and last_change.flags.c_contiguous and last_change.shape == tokens.shape
    return last_change


@dataclass
class RowStats:
    argmax: np.ndarray  # int32 [N]
    pmax: np.ndarray  # float64 [N]
    ptarget: np.ndarray  # float64 [N]
    gap: np.ndarray  # float64 [N] top-1 minus top-2 logit
    maxlogit: np.ndarray  # float64 [N]
    logz: np.ndarray  # float64 [N]
    entropy: np.ndarray  # float64 [N], -sum p log p


@dataclass
class StepResult:
    tokens: np.ndarray
    counts: np.ndarray
    flags: np.ndarray
    argmax: np.ndarray
    pmax: np.ndarray
    ptarget: np.ndarray
    gap: np.ndarray


class Oracle:
    """ctypes view of one compiled copy of ``wino_oracle.c``."""

    def __init__(self, path: str | None = None):
        L = C.CDLL(str(path or _build()))
        i64, i32, dbl, vp = C.c_int64, C.c_int32, C.c_double, C.c_void_p
        L.oracle_bf16_to_double.restype = dbl
        L.oracle_bf16_to_double.argtypes = [C.c_uint16]
        L.oracle_logits_row.restype = None
        L.oracle_logits_row.argtypes = [vp, vp, i64, i64, vp]
        L.oracle_score_rows.restype = C.c_int
        L.oracle_score_rows.argtypes = [vp, vp, i64, i64, i64, vp, vp, vp, vp, vp, vp, vp, vp, C.c_int]
        L.oracle_row_targets.restype = C.c_int
        L.oracle_row_targets.argtypes = [vp, i64, i64, i64, i64, i32, vp]
        L.oracle_draft_verify.restype = C.c_int
        L.oracle_draft_verify.argtypes = [vp, i64, i64, i64, i64, i32, dbl, dbl, vp, vp, vp, vp, vp, C.c_int,
                                          C.c_int, i32, vp, i64]
        L.oracle_step.restype = C.c_int
        L.oracle_step.argtypes = [vp, vp, i64, i64, vp, i64, i64, i64, i64, i32, dbl, dbl, vp, vp, vp, vp, vp,
                                  vp, C.c_int, C.c_int, C.c_int, i32, vp, i64]
        L.oracle_num_threads.restype = C.c_int
        L.oracle_num_threads.argtypes = []
        self.L = L

    def num_threads(self) -> int:
        return self.L.oracle_num_threads()

    def bf16_to_double(self, bits: int) -> float:
        return self.L.oracle_bf16_to_double(int(bits) & 0xFFFF)

    def logits_row(self, h_bits: np.ndarray, W_bits: np.ndarray) -> np.ndarray:
        """fp64 logits of one row."""
        h, W = _c(h_bits, np.uint16), _c(W_bits, np.uint16)
        V, d = W.shape
        assert h.shape == (d,)
        out = np.empty(V, dtype=np.float64)
        self.L.oracle_logits_row(_p(h), _p(W), d, V, _p(out))
        return out

    def score_rows(self, H_bits: np.ndarray, W_bits: np.ndarray, target: np.ndarray | None = None,
                   nthreads: int = 0) -> RowStats:
        H, W = _c(H_bits, np.uint16), _c(W_bits, np.uint16)
        N, d = H.shape
        V, d2 = W.shape
        assert d == d2
        t = None if target is None else _c(target, np.int32)
        if t is not None:
            assert t.shape == (N,)
        out = RowStats(np.empty(N, np.int32), *(np.empty(N, np.float64) for _ in range(6)))
        rc = self.L.oracle_score_rows(_p(H), _p(W), N, d, V, _p(t), _p(out.argmax), _p(out.pmax),
                                      _p(out.ptarget), _p(out.gap), _p(out.maxlogit), _p(out.logz),
                                      _p(out.entropy), nthreads)
        if rc != 0:
            raise RuntimeError(f"oracle_score_rows failed: {rc}")
        return out

    def row_targets(self, tokens: np.ndarray, blk_start: int, blk_len: int, mask_id: int) -> np.ndarray:
        tok = _c(tokens, np.int32)
        n_seq, S = tok.shape
        out = np.empty(n_seq * 2 * blk_len, np.int32)
        rc = self.L.oracle_row_targets(_p(tok), n_seq, S, blk_start, blk_len, mask_id, _p(out))
        if rc != 0:
            raise RuntimeError(f"oracle_row_targets failed: {rc}")
        return out

    def draft_verify(self, tokens: np.ndarray, blk_start: int, blk_len: int, mask_id: int, tau1: float,
                     tau2: float, argmax: np.ndarray, pmax: np.ndarray, ptarget: np.ndarray,
                     freeze_finished: bool = False, step_index: int = 0, last_change: np.ndarray | None = None,
                     no_shadow: bool = False, draft_m: int = 0):
        """Eq. 4 on a copy of ``tokens``; returns (new_tokens, counts [n_seq,3], flags [n_seq, blk_len]).
        ``last_change`` (int32 [n_seq, seq_len], updated in place) gets ``step_index`` where a token changes.
        ``no_shadow``: WINO+ inference, rows are block rows only and ``ptarget`` may be None.
        ``draft_m`` > 0: draft the ``draft_m`` most confident masked positions instead (naive parallel
        sampling, Sec. 3; 1 = greedy, Eq. 1)."""
        tok = np.array(tokens, dtype=np.int32, copy=True, order="C")
        n_seq, S = tok.shape
        N = n_seq * (1 if no_shadow else 2) * blk_len
        am, pm = _c(argmax, np.int32), _c(pmax, np.float64)
        pt = None if ptarget is None else _c(ptarget, np.float64)
        assert am.shape == pm.shape == (N,) and (pt is None or pt.shape == (N,))
        counts = np.empty((n_seq, 3), np.int32)
        flags = np.empty((n_seq, blk_len), np.int8)
        rc = self.L.oracle_draft_verify(_p(tok), n_seq, S, blk_start, blk_len, mask_id, float(tau1),
                                        float(tau2), _p(am), _p(pm), _p(pt), _p(counts), _p(flags),
                                        int(bool(freeze_finished)), int(bool(no_shadow)), int(step_index),
                                        _p(_lc(last_change, tok)), int(draft_m))
        if rc != 0:
            raise RuntimeError(f"oracle_draft_verify failed: {rc}")
        return tok, counts, flags

    def step(self, H_bits: np.ndarray, W_bits: np.ndarray, tokens: np.ndarray, blk_start: int, blk_len: int,
             mask_id: int, tau1: float, tau2: float, nthreads: int = 0, freeze_finished: bool = False,
             step_index: int = 0, last_change: np.ndarray | None = None, no_shadow: bool = False,
             draft_m: int = 0) -> StepResult:
        """One whole WINO step on a copy of ``tokens`` (``last_change``, ``no_shadow``, ``draft_m`` as in
        draft_verify)."""
        H, W = _c(H_bits, np.uint16), _c(W_bits, np.uint16)
        tok = np.array(tokens, dtype=np.int32, copy=True, order="C")
        n_seq, S = tok.shape
        N = n_seq * (1 if no_shadow else 2) * blk_len
        V, d = W.shape
        assert H.shape == (N, d)
        r = StepResult(tok, np.empty((n_seq, 3), np.int32), np.empty((n_seq, blk_len), np.int8),
                       np.empty(N, np.int32), np.empty(N, np.float64), np.empty(N, np.float64),
                       np.empty(N, np.float64))
        rc = self.L.oracle_step(_p(H), _p(W), d, V, _p(tok), n_seq, S, blk_start, blk_len, mask_id, float(tau1),
                                float(tau2), _p(r.counts), _p(r.flags), _p(r.argmax), _p(r.pmax), _p(r.ptarget),
                                _p(r.gap), nthreads, int(bool(freeze_finished)), int(bool(no_shadow)),
                                int(step_index), _p(_lc(last_change, tok)), int(draft_m))
        if rc != 0:
            raise RuntimeError(f"oracle_step failed: {rc}")
        return r


_default: Oracle | None = None


def default() -> Oracle:
    global _default
    if _default is None:
        _default = Oracle()
    return _default


def num_threads() -> int:
    return default().num_threads()


def bf16_to_double(bits: int) -> float:
    return default().bf16_to_double(bits)


def logits_row(h_bits, W_bits):
    return default().logits_row(h_bits, W_bits)


def score_rows(H_bits, W_bits, target=None, nthreads: int = 0) -> RowStats:
    return default().score_rows(H_bits, W_bits, target, nthreads)


def row_targets(tokens, blk_start: int, blk_len: int, mask_id: int):
    return default().row_targets(tokens, blk_start, blk_len, mask_id)


def draft_verify(tokens, blk_start, blk_len, mask_id, tau1, tau2, argmax, pmax, ptarget, freeze_finished=False,
                 step_index=0, last_change=None, no_shadow=False, draft_m=0):
    return default().draft_verify(tokens, blk_start, blk_len, mask_id, tau1, tau2, argmax, pmax, ptarget,
                                  freeze_finished, step_index, last_change, no_shadow, draft_m)


def step(H_bits, W_bits, tokens, blk_start, blk_len, mask_id, tau1, tau2, nthreads: int = 0,
         freeze_finished: bool = False, step_index: int = 0, last_change=None, no_shadow: bool = False,
         draft_m: int = 0) -> StepResult:
    return default().step(H_bits, W_bits, tokens, blk_start, blk_len, mask_id, tau1, tau2, nthreads, freeze_finished,
                          step_index, last_change, no_shadow, draft_m)
