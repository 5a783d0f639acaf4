"""Helpers for the GPU parity tests: upload seeded inputs, run the C ABI,
compare with the oracle under the stated tolerances.

Tolerances: per-row probabilities within 1e-3 absolute of the fp64 oracle;
argmax and the integer token state bit-exact, except where the oracle's
top-2 logits differ by less than 1e-3 (argmax near-tie) or a decision's
probability lies within 1e-3 of its threshold; those positions are counted
and reported, not failed.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

import oracle
import paper_2605_16941_gb300 as wino

PROB_TOL = 1e-3
TIE_TOL = 1e-3


def dev(a: np.ndarray) -> torch.Tensor:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy()


def f32(x: float) -> float:
    """The double value of x rounded to float32: the kernels compare in fp32."""
    return float(np.float32(x))


@dataclass
class GpuStats:
    argmax: np.ndarray
    pmax: np.ndarray
    ptarget: np.ndarray
    entropy: np.ndarray | None = None


def gpu_score(Hd: torch.Tensor, Wd: torch.Tensor, target: np.ndarray | None, canary: int = 64,
              entropy: bool = False) -> GpuStats:
    """wino_score_rows with guard zones after every output (checked untouched)."""
    N, d = Hd.shape
    V = Wd.shape[0]
    t = dev(target.astype(np.int32)) if target is not None else None
    am = torch.full((N + canary,), -777, dtype=torch.int32, device="cuda")
    pm = torch.full((N + canary,), -7.0, dtype=torch.float32, device="cuda")
    pt = torch.full((N + canary,), -7.0, dtype=torch.float32, device="cuda")
    en = torch.full((N + canary,), -7.0, dtype=torch.float32, device="cuda") if entropy else None
    ws = wino.workspace(N, d, V)
    wino.wino_score_rows(Hd, Wd, t, am, pm, pt, ws, entropy=en, N=N, d=d, V=V)
    torch.cuda.synchronize()
    assert wino.wino_read_device_status(ws) == wino.WINO_OK
    am, pm, pt = host(am), host(pm), host(pt)
    assert np.all(am[N:] == -777) and np.all(pm[N:] == -7.0) and np.all(pt[N:] == -7.0), "output guard zone written"
    ent = None
    if entropy:
        ent = host(en)
        assert np.all(ent[N:] == -7.0), "entropy guard zone written"
        ent = ent[:N]
    return GpuStats(am[:N], pm[:N], pt[:N], ent)


def compare_rows(o: oracle.RowStats, g: GpuStats, rows=None) -> dict:
    """Row statistics against the oracle; returns counts of flagged near-ties."""
    idx = np.arange(len(o.pmax)) if rows is None else np.asarray(rows)
    am, pm, pt = g.argmax[idx], g.pmax[idx], g.ptarget[idx]
    assert np.all(np.isfinite(pm)) and np.all(np.isfinite(pt))
    dp = np.abs(pm.astype(np.float64) - o.pmax)
    dt = np.abs(pt.astype(np.float64) - o.ptarget)
    assert dp.max(initial=0) <= PROB_TOL, f"pmax off by {dp.max()} at row {idx[dp.argmax()]}"
    assert dt.max(initial=0) <= PROB_TOL, f"ptarget off by {dt.max()} at row {idx[dt.argmax()]}"
    if g.entropy is not None:
        de = np.abs(g.entropy[idx].astype(np.float64) - o.entropy)
        assert np.all(np.isfinite(g.entropy[idx])) and de.max(initial=0) <= PROB_TOL, \
            f"entropy off by {de.max()} at row {idx[de.argmax()]}"
    near = o.gap < TIE_TOL
    bad = (am != o.argmax) & ~near
    assert not bad.any(), f"argmax differs at rows {idx[bad][:10]}: gpu {am[bad][:10]} oracle {o.argmax[bad][:10]}"
    return {"rows": len(idx), "argmax_near_ties": int(near.sum()), "argmax_tie_mismatch": int((am != o.argmax).sum()),
            "max_dpmax": float(dp.max(initial=0)), "max_dptarget": float(dt.max(initial=0))}


def flagged_positions(tokens_pre: np.ndarray, o: oracle.StepResult, blk_start: int, blk_len: int, mask_id: int,
                      tau1: float, tau2: float) -> np.ndarray:
    """[n_seq, blk_len] bool: positions whose Eq. 4 decision is within tolerance of a tie."""
    n_seq = tokens_pre.shape[0]
    L = blk_len
    pm = o.pmax.reshape(n_seq, 2, L)[:, 0, :]
    pt = o.ptarget.reshape(n_seq, 2, L)[:, 1, :]
    gap = o.gap.reshape(n_seq, 2, L)[:, 0, :]
    y = tokens_pre[:, blk_start:blk_start + L]
    masked = y == mask_id
    flag = np.zeros((n_seq, L), bool)
    flag |= masked & (np.abs(pm - tau1) < PROB_TOL)
    flag |= masked & (gap < TIE_TOL)
    flag |= ~masked & (np.abs(pt - tau2) < PROB_TOL)
    # the at-least-one rule: if the two most confident masked positions are close, the choice is flagged
    for s in range(n_seq):
        c = np.where(masked[s], pm[s], -np.inf)
        if masked[s].sum() >= 2 and not (masked[s] & (pm[s] > tau1 + PROB_TOL)).any():
            srt = np.sort(c)[::-1]
            if srt[0] - srt[1] < PROB_TOL:
                flag[s] |= masked[s] & (c >= srt[0] - PROB_TOL)
    return flag


def compare_step(tokens_pre: np.ndarray, tok_gpu: np.ndarray, cnt_gpu: np.ndarray, o: oracle.StepResult,
                 blk_start: int, blk_len: int, mask_id: int, tau1: float, tau2: float) -> dict:
    """Token state and counts of a GPU step against the oracle's step from the same state."""
    L = blk_len
    outside = np.ones(tokens_pre.shape[1], bool)
    outside[blk_start:blk_start + L] = False
    assert np.array_equal(tok_gpu[:, outside], tokens_pre[:, outside]), "a position outside the block changed"
    flag = flagged_positions(tokens_pre, o, blk_start, blk_len, mask_id, tau1, tau2)
    g = tok_gpu[:, blk_start:blk_start + L]
    r = o.tokens[:, blk_start:blk_start + L]
    bad = (g != r) & ~flag
    assert not bad.any(), f"token state differs at {np.argwhere(bad)[:10].tolist()}"
    seq_clean = ~flag.any(1)
    assert np.array_equal(cnt_gpu[seq_clean], o.counts[seq_clean]), (cnt_gpu[seq_clean], o.counts[seq_clean])
    return {"flagged_positions": int(flag.sum()), "flagged_mismatch": int(((g != r) & flag).sum()),
            "drafted": int(o.counts[:, 0].sum()), "remasked": int(o.counts[:, 1].sum()),
            "fallback": int((o.flags == oracle.FLAG_DRAFT_FALLBACK).sum()),
            "threshold_drafts": int((o.flags == oracle.FLAG_DRAFT).sum()),
            "kept_decoded": int(((tokens_pre[:, blk_start:blk_start + L] != mask_id) & (o.flags == 0)).sum())}
