"""Semi-autoregressive WINO decode loop over the C ABI (Sec. 3 and Sec. 4.2.3).

Blocks are decoded left to right; inside a block ``wino_step`` is repeated
until no position of the block is MASK in any sequence of the batch.  A
sequence whose block is complete is frozen (WINO_OPT_FREEZE_FINISHED): its
own loop has ended, so it is not re-verified while the rest of the batch
finishes the block.  The
only device-to-host traffic per step is the [n_seq, 3] counts array, read to
decide whether the block is finished (plus the token state when a trajectory
is recorded).  The hidden states of each step come
from a caller-supplied function (the transformer forward with the
shadow-block attention mask is outside this library).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable

from ._abi import (WINO_ERR_MAX_STEPS, WINO_OK, WinoError, make_params, wino_decode, wino_step,
                   wino_workspace_size_step)


@dataclass
class BlockStats:
    block: int
    blk_start: int
    steps: int = 0
    drafted: int = 0
    remasked: int = 0
    fallback: int = 0  # drafts made by the at-least-one rule (no masked position cleared tau1)


@dataclass
class LoopStats:
    blocks: list = field(default_factory=list)
    total_steps: int = 0  # steps this call ran
    rows_scored: int = 0
    next_step: int = 0  # global index of the step after the last one run


def resume_point(k: int, blk_start: int, counts, *, prompt_len: int, blk_len: int) -> tuple[int, int]:
    """(start_block, start_step) that continue a decode after its global step ``k``, from the arguments
    ``on_step`` receives.  A checkpoint of a decode is the token state (and ``last_change``) after step
    ``k`` together with this pair: the hidden states of later steps depend only on the step index and
    the block, so a decode resumed from it replays the uninterrupted one exactly."""
    import numpy as np
    b = (blk_start - prompt_len) // blk_len
    done = bool((np.asarray(counts)[:, 2] == 0).all())
    return (b + 1 if done else b), k + 1


def _head_dims(W, w_panels: bool) -> tuple[int, int]:
    """(d, V) of an LM head given row-major [V, d] or as a panel copy [d/64, V, 64]."""
    if w_panels:
        return int(W.shape[0]) * 64, int(W.shape[1])
    return int(W.shape[1]), int(W.shape[0])


def decode(W, tokens, *, prompt_len: int, blk_len: int, n_blocks: int, tau1: float, tau2: float, mask_id: int,
           hidden: Callable[[int, int], object], max_steps: int = 4096, stream=None,
           on_step: Callable | None = None, last_change=None, no_shadow: bool = False,
           compact: bool = False, draft_m: int = 0, trajectory: list | None = None, start_block: int = 0,
           start_step: int = 0, skip_finished: bool = False, w_panels: bool = False) -> LoopStats:
    """Decode ``n_blocks`` blocks of ``tokens`` (int32 [n_seq, S], device) in place.

    ``hidden(k, blk_start)`` returns the device bf16 hidden states [2*n_seq*blk_len, d]
    for global step ``k`` (0-based; the step produces state Y^(k+1)).  ``on_step(k,
    blk_start, counts_host, flags)`` is called after every step (for tests and
    statistics).  ``last_change`` (device int32 [n_seq, S], zeros at the start)
    receives, per position, the last step that changed it: after the decode, each
    position's WINO finalization step t_l (Sec. 5.1).  ``no_shadow``: WINO+ inference
    (Sec. 5.3): ``hidden`` returns only the n_seq*blk_len block rows, drafting uses the
    single threshold ``tau1`` and nothing is re-masked.  ``compact``: score only the row
    each position's update reads (WINO_OPT_COMPACT), same results.  ``draft_m`` > 0: draft
    a fixed number of the most confident masked positions per step instead of Eq. 2 (naive
    parallel sampling, Sec. 3; with ``no_shadow`` the irreversible baseline decoder, 1 =
    greedy Eq. 1).  ``trajectory``: a list that receives the host copy of the state
    Y^(0), Y^(1), ... (int32 [n_seq, S] arrays), one per step, for building WINO+ training
    states (Sec. 5.1-5.2); it costs one extra device-to-host copy of ``tokens`` per step.
    ``start_block``, ``start_step``: resume a checkpointed decode (see ``resume_point``): blocks
    before ``start_block`` are taken as done and the global step count starts at ``start_step``.
    ``skip_finished``: each step scores only the sequences whose block still has a MASK (an
    active-sequence list, ``wino_params.active_seq``); the states are those of the frozen
    sequences without it, and ``on_step`` sees zero counts for the sequences left out.
    ``w_panels``: ``W`` is the panel copy of ``wino_lm_head_panels`` ([d/64, V, 64]), same results.
    """
    import numpy as np
    import torch

    n_seq, S = int(tokens.shape[0]), int(tokens.shape[1])
    d, V = _head_dims(W, w_panels)
    rows_per_seq = (1 if (no_shadow or compact) else 2) * blk_len  # rows scored per sequence and step
    dev = tokens.device
    ts = stream if stream is not None else torch.cuda.current_stream(dev)  # every copy goes on the step's stream
    active_d = torch.arange(n_seq, dtype=torch.int32, device=dev) if skip_finished else None
    active_h = torch.zeros(n_seq, dtype=torch.int32, pin_memory=True) if skip_finished else None
    p0 = make_params(tau1, tau2, mask_id, n_seq, S, prompt_len, blk_len, no_shadow=no_shadow, compact=compact,
                     draft_m=draft_m, active_seq=active_d, n_active=n_seq if skip_finished else None,
                     w_panels=w_panels)
    ws = torch.zeros(wino_workspace_size_step(p0, d, V), dtype=torch.uint8, device=dev)
    counts = torch.zeros((n_seq, 3), dtype=torch.int32, device=dev)
    flags = torch.zeros((n_seq, blk_len), dtype=torch.int8, device=dev)
    counts_host = torch.zeros((n_seq, 3), dtype=torch.int32, pin_memory=True)
    flags_host = torch.zeros((n_seq, blk_len), dtype=torch.int8, pin_memory=True)
    tokens_host = torch.zeros((n_seq, S), dtype=torch.int32, pin_memory=True) if trajectory is not None else None
    if trajectory is not None:
        with torch.cuda.stream(ts):
            tokens_host.copy_(tokens)
        ts.synchronize()
        trajectory.append(tokens_host.numpy().copy())
    stats = LoopStats()
    k = start_step
    for b in range(start_block, n_blocks):
        b0 = prompt_len + b * blk_len
        p = make_params(tau1, tau2, mask_id, n_seq, S, b0, blk_len, max_steps, freeze_finished=True,
                        last_change=last_change, no_shadow=no_shadow, compact=compact, draft_m=draft_m,
                        w_panels=w_panels)
        bs = BlockStats(block=b, blk_start=b0)
        active = list(range(n_seq))  # a new block: every sequence takes part
        while True:
            if bs.steps >= max_steps:
                raise WinoError(WINO_ERR_MAX_STEPS, f"decode: block {b} not finished after {max_steps} steps")
            H = hidden(k, b0)
            p.step_index = k + 1
            if skip_finished:
                active_h[:len(active)] = torch.tensor(active, dtype=torch.int32)
                with torch.cuda.stream(ts):
                    active_d[:len(active)].copy_(active_h[:len(active)], non_blocking=True)
                p.active_seq, p.n_active = active_d.data_ptr(), len(active)
            wino_step(H, W, tokens, p, counts, ws, flags=flags, stream=ts)
            with torch.cuda.stream(ts):
                counts_host.copy_(counts, non_blocking=True)
                flags_host.copy_(flags, non_blocking=True)
                if tokens_host is not None:
                    tokens_host.copy_(tokens, non_blocking=True)
            ts.synchronize()
            c = counts_host.numpy().copy()
            fl = flags_host.numpy().copy()
            if skip_finished:  # the sequences left out were not stepped: no counts, no flags
                left_out = np.ones(n_seq, bool)
                left_out[active] = False
                c[left_out] = 0
                fl[left_out] = 0
            if tokens_host is not None:
                trajectory.append(tokens_host.numpy().copy())
            if (c < 0).any():
                raise WinoError(int(c.min()), f"decode: device status at step {k}")
            bs.steps += 1
            bs.drafted += int(c[:, 0].sum())
            bs.remasked += int(c[:, 1].sum())
            bs.fallback += int((fl == 2).sum())
            stats.rows_scored += rows_per_seq * len(active)
            if on_step is not None:
                on_step(k, b0, c.copy(), flags)
            k += 1
            if (c[:, 2] == 0).all():
                break
            if skip_finished:
                active = [i for i in active if c[i, 2] != 0]
        stats.blocks.append(bs)
    stats.total_steps = k - start_step
    stats.next_step = k
    return stats


def decode_native(W, tokens, *, prompt_len: int, blk_len: int, n_blocks: int, tau1: float, tau2: float,
                  mask_id: int, hidden: Callable[[int, int], object], max_steps: int = 4096, stream=None,
                  last_change=None, no_shadow: bool = False, compact: bool = False, draft_m: int = 0,
                  start_block: int = 0, start_step: int = 0, skip_finished: bool = False,
                  w_panels: bool = False) -> LoopStats:
    """``decode`` with the step loop run by the library (``wino_decode``): the same steps, states and
    statistics, with one callback into Python per step (for the hidden states) instead of the whole
    per-step bookkeeping.  No ``on_step`` or ``trajectory``; errors raise ``WinoError``.
    ``skip_finished`` as in ``decode``: the library keeps the active-sequence list; ``w_panels`` as in ``decode``."""
    import torch

    n_seq, S = int(tokens.shape[0]), int(tokens.shape[1])
    d, V = _head_dims(W, w_panels)
    rows_per_seq = (1 if (no_shadow or compact) else 2) * blk_len
    dev = tokens.device
    ts = stream if stream is not None else torch.cuda.current_stream(dev)
    p = make_params(tau1, tau2, mask_id, n_seq, S, prompt_len, blk_len, max_steps, freeze_finished=True,
                    last_change=last_change, no_shadow=no_shadow, compact=compact, draft_m=draft_m,
                    w_panels=w_panels)
    active_buf = torch.zeros(n_seq, dtype=torch.int32, device=dev) if skip_finished else None
    p_ws = make_params(tau1, tau2, mask_id, n_seq, S, prompt_len, blk_len, no_shadow=no_shadow, compact=compact,
                       active_seq=active_buf, n_active=n_seq if skip_finished else None)  # sized for every list
    ws = torch.zeros(wino_workspace_size_step(p_ws, d, V), dtype=torch.uint8, device=dev)
    counts = torch.zeros((n_seq, 3), dtype=torch.int32, device=dev)
    counts_host = torch.zeros((n_seq, 3), dtype=torch.int32, pin_memory=True)
    flags = torch.zeros((n_seq, blk_len), dtype=torch.int8, device=dev)
    flags_host = torch.zeros((n_seq, blk_len), dtype=torch.int8, pin_memory=True)
    torch.cuda.current_stream(dev).synchronize()  # the buffers above are ready before the library's stream runs
    rc, blocks, nxt = wino_decode(W, tokens, p, n_blocks, hidden, counts, counts_host, ws, flags=flags,
                                  flags_host=flags_host, active_buf=active_buf, stream=ts, first_block=start_block,
                                  first_step=start_step)
    if rc != WINO_OK:
        raise WinoError(rc, f"wino_decode (stopped at step {nxt})")
    stats = LoopStats()
    for b in range(start_block, n_blocks):
        steps, drafted, remasked, fallback, seq_steps = blocks[b]
        stats.blocks.append(BlockStats(block=b, blk_start=prompt_len + b * blk_len, steps=steps, drafted=drafted,
                                       remasked=remasked, fallback=fallback))
        stats.rows_scored += rows_per_seq * seq_steps
    stats.total_steps = nxt - start_step
    stats.next_step = nxt
    return stats
