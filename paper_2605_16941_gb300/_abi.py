"""ctypes binding of ``libwino.so`` (declared in ``include/wino.h``).

Argument marshalling only: every function forwards to the C entry point of
the same name, passing device pointers (``torch.Tensor.data_ptr()`` or raw
integers), sizes and a ``cudaStream_t`` handle.  All computation happens in
the library's CUDA kernels.  If the library has not been built, loading it
raises ``RuntimeError``; there is no fallback.
"""
from __future__ import annotations

import ctypes as C
from pathlib import Path

_LIB_PATH = Path(__file__).resolve().parent / "_build" / "libwino.so"
_lib = None

WINO_OK = 0
WINO_ERR_ARG = -1
WINO_ERR_SHAPE = -2
WINO_ERR_WORKSPACE = -3
WINO_ERR_CUDA = -4
WINO_ERR_MAX_STEPS = -5
WINO_ERR_DEVICE_TIMEOUT = -6
WINO_ERR_UNSUPPORTED = -7

# per-position outcome codes written to `flags`
FLAG_NONE, FLAG_DRAFT, FLAG_DRAFT_FALLBACK, FLAG_REMASK, FLAG_DRAFT_IS_MASK, FLAG_DRAFT_TOP_M = 0, 1, 2, 3, 4, 5

# wino_params.options
WINO_OPT_FREEZE_FINISHED = 1
WINO_OPT_NO_SHADOW = 2
WINO_OPT_COMPACT = 4
WINO_OPT_W_PANELS = 8

EXPORTS = ("wino_workspace_size", "wino_workspace_size_step", "wino_score_rows", "wino_draft_verify", "wino_step",
           "wino_step_static_scratch", "wino_read_device_status", "wino_profile_begin", "wino_profile_end",
           "wino_selftest_wait_timeout", "wino_status_string", "wino_version", "wino_decode", "wino_timeline_begin",
           "wino_timeline_end", "wino_score_plan", "wino_score_plan_host", "wino_lm_head_panels")

# 64-bit words per CTA in a score-kernel timeline (wino_timeline_begin)
TIMELINE_WORDS = 8

# size of the fixed device array behind wino_step_static_scratch
WINO_STATIC_SCRATCH_BYTES = 16 << 20


class WinoError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {wino_status_string(status)} ({status})")


class WinoParams(C.Structure):
    _fields_ = [("tau1", C.c_float), ("tau2", C.c_float), ("mask_id", C.c_int32), ("n_seq", C.c_int32),
                ("seq_len", C.c_int32), ("blk_start", C.c_int32), ("blk_len", C.c_int32),
                ("max_steps", C.c_int32), ("options", C.c_int32), ("step_index", C.c_int32),
                ("last_change", C.c_void_p), ("draft_m", C.c_int32), ("active_seq", C.c_void_p),
                ("n_active", C.c_int32)]


class WinoBlockStats(C.Structure):
    _fields_ = [("steps", C.c_int32), ("drafted", C.c_int32), ("remasked", C.c_int32), ("fallback", C.c_int32),
                ("seq_steps", C.c_int32)]


# const uint16_t *(*)(void *user, int32_t step, int32_t blk_start)
HIDDEN_FN = C.CFUNCTYPE(C.c_void_p, C.c_void_p, C.c_int32, C.c_int32)


def library_path() -> Path:
    return _LIB_PATH


def lib() -> C.CDLL:
    """Load libwino.so (built in-tree by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is None:
        if not _LIB_PATH.exists():
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with paper_2605_16941_gb300.build.build()")
        L = C.CDLL(str(_LIB_PATH))
        i64, vp, sz = C.c_int64, C.c_void_p, C.c_size_t
        L.wino_workspace_size.restype = C.c_int
        L.wino_workspace_size.argtypes = [i64, i64, i64, C.POINTER(sz)]
        L.wino_workspace_size_step.restype = C.c_int
        L.wino_workspace_size_step.argtypes = [C.POINTER(WinoParams), i64, i64, C.POINTER(sz)]
        L.wino_score_rows.restype = C.c_int
        L.wino_score_rows.argtypes = [vp, vp, i64, i64, i64, vp, vp, vp, vp, vp, vp, sz, vp]
        L.wino_draft_verify.restype = C.c_int
        L.wino_draft_verify.argtypes = [vp, vp, vp, vp, C.POINTER(WinoParams), vp, vp, vp]
        L.wino_step.restype = C.c_int
        L.wino_step.argtypes = [vp, vp, i64, i64, vp, C.POINTER(WinoParams), vp, vp, vp, sz, vp]
        L.wino_lm_head_panels.restype = C.c_int
        L.wino_lm_head_panels.argtypes = [vp, i64, i64, vp, vp]
        L.wino_step_static_scratch.restype = C.c_int
        L.wino_step_static_scratch.argtypes = [vp, vp, i64, i64, vp, C.POINTER(WinoParams), vp, vp, vp]
        L.wino_read_device_status.restype = C.c_int
        L.wino_read_device_status.argtypes = [vp, vp, C.POINTER(C.c_int)]
        L.wino_profile_begin.restype = C.c_int
        L.wino_profile_begin.argtypes = [C.c_int]
        L.wino_profile_end.restype = C.c_int
        L.wino_profile_end.argtypes = [C.POINTER(C.c_double), C.POINTER(C.c_int)]
        L.wino_score_plan_host.restype = C.c_int
        L.wino_score_plan_host.argtypes = [i64, i64, i64, C.c_int32, C.c_int32, C.POINTER(C.c_int32)]
        L.wino_score_plan.restype = C.c_int
        L.wino_score_plan.argtypes = [i64, i64, i64, C.POINTER(C.c_int32)]
        L.wino_timeline_begin.restype = C.c_int
        L.wino_timeline_begin.argtypes = [vp, i64, i64]
        L.wino_timeline_end.restype = C.c_int
        L.wino_timeline_end.argtypes = [C.POINTER(i64)]
        L.wino_selftest_wait_timeout.restype = C.c_int
        L.wino_selftest_wait_timeout.argtypes = [vp, i64, vp]
        L.wino_status_string.restype = C.c_char_p
        L.wino_status_string.argtypes = [C.c_int]
        L.wino_version.restype = C.c_int
        L.wino_version.argtypes = []
        L.wino_decode.restype = C.c_int
        L.wino_decode.argtypes = [vp, i64, i64, vp, C.POINTER(WinoParams), C.c_int32, C.c_int32, C.c_int32,
                                  HIDDEN_FN, vp, vp, vp, vp, vp, vp, vp, sz, vp, C.POINTER(WinoBlockStats),
                                  C.POINTER(C.c_int32)]
        _lib = L
    return _lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int, where: str) -> None:
    if status != WINO_OK:
        raise WinoError(status, where)


def wino_status_string(status: int) -> str:
    return lib().wino_status_string(int(status)).decode()


def wino_version() -> int:
    return lib().wino_version()


def wino_workspace_size(N: int, d: int, V: int) -> int:
    out = C.c_size_t(0)
    _check(lib().wino_workspace_size(N, d, V, C.byref(out)), "wino_workspace_size")
    return out.value


def wino_workspace_size_step(params: WinoParams, d: int, V: int) -> int:
    out = C.c_size_t(0)
    _check(lib().wino_workspace_size_step(C.byref(params), d, V, C.byref(out)), "wino_workspace_size_step")
    return out.value


def step_workspace(params: WinoParams, d: int, V: int, device=None):
    """A zeroed uint8 device tensor of wino_workspace_size_step bytes (allocated by PyTorch)."""
    import torch
    return torch.zeros(wino_workspace_size_step(params, d, V), dtype=torch.uint8, device=device or "cuda")


def workspace(N: int, d: int, V: int, device=None):
    """A zeroed uint8 device tensor of wino_workspace_size(N, d, V) bytes (allocated by PyTorch)."""
    import torch
    return torch.zeros(wino_workspace_size(N, d, V), dtype=torch.uint8, device=device or "cuda")


def make_params(tau1: float, tau2: float, mask_id: int, n_seq: int, seq_len: int, blk_start: int, blk_len: int,
                max_steps: int = 4096, freeze_finished: bool = False, step_index: int = 0,
                last_change=None, no_shadow: bool = False, compact: bool = False, draft_m: int = 0,
                active_seq=None, n_active: int | None = None, w_panels: bool = False) -> WinoParams:
    """wino_params; ``draft_m`` > 0 selects fixed-M drafting (naive parallel sampling, Sec. 3);
    ``active_seq`` (device int32) lists the sequences a wino_step scores and updates (default: all);
    ``w_panels``: the W passed to the step is the panel copy of ``wino_lm_head_panels``."""
    opts = ((WINO_OPT_FREEZE_FINISHED if freeze_finished else 0) | (WINO_OPT_NO_SHADOW if no_shadow else 0) |
            (WINO_OPT_COMPACT if compact else 0) | (WINO_OPT_W_PANELS if w_panels else 0))
    if active_seq is not None and n_active is None:
        n_active = int(active_seq.numel())
    return WinoParams(tau1, tau2, mask_id, n_seq, seq_len, blk_start, blk_len, max_steps, opts, step_index,
                      _ptr(last_change), draft_m, _ptr(active_seq), n_active or 0)


def wino_score_rows(H, W, target, argmax, pmax, ptarget, ws, stream=None, *, entropy=None, N: int | None = None,
                    d: int | None = None, V: int | None = None) -> None:
    """Fused LM-head + full-vocabulary softmax statistics (and, given ``entropy``, H(p) per row);
    shapes default to H.shape / W.shape."""
    N = int(H.shape[0]) if N is None else N
    d = int(H.shape[1]) if d is None else d
    V = int(W.shape[0]) if V is None else V
    ws_bytes = ws.numel() * ws.element_size()
    _check(lib().wino_score_rows(_ptr(H), _ptr(W), N, d, V, _ptr(target), _ptr(argmax), _ptr(pmax), _ptr(ptarget),
                                 _ptr(entropy), _ptr(ws), ws_bytes, _stream(stream)), "wino_score_rows")


def wino_draft_verify(tokens, argmax, pmax, ptarget, params: WinoParams, counts, flags=None, stream=None) -> None:
    """Eq. 4 in place on ``tokens`` from per-row statistics."""
    _check(lib().wino_draft_verify(_ptr(tokens), _ptr(argmax), _ptr(pmax), _ptr(ptarget), C.byref(params),
                                   _ptr(counts), _ptr(flags), _stream(stream)), "wino_draft_verify")


def _vocab(W, params: WinoParams) -> int:
    """V from W's shape: [V, d] row-major, or [d/64, V, 64] for a panel copy (WINO_OPT_W_PANELS)."""
    return int(W.shape[1] if params.options & WINO_OPT_W_PANELS else W.shape[0])


def wino_lm_head_panels(W, Wp=None, stream=None):
    """The panel copy Wp[k][v][c] = W[v][64k + c] of a [V, d] bf16 LM head, as a [d/64, V, 64] tensor (written
    into ``Wp`` when given, else allocated by PyTorch); pass it as W with ``make_params(..., w_panels=True)``."""
    import torch
    V, d = int(W.shape[0]), int(W.shape[1])
    if Wp is None:
        Wp = torch.empty((d // 64, V, 64), dtype=W.dtype, device=W.device)
    _check(lib().wino_lm_head_panels(_ptr(W), d, V, _ptr(Wp), _stream(stream)), "wino_lm_head_panels")
    return Wp


def wino_step(H, W, tokens, params: WinoParams, counts, ws, flags=None, stream=None, *, d: int | None = None,
              V: int | None = None) -> None:
    """One whole WINO step in place on ``tokens``."""
    d = int(H.shape[1]) if d is None else d
    V = _vocab(W, params) if V is None else V
    ws_bytes = ws.numel() * ws.element_size()
    _check(lib().wino_step(_ptr(H), _ptr(W), d, V, _ptr(tokens), C.byref(params), _ptr(counts), _ptr(flags),
                           _ptr(ws), ws_bytes, _stream(stream)), "wino_step")


def wino_step_static_scratch(H, W, tokens, params: WinoParams, counts, flags=None, stream=None, *,
                             d: int | None = None, V: int | None = None) -> None:
    """wino_step with the library's fixed device scratch instead of a caller workspace (allocates nothing)."""
    d = int(H.shape[1]) if d is None else d
    V = _vocab(W, params) if V is None else V
    _check(lib().wino_step_static_scratch(_ptr(H), _ptr(W), d, V, _ptr(tokens), C.byref(params), _ptr(counts),
                                          _ptr(flags), _stream(stream)), "wino_step_static_scratch")


def wino_decode(W, tokens, params: WinoParams, n_blocks: int, hidden, counts, counts_host, ws, flags=None,
                stream=None, *, flags_host=None, active_buf=None, first_block: int = 0, first_step: int = 0,
                d: int | None = None, V: int | None = None):
    """The library's decode loop (wino_decode).  ``hidden(k, blk_start)`` returns step k's device bf16
    hidden states (a tensor, kept alive until the next call); ``counts_host`` is a host int32 [n_seq, 3]
    tensor (pinned for speed); with ``flags`` and a host int8 ``flags_host`` the at-least-one drafts are
    counted too; with a device int32 [n_seq] ``active_buf`` only the sequences whose block still has a
    MASK are stepped.  Returns (status, per-block (steps, drafted, re-masked, at-least-one drafts,
    sequences stepped summed over the steps), next step index); the status is
    WINO_OK or the error that stopped the loop (an exception raised by ``hidden`` is re-raised)."""
    if params.options & WINO_OPT_W_PANELS:  # [d/64, V, 64]
        d = int(W.shape[0]) * 64 if d is None else d
    else:
        d = int(W.shape[1]) if d is None else d
    V = _vocab(W, params) if V is None else V
    held, failure = [None], []

    def cb(user, k, blk_start):
        try:
            H = hidden(int(k), int(blk_start))
            held[0] = H
            return _ptr(H)
        except BaseException as e:  # reported after the call: an exception cannot cross the C frame
            failure.append(e)
            return None

    fn = HIDDEN_FN(cb)
    stats = (WinoBlockStats * n_blocks)()
    nxt = C.c_int32(0)
    ws_bytes = ws.numel() * ws.element_size()
    rc = lib().wino_decode(_ptr(W), d, V, _ptr(tokens), C.byref(params), n_blocks, first_block, first_step, fn,
                           None, _ptr(counts), _ptr(counts_host), _ptr(flags), _ptr(flags_host), _ptr(active_buf),
                           _ptr(ws), ws_bytes, _stream(stream),
                           stats, C.byref(nxt))
    if failure:
        raise failure[0]
    return rc, [(b.steps, b.drafted, b.remasked, b.fallback, b.seq_steps) for b in stats], nxt.value


def wino_read_device_status(ws, stream=None) -> int:
    out = C.c_int(0)
    _check(lib().wino_read_device_status(_ptr(ws), _stream(stream), C.byref(out)), "wino_read_device_status")
    return out.value


def wino_profile_begin(max_launches: int) -> None:
    _check(lib().wino_profile_begin(int(max_launches)), "wino_profile_begin")


def wino_profile_end() -> tuple[float, int]:
    """(summed score-kernel milliseconds, number of launches timed)."""
    ms, n = C.c_double(0), C.c_int(0)
    _check(lib().wino_profile_end(C.byref(ms), C.byref(n)), "wino_profile_end")
    return ms.value, n.value


def wino_score_plan(N: int, d: int, V: int) -> dict:
    """The score kernel's work split for N rows over V entries on the current device."""
    out = (C.c_int32 * 8)()
    _check(lib().wino_score_plan(int(N), int(d), int(V), out), "wino_score_plan")
    return dict(zip(("bn", "n_vt", "n_mb", "n_groups", "G", "ctas", "two", "stages"), list(out)))


def wino_score_plan_host(N: int, d: int, V: int, sm_count: int = 152, max_pairs: int = 76) -> dict:
    """The score kernel's work split for a device with sm_count SMs and max_pairs resident pairs (no device)."""
    out = (C.c_int32 * 10)()
    _check(lib().wino_score_plan_host(int(N), int(d), int(V), int(sm_count), int(max_pairs), out),
           "wino_score_plan_host")
    return dict(zip(("bn", "n_vt", "n_mb", "n_groups", "G", "ctas", "two", "stages", "stage_bytes",
                     "records_per_row"), list(out)))


def wino_timeline_begin(buf, n_launches: int, ctas_per_launch: int) -> None:
    """Start recording per-CTA score-kernel stamps into the device uint64 tensor ``buf``
    (n_launches * ctas_per_launch * TIMELINE_WORDS words)."""
    _check(lib().wino_timeline_begin(_ptr(buf), int(n_launches), int(ctas_per_launch)), "wino_timeline_begin")


def wino_timeline_end() -> int:
    """Stop recording; returns the number of score launches counted."""
    n = C.c_int64(0)
    _check(lib().wino_timeline_end(C.byref(n)), "wino_timeline_end")
    return n.value


def wino_selftest_wait_timeout(status, limit_ns: int, stream=None) -> None:
    """Run the bounded-wait timeout self-test; ``status`` (device int32) receives the outcome."""
    _check(lib().wino_selftest_wait_timeout(_ptr(status), int(limit_ns), _stream(stream)),
           "wino_selftest_wait_timeout")
