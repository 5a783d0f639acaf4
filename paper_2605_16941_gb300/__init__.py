"""GB300-native (sm_103a) WINO scoring-and-revoke step.

WINO ("Wide-In, Narrow-Out", arXiv 2605.16941, Sec. 4) is a revokable
decoding rule for diffusion LLMs: per step it drafts every masked position
whose confidence exceeds tau1 (Eq. 2), re-masks every decoded position whose
shadow-block verification probability is below tau2 (Eq. 3), both from one
forward pass (Eq. 4).  This package is the per-step hot path after the
transformer: the LM-head GEMM fused with a full-vocabulary online softmax,
the cross-tile merge, and the in-place state update, as CUDA kernels behind
a C ABI (``include/wino.h``).  The Python side marshals arguments only.
"""
from ._abi import (EXPORTS, WINO_STATIC_SCRATCH_BYTES, FLAG_DRAFT, FLAG_DRAFT_FALLBACK, FLAG_DRAFT_IS_MASK, FLAG_NONE, FLAG_REMASK,
                   FLAG_DRAFT_TOP_M, TIMELINE_WORDS, wino_timeline_begin, wino_timeline_end, wino_score_plan, wino_score_plan_host,
                   WINO_ERR_ARG, WINO_ERR_CUDA, WINO_ERR_DEVICE_TIMEOUT, WINO_ERR_MAX_STEPS, WINO_ERR_SHAPE,
                   WINO_ERR_UNSUPPORTED, WINO_ERR_WORKSPACE, WINO_OK, WINO_OPT_FREEZE_FINISHED, WINO_OPT_NO_SHADOW, WINO_OPT_COMPACT, WINO_OPT_W_PANELS, wino_lm_head_panels, step_workspace, wino_workspace_size_step, WinoError, WinoParams, lib, library_path,
                   make_params, wino_draft_verify, wino_profile_begin, wino_profile_end, wino_read_device_status, wino_score_rows, wino_status_string, wino_step_static_scratch, wino_selftest_wait_timeout,
                   wino_step, wino_version, wino_workspace_size, workspace, wino_decode, WinoBlockStats)

__all__ = [
    "EXPORTS", "WINO_STATIC_SCRATCH_BYTES", "FLAG_DRAFT", "FLAG_DRAFT_FALLBACK", "FLAG_DRAFT_IS_MASK", "FLAG_NONE", "FLAG_REMASK",
    "FLAG_DRAFT_TOP_M", "TIMELINE_WORDS", "wino_timeline_begin", "wino_timeline_end", "wino_score_plan", "wino_score_plan_host",
    "WINO_ERR_ARG", "WINO_ERR_CUDA", "WINO_ERR_DEVICE_TIMEOUT", "WINO_ERR_MAX_STEPS", "WINO_ERR_SHAPE",
    "WINO_ERR_UNSUPPORTED", "WINO_ERR_WORKSPACE", "WINO_OK", "WINO_OPT_FREEZE_FINISHED", "WINO_OPT_NO_SHADOW", "WINO_OPT_COMPACT", "WINO_OPT_W_PANELS", "wino_lm_head_panels", "step_workspace", "wino_workspace_size_step", "WinoError", "WinoParams", "lib", "library_path",
    "make_params", "wino_draft_verify", "wino_profile_begin", "wino_profile_end", "wino_read_device_status", "wino_score_rows", "wino_status_string", "wino_step_static_scratch", "wino_selftest_wait_timeout",
    "wino_step", "wino_version", "wino_workspace_size", "workspace", "wino_decode", "WinoBlockStats",
]
