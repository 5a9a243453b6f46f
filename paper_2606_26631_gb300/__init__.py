"""PRCR visual-revisit path for GB300 (sm_103a): Python binding of libprcr.so.

The C ABI (include/prcr.h) does the work: position reassignment of revisited
visual tokens (Sec. 3.2), M-RoPE rebinding of their raw keys and injection of
K/V into the active decoder cache (Sec. 3.3). This package only marshals torch
tensors into those calls; it has no CPU fallback.
"""
from ._binding import (  # noqa: F401
    CACHE_CONTIGUOUS, CACHE_PAGED, EXPORTS, FLAG_DEGENERATE_CENTER, LAYOUT_INTERLEAVED,
    LAYOUT_SECTIONED, MODE_LPA, MODE_ORIGINAL, MODE_PCR, MODE_UIR, ST_CAPACITY, ST_CSR,
    ST_IDX_RANGE, ST_NO_BLOCK, ST_POS_RANGE, PrcrError, cache_contiguous, cache_paged,
    decode_attention, decode_workspace_size, lib,
    next_text_pos, outputs, plan, prefill_capture, rebind_apply, rebind_inject, rebind_inject_static,
    revisit_batch, rope_cfg, select_topk, select_topk_cached, select_workspace_size,
    store_desc, store_raw, version, workspace_size)
from .revisit import Revisit  # noqa: F401
