"""ctypes binding of libprcr.so (argument marshalling only).

Every function here has the name of the C entry point it wraps (without the
``prcr_`` prefix) and forwards torch tensors as raw device pointers; all of
the work runs in the library's CUDA kernels. There is no fallback: if the
library is missing or cannot be loaded, ``lib()`` raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libprcr.so")

# return codes / status bits / modes / flags / layouts / cache kinds (mirror include/prcr.h)
OK, EINVAL, EALIGN, EWORKSPACE, ECUDA = 0, -1, -2, -3, -4
ST_IDX_RANGE, ST_NO_BLOCK, ST_CAPACITY, ST_CSR, ST_POS_RANGE = 1, 2, 4, 8, 16
MODE_PCR, MODE_ORIGINAL, MODE_UIR, MODE_LPA = 0, 1, 2, 3
FLAG_DEGENERATE_CENTER = 1
LAYOUT_SECTIONED, LAYOUT_INTERLEAVED = 0, 1
CACHE_CONTIGUOUS, CACHE_PAGED = 0, 1

EXPORTS = ("prcr_workspace_size", "prcr_rebind_inject", "prcr_plan", "prcr_rebind_apply",
           "prcr_store_raw", "prcr_next_text_pos", "prcr_error_string", "prcr_version",
           "prcr_rebind_inject_static", "prcr_prefill_capture", "prcr_decode_workspace_size",
           "prcr_decode_attention", "prcr_select_workspace_size", "prcr_select_topk",
           "prcr_select_topk_cached")
STATIC_MAX_TOKENS = 65536


class RopeCfg(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32),
                ("sections", C.c_int32 * 3), ("layout", C.c_int32), ("reserved", C.c_int32),
                ("theta", C.c_double)]


class StoreDesc(C.Structure):
    _fields_ = [("k", C.c_void_p), ("v", C.c_void_p), ("coords", C.c_void_p),
                ("seq_stride", C.c_int64), ("layer_stride", C.c_int64),
                ("token_stride", C.c_int64), ("coord_seq_stride", C.c_int64),
                ("n_seqs", C.c_int32), ("n_tokens", C.c_int32)]


class CacheDesc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("block_size", C.c_int32), ("k", C.c_void_p),
                ("v", C.c_void_p), ("seq_stride", C.c_int64), ("layer_stride", C.c_int64),
                ("block_stride", C.c_int64), ("slot_stride", C.c_int64),
                ("block_table", C.c_void_p), ("bt_stride", C.c_int32), ("n_blocks", C.c_int32),
                ("max_slots", C.c_int32), ("n_seqs", C.c_int32)]


class RevisitBatch(C.Structure):
    _fields_ = [("seq_rev_off", C.c_void_p), ("rev_tok_off", C.c_void_p), ("idx", C.c_void_p),
                ("p_txt", C.c_void_p), ("cache_len_in", C.c_void_p), ("n_seqs", C.c_int32),
                ("n_revisits", C.c_int32), ("total_k", C.c_int64)]


class Outputs(C.Structure):
    _fields_ = [("cache_len_out", C.c_void_p), ("next_pos_out", C.c_void_p),
                ("pos_out", C.c_void_p), ("slot_out", C.c_void_p), ("status", C.c_void_p)]


_lib = None


def lib():
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libprcr.so not built ({LIB_PATH}); run __graft_entry__.build()")
    L = C.CDLL(LIB_PATH)
    P = C.POINTER
    L.prcr_workspace_size.argtypes = [C.c_int64]
    L.prcr_workspace_size.restype = C.c_size_t
    call = [P(RopeCfg), P(StoreDesc), P(CacheDesc), P(RevisitBatch), P(Outputs), C.c_int32,
            C.c_int32, C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p]
    for name in ("prcr_rebind_inject", "prcr_plan", "prcr_rebind_apply"):
        getattr(L, name).argtypes = call
        getattr(L, name).restype = C.c_int
    L.prcr_rebind_inject_static.argtypes = call[:8] + [C.c_void_p]
    L.prcr_rebind_inject_static.restype = C.c_int
    L.prcr_store_raw.argtypes = [P(RopeCfg), P(StoreDesc), C.c_int32, C.c_int32, C.c_int32,
                                 C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_int64,
                                 C.c_int64, C.c_void_p, C.c_void_p]
    L.prcr_store_raw.restype = C.c_int
    L.prcr_prefill_capture.argtypes = [P(RopeCfg), P(StoreDesc), P(CacheDesc), C.c_int32,
                                       C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                       C.c_void_p, C.c_void_p, C.c_int64, C.c_int64, C.c_void_p,
                                       C.c_void_p, C.c_void_p]
    L.prcr_prefill_capture.restype = C.c_int
    L.prcr_decode_workspace_size.argtypes = [P(RopeCfg), C.c_int32, C.c_int32, C.c_int64]
    L.prcr_decode_workspace_size.restype = C.c_size_t
    L.prcr_decode_attention.argtypes = [P(RopeCfg), P(CacheDesc), C.c_int32, C.c_int32,
                                        C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64,
                                        C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t,
                                        C.c_void_p]
    L.prcr_decode_attention.restype = C.c_int
    L.prcr_select_workspace_size.argtypes = [C.c_int32, C.c_int32, C.c_int32]
    L.prcr_select_workspace_size.restype = C.c_size_t
    L.prcr_select_topk.argtypes = [P(RopeCfg), P(StoreDesc), C.c_int32, C.c_int32, C.c_int32,
                                   C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p,
                                   C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]
    L.prcr_select_topk.restype = C.c_int
    L.prcr_select_topk_cached.argtypes = [P(RopeCfg), P(CacheDesc), C.c_int32, C.c_int32,
                                          C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                          C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                          C.c_size_t, C.c_void_p]
    L.prcr_select_topk_cached.restype = C.c_int
    L.prcr_next_text_pos.argtypes = [C.c_int64, C.c_int64, C.c_int32]
    L.prcr_next_text_pos.restype = C.c_int64
    L.prcr_error_string.argtypes = [C.c_int]
    L.prcr_error_string.restype = C.c_char_p
    L.prcr_version.argtypes = []
    L.prcr_version.restype = C.c_int
    _lib = L
    return L


class PrcrError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {lib().prcr_error_string(code).decode()} ({code})")
        self.code = code


def _check(code: int, where: str) -> int:
    if code != OK:
        raise PrcrError(code, where)
    return code


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ----------------------------------------------------------------------------
# descriptors built from torch tensors
# ----------------------------------------------------------------------------
def rope_cfg(n_layers: int, n_kv_heads: int, head_dim: int, sections, theta: float = 1e6,
             layout: int = LAYOUT_SECTIONED) -> RopeCfg:
    c = RopeCfg()
    c.n_layers, c.n_kv_heads, c.head_dim = n_layers, n_kv_heads, head_dim
    c.sections[0], c.sections[1], c.sections[2] = (int(s) for s in sections)
    c.layout, c.reserved, c.theta = layout, 0, float(theta)
    return c


def _bf16(t: torch.Tensor, name: str):
    if t.dtype != torch.bfloat16:
        raise TypeError(f"{name} must be bfloat16")
    if t.stride(-1) != 1 or t.stride(-2) != t.shape[-1]:
        raise ValueError(f"{name}: a [heads, head_dim] row must be contiguous")


def store_desc(k: torch.Tensor, v: torch.Tensor, coords: torch.Tensor) -> StoreDesc:
    """k, v: [B, n_L, M, H, D] bf16 (row-contiguous, equal strides); coords: [B, M, 3] int32."""
    _bf16(k, "store k"); _bf16(v, "store v")
    if k.stride() != v.stride() or k.shape != v.shape:
        raise ValueError("store k and v must have the same shape and strides")
    if coords.dtype != torch.int32 or coords.stride(-1) != 1 or coords.stride(-2) != 3:
        raise ValueError("coords must be int32 [B, M, 3] with contiguous rows")
    d = StoreDesc()
    d.k, d.v, d.coords = k.data_ptr(), v.data_ptr(), coords.data_ptr()
    d.seq_stride, d.layer_stride, d.token_stride = k.stride(0), k.stride(1), k.stride(2)
    d.coord_seq_stride = coords.stride(0)
    d.n_seqs, d.n_tokens = k.shape[0], k.shape[2]
    d._keep = (k, v, coords)
    return d


def cache_contiguous(k: torch.Tensor, v: torch.Tensor) -> CacheDesc:
    """k, v: [B, n_L, S, H, D] bf16."""
    _bf16(k, "cache k"); _bf16(v, "cache v")
    if k.stride() != v.stride() or k.shape != v.shape:
        raise ValueError("cache k and v must have the same shape and strides")
    d = CacheDesc()
    d.kind, d.block_size = CACHE_CONTIGUOUS, 1
    d.k, d.v = k.data_ptr(), v.data_ptr()
    d.seq_stride, d.layer_stride, d.slot_stride = k.stride(0), k.stride(1), k.stride(2)
    d.block_stride, d.block_table, d.bt_stride, d.n_blocks = 0, None, 0, 0
    d.max_slots, d.n_seqs = k.shape[2], k.shape[0]
    d._keep = (k, v)
    return d


def cache_paged(k: torch.Tensor, v: torch.Tensor, block_table: torch.Tensor) -> CacheDesc:
    """k, v: [n_L, n_blocks, block_size, H, D] bf16; block_table: [B, max_blocks] int32."""
    _bf16(k, "cache k"); _bf16(v, "cache v")
    if k.stride() != v.stride() or k.shape != v.shape:
        raise ValueError("cache k and v must have the same shape and strides")
    if block_table.dtype != torch.int32 or block_table.stride(-1) != 1:
        raise ValueError("block_table must be int32 [B, max_blocks] with contiguous rows")
    d = CacheDesc()
    d.kind, d.block_size = CACHE_PAGED, k.shape[2]
    d.k, d.v = k.data_ptr(), v.data_ptr()
    d.seq_stride, d.layer_stride = 0, k.stride(0)
    d.block_stride, d.slot_stride = k.stride(1), k.stride(2)
    d.block_table, d.bt_stride = block_table.data_ptr(), block_table.stride(0)
    d.n_blocks, d.max_slots, d.n_seqs = k.shape[1], 0, block_table.shape[0]
    d._keep = (k, v, block_table)
    return d


def revisit_batch(seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in) -> RevisitBatch:
    for name, t, dt in (("seq_rev_off", seq_rev_off, torch.int32), ("rev_tok_off", rev_tok_off, torch.int32),
                        ("idx", idx, torch.int32), ("p_txt", p_txt, torch.int64),
                        ("cache_len_in", cache_len_in, torch.int32)):
        if t.dtype != dt or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous {dt} tensor")
    b = RevisitBatch()
    b.seq_rev_off, b.rev_tok_off = seq_rev_off.data_ptr(), rev_tok_off.data_ptr()
    b.idx = idx.data_ptr() if idx.numel() else None
    b.p_txt, b.cache_len_in = p_txt.data_ptr(), cache_len_in.data_ptr()
    b.n_seqs, b.n_revisits, b.total_k = seq_rev_off.numel() - 1, rev_tok_off.numel() - 1, idx.numel()
    b._keep = (seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in)
    return b


def outputs(cache_len_out, next_pos_out, status, pos_out=None, slot_out=None) -> Outputs:
    o = Outputs()
    o.cache_len_out, o.next_pos_out, o.status = (cache_len_out.data_ptr(), next_pos_out.data_ptr(),
                                                 status.data_ptr())
    o.pos_out, o.slot_out = _ptr(pos_out), _ptr(slot_out)
    o._keep = (cache_len_out, next_pos_out, status, pos_out, slot_out)
    return o


# ----------------------------------------------------------------------------
# entry points
# ----------------------------------------------------------------------------
def workspace_size(total_k: int) -> int:
    return int(lib().prcr_workspace_size(int(total_k)))


def _call(name, cfg, store, cache, batch, out, mode, L, flags, workspace, stream):
    ws = None if workspace is None else workspace.data_ptr()
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = getattr(lib(), name)(C.byref(cfg), C.byref(store), C.byref(cache), C.byref(batch),
                              C.byref(out), int(mode), int(L), int(flags), ws, nbytes,
                              _stream(stream))
    return _check(rc, name)


def rebind_inject(cfg, store, cache, batch, out, mode=MODE_PCR, L=2, flags=0, workspace=None,
                  stream=None):
    """prcr_rebind_inject: plan + rebind/inject on ``stream`` (default: torch's current)."""
    return _call("prcr_rebind_inject", cfg, store, cache, batch, out, mode, L, flags, workspace, stream)


def plan(cfg, store, cache, batch, out, mode=MODE_PCR, L=2, flags=0, workspace=None, stream=None):
    """prcr_plan: positions, slots and per-sequence outputs only."""
    return _call("prcr_plan", cfg, store, cache, batch, out, mode, L, flags, workspace, stream)


def rebind_apply(cfg, store, cache, batch, out, mode=MODE_PCR, L=2, flags=0, workspace=None,
                 stream=None):
    """prcr_rebind_apply: the row-moving half, consuming a preceding prcr_plan."""
    return _call("prcr_rebind_apply", cfg, store, cache, batch, out, mode, L, flags, workspace, stream)


def rebind_inject_static(cfg, store, cache, batch, out, mode=MODE_PCR, L=2, flags=0, stream=None):
    """prcr_rebind_inject_static: the same call with the library's own fixed
    scratch instead of a caller workspace (for callers that cannot allocate
    device memory); at most STATIC_MAX_TOKENS selected tokens per call, and
    calls must not overlap on the GPU."""
    rc = lib().prcr_rebind_inject_static(C.byref(cfg), C.byref(store), C.byref(cache),
                                         C.byref(batch), C.byref(out), int(mode), int(L),
                                         int(flags), _stream(stream))
    return _check(rc, "prcr_rebind_inject_static")


def store_raw(cfg, store, seq: int, layer_begin: int, m_begin: int, k_src: torch.Tensor,
              v_src: torch.Tensor, coords_src: Optional[torch.Tensor] = None, stream=None):
    """prcr_store_raw: k_src / v_src are [n_layers, m_count, H, D] bf16 (row-contiguous)."""
    _bf16(k_src, "k_src"); _bf16(v_src, "v_src")
    if k_src.stride() != v_src.stride() or k_src.shape != v_src.shape:
        raise ValueError("k_src and v_src must have the same shape and strides")
    if coords_src is not None and (coords_src.dtype != torch.int32 or not coords_src.is_contiguous()):
        raise TypeError("coords_src must be a contiguous int32 [m_count, 3] tensor")
    rc = lib().prcr_store_raw(C.byref(cfg), C.byref(store), int(seq), int(layer_begin),
                              int(k_src.shape[0]), int(m_begin), int(k_src.shape[1]),
                              k_src.data_ptr(), v_src.data_ptr(), k_src.stride(0), k_src.stride(1),
                              _ptr(coords_src), _stream(stream))
    return _check(rc, "prcr_store_raw")


def prefill_capture(cfg, store, cache, seq: int, layer_begin: int, m_begin: int, slot_begin: int,
                    k_src: torch.Tensor, v_src: torch.Tensor, coords_src: torch.Tensor,
                    status: torch.Tensor, stream=None):
    """prcr_prefill_capture: k_src / v_src are the prefill's pre-rotation rows
    [n_layers, m_count, H, D] bf16 (row-contiguous); coords_src [m_count, 3] int32."""
    _bf16(k_src, "k_src"); _bf16(v_src, "v_src")
    if k_src.stride() != v_src.stride() or k_src.shape != v_src.shape:
        raise ValueError("k_src and v_src must have the same shape and strides")
    if coords_src.dtype != torch.int32 or not coords_src.is_contiguous():
        raise TypeError("coords_src must be a contiguous int32 [m_count, 3] tensor")
    rc = lib().prcr_prefill_capture(C.byref(cfg), C.byref(store), C.byref(cache), int(seq),
                                    int(layer_begin), int(k_src.shape[0]), int(m_begin),
                                    int(k_src.shape[1]), int(slot_begin), k_src.data_ptr(),
                                    v_src.data_ptr(), k_src.stride(0), k_src.stride(1),
                                    coords_src.data_ptr(), status.data_ptr(), _stream(stream))
    return _check(rc, "prcr_prefill_capture")


def decode_workspace_size(cfg, n_seqs: int, n_q_heads: int, max_len: int) -> int:
    return int(lib().prcr_decode_workspace_size(C.byref(cfg), int(n_seqs), int(n_q_heads),
                                                int(max_len)))


def decode_attention(cfg, cache, q: torch.Tensor, q_pos: torch.Tensor, seq_len: torch.Tensor,
                     max_len: int, out: torch.Tensor, status: torch.Tensor,
                     workspace: Optional[torch.Tensor] = None, stream=None):
    """prcr_decode_attention: q [B, n_layers, Hq, D] bf16 (contiguous), q_pos int64 [B],
    seq_len int32 [B], out float32 [B, n_layers, Hq, D]."""
    if q.dtype != torch.bfloat16 or not q.is_contiguous():
        raise TypeError("q must be a contiguous bfloat16 [B, n_layers, Hq, D] tensor")
    if out.dtype != torch.float32 or not out.is_contiguous() or out.shape != q.shape:
        raise TypeError("out must be a contiguous float32 tensor shaped like q")
    if q_pos.dtype != torch.int64 or seq_len.dtype != torch.int32:
        raise TypeError("q_pos must be int64 and seq_len int32")
    ws = None if workspace is None else workspace.data_ptr()
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = lib().prcr_decode_attention(C.byref(cfg), C.byref(cache), int(q.shape[0]), int(q.shape[2]),
                                     q.data_ptr(), q_pos.data_ptr(), seq_len.data_ptr(),
                                     int(max_len), out.data_ptr(), status.data_ptr(), ws, nbytes,
                                     _stream(stream))
    return _check(rc, "prcr_decode_attention")


def select_workspace_size(n_seqs: int, n_q_heads: int, n_tokens: int) -> int:
    return int(lib().prcr_select_workspace_size(int(n_seqs), int(n_q_heads), int(n_tokens)))


def select_topk(cfg, store, layer: int, q: torch.Tensor, q_pos: torch.Tensor, k: int,
                idx_out: torch.Tensor, seq_rev_off: torch.Tensor, rev_tok_off: torch.Tensor,
                workspace: torch.Tensor, score_out: Optional[torch.Tensor] = None, stream=None):
    """prcr_select_topk: q [B, Hq, D] bf16 (contiguous); q_pos int64 [B]; outputs
    idx_out int32 [B * k], seq_rev_off / rev_tok_off int32 [B + 1]."""
    if q.dtype != torch.bfloat16 or not q.is_contiguous():
        raise TypeError("q must be a contiguous bfloat16 [B, Hq, D] tensor")
    for name, t in (("idx_out", idx_out), ("seq_rev_off", seq_rev_off), ("rev_tok_off", rev_tok_off)):
        if t.dtype != torch.int32 or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous int32 tensor")
    rc = lib().prcr_select_topk(C.byref(cfg), C.byref(store), int(q.shape[0]), int(layer),
                                int(q.shape[1]), q.data_ptr(), q_pos.data_ptr(), int(k),
                                idx_out.data_ptr(), seq_rev_off.data_ptr(), rev_tok_off.data_ptr(),
                                _ptr(score_out), workspace.data_ptr(),
                                workspace.numel() * workspace.element_size(), _stream(stream))
    return _check(rc, "prcr_select_topk")


def select_topk_cached(cfg, cache, layer: int, q: torch.Tensor, q_pos: torch.Tensor,
                       img_slot0: torch.Tensor, n_tokens: int, k: int, idx_out: torch.Tensor,
                       seq_rev_off: torch.Tensor, rev_tok_off: torch.Tensor, status: torch.Tensor,
                       workspace: torch.Tensor, score_out: Optional[torch.Tensor] = None,
                       stream=None):
    """prcr_select_topk_cached: the selection read from the position-bound
    cache `cache`; sequence b's n_tokens visual tokens occupy slots
    img_slot0[b] .. (int32 [B]). Other arguments as select_topk; status is
    the device status word (int32 [1])."""
    if q.dtype != torch.bfloat16 or not q.is_contiguous():
        raise TypeError("q must be a contiguous bfloat16 [B, Hq, D] tensor")
    for name, t in (("idx_out", idx_out), ("seq_rev_off", seq_rev_off), ("rev_tok_off", rev_tok_off),
                    ("img_slot0", img_slot0)):
        if t.dtype != torch.int32 or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous int32 tensor")
    rc = lib().prcr_select_topk_cached(C.byref(cfg), C.byref(cache), int(q.shape[0]), int(layer),
                                       int(q.shape[1]), int(n_tokens), img_slot0.data_ptr(),
                                       q.data_ptr(), q_pos.data_ptr(), int(k), idx_out.data_ptr(),
                                       seq_rev_off.data_ptr(), rev_tok_off.data_ptr(),
                                       _ptr(score_out), status.data_ptr(), workspace.data_ptr(),
                                       workspace.numel() * workspace.element_size(), _stream(stream))
    return _check(rc, "prcr_select_topk_cached")


def next_text_pos(p_txt: int, k_seq: int, mode: int = MODE_PCR) -> int:
    return int(lib().prcr_next_text_pos(int(p_txt), int(k_seq), int(mode)))


def version() -> int:
    return int(lib().prcr_version())
