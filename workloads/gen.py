"""Seeded synthetic inputs for the revisit path.

Shared by the CUDA path's tests/bench and by the oracle's tests. It only makes
inputs: the raw visual store (pre-rotation K/V, Eq. "raw_kv"), each visual
token's original (t, h, w) coordinate, the revisited index sets (Eq. 3), the
current text position and the existing decoder cache with its block table.
It holds none of the method's arithmetic: no coordinate range, no position
reassignment, no rotation, no slot computation.

Seeds: K/V draw from a torch generator seeded ``seed`` on the target device;
selections use numpy PCG64 seeded ``seed + 1``; text positions and the block
shuffle use numpy PCG64 seeded ``seed + 2``.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional, Tuple

import numpy as np
import torch

from .configs import Workload

CANARY_BITS = -1  # int16 bit pattern 0xFFFF (a bf16 NaN) marks cache slots nobody wrote
IMAGE_BASE = 16   # position of the first visual token (a short text prefix precedes it)
IMAGE_GAP = 24    # text tokens between two images of one sequence


@dataclass
class Batch:
    wl: Workload
    store_k: torch.Tensor          # bf16 [B, n_L, M, H, D]
    store_v: torch.Tensor          # bf16 [B, n_L, M, H, D]
    coords: torch.Tensor           # int32 [B, M, 3], original (t, h, w)
    seq_rev_off: torch.Tensor      # int32 [B+1]
    rev_tok_off: torch.Tensor      # int32 [R+1]
    idx: torch.Tensor              # int32 [sum K]
    p_txt: torch.Tensor            # int64 [B]
    cache_len_in: torch.Tensor     # int32 [B]
    cache_k: torch.Tensor          # bf16 contiguous [B, n_L, S, H, D] or paged [n_L, NB, bs, H, D]
    cache_v: torch.Tensor
    block_table: Optional[torch.Tensor]  # int32 [B, max_blocks] (paged), -1 = unmapped
    revisits: List[Tuple[int, np.ndarray]]  # host copy: (sequence, token ids) per revisit

    @property
    def n_revisits(self) -> int:
        return int(self.rev_tok_off.numel() - 1)

    @property
    def total_k(self) -> int:
        return int(self.idx.numel())

    @property
    def paged(self) -> bool:
        return self.block_table is not None

    def algorithmic_bytes(self) -> int:
        """Bytes the path must move: read K_raw and V_raw, write K and V, per
        (token, layer, kv-head) row of D bf16 elements."""
        wl = self.wl
        return self.total_k * wl.n_layers * wl.n_kv_heads * wl.head_dim * 8


# ----------------------------------------------------------------------------
# visual grids and coordinates
# ----------------------------------------------------------------------------
def grid_layout(wl: Workload):
    """Per grid: (first token id, frames, rows, cols, coordinate base)."""
    out = []
    m0, base = 0, IMAGE_BASE
    for f, r, c in wl.grids:
        out.append((m0, f, r, c, base))
        m0 += f * r * c
        base += max(f, r, c) + IMAGE_GAP
    return out


def token_coords(wl: Workload) -> np.ndarray:
    """[M, 3] int32 original coordinates: token (frame, row, col) of a grid with
    base s sits at (s + frame, s + row, s + col), the layout Qwen2-VL style
    multimodal RoPE gives visual tokens."""
    coords = np.zeros((wl.n_tokens, 3), dtype=np.int32)
    for m0, f, r, c, s in grid_layout(wl):
        ff, rr, cc = np.meshgrid(np.arange(f), np.arange(r), np.arange(c), indexing="ij")
        n = f * r * c
        coords[m0:m0 + n, 0] = s + ff.reshape(-1)
        coords[m0:m0 + n, 1] = s + rr.reshape(-1)
        coords[m0:m0 + n, 2] = s + cc.reshape(-1)
    return coords


def _tok(layout, g, f, r, c) -> int:
    m0, _, rows, cols, _ = layout[g]
    return m0 + (f * rows + r) * cols + c


def _rect_ids(layout, g, f0, nf, r0, nr, c0, nc) -> np.ndarray:
    ids = [_tok(layout, g, f, r, c)
           for f in range(f0, f0 + nf) for r in range(r0, r0 + nr) for c in range(c0, c0 + nc)]
    return np.asarray(ids, dtype=np.int32)


def _disjoint_rects(rng, rows, cols, areas) -> List[Tuple[int, int, int, int]]:
    """Non-overlapping rectangles (r0, nr, c0, nc) with roughly the given areas."""
    taken = np.zeros((rows, cols), dtype=bool)
    rects = []
    for area in areas:
        for _ in range(10000):
            nr = int(rng.integers(max(2, area // cols + 1), min(rows, max(3, area // 2)) + 1))
            nc = max(1, min(cols, int(round(area / nr))))
            r0 = int(rng.integers(0, rows - nr + 1))
            c0 = int(rng.integers(0, cols - nc + 1))
            if not taken[r0:r0 + nr, c0:c0 + nc].any():
                taken[r0:r0 + nr, c0:c0 + nc] = True
                rects.append((r0, nr, c0, nc))
                break
        else:
            raise RuntimeError("could not place rectangle")
    return rects


def selections(wl: Workload, rng, rects_out: Optional[list] = None) -> List[List[np.ndarray]]:
    """Per sequence, the list of revisited index sets (Eq. 3), each in the
    order a caller would hand them over (rectangle by rectangle, row-major).
    If ``rects_out`` is a list, it receives per sequence, per revisit, the
    rectangles as drawn: (grid, first frame, frames, first row, rows, first
    column, columns) each, or an empty list for scattered tokens."""
    layout = grid_layout(wl)
    out = []
    for _ in range(wl.n_seqs):
        revs = []
        drawn = []
        if wl.selection == "rect4x4":
            r0 = int(rng.integers(0, 5)); c0 = int(rng.integers(0, 5))
            revs.append(_rect_ids(layout, 0, 0, 1, r0, 4, c0, 4))
            drawn.append([(0, 0, 1, r0, 4, c0, 4)])
        elif wl.selection in ("rects3_256", "rectset512"):
            _, _, rows, cols, _ = layout[0]
            if wl.selection == "rects3_256":
                areas = [85, 85, 86]
            else:
                n = int(rng.integers(2, 5))
                areas = [512 // n] * n
            rects = _disjoint_rects(rng, rows, cols, areas)
            revs.append(np.concatenate([_rect_ids(layout, 0, 0, 1, *rc) for rc in rects]))
            drawn.append([(0, 0, 1) + tuple(rc) for rc in rects])
        elif wl.selection == "rev4_256_1024":
            for _ in range(4):
                g = int(rng.integers(0, len(layout)))
                _, _, rows, cols, _ = layout[g]
                area = int(rng.integers(256, 1025))
                nr = int(rng.integers(max(4, -(-area // cols)), min(rows, area // 4) + 1))
                nc = min(cols, max(1, int(round(area / nr))))
                r0 = int(rng.integers(0, rows - nr + 1)); c0 = int(rng.integers(0, cols - nc + 1))
                revs.append(_rect_ids(layout, g, 0, 1, r0, nr, c0, nc))
                drawn.append([(g, 0, 1, r0, nr, c0, nc)])
        elif wl.selection == "video_stress":
            _, frames, rows, cols, _ = layout[0]
            fr = rng.choice(frames, size=2, replace=False)
            for f in fr:
                revs.append(_rect_ids(layout, 0, int(f), 1, 0, rows, 0, cols))
                drawn.append([(0, int(f), 1, 0, rows, 0, cols)])
            f0 = int(rng.integers(0, frames - 8 + 1))
            r0 = int(rng.integers(0, rows - 16 + 1)); c0 = int(rng.integers(0, cols - 16 + 1))
            revs.append(_rect_ids(layout, 0, f0, 8, r0, 16, c0, 16))
            drawn.append([(0, f0, 8, r0, 16, c0, 16)])
        elif wl.selection in ("rect_k32", "rect_k128"):
            nr, nc = (4, 8) if wl.selection == "rect_k32" else (8, 16)
            _, _, rows, cols, _ = layout[0]
            r0 = int(rng.integers(0, rows - nr + 1)); c0 = int(rng.integers(0, cols - nc + 1))
            revs.append(_rect_ids(layout, 0, 0, 1, r0, nr, c0, nc))
            drawn.append([(0, 0, 1, r0, nr, c0, nc)])
        elif wl.selection == "random":
            # extra = (min revisits, max revisits, min K, max K): distinct random tokens
            rmin, rmax, kmin, kmax = wl.extra
            for _ in range(int(rng.integers(rmin, rmax + 1))):
                k = min(int(rng.integers(kmin, kmax + 1)), wl.n_tokens)
                revs.append(rng.choice(wl.n_tokens, size=k, replace=False).astype(np.int32))
                drawn.append([])
        else:
            raise ValueError(wl.selection)
        out.append(revs)
        if rects_out is not None:
            rects_out.append(drawn)
    return out


def text_positions(wl: Workload, rng) -> np.ndarray:
    kind = wl.cur_pos[0]
    if kind == "fixed":
        p = np.full(wl.n_seqs, wl.cur_pos[1], dtype=np.int64)
    elif kind == "around":
        c, s = wl.cur_pos[1], wl.cur_pos[2]
        p = c + rng.integers(-s, s + 1, size=wl.n_seqs)
    elif kind == "uniform":
        p = rng.integers(wl.cur_pos[1], wl.cur_pos[2] + 1, size=wl.n_seqs)
    else:
        raise ValueError(kind)
    return p.astype(np.int64)


# ----------------------------------------------------------------------------
# raw visual store
# ----------------------------------------------------------------------------
def fill_store(wl: Workload, store_k: torch.Tensor, store_v: torch.Tensor, seed: int) -> None:
    """K, V ~ N(0, 1) (or N(0, 1) times a fixed per-(layer, head, channel)
    scale ~ U(0.5, 4) for "channel_scale", mimicking outlier channels), drawn
    on the store's device sequence by sequence, layer by layer."""
    dev = store_k.device
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    B, nL, M, H, D = store_k.shape
    scale = None
    if wl.kv_dist == "channel_scale":
        scale = torch.rand((2, nL, H, D), generator=g, device=dev, dtype=torch.float32) * 3.5 + 0.5
    for b in range(B):
        for l in range(nL):
            for which, dst in ((0, store_k), (1, store_v)):
                x = torch.randn((M, H, D), generator=g, device=dev, dtype=torch.float32)
                if scale is not None:
                    x.mul_(scale[which, l])
                dst[b, l].copy_(x.to(torch.bfloat16))


# ----------------------------------------------------------------------------
# whole batch
# ----------------------------------------------------------------------------
def make_batch(wl: Workload, device="cpu", seed: int = 0, store: bool = True,
               context: str = "canary") -> Batch:
    device = torch.device(device)
    rng_sel = np.random.Generator(np.random.PCG64(seed + 1))
    rng_pos = np.random.Generator(np.random.PCG64(seed + 2))

    sels = selections(wl, rng_sel)
    p_txt = text_positions(wl, rng_pos)
    cache_len_in = (p_txt + 1).astype(np.int32)  # the cache holds the context up to p_txt

    seq_rev_off = [0]
    rev_tok_off = [0]
    idx_list = []
    revisits = []
    for b, revs in enumerate(sels):
        for ids in revs:
            idx_list.append(ids)
            rev_tok_off.append(rev_tok_off[-1] + len(ids))
            revisits.append((b, ids))
        seq_rev_off.append(len(rev_tok_off) - 1)
    idx = np.concatenate(idx_list).astype(np.int32) if idx_list else np.zeros(0, np.int32)
    k_per_seq = np.array([sum(len(x) for x in revs) for revs in sels], dtype=np.int64)

    B, nL, M, H, D = wl.n_seqs, wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    coords = np.broadcast_to(token_coords(wl), (B, M, 3)).copy()

    shape = (B, nL, M, H, D)
    if store:
        store_k = torch.empty(shape, dtype=torch.bfloat16, device=device)
        store_v = torch.empty(shape, dtype=torch.bfloat16, device=device)
        fill_store(wl, store_k, store_v, seed)
    else:
        store_k = store_v = torch.empty((0,), dtype=torch.bfloat16, device=device)

    # context="canary": only the appended span is backed (paged) and every
    # cache row holds the canary; context="random": every slot up to the end of
    # the appended span is backed and the existing context rows hold N(0, 1)
    # values standing in for the model's already-rotated entries.
    full = context == "random"
    bs = wl.block_size
    if wl.cache == "contiguous":
        S = int(np.max(cache_len_in.astype(np.int64) + k_per_seq))
        S = (S + 16 + 15) // 16 * 16
        cshape = (B, nL, S, H, D)
        block_table = None
    else:
        first = cache_len_in.astype(np.int64) // bs
        last = (cache_len_in.astype(np.int64) + k_per_seq - 1) // bs
        if full:
            last = np.maximum(last, (cache_len_in.astype(np.int64) - 1) // bs)
            first = np.zeros_like(first)
            n_span = last - first + 1
        else:
            n_span = np.where(k_per_seq > 0, last - first + 1, 0)
        n_blocks = int(n_span.sum())
        max_blocks = int(np.max(np.where(k_per_seq > 0, last + 1, first + 1))) + 1
        perm = rng_pos.permutation(n_blocks).astype(np.int32)
        bt = np.full((B, max_blocks), -1, dtype=np.int32)
        k = 0
        for b in range(B):
            for j in range(int(n_span[b])):
                bt[b, first[b] + j] = perm[k]
                k += 1
        cshape = (nL, max(n_blocks, 1), bs, H, D)
        block_table = torch.from_numpy(bt).to(device)
    if full:
        g = torch.Generator(device=device)
        g.manual_seed(seed + 3)
        cache_k = torch.randn(cshape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
        cache_v = torch.randn(cshape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    else:
        cache_k = torch.full(cshape, CANARY_BITS, dtype=torch.int16, device=device).view(torch.bfloat16)
        cache_v = torch.full(cshape, CANARY_BITS, dtype=torch.int16, device=device).view(torch.bfloat16)

    t = lambda a, dt: torch.as_tensor(np.asarray(a), dtype=dt).to(device)
    return Batch(
        wl=wl, store_k=store_k, store_v=store_v,
        coords=t(coords, torch.int32),
        seq_rev_off=t(seq_rev_off, torch.int32), rev_tok_off=t(rev_tok_off, torch.int32),
        idx=t(idx, torch.int32), p_txt=t(p_txt, torch.int64),
        cache_len_in=t(cache_len_in, torch.int32),
        cache_k=cache_k, cache_v=cache_v, block_table=block_table, revisits=revisits)


def make_decode_inputs(n_seqs: int, n_layers: int, n_kv_heads: int, n_q_heads: int, head_dim: int,
                       max_len: int, paged: bool, device="cpu", seed: int = 0,
                       block_size: int = 16) -> dict:
    """A populated decoder cache (N(0, 1) bf16 rows in every slot each sequence
    attends), raw queries N(0, 1) bf16 [B, n_L, Hq, D], per-sequence lengths
    (the last sequence at max_len) and query positions at or after them."""
    device = torch.device(device)
    rng = np.random.Generator(np.random.PCG64(seed + 1))
    seq_len = rng.integers(1, max_len + 1, size=n_seqs)
    seq_len[-1] = max_len
    q_pos = seq_len + rng.integers(0, 20000, size=n_seqs)
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    H, D = n_kv_heads, head_dim
    if paged:
        nblk = [(int(n) + block_size - 1) // block_size for n in seq_len]
        total = sum(nblk)
        perm = rng.permutation(total + 3)[:total]  # a few pool blocks stay unused
        bt = np.full((n_seqs, max(nblk) + 2), -1, dtype=np.int32)
        k = 0
        for b in range(n_seqs):
            bt[b, :nblk[b]] = perm[k:k + nblk[b]]
            k += nblk[b]
        shape = (n_layers, total + 3, block_size, H, D)
        block_table = torch.from_numpy(bt).to(device)
    else:
        shape = (n_seqs, n_layers, max_len + 8, H, D)
        block_table = None
    cache_k = torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    cache_v = torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    q = torch.randn((n_seqs, n_layers, n_q_heads, D), generator=g, device=device,
                    dtype=torch.float32).to(torch.bfloat16)
    return dict(cache_k=cache_k, cache_v=cache_v, block_table=block_table, q=q,
                q_pos=torch.as_tensor(q_pos, dtype=torch.int64).to(device),
                seq_len=torch.as_tensor(seq_len, dtype=torch.int32).to(device),
                max_len=int(max_len), block_size=block_size)
