"""Workload shapes for the revisit path, modelled on the paper's MLLM setups.

The paper evaluates Qwen3-VL / InternVL3.5 models on image reasoning benchmarks
(Sec. 4.1); neither the benchmarks nor the weights are used here. Each workload
below fixes the decoder geometry (layers, KV heads, head dim, M-RoPE sections),
the visual grids that fill the raw visual store (Eq. 4, "global_raw_memory"),
how the revisited index sets are drawn (Sec. 2.1, Eq. 3) and the cache kind
(Eq. "active_cache"). The arrays themselves are made by ``workloads.gen``.

Nothing in this module computes any part of the method.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Tuple


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_kv_heads: int
    head_dim: int
    sections: Tuple[int, int, int]       # rotation pairs given to the t, h, w axes
    n_seqs: int
    grids: Tuple[Tuple[int, int, int], ...]  # per image/video of one sequence: (frames, rows, cols)
    selection: str                      # name of the index-set recipe (see gen.py)
    cache: str                          # "contiguous" or "paged"
    cur_pos: Tuple                      # ("fixed", p) | ("around", p, spread) | ("uniform", lo, hi)
    theta: float = 1.0e6
    block_size: int = 16
    kv_dist: str = "normal"             # "normal" or "channel_scale"
    L: int = 2                          # left extension; the paper's default (Sec. 4.4)
    extra: Tuple = field(default=())

    @property
    def n_tokens(self) -> int:
        """M: visual tokens per sequence."""
        return sum(f * r * c for f, r, c in self.grids)

    @property
    def row_elems(self) -> int:
        return self.n_kv_heads * self.head_dim


TINY = Workload(
    name="tiny", n_layers=2, n_kv_heads=2, head_dim=64, sections=(8, 12, 12),
    n_seqs=1, grids=((1, 8, 8),), selection="rect4x4", cache="contiguous",
    cur_pos=("fixed", 200))

QWEN2VL_2B = Workload(
    name="qwen2vl-2b", n_layers=28, n_kv_heads=2, head_dim=128, sections=(16, 24, 24),
    n_seqs=1, grids=((1, 32, 32),), selection="rects3_256", cache="contiguous",
    cur_pos=("around", 1500, 64))

QWEN25VL_7B = Workload(
    name="qwen25vl-7b", n_layers=28, n_kv_heads=4, head_dim=128, sections=(16, 24, 24),
    n_seqs=8, grids=((1, 46, 46),), selection="rectset512", cache="paged",
    cur_pos=("uniform", 1000, 4000), kv_dist="channel_scale")

QWEN3VL_8B = Workload(
    name="qwen3vl-8b", n_layers=36, n_kv_heads=8, head_dim=128, sections=(24, 20, 20),
    n_seqs=16, grids=((1, 64, 64), (1, 64, 64)), selection="rev4_256_1024", cache="paged",
    cur_pos=("uniform", 1000, 4000))

STRESS = Workload(
    name="stress", n_layers=36, n_kv_heads=8, head_dim=128, sections=(24, 20, 20),
    n_seqs=32, grids=((16, 32, 32),), selection="video_stress", cache="paged",
    cur_pos=("uniform", 8000, 30000))

# Table 3 shape: Qwen3-VL-8B dimensions, a 768-token image, K in {32, 128}.
PAPER_8B_K32 = Workload(
    name="paper-8b-k32", n_layers=36, n_kv_heads=8, head_dim=128, sections=(24, 20, 20),
    n_seqs=1, grids=((1, 24, 32),), selection="rect_k32", cache="contiguous",
    cur_pos=("fixed", 900))

PAPER_8B_K128 = Workload(
    name="paper-8b-k128", n_layers=36, n_kv_heads=8, head_dim=128, sections=(24, 20, 20),
    n_seqs=1, grids=((1, 24, 32),), selection="rect_k128", cache="contiguous",
    cur_pos=("fixed", 900))

ALL = {w.name: w for w in (TINY, QWEN2VL_2B, QWEN25VL_7B, QWEN3VL_8B, STRESS,
                           PAPER_8B_K32, PAPER_8B_K128)}


def get(name: str) -> Workload:
    return ALL[name]
