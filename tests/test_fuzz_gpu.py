"""Seeded random shapes through prcr_rebind_inject, each compared completely
with the oracle (every position, slot, length, K/V row and untouched cache
row), as the fixed-workload parity tests do.

Each case draws its own decoder shape (layers, KV heads, head_dim 16..256,
rotary sections, theta), sequences with one or two images or videos,
revisits of random token sets (empty revisits and sequences included),
contiguous or paged caches with block sizes 1..32, the position rule (PCR,
ORIGINAL, UIR, LPA), L, the degenerate-axis reading and the band layout.
Most cases are small enough for the one-kernel path; the last ones select
more than 2048 tokens and take the plan + rebind kernels.
"""
import numpy as np
import pytest

from oracle import prcr_oracle as O
from workloads import Workload, make_batch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
N_SMALL, N_LARGE = 20, 4


def _case(i: int):
    rng = np.random.default_rng(1000 + i)
    large = i >= N_SMALL
    D = int(rng.choice([16, 32, 48, 64, 128] + ([256] if not large else [])))
    P = D // 2
    cut = np.sort(rng.integers(0, P + 1, size=2))
    sections = (int(cut[0]), int(cut[1] - cut[0]), int(P - cut[1]))
    H = int(rng.choice([1, 2, 3, 4, 8]))
    while H * D > 8192:
        H //= 2
    n_layers = int(rng.integers(1, 7))
    n_seqs = int(rng.integers(1, 7)) if not large else int(rng.integers(2, 5))
    if large:
        grids = ((int(rng.integers(2, 5)), 24, 32),)
    else:
        grids = tuple((int(rng.integers(1, 4)), int(rng.integers(2, 10)), int(rng.integers(2, 10)))
                      for _ in range(int(rng.integers(1, 3))))
    M = sum(f * r * c for f, r, c in grids)
    kmax = min(M, 1200) if large else M
    extra = (2, 3, 800, kmax) if large else (int(rng.integers(0, 2)), int(rng.integers(1, 4)), 0, kmax)
    paged = bool(rng.integers(0, 2))
    block_size = int(rng.choice([1, 3, 7, 16, 32])) if paged else 16
    wl = Workload(name=f"fuzz{i}", n_layers=n_layers, n_kv_heads=H, head_dim=D, sections=sections,
                  n_seqs=n_seqs, grids=grids, selection="random",
                  cache="paged" if paged else "contiguous",
                  cur_pos=("uniform", M + 10, M + 50000), block_size=block_size, extra=extra,
                  theta=float(rng.choice([1e4, 5e5, 1e6])))
    mode = int(rng.choice([O.MODE_PCR, O.MODE_PCR, O.MODE_ORIGINAL, O.MODE_UIR, O.MODE_LPA]))
    L = int(rng.choice([0, 1, 2, 5]))
    center = bool(rng.integers(0, 2))
    layout = int(rng.choice([O.LAYOUT_SECTIONED, O.LAYOUT_INTERLEAVED]))
    return wl, mode, L, center, layout


@pytest.mark.parametrize("i", range(N_SMALL + N_LARGE))
def test_fuzz_rebind_inject(i):
    import parity_util as pu
    wl, mode, L, center, layout = _case(i)
    batch = make_batch(wl, device=DEV, seed=50 + i)
    if i >= N_SMALL:
        assert batch.total_k > 2048  # the two-kernel path
    rv = pu.make_revisit(batch, mode=mode, L=L, flags=1 if center else 0, layout=layout)
    rv.run()
    import torch
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    pu.full_check(batch, rv, mode=mode, L=L, degenerate="center" if center else "zero",
                  layout=layout)
