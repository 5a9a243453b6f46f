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


def _decode_case(i: int):
    rng = np.random.default_rng(2000 + i)
    D = int(rng.choice([64, 128, 256]))
    H = int(rng.choice([1, 2, 3, 4, 8]))
    g = int(rng.choice([1, 2, 3, 4, 7, 8]))
    while H * g * D > 8192:
        g = max(1, g // 2)
    B = int(rng.integers(1, 6))
    nL = int(rng.integers(1, 5))
    max_len = int(rng.choice([17, 64, 300, 933, 2500, 6000]))
    paged = bool(rng.integers(0, 2))
    bs = int(rng.choice([1, 7, 16, 32])) if paged else 16
    P = D // 2
    cut = np.sort(rng.integers(0, P + 1, size=2))
    sec = (int(cut[0]), int(cut[1] - cut[0]), int(P - cut[1]))
    return B, nL, H, H * g, D, max_len, paged, bs, sec


@pytest.mark.parametrize("i", range(12))
def test_fuzz_decode(i):
    """Random decode shapes (chunking, head split, merge kernels and the
    CUDA-core kernel all vary with them) against the oracle."""
    import torch
    import paper_2606_26631_gb300 as prcr
    from workloads import make_decode_inputs
    B, nL, H, Hq, D, max_len, paged, bs, sec = _decode_case(i)
    inp = make_decode_inputs(B, nL, H, Hq, D, max_len, paged, device=DEV, seed=60 + i, block_size=bs)
    cfg = prcr.rope_cfg(nL, H, D, sec, 1e6)
    cd = (prcr.cache_paged(inp["cache_k"], inp["cache_v"], inp["block_table"]) if paged
          else prcr.cache_contiguous(inp["cache_k"], inp["cache_v"]))
    out = torch.full(inp["q"].shape, float("nan"), dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(max(prcr.decode_workspace_size(cfg, B, Hq, max_len), 16), dtype=torch.uint8,
                     device=DEV)
    prcr.decode_attention(cfg, cd, inp["q"], inp["q_pos"], inp["seq_len"], max_len, out, status, ws)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got = out.cpu().numpy()
    qv = O.bf16_bits_to_f64(inp["q"].view(torch.int16).cpu().numpy())
    for b in range(B):
        n = int(inp["seq_len"][b])
        s = torch.arange(n, device=DEV)
        if paged:
            blk = inp["block_table"][b][s // bs].long()
            K = inp["cache_k"][:, blk, s % bs].transpose(0, 1)
            V = inp["cache_v"][:, blk, s % bs].transpose(0, 1)
        else:
            K = inp["cache_k"][b, :, :n].transpose(0, 1)
            V = inp["cache_v"][b, :, :n].transpose(0, 1)
        K = O.bf16_bits_to_f64(K.contiguous().view(torch.int16).cpu().numpy())
        V = O.bf16_bits_to_f64(V.contiguous().view(torch.int16).cpu().numpy())
        for l in range(nL):
            ref = O.decode_attention(qv[b, l], int(inp["q_pos"][b]), K[:, l], V[:, l], D, sec, 1e6)
            assert np.abs(got[b, l] - ref).max() / np.abs(V[:, l]).max() <= 1e-4, (b, l)


def _select_case(i: int):
    rng = np.random.default_rng(3000 + i)
    D = int(rng.choice([64, 128, 256]))
    H = int(rng.choice([1, 2, 3, 4, 8]))
    g = int(rng.choice([1, 2, 3, 4, 7, 8]))
    while H * g * D > 8192:
        g = max(1, g // 2)
    B = int(rng.integers(1, 6))
    M = int(rng.choice([1, 15, 16, 17, 100, 767, 1024, 1025, 4099, 9000]))
    k = int(rng.integers(1, M + 1))
    P = D // 2
    cut = np.sort(rng.integers(0, P + 1, size=2))
    sec = (int(cut[0]), int(cut[1] - cut[0]), int(P - cut[1]))
    return B, H, H * g, D, M, k, sec, bool(i % 2)


@pytest.mark.parametrize("i", range(12))
def test_fuzz_select(i):
    """Random selection shapes from the raw store (even cases) and from the
    cache (odd cases): relevance against the oracle, the set the exact top-k
    of the reported relevance and a valid top-k of the oracle's."""
    import torch
    import paper_2606_26631_gb300 as prcr
    B, H, Hq, D, M, k, sec, cached = _select_case(i)
    g = torch.Generator(device=DEV).manual_seed(70 + i)
    sk = torch.randn((B, 1, M, H, D), device=DEV, generator=g).to(torch.bfloat16)
    coords = torch.randint(0, 64, (B, M, 3), device=DEV, generator=g, dtype=torch.int32)
    q = (2.0 * torch.randn((B, Hq, D), device=DEV, generator=g)).to(torch.bfloat16)
    q_pos = torch.randint(100, 20000, (B,), device=DEV, generator=g, dtype=torch.int64)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    idx = torch.full((B * k,), -7, dtype=torch.int32, device=DEV)
    sro = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    rto = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    score = torch.full((B, M), -1.0, dtype=torch.float32, device=DEV)
    ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=DEV)
    if cached:
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        img0 = torch.zeros(B, dtype=torch.int32, device=DEV)
        prcr.select_topk_cached(cfg, prcr.cache_contiguous(sk, sk), 0, q, q_pos, img0, M, k, idx, sro,
                                rto, status, ws, score)
    else:
        prcr.select_topk(cfg, prcr.store_desc(sk, sk, coords), 0, q, q_pos, k, idx, sro, rto, ws, score)
    torch.cuda.synchronize()
    if cached:
        assert int(status.item()) == 0
    idx = idx.view(B, k).cpu().numpy()
    score = score.cpu().numpy()
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    kb = sk.view(torch.int16).cpu().numpy()
    crd = coords.cpu().numpy()
    for b in range(B):
        if cached:
            ref = O.ads_relevance_cached(qv[b], int(q_pos[b]), O.bf16_bits_to_f64(kb[b, 0]), D, sec, 1e6)
        else:
            ref = O.ads_relevance(qv[b], int(q_pos[b]), kb[b, 0], crd[b], D, sec, 1e6)
        assert (np.abs(score[b] - ref) / ref).max() <= 1e-4
        sel = idx[b]
        order = np.lexsort((np.arange(M), -score[b].astype(np.float64)))
        assert np.array_equal(sel, np.sort(order[:k]))
        if k < M:
            tol = 2 * np.abs(score[b] - ref).max() + 1e-12
            chosen = np.zeros(M, dtype=bool)
            chosen[sel] = True
            assert ref[chosen].min() >= ref[~chosen].max() - tol
