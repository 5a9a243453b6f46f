"""GPU checks of prcr_select_topk (attention-driven selection, Sec. 2.1 /
Eq. 3, under the reading in the oracle's header).

Relevance: float32 on the GPU against the oracle's float64 ads_relevance,
relative error <= 1e-4. Selection: where floating point decides an integer,
the check is that (a) the set is exactly the top-k of the relevance the
kernel itself reports (ties to the lower index), (b) it is a valid top-k of
the oracle's relevance up to the measured relevance error, and (c) it equals
the oracle's ads_select whenever the oracle's k-th and (k+1)-th values are
further apart than that error. Ties are forced with an all-zero key layer.
"""
import numpy as np
import pytest
import torch

from oracle import prcr_oracle as O
from workloads import Workload, get, make_batch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _select(batch, layer, Hq, k, q, q_pos):
    import paper_2606_26631_gb300 as prcr
    wl = batch.wl
    B, M = wl.n_seqs, wl.n_tokens
    cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta)
    sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
    idx = torch.full((B * k,), -7, dtype=torch.int32, device=DEV)
    sro = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    rto = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    score = torch.full((B, M), -1.0, dtype=torch.float32, device=DEV)
    ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=DEV)
    prcr.select_topk(cfg, sd, layer, q, q_pos, k, idx, sro, rto, ws, score)
    torch.cuda.synchronize()
    return idx.view(B, k).cpu().numpy(), sro.cpu().numpy(), rto.cpu().numpy(), score.cpu().numpy()


def _topk_by(values, k):
    order = np.lexsort((np.arange(len(values)), -values))
    return np.sort(order[:k])


# odd shapes: head_dim 48 (3 of 4 lanes per row active), 3 KV heads with a
# GQA group of 3, two grids per sequence; head_dim 256 with a group of 2;
# token counts that leave a ragged last tile
SHAPES = {
    "sel-odd": Workload(name="sel-odd", n_layers=2, n_kv_heads=3, head_dim=48, sections=(8, 8, 8),
                        n_seqs=3, grids=((3, 5, 5), (1, 4, 4)), selection="random",
                        cache="contiguous", cur_pos=("uniform", 100, 4000), extra=(0, 3, 0, 37)),
    "sel-d256": Workload(name="sel-d256", n_layers=1, n_kv_heads=2, head_dim=256,
                         sections=(40, 44, 44), n_seqs=2, grids=((2, 10, 13),), selection="random",
                         cache="contiguous", cur_pos=("uniform", 500, 900), extra=(1, 2, 1, 40)),
    # 1500 tokens over 24 tiles of 64 (ragged last tile), 16 query heads
    "sel-1500": Workload(name="sel-1500", n_layers=1, n_kv_heads=4, head_dim=128,
                         sections=(16, 24, 24), n_seqs=2, grids=((1, 30, 50),), selection="random",
                         cache="contiguous", cur_pos=("uniform", 2000, 9000), extra=(1, 1, 1, 40)),
}


@pytest.mark.parametrize("name,Hq,k,layer", [("qwen25vl-7b", 28, 64, 5), ("qwen3vl-8b", 32, 300, 35),
                                             ("tiny", 2, 16, 1), ("qwen2vl-2b", 4, 100, 20),
                                             ("sel-odd", 9, 20, 1), ("sel-d256", 4, 30, 0),
                                             ("sel-1500", 16, 200, 0)])
def test_select_parity(name, Hq, k, layer):
    wl = SHAPES.get(name) or get(name)
    batch = make_batch(wl, device=DEV)
    B, M, D = wl.n_seqs, wl.n_tokens, wl.head_dim
    g = torch.Generator(device=DEV)
    g.manual_seed(17)
    q = (3.0 * torch.randn((B, Hq, D), generator=g, device=DEV)).to(torch.bfloat16)
    idx, sro, rto, score = _select(batch, layer, Hq, k, q, batch.p_txt)
    assert np.array_equal(sro, np.arange(B + 1))
    assert np.array_equal(rto, k * np.arange(B + 1))
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    coords = batch.coords.cpu().numpy()
    for b in range(min(B, 4)):
        k_raw = batch.store_k[b, layer].view(torch.int16).cpu().numpy()
        ref = O.ads_relevance(qv[b], int(batch.p_txt[b]), k_raw, coords[b], D, wl.sections, wl.theta)
        rel_err = np.abs(score[b] - ref) / ref
        assert rel_err.max() <= 1e-4, rel_err.max()
        sel = idx[b]
        assert len(set(sel.tolist())) == k and np.all(np.diff(sel) > 0)
        assert np.array_equal(sel, _topk_by(score[b].astype(np.float64), k))  # (a)
        tol = 2 * np.abs(score[b] - ref).max() + 1e-12
        chosen = np.zeros(M, dtype=bool)
        chosen[sel] = True
        if k < M:
            assert ref[chosen].min() >= ref[~chosen].max() - tol  # (b)
            srt = np.sort(ref)[::-1]
            if srt[k - 1] - srt[k] > tol:
                assert np.array_equal(sel, O.ads_select(ref, k))  # (c)


def test_select_ties_and_full_set():
    wl = get("qwen2vl-2b")
    batch = make_batch(wl, device=DEV)
    batch.store_k[:, 3].zero_()  # every logit of layer 3 is 0: all relevances tie
    B, M, D = 1, wl.n_tokens, wl.head_dim
    q = torch.randn((B, 2, D), device=DEV).to(torch.bfloat16)
    idx, _, _, score = _select(batch, 3, 2, 100, q, batch.p_txt)
    assert np.array_equal(idx[0], np.arange(100))
    assert np.allclose(score[0], 1.0 / M, rtol=1e-6)
    idx, _, _, _ = _select(batch, 7, 2, M, q, batch.p_txt)
    assert np.array_equal(idx[0], np.arange(M))


def test_select_feeds_rebind_inject():
    """The selection's outputs are a valid revisit batch for prcr_rebind_inject."""
    import paper_2606_26631_gb300 as prcr
    wl = get("qwen25vl-7b")
    batch = make_batch(wl, device=DEV)
    B, k = wl.n_seqs, 48
    q = torch.randn((B, 4, wl.head_dim), device=DEV).to(torch.bfloat16)
    cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta)
    sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
    idx = torch.empty(B * k, dtype=torch.int32, device=DEV)
    sro = torch.empty(B + 1, dtype=torch.int32, device=DEV)
    rto = torch.empty(B + 1, dtype=torch.int32, device=DEV)
    ws = torch.empty(prcr.select_workspace_size(B, 4, wl.n_tokens), dtype=torch.uint8, device=DEV)
    prcr.select_topk(cfg, sd, 0, q, batch.p_txt, k, idx, sro, rto, ws)
    # a cache with room for k slots after each sequence's context
    clen = batch.cache_len_in
    nblk = int(((clen.max() + k) // 16 + 2).item())
    bt = torch.arange(B * nblk, dtype=torch.int32, device=DEV).view(B, nblk).contiguous()
    ck = torch.full((wl.n_layers, B * nblk, 16, wl.n_kv_heads, wl.head_dim), -1,
                    dtype=torch.int16, device=DEV).view(torch.bfloat16)
    cv = ck.clone()
    rv = prcr.Revisit(cfg, batch.store_k, batch.store_v, batch.coords, ck, cv, bt, sro, rto, idx,
                      batch.p_txt, clen)
    rv.run()
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    assert torch.equal(rv.cache_len_out, clen + k)
    assert torch.equal(rv.next_pos, batch.p_txt + 1)
    written = int((ck.view(torch.int16) != -1).sum().item())
    assert written == B * k * wl.n_layers * wl.n_kv_heads * wl.head_dim


@pytest.mark.slow
def test_select_full_size_sampled():
    """The selection configuration bench.py times on the stress shape (32
    sequences x 16,384 tokens, 32 query heads, k = 4096, last layer); sampled
    sequences checked like test_select_parity."""
    wl = get("stress")
    batch = make_batch(wl, device=DEV)
    B, M, H, D = wl.n_seqs, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    Hq, k, layer = 4 * H, batch.total_k // B, wl.n_layers - 1
    q = torch.randn((B, Hq, D), device=DEV, generator=torch.Generator(device=DEV).manual_seed(3)
                    ).to(torch.bfloat16)
    idx, sro, rto, score = _select(batch, layer, Hq, k, q, batch.p_txt)
    assert np.array_equal(sro, np.arange(B + 1))
    assert np.array_equal(rto, k * np.arange(B + 1))
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    coords = batch.coords.cpu().numpy()
    for b in (0, B // 2, B - 1):
        k_raw = batch.store_k[b, layer].view(torch.int16).cpu().numpy()
        ref = O.ads_relevance(qv[b], int(batch.p_txt[b]), k_raw, coords[b], D, wl.sections, wl.theta)
        assert (np.abs(score[b] - ref) / ref).max() <= 1e-4
        sel = idx[b]
        assert np.array_equal(sel, _topk_by(score[b].astype(np.float64), k))
        tol = 2 * np.abs(score[b] - ref).max() + 1e-12
        chosen = np.zeros(M, dtype=bool)
        chosen[sel] = True
        assert ref[chosen].min() >= ref[~chosen].max() - tol
    del batch
    torch.cuda.empty_cache()


def test_select_interleaved_layout():
    """The interleaved M-RoPE band layout (pair i to h when i % 3 == 1, to w
    when i % 3 == 2, within their sections) on both logits kernels: head_dim
    128 (tensor cores) and 48 (CUDA cores)."""
    import paper_2606_26631_gb300 as prcr
    for wl, Hq, k, layer in ((get("qwen2vl-2b"), 8, 100, 9), (SHAPES["sel-odd"], 9, 20, 1)):
        batch = make_batch(wl, device=DEV)
        B, M, D = wl.n_seqs, wl.n_tokens, wl.head_dim
        cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, D, wl.sections, wl.theta,
                            O.LAYOUT_INTERLEAVED)
        sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
        q = (3.0 * torch.randn((B, Hq, D), device=DEV,
                               generator=torch.Generator(device=DEV).manual_seed(8))).to(torch.bfloat16)
        idx = torch.empty(B * k, dtype=torch.int32, device=DEV)
        sro = torch.empty(B + 1, dtype=torch.int32, device=DEV)
        rto = torch.empty(B + 1, dtype=torch.int32, device=DEV)
        score = torch.empty((B, M), dtype=torch.float32, device=DEV)
        ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=DEV)
        prcr.select_topk(cfg, sd, layer, q, batch.p_txt, k, idx, sro, rto, ws, score)
        torch.cuda.synchronize()
        qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
        coords = batch.coords.cpu().numpy()
        sc = score.cpu().numpy()
        sel = idx.view(B, k).cpu().numpy()
        for b in range(B):
            k_raw = batch.store_k[b, layer].view(torch.int16).cpu().numpy()
            ref = O.ads_relevance(qv[b], int(batch.p_txt[b]), k_raw, coords[b], D, wl.sections,
                                  wl.theta, O.LAYOUT_INTERLEAVED)
            assert (np.abs(sc[b] - ref) / ref).max() <= 1e-4, wl.name
            assert np.array_equal(sel[b], _topk_by(sc[b].astype(np.float64), k))


# Coordinate structures beyond one image per sequence: two images of widths
# 4 and 16 in one sequence, a 24-wide video with a t section that ends inside
# an 8-pair group, head_dim 64 with a GQA group of 8, and a sequence whose
# coordinates are shuffled (no token shares a row or column with its index
# neighbours). The relevance must not depend on any grid regularity.
GRID_SHAPES = {
    "rot-w4-w16": (Workload(name="rot-w4-w16", n_layers=1, n_kv_heads=2, head_dim=128,
                            sections=(24, 20, 20), n_seqs=2, grids=((2, 6, 4), (1, 9, 16)),
                            selection="random", cache="contiguous", cur_pos=("uniform", 300, 5000),
                            extra=(1, 1, 1, 20)), 8, False),
    "rot-t20": (Workload(name="rot-t20", n_layers=1, n_kv_heads=4, head_dim=128,
                         sections=(20, 20, 24), n_seqs=2, grids=((3, 11, 24),), selection="random",
                         cache="contiguous", cur_pos=("uniform", 300, 5000), extra=(1, 1, 1, 20)),
                16, False),
    "rot-d64-g8": (Workload(name="rot-d64-g8", n_layers=1, n_kv_heads=2, head_dim=64,
                            sections=(8, 12, 12), n_seqs=2, grids=((1, 20, 24),), selection="random",
                            cache="contiguous", cur_pos=("uniform", 300, 5000), extra=(1, 1, 1, 20)),
                   16, False),
    "rot-shuffled": (get("qwen2vl-2b"), 8, True),
}


@pytest.mark.parametrize("name", sorted(GRID_SHAPES))
def test_select_coordinate_structures(name):
    wl, Hq, shuffle = GRID_SHAPES[name]
    batch = make_batch(wl, device=DEV)
    B, M, D = wl.n_seqs, wl.n_tokens, wl.head_dim
    if shuffle:
        perm = torch.randperm(M, generator=torch.Generator().manual_seed(5)).to(DEV)
        batch.coords[0] = batch.coords[0][perm].clone()
    k = min(40, M - 1)
    g = torch.Generator(device=DEV)
    g.manual_seed(29)
    q = (3.0 * torch.randn((B, Hq, D), generator=g, device=DEV)).to(torch.bfloat16)
    idx, sro, rto, score = _select(batch, 0, Hq, k, q, batch.p_txt)
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    coords = batch.coords.cpu().numpy()
    for b in range(B):
        k_raw = batch.store_k[b, 0].view(torch.int16).cpu().numpy()
        ref = O.ads_relevance(qv[b], int(batch.p_txt[b]), k_raw, coords[b], D, wl.sections, wl.theta)
        rel_err = np.abs(score[b] - ref) / ref
        assert rel_err.max() <= 1e-4, (b, rel_err.max())
        assert np.array_equal(idx[b], _topk_by(score[b].astype(np.float64), k))


# Shapes whose logits work divides unevenly over the persistent grid of a
# 152-SM GB300 (two CTAs per SM): the last items are split in halves by KV
# heads, here over groups of 3 KV heads (halves of 2 and 1) and 5 (3 and 2,
# then 2 and 1 for the group of 2). The split items are the last ones, i.e.
# the last sequences', which the test checks against the oracle.
HALVES = {
    "halves-h6": (Workload(name="halves-h6", n_layers=1, n_kv_heads=6, head_dim=128,
                           sections=(16, 24, 24), n_seqs=24, grids=((1, 40, 40),), selection="random",
                           cache="contiguous", cur_pos=("uniform", 2000, 9000), extra=(1, 1, 1, 40)), 12),
    "halves-h5-d64": (Workload(name="halves-h5-d64", n_layers=1, n_kv_heads=5, head_dim=64,
                               sections=(8, 12, 12), n_seqs=20, grids=((1, 40, 50),), selection="random",
                               cache="contiguous", cur_pos=("uniform", 2000, 9000), extra=(1, 1, 1, 40)), 15),
}


@pytest.mark.parametrize("name", sorted(HALVES))
def test_select_leftover_halves(name):
    wl, Hq = HALVES[name]
    batch = make_batch(wl, device=DEV)
    B, M, D = wl.n_seqs, wl.n_tokens, wl.head_dim
    k = 100
    g = torch.Generator(device=DEV)
    g.manual_seed(29)
    q = (3.0 * torch.randn((B, Hq, D), generator=g, device=DEV)).to(torch.bfloat16)
    idx, _, _, score = _select(batch, 0, Hq, k, q, batch.p_txt)
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    coords = batch.coords.cpu().numpy()
    for b in (0, B - 3, B - 2, B - 1):
        k_raw = batch.store_k[b, 0].view(torch.int16).cpu().numpy()
        ref = O.ads_relevance(qv[b], int(batch.p_txt[b]), k_raw, coords[b], D, wl.sections, wl.theta)
        assert (np.abs(score[b] - ref) / ref).max() <= 1e-4, b
        assert np.array_equal(idx[b], _topk_by(score[b].astype(np.float64), k))
