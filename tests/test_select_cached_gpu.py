"""GPU checks of prcr_select_topk_cached: the attention-driven selection read
from the decoder's position-bound cache (Sec. 2.1 / Eq. 3, second reading in
the oracle's header), against the oracle's float64 ads_relevance_cached on
the same bf16 cache rows.

Caches are filled with random bf16 rows directly (contiguous, and paged with
shuffled blocks of 16 or 7 slots; head_dim 64, 128 and 256), so nothing but
this call is under test.
Relevance: relative error <= 1e-4. Selection: as for the raw-store call,
(a) the set is exactly the top-k of the relevance the kernel reports (ties to
the lower index), (b) it is a valid top-k of the oracle's relevance up to
the measured relevance error, (c) it equals the oracle's ads_select whenever
the k-th and (k+1)-th oracle values are further apart than that error.
"""
import numpy as np
import pytest
import torch

from oracle import prcr_oracle as O

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _topk_by(values, k):
    order = np.lexsort((np.arange(len(values)), -values))
    return np.sort(order[:k])


def _make_cache(B, nL, H, D, M, paged, block_size, seed):
    """A cache of random bf16 rows and each sequence's first image slot; the
    image rows of sequence b are slots img_slot0[b] .. img_slot0[b] + M - 1."""
    g = torch.Generator(device=DEV).manual_seed(seed)
    img0 = [3 + 5 * b for b in range(B)]
    S = max(img0) + M + 9
    if not paged:
        k = torch.randn((B, nL, S, H, D), device=DEV, generator=g).to(torch.bfloat16)
        return k, None, torch.tensor(img0, dtype=torch.int32, device=DEV)
    nblk = (S + block_size - 1) // block_size
    NB = B * nblk + 2
    k = torch.randn((nL, NB, block_size, H, D), device=DEV, generator=g).to(torch.bfloat16)
    perm = torch.randperm(NB, device=DEV, generator=g)[: B * nblk].to(torch.int32)
    bt = perm.view(B, nblk).contiguous()
    return k, bt, torch.tensor(img0, dtype=torch.int32, device=DEV)


def _image_rows(cache_k, bt, img0, b, layer, M):
    """[M, H, D] float64 values of sequence b's image rows at `layer`."""
    s = torch.arange(M, device=DEV) + int(img0[b])
    if bt is None:
        rows = cache_k[b, layer, s]
    else:
        bs = cache_k.shape[2]
        rows = cache_k[layer, bt[b][s // bs].long(), s % bs]
    return O.bf16_bits_to_f64(rows.contiguous().view(torch.int16).cpu().numpy())


def _run(cfg, cache_desc, layer, q, q_pos, img0, M, k):
    import paper_2606_26631_gb300 as prcr
    B = q.shape[0]
    idx = torch.full((B * k,), -7, dtype=torch.int32, device=DEV)
    sro = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    rto = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    score = torch.full((B, M), -1.0, dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(prcr.select_workspace_size(B, q.shape[1], M), dtype=torch.uint8, device=DEV)
    prcr.select_topk_cached(cfg, cache_desc, layer, q, q_pos, img0, M, k, idx, sro, rto, status, ws,
                            score)
    torch.cuda.synchronize()
    return (idx.view(B, k).cpu().numpy(), sro.cpu().numpy(), rto.cpu().numpy(),
            score.cpu().numpy(), int(status.item()))


def _check_seq(score_b, ref, sel, k, M):
    rel_err = np.abs(score_b - ref) / ref
    assert rel_err.max() <= 1e-4, rel_err.max()
    assert len(set(sel.tolist())) == k and np.all(np.diff(sel) > 0)
    assert np.array_equal(sel, _topk_by(score_b.astype(np.float64), k))  # (a)
    tol = 2 * np.abs(score_b - ref).max() + 1e-12
    chosen = np.zeros(M, dtype=bool)
    chosen[sel] = True
    if k < M:
        assert ref[chosen].min() >= ref[~chosen].max() - tol  # (b)
        srt = np.sort(ref)[::-1]
        if srt[k - 1] - srt[k] > tol:
            assert np.array_equal(sel, O.ads_select(ref, k))  # (c)


CASES = [  # (B, n_layers, layer, H, Hq, D, M, k, paged, block_size, sections, theta)
    (2, 4, 3, 8, 32, 128, 768, 32, False, 0, (24, 20, 20), 1e6),
    (3, 2, 1, 4, 16, 128, 2116, 300, True, 16, (16, 24, 24), 1e6),
    (3, 1, 0, 2, 14, 64, 91, 20, True, 7, (8, 12, 12), 5e5),
    (1, 2, 0, 3, 9, 64, 1500, 200, False, 0, (8, 12, 12), 1e6),
    (2, 1, 0, 4, 16, 256, 700, 64, True, 16, (40, 44, 44), 1e6),
]


@pytest.mark.parametrize("case", CASES, ids=[
    f"B{c[0]}H{c[3]}Hq{c[4]}D{c[5]}M{c[6]}k{c[7]}{'p' + str(c[9]) if c[8] else 'c'}" for c in CASES])
def test_select_cached_parity(case):
    import paper_2606_26631_gb300 as prcr
    B, nL, layer, H, Hq, D, M, k, paged, bs, sec, theta = case
    cache_k, bt, img0 = _make_cache(B, nL, H, D, M, paged, bs, seed=31 + M)
    cache_v = torch.zeros_like(cache_k)
    cd = prcr.cache_paged(cache_k, cache_v, bt) if paged else prcr.cache_contiguous(cache_k, cache_v)
    cfg = prcr.rope_cfg(nL, H, D, sec, theta)
    g = torch.Generator(device=DEV).manual_seed(5 + B)
    q = (3.0 * torch.randn((B, Hq, D), device=DEV, generator=g)).to(torch.bfloat16)
    q_pos = torch.tensor([900 + 4111 * b for b in range(B)], dtype=torch.int64, device=DEV)
    idx, sro, rto, score, st = _run(cfg, cd, layer, q, q_pos, img0, M, k)
    assert st == 0
    assert np.array_equal(sro, np.arange(B + 1)) and np.array_equal(rto, k * np.arange(B + 1))
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    for b in range(B):
        kc = _image_rows(cache_k, bt, img0.cpu().numpy(), b, layer, M)
        ref = O.ads_relevance_cached(qv[b], int(q_pos[b]), kc, D, sec, theta)
        _check_seq(score[b], ref, idx[b], k, M)


def test_select_cached_missing_rows():
    """Image slots past the capacity (contiguous) and in an unmapped block
    (paged) set their status bit and get relevance 0; the others keep the
    oracle's relevance over the readable tokens."""
    import paper_2606_26631_gb300 as prcr
    D, H, Hq, M, k, sec = 64, 2, 8, 40, 5, (8, 12, 12)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    g = torch.Generator(device=DEV).manual_seed(8)
    q = torch.randn((1, Hq, D), device=DEV, generator=g).to(torch.bfloat16)
    q_pos = torch.tensor([300], dtype=torch.int64, device=DEV)
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    # contiguous: 50 slots, the image starts at slot 20, so tokens 30..39 are beyond the capacity
    ck = torch.randn((1, 1, 50, H, D), device=DEV, generator=g).to(torch.bfloat16)
    img0 = torch.tensor([20], dtype=torch.int32, device=DEV)
    cd = prcr.cache_contiguous(ck, torch.zeros_like(ck))
    idx, _, _, score, st = _run(cfg, cd, 0, q, q_pos, img0, M, k)
    assert st & prcr.ST_CAPACITY
    assert np.all(score[0, 30:] == 0.0)
    kc = O.bf16_bits_to_f64(ck[0, 0, 20:50].contiguous().view(torch.int16).cpu().numpy())
    ref = O.ads_relevance_cached(qv[0], 300, kc, D, sec, 1e6)
    assert (np.abs(score[0, :30] - ref) / ref).max() <= 1e-4
    assert np.all(idx[0] < 30)
    # paged, blocks of 8: the block of slots 16..23 is unmapped
    pk = torch.randn((1, 8, 8, H, D), device=DEV, generator=g).to(torch.bfloat16)
    bt = torch.tensor([[3, 1, -1, 0, 6, 2, 7]], dtype=torch.int32, device=DEV)
    img0 = torch.tensor([4], dtype=torch.int32, device=DEV)
    cd = prcr.cache_paged(pk, torch.zeros_like(pk), bt)
    idx, _, _, score, st = _run(cfg, cd, 0, q, q_pos, img0, M, k)
    assert st & prcr.ST_NO_BLOCK
    missing = np.arange(M)[(np.arange(M) + 4) // 8 == 2]
    assert np.all(score[0, missing] == 0.0)
    keep = np.setdiff1d(np.arange(M), missing)
    slots = keep + 4
    rows = pk[0, bt[0][torch.as_tensor(slots // 8, device=DEV)].long(),
              torch.as_tensor(slots % 8, device=DEV)]
    kc = O.bf16_bits_to_f64(rows.contiguous().view(torch.int16).cpu().numpy())
    ref = O.ads_relevance_cached(qv[0], 300, kc, D, sec, 1e6)
    assert (np.abs(score[0, keep] - ref) / ref).max() <= 1e-4
    assert not set(idx[0].tolist()) & set(missing.tolist())


def test_select_cached_full_size_sampled():
    """Stress-shaped batch (32 sequences x 16,384 visual tokens, 8 KV heads,
    32 query heads, head_dim 128, paged): every sequence's selection is
    well formed; sampled sequences match the oracle."""
    import paper_2606_26631_gb300 as prcr
    B, H, Hq, D, M, k, sec = 32, 8, 32, 128, 16384, 4096, (24, 20, 20)
    cache_k, bt, img0 = _make_cache(B, 1, H, D, M, True, 16, seed=77)
    cd = prcr.cache_paged(cache_k, torch.zeros_like(cache_k), bt)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    g = torch.Generator(device=DEV).manual_seed(6)
    q = (2.0 * torch.randn((B, Hq, D), device=DEV, generator=g)).to(torch.bfloat16)
    q_pos = torch.randint(8000, 30000, (B,), device=DEV, generator=g, dtype=torch.int64)
    idx, sro, rto, score, st = _run(cfg, cd, 0, q, q_pos, img0, M, k)
    assert st == 0
    assert np.array_equal(rto, k * np.arange(B + 1))
    for b in range(B):
        assert np.all(np.diff(idx[b]) > 0) and idx[b][0] >= 0 and idx[b][-1] < M
        assert np.array_equal(idx[b], _topk_by(score[b].astype(np.float64), k))
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    for b in (0, 17, 31):
        kc = _image_rows(cache_k, bt, img0.cpu().numpy(), b, 0, M)
        ref = O.ads_relevance_cached(qv[b], int(q_pos[b]), kc, D, sec, 1e6)
        _check_seq(score[b], ref, idx[b], k, M)


def test_select_cached_after_prefill_capture():
    """The cache written by prcr_prefill_capture from the raw store: the
    cached-key relevance is the raw-store relevance up to the bf16 rounding
    of the rotated keys, and equals the oracle on the rows actually stored."""
    import paper_2606_26631_gb300 as prcr
    from workloads import get, make_batch
    wl = get("qwen2vl-2b")
    batch = make_batch(wl, device=DEV)
    B, nL, M, H, D = wl.n_seqs, wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    layer, Hq, k = 11, 12, 100
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta)
    sd = prcr.store_desc(batch.store_k, batch.store_v, batch.coords)
    S = M + 16
    ck = torch.zeros((B, nL, S, H, D), dtype=torch.bfloat16, device=DEV)
    cv = torch.zeros_like(ck)
    cd = prcr.cache_contiguous(ck, cv)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    # this workload's store holds the raw rows already: capture them again
    # from a copy into the cache at slots 16 .. 16 + M - 1
    for b in range(B):
        src_k = batch.store_k[b].clone()  # [nL, M, H, D]
        src_v = batch.store_v[b].clone()
        prcr.prefill_capture(cfg, sd, cd, b, 0, 0, 16, src_k, src_v, batch.coords[b].contiguous(),
                             status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    g = torch.Generator(device=DEV).manual_seed(12)
    q = (3.0 * torch.randn((B, Hq, D), device=DEV, generator=g)).to(torch.bfloat16)
    img0 = torch.full((B,), 16, dtype=torch.int32, device=DEV)
    idx, _, _, score, st = _run(cfg, cd, layer, q, batch.p_txt, img0, M, k)
    assert st == 0
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    coords = batch.coords.cpu().numpy()
    for b in range(B):
        kc = _image_rows(ck, None, img0.cpu().numpy(), b, layer, M)
        ref = O.ads_relevance_cached(qv[b], int(batch.p_txt[b]), kc, D, wl.sections, wl.theta)
        _check_seq(score[b], ref, idx[b], k, M)
        raw = O.ads_relevance(qv[b], int(batch.p_txt[b]),
                              batch.store_k[b, layer].view(torch.int16).cpu().numpy(), coords[b], D,
                              wl.sections, wl.theta)
        # bf16 keys carry 2^-9 relative rounding: for these query and key
        # scales a logit moves by ~6e-3 (one sigma), the relevance by as much
        assert (np.abs(score[b] - raw) / raw).max() <= 5e-2


def test_select_single_token_both_sources():
    """One visual token, k = 1: the softmax over one token is 1 for every
    head, so the relevance is exactly 1 (4 heads x 0.25) and the token is
    selected, from the raw store and from the cache alike."""
    import paper_2606_26631_gb300 as prcr
    B, H, Hq, D, M, sec = 2, 2, 4, 64, 1, (8, 12, 12)
    g = torch.Generator(device=DEV).manual_seed(2)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    q = torch.randn((B, Hq, D), device=DEV, generator=g).to(torch.bfloat16)
    q_pos = torch.tensor([50, 70], dtype=torch.int64, device=DEV)
    ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=DEV)
    sk = torch.randn((B, 1, M, H, D), device=DEV, generator=g).to(torch.bfloat16)
    coords = torch.tensor([[[0, 3, 4]], [[0, 5, 6]]], dtype=torch.int32, device=DEV)
    for source in ("raw", "cache"):
        idx = torch.full((B,), -7, dtype=torch.int32, device=DEV)
        sro = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
        rto = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
        score = torch.full((B, M), -1.0, dtype=torch.float32, device=DEV)
        if source == "raw":
            prcr.select_topk(cfg, prcr.store_desc(sk, sk, coords), 0, q, q_pos, 1, idx, sro, rto, ws,
                             score)
        else:
            status = torch.zeros(1, dtype=torch.int32, device=DEV)
            img0 = torch.zeros(B, dtype=torch.int32, device=DEV)
            prcr.select_topk_cached(cfg, prcr.cache_contiguous(sk, sk), 0, q, q_pos, img0, M, 1, idx,
                                    sro, rto, status, ws, score)
        torch.cuda.synchronize()
        assert idx.tolist() == [0, 0], source
        assert sro.tolist() == [0, 1, 2] and rto.tolist() == [0, 1, 2], source
        assert score.cpu().tolist() == [[1.0], [1.0]], source


@pytest.mark.parametrize("cached", [False, True])
def test_select_most_query_heads(cached):
    """128 query heads (16 KV heads x 8, head_dim 64: the largest head count
    the selection takes) from the raw store and from the cache."""
    import paper_2606_26631_gb300 as prcr
    B, H, Hq, D, M, k, sec = 2, 16, 128, 64, 300, 40, (8, 12, 12)
    g = torch.Generator(device=DEV).manual_seed(21)
    sk = torch.randn((B, 1, M, H, D), device=DEV, generator=g).to(torch.bfloat16)
    coords = torch.randint(0, 40, (B, M, 3), device=DEV, generator=g, dtype=torch.int32)
    q = (2.0 * torch.randn((B, Hq, D), device=DEV, generator=g)).to(torch.bfloat16)
    q_pos = torch.tensor([700, 3000], dtype=torch.int64, device=DEV)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    ws = torch.empty(prcr.select_workspace_size(B, Hq, M), dtype=torch.uint8, device=DEV)
    idx = torch.full((B * k,), -7, dtype=torch.int32, device=DEV)
    sro = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    rto = torch.full((B + 1,), -7, dtype=torch.int32, device=DEV)
    score = torch.full((B, M), -1.0, dtype=torch.float32, device=DEV)
    if cached:
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        prcr.select_topk_cached(cfg, prcr.cache_contiguous(sk, sk), 0, q, q_pos,
                                torch.zeros(B, dtype=torch.int32, device=DEV), M, k, idx, sro, rto,
                                status, ws, score)
    else:
        prcr.select_topk(cfg, prcr.store_desc(sk, sk, coords), 0, q, q_pos, k, idx, sro, rto, ws, score)
    torch.cuda.synchronize()
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    kb = sk.view(torch.int16).cpu().numpy()
    idx = idx.view(B, k).cpu().numpy()
    score = score.cpu().numpy()
    for b in range(B):
        if cached:
            ref = O.ads_relevance_cached(qv[b], int(q_pos[b]), O.bf16_bits_to_f64(kb[b, 0]), D, sec, 1e6)
        else:
            ref = O.ads_relevance(qv[b], int(q_pos[b]), kb[b, 0], coords[b].cpu().numpy(), D, sec, 1e6)
        _check_seq(score[b], ref, idx[b], k, M)


def test_select_cached_query_position_range():
    """A query position of 2^31 or more sets PRCR_ST_POS_RANGE; every token of
    that sequence gets relevance 0, so it selects its first k tokens (equal
    relevance: lower index first), while the other sequence of the batch keeps
    the oracle's relevance and a valid selection."""
    import paper_2606_26631_gb300 as prcr
    D, H, Hq, M, k, sec = 64, 2, 8, 40, 5, (8, 12, 12)
    cache_k, bt, img0 = _make_cache(2, 1, H, D, M, False, 0, seed=3)
    cfg = prcr.rope_cfg(1, H, D, sec, 1e6)
    q = torch.randn((2, Hq, D), device=DEV).to(torch.bfloat16)
    qv = O.bf16_bits_to_f64(q.view(torch.int16).cpu().numpy())
    cd = prcr.cache_contiguous(cache_k, cache_k)
    for pos, bad in ((2 ** 31 + 7, True), (-(2 ** 31), True), (2 ** 31 - 1, False)):
        qp = torch.tensor([pos, 700], dtype=torch.int64, device=DEV)
        idx, _, _, score, st = _run(cfg, cd, 0, q, qp, img0, M, k)
        assert st == (prcr.ST_POS_RANGE if bad else 0)
        if bad:
            assert np.all(score[0] == 0.0)
            assert np.array_equal(idx[0], np.arange(k))
        kc = _image_rows(cache_k, None, img0.cpu().numpy(), 1, 0, M)
        ref = O.ads_relevance_cached(qv[1], 700, kc, D, sec, 1e6)
        _check_seq(score[1], ref, idx[1], k, M)
