"""GPU parity of prcr_decode_attention (Eq. "decode_with_active_cache")
against the oracle's fp64 decode_attention.

1. Decode over a populated input cache (contiguous and paged, GQA groups
   1 / 4 / 7, head_dim 64 / 128 / 256, sequences long enough to be split).
   Bar: max |o_gpu - o_ref| <= 1e-4 * max |V| (float32 logits, exp and
   accumulation over at most a few thousand slots per chunk stay ~1e-6).
2. End to end: revisit rows appended by prcr_rebind_inject into a cache whose
   context rows are data, then decoded at next_pos over cache_len_out. The
   expected cache is the context plus the oracle's rebound keys rounded to
   bf16 (the value a correct kernel stores); bar 1e-3 * max |V|.
3. Relative positions only (Eq. "direct_reuse_score"): a cache made only of
   revisited rows decoded at p + 1 gives the same output when the text
   position moves by a constant (up to the bf16 rounding of the keys).
"""
import numpy as np
import pytest
import torch

from oracle import prcr_oracle as O
from workloads import Workload, get, make_batch, make_decode_inputs

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _f64(t):
    return O.bf16_bits_to_f64(t.contiguous().view(torch.int16).cpu().numpy())


def _cache_rows(cache_k, cache_v, block_table, b, n, paged):
    """[n, n_L, H, D] value arrays of slots 0..n-1 of sequence b (input data)."""
    s = torch.arange(n, device=cache_k.device)
    if not paged:
        return _f64(cache_k[b, :, :n].transpose(0, 1)), _f64(cache_v[b, :, :n].transpose(0, 1))
    bs = cache_k.shape[2]
    blk = block_table[b][s // bs].long()
    off = s % bs
    return _f64(cache_k[:, blk, off].transpose(0, 1)), _f64(cache_v[:, blk, off].transpose(0, 1))


def _run_decode(cfg, cache_desc, q, q_pos, seq_len, max_len):
    import paper_2606_26631_gb300 as prcr
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    nbytes = prcr.decode_workspace_size(cfg, q.shape[0], q.shape[2], max_len)
    ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
    prcr.decode_attention(cfg, cache_desc, q, q_pos, seq_len, max_len, out, status, ws)
    torch.cuda.synchronize()
    return out, int(status.item())


CASES = [  # (B, layers, H, Hq, D, max_len, paged)
    (3, 3, 8, 32, 128, 3000, True),
    (2, 2, 2, 14, 64, 700, False),
    (2, 2, 4, 4, 256, 1200, True),
    (5, 1, 4, 28, 128, 9000, True),
    # one sequence of the Table 3 shape (small batch: KV heads split over
    # CTAs, chunk rows requested into L2 ahead of the tile loop)
    (1, 36, 8, 32, 128, 933, False),
    (2, 2, 8, 16, 64, 500, True),
    # the head-split kernel at the ends of the GQA range: 1 and 8 query heads per KV head
    (1, 2, 8, 8, 128, 500, False),
    (1, 2, 8, 64, 128, 300, True),
]


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}L{c[1]}H{c[2]}Hq{c[3]}D{c[4]}S{c[5]}{'p' if c[6] else 'c'}" for c in CASES])
def test_decode_parity(case):
    import paper_2606_26631_gb300 as prcr
    B, nL, H, Hq, D, max_len, paged = case
    sec = (D // 8, D // 8 + (D // 2 - 3 * (D // 8)) // 2, 0)
    sec = (sec[0], sec[1], D // 2 - sec[0] - sec[1])
    inp = make_decode_inputs(B, nL, H, Hq, D, max_len, paged, device=DEV, seed=7)
    cfg = prcr.rope_cfg(nL, H, D, sec, 1e6)
    cd = (prcr.cache_paged(inp["cache_k"], inp["cache_v"], inp["block_table"]) if paged
          else prcr.cache_contiguous(inp["cache_k"], inp["cache_v"]))
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], inp["seq_len"], max_len)
    assert st == 0
    got = out.cpu().numpy()
    qv = _f64(inp["q"])
    for b in range(B):
        n = int(inp["seq_len"][b])
        K, V = _cache_rows(inp["cache_k"], inp["cache_v"], inp["block_table"], b, n, paged)
        for l in range(nL):
            ref = O.decode_attention(qv[b, l], int(inp["q_pos"][b]), K[:, l], V[:, l], D, sec, 1e6)
            err = np.abs(got[b, l] - ref).max() / np.abs(V[:, l]).max()
            assert err <= 1e-4, (b, l, err)


@pytest.mark.parametrize("H,Hq,D,paged", [(8, 32, 128, False), (4, 16, 128, True), (2, 14, 64, False),
                                         (4, 8, 256, True)])
def test_decode_empty_and_single_slot(H, Hq, D, paged):
    """A sequence with no slots gets zeros; one with a single slot gets that
    slot's V row exactly (its softmax weight is exactly 1); a longer one
    beside them still matches the oracle. Covers the head-split kernel
    (8 KV heads), the one-CTA-per-chunk kernel, head_dim 64 and the
    CUDA-core kernel (head_dim 256)."""
    import paper_2606_26631_gb300 as prcr
    B, nL, max_len = 3, 2, 300
    sec = (D // 8, D // 8 + (D // 2 - 3 * (D // 8)) // 2, 0)
    sec = (sec[0], sec[1], D // 2 - sec[0] - sec[1])
    inp = make_decode_inputs(B, nL, H, Hq, D, max_len, paged, device=DEV, seed=19)
    seq_len = torch.tensor([0, 1, max_len], dtype=torch.int32, device=DEV)
    cfg = prcr.rope_cfg(nL, H, D, sec, 1e6)
    cd = (prcr.cache_paged(inp["cache_k"], inp["cache_v"], inp["block_table"]) if paged
          else prcr.cache_contiguous(inp["cache_k"], inp["cache_v"]))
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], seq_len, max_len)
    assert st == 0
    got = out.cpu().numpy()
    assert np.all(got[0] == 0.0)
    g = Hq // H
    K1, V1 = _cache_rows(inp["cache_k"], inp["cache_v"], inp["block_table"], 1, 1, paged)
    for l in range(nL):
        for h in range(Hq):
            assert np.array_equal(got[1, l, h], V1[0, l, h // g].astype(np.float32)), (l, h)
    K, V = _cache_rows(inp["cache_k"], inp["cache_v"], inp["block_table"], 2, max_len, paged)
    qv = _f64(inp["q"])
    for l in range(nL):
        ref = O.decode_attention(qv[2, l], int(inp["q_pos"][2]), K[:, l], V[:, l], D, sec, 1e6)
        assert np.abs(got[2, l] - ref).max() / np.abs(V[:, l]).max() <= 1e-4


def test_decode_device_errors():
    """Device-detected errors: an unmapped block in a sequence's range sets
    PRCR_ST_NO_BLOCK and its slots are left out of the softmax; a length
    beyond the capacity sets PRCR_ST_CAPACITY and is clamped to it; a length
    above max_len sets PRCR_ST_CAPACITY too. Outputs stay the oracle's
    attention over the slots that remain (where those are defined)."""
    import paper_2606_26631_gb300 as prcr
    nL, H, Hq, D, sec = 2, 2, 8, 64, (8, 12, 12)
    cfg = prcr.rope_cfg(nL, H, D, sec, 1e6)
    # (a) paged: block 3 of sequence 1 (its slots 48..63) unmapped
    inp = make_decode_inputs(2, nL, H, Hq, D, 200, True, device=DEV, seed=23)
    bt = inp["block_table"].clone()
    bt[1, 3] = -1
    cd = prcr.cache_paged(inp["cache_k"], inp["cache_v"], bt)
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], inp["seq_len"], 200)
    assert st & prcr.ST_NO_BLOCK
    got = out.cpu().numpy()
    qv = _f64(inp["q"])
    n1 = int(inp["seq_len"][1])
    K, V = _cache_rows(inp["cache_k"], inp["cache_v"], inp["block_table"], 1, n1, True)
    keep = np.array([s for s in range(n1) if s // 16 != 3])
    for l in range(nL):
        ref = O.decode_attention(qv[1, l], int(inp["q_pos"][1]), K[keep, l], V[keep, l], D, sec, 1e6)
        assert np.abs(got[1, l] - ref).max() / np.abs(V[:, l]).max() <= 1e-4
    K0, V0 = _cache_rows(inp["cache_k"], inp["cache_v"], inp["block_table"], 0, int(inp["seq_len"][0]),
                         True)
    for l in range(nL):
        ref = O.decode_attention(qv[0, l], int(inp["q_pos"][0]), K0[:, l], V0[:, l], D, sec, 1e6)
        assert np.abs(got[0, l] - ref).max() / np.abs(V0[:, l]).max() <= 1e-4
    # (b) contiguous, capacity 208 slots: a length of 300 is clamped to 208
    inp = make_decode_inputs(1, nL, H, Hq, D, 200, False, device=DEV, seed=24)
    cap = inp["cache_k"].shape[2]
    cd = prcr.cache_contiguous(inp["cache_k"], inp["cache_v"])
    seq_len = torch.tensor([300], dtype=torch.int32, device=DEV)
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], seq_len, cap)
    assert st & prcr.ST_CAPACITY
    got = out.cpu().numpy()
    qv = _f64(inp["q"])
    K, V = _cache_rows(inp["cache_k"], inp["cache_v"], None, 0, cap, False)
    for l in range(nL):
        ref = O.decode_attention(qv[0, l], int(inp["q_pos"][0]), K[:, l], V[:, l], D, sec, 1e6)
        assert np.abs(got[0, l] - ref).max() / np.abs(V[:, l]).max() <= 1e-4
    # (c) a length above the max_len the call was split for
    seq_len = torch.tensor([150], dtype=torch.int32, device=DEV)
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], seq_len, 100)
    assert st & prcr.ST_CAPACITY
    assert torch.isfinite(out).all()


def test_decode_query_position_range():
    """A query position of 2^31 or more is beyond the fixed-point angle
    reduction: PRCR_ST_POS_RANGE, and that sequence reads no slot (its output
    is zeros) while the other sequence of the batch matches the oracle.
    Head-split and one-CTA-per-chunk kernels, split and unsplit sequences."""
    import paper_2606_26631_gb300 as prcr
    sec = (16, 24, 24)
    for H, Hq, max_len in ((8, 32, 300), (2, 8, 300), (8, 32, 3000)):
        inp = make_decode_inputs(2, 2, H, Hq, 128, max_len, False, device=DEV, seed=5)
        cfg = prcr.rope_cfg(2, H, 128, sec, 1e6)
        cd = prcr.cache_contiguous(inp["cache_k"], inp["cache_v"])
        qp = inp["q_pos"].clone()
        qp[0] = 2 ** 31
        out, st = _run_decode(cfg, cd, inp["q"], qp, inp["seq_len"], max_len)
        assert st == prcr.ST_POS_RANGE
        got = out.cpu().numpy()
        assert np.all(got[0] == 0.0)
        n = int(inp["seq_len"][1])
        K, V = _cache_rows(inp["cache_k"], inp["cache_v"], None, 1, n, False)
        qv = _f64(inp["q"])
        for l in range(2):
            ref = O.decode_attention(qv[1, l], int(qp[1]), K[:, l], V[:, l], 128, sec, 1e6)
            assert np.abs(got[1, l] - ref).max() / np.abs(V[:, l]).max() <= 1e-4
        qp[0] = -(2 ** 31)
        out, st = _run_decode(cfg, cd, inp["q"], qp, inp["seq_len"], max_len)
        assert st == prcr.ST_POS_RANGE and bool((out[0] == 0).all().item())
        qp[0] = 2 ** 31 - 1
        _, st = _run_decode(cfg, cd, inp["q"], qp, inp["seq_len"], max_len)
        assert st == 0


def test_decode_unaligned_query():
    """Query rows only 4-byte aligned (the ABI's minimum) take the scalar
    loads of the rotation: the output is bit-identical to the aligned call."""
    import paper_2606_26631_gb300 as prcr
    B, nL, H, Hq, D, max_len = 1, 4, 8, 32, 128, 933
    inp = make_decode_inputs(B, nL, H, Hq, D, max_len, False, device=DEV, seed=3)
    cfg = prcr.rope_cfg(nL, H, D, (16, 24, 24), 1e6)
    cd = prcr.cache_contiguous(inp["cache_k"], inp["cache_v"])
    q = inp["q"]
    buf = torch.empty(q.numel() + 2, dtype=torch.bfloat16, device=DEV)
    q_odd = buf[2:].view(q.shape)
    q_odd.copy_(q)
    assert q_odd.data_ptr() % 16 == 4
    ref, st0 = _run_decode(cfg, cd, q, inp["q_pos"], inp["seq_len"], max_len)
    got, st1 = _run_decode(cfg, cd, q_odd, inp["q_pos"], inp["seq_len"], max_len)
    assert st0 == 0 and st1 == 0
    assert torch.equal(ref, got)


def test_inject_then_decode():
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    for name in ("qwen2vl-2b", "qwen25vl-7b"):
        wl = get(name)
        batch = make_batch(wl, device=DEV, context="random")
        B, nL, H, D = wl.n_seqs, wl.n_layers, wl.n_kv_heads, wl.head_dim
        Hq = {"qwen2vl-2b": 12, "qwen25vl-7b": 28}[name]
        # expected cache: context rows as given + the oracle's rows at the slots
        ctx_k = batch.cache_k.clone()
        ctx_v = batch.cache_v.clone()
        rv = pu.make_revisit(batch)
        rv.run()
        torch.cuda.synchronize()
        assert rv.status_value() == 0
        pl = pu.oracle_plan(batch)
        g = torch.Generator(device=DEV)
        g.manual_seed(11)
        q = torch.randn((B, nL, Hq, D), generator=g, device=DEV).to(torch.bfloat16)
        max_len = int(pl["cache_len_out"].max())
        cfg = rv.cfg
        out, st = _run_decode(cfg, rv.cache, q, rv.next_pos, rv.cache_len_out, max_len)
        assert st == 0
        got = out.cpu().numpy()
        qv = _f64(q)
        idx = batch.idx.cpu().numpy()
        for b in range(B):
            n_ctx = int(batch.cache_len_in[b])
            n_all = int(pl["cache_len_out"][b])
            K, V = _cache_rows(ctx_k, ctx_v, batch.block_table, b, n_all, batch.paged)
            toks = np.nonzero(pl["seq"] == b)[0]
            slots = pl["slot"][toks]
            k_raw = pu.bits(batch.store_k[b][:, torch.as_tensor(idx[toks], device=DEV).long()]
                            .transpose(0, 1))
            v_raw = pu.bits(batch.store_v[b][:, torch.as_tensor(idx[toks], device=DEV).long()]
                            .transpose(0, 1))
            k_hat = O.rebind_keys(k_raw, pl["pos"][toks], D, wl.sections, wl.theta)
            K[slots] = O.f64_to_bf16_rne(k_hat)
            V[slots] = O.bf16_bits_to_f64(v_raw)
            assert n_ctx + len(toks) == n_all
            for l in range(nL):
                ref = O.decode_attention(qv[b, l], int(pl["next_pos"][b]), K[:, l], V[:, l], D,
                                         wl.sections, wl.theta)
                err = np.abs(got[b, l] - ref).max() / np.abs(V[:, l]).max()
                assert err <= 1e-3, (name, b, l, err)


def test_decode_sees_only_relative_positions():
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    wl = Workload(name="rel", n_layers=2, n_kv_heads=4, head_dim=128, sections=(16, 24, 24),
                  n_seqs=2, grids=((1, 24, 24),), selection="random", cache="contiguous",
                  cur_pos=("fixed", 3000), extra=(1, 1, 200, 300))
    outs = []
    for shift in (0, 12345):
        batch = make_batch(wl, device=DEV, seed=3)
        batch.p_txt += shift
        batch.cache_len_in.zero_()  # the cache holds only the revisited rows
        rv = pu.make_revisit(batch)
        rv.run()
        g = torch.Generator(device=DEV)
        g.manual_seed(5)
        q = torch.randn((2, 2, 16, 128), generator=g, device=DEV).to(torch.bfloat16)
        out, st = _run_decode(rv.cfg, rv.cache, q, rv.next_pos, rv.cache_len_out,
                              int(rv.cache_len_out.max()))
        assert st == 0 and rv.status_value() == 0
        outs.append(out.cpu().numpy())
    vmax = float(torch.abs(batch.store_v.float()).max())
    assert np.abs(outs[0] - outs[1]).max() / vmax <= 2e-3


def _layer_rows(inp, b, l, n):
    """[n, H, D] value arrays of slots 0..n-1 of sequence b at layer l (paged)."""
    s = torch.arange(n, device=inp["cache_k"].device)
    bs = inp["cache_k"].shape[2]
    blk = inp["block_table"][b][s // bs].long()
    off = s % bs
    return _f64(inp["cache_k"][l, blk, off]), _f64(inp["cache_v"][l, blk, off])


@pytest.mark.slow
def test_decode_full_size_sampled():
    """The decode configuration bench.py times (qwen3vl-8b shape: 16 sequences
    of up to 8192 slots, 36 layers, 8 KV heads, 32 query heads, paged, the same
    seed, so the same chunk split and merge launch); sampled (sequence, layer)
    pairs, every query head, against the oracle."""
    import paper_2606_26631_gb300 as prcr
    wl = get("qwen3vl-8b")
    B, nL, H, D = wl.n_seqs, wl.n_layers, wl.n_kv_heads, wl.head_dim
    Hq, max_len = 4 * H, 8192
    inp = make_decode_inputs(B, nL, H, Hq, D, max_len, True, device=DEV, seed=1)
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta)
    cd = prcr.cache_paged(inp["cache_k"], inp["cache_v"], inp["block_table"])
    out, st = _run_decode(cfg, cd, inp["q"], inp["q_pos"], inp["seq_len"], max_len)
    assert st == 0
    got = out.cpu().numpy()
    qv = _f64(inp["q"])
    for b in (0, B // 2, B - 1):
        n = int(inp["seq_len"][b])
        for l in (0, nL // 2, nL - 1):
            K, V = _layer_rows(inp, b, l, n)
            ref = O.decode_attention(qv[b, l], int(inp["q_pos"][b]), K, V, D, wl.sections, wl.theta)
            err = np.abs(got[b, l] - ref).max() / np.abs(V).max()
            assert err <= 1e-4, (b, l, n, err)
    del inp
    torch.cuda.empty_cache()
