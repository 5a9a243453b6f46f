"""GPU parity of prcr_prefill_capture (Sec. 3.1 with Eq.
"historical_position_bound_kv") against the oracle's prefill_capture: the
store receives the raw rows and coordinates bit for bit; the cache receives
the key rotated at the original coordinate (within the K tolerance) and the
value bit for bit at consecutive slots; nothing else in the cache changes."""
import numpy as np
import pytest
import torch

from oracle import prcr_oracle as O
from workloads import CANARY_BITS, get, make_batch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _cache(wl, B, slot_begin, M, paged, rng):
    nL, H, D = wl.n_layers, wl.n_kv_heads, wl.head_dim
    if not paged:
        S = int(max(slot_begin) + M + 5)
        shape = (B, nL, S, H, D)
        bt = None
    else:
        bs = 16
        first = [s // bs for s in slot_begin]
        last = [(s + M - 1) // bs for s in slot_begin]
        n = sum(l - f + 1 for f, l in zip(first, last))
        perm = rng.permutation(n)
        bt = np.full((B, max(last) + 2), -1, dtype=np.int32)
        k = 0
        for b in range(B):
            for lb in range(first[b], last[b] + 1):
                bt[b, lb] = perm[k]
                k += 1
        shape = (nL, n, bs, H, D)
        bt = torch.from_numpy(bt).to(DEV)
    ck = torch.full(shape, CANARY_BITS, dtype=torch.int16, device=DEV).view(torch.bfloat16)
    cv = torch.full(shape, CANARY_BITS, dtype=torch.int16, device=DEV).view(torch.bfloat16)
    return ck, cv, bt


def _rows(ck, bt, b, slots, layers, paged):
    lay = torch.as_tensor(list(layers), device=DEV)
    s = torch.as_tensor(slots, device=DEV)
    if not paged:
        return ck[b][lay[None, :], s[:, None]]
    blk = bt[b][s // 16].long()
    return ck[lay[None, :], blk[:, None], (s % 16)[:, None]]


@pytest.mark.parametrize("name,paged,layers", [("qwen2vl-2b", False, None),
                                               ("qwen25vl-7b", True, (0, 13, 27)),
                                               ("tiny", True, None)])
def test_prefill_capture_parity(name, paged, layers):
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    wl = get(name)
    src = make_batch(wl, device=DEV)  # its raw store stands in for the prefill projections
    B, nL, M = wl.n_seqs, wl.n_layers, wl.n_tokens
    rng = np.random.default_rng(4)
    slot_begin = [16 + 5 * b for b in range(B)]
    ck, cv, bt = _cache(wl, B, slot_begin, M, paged, rng)
    store_k = torch.full_like(src.store_k.view(torch.int16), 7).view(torch.bfloat16)
    store_v = torch.full_like(src.store_v.view(torch.int16), 7).view(torch.bfloat16)
    coords = torch.zeros_like(src.coords)
    cfg = prcr.rope_cfg(nL, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta)
    sd = prcr.store_desc(store_k, store_v, coords)
    cd = prcr.cache_paged(ck, cv, bt) if paged else prcr.cache_contiguous(ck, cv)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    half, lh = M // 3, nL // 2
    for b in range(B):
        # two token ranges x two layer ranges, as a layer-by-layer prefill would call it
        for (m0, m1) in ((0, half), (half, M)):
            for (l0, l1) in ((0, lh), (lh, nL)):
                prcr.prefill_capture(cfg, sd, cd, b, l0, m0, slot_begin[b] + m0,
                                     src.store_k[b, l0:l1, m0:m1], src.store_v[b, l0:l1, m0:m1],
                                     src.coords[b, m0:m1].contiguous(), status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(store_k.view(torch.int16), src.store_k.view(torch.int16))
    assert torch.equal(store_v.view(torch.int16), src.store_v.view(torch.int16))
    assert torch.equal(coords, src.coords)
    layers = list(range(nL)) if layers is None else list(layers)
    for b in range(B):
        k_raw = pu.bits(src.store_k[b].transpose(0, 1)[:, layers])  # [M, L, H, D]
        v_raw = pu.bits(src.store_v[b].transpose(0, 1)[:, layers])
        crd = src.coords[b].cpu().numpy()
        _, _, k_want, v_want = O.prefill_capture(k_raw, v_raw, crd, wl.head_dim, wl.sections,
                                                 wl.theta)
        slots = np.arange(M) + slot_begin[b]
        k_got = pu.bits(_rows(ck, bt, b, slots, layers, paged))
        v_got = pu.bits(_rows(cv, bt, b, slots, layers, paged))
        assert np.array_equal(v_got, v_want)
        e = pu.k_error(k_got, k_want, k_raw)
        assert e["max_err"] <= pu.K_TOL, e
    # untouched: exactly B * M rows per layer were written
    row = wl.n_kv_heads * wl.head_dim
    for c in (ck, cv):
        c16 = c.view(torch.int16)
        for l in range(nL):
            lay = c16[:, l] if not paged else c16[l]
            assert int((lay == CANARY_BITS).sum().item()) == lay.numel() - B * M * row


def test_prefill_capture_capacity_error():
    import paper_2606_26631_gb300 as prcr
    wl = get("tiny")
    src = make_batch(wl, device=DEV)
    M = wl.n_tokens
    ck = torch.full((1, 2, M + 10, 2, 64), CANARY_BITS, dtype=torch.int16, device=DEV).view(torch.bfloat16)
    cv = ck.clone()
    store_k = torch.zeros_like(src.store_k); store_v = torch.zeros_like(src.store_v)
    coords = torch.zeros_like(src.coords)
    cfg = prcr.rope_cfg(2, 2, 64, wl.sections, wl.theta)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    prcr.prefill_capture(cfg, prcr.store_desc(store_k, store_v, coords),
                         prcr.cache_contiguous(ck, cv), 0, 0, 0, 20, src.store_k[0], src.store_v[0],
                         src.coords[0].contiguous(), status)
    torch.cuda.synchronize()
    assert int(status.item()) & prcr.ST_CAPACITY
    # the store is complete; the cache got exactly the slots that fit (20 .. M+9)
    assert torch.equal(store_k.view(torch.int16), src.store_k.view(torch.int16))
    fit = M + 10 - 20
    for c in (ck, cv):
        n = int((c.view(torch.int16) == CANARY_BITS).sum().item())
        assert n == c.numel() - fit * 2 * 128


@pytest.mark.slow
def test_prefill_capture_full_size_sampled():
    """The capture configuration bench.py times (qwen3vl-8b: 16 sequences x
    8192 tokens x 36 layers, one call per sequence over all layers into a
    shuffled paged cache from slot 0); store bit-exact everywhere, cache rows
    on sampled sequences, tokens and layers against the oracle."""
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    wl = get("qwen3vl-8b")
    src = make_batch(wl, device=DEV)
    B, nL, M, H, D = wl.n_seqs, wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    store_k = torch.empty_like(src.store_k)
    store_v = torch.empty_like(src.store_v)
    coords = torch.empty_like(src.coords)
    bs = 16
    nblk = (M + bs - 1) // bs
    perm = torch.randperm(B * nblk, device=DEV, generator=torch.Generator(device=DEV).manual_seed(2))
    bt = perm.view(B, nblk).to(torch.int32).contiguous()
    ck = torch.empty((nL, B * nblk, bs, H, D), dtype=torch.bfloat16, device=DEV)
    cv = torch.empty_like(ck)
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta)
    sd = prcr.store_desc(store_k, store_v, coords)
    cd = prcr.cache_paged(ck, cv, bt)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    for b in range(B):
        prcr.prefill_capture(cfg, sd, cd, b, 0, 0, 0, src.store_k[b], src.store_v[b], src.coords[b],
                             status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(store_k.view(torch.int16), src.store_k.view(torch.int16))
    assert torch.equal(store_v.view(torch.int16), src.store_v.view(torch.int16))
    assert torch.equal(coords, src.coords)
    rng = np.random.default_rng(9)
    layers = [0, nL // 2, nL - 1]
    for b in (0, B // 2, B - 1):
        toks = np.sort(rng.choice(M, size=512, replace=False))
        t_dev = torch.as_tensor(toks, device=DEV)
        k_raw = pu.bits(src.store_k[b][:, t_dev].transpose(0, 1)[:, layers])  # [n, L, H, D]
        v_raw = pu.bits(src.store_v[b][:, t_dev].transpose(0, 1)[:, layers])
        crd = src.coords[b].cpu().numpy()[toks]
        _, _, k_want, v_want = O.prefill_capture(k_raw, v_raw, crd, D, wl.sections, wl.theta)
        k_got = pu.bits(_rows(ck, bt, b, toks, layers, True))
        v_got = pu.bits(_rows(cv, bt, b, toks, layers, True))
        assert np.array_equal(v_got, v_want)
        e = pu.k_error(k_got, k_want, k_raw)
        assert e["max_err"] <= pu.K_TOL, e
    del src, store_k, store_v, ck, cv
    torch.cuda.empty_cache()


def test_prefill_capture_interleaved_layout():
    """The cache keys rotated with the interleaved M-RoPE band layout."""
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    wl = get("qwen2vl-2b")
    src = make_batch(wl, device=DEV)
    nL, M, H, D = wl.n_layers, wl.n_tokens, wl.n_kv_heads, wl.head_dim
    rng = np.random.default_rng(6)
    ck, cv, bt = _cache(wl, 1, [7], M, False, rng)
    store_k = torch.empty_like(src.store_k)
    store_v = torch.empty_like(src.store_v)
    coords = torch.empty_like(src.coords)
    cfg = prcr.rope_cfg(nL, H, D, wl.sections, wl.theta, O.LAYOUT_INTERLEAVED)
    sd = prcr.store_desc(store_k, store_v, coords)
    cd = prcr.cache_contiguous(ck, cv)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    prcr.prefill_capture(cfg, sd, cd, 0, 0, 0, 7, src.store_k[0], src.store_v[0], src.coords[0],
                         status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    layers = [0, nL // 2, nL - 1]
    k_raw = pu.bits(src.store_k[0].transpose(0, 1)[:, layers])
    v_raw = pu.bits(src.store_v[0].transpose(0, 1)[:, layers])
    _, _, k_want, v_want = O.prefill_capture(k_raw, v_raw, src.coords[0].cpu().numpy(), D,
                                             wl.sections, wl.theta, O.LAYOUT_INTERLEAVED)
    slots = np.arange(M) + 7
    assert np.array_equal(pu.bits(_rows(cv, bt, 0, slots, layers, False)), v_want)
    e = pu.k_error(pu.bits(_rows(ck, bt, 0, slots, layers, False)), k_want, k_raw)
    assert e["max_err"] <= pu.K_TOL, e
