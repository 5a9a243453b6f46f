"""GPU parity: the CUDA path through the C ABI against the CPU oracle.

Small and medium workloads are compared completely (every position, slot,
token x layer x head row and every untouched cache row). The two largest
workloads run at full size, in the launch configuration the benchmark times;
there every position/slot/length is compared, K/V rows on sampled
(sequence, layer) pairs, and the untouched-row property over the whole cache.
"""
import gc

import re

import numpy as np
import pytest
import torch

from oracle import prcr_oracle as O
from workloads import Workload, get, make_batch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _run(batch, **kw):
    import parity_util as pu
    rv = pu.make_revisit(batch, **kw)
    rv.run()
    torch.cuda.synchronize()
    return rv


def _free():
    gc.collect()
    torch.cuda.empty_cache()


@pytest.fixture(autouse=True)
def _cleanup():
    yield
    _free()


@pytest.mark.parametrize("name", ["tiny", "qwen2vl-2b", "paper-8b-k32", "paper-8b-k128",
                                  "qwen25vl-7b"])
def test_full_parity(name):
    import parity_util as pu
    batch = make_batch(get(name), device=DEV)
    rv = _run(batch)
    assert rv.status_value() == 0
    e = pu.full_check(batch, rv)
    assert e["n"] == batch.total_k * batch.wl.n_layers * batch.wl.row_elems
    print(name, e)


def test_tiny_matches_oracle_whole_call():
    """Tiny end to end against the oracle's own Algorithm 1 (its own gather)."""
    import parity_util as pu
    batch = make_batch(get("tiny"), device=DEV)
    rv = _run(batch)
    ref = pu.full_oracle_call(batch)
    pl = pu.oracle_plan(batch)
    pu.check_plan(rv, ref)
    tokens = np.arange(batch.total_k)
    k_got = pu.bits(pu.gather_cache(batch, batch.cache_k, tokens, pl, range(2)))
    v_got = pu.bits(pu.gather_cache(batch, batch.cache_v, tokens, pl, range(2)))
    assert np.array_equal(v_got, ref["v_hat"].astype(np.int16))
    e = pu.k_error(k_got, ref["k_hat"], ref["k_raw"])
    assert e["max_err"] <= pu.K_TOL
    # positions are the hand-worked values 198 + {3, 18, 33, 48}/17 (rows/cols), t = 198 + 3/17
    vals = sorted(set(np.round(rv.pos.cpu().numpy()[:, 1], 9)))
    assert vals == sorted(set(np.round([198 + x / 17 for x in (3, 18, 33, 48)], 9)))
    assert int(rv.next_pos.item()) == 201


EDGE = [
    # smallest head (D=16, one head, one layer), empty revisits and empty sequences, contiguous
    Workload(name="edge-d16", n_layers=1, n_kv_heads=1, head_dim=16, sections=(2, 3, 3),
             n_seqs=5, grids=((1, 3, 3),), selection="random", cache="contiguous",
             cur_pos=("uniform", 10, 60), extra=(0, 3, 0, 9)),
    # widest row (H*D = 8192: 512 threads per token), paged, two frames (t non-degenerate)
    Workload(name="edge-maxrow", n_layers=3, n_kv_heads=32, head_dim=256, sections=(40, 44, 44),
             n_seqs=2, grids=((2, 4, 6),), selection="random", cache="paged",
             cur_pos=("uniform", 500, 900), extra=(1, 2, 1, 40)),
    # odd sizes: D=48, 3 heads, 5 layers, block size 7, two grids, ragged everything
    Workload(name="edge-odd", n_layers=5, n_kv_heads=3, head_dim=48, sections=(8, 8, 8),
             n_seqs=4, grids=((3, 5, 5), (1, 4, 4)), selection="random", cache="paged",
             cur_pos=("uniform", 100, 40000), block_size=7, extra=(0, 3, 0, 37)),
    # many tokens over several tiles, many layer groups, large positions
    Workload(name="edge-long", n_layers=7, n_kv_heads=2, head_dim=64, sections=(8, 12, 12),
             n_seqs=3, grids=((4, 16, 16),), selection="random", cache="contiguous",
             cur_pos=("uniform", 20000, 2000000), extra=(1, 3, 100, 700)),
]


def test_one_tile_touching_64_revisits():
    """One-kernel path where a single CTA's tile (256 tokens at one thread per
    token: one KV head of head_dim 16) spans all 64 revisits of the batch, so
    that the CTA reduces 64 coordinate ranges at once (more range slots than
    it has threads); every output against the oracle."""
    import parity_util as pu
    wl = Workload(name="edge-manyrev", n_layers=2, n_kv_heads=1, head_dim=16, sections=(2, 3, 3),
                  n_seqs=4, grids=((2, 8, 8),), selection="random", cache="contiguous",
                  cur_pos=("uniform", 50, 5000), extra=(16, 16, 1, 4))
    batch = make_batch(wl, device=DEV, seed=9)
    assert batch.n_revisits == 64 and batch.total_k <= 256
    rv = pu.make_revisit(batch)
    assert _kernel_names(rv.run) == ["fused_kernel"]
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    pu.full_check(batch, rv)


@pytest.mark.parametrize("wl", EDGE, ids=[w.name for w in EDGE])
def test_edge_shapes(wl):
    import parity_util as pu
    batch = make_batch(wl, device=DEV, seed=5)
    rv = _run(batch)
    assert rv.status_value() == 0
    pu.full_check(batch, rv)


@pytest.mark.parametrize("mode", [O.MODE_ORIGINAL, O.MODE_UIR, O.MODE_LPA])
@pytest.mark.parametrize("name", ["tiny", "edge-odd"])
def test_other_modes(mode, name):
    import parity_util as pu
    wl = get(name) if name != "edge-odd" else EDGE[2]
    batch = make_batch(wl, device=DEV, seed=3)
    rv = _run(batch, mode=mode)
    assert rv.status_value() == 0
    pu.full_check(batch, rv, mode=mode)


def test_original_mode_is_position_bound_cache():
    """mode ORIGINAL reproduces RoPE(k_raw, p_m) at the stored coordinates."""
    import parity_util as pu
    batch = make_batch(get("qwen2vl-2b"), device=DEV)
    rv = _run(batch, mode=O.MODE_ORIGINAL)
    pl = pu.oracle_plan(batch, mode=O.MODE_ORIGINAL)
    coords = batch.coords.cpu().numpy()[pl["seq"], batch.idx.cpu().numpy()]
    assert np.array_equal(rv.pos.cpu().numpy(), coords.astype(np.float64))
    tokens = np.arange(batch.total_k)
    k_raw = pu.bits(pu.raw_rows(batch, batch.store_k, tokens, pl, range(28)))
    want = O.position_bound_keys(k_raw, coords, 128, batch.wl.sections, batch.wl.theta)
    got = pu.bits(pu.gather_cache(batch, batch.cache_k, tokens, pl, range(28)))
    assert pu.k_error(got, want, k_raw)["max_err"] <= pu.K_TOL


@pytest.mark.parametrize("name", ["tiny", "edge-odd"])
def test_degenerate_center_and_L(name):
    import parity_util as pu
    wl = get(name) if name != "edge-odd" else EDGE[2]
    for L, flags, deg in ((0, 0, "zero"), (5, 1, "center"), (2, 1, "center")):
        batch = make_batch(wl, device=DEV, seed=9)
        rv = _run(batch, L=L, flags=flags)
        pu.full_check(batch, rv, L=L, degenerate=deg)


def test_interleaved_layout():
    import parity_util as pu
    wl = Workload(name="il", n_layers=4, n_kv_heads=8, head_dim=128, sections=(24, 20, 20),
                  n_seqs=3, grids=((4, 8, 8),), selection="random", cache="paged",
                  cur_pos=("uniform", 8000, 30000), extra=(1, 3, 5, 120))
    batch = make_batch(wl, device=DEV, seed=13)
    rv = _run(batch, layout=O.LAYOUT_INTERLEAVED)
    pu.full_check(batch, rv, layout=O.LAYOUT_INTERLEAVED)


def test_rerun_and_split_calls_agree():
    """The call is re-runnable, and plan + apply equals the fused entry point."""
    import parity_util as pu
    batch = make_batch(get("qwen25vl-7b"), device=DEV)
    rv = _run(batch)
    k1 = batch.cache_k.clone(); v1 = batch.cache_v.clone()
    rv.run(); torch.cuda.synchronize()
    assert torch.equal(k1.view(torch.int16), batch.cache_k.view(torch.int16))
    batch.cache_k.view(torch.int16).fill_(-1); batch.cache_v.view(torch.int16).fill_(-1)
    rv.run_plan(); rv.run_apply(); torch.cuda.synchronize()
    assert torch.equal(k1.view(torch.int16), batch.cache_k.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), batch.cache_v.view(torch.int16))
    assert rv.status_value() == 0


def test_run_from_host_matches():
    import parity_util as pu
    batch = make_batch(get("qwen2vl-2b"), device=DEV)
    rv = pu.make_revisit(batch)
    st = rv.run_from_host()
    assert st == 0
    h = rv.host_inputs()
    pl = pu.oracle_plan(batch)
    assert np.array_equal(h["next_pos"].numpy(), pl["next_pos"])
    assert np.array_equal(h["cache_len_out"].numpy().astype(np.int64), pl["cache_len_out"])
    pu.full_check(batch, rv)


def test_store_raw_copies_bit_exact():
    import paper_2606_26631_gb300 as prcr
    wl = get("qwen25vl-7b")
    batch = make_batch(wl, device=DEV)
    store_k = torch.empty_like(batch.store_k).view(torch.int16).fill_(7).view(torch.bfloat16)
    store_v = torch.empty_like(batch.store_v).view(torch.int16).fill_(7).view(torch.bfloat16)
    coords = torch.zeros_like(batch.coords)
    cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta)
    desc = prcr.store_desc(store_k, store_v, coords)
    # fill in two pieces per sequence: layers [0, 11) tokens [0, 1000), then the rest
    for b in range(wl.n_seqs):
        for (l0, l1, m0, m1) in ((0, 11, 0, 1000), (11, 28, 0, 1000), (0, 28, 1000, wl.n_tokens)):
            prcr.store_raw(cfg, desc, b, l0, m0, batch.store_k[b, l0:l1, m0:m1],
                           batch.store_v[b, l0:l1, m0:m1],
                           batch.coords[b, m0:m1].contiguous() if l0 == 0 else None)
    torch.cuda.synchronize()
    assert torch.equal(store_k.view(torch.int16), batch.store_k.view(torch.int16))
    assert torch.equal(store_v.view(torch.int16), batch.store_v.view(torch.int16))
    assert torch.equal(coords, batch.coords)


# ----------------------------------------------------------------------------
# device-side error paths: status bits, no out-of-bounds writes, no trap
# ----------------------------------------------------------------------------
def test_bad_index_and_missing_block_and_capacity():
    import parity_util as pu
    wl = get("qwen25vl-7b")
    batch = make_batch(wl, device=DEV)
    pl = pu.oracle_plan(batch)
    idx = batch.idx.clone()
    bad_idx_tok = 5
    batch.idx[bad_idx_tok] = wl.n_tokens + 3  # out of range
    # unmap the block holding the last token of sequence 2
    b2_last = int(batch.rev_tok_off[int(batch.seq_rev_off[3])].item()) - 1
    s = int(pl["slot"][b2_last])
    batch.block_table[2, s // 16] = -1
    rv = _run(batch)
    st = rv.status_value()
    assert st & pu.prcr.ST_IDX_RANGE and st & pu.prcr.ST_NO_BLOCK
    assert not st & pu.prcr.ST_CSR
    unmapped = [j for j in range(batch.total_k)
                if pl["seq"][j] == 2 and pl["slot"][j] // 16 == s // 16]
    written = [j for j in range(batch.total_k) if j != bad_idx_tok and j not in unmapped]
    # the bad token's revisit gets its coordinate range from its valid tokens
    # only, so compare rows outside that revisit (revisit 0)
    r0_end = int(batch.rev_tok_off[1].item())
    assert bad_idx_tok < r0_end
    checked = [j for j in written if j >= r0_end]
    batch.idx.copy_(idx)
    pu.check_rows(batch, rv, pl, checked, range(wl.n_layers))
    pu.check_untouched(batch, pl, written=np.asarray(written))
    # capacity: a contiguous cache one slot too small for sequence 0
    wl2 = get("qwen2vl-2b")
    b2 = make_batch(wl2, device=DEV)
    pl2 = pu.oracle_plan(b2)
    cap = int(pl2["slot"].max())  # the last token's slot no longer fits
    ck = b2.cache_k[:, :, :cap].clone(); cv = b2.cache_v[:, :, :cap].clone()
    b2.cache_k, b2.cache_v = ck, cv
    rv2 = _run(b2)
    assert rv2.status_value() & pu.prcr.ST_CAPACITY
    good2 = np.arange(b2.total_k - 1)
    pu.check_rows(b2, rv2, pl2, good2, range(wl2.n_layers))
    pu.check_untouched(b2, pl2, written=good2)


def test_malformed_offsets_write_nothing():
    import parity_util as pu
    batch = make_batch(get("qwen25vl-7b"), device=DEV)
    batch.rev_tok_off[3] = batch.rev_tok_off[2] - 1  # not monotone
    rv = _run(batch)
    assert rv.status_value() & pu.prcr.ST_CSR
    for c in (batch.cache_k, batch.cache_v):
        assert bool((c.view(torch.int16) == -1).all().item())


def test_empty_batch():
    import paper_2606_26631_gb300 as prcr
    wl = Workload(name="empty", n_layers=2, n_kv_heads=2, head_dim=64, sections=(8, 12, 12),
                  n_seqs=3, grids=((1, 4, 4),), selection="random", cache="paged",
                  cur_pos=("fixed", 50), extra=(0, 0, 0, 0))
    batch = make_batch(wl, device=DEV)
    assert batch.total_k == 0
    import parity_util as pu
    rv = _run(batch)
    assert rv.status_value() == 0
    assert rv.next_pos.cpu().tolist() == [51, 51, 51]
    assert rv.cache_len_out.cpu().tolist() == batch.cache_len_in.cpu().tolist()
    for c in (batch.cache_k, batch.cache_v):
        assert bool((c.view(torch.int16) == -1).all().item())


# ----------------------------------------------------------------------------
# full-size workloads, the benchmark's launch configuration
# ----------------------------------------------------------------------------
@pytest.mark.slow
@pytest.mark.parametrize("name,seqs,layers", [("qwen3vl-8b", (0, 7, 15), (0, 17, 35)),
                                              ("stress", (0, 13, 31), (0, 18, 35))])
def test_full_size(name, seqs, layers):
    import parity_util as pu
    batch = make_batch(get(name), device=DEV)
    rv = pu.make_revisit(batch)
    rv.run_plan(); rv.run_apply()
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    pl = pu.oracle_plan(batch)
    pu.check_plan(rv, pl)
    tokens = np.nonzero(np.isin(pl["seq"], np.asarray(seqs)))[0]
    e = pu.check_rows(batch, rv, pl, tokens, layers)
    print(name, e)
    pu.check_untouched(batch, pl)


@pytest.mark.parametrize("name", ["tiny", "qwen25vl-7b"])
def test_graph_replay_matches(name):
    """The call captured in a CUDA graph (plan + PDL-launched rebind) and
    replayed gives the oracle's results."""
    import parity_util as pu
    batch = make_batch(get(name), device=DEV)
    rv = pu.make_revisit(batch)
    rv.run()  # warm-up outside capture (first-call set-up)
    torch.cuda.synchronize()
    batch.cache_k.view(torch.int16).fill_(-1)
    batch.cache_v.view(torch.int16).fill_(-1)
    rv.pos.zero_(); rv.slot.zero_(); rv.next_pos.zero_(); rv.cache_len_out.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        rv.run()
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    pu.full_check(batch, rv)


def _kernel_names(fn):
    """Names of this library's CUDA kernels that fn launches, as the profiler
    (CUPTI) records them."""
    from torch.profiler import ProfilerActivity, profile
    for _ in range(3):  # the first session of a process records no kernels
        with profile(activities=[ProfilerActivity.CPU, ProfilerActivity.CUDA]) as prof:
            fn()
            torch.cuda.synchronize()
        names = set()
        for e in prof.key_averages():
            if e.device_type.name == "CUDA":
                names.update(re.findall(r"\bprcr::.*?\b(\w+_kernel)\b", e.key))
        if names:
            return sorted(names)
    return []


SMALL = ["tiny", "qwen2vl-2b", "paper-8b-k32", "paper-8b-k128", "edge-d16", "edge-odd"]


def _small_wl(name):
    return {w.name: w for w in EDGE}.get(name) or get(name)


@pytest.mark.parametrize("mode", [O.MODE_PCR, O.MODE_ORIGINAL, O.MODE_UIR, O.MODE_LPA])
@pytest.mark.parametrize("name", SMALL)
def test_fused_path_matches_two_kernel_path(name, mode):
    """Small batches take the one-kernel path in prcr_rebind_inject; its
    results equal the plan + rebind kernels' bit for bit (prcr_plan followed
    by prcr_rebind_apply always runs the two kernels)."""
    import parity_util as pu
    batch = make_batch(_small_wl(name), device=DEV, seed=21)
    assert batch.total_k <= 2048 and batch.n_revisits <= 64
    pristine_k = batch.cache_k.clone(); pristine_v = batch.cache_v.clone()
    fused = pu.make_revisit(batch, mode=mode)
    assert _kernel_names(fused.run) == ["fused_kernel"]
    fk, fv = batch.cache_k.clone(), batch.cache_v.clone()
    batch.cache_k.copy_(pristine_k); batch.cache_v.copy_(pristine_v)
    two = pu.make_revisit(batch, mode=mode)
    two.run_plan(); two.run_apply()
    torch.cuda.synchronize()
    assert fused.status_value() == two.status_value() == 0
    assert torch.equal(fk.view(torch.int16), batch.cache_k.view(torch.int16))
    assert torch.equal(fv.view(torch.int16), batch.cache_v.view(torch.int16))
    assert torch.equal(fused.pos.view(torch.int64), two.pos.view(torch.int64))
    assert torch.equal(fused.slot, two.slot)
    assert torch.equal(fused.cache_len_out, two.cache_len_out)
    assert torch.equal(fused.next_pos, two.next_pos)


def test_large_batch_takes_two_kernels():
    """A batch past the fused path's limits runs the plan kernel, then the
    rebind + inject kernel."""
    import parity_util as pu
    batch = make_batch(get("qwen25vl-7b"), device=DEV)
    assert batch.total_k > 2048
    rv = pu.make_revisit(batch)
    assert _kernel_names(rv.run) == ["plan_kernel", "rebind_kernel"]
    assert rv.status_value() == 0


def test_malformed_offsets_small_batch_write_nothing():
    import parity_util as pu
    batch = make_batch(_small_wl("edge-odd"), device=DEV, seed=5)
    r = int(batch.rev_tok_off.numel()) - 1
    assert r >= 3 and batch.total_k <= 2048
    batch.rev_tok_off[2] = batch.rev_tok_off[3] + 1  # not monotone
    rv = _run(batch)
    assert rv.status_value() & pu.prcr.ST_CSR
    for c in (batch.cache_k, batch.cache_v):
        assert bool((c.view(torch.int16) == -1).all().item())


def test_bad_index_small_batch():
    """Fused path: an out-of-range index is reported and its rows skipped;
    the other revisits' rows are right."""
    import parity_util as pu
    batch = make_batch(get("paper-8b-k128"), device=DEV)
    pl = pu.oracle_plan(batch)
    batch.idx[7] = batch.wl.n_tokens + 1
    rv = _run(batch)
    assert rv.status_value() & pu.prcr.ST_IDX_RANGE
    written = np.array([j for j in range(batch.total_k) if j != 7])
    pu.check_untouched(batch, pl, written=written)


def test_position_beyond_angle_range_is_flagged():
    """Text positions of 2^31 and more are beyond the fixed-point angle
    reduction: the call sets PRCR_ST_POS_RANGE and skips those tokens' rows
    (they keep the canary), while the other sequences of the same batch get
    the oracle's positions and rows. One-kernel path (2 sequences, ~1000
    tokens) and two-kernel path (8 sequences); a position well inside the
    range sets nothing."""
    import dataclasses
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    for n_seqs, bad_seqs in ((2, [1]), (8, [0, 5])):
        wl = dataclasses.replace(get("qwen25vl-7b"), n_seqs=n_seqs, n_layers=3)
        batch = make_batch(wl, device=DEV, seed=4)
        for b in bad_seqs:
            batch.p_txt[b] = 2 ** 31 + 100 + b
        pl = pu.oracle_plan(batch)
        rv = pu.make_revisit(batch)
        launched = _kernel_names(rv.run)  # runs the call once
        assert launched == (["fused_kernel"] if n_seqs == 2 else ["plan_kernel", "rebind_kernel"]), launched
        assert rv.status_value() == prcr.ST_POS_RANGE, (n_seqs, rv.status_value())
        good = np.nonzero(~np.isin(pl["seq"], bad_seqs))[0]
        assert 0 < len(good) < batch.total_k
        got_pos = rv.pos.cpu().numpy()
        assert np.array_equal(got_pos[good].view(np.int64), pl["pos"][good].view(np.int64))
        assert np.array_equal(rv.slot.cpu().numpy()[good].astype(np.int64), pl["slot"][good])
        assert np.array_equal(rv.cache_len_out.cpu().numpy().astype(np.int64), pl["cache_len_out"])
        assert np.array_equal(rv.next_pos.cpu().numpy(), pl["next_pos"])
        pu.check_rows(batch, rv, pl, good, range(wl.n_layers))
        pu.check_untouched(batch, pl, written=good)
    for name in ("tiny", "qwen25vl-7b"):
        batch = make_batch(get(name), device=DEV, seed=4)
        batch.p_txt.fill_(2 ** 31 - 2 ** 20)
        rv = _run(batch)
        assert rv.status_value() == 0, name
