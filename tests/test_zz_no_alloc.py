"""GPU test of prcr_rebind_inject_static, the allocation-free form of the call.

Some callers cannot allocate device memory themselves (a plugin whose host
framework owns all device memory through its own pool, or a decode loop where
cudaMalloc/cudaFree, which may synchronise the device, are not allowed). For
them the library keeps the per-token plan in its own fixed device array
instead of a caller workspace. This test calls that entry point through the C
ABI twice in a row, on two different workloads, and checks each result
against the workspace-based prcr_rebind_inject on the same inputs: positions,
slots, lengths and V bit for bit, K within the tolerance the parity tests use,
every row neither call should write left untouched. Both launch forms are
covered: the plan kernel, which keeps its per-token plan in the array, and
the one-kernel form small batches take. It also checks that device memory in
use does not change across static calls, that a batch above the array's
capacity is refused before anything runs, and that a malformed call gets the
same error code as prcr_rebind_inject.

The file name sorts last so that a run stopping at the first failure has run
every other test before this one; it passes alone in a fresh process too.
"""
import ctypes as C
import dataclasses

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _compare_with_workspace_call(wl, plan_kernel=True):
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    from workloads import make_batch

    batch = make_batch(wl, device=DEV)
    # batches above 2048 tokens use the plan kernel and its per-token scratch;
    # smaller ones the one-kernel form
    assert (batch.total_k > 2048) == plan_kernel
    pristine_k = batch.cache_k.clone()
    pristine_v = batch.cache_v.clone()

    ref = pu.make_revisit(batch)  # caller-provided workspace
    ref.run()
    torch.cuda.synchronize()

    other = dataclasses.replace(batch, cache_k=pristine_k, cache_v=pristine_v)
    st = pu.make_revisit(other)
    prcr.rebind_inject_static(st.cfg, st.store, st.cache, st.batch, st.out, st.mode, st.L, st.flags)
    torch.cuda.synchronize()

    assert ref.status_value() == 0 and st.status_value() == 0
    assert torch.equal(st.pos.view(torch.int64), ref.pos.view(torch.int64))
    assert torch.equal(st.slot, ref.slot)
    assert torch.equal(st.cache_len_out, ref.cache_len_out)
    assert torch.equal(st.next_pos, ref.next_pos)
    assert torch.equal(other.cache_v.view(torch.int16), batch.cache_v.view(torch.int16))

    pl = pu.oracle_plan(batch)
    tokens = np.arange(batch.total_k)
    layers = range(batch.wl.n_layers)
    k_raw = pu.bits(pu.raw_rows(batch, batch.store_k, tokens, pl, layers))
    k_ref = pu.bits(pu.gather_cache(batch, batch.cache_k, tokens, pl, layers))
    k_st = pu.bits(pu.gather_cache(other, other.cache_k, tokens, pl, layers))
    from oracle import prcr_oracle as O
    e = pu.k_error(k_st, O.bf16_bits_to_f64(k_ref), k_raw)
    assert e["max_err"] <= pu.K_TOL, e
    pu.check_untouched(other, pl)
    return st


def test_static_scratch_two_calls_in_a_row():
    from workloads import get
    first = _compare_with_workspace_call(get("qwen25vl-7b"))  # paged, 4093 tokens
    second = _compare_with_workspace_call(                    # contiguous, 12 x 259 tokens
        dataclasses.replace(get("qwen2vl-2b"), n_seqs=12))
    assert first.batch.total_k != second.batch.total_k


def test_static_small_batches_two_calls_in_a_row():
    import dataclasses as dc
    from workloads import get
    first = _compare_with_workspace_call(get("paper-8b-k32"), plan_kernel=False)
    second = _compare_with_workspace_call(dc.replace(get("qwen25vl-7b"), n_seqs=2, n_layers=4),
                                          plan_kernel=False)
    assert first.batch.total_k != second.batch.total_k


def test_static_calls_allocate_no_device_memory():
    """After a first call of each launch form (which may load the library's
    module and looks up the array's address), further calls leave the device
    memory in use unchanged, as torch's allocator and the driver see it."""
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    from workloads import get, make_batch

    rvs = []
    for name in ("qwen25vl-7b", "paper-8b-k32"):
        rv = pu.make_revisit(make_batch(get(name), device=DEV))
        rvs.append(rv)
    for rv in rvs:  # warm-up: first call of each form
        prcr.rebind_inject_static(rv.cfg, rv.store, rv.cache, rv.batch, rv.out, rv.mode, rv.L,
                                  rv.flags)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    alloc0 = torch.cuda.memory_stats().get("allocated_bytes.all.current", 0)
    reserved0 = torch.cuda.memory_reserved()
    for _ in range(3):
        for rv in rvs:
            prcr.rebind_inject_static(rv.cfg, rv.store, rv.cache, rv.batch, rv.out, rv.mode, rv.L,
                                      rv.flags)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert torch.cuda.memory_stats().get("allocated_bytes.all.current", 0) == alloc0
    assert torch.cuda.memory_reserved() == reserved0
    for rv in rvs:
        assert rv.status_value() == 0


def test_static_scratch_refuses_oversized_batch():
    import paper_2606_26631_gb300 as prcr
    import parity_util as pu
    from paper_2606_26631_gb300 import _binding as B
    from workloads import get, make_batch

    batch = make_batch(get("tiny"), device=DEV)
    rv = pu.make_revisit(batch)
    big = B.RevisitBatch.from_buffer_copy(rv.batch)
    big.total_k = B.STATIC_MAX_TOKENS + 1
    rc = prcr.lib().prcr_rebind_inject_static(C.byref(rv.cfg), C.byref(rv.store),
                                              C.byref(rv.cache), C.byref(big), C.byref(rv.out),
                                              0, 2, 0, None)
    assert rc == B.EWORKSPACE
    # a malformed call is refused with prcr_rebind_inject's code, whatever its size
    for mode in (7, -1):
        rc = prcr.lib().prcr_rebind_inject_static(C.byref(rv.cfg), C.byref(rv.store),
                                                  C.byref(rv.cache), C.byref(big), C.byref(rv.out),
                                                  mode, 2, 0, None)
        assert rc == B.EINVAL
    torch.cuda.synchronize()
    assert rv.status_value() == 0
    assert bool((batch.cache_k.view(torch.int16) == -1).all().item())
