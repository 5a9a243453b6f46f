"""The library keeps no per-call state on the device and only read-mostly
caches on the host (turn rates per (theta, head_dim), occupancy per kernel
shape, both behind a mutex), so independent calls may overlap: on several
CUDA streams, and from several host threads at once. Both must give exactly
the results of the same calls made one after another."""
import threading

import pytest
import torch

from workloads import Workload, get, make_batch

pytestmark = pytest.mark.gpu

DEV = "cuda:0"

# different shapes, cache kinds, paths (one-kernel and two-kernel) and rotary
# bases, so the host caches see distinct entries
SHAPES = [
    get("qwen2vl-2b"),
    get("qwen25vl-7b"),
    Workload(name="odd", n_layers=5, n_kv_heads=3, head_dim=48, sections=(8, 8, 8), n_seqs=4,
             grids=((3, 5, 5), (1, 4, 4)), selection="random", cache="paged",
             cur_pos=("uniform", 100, 40000), block_size=7, extra=(0, 3, 0, 37), theta=5e5),
    Workload(name="tiny-b", n_layers=2, n_kv_heads=2, head_dim=64, sections=(8, 12, 12), n_seqs=1,
             grids=((1, 8, 8),), selection="rect4x4", cache="contiguous", cur_pos=("fixed", 200),
             theta=2e4),
]


def _fresh():
    """One batch per shape with its Revisit, and the pristine caches."""
    import parity_util as pu
    out = []
    for i, wl in enumerate(SHAPES):
        batch = make_batch(wl, device=DEV, seed=40 + i)
        out.append((batch, pu.make_revisit(batch), batch.cache_k.clone(), batch.cache_v.clone()))
    return out


def _results(items):
    return [(b.cache_k.view(torch.int16).clone(), b.cache_v.view(torch.int16).clone(),
             rv.pos.clone(), rv.slot.clone(), rv.next_pos.clone(), rv.cache_len_out.clone(),
             rv.status_value()) for b, rv, _, _ in items]


def _reset(items):
    for b, rv, k0, v0 in items:
        b.cache_k.copy_(k0)
        b.cache_v.copy_(v0)
        rv.status.zero_()
    torch.cuda.synchronize()


def _same(x, y):
    for a, b in zip(x, y):
        for u, v in zip(a[:6], b[:6]):
            assert torch.equal(u, v)
        assert a[6] == b[6] == 0


def test_streams_overlap():
    items = _fresh()
    for _, rv, _, _ in items:
        rv.run()
    torch.cuda.synchronize()
    want = _results(items)
    _reset(items)
    streams = [torch.cuda.Stream() for _ in items]
    for _ in range(3):  # re-running is harmless: the call is a pure function of its inputs
        for (_, rv, _, _), s in zip(items, streams):
            rv.run(stream=s)
    torch.cuda.synchronize()
    _same(want, _results(items))


def test_host_threads():
    items = _fresh()
    for _, rv, _, _ in items:
        rv.run()
    torch.cuda.synchronize()
    want = _results(items)
    _reset(items)
    errors = []

    def work(rv):
        try:
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                for _ in range(5):
                    rv.run(stream=s)
            s.synchronize()
        except Exception as e:  # pragma: no cover - reported below
            errors.append(e)

    threads = [threading.Thread(target=work, args=(rv,)) for _, rv, _, _ in items]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    torch.cuda.synchronize()
    _same(want, _results(items))
