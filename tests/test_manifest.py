"""The committed selection manifests (workloads/manifests/) describe exactly
the revisits the seeded workloads draw: each file equals a fresh draw, and for
the workloads small enough to build here the manifest's K values, token-id
hashes, text positions and cache lengths match the batch make_batch returns
(the batch bench.py and the parity tests use)."""
import hashlib
import json

import numpy as np
import pytest

from workloads import ALL, get, make_batch
from workloads import manifest as MF


@pytest.mark.parametrize("name", sorted(ALL))
def test_committed_manifest_is_a_fresh_draw(name):
    with open(MF.path_for(name, 0)) as f:
        assert f.read() == MF.dumps(MF.manifest(get(name), 0))


@pytest.mark.parametrize("name", ["tiny", "qwen2vl-2b", "qwen25vl-7b", "paper-8b-k32", "paper-8b-k128"])
def test_manifest_matches_the_batch(name):
    wl = get(name)
    m = json.loads(MF.dumps(MF.manifest(wl, 0)))
    batch = make_batch(wl, device="cpu", seed=0, store=False)
    sro = batch.seq_rev_off.numpy()
    rto = batch.rev_tok_off.numpy()
    idx = batch.idx.numpy().astype(np.int32)
    assert m["n_seqs"] == wl.n_seqs and m["n_revisits"] == batch.n_revisits
    assert m["total_k"] == batch.total_k
    for b, seq in enumerate(m["sequences"]):
        assert seq["p_txt"] == int(batch.p_txt[b]) and seq["cache_len_in"] == int(batch.cache_len_in[b])
        revs = list(range(sro[b], sro[b + 1]))
        assert len(revs) == len(seq["revisits"])
        for r, rec in zip(revs, seq["revisits"]):
            ids = np.ascontiguousarray(idx[rto[r]:rto[r + 1]])
            assert rec["K"] == ids.size
            assert rec["ids_sha256"] == hashlib.sha256(ids.tobytes()).hexdigest()
            # the rectangles as drawn cover exactly the revisit's tokens
            if rec["rects"]:
                assert sum(r_[2] * r_[4] * r_[6] for r_ in rec["rects"]) == ids.size
