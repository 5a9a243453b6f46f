"""JSON manifest of the revisits a workload's batch selects (the record of
what a benchmark line timed).

For each sequence: its text position and existing cache length; for each of
its revisits, in call order: the number of tokens K, the rectangles the
generator drew (grid, first frame, frames, first row, rows, first column,
columns; empty for scattered tokens), the first and last token ids and the
sha256 of the int32 id list. Everything comes from the seeded generator in
``workloads.gen`` (selections: PCG64 seed + 1; text positions: seed + 2), on
the host, without building the store or the cache; nothing here computes any
part of the method.

    python -m workloads.manifest            # rewrite workloads/manifests/*_seed0.json
    python -m workloads.manifest --check    # compare them with a fresh draw
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import sys

import numpy as np

from .configs import ALL, Workload
from .gen import selections, text_positions

HERE = os.path.dirname(os.path.abspath(__file__))
MANIFEST_DIR = os.path.join(HERE, "manifests")


def manifest(wl: Workload, seed: int = 0) -> dict:
    rng_sel = np.random.Generator(np.random.PCG64(seed + 1))
    rng_pos = np.random.Generator(np.random.PCG64(seed + 2))
    rects = []
    sels = selections(wl, rng_sel, rects)
    p_txt = text_positions(wl, rng_pos)
    seqs = []
    total = 0
    for b, revs in enumerate(sels):
        out = []
        for ids, rc in zip(revs, rects[b]):
            ids = np.ascontiguousarray(ids, dtype=np.int32)
            out.append(dict(K=int(ids.size), rects=[list(map(int, r)) for r in rc],
                            first_id=int(ids[0]) if ids.size else None,
                            last_id=int(ids[-1]) if ids.size else None,
                            ids_sha256=hashlib.sha256(ids.tobytes()).hexdigest()))
            total += int(ids.size)
        seqs.append(dict(seq=b, p_txt=int(p_txt[b]), cache_len_in=int(p_txt[b]) + 1, revisits=out))
    return dict(workload=wl.name, seed=seed,
                decoder=dict(n_layers=wl.n_layers, n_kv_heads=wl.n_kv_heads,
                             head_dim=wl.head_dim, sections=list(wl.sections), theta=wl.theta),
                grids=[list(g) for g in wl.grids], selection=wl.selection, cache=wl.cache,
                block_size=wl.block_size, L=wl.L, n_seqs=wl.n_seqs,
                n_revisits=sum(len(s["revisits"]) for s in seqs), total_k=total,
                rect_fields=["grid", "frame0", "frames", "row0", "rows", "col0", "cols"],
                sequences=seqs)


def dumps(m: dict) -> str:
    return json.dumps(m, indent=1, sort_keys=True) + "\n"


def sha256_of(text: str) -> str:
    return hashlib.sha256(text.encode()).hexdigest()


def path_for(name: str, seed: int = 0) -> str:
    return os.path.join(MANIFEST_DIR, f"{name}_seed{seed}.json")


def main(argv=None) -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--check", action="store_true")
    args = ap.parse_args(argv)
    os.makedirs(MANIFEST_DIR, exist_ok=True)
    bad = 0
    for name, wl in sorted(ALL.items()):
        text = dumps(manifest(wl, 0))
        p = path_for(name, 0)
        if args.check:
            ok = os.path.exists(p) and open(p).read() == text
            bad += not ok
            print(f"{name}: {'ok' if ok else 'DIFFERS'}")
        else:
            with open(p, "w") as f:
                f.write(text)
            print(f"{p}: {sha256_of(text)[:16]}")
    return 1 if bad else 0


if __name__ == "__main__":
    sys.exit(main())
