"""Helpers for GPU-vs-oracle parity checks (used by the -m gpu tests, smoke()
and bench.py's self-check).

The GPU side always goes through the C ABI (paper_2606_26631_gb300). The
expected side is the CPU oracle (oracle/prcr_oracle.py) fed with the same
seeded inputs. Bars:
  * positions (float64), slots, cache_len_out, next_pos, V rows: bit-exact;
  * K rows: err = |g - o| / max(|o|, 2^-7 * rho) <= 8e-3 per element, where
    rho is the norm of the element's rotation pair (invariant under the
    rotation); 8e-3 is about one bf16 ulp (2^-7), the output rounding alone
    contributing at most half of it;
  * every cache row the call must not touch still holds the canary pattern.
"""
from __future__ import annotations

from typing import Iterable, Optional

import numpy as np
import torch

import paper_2606_26631_gb300 as prcr
from oracle import prcr_oracle as O
from workloads import CANARY_BITS, Batch

K_TOL = 8e-3
NEAR_ZERO = 2.0 ** -7


def make_revisit(batch: Batch, mode=O.MODE_PCR, L: Optional[int] = None, flags=0,
                 layout=O.LAYOUT_SECTIONED) -> prcr.Revisit:
    wl = batch.wl
    cfg = prcr.rope_cfg(wl.n_layers, wl.n_kv_heads, wl.head_dim, wl.sections, wl.theta, layout)
    return prcr.Revisit(cfg, batch.store_k, batch.store_v, batch.coords, batch.cache_k,
                        batch.cache_v, batch.block_table, batch.seq_rev_off, batch.rev_tok_off,
                        batch.idx, batch.p_txt, batch.cache_len_in, mode=mode,
                        L=wl.L if L is None else L, flags=flags)


def oracle_plan(batch: Batch, mode=O.MODE_PCR, L: Optional[int] = None, degenerate="zero"):
    wl = batch.wl
    return O.plan(batch.coords.cpu().numpy(), batch.seq_rev_off.cpu().numpy(),
                  batch.rev_tok_off.cpu().numpy(), batch.idx.cpu().numpy(),
                  batch.p_txt.cpu().numpy(), batch.cache_len_in.cpu().numpy(),
                  wl.L if L is None else L, mode, degenerate)


def _rows_of(batch: Batch, slots: np.ndarray, seqs: np.ndarray):
    """Cache row coordinates of (seq, slot): (b, s) contiguous, (blk, off) paged."""
    if not batch.paged:
        return seqs, slots
    bt = batch.block_table.cpu().numpy()
    bs = batch.wl.block_size
    blk = bt[seqs, slots // bs]
    return blk.astype(np.int64), (slots % bs).astype(np.int64)


def gather_cache(batch: Batch, which: torch.Tensor, tokens: np.ndarray, pl, layers) -> torch.Tensor:
    """GPU cache rows of the given tokens (at the oracle's slots): [n, len(layers), H, D]."""
    a, b = _rows_of(batch, pl["slot"][tokens], pl["seq"][tokens])
    a = torch.as_tensor(a, device=which.device)
    b = torch.as_tensor(b, device=which.device)
    lay = torch.as_tensor(list(layers), device=which.device)
    if not batch.paged:
        return which[a[:, None], lay[None, :], b[:, None]]
    return which[lay[None, :], a[:, None], b[:, None]]


def raw_rows(batch: Batch, store: torch.Tensor, tokens: np.ndarray, pl, layers) -> torch.Tensor:
    """Raw store rows of the given tokens: [n, len(layers), H, D] (input data)."""
    dev = store.device
    seq = torch.as_tensor(pl["seq"][tokens], device=dev)
    m = batch.idx[torch.as_tensor(tokens, device=dev)].long()
    lay = torch.as_tensor(list(layers), device=dev)
    return store[seq[:, None], lay[None, :], m[:, None]]


def bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy()


def k_error(got_bits: np.ndarray, want: np.ndarray, raw_bits: np.ndarray) -> dict:
    g = O.bf16_bits_to_f64(got_bits)
    rho = O.pair_norms(raw_bits)
    diff = np.abs(g - want)
    den = np.maximum(np.abs(want), NEAR_ZERO * rho)
    err = np.zeros_like(diff)
    nz = den > 0
    err[nz] = diff[nz] / den[nz]
    err[~nz & (diff > 0)] = np.inf
    sig = (np.abs(want) >= NEAR_ZERO * rho) & (want != 0)
    rel = np.zeros_like(diff)
    rel[sig] = diff[sig] / np.abs(want[sig])
    return dict(max_err=float(err.max()) if err.size else 0.0,
                max_rel=float(rel.max()) if rel.size else 0.0,
                n_rne=int(np.sum(g == O.f64_to_bf16_rne(want))), n=int(g.size))


def merge(a: dict, b: dict) -> dict:
    return dict(max_err=max(a["max_err"], b["max_err"]), max_rel=max(a["max_rel"], b["max_rel"]),
                n_rne=a["n_rne"] + b["n_rne"], n=a["n"] + b["n"])


def check_plan(rv: prcr.Revisit, pl) -> None:
    got_pos = rv.pos.cpu().numpy()
    assert np.array_equal(got_pos.view(np.int64), pl["pos"].view(np.int64)), "positions differ"
    assert np.array_equal(rv.slot.cpu().numpy().astype(np.int64), pl["slot"]), "slots differ"
    assert np.array_equal(rv.cache_len_out.cpu().numpy().astype(np.int64), pl["cache_len_out"])
    assert np.array_equal(rv.next_pos.cpu().numpy(), pl["next_pos"])


def check_rows(batch: Batch, rv: prcr.Revisit, pl, tokens: Iterable[int], layers: Iterable[int],
               layout=O.LAYOUT_SECTIONED, chunk_elems: int = 1 << 24) -> dict:
    """K within K_TOL and V bit-exact for the given tokens x layers."""
    tokens = np.asarray(list(tokens), dtype=np.int64)
    layers = list(layers)
    stats = dict(max_err=0.0, max_rel=0.0, n_rne=0, n=0)
    if tokens.size == 0 or not layers:
        return stats
    wl = batch.wl
    row = wl.n_kv_heads * wl.head_dim
    tok_chunk = max(1, chunk_elems // (row * len(layers)))
    for t0 in range(0, tokens.size, tok_chunk):
        tk = tokens[t0:t0 + tok_chunk]
        k_raw = bits(raw_rows(batch, batch.store_k, tk, pl, layers))
        v_raw = bits(raw_rows(batch, batch.store_v, tk, pl, layers))
        k_got = bits(gather_cache(batch, batch.cache_k, tk, pl, layers))
        v_got = bits(gather_cache(batch, batch.cache_v, tk, pl, layers))
        assert np.array_equal(v_got, v_raw), "V rows differ"
        want = O.rebind_keys(k_raw, pl["pos"][tk], wl.head_dim, wl.sections, wl.theta, layout)
        stats = merge(stats, k_error(k_got, want, k_raw))
    assert stats["max_err"] <= K_TOL, f"K error {stats}"
    return stats


def check_untouched(batch: Batch, pl, written: Optional[np.ndarray] = None) -> None:
    """Rows the call must not write still hold the canary; written rows do not."""
    tokens = np.arange(len(pl["slot"])) if written is None else written
    a, b = _rows_of(batch, pl["slot"][tokens], pl["seq"][tokens])
    row = batch.wl.n_kv_heads * batch.wl.head_dim
    for cache in (batch.cache_k, batch.cache_v):
        c16 = cache.view(torch.int16)
        nL = batch.wl.n_layers
        for l in range(nL):
            lay = c16[:, l] if not batch.paged else c16[l]
            total = lay.numel()
            n_canary = int((lay == CANARY_BITS).sum().item())
            assert n_canary == total - len(tokens) * row, (l, n_canary, total, len(tokens))
        # written rows carry data (a rotated or copied finite value is never 0xFFFF)
        if len(tokens):
            aa = torch.as_tensor(a, device=cache.device)
            bb = torch.as_tensor(b, device=cache.device)
            if not batch.paged:
                w = c16[aa, :, bb]
            else:
                w = c16[:, aa, bb]
            assert not bool((w == CANARY_BITS).any().item())


def full_check(batch: Batch, rv: prcr.Revisit, mode=O.MODE_PCR, L=None, degenerate="zero",
               layout=O.LAYOUT_SECTIONED) -> dict:
    """Complete comparison: plan, every token x layer row, untouched rows."""
    pl = oracle_plan(batch, mode, L, degenerate)
    check_plan(rv, pl)
    e = check_rows(batch, rv, pl, range(batch.total_k), range(batch.wl.n_layers), layout)
    check_untouched(batch, pl)
    return e


def full_oracle_call(batch: Batch, mode=O.MODE_PCR, L=None, degenerate="zero",
                     layout=O.LAYOUT_SECTIONED):
    """The oracle's whole Algorithm 1 (including its own gather) on host copies."""
    wl = batch.wl
    return O.rebind_inject(bits(batch.store_k), bits(batch.store_v), batch.coords.cpu().numpy(),
                           batch.seq_rev_off.cpu().numpy(), batch.rev_tok_off.cpu().numpy(),
                           batch.idx.cpu().numpy(), batch.p_txt.cpu().numpy(),
                           batch.cache_len_in.cpu().numpy(), wl.head_dim, wl.sections, wl.theta,
                           wl.L if L is None else L, mode, degenerate, layout)
