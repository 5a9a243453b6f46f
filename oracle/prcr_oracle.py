"""Plain CPU oracle for PRCR's visual-revisit path (test infrastructure).

This module is test infrastructure. Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline leg (and its ``--impl reference`` arm) may
import it. The library path never calls it, and it shares no code with the
CUDA path: it is written from the paper's equations alone, in float64, with
positions kept as exact rationals until the single final rounding.

What it computes (paper sections / equations):

* Gather of the selected raw memory, M_tau = M[I_tau]            (Sec. 3.1, Eq. 7 "selected_raw_kv")
* Per-axis coordinate range over the selected set                (Sec. 3.2, Eq. "selected_coord_range")
* Normalised relative coordinate u                               (Sec. 3.2, Eq. "normalized_coord")
* PCR re-anchoring into (p_txt - L, p_txt + 1)                   (Sec. 3.2, Eq. "image_range_fractional_reinsert")
* Key rebinding with rotary embedding, values reused unchanged   (Sec. 3.3, Eq. "cache_reconstruction")
* Concatenation onto the existing decoder cache                  (Sec. 3.3, Eq. "active_cache")
* Next text position p_txt + 1                                   (Sec. 3.2 and 3.3, before Eq. "decode_with_active_cache")
* The position-bound historical key RoPE(k_raw, p_m)             (Sec. 2.3, Eq. "historical_position_bound_kv")
* Prefill capture: raw rows kept + position-bound cache rows       (Sec. 3.1, Eq. "raw_kv", "global_raw_memory")
* First decode step over the active cache                         (Sec. 3.3, Eq. "decode_with_active_cache")
* Attention-driven selection of the revisited set I_tau            (Sec. 2.1, Eq. 3; reading below)

Readings taken where the paper is silent (each is a named choice below):

* Three axes (t, h, w): the per-axis rule of Sec. 3.2 is applied to t as well
  as h and w, and a text position p is the triple (p, p, p).
* Degenerate axis (max == min, e.g. t inside one image): u = 0 by default
  ("zero"), or u = 1/2 ("center").
* K in Eq. "image_range_fractional_reinsert" is |I_tau| of that revisit.
* Rotary convention: rotate-half pairs (i, i + D/2) with inverse frequency
  theta^(-2i/D); sectioned M-RoPE gives the first s_t pairs to t, the next
  s_h to h, the rest to w. The interleaved band layout gives pair i to h when
  i % 3 == 1 and i < 3 s_h, to w when i % 3 == 2 and i < 3 s_w, else to t.
* Several revisits of one sequence in one call are reassigned independently
  (own range, own K) against the same p_txt; their tokens are appended in
  call order.
* UIR (Sec. 3.2, compared in Table 2; its formula is not printed): the j-th of
  K entries of a revisit goes to p_txt + j / (K + 1), next text position
  p_txt + 1.
* LPA (Sec. 3.2, Table 2; formula not printed): the r-th token appended to a
  sequence in this call goes to p_txt + r (r = 1, 2, ...) on all axes, and the
  next text position becomes p_txt + K_seq + 1.
* Attention-driven selection (Sec. 2.1 names it, its formula is outside the
  paper): the relevance of visual token m is the trigger query's attention
  on m at one layer, softmax over the M visual tokens' position-bound keys
  RoPE(k_raw, p_m), averaged over the query heads; the K most relevant tokens
  are selected (ties to the lower index) and listed in ascending token order.
  Second reading (``ads_relevance_cached``): the same attention computed
  over the keys the decoder's position-bound cache holds for the visual
  tokens (RoPE(k_raw, p_m) as stored, e.g. in bf16), only the query rotated.

Every function here is pinned in tests/test_oracle_pins.py against facts
from outside this module (no function is "parity unpinned"):

* coord_range, normalized_coord, pcr_position, reassign_revisit: hand-worked
  4x4 and 2x2 rectangles (tests/golden), closed forms of the PCR rule, the
  centre reading, the other position rules (pin_worked_rect*,
  pin_pcr_closed_forms, pin_degenerate_center, pin_other_modes)
* next_text_pos, plan: pin_worked_rect4x4, pin_other_modes,
  pin_plan_slots_and_continuity
* inv_freq, pair_axes, angles, rope, rebind_keys: textbook rotary values and
  complex-number RoPE, band membership, norm preservation, R(a)R(b) = R(a+b),
  the relative-offset logit identity (pin_rope_closed_forms,
  pin_mrope_equal_axes_is_textbook, pin_mrope_sections, pin_rope_invariants)
* bf16_bits_to_f64, f64_to_bf16_rne: pin_bf16_helpers
* rebind_inject, position_bound_keys, prefill_capture: a pure-Python brute
  force on a 2x2 region, the ORIGINAL rule against Eq.
  "historical_position_bound_kv" (pin_brute_force_2x2,
  pin_original_mode_is_position_bound_cache, pin_prefill_capture)
* decode_attention: a direct softmax and the relative-offset identity
  (pin_decode_attention)
* ads_relevance, ads_relevance_cached, ads_select: pin_ads, pin_ads_cached
* pair_norms: hand-worked rows (tests/golden/pair_norms.txt) and the norm
  kept by any rotation (pin_pair_norms)

Planted mistakes in each of them are caught by some pin
(test_planted_mistakes).
"""
from __future__ import annotations

from fractions import Fraction
from typing import Dict, List, Sequence

import numpy as np

MODE_PCR = 0
MODE_ORIGINAL = 1
MODE_UIR = 2
MODE_LPA = 3

LAYOUT_SECTIONED = 0
LAYOUT_INTERLEAVED = 1

AXES = ("t", "h", "w")


# ----------------------------------------------------------------------------
# Position reassignment (Sec. 3.2)
# ----------------------------------------------------------------------------
def coord_range(sel_coords: Sequence[Sequence[int]]):
    """Eq. "selected_coord_range": per-axis minimum and maximum over I_tau."""
    lo = [min(int(c[a]) for c in sel_coords) for a in range(3)]
    hi = [max(int(c[a]) for c in sel_coords) for a in range(3)]
    return lo, hi


def normalized_coord(c: int, lo: int, hi: int, degenerate: str = "zero") -> Fraction:
    """Eq. "normalized_coord": u = (p_m - p_min) / (p_max - p_min).

    The paper defines u only for p_max > p_min; for a degenerate axis the
    reading is u = 0 ("zero") or u = 1/2 ("center")."""
    if hi > lo:
        return Fraction(int(c) - lo, hi - lo)
    if degenerate == "zero":
        return Fraction(0)
    if degenerate == "center":
        return Fraction(1, 2)
    raise ValueError(degenerate)


def pcr_position(u: Fraction, K: int, p_txt: int, L: int) -> Fraction:
    """Eq. "image_range_fractional_reinsert":
    p_hat = (p_txt - L) + (L + 1) * (1 + (K - 1) u) / (K + 1)."""
    return Fraction(p_txt - L) + Fraction(L + 1) * (1 + (K - 1) * u) / (K + 1)


def reassign_revisit(sel_coords, p_txt: int, L: int, mode: int = MODE_PCR,
                     degenerate: str = "zero", seq_rank0: int = 0) -> List[List[Fraction]]:
    """Reassigned (t, h, w) position of every token of one revisit, exact.

    ``sel_coords`` lists the stored original coordinates of the K selected
    tokens in call order; ``seq_rank0`` is how many tokens of the same
    sequence precede this revisit in the call (used by LPA only)."""
    K = len(sel_coords)
    if K == 0:
        return []
    if mode == MODE_PCR:
        lo, hi = coord_range(sel_coords)
        return [[pcr_position(normalized_coord(c[a], lo[a], hi[a], degenerate), K, p_txt, L)
                 for a in range(3)] for c in sel_coords]
    if mode == MODE_ORIGINAL:
        return [[Fraction(int(c[a])) for a in range(3)] for c in sel_coords]
    if mode == MODE_UIR:
        return [[Fraction(p_txt) + Fraction(j + 1, K + 1)] * 3 for j in range(K)]
    if mode == MODE_LPA:
        return [[Fraction(p_txt + seq_rank0 + j + 1)] * 3 for j in range(K)]
    raise ValueError(mode)


def next_text_pos(p_txt: int, k_seq: int, mode: int = MODE_PCR) -> int:
    """Next text position after the revisit: p_txt + 1 (Sec. 3.2, Sec. 3.3);
    LPA shifts it past the appended entries."""
    if mode == MODE_LPA:
        return p_txt + k_seq + 1
    return p_txt + 1


def plan(coords, seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in, L: int,
         mode: int = MODE_PCR, degenerate: str = "zero") -> Dict[str, object]:
    """Positions, cache slots and per-sequence outputs of one call.

    coords: [B, M, 3] int; seq_rev_off: [B+1]; rev_tok_off: [R+1]; idx: [sum K].
    Returns exact positions (Fractions), their float64 values (each rounded
    once from the exact rational), the slot of every token (the cache length
    before the call plus the token's rank among its sequence's tokens in this
    call: the Concat of Eq. "active_cache"), and cache_len_out / next_pos."""
    coords = np.asarray(coords)
    seq_rev_off = [int(x) for x in np.asarray(seq_rev_off)]
    rev_tok_off = [int(x) for x in np.asarray(rev_tok_off)]
    idx = np.asarray(idx)
    B = len(seq_rev_off) - 1
    total = rev_tok_off[-1]
    frac = [None] * total
    slot = np.zeros(total, dtype=np.int64)
    seq_of = np.zeros(total, dtype=np.int64)
    cache_len_out = np.zeros(B, dtype=np.int64)
    next_pos = np.zeros(B, dtype=np.int64)
    for b in range(B):
        t0 = rev_tok_off[seq_rev_off[b]]
        t1 = rev_tok_off[seq_rev_off[b + 1]]
        for r in range(seq_rev_off[b], seq_rev_off[b + 1]):
            j0, j1 = rev_tok_off[r], rev_tok_off[r + 1]
            sel = [coords[b, int(idx[j])] for j in range(j0, j1)]
            pos = reassign_revisit(sel, int(p_txt[b]), L, mode, degenerate, seq_rank0=j0 - t0)
            for j in range(j0, j1):
                frac[j] = pos[j - j0]
                slot[j] = int(cache_len_in[b]) + (j - t0)
                seq_of[j] = b
        cache_len_out[b] = int(cache_len_in[b]) + (t1 - t0)
        next_pos[b] = next_text_pos(int(p_txt[b]), t1 - t0, mode)
    pos64 = np.array([[float(x) for x in f] for f in frac], dtype=np.float64).reshape(total, 3)
    return dict(frac=frac, pos=pos64, slot=slot, seq=seq_of,
                cache_len_out=cache_len_out, next_pos=next_pos)


# ----------------------------------------------------------------------------
# Rotary rebinding (Sec. 3.3) and the position-bound cache (Sec. 2.3)
# ----------------------------------------------------------------------------
def inv_freq(head_dim: int, theta: float) -> np.ndarray:
    """theta^(-2i/D) for rotation pair i = 0 .. D/2 - 1, float64."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(theta), -2.0 * i / head_dim)


def pair_axes(head_dim: int, sections, layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Axis (0 = t, 1 = h, 2 = w) whose position drives rotation pair i."""
    P = head_dim // 2
    st, sh, sw = (int(s) for s in sections)
    assert st + sh + sw == P
    i = np.arange(P)
    if layout == LAYOUT_SECTIONED:
        return np.where(i < st, 0, np.where(i < st + sh, 1, 2))
    if layout == LAYOUT_INTERLEAVED:
        ax = np.zeros(P, dtype=np.int64)
        ax[(i % 3 == 1) & (i < 3 * sh)] = 1
        ax[(i % 3 == 2) & (i < 3 * sw)] = 2
        return ax
    raise ValueError(layout)


def angles(pos: np.ndarray, head_dim: int, sections, theta: float,
           layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """[N, P] float64 rotation angle of pair i: position on axis(i) x inv_freq_i."""
    pos = np.asarray(pos, dtype=np.float64).reshape(-1, 3)
    ax = pair_axes(head_dim, sections, layout)
    return pos[:, ax] * inv_freq(head_dim, theta)[None, :]


def rope(x: np.ndarray, ang: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE in float64. x: [N, ..., D]; ang: [N, D/2].
    Pair (x_i, x_{i+D/2}) is rotated by ang_i:
    (x_i cos - x_{i+D/2} sin, x_{i+D/2} cos + x_i sin)."""
    x = np.asarray(x, dtype=np.float64)
    P = x.shape[-1] // 2
    shp = (ang.shape[0],) + (1,) * (x.ndim - 2) + (P,)
    c = np.cos(ang).reshape(shp)
    s = np.sin(ang).reshape(shp)
    a, b = x[..., :P], x[..., P:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (int16/uint16) as float64."""
    u = np.asarray(bits).astype(np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def f64_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    """Round float64 to the nearest bf16 value (ties to even), returned as
    float64; finite normal range only (used for reporting)."""
    m, e = np.frexp(np.asarray(x, dtype=np.float64))
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def rebind_keys(k_raw_bits: np.ndarray, pos: np.ndarray, head_dim: int, sections,
                theta: float, layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Eq. "cache_reconstruction": K_hat = RoPE(K_raw, P_hat), float64.
    k_raw_bits: [N, ..., D] bf16 bit patterns of the gathered raw keys of N
    tokens; pos: [N, 3] reassigned positions."""
    return rope(bf16_bits_to_f64(k_raw_bits), angles(pos, head_dim, sections, theta, layout))


def position_bound_keys(k_raw_bits, coords, head_dim, sections, theta,
                        layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Eq. "historical_position_bound_kv": k_tilde = RoPE(k_raw, p_m)."""
    return rebind_keys(k_raw_bits, np.asarray(coords, dtype=np.float64), head_dim, sections,
                       theta, layout)


def prefill_capture(k_raw_bits, v_raw_bits, coords, head_dim, sections, theta,
                    layout: int = LAYOUT_SECTIONED):
    """Sec. 3.1: during prefill the raw projections of every visual token are
    kept as they are (Eq. "raw_kv", "global_raw_memory") while the ordinary
    cache receives the position-bound entries of Eq.
    "historical_position_bound_kv" (key rotated at the original coordinate,
    value unchanged). Inputs [M, ..., D] bf16 bit patterns and [M, 3] coords;
    returns (store K bits, store V bits, cache K float64, cache V bits)."""
    k_raw_bits = np.asarray(k_raw_bits)
    v_raw_bits = np.asarray(v_raw_bits)
    k_cache = position_bound_keys(k_raw_bits, coords, head_dim, sections, theta, layout)
    return k_raw_bits.copy(), v_raw_bits.copy(), k_cache, v_raw_bits.copy()


def decode_attention(q_raw: np.ndarray, q_pos: int, k_act: np.ndarray, v_act: np.ndarray,
                     head_dim: int, sections, theta: float,
                     layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Eq. "decode_with_active_cache" for one sequence and one layer:
    o = softmax(RoPE(q_raw, p_next) K_act^T / sqrt(d_k)) V_act.

    q_raw: [Hq, D] raw query (values); q_pos: the query's text position, the
    triple (p, p, p) under M-RoPE; k_act, v_act: [S, H, D] active cache
    (values). Query head hq reads KV head hq // (Hq / H). Returns [Hq, D]."""
    q_raw = np.asarray(q_raw, dtype=np.float64)
    k_act = np.asarray(k_act, dtype=np.float64)
    v_act = np.asarray(v_act, dtype=np.float64)
    Hq = q_raw.shape[0]
    H = k_act.shape[1]
    group = Hq // H
    pos = np.full((Hq, 3), float(q_pos))
    q = rope(q_raw, angles(pos, head_dim, sections, theta, layout))
    out = np.zeros((Hq, head_dim))
    for hq in range(Hq):
        kh = hq // group
        logits = k_act[:, kh, :] @ q[hq] / np.sqrt(head_dim)
        w = np.exp(logits - logits.max())
        out[hq] = (w / w.sum()) @ v_act[:, kh, :]
    return out


def ads_relevance(q_raw: np.ndarray, q_pos: int, k_raw_bits: np.ndarray, coords, head_dim: int,
                  sections, theta: float, layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Relevance of each visual token to the trigger query (the reading of the
    attention-driven selection named in Sec. 2.1): q_raw [Hq, D] values at
    text position q_pos; k_raw_bits [M, H, D] raw keys of one layer; coords
    [M, 3]. r_m = mean over query heads h of softmax_m(RoPE(q_h, (p,p,p)) .
    RoPE(k_m, p_m) / sqrt(D)), query head h reading KV head h // (Hq / H)."""
    q_raw = np.asarray(q_raw, dtype=np.float64)
    Hq = q_raw.shape[0]
    k = position_bound_keys(k_raw_bits, coords, head_dim, sections, theta, layout)  # [M, H, D]
    H = k.shape[1]
    group = Hq // H
    q = rope(q_raw, angles(np.full((Hq, 3), float(q_pos)), head_dim, sections, theta, layout))
    r = np.zeros(k.shape[0])
    for h in range(Hq):
        lg = k[:, h // group, :] @ q[h] / np.sqrt(head_dim)
        w = np.exp(lg - lg.max())
        r += w / w.sum()
    return r / Hq


def ads_relevance_cached(q_raw: np.ndarray, q_pos: int, k_cached: np.ndarray, head_dim: int,
                         sections, theta: float, layout: int = LAYOUT_SECTIONED) -> np.ndarray:
    """Relevance read from the decoder's position-bound cache (second reading
    of the attention-driven selection named in Sec. 2.1): k_cached [M, H, D]
    holds the visual tokens' keys as that cache keeps them, already rotated at
    their own coordinates (Eq. "historical_position_bound_kv"), so only the
    query is rotated: r_m = mean over query heads h of
    softmax_m(RoPE(q_h, (p,p,p)) . k_m / sqrt(D)), query head h reading KV
    head h // (Hq / H)."""
    q_raw = np.asarray(q_raw, dtype=np.float64)
    k = np.asarray(k_cached, dtype=np.float64)
    Hq = q_raw.shape[0]
    group = Hq // k.shape[1]
    q = rope(q_raw, angles(np.full((Hq, 3), float(q_pos)), head_dim, sections, theta, layout))
    r = np.zeros(k.shape[0])
    for h in range(Hq):
        lg = k[:, h // group, :] @ q[h] / np.sqrt(head_dim)
        w = np.exp(lg - lg.max())
        r += w / w.sum()
    return r / Hq


def ads_select(relevance: np.ndarray, K: int) -> np.ndarray:
    """I_tau of Eq. 3: the K most relevant tokens (equal relevance: lower
    token index first), in ascending token order."""
    order = sorted(range(len(relevance)), key=lambda m: (-relevance[m], m))
    return np.array(sorted(order[:K]), dtype=np.int64)


# ----------------------------------------------------------------------------
# Whole call on small inputs: gather, reassign, rebind, concat
# ----------------------------------------------------------------------------
def rebind_inject(store_k_bits, store_v_bits, coords, seq_rev_off, rev_tok_off, idx,
                  p_txt, cache_len_in, head_dim, sections, theta, L, mode=MODE_PCR,
                  degenerate="zero", layout=LAYOUT_SECTIONED, layers=None):
    """Algorithm 1 end to end on host arrays.

    store_*_bits: [B, n_L, M, H, D] bf16 bit patterns (raw, pre-rotation).
    Returns the plan (see ``plan``) plus, for every selected token and every
    layer in ``layers`` (default all), the rebound keys K_hat (float64) and the
    reused values V_hat (bit patterns): arrays [sum K, len(layers), H, D]."""
    pl = plan(coords, seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in, L, mode, degenerate)
    store_k_bits = np.asarray(store_k_bits)
    store_v_bits = np.asarray(store_v_bits)
    if layers is None:
        layers = list(range(store_k_bits.shape[1]))
    seq = pl["seq"]
    idx = np.asarray(idx).astype(np.int64)
    # Gather: M_tau = M[I_tau], for every requested layer (Eq. 7).
    k_sel = store_k_bits[seq[:, None], np.asarray(layers)[None, :], idx[:, None]]
    v_sel = store_v_bits[seq[:, None], np.asarray(layers)[None, :], idx[:, None]]
    k_hat = rebind_keys(k_sel, pl["pos"], head_dim, sections, theta, layout)
    pl.update(k_hat=k_hat, v_hat=v_sel, layers=list(layers), k_raw=k_sel)
    return pl


def pair_norms(k_raw_bits: np.ndarray) -> np.ndarray:
    """Norm of each rotation pair (x_i, x_{i+D/2}) of the raw keys, repeated on
    both of its elements: the quantity a rotary embedding preserves (Sec. 2.3
    and Sec. 3.3, Eq. "cache_reconstruction": the rebound key differs from the
    raw key by a rotation of each pair). Used to scale errors near zero."""
    x = bf16_bits_to_f64(k_raw_bits)
    P = x.shape[-1] // 2
    r = np.sqrt(x[..., :P] ** 2 + x[..., P:] ** 2)
    return np.concatenate([r, r], axis=-1)

