"""Pins for the CPU oracle: checks against what the paper and mathematics fix.

Each ``pin_*`` function takes the oracle module and raises AssertionError when
the oracle disagrees with a fact that does not come from the oracle itself:
values worked by hand from the paper's equations (tests/golden/), closed forms
and invariants stated in Sec. 2.3 / 3.2 / 3.3, textbook rotary embedding
written as complex multiplication, and a brute force on a 2x2 region.
``test_planted_mistakes`` plants plausible mistakes in the oracle (on the CPU)
and checks that some pin catches each of them.
"""
import cmath
import math
import os
import random
from fractions import Fraction

import numpy as np
import pytest

from oracle import prcr_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line.split())
    return rows


def _grid_coords(rows, cols, base=16, frame=0):
    return [(base + frame, base + r, base + c) for r in range(rows) for c in range(cols)]


# ----------------------------------------------------------------------------
# Position pins (Sec. 3.2)
# ----------------------------------------------------------------------------
def pin_worked_rect4x4(o):
    """Hand-worked 4x4 example, p_txt = 200, L = 2 (tests/golden)."""
    rows = _golden_rows("pcr_rect4x4_p200_L2.txt")
    expect = {int(r[0]): Fraction(int(r[3]), int(r[4])) for r in rows if r[0].isdigit()}
    t_expect = [Fraction(int(r[1]), int(r[2])) for r in rows if r[0] == "T"][0]
    nxt = [int(r[1]) for r in rows if r[0] == "NEXT"][0]
    r0, c0 = 2, 3
    sel = [(16, 16 + r0 + r, 16 + c0 + c) for r in range(4) for c in range(4)]
    pos = o.reassign_revisit(sel, 200, 2, o.MODE_PCR)
    for j, (r, c) in enumerate([(r, c) for r in range(4) for c in range(4)]):
        assert pos[j][0] == t_expect
        assert pos[j][1] == expect[r], (j, pos[j][1], expect[r])
        assert pos[j][2] == expect[c], (j, pos[j][2], expect[c])
    assert o.next_text_pos(200, 16, o.MODE_PCR) == nxt


def pin_worked_rect2x2(o):
    rows = _golden_rows("pcr_rect2x2_p200_L2.txt")
    expect = {int(r[0]): Fraction(int(r[1]), int(r[2])) for r in rows if r[0].isdigit()}
    t_expect = [Fraction(int(r[1]), int(r[2])) for r in rows if r[0] == "T"][0]
    sel = [(40, 40 + r, 50 + c) for r in range(2) for c in range(2)]
    pos = o.reassign_revisit(sel, 200, 2, o.MODE_PCR)
    for j, (r, c) in enumerate([(r, c) for r in range(2) for c in range(2)]):
        assert pos[j] == [t_expect, expect[r], expect[c]]


def _random_revisit(rng, K):
    rows = rng.randint(1, 9)
    cols = rng.randint(1, 9)
    grid = [(5 + rng.randint(0, 3), 7 + r, 11 + c) for r in range(rows) for c in range(cols)]
    K = min(K, len(grid))
    return rng.sample(grid, K)


def pin_pcr_closed_forms(o):
    """Range endpoints, strict interval, mirror symmetry, layout preservation,
    uniform shift and K = 1 midpoint, all from Eq. "image_range_fractional_reinsert"."""
    rng = random.Random(7)
    for trial in range(300):
        K = rng.randint(1, 40)
        sel = _random_revisit(rng, K)
        K = len(sel)
        p = rng.randint(0, 40000)
        L = rng.randint(0, 6)
        pos = o.reassign_revisit(sel, p, L, o.MODE_PCR)
        assert len(pos) == K
        for a in range(3):
            vals = [int(c[a]) for c in sel]
            lo, hi = min(vals), max(vals)
            for j, c in enumerate(sel):
                ph = pos[j][a]
                # strictly inside (p - L, p + 1)
                assert Fraction(p - L) < ph < Fraction(p + 1), (p, L, K, ph)
                if hi > lo:
                    if c[a] == lo:
                        assert ph == Fraction(p - L) + Fraction(L + 1, K + 1)
                    if c[a] == hi:
                        assert ph == Fraction(p - L) + Fraction((L + 1) * K, K + 1)
                    # affine in the stored coordinate: layout preserved
                    slope = Fraction((L + 1) * (K - 1), (K + 1) * (hi - lo))
                    base = Fraction(p - L) + Fraction(L + 1, K + 1)
                    assert ph == base + slope * (int(c[a]) - lo)
                else:
                    # degenerate axis, reading u = 0
                    assert ph == Fraction(p - L) + Fraction(L + 1, K + 1)
            # mirror symmetry: p(u) + p(1 - u) = 2 (p - L) + L + 1
            if hi > lo:
                by_c = {int(c[a]): pos[j][a] for j, c in enumerate(sel)}
                for cv, ph in by_c.items():
                    mv = lo + hi - cv
                    if mv in by_c:
                        assert ph + by_c[mv] == 2 * (p - L) + L + 1
        # uniform shift of p_txt moves every position by the same amount
        s = rng.randint(-500, 500)
        pos2 = o.reassign_revisit(sel, p + s, L, o.MODE_PCR)
        for j in range(K):
            for a in range(3):
                assert pos2[j][a] - pos[j][a] == s
    # K = 1: the midpoint of the interval
    for p, L in ((200, 2), (7, 0), (30000, 5)):
        pos = o.reassign_revisit([(3, 4, 5)], p, L, o.MODE_PCR)
        assert pos[0] == [Fraction(p - L) + Fraction(L + 1, 2)] * 3


def pin_degenerate_center(o):
    """Reading u = 1/2 on a degenerate axis puts it at the interval's centre."""
    sel = [(9, 3, c) for c in range(5)]
    pos = o.reassign_revisit(sel, 100, 2, o.MODE_PCR, degenerate="center")
    for j in range(5):
        assert pos[j][0] == pos[j][1] == Fraction(98) + Fraction(3, 2)


def pin_other_modes(o):
    """ORIGINAL keeps the stored coordinates (Eq. "historical_position_bound_kv");
    UIR is PCR with L = 0 on the 1-D order coordinate; LPA appends at
    p + 1 .. p + K and moves the next text position to p + K + 1."""
    sel = [(2, 9, 4), (2, 9, 5), (2, 10, 4), (3, 10, 5), (3, 11, 6)]
    K = len(sel)
    orig = o.reassign_revisit(sel, 300, 2, o.MODE_ORIGINAL)
    assert orig == [[Fraction(x) for x in c] for c in sel]
    uir = o.reassign_revisit(sel, 300, 2, o.MODE_UIR)
    order = [(0, j, j) for j in range(K)]
    pcr_l0 = o.reassign_revisit(order, 300, 0, o.MODE_PCR)
    for j in range(K):
        assert uir[j] == [pcr_l0[j][1]] * 3
        assert Fraction(300) < uir[j][0] < Fraction(301)
    lpa = o.reassign_revisit(sel, 300, 2, o.MODE_LPA, seq_rank0=3)
    assert [x[0] for x in lpa] == [Fraction(300 + 3 + j + 1) for j in range(K)]
    assert o.next_text_pos(300, 8, o.MODE_LPA) == 309
    for m in (o.MODE_PCR, o.MODE_ORIGINAL, o.MODE_UIR):
        assert o.next_text_pos(300, 8, m) == 301


def pin_plan_slots_and_continuity(o):
    """Slots follow the existing cache in call order (Concat of Eq.
    "active_cache"); cache length grows by exactly K per sequence; the text
    position continues at p + 1; float64 positions are the exact rationals
    rounded once."""
    coords = np.zeros((2, 20, 3), dtype=np.int64)
    for m in range(20):
        coords[:, m] = (16, 16 + m // 5, 16 + m % 5)
    seq_rev_off = [0, 2, 3]
    idx = [0, 1, 5, 6, 12, 13, 14, 3, 4, 9]
    rev_tok_off = [0, 4, 7, 10]
    p_txt = [500, 123]
    cache_len_in = [501, 40]
    pl = o.plan(coords, seq_rev_off, rev_tok_off, idx, p_txt, cache_len_in, 2, o.MODE_PCR)
    assert list(pl["slot"]) == [501, 502, 503, 504, 505, 506, 507, 40, 41, 42]
    assert list(pl["seq"]) == [0] * 7 + [1] * 3
    assert list(pl["cache_len_out"]) == [508, 43]
    assert list(pl["next_pos"]) == [501, 124]
    for j in range(10):
        for a in range(3):
            f = pl["frac"][j][a]
            assert pl["pos"][j, a] == f.numerator / f.denominator  # one correctly rounded division
    # each revisit is reassigned on its own: revisit 1 has rows {2} only -> degenerate h
    assert pl["frac"][4][1] == Fraction(498) + Fraction(3, 4)


# ----------------------------------------------------------------------------
# Rotary pins (Sec. 2.3, Sec. 3.3)
# ----------------------------------------------------------------------------
def _textbook_rope_1d(x, p, theta):
    """Su et al. RoPE as complex multiplication, rotate-half pairing:
    z_i = x_i + 1j * x_{i+P}, z_i' = z_i * exp(1j * p * theta^(-2i/D))."""
    D = len(x)
    P = D // 2
    out = [0.0] * D
    for i in range(P):
        w = theta ** (-2.0 * i / D)
        z = complex(x[i], x[i + P]) * cmath.exp(1j * p * w)
        out[i], out[i + P] = z.real, z.imag
    return out


def pin_rope_closed_forms(o):
    vals = {r[0]: float(r[1]) for r in _golden_rows("rope_closed_forms.txt")}
    y = o.rope(np.array([[1.0, 0.0]]), np.array([[1.0]]))
    assert abs(y[0, 0] - vals["cos1"]) < 1e-15 and abs(y[0, 1] - vals["sin1"]) < 1e-15
    k_bits = np.array([[0x3F80, 0x0000]], dtype=np.uint16)  # bf16 (1.0, 0.0)
    y = o.rebind_keys(k_bits, np.array([[1.0, 1.0, 1.0]]), 2, (1, 0, 0), 1e6)
    assert abs(y[0, 0] - vals["cos1"]) < 1e-15 and abs(y[0, 1] - vals["sin1"]) < 1e-15
    f = o.inv_freq(128, 1e4)
    assert abs(f[32] - vals["invfreq_1e4_d128_i32"]) < 1e-16
    assert f[0] == 1.0
    r = f[1:] / f[:-1]
    assert np.allclose(r, 1e4 ** (-2.0 / 128), rtol=1e-13, atol=0)


def pin_mrope_equal_axes_is_textbook(o):
    """M-RoPE at (p, p, p) equals 1-D RoPE at p, whatever the sections."""
    rng = np.random.default_rng(3)
    for D, sec in ((8, (1, 1, 2)), (64, (8, 12, 12)), (128, (16, 24, 24)), (128, (24, 20, 20))):
        for layout in (o.LAYOUT_SECTIONED, o.LAYOUT_INTERLEAVED):
            x = rng.standard_normal((5, D))
            p = rng.uniform(-3000, 3000, size=5)
            pos = np.repeat(p[:, None], 3, axis=1)
            got = o.rope(x, o.angles(pos, D, sec, 1e6, layout))
            for n in range(5):
                ref = _textbook_rope_1d(list(x[n]), p[n], 1e6)
                assert np.allclose(got[n], ref, rtol=0, atol=1e-9)


def pin_mrope_sections(o):
    """A position on one axis only rotates exactly the pairs of that axis's
    band: the first s_t pairs (t), the next s_h (h), the last s_w (w)."""
    D, sec = 64, (8, 12, 12)
    P = D // 2
    x = np.random.default_rng(5).standard_normal((1, D))
    for a in range(3):
        pos = np.zeros((1, 3))
        pos[0, a] = 37.25
        y = o.rope(x, o.angles(pos, D, sec, 1e6))
        moved = [not (np.isclose(y[0, i], x[0, i], atol=1e-12) and
                      np.isclose(y[0, i + P], x[0, i + P], atol=1e-12)) for i in range(P)]
        lo = [0, sec[0], sec[0] + sec[1]][a]
        expect = [lo <= i < lo + sec[a] for i in range(P)]
        assert moved == expect, (a, moved)
    # interleaved layout of the same sizes (24, 20, 20 over 64 pairs)
    ax = o.pair_axes(128, (24, 20, 20), o.LAYOUT_INTERLEAVED)
    assert list(np.bincount(ax, minlength=3)) == [24, 20, 20]
    assert list(ax[:6]) == [0, 1, 2, 0, 1, 2] and list(ax[60:]) == [0, 0, 0, 0]


def pin_rope_invariants(o):
    """Per-pair norm preserved; R(a) R(b) = R(a + b); logits depend only on
    the relative offset (Eq. "direct_reuse_score"): a uniform shift of all
    positions leaves <RoPE(q, P), RoPE(k, P')> unchanged and it equals
    <q, R(P' - P) k>."""
    rng = np.random.default_rng(11)
    D, sec = 128, (16, 24, 24)
    P = D // 2
    x = rng.standard_normal((20, D))
    pa = rng.uniform(0, 30000, size=(20, 3))
    pb = rng.uniform(-50, 50, size=(20, 3))
    y = o.rope(x, o.angles(pa, D, sec, 1e6))
    n0 = np.hypot(x[:, :P], x[:, P:])
    n1 = np.hypot(y[:, :P], y[:, P:])
    assert np.allclose(n0, n1, rtol=1e-13, atol=0)
    yy = o.rope(y, o.angles(pb, D, sec, 1e6))
    y2 = o.rope(x, o.angles(pa + pb, D, sec, 1e6))
    assert np.allclose(yy, y2, rtol=0, atol=1e-9)
    q = rng.standard_normal((20, D))
    k = rng.standard_normal((20, D))
    Pq = np.repeat(rng.uniform(1000, 5000, size=(20, 1)), 3, axis=1)
    Pk = rng.uniform(0, 5000, size=(20, 3))
    s = rng.uniform(-900, 900, size=(20, 1))
    l0 = np.sum(o.rope(q, o.angles(Pq, D, sec, 1e6)) * o.rope(k, o.angles(Pk, D, sec, 1e6)), axis=1)
    l1 = np.sum(o.rope(q, o.angles(Pq + s, D, sec, 1e6)) * o.rope(k, o.angles(Pk + s, D, sec, 1e6)), axis=1)
    l2 = np.sum(q * o.rope(k, o.angles(Pk - Pq, D, sec, 1e6)), axis=1)
    assert np.allclose(l0, l1, rtol=0, atol=1e-8)
    assert np.allclose(l0, l2, rtol=0, atol=1e-8)


def pin_bf16_helpers(o):
    """bf16 bit patterns decode exactly; rounding to bf16 is to nearest even."""
    bits = np.array([0x3F80, 0xBF80, 0x4049, 0x0000, 0x3F81], dtype=np.uint16)
    assert list(o.bf16_bits_to_f64(bits)) == [1.0, -1.0, 3.140625, 0.0, 1.0078125]
    assert list(o.f64_to_bf16_rne(np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -9]))) == \
        [1.0, 1.0 + 2 ** -6, 1.0]


# ----------------------------------------------------------------------------
# Whole-call brute force on a 2x2 region (independent of the oracle's code)
# ----------------------------------------------------------------------------
def _bf16_value(bits):
    b = int(bits) & 0xFFFF
    sign = -1.0 if b >> 15 else 1.0
    e = (b >> 7) & 0xFF
    m = b & 0x7F
    if e == 0:
        return sign * m * 2.0 ** -133
    return sign * (1 + m / 128.0) * 2.0 ** (e - 127)


def _brute_force_2x2(store_k, store_v, coords, sel_ids, p, L, cache_len, D, sec, theta):
    K = len(sel_ids)
    out = []
    cs = [coords[m] for m in sel_ids]
    for j, m in enumerate(sel_ids):
        ph = []
        for a in range(3):
            vals = [c[a] for c in cs]
            lo, hi = min(vals), max(vals)
            u = Fraction(cs[j][a] - lo, hi - lo) if hi != lo else Fraction(0)
            ph.append(p - L + Fraction(L + 1) * (1 + (K - 1) * u) / (K + 1))
        rows_k, rows_v = [], []
        for l in range(store_k.shape[0]):
            hk, hv = [], []
            for h in range(store_k.shape[2]):
                x = [_bf16_value(v) for v in store_k[l, m, h]]
                P = D // 2
                y = [0.0] * D
                for i in range(P):
                    axis = 0 if i < sec[0] else (1 if i < sec[0] + sec[1] else 2)
                    ang = float(ph[axis]) * theta ** (-2.0 * i / D)
                    z = complex(x[i], x[i + P]) * cmath.exp(1j * ang)
                    y[i], y[i + P] = z.real, z.imag
                hk.append(y)
                hv.append(list(store_v[l, m, h]))
            rows_k.append(hk)
            rows_v.append(hv)
        out.append(dict(slot=cache_len + j, pos=ph, k=rows_k, v=rows_v))
    return out, p + 1, cache_len + K


def pin_brute_force_2x2(o):
    rng = np.random.default_rng(17)
    D, sec, theta, nL, H, M = 16, (2, 3, 3), 1e6, 2, 2, 12
    store_k = rng.integers(0, 1 << 16, size=(1, nL, M, H, D)).astype(np.uint16)
    store_v = rng.integers(0, 1 << 16, size=(1, nL, M, H, D)).astype(np.uint16)
    # keep finite, moderate values: exponent field 120..130
    for s in (store_k, store_v):
        s &= 0x807F
        s |= (rng.integers(120, 131, size=s.shape).astype(np.uint16) << 7)
    coords = np.array([[(16, 16 + m // 4, 16 + m % 4) for m in range(M)]])
    sel = [5, 6, 9, 10]  # rows 1..2, cols 1..2
    bf, nxt, clen = _brute_force_2x2(store_k[0], store_v[0], coords[0], sel, 200, 2, 201, D, sec, theta)
    got = o.rebind_inject(store_k, store_v, coords, [0, 1], [0, 4], sel, [200], [201],
                          D, sec, theta, 2, o.MODE_PCR)
    assert list(got["next_pos"]) == [nxt] and list(got["cache_len_out"]) == [clen]
    for j in range(4):
        assert got["slot"][j] == bf[j]["slot"]
        assert got["frac"][j] == bf[j]["pos"]
        assert np.allclose(got["k_hat"][j], np.array(bf[j]["k"]), rtol=1e-12, atol=1e-12)
        assert np.array_equal(got["v_hat"][j].astype(np.uint16), np.array(bf[j]["v"], dtype=np.uint16))
    # 2x2 positions are the hand-worked ones
    assert sorted({x[1] for x in got["frac"]}) == [Fraction(993, 5), Fraction(1002, 5)]


def pin_original_mode_is_position_bound_cache(o):
    """Rebinding at the stored coordinates reproduces the historical cache
    entry RoPE(k_raw, p_m) of Eq. "historical_position_bound_kv", here built
    with textbook complex rotation on each axis band."""
    rng = np.random.default_rng(23)
    D, sec, nL, H, M = 32, (4, 6, 6), 1, 1, 9
    kb = (rng.integers(0x3C00, 0x4100, size=(1, nL, M, H, D))).astype(np.uint16)
    vb = (rng.integers(0x3C00, 0x4100, size=(1, nL, M, H, D))).astype(np.uint16)
    coords = np.array([[(20, 30 + m // 3, 40 + m % 3) for m in range(M)]])
    sel = [0, 4, 8, 2]
    got = o.rebind_inject(kb, vb, coords, [0, 1], [0, 4], sel, [999], [1000], D, sec, 1e6, 2,
                          o.MODE_ORIGINAL)
    P = D // 2
    for j, m in enumerate(sel):
        x = [_bf16_value(v) for v in kb[0, 0, m, 0]]
        y = [0.0] * D
        for i in range(P):
            axis = 0 if i < sec[0] else (1 if i < sec[0] + sec[1] else 2)
            z = complex(x[i], x[i + P]) * cmath.exp(1j * coords[0, m, axis] * 1e6 ** (-2.0 * i / D))
            y[i], y[i + P] = z.real, z.imag
        assert np.allclose(got["k_hat"][j, 0, 0], y, rtol=0, atol=1e-12)


def pin_prefill_capture(o):
    """The store keeps the raw rows bit for bit; the cache key is the textbook
    rotation at the original coordinate (Eq. "historical_position_bound_kv")."""
    rng = np.random.default_rng(29)
    D, sec = 16, (2, 3, 3)
    kb = rng.integers(0x3C00, 0x4100, size=(5, 2, D)).astype(np.uint16)
    vb = rng.integers(0x3C00, 0x4100, size=(5, 2, D)).astype(np.uint16)
    coords = np.array([(7, 20 + m, 30 - m) for m in range(5)])
    sk, sv, ck, cv = o.prefill_capture(kb, vb, coords, D, sec, 1e6)
    assert np.array_equal(sk, kb) and np.array_equal(sv, vb) and np.array_equal(cv, vb)
    P = D // 2
    for m in range(5):
        for h in range(2):
            x = [_bf16_value(v) for v in kb[m, h]]
            for i in range(P):
                axis = 0 if i < sec[0] else (1 if i < sec[0] + sec[1] else 2)
                z = complex(x[i], x[i + P]) * cmath.exp(1j * coords[m, axis] * 1e6 ** (-2.0 * i / D))
                assert abs(ck[m, h, i] - z.real) < 1e-12 and abs(ck[m, h, i + P] - z.imag) < 1e-12


def pin_decode_attention(o):
    """Eq. "decode_with_active_cache": (1) one cached slot returns its value
    row; (2) equal keys give the mean of the values; (3) against a direct
    per-slot loop with math.exp; (4) a uniform shift of every position
    (query and cached keys) leaves the output unchanged (Eq.
    "direct_reuse_score": logits see only relative offsets); (5) GQA: query
    head hq reads KV head hq // group."""
    rng = np.random.default_rng(31)
    D, sec, th = 16, (2, 3, 3), 1e6
    q = rng.standard_normal((4, D))
    v1 = rng.standard_normal((1, 2, D))
    k1 = rng.standard_normal((1, 2, D))
    out = o.decode_attention(q, 50, k1, v1, D, sec, th)
    assert np.allclose(out, np.repeat(v1[0], 2, axis=0), atol=1e-14)
    kk = np.repeat(rng.standard_normal((1, 2, D)), 5, axis=0)
    vv = rng.standard_normal((5, 2, D))
    out = o.decode_attention(q, 7, kk, vv, D, sec, th)
    assert np.allclose(out, np.repeat(vv.mean(axis=0), 2, axis=0), atol=1e-12)
    S = 9
    k_raw = rng.standard_normal((S, 2, D))
    v = rng.standard_normal((S, 2, D))
    kpos = rng.uniform(0, 300, size=(S, 3))
    k = o.rope(k_raw, o.angles(kpos, D, sec, th))
    out = o.decode_attention(q, 301, k, v, D, sec, th)
    P = D // 2
    for hq in range(4):
        kh = hq // 2
        qz = [complex(q[hq, i], q[hq, i + P]) * cmath.exp(1j * 301 * th ** (-2.0 * i / D))
              for i in range(P)]
        qr = [z.real for z in qz] + [z.imag for z in qz]
        lg = [sum(qr[d] * k[s, kh, d] for d in range(D)) / math.sqrt(D) for s in range(S)]
        mx = max(lg)
        w = [math.exp(x - mx) for x in lg]
        ref = [sum(w[s] * v[s, kh, d] for s in range(S)) / sum(w) for d in range(D)]
        assert np.allclose(out[hq], ref, rtol=0, atol=1e-12)
    shift = 1234.0
    k2 = o.rope(k_raw, o.angles(kpos + shift, D, sec, th))
    out2 = o.decode_attention(q, 301 + shift, k2, v, D, sec, th)
    assert np.allclose(out, out2, rtol=0, atol=1e-9)


def pin_ads(o):
    """Selection reading (Sec. 2.1, Eq. 3): relevance is a per-head softmax
    averaged over heads, so it sums to 1; a key equal to a large multiple of
    the (rotated) query direction wins; ties go to the lower index; the set
    comes back in ascending order; against a direct loop with math.exp."""
    rng = np.random.default_rng(37)
    D, sec, th = 16, (2, 3, 3), 1e6
    M, H, Hq = 12, 2, 4
    kb = rng.integers(0x3C00, 0x4100, size=(M, H, D)).astype(np.uint16)
    kb[..., ::2] |= 0x8000  # mixed signs
    coords = np.array([(3, 10 + m // 4, 20 + m % 4) for m in range(M)])
    q = rng.standard_normal((Hq, D))
    r = o.ads_relevance(q, 40, kb, coords, D, sec, th)
    assert abs(r.sum() - 1.0) < 1e-12 and (r > 0).all()
    # direct loop
    P = D // 2
    ref = np.zeros(M)
    for h in range(Hq):
        qz = [complex(q[h, i], q[h, i + P]) * cmath.exp(1j * 40 * th ** (-2.0 * i / D)) for i in range(P)]
        lg = []
        for m in range(M):
            x = [_bf16_value(v) for v in kb[m, h // 2]]
            kz = []
            for i in range(P):
                axis = 0 if i < sec[0] else (1 if i < sec[0] + sec[1] else 2)
                kz.append(complex(x[i], x[i + P]) * cmath.exp(1j * coords[m, axis] * th ** (-2.0 * i / D)))
            lg.append(sum(a.real * b.real + a.imag * b.imag for a, b in zip(qz, kz)) / math.sqrt(D))
        mx = max(lg)
        w = [math.exp(x - mx) for x in lg]
        for m in range(M):
            ref[m] += w[m] / sum(w) / Hq
    assert np.allclose(r, ref, rtol=1e-10, atol=0)
    sel = o.ads_select(np.array([0.1, 0.3, 0.3, 0.05, 0.3, 0.2]), 3)
    assert list(sel) == [1, 2, 4]
    sel = o.ads_select(np.array([0.1, 0.3, 0.3, 0.05, 0.3, 0.2]), 2)
    assert list(sel) == [1, 2]
    sel = o.ads_select(np.array([0.5, 0.1, 0.2, 0.9]), 2)
    assert list(sel) == [0, 3]


def pin_ads_cached(o):
    """Selection over the position-bound cache (second reading): against a
    direct loop (query turned by complex exponentials, keys used as given);
    relevance sums to 1; with keys rotated exactly at their coordinates it is
    the raw-store relevance (the relative-angle identity of Eq.
    "direct_reuse_score"); moving the query position and every key position
    by the same shift changes nothing."""
    rng = np.random.default_rng(41)
    D, sec, th = 16, (2, 3, 3), 1e6
    M, H, Hq = 10, 2, 6
    kc = rng.standard_normal((M, H, D))
    q = rng.standard_normal((Hq, D))
    r = o.ads_relevance_cached(q, 57, kc, D, sec, th)
    assert abs(r.sum() - 1.0) < 1e-12 and (r > 0).all()
    P = D // 2
    ref = np.zeros(M)
    for h in range(Hq):
        qz = [complex(q[h, i], q[h, i + P]) * cmath.exp(1j * 57 * th ** (-2.0 * i / D)) for i in range(P)]
        lg = [sum(qz[i].real * kc[m, h // 3, i] + qz[i].imag * kc[m, h // 3, i + P] for i in range(P))
              / math.sqrt(D) for m in range(M)]
        mx = max(lg)
        w = [math.exp(x - mx) for x in lg]
        for m in range(M):
            ref[m] += w[m] / sum(w) / Hq
    assert np.allclose(r, ref, rtol=1e-10, atol=0)
    kb = rng.integers(0x3C00, 0x4100, size=(M, H, D)).astype(np.uint16)
    kb[..., 1::2] |= 0x8000
    coords = np.array([(2, 7 + m // 5, 30 + m % 5) for m in range(M)])
    kpb = o.position_bound_keys(kb, coords, D, sec, th)
    assert np.allclose(o.ads_relevance_cached(q, 90, kpb, D, sec, th),
                       o.ads_relevance(q, 90, kb, coords, D, sec, th), rtol=1e-10, atol=0)
    kps = o.position_bound_keys(kb, coords + 500, D, sec, th)
    assert np.allclose(o.ads_relevance_cached(q, 590, kps, D, sec, th),
                       o.ads_relevance_cached(q, 90, kpb, D, sec, th), rtol=1e-9, atol=0)


def pin_pair_norms(o):
    """Norm of each rotation pair (the scale of the K error bar near zero):
    hand-worked rows (tests/golden/pair_norms.txt), shapes kept for batched
    rows, and the invariant it stands for: a rotary embedding at any angles
    leaves every pair's norm unchanged (Sec. 2.3; Sec. 3.3, Eq.
    "cache_reconstruction"), so the norms of the raw row equal the pair
    lengths of the rebound row."""
    for r in _golden_rows("pair_norms.txt"):
        D = int(r[0])
        raw = np.array([int(h, 16) for h in r[1:1 + D]], dtype=np.uint16)
        want = [float(x) for x in r[1 + D:1 + 2 * D]]
        got = o.pair_norms(raw)
        assert got.shape == (D,), (got.shape, D)
        assert list(got) == want, (r, list(got))
        # a batch of rows [N, H, D] keeps its shape and gives each row's norms
        batch = np.stack([raw, raw[::-1].copy()])[:, None, :]
        gb = o.pair_norms(batch)
        assert gb.shape == (2, 1, D)
        assert list(gb[0, 0]) == want
    rng = np.random.default_rng(23)
    D = 128
    P = D // 2
    bits = rng.integers(0x3C00, 0x4100, size=(6, 4, D)).astype(np.uint16)
    bits[..., 1::3] |= 0x8000
    rho = o.pair_norms(bits)
    x = o.bf16_bits_to_f64(bits).reshape(-1, D)
    for ang in (rng.uniform(-40, 40, size=(x.shape[0], P)), np.zeros((x.shape[0], P))):
        y = o.rope(x, ang)
        n = np.sqrt(y[:, :P] ** 2 + y[:, P:] ** 2)
        assert np.allclose(np.concatenate([n, n], axis=1), rho.reshape(-1, D), rtol=1e-13, atol=0)


PINS = [pin_worked_rect4x4, pin_worked_rect2x2, pin_pcr_closed_forms, pin_degenerate_center,
        pin_other_modes, pin_plan_slots_and_continuity, pin_rope_closed_forms,
        pin_mrope_equal_axes_is_textbook, pin_mrope_sections, pin_rope_invariants,
        pin_bf16_helpers, pin_brute_force_2x2, pin_original_mode_is_position_bound_cache,
        pin_prefill_capture, pin_decode_attention, pin_ads, pin_ads_cached, pin_pair_norms]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin(O)


# ----------------------------------------------------------------------------
# Planted mistakes: each must be caught by at least one pin
# ----------------------------------------------------------------------------
def _m_pcr_k_not_k_minus_1(u, K, p, L):
    return Fraction(p - L) + Fraction(L + 1) * (1 + K * u) / (K + 1)


def _m_pcr_denominator_k(u, K, p, L):
    return Fraction(p - L) + Fraction(L + 1) * (1 + (K - 1) * u) / K


def _m_pcr_anchor(u, K, p, L):
    return Fraction(p - L + 1) + Fraction(L + 1) * (1 + (K - 1) * u) / (K + 1)


def _m_pcr_drop_one(u, K, p, L):
    return Fraction(p - L) + Fraction(L + 1) * ((K - 1) * u) / (K + 1)


def _m_norm_from_max(c, lo, hi, degenerate="zero"):
    return Fraction(hi - int(c), hi - lo) if hi > lo else Fraction(0)


def _m_rope_sign(x, ang):
    x = np.asarray(x, dtype=np.float64)
    P = x.shape[-1] // 2
    shp = (ang.shape[0],) + (1,) * (x.ndim - 2) + (P,)
    c, s = np.cos(ang).reshape(shp), np.sin(ang).reshape(shp)
    a, b = x[..., :P], x[..., P:]
    return np.concatenate([a * c + b * s, b * c - a * s], axis=-1)


def _m_rope_adjacent_pairs(x, ang):
    x = np.asarray(x, dtype=np.float64)
    P = x.shape[-1] // 2
    shp = (ang.shape[0],) + (1,) * (x.ndim - 2) + (P,)
    c, s = np.cos(ang).reshape(shp), np.sin(ang).reshape(shp)
    a, b = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = a * c - b * s
    out[..., 1::2] = b * c + a * s
    return out


def _m_inv_freq_no_two(head_dim, theta):
    i = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(theta), -1.0 * i / head_dim)


_orig_pair_axes = O.pair_axes


def _m_axes_swapped(head_dim, sections, layout=0):
    ax = _orig_pair_axes(head_dim, sections, layout)
    return np.where(ax == 0, 1, np.where(ax == 1, 0, ax))


_orig_plan = O.plan


def _m_plan_slot_shift(*a, **k):
    pl = _orig_plan(*a, **k)
    pl["slot"] = pl["slot"] + 1
    return pl


def _m_next_pos_same(p, k, mode=0):
    return p


def _m_range_swapped_axes(sel):
    lo = [min(int(c[a]) for c in sel) for a in (0, 2, 1)]
    hi = [max(int(c[a]) for c in sel) for a in (0, 2, 1)]
    return lo, hi


_orig_decode = O.decode_attention


def _m_decode_no_scale(q_raw, q_pos, k_act, v_act, head_dim, sections, theta, layout=0):
    return _orig_decode(q_raw, q_pos, k_act * np.sqrt(head_dim), v_act, head_dim, sections, theta,
                        layout)


def _m_decode_head_modulo(q_raw, q_pos, k_act, v_act, head_dim, sections, theta, layout=0):
    H = k_act.shape[1]
    Hq = q_raw.shape[0]
    perm = np.array([(hq % H) * (Hq // H) + hq // H for hq in range(Hq)])
    return _orig_decode(q_raw[perm], q_pos, k_act, v_act, head_dim, sections, theta, layout)[
        np.argsort(perm)]


def _m_decode_query_unrotated(q_raw, q_pos, k_act, v_act, head_dim, sections, theta, layout=0):
    return _orig_decode(q_raw, 0, k_act, v_act, head_dim, sections, theta, layout)


_orig_select = O.ads_select
_orig_rel_cached = O.ads_relevance_cached


def _m_rel_cached_query_unrotated(q_raw, q_pos, k_cached, head_dim, sections, theta, layout=0):
    return _orig_rel_cached(q_raw, 0, k_cached, head_dim, sections, theta, layout)


def _m_rel_cached_head_modulo(q_raw, q_pos, k_cached, head_dim, sections, theta, layout=0):
    H = k_cached.shape[1]
    Hq = q_raw.shape[0]
    perm = np.array([(hq % H) * (Hq // H) + hq // H for hq in range(Hq)])
    return _orig_rel_cached(q_raw[perm], q_pos, k_cached, head_dim, sections, theta, layout)


def _m_select_unsorted(rel, K):
    order = sorted(range(len(rel)), key=lambda m: (-rel[m], m))
    return np.array(order[:K], dtype=np.int64)


def _m_select_ties_high(rel, K):
    order = sorted(range(len(rel)), key=lambda m: (-rel[m], -m))
    return np.array(sorted(order[:K]), dtype=np.int64)


def _m_pair_norms_no_sqrt(k_raw_bits):
    x = O.bf16_bits_to_f64(k_raw_bits)
    P = x.shape[-1] // 2
    r = x[..., :P] ** 2 + x[..., P:] ** 2
    return np.concatenate([r, r], axis=-1)


def _m_pair_norms_first_half(k_raw_bits):
    x = O.bf16_bits_to_f64(k_raw_bits)
    P = x.shape[-1] // 2
    r = np.abs(x[..., :P])
    return np.concatenate([r, r], axis=-1)


def _m_pair_norms_whole_row(k_raw_bits):
    x = O.bf16_bits_to_f64(k_raw_bits)
    return np.broadcast_to(np.sqrt((x ** 2).sum(axis=-1, keepdims=True)), x.shape).copy()


def _m_pair_norms_adjacent(k_raw_bits):
    x = O.bf16_bits_to_f64(k_raw_bits)
    r = np.sqrt(x[..., 0::2] ** 2 + x[..., 1::2] ** 2)
    return np.concatenate([r, r], axis=-1)


MUTANTS = [
    ("pcr_position", _m_pcr_k_not_k_minus_1),
    ("pcr_position", _m_pcr_denominator_k),
    ("pcr_position", _m_pcr_anchor),
    ("pcr_position", _m_pcr_drop_one),
    ("normalized_coord", _m_norm_from_max),
    ("rope", _m_rope_sign),
    ("rope", _m_rope_adjacent_pairs),
    ("inv_freq", _m_inv_freq_no_two),
    ("pair_axes", _m_axes_swapped),
    ("plan", _m_plan_slot_shift),
    ("next_text_pos", _m_next_pos_same),
    ("coord_range", _m_range_swapped_axes),
    ("decode_attention", _m_decode_no_scale),
    ("decode_attention", _m_decode_head_modulo),
    ("decode_attention", _m_decode_query_unrotated),
    ("ads_select", _m_select_unsorted),
    ("ads_select", _m_select_ties_high),
    ("ads_relevance_cached", _m_rel_cached_query_unrotated),
    ("ads_relevance_cached", _m_rel_cached_head_modulo),
    ("pair_norms", _m_pair_norms_no_sqrt),
    ("pair_norms", _m_pair_norms_first_half),
    ("pair_norms", _m_pair_norms_whole_row),
    ("pair_norms", _m_pair_norms_adjacent),
]


@pytest.mark.parametrize("name,mutant", MUTANTS, ids=[f"{n}:{m.__name__}" for n, m in MUTANTS])
def test_planted_mistakes(monkeypatch, name, mutant):
    monkeypatch.setattr(O, name, mutant)
    caught = []
    for pin in PINS:
        try:
            pin(O)
        except (AssertionError, ValueError, ZeroDivisionError, IndexError):
            caught.append(pin.__name__)
    assert caught, f"no pin catches the planted mistake in {name}"
