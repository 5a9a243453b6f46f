// Device helpers shared by the revisit kernels: row streaming with the
// rotate-half rotation, and the exact position arithmetic of Sec. 3.2.
#pragma once

#include <climits>
#include <cmath>

#include <cuda_bf16.h>

#include "prcr_internal.h"

namespace prcr {

__device__ __forceinline__ uint4 ld_stream(const uint16_t* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ void st_row(uint16_t* p, const uint4& v) {
    asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};"
                 :
                 : "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ float lo_f32(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_f32(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

// Two floats as bf16 pairs: a head (round to nearest even) and the rounded
// remainder, so that head + remainder keeps ~16 significant bits.
__device__ __forceinline__ void split_bf16x2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    hi = pack_bf16x2(x0, x1);
    lo = pack_bf16x2(x0 - lo_f32(hi), x1 - hi_f32(hi));
}

// D += A B on tensor cores: mma.sync m16n8k16, bf16 operands, float32
// accumulate (fragment layouts of the PTX ISA for this shape).
__device__ __forceinline__ void mma_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                          uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Rotate four bf16 pairs held as (first-half word x, second-half word y):
// x' = x cos - y sin, y' = y cos + x sin, float32, bf16 round-to-nearest-even.
__device__ __forceinline__ void rotate_word(uint32_t x, uint32_t y, float c0, float s0, float c1,
                                           float s1, uint32_t& xo, uint32_t& yo) {
    const float x0 = lo_f32(x), x1 = hi_f32(x);
    const float y0 = lo_f32(y), y1 = hi_f32(y);
    const float a0 = fmaf(x0, c0, -y0 * s0);
    const float a1 = fmaf(x1, c1, -y1 * s1);
    const float b0 = fmaf(y0, c0, x0 * s0);
    const float b1 = fmaf(y1, c1, x1 * s1);
    xo = pack_bf16x2(a0, a1);
    yo = pack_bf16x2(b0, b1);
}

__device__ __forceinline__ void rotate_vec(const uint4& x, const uint4& y, const float (&c)[8],
                                           const float (&s)[8], uint4& xo, uint4& yo) {
    rotate_word(x.x, y.x, c[0], s[0], c[1], s[1], xo.x, yo.x);
    rotate_word(x.y, y.y, c[2], s[2], c[3], s[3], xo.y, yo.y);
    rotate_word(x.z, y.z, c[4], s[4], c[5], s[5], xo.z, yo.z);
    rotate_word(x.w, y.w, c[6], s[6], c[7], s[7], xo.w, yo.w);
}

__device__ __forceinline__ int pair_axis(int i, int layout, int st, int sh, int sw) {
    if (layout == PRCR_LAYOUT_SECTIONED) return i < st ? 0 : (i < st + sh ? 1 : 2);
    const int r = i % 3;
    if (r == 1 && i < 3 * sh) return 1;
    if (r == 2 && i < 3 * sw) return 2;
    return 0;
}

// One (token, head, 16-byte vector) lane through n consecutive layers: the
// first-half vector of K and its rotate-half partner (half elements away) and
// the same two vectors of V are gathered, K is rotated, both are written.
// Two layers are in flight per iteration.
__device__ __forceinline__ void stream_layers(const uint16_t* sk, const uint16_t* sv, uint16_t* ck,
                                              uint16_t* cv, int64_t sls, int64_t cls, int half,
                                              int n, const float (&c)[8], const float (&s)[8]) {
    int l = 0;
    for (; l + 2 <= n; l += 2) {
        const uint4 k0a = ld_stream(sk), k1a = ld_stream(sk + half);
        const uint4 v0a = ld_stream(sv), v1a = ld_stream(sv + half);
        const uint4 k0b = ld_stream(sk + sls), k1b = ld_stream(sk + sls + half);
        const uint4 v0b = ld_stream(sv + sls), v1b = ld_stream(sv + sls + half);
        uint4 o0, o1;
        rotate_vec(k0a, k1a, c, s, o0, o1);
        st_row(ck, o0);
        st_row(ck + half, o1);
        st_row(cv, v0a);
        st_row(cv + half, v1a);
        rotate_vec(k0b, k1b, c, s, o0, o1);
        st_row(ck + cls, o0);
        st_row(ck + cls + half, o1);
        st_row(cv + cls, v0b);
        st_row(cv + cls + half, v1b);
        sk += 2 * sls; sv += 2 * sls; ck += 2 * cls; cv += 2 * cls;
    }
    if (l < n) {
        const uint4 k0 = ld_stream(sk), k1 = ld_stream(sk + half);
        const uint4 v0 = ld_stream(sv), v1 = ld_stream(sv + half);
        uint4 o0, o1;
        rotate_vec(k0, k1, c, s, o0, o1);
        st_row(ck, o0);
        st_row(ck + half, o1);
        st_row(cv, v0);
        st_row(cv + half, v1);
    }
}

constexpr int kTokPerThread = 4;   // tokens of a revisit each thread keeps in registers
constexpr int kPosTable = 1024;    // exact PCR positions tabulated per axis when span < this

// True when (|p - L| + L + 1) * Q < 2^52 (Q >= 1), i.e. every integer formed
// for p_hat = ((p - L) * Q + tail) / Q with 0 <= tail <= (L+1) * Q stays
// below 2^52 in magnitude, so that the integer products cannot overflow and
// the float64 division sees exact operands. Integer arithmetic only (GB300's
// float64 pipe is narrow and shared by every warp of an SM sub-partition).
__device__ __forceinline__ bool exact_ok(int64_t p_minus_l, int32_t L, uint64_t Q) {
    const int64_t lim = int64_t(1) << 62;
    if (p_minus_l <= -lim || p_minus_l >= lim) return false;
    const uint64_t a = uint64_t(p_minus_l < 0 ? -p_minus_l : p_minus_l) + uint64_t(L) + 1u;
    return __umul64hi(a, Q) == 0 && a * Q < (uint64_t(1) << 52);
}

// The denominator Q of the PCR position on an axis of the given span:
// (K+1) * span, or (K+1) (2 (K+1) with the centre reading) when the axis is
// degenerate (span <= 0).
__device__ __forceinline__ uint64_t pcr_denominator(int64_t K, int64_t span, bool center) {
    return span > 0 ? uint64_t(K + 1) * uint64_t(span) : uint64_t(center ? 2 * (K + 1) : K + 1);
}

__device__ __forceinline__ double pcr_position(int64_t p, int32_t L, int64_t K, int32_t c,
                                               int32_t lo, int32_t hi, bool center,
                                               uint32_t& err) {
    // The numerator and denominator are selected, not branched on, so that
    // the lanes of a warp (whose axes may be degenerate or not) share one
    // float64 division.
    const int64_t span = int64_t(hi) - int64_t(lo);
    const int64_t pl = p - L;
    const bool deg = span <= 0;  // degenerate axis: u = 0, or u = 1/2 with the centre reading
    const uint64_t Q = pcr_denominator(K, span, center);
    const int64_t tail = deg ? (center ? int64_t(L + 1) * (K + 1) : int64_t(L + 1))
                             : int64_t(L + 1) * (span + (K - 1) * (int64_t(c) - lo));
    if (exact_ok(pl, L, Q)) return exact_f64(pl * int64_t(Q) + tail) / exact_f64(int64_t(Q));
    err |= PRCR_ST_POS_RANGE;
    if (deg) return double(pl) + double(tail) / double(Q);
    const double u = double(int64_t(c) - lo) / double(span);
    return double(pl) + double(L + 1) * (1.0 + double(K - 1) * u) / double(K + 1);
}

// p + num / (K + 1), exact while representable (UIR).
__device__ __forceinline__ double uir_position(int64_t p, int64_t num, int64_t K, uint32_t& err) {
    if (exact_ok(p, 0, uint64_t(K + 1)))
        return exact_f64(p * (K + 1) + num) / exact_f64(K + 1);
    err |= PRCR_ST_POS_RANGE;
    return double(p) + double(num) / double(K + 1);
}

__device__ __forceinline__ void block_minmax(int (&mn)[3], int (&mx)[3], int* s_part) {
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int a = 0; a < 3; ++a) {
        mn[a] = __reduce_min_sync(0xffffffffu, mn[a]);
        mx[a] = __reduce_max_sync(0xffffffffu, mx[a]);
    }
    if (lane == 0) {
#pragma unroll
        for (int a = 0; a < 3; ++a) {
            s_part[warp * 6 + a] = mn[a];
            s_part[warp * 6 + 3 + a] = mx[a];
        }
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int a = 0; a < 3; ++a) {
            int vmn = lane < nwarps ? s_part[lane * 6 + a] : INT_MAX;
            int vmx = lane < nwarps ? s_part[lane * 6 + 3 + a] : INT_MIN;
            vmn = __reduce_min_sync(0xffffffffu, vmn);
            vmx = __reduce_max_sync(0xffffffffu, vmx);
            if (lane == 0) {
                s_part[32 * 6 + a] = vmn;
                s_part[32 * 6 + 3 + a] = vmx;
            }
        }
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < 3; ++a) {
        mn[a] = s_part[32 * 6 + a];
        mx[a] = s_part[32 * 6 + 3 + a];
    }
    __syncthreads();  // s_part is reused by the next revisit
}

struct RevisitCtx {
    int b, beg, end, t0;
    int64_t K, p, clen, capacity;
    int lo[3], hi[3];
    bool tab[3];
    bool center;
    bool inexact;  // some position of this revisit cannot be formed exactly
};

// |pos| < 2^31 (and not NaN), tested on the bits (no float64 instruction).
__device__ __forceinline__ bool pos_in_range(double pos) {
    return (static_cast<unsigned long long>(__double_as_longlong(pos)) & 0x7fffffffffffffffull) <
           0x41e0000000000000ull;
}

// Whether every position of revisit r is an exact rational with operands
// below 2^52 (the condition pcr_position / uir_position test per token; it
// depends only on the revisit: p, L, K and the axis spans). Needs r.lo/r.hi.
__device__ __forceinline__ void revisit_exactness(const PlanArgs& a, RevisitCtx& r) {
    bool ok = true;
    if (a.mode == PRCR_MODE_PCR) {
#pragma unroll
        for (int ax = 0; ax < 3; ++ax)
            ok = ok && exact_ok(r.p - a.L, a.L,
                                pcr_denominator(r.K, int64_t(r.hi[ax]) - int64_t(r.lo[ax]), r.center));
    } else if (a.mode == PRCR_MODE_UIR) {
        ok = exact_ok(r.p, 0, uint64_t(r.K + 1));
    }
    r.inexact = !ok;
}

// Physical destination row offset of `slot` (layer term excluded), or -1.
__device__ __forceinline__ int64_t dest_row(const PlanArgs& a, const RevisitCtx& r, int64_t slot,
                                            int32_t blk, uint32_t& err) {
    if (r.clen < 0 || slot >= r.capacity) {
        err |= PRCR_ST_CAPACITY;
        return -1;
    }
    if (a.cache_kind == PRCR_CACHE_CONTIGUOUS)
        return int64_t(r.b) * a.cache_seq_stride + slot * a.slot_stride;
    if (blk < 0 || blk >= a.n_blocks) {
        err |= PRCR_ST_NO_BLOCK;
        return -1;
    }
    const int64_t lb = slot / a.block_size;
    return int64_t(blk) * a.block_stride + (slot - lb * a.block_size) * a.slot_stride;
}

// Block id holding `slot` (paged caches), read early so the load overlaps others.
__device__ __forceinline__ int32_t block_of(const PlanArgs& a, const RevisitCtx& r, int64_t slot) {
    if (a.cache_kind != PRCR_CACHE_PAGED || r.clen < 0 || slot >= r.capacity) return -1;
    return a.block_table[int64_t(r.b) * a.bt_stride + slot / a.block_size];
}

__device__ __forceinline__ void load_coords(const int32_t* crd, int m, int n_tokens, int (&c)[3]) {
    if (m >= 0 && m < n_tokens) {
        const int32_t* q = crd + 3 * int64_t(m);
        c[0] = q[0];
        c[1] = q[1];
        c[2] = q[2];
    } else {
        c[0] = c[1] = c[2] = 0;
    }
}

// Reassigned position, store row, cache row and slot of token j of revisit
// r (m: its store index, c: its stored coordinate, blk: the block holding its
// slot). PCR positions come from the per-revisit table when it holds the
// axis (tab non-null and r.tab), else from one exact division each.
__device__ __forceinline__ void token_plan(const PlanArgs& a, const RevisitCtx& r,
                                           const double (*tab)[kPosTable], int j, int m,
                                           const int (&c)[3], int32_t blk, uint32_t& err,
                                           double (&pos)[3], int64_t& src, int64_t& dst,
                                           int64_t& slot) {
    slot = r.clen + (j - r.t0);
    src = 0;
    dst = -1;
    if (m < 0 || m >= a.n_tokens) {
        err |= PRCR_ST_IDX_RANGE;
        pos[0] = pos[1] = pos[2] = __longlong_as_double(0x7ff8000000000000LL);
        return;
    }
    switch (a.mode) {
        case PRCR_MODE_PCR:
#pragma unroll
            for (int ax = 0; ax < 3; ++ax)
                pos[ax] = (tab && r.tab[ax]) ? tab[ax][c[ax] - r.lo[ax]]
                                             : pcr_position(r.p, a.L, r.K, c[ax], r.lo[ax],
                                                            r.hi[ax], r.center, err);
            break;
        case PRCR_MODE_ORIGINAL:
#pragma unroll
            for (int ax = 0; ax < 3; ++ax) pos[ax] = double(c[ax]);
            break;
        case PRCR_MODE_UIR: {
            // p + (j' + 1) / (K + 1), j' the token's rank in its revisit
            const double v = uir_position(r.p, int64_t(j - r.beg + 1), r.K, err);
            pos[0] = pos[1] = pos[2] = v;
            break;
        }
        default: {  // PRCR_MODE_LPA: p + rank in sequence + 1
            const double v = double(r.p + (j - r.t0) + 1);
            pos[0] = pos[1] = pos[2] = v;
            break;
        }
    }
    src = int64_t(r.b) * a.store_seq_stride + int64_t(m) * a.store_token_stride;
    // The rotation reduces angles in 32.32 fixed point (|position| < 2^31),
    // and a position must be the correctly rounded exact value: otherwise the
    // status bit is set and the token's rows are skipped (its position
    // outputs keep the value computed).
    if (r.inexact || !(pos_in_range(pos[0]) && pos_in_range(pos[1]) && pos_in_range(pos[2]))) {
        err |= PRCR_ST_POS_RANGE;
        return;
    }
    dst = dest_row(a, r, slot, blk, err);
}

// Context of revisit r: its token range, sequence (the last b with
// seq_rev_off[b] <= r), the sequence's first token, text position, cache
// length and capacity. False (uniform over the CTA) when the offsets around
// r are inconsistent.
__device__ __forceinline__ bool revisit_ctx(const PlanArgs& a, int r, RevisitCtx& x) {
    x.beg = a.rev_tok_off[r];
    x.end = a.rev_tok_off[r + 1];
    int lo = 0, hi = a.n_seqs;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (a.seq_rev_off[mid] <= r) lo = mid; else hi = mid;
    }
    x.b = lo;
    const int r_first = a.seq_rev_off[x.b];
    bool ok = x.beg >= 0 && x.beg <= x.end && int64_t(x.end) <= a.total_k &&
              r_first <= r && r < a.seq_rev_off[x.b + 1] && r_first >= 0;
    x.t0 = ok ? a.rev_tok_off[r_first] : 0;
    ok = ok && x.t0 >= 0 && x.t0 <= x.beg;
    if (!ok) return false;
    x.K = x.end - x.beg;
    x.p = a.p_txt[x.b];
    x.clen = a.cache_len_in[x.b];
    x.center = (a.flags & PRCR_FLAG_DEGENERATE_CENTER) != 0;
    x.capacity = a.cache_kind == PRCR_CACHE_CONTIGUOUS ? int64_t(a.max_slots)
                                                       : int64_t(a.bt_stride) * a.block_size;
    x.inexact = false;
    return true;
}

}  // namespace prcr
