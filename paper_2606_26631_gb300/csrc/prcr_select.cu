// Attention-driven selection of the revisited set (Sec. 2.1, Eq. 3).
//
// The paper names the selection module and what it does (rank the visual
// tokens by relevance to the current decoding context, keep K of them) but
// not its formula. Reading implemented here: relevance of visual token m is
// the trigger query's attention on m at one layer, a softmax over the M
// visual tokens of RoPE(q_h, (p, p, p)) . RoPE(k_m, p_m) / sqrt(D) per query
// head h (GQA: head h reads KV head h / group), averaged over the heads. The
// K most relevant tokens (equal relevance: lower token index first) are
// written in ascending token order, one revisit per sequence, as the offsets
// and indices prcr_rebind_inject takes.
//
// Kernel 1 (logits): a CTA owns 16 tokens of one sequence and all KV heads;
// it rotates the sequence's query heads once into shared memory (pre-scaled
// by 1/sqrt(D)) and computes each token's cos/sin once; thread (token, KV
// head) rotates its raw key row on the fly and forms the logits of the
// group's query heads. Kernel 2 (select): a CTA per sequence reduces each
// head's softmax normaliser, averages the heads into the relevance (kept in
// shared memory), finds the K-th largest relevance with a 4-pass 8-bit radix
// select on the float bits (relevance >= 0, so bit order is value order),
// and compacts the selection in index order with block-wide scans.
#include <cmath>

#include "prcr_internal.h"

namespace prcr {
namespace {

constexpr double kTwoPiHi = 6.283185307179586;
constexpr double kTwoPiLo = 2.4492935982947064e-16;
constexpr double kInvTwoPi = 0.15915494309189535;
constexpr int kTokTile = 16;

__device__ __forceinline__ void sincos_reduced(double ang, float* s, float* c) {
    const double k = rint(ang * kInvTwoPi);
    double r = fma(-k, kTwoPiHi, ang);
    r = fma(-k, kTwoPiLo, r);
    sincosf(float(r), s, c);
}

__device__ __forceinline__ int pair_axis(int i, int layout, int st, int sh, int sw) {
    if (layout == PRCR_LAYOUT_SECTIONED) return i < st ? 0 : (i < st + sh ? 1 : 2);
    const int r = i % 3;
    if (r == 1 && i < 3 * sh) return 1;
    if (r == 2 && i < 3 * sw) return 2;
    return 0;
}

__global__ void __launch_bounds__(256) ads_logits_kernel(const __grid_constant__ SelectArgs a) {
    extern __shared__ __align__(16) float sm[];
    const int D = a.head_dim, P = D >> 1, Hq = a.n_q_heads, H = a.n_kv_heads;
    const int qs = D + 4;  // padded row strides
    const int cs = P + 4;
    float* q_s = sm;                 // [Hq][D + 4]
    float* cos_s = q_s + Hq * qs;    // [kTokTile][P + 4]
    float* sin_s = cos_s + kTokTile * cs;
    const int b = blockIdx.y;
    const int m0 = blockIdx.x * kTokTile;

    // the query sits at (p, p, p): pair i turns by p * inv_freq_i for every head
    __shared__ float s_qc[kMaxPairs], s_qs[kMaxPairs];
    const int64_t p = a.q_pos[b];
    for (int i = threadIdx.x; i < P; i += blockDim.x) sincos_reduced(double(p) * a.inv_freq[i], &s_qs[i], &s_qc[i]);
    __syncthreads();
    const uint16_t* qb = a.q + int64_t(b) * Hq * D;
    for (int e = threadIdx.x; e < Hq * P; e += blockDim.x) {
        const int hq = e / P, i = e - (e / P) * P;
        const float sn = s_qs[i], cn = s_qc[i];
        const float x = __uint_as_float(uint32_t(qb[hq * D + i]) << 16);
        const float y = __uint_as_float(uint32_t(qb[hq * D + i + P]) << 16);
        q_s[hq * qs + i] = fmaf(x, cn, -y * sn) * a.scale;
        q_s[hq * qs + i + P] = fmaf(y, cn, x * sn) * a.scale;
    }
    const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride;
    for (int e = threadIdx.x; e < kTokTile * P; e += blockDim.x) {
        const int t = e / P, i = e - (e / P) * P;
        const int m = m0 + t;
        float sn = 0.0f, cn = 1.0f;
        if (m < a.n_tokens) {
            const int ax = pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w);
            sincos_reduced(double(crd[3 * int64_t(m) + ax]) * a.inv_freq[i], &sn, &cn);
        }
        cos_s[t * cs + i] = cn;
        sin_s[t * cs + i] = sn;
    }
    __syncthreads();

    const int g = Hq / H;
    for (int e = threadIdx.x; e < kTokTile * H; e += blockDim.x) {
        const int t = e / H, kh = e - (e / H) * H;
        const int m = m0 + t;
        if (m >= a.n_tokens) continue;
        const uint16_t* kr = a.store_k + int64_t(b) * a.store_seq_stride +
                             int64_t(a.layer) * a.store_layer_stride +
                             int64_t(m) * a.store_token_stride + int64_t(kh) * D;
        float acc[8];
#pragma unroll
        for (int h = 0; h < 8; ++h) acc[h] = 0.0f;
        for (int i0 = 0; i0 < P; i0 += 8) {
            const uint4 lo = *reinterpret_cast<const uint4*>(kr + i0);
            const uint4 hi = *reinterpret_cast<const uint4*>(kr + i0 + P);
            const uint32_t lw[4] = {lo.x, lo.y, lo.z, lo.w};
            const uint32_t hw[4] = {hi.x, hi.y, hi.z, hi.w};
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = i0 + j;
                const uint32_t wl = lw[j >> 1], wh = hw[j >> 1];
                const float x = __uint_as_float((j & 1) ? (wl & 0xffff0000u) : (wl << 16));
                const float y = __uint_as_float((j & 1) ? (wh & 0xffff0000u) : (wh << 16));
                const float cn = cos_s[t * cs + i], sn = sin_s[t * cs + i];
                const float kx = fmaf(x, cn, -y * sn);
                const float ky = fmaf(y, cn, x * sn);
#pragma unroll
                for (int h = 0; h < 8; ++h) {
                    if (h < g) {
                        const float* qh = q_s + (kh * g + h) * qs;
                        acc[h] = fmaf(qh[i], kx, fmaf(qh[i + P], ky, acc[h]));
                    }
                }
            }
        }
#pragma unroll
        for (int h = 0; h < 8; ++h)
            if (h < g) a.logits[(int64_t(b) * Hq + kh * g + h) * a.n_tokens + m] = acc[h];
    }
}

// Block-wide exclusive scan of one int per thread; returns the total.
__device__ __forceinline__ int block_scan(int v, int* s_warp, int* out_excl) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < nw ? s_warp[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < nw) s_warp[lane] = w;  // inclusive prefix of warp totals
    }
    __syncthreads();
    const int total = s_warp[nw - 1];
    *out_excl = x - v + (warp > 0 ? s_warp[warp - 1] : 0);
    __syncthreads();
    return total;
}

__global__ void __launch_bounds__(1024) ads_select_kernel(const __grid_constant__ SelectArgs a) {
    extern __shared__ __align__(16) float rel[];  // [n_tokens]
    __shared__ float s_max[kSelectMaxQHeads], s_inv[kSelectMaxQHeads];
    __shared__ float s_red[64];
    __shared__ int s_warp[32];
    __shared__ unsigned int s_hist[256];
    __shared__ unsigned int s_prefix, s_kleft;
    const int b = blockIdx.x;
    const int M = a.n_tokens, Hq = a.n_q_heads;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const float* lg = a.logits + int64_t(b) * Hq * M;

    // 1. per query head: softmax max and normaliser over the M visual tokens
    for (int h = 0; h < Hq; ++h) {
        float mx = -INFINITY;
        for (int m = threadIdx.x; m < M; m += blockDim.x) mx = fmaxf(mx, lg[int64_t(h) * M + m]);
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if (lane == 0) s_red[warp] = mx;
        __syncthreads();
        if (threadIdx.x == 0) {
            float v = -INFINITY;
            for (int w = 0; w < nw; ++w) v = fmaxf(v, s_red[w]);
            s_max[h] = v;
        }
        __syncthreads();
        const float hm = s_max[h];
        float sum = 0.0f;
        for (int m = threadIdx.x; m < M; m += blockDim.x) sum += expf(lg[int64_t(h) * M + m] - hm);
#pragma unroll
        for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) s_red[32 + warp] = sum;
        __syncthreads();
        if (threadIdx.x == 0) {
            float v = 0.0f;
            for (int w = 0; w < nw; ++w) v += s_red[32 + w];
            s_inv[h] = 1.0f / (v * float(Hq));
        }
        __syncthreads();
    }
    // 2. relevance = mean over heads of the per-head softmax
    for (int m = threadIdx.x; m < M; m += blockDim.x) {
        float r = 0.0f;
        for (int h = 0; h < Hq; ++h) r = fmaf(expf(lg[int64_t(h) * M + m] - s_max[h]), s_inv[h], r);
        rel[m] = r;
        if (a.score_out) a.score_out[int64_t(b) * M + m] = r;
    }
    if (threadIdx.x == 0) {
        s_prefix = 0u;
        s_kleft = unsigned(a.k);
    }
    __syncthreads();

    // 3. radix select of the K-th largest relevance (bits of a float >= 0)
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += blockDim.x) s_hist[i] = 0u;
        __syncthreads();
        const unsigned int prefix = s_prefix;
        const unsigned int hi_mask = shift == 24 ? 0u : (0xffffffffu << (shift + 8));
        for (int m = threadIdx.x; m < M; m += blockDim.x) {
            const unsigned int key = __float_as_uint(rel[m]);
            if ((key & hi_mask) == prefix) atomicAdd(&s_hist[(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            unsigned int left = s_kleft, acc = 0u;
            int bin = 255;
            for (; bin > 0; --bin) {
                if (acc + s_hist[bin] >= left) break;
                acc += s_hist[bin];
            }
            s_kleft = left - acc;
            s_prefix = prefix | (unsigned(bin) << shift);
        }
        __syncthreads();
    }
    const unsigned int thr = s_prefix;   // the K-th largest key
    const int need_eq = int(s_kleft);    // how many keys equal to thr are taken

    // 4. ordered compaction: all keys > thr, then the first need_eq keys == thr
    const int per = (M + blockDim.x - 1) / blockDim.x;
    const int beg = threadIdx.x * per;
    const int end = min(M, beg + per);
    int n_eq = 0;
    for (int m = beg; m < end; ++m) n_eq += __float_as_uint(rel[m]) == thr;
    int eq_before = 0;
    block_scan(n_eq, s_warp, &eq_before);
    int n_sel = 0;
    {
        int e = eq_before;
        for (int m = beg; m < end; ++m) {
            const unsigned int key = __float_as_uint(rel[m]);
            if (key > thr) ++n_sel;
            else if (key == thr) { if (e < need_eq) ++n_sel; ++e; }
        }
    }
    int sel_before = 0;
    block_scan(n_sel, s_warp, &sel_before);
    int32_t* out = a.idx_out + int64_t(b) * a.k;
    {
        int e = eq_before, o = sel_before;
        for (int m = beg; m < end; ++m) {
            const unsigned int key = __float_as_uint(rel[m]);
            bool take = key > thr;
            if (key == thr) { take = e < need_eq; ++e; }
            if (take) out[o++] = m;
        }
    }
    if (threadIdx.x == 0) {
        a.rev_tok_off[b] = b * a.k;
        a.seq_rev_off[b] = b;
        if (b == gridDim.x - 1) {
            a.rev_tok_off[b + 1] = (b + 1) * a.k;
            a.seq_rev_off[b + 1] = b + 1;
        }
    }
}

}  // namespace

cudaError_t launch_select(const SelectArgs& a, int n_seqs, cudaStream_t stream) {
    const int D = a.head_dim, P = D / 2;
    const size_t smem1 = (size_t(a.n_q_heads) * (D + 4) + 2 * size_t(kTokTile) * (P + 4)) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(ads_logits_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         int(smem1));
    if (e != cudaSuccess) return e;
    const dim3 g1((a.n_tokens + kTokTile - 1) / kTokTile, n_seqs, 1);
    ads_logits_kernel<<<g1, 256, smem1, stream>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const size_t smem2 = size_t(a.n_tokens) * sizeof(float);
    e = cudaFuncSetAttribute(ads_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(smem2));
    if (e != cudaSuccess) return e;
    ads_select_kernel<<<n_seqs, 1024, smem2, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
