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
// Kernel 0 rotates each sequence's trigger queries once. Kernel 1 (logits):
// a CTA owns 256 / H (16..64) tokens of one sequence and all H KV heads, one
// thread per (token, KV head); it copies the rotated queries (pre-scaled by
// 1/sqrt(D)) into shared memory and computes each token's cos/sin once;
// thread (token, KV head) rotates its raw key row on the fly and forms the logits of the
// group's query heads, plus the tile's per-head softmax statistics (max, sum
// of exp). Kernel 2 (norm) merges the tiles' statistics into each head's
// normaliser; kernel 3 (relevance) averages every token's per-head softmax
// weight; kernel 4 (select), one CTA per sequence, finds the K-th largest
// relevance with a 4-pass 8-bit radix select on the float bits (relevance >=
// 0, so bit order is value order) and compacts the selection in index order
// with block-wide scans.
#include <cmath>

#include "prcr_internal.h"

namespace prcr {
namespace {

__device__ __forceinline__ int pair_axis(int i, int layout, int st, int sh, int sw) {
    if (layout == PRCR_LAYOUT_SECTIONED) return i < st ? 0 : (i < st + sh ? 1 : 2);
    const int r = i % 3;
    if (r == 1 && i < 3 * sh) return 1;
    if (r == 2 && i < 3 * sw) return 2;
    return 0;
}

// The trigger queries of each sequence, rotated at (p, p, p) (pair i turns by
// p * inv_freq_i for every head) and scaled by 1/sqrt(D), once per sequence.
__global__ void __launch_bounds__(256) ads_query_kernel(const __grid_constant__ SelectArgs a) {
    __shared__ float s_c[kMaxPairs], s_s[kMaxPairs];
    const int b = blockIdx.x;
    const int D = a.head_dim, P = D >> 1, Hq = a.n_q_heads;
    const int64_t p = a.q_pos[b];
    for (int i = threadIdx.x; i < P; i += blockDim.x) sincos_turns(double(p), a.turn_freq[i], &s_s[i], &s_c[i]);
    __syncthreads();
    const uint16_t* qb = a.q + int64_t(b) * Hq * D;
    float* qo = a.qrot + int64_t(b) * Hq * D;
    for (int e = threadIdx.x; e < Hq * P; e += blockDim.x) {
        const int hq = e / P, i = e - (e / P) * P;
        const float x = __uint_as_float(uint32_t(qb[hq * D + i]) << 16);
        const float y = __uint_as_float(uint32_t(qb[hq * D + i + P]) << 16);
        qo[hq * D + i] = fmaf(x, s_c[i], -y * s_s[i]) * a.scale;
        qo[hq * D + i + P] = fmaf(y, s_c[i], x * s_s[i]) * a.scale;
    }
}

// NV: upper bound of the 16-byte vectors in half a head row (head_dim / 16).
template <int NV>
__global__ void __launch_bounds__(256) ads_logits_kernel(const __grid_constant__ SelectArgs a) {
    extern __shared__ __align__(16) float sm[];
    const int D = a.head_dim, P = D >> 1, Hq = a.n_q_heads, H = a.n_kv_heads;
    const int T = a.tok_tile;
    const int qs = D + 4;  // padded row strides (multiples of 4: float4 rows)
    const int cs = P + 4;
    float* q_s = sm;                 // [Hq][D + 4]
    float* cos_s = q_s + Hq * qs;    // [T][P + 4]
    float* sin_s = cos_s + T * cs;
    float* lg_s = sin_s + T * cs;    // [Hq][T + 1] this tile's logits (padded rows)
    const int b = blockIdx.y;
    const int m0 = blockIdx.x * T;

    // rotated queries of the sequence (ads_query_kernel) and the tile's coordinates
    __shared__ int s_crd[3 * 64];
    {
        const float4* src = reinterpret_cast<const float4*>(a.qrot + int64_t(b) * Hq * D);
        const int nv = Hq * D / 4;
        // row of query head hq = kh * g + h is h * H + kh: the rows the 8 lanes of a
        // quarter-warp read together (same h, consecutive kh) fall in distinct banks
        const int g = Hq / H;
#pragma unroll 4
        for (int e = threadIdx.x; e < nv; e += blockDim.x) {
            const int hq = (4 * e) / D, d = 4 * e - hq * D;
            *reinterpret_cast<float4*>(q_s + ((hq % g) * H + hq / g) * qs + d) = src[e];
        }
        const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride + 3 * int64_t(m0);
        const int nc = 3 * min(T, a.n_tokens - m0);
        for (int e = threadIdx.x; e < nc; e += blockDim.x) s_crd[e] = crd[e];
    }
    __syncthreads();
    for (int e = threadIdx.x; e < T * P; e += blockDim.x) {
        const int t = e / P, i = e - (e / P) * P;
        const int m = m0 + t;
        float sn = 0.0f, cn = 1.0f;
        if (m < a.n_tokens) {
            const int ax = pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w);
            sincos_turns(double(s_crd[3 * t + ax]), a.turn_freq[i], &sn, &cn);
        }
        cos_s[t * cs + i] = cn;
        sin_s[t * cs + i] = sn;
    }
    __syncthreads();

    const int g = Hq / H;
    for (int e = threadIdx.x; e < T * H; e += blockDim.x) {
        const int t = e / H, kh = e - (e / H) * H;
        const int m = m0 + t;
        if (m >= a.n_tokens) continue;
        const uint16_t* kr = a.store_k + int64_t(b) * a.store_seq_stride +
                             int64_t(a.layer) * a.store_layer_stride +
                             int64_t(m) * a.store_token_stride + int64_t(kh) * D;
        const float4* c4 = reinterpret_cast<const float4*>(cos_s + t * cs);
        const float4* s4 = reinterpret_cast<const float4*>(sin_s + t * cs);
        float acc[8];
#pragma unroll
        for (int h = 0; h < 8; ++h) acc[h] = 0.0f;
        // the whole row is requested before any of it is used: one load latency
        uint4 klo[NV], khi[NV];
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            if (8 * v < P) {
                klo[v] = __ldg(reinterpret_cast<const uint4*>(kr + 8 * v));
                khi[v] = __ldg(reinterpret_cast<const uint4*>(kr + 8 * v + P));
            }
        }
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            if (8 * v >= P) break;
            const int i0 = 8 * v;
            const uint4 lo = klo[v];
            const uint4 hi = khi[v];
            const float4 ca = c4[i0 / 4], cb = c4[i0 / 4 + 1];
            const float4 sa = s4[i0 / 4], sb = s4[i0 / 4 + 1];
            const uint32_t lw[4] = {lo.x, lo.y, lo.z, lo.w};
            const uint32_t hw[4] = {hi.x, hi.y, hi.z, hi.w};
            const float cc[8] = {ca.x, ca.y, ca.z, ca.w, cb.x, cb.y, cb.z, cb.w};
            const float ss[8] = {sa.x, sa.y, sa.z, sa.w, sb.x, sb.y, sb.z, sb.w};
            float kx[8], ky[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const uint32_t wl = lw[j >> 1], wh = hw[j >> 1];
                const float x = __uint_as_float((j & 1) ? (wl & 0xffff0000u) : (wl << 16));
                const float y = __uint_as_float((j & 1) ? (wh & 0xffff0000u) : (wh << 16));
                kx[j] = fmaf(x, cc[j], -y * ss[j]);
                ky[j] = fmaf(y, cc[j], x * ss[j]);
            }
#pragma unroll
            for (int h = 0; h < 8; ++h) {
                if (h < g) {
                    const float4* qh = reinterpret_cast<const float4*>(q_s + (h * H + kh) * qs);
                    const float4 qa = qh[i0 / 4], qb2 = qh[i0 / 4 + 1];
                    const float4 qc = qh[(i0 + P) / 4], qd = qh[(i0 + P) / 4 + 1];
                    float r = acc[h];
                    r = fmaf(qa.x, kx[0], r); r = fmaf(qa.y, kx[1], r);
                    r = fmaf(qa.z, kx[2], r); r = fmaf(qa.w, kx[3], r);
                    r = fmaf(qb2.x, kx[4], r); r = fmaf(qb2.y, kx[5], r);
                    r = fmaf(qb2.z, kx[6], r); r = fmaf(qb2.w, kx[7], r);
                    r = fmaf(qc.x, ky[0], r); r = fmaf(qc.y, ky[1], r);
                    r = fmaf(qc.z, ky[2], r); r = fmaf(qc.w, ky[3], r);
                    r = fmaf(qd.x, ky[4], r); r = fmaf(qd.y, ky[5], r);
                    r = fmaf(qd.z, ky[6], r); r = fmaf(qd.w, ky[7], r);
                    acc[h] = r;
                }
            }
        }
#pragma unroll
        for (int h = 0; h < 8; ++h)
            if (h < g) {
                a.logits[(int64_t(b) * Hq + kh * g + h) * a.n_tokens + m] = acc[h];
                lg_s[(kh * g + h) * (T + 1) + t] = acc[h];
            }
    }
    __syncthreads();
    // this tile's softmax statistics per query head: max and sum of exp
    const int nt = min(T, a.n_tokens - m0);
    for (int hq = threadIdx.x; hq < Hq; hq += blockDim.x) {
        float mx = -INFINITY;
        for (int t = 0; t < nt; ++t) mx = fmaxf(mx, lg_s[hq * (T + 1) + t]);
        float sm2 = 0.0f;
        for (int t = 0; t < nt; ++t) sm2 += expf(lg_s[hq * (T + 1) + t] - mx);
        float* ts = a.tile_stats + ((int64_t(b) * Hq + hq) * a.n_tiles + blockIdx.x) * 2;
        ts[0] = mx;
        ts[1] = sm2;
    }
}

// Softmax normaliser of each (sequence, query head) from the tiles' statistics.
__global__ void __launch_bounds__(256) ads_norm_kernel(const __grid_constant__ SelectArgs a) {
    __shared__ float s_m[8], s_z[8];
    const int hq = blockIdx.x, b = blockIdx.y;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const float* ts = a.tile_stats + (int64_t(b) * a.n_q_heads + hq) * a.n_tiles * 2;
    float mx = -INFINITY;
    for (int i = threadIdx.x; i < a.n_tiles; i += blockDim.x) mx = fmaxf(mx, ts[2 * i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) s_m[warp] = mx;
    __syncthreads();
    mx = s_m[0];
    for (int w = 1; w < nw; ++w) mx = fmaxf(mx, s_m[w]);
    float z = 0.0f;
    for (int i = threadIdx.x; i < a.n_tiles; i += blockDim.x) z += ts[2 * i + 1] * expf(ts[2 * i] - mx);
#pragma unroll
    for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) s_z[warp] = z;
    __syncthreads();
    if (threadIdx.x == 0) {
        float zt = 0.0f;
        for (int w = 0; w < nw; ++w) zt += s_z[w];
        float* nrm = a.norm + (int64_t(b) * a.n_q_heads + hq) * 2;
        nrm[0] = mx;
        nrm[1] = 1.0f / (zt * float(a.n_q_heads));
    }
}

// Relevance of every token: mean over the query heads of its softmax weight.
__global__ void __launch_bounds__(256) ads_relevance_kernel(const __grid_constant__ SelectArgs a) {
    __shared__ float s_n[2 * kSelectMaxQHeads];
    const int b = blockIdx.y;
    const int Hq = a.n_q_heads, M = a.n_tokens;
    for (int i = threadIdx.x; i < 2 * Hq; i += blockDim.x) s_n[i] = a.norm[int64_t(b) * Hq * 2 + i];
    __syncthreads();
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M) return;
    const float* lg = a.logits + int64_t(b) * Hq * M + m;
    float r = 0.0f;
    for (int h = 0; h < Hq; ++h) r = fmaf(expf(lg[int64_t(h) * M] - s_n[2 * h]), s_n[2 * h + 1], r);
    a.rel[int64_t(b) * M + m] = r;
    if (a.score_out) a.score_out[int64_t(b) * M + m] = r;
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
    __shared__ int s_warp[32];
    __shared__ unsigned int s_hist[256];
    __shared__ unsigned int s_prefix, s_kleft;
    const int b = blockIdx.x;
    const int M = a.n_tokens;

    // relevance of this sequence's tokens (from the relevance kernel)
    const float* rs = a.rel + int64_t(b) * M;
    for (int m = threadIdx.x; m < M; m += blockDim.x) rel[m] = rs[m];
    if (threadIdx.x == 0) {
        s_prefix = 0u;
        s_kleft = unsigned(a.k);
    }
    __syncthreads();

    // 1. radix select of the K-th largest relevance (bits of a float >= 0)
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

    // 2. ordered compaction: all keys > thr, then the first need_eq keys == thr
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
    const size_t smem1 = (size_t(a.n_q_heads) * (D + 4) + 2 * size_t(a.tok_tile) * (P + 4) +
                          size_t(a.n_q_heads) * (a.tok_tile + 1)) * sizeof(float);
    const dim3 g1(a.n_tiles, n_seqs, 1);
    ads_query_kernel<<<n_seqs, 256, 0, stream>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (D <= 64) {
        e = cudaFuncSetAttribute(ads_logits_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem1));
        if (e == cudaSuccess) ads_logits_kernel<4><<<g1, 256, smem1, stream>>>(a);
    } else if (D <= 128) {
        e = cudaFuncSetAttribute(ads_logits_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem1));
        if (e == cudaSuccess) ads_logits_kernel<8><<<g1, 256, smem1, stream>>>(a);
    } else {
        e = cudaFuncSetAttribute(ads_logits_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem1));
        if (e == cudaSuccess) ads_logits_kernel<16><<<g1, 256, smem1, stream>>>(a);
    }
    if (e != cudaSuccess) return e;
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    ads_norm_kernel<<<dim3(a.n_q_heads, n_seqs, 1), 256, 0, stream>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    ads_relevance_kernel<<<dim3((a.n_tokens + 255) / 256, n_seqs, 1), 256, 0, stream>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const size_t smem2 = size_t(a.n_tokens) * sizeof(float);
    e = cudaFuncSetAttribute(ads_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(smem2));
    if (e != cudaSuccess) return e;
    ads_select_kernel<<<n_seqs, 1024, smem2, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
