// First decode step over the active cache (Sec. 3.3, Eq.
// "decode_with_active_cache"): for every sequence, layer and query head,
//   o = softmax(RoPE(q_raw, (p, p, p)) K_act^T / sqrt(D)) V_act
// over the sequence's cache slots [0, len), the revisited rows included.
//
// Work layout (memory-bound: every cached K/V row is read once per step).
// A CTA owns (sequence, layer, slot chunk). Its prologue rotates the layer's
// query heads at the text position (float64 angle reduced modulo 2*pi,
// float32 sincos), pre-scales them by 1/sqrt(D) into shared memory, and
// resolves the chunk's cache rows (block table for paged caches). Each warp
// then serves one KV head and the `group` query heads that share it (GQA):
// lane i holds D/32 consecutive dimensions, so every K or V row of the head
// is one fully coalesced warp load. S = 32 / GP slots are processed per
// iteration (GP = 4 for groups up to 4, else 8): each lane forms its
// partial dot products for all GP x S (head, slot) pairs, and a butterfly
// transpose-reduction (31 shuffles) leaves lane l with the complete logit of
// pair l. The online softmax then runs per head, and P V accumulates in
// float32 per lane. Chunks of one (sequence, layer) are merged by a second
// kernel from (max, sum, accumulator) partials when the sequence is split.
#include <cmath>

#include <cuda_bf16.h>

#include "prcr_internal.h"

namespace prcr {
namespace {

constexpr double kTwoPiHi = 6.283185307179586;
constexpr double kTwoPiLo = 2.4492935982947064e-16;
constexpr double kInvTwoPi = 0.15915494309189535;
constexpr unsigned kFull = 0xffffffffu;
constexpr int kDecodeThreads = 128;

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// EPL consecutive bf16 of a row as EPL / 2 packed words.
template <int EPL>
__device__ __forceinline__ void load_row(const uint16_t* p, uint32_t (&w)[EPL / 2]) {
    if constexpr (EPL == 2) {
        w[0] = __ldg(reinterpret_cast<const unsigned int*>(p));
    } else if constexpr (EPL == 4) {
        const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
        w[0] = v.x; w[1] = v.y;
    } else {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
        w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
    }
}

template <int GP, int EPL>
__global__ void __launch_bounds__(kDecodeThreads, 3) decode_kernel(const __grid_constant__ DecodeArgs a) {
    constexpr int S = 32 / GP;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int D = a.head_dim;
    const int P = D >> 1;
    const int Hq = a.n_q_heads;
    float* q_s = reinterpret_cast<float*>(smem_raw);
    int64_t* row_s = reinterpret_cast<int64_t*>(smem_raw + size_t(Hq) * D * sizeof(float));
    const int b = blockIdx.z;
    const int l = blockIdx.y;
    const int split = blockIdx.x;
    uint32_t err = 0;

    int64_t len = a.seq_len[b];
    if (len < 0 || len > a.capacity) {
        err |= PRCR_ST_CAPACITY;
        len = len < 0 ? 0 : a.capacity;
    }
    const int64_t s_begin = int64_t(split) * a.chunk;
    const int64_t s_end = min(len, s_begin + a.chunk);

    // Query heads of (b, l), rotated at (p, p, p) and scaled by 1/sqrt(D).
    // With the same position on every axis, pair i turns by p * inv_freq_i
    // whatever its band, so each pair's cos/sin serves all heads.
    __shared__ float s_cos[kMaxPairs], s_sin[kMaxPairs];
    const int64_t p = a.q_pos[b];
    for (int i = threadIdx.x; i < P; i += blockDim.x) {
        const double ang = double(p) * a.inv_freq[i];
        const double k = rint(ang * kInvTwoPi);
        double r = fma(-k, kTwoPiHi, ang);
        r = fma(-k, kTwoPiLo, r);
        sincosf(float(r), &s_sin[i], &s_cos[i]);
    }
    __syncthreads();
    const uint16_t* qb = a.q + (int64_t(b) * a.n_layers + l) * Hq * D;
    for (int e = threadIdx.x; e < Hq * P; e += blockDim.x) {
        const int hq = e / P;
        const int i = e - hq * P;
        const float sn = s_sin[i], cs = s_cos[i];
        const float x = __uint_as_float(uint32_t(qb[hq * D + i]) << 16);
        const float y = __uint_as_float(uint32_t(qb[hq * D + i + P]) << 16);
        q_s[hq * D + i] = fmaf(x, cs, -y * sn) * a.scale;
        q_s[hq * D + i + P] = fmaf(y, cs, x * sn) * a.scale;
    }
    // Cache rows of this chunk (layer term excluded), -1 when unmapped.
    for (int64_t s = s_begin + threadIdx.x; s < s_end; s += blockDim.x) {
        int64_t row;
        if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
            row = int64_t(b) * a.seq_stride + s * a.slot_stride;
        } else {
            const int64_t lb = s / a.block_size;
            const int32_t blk = a.block_table[int64_t(b) * a.bt_stride + lb];
            if (blk < 0 || blk >= a.n_blocks) {
                err |= PRCR_ST_NO_BLOCK;
                row = -1;
            } else {
                row = int64_t(blk) * a.block_stride + (s - lb * a.block_size) * a.slot_stride;
            }
        }
        row_s[s - s_begin] = row;
    }
    if (err) atomicOr(a.status, err);
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int g = a.group;
    const int my_h = lane / S;
    const int my_si = lane - my_h * S;
    const int64_t lstride = int64_t(l) * a.layer_stride;

    for (int kh = warp; kh < a.n_kv_heads; kh += nwarps) {
        float qf[GP][EPL];
#pragma unroll
        for (int h = 0; h < GP; ++h)
#pragma unroll
            for (int e = 0; e < EPL; ++e)
                qf[h][e] = h < g ? q_s[(kh * g + h) * D + lane * EPL + e] : 0.0f;
        float m[GP], lsum[GP], acc[GP][EPL];
#pragma unroll
        for (int h = 0; h < GP; ++h) {
            m[h] = -INFINITY;
            lsum[h] = 0.0f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) acc[h][e] = 0.0f;
        }
        const uint16_t* kbase = a.cache_k + lstride + int64_t(kh) * D + lane * EPL;
        const uint16_t* vbase = a.cache_v + lstride + int64_t(kh) * D + lane * EPL;

        // Software pipeline: the K/V rows of the next S slots are requested
        // before the current S slots are reduced, so every warp keeps its
        // loads in flight while it runs the shuffle and softmax work.
        uint32_t kn[S][EPL / 2], vn[S][EPL / 2];
        bool okn[S];
        auto fetch = [&](int64_t s0) {
#pragma unroll
            for (int si = 0; si < S; ++si) {
                const int64_t s = s0 + si;
                const int64_t row = s < s_end ? row_s[s - s_begin] : -1;
                okn[si] = row >= 0;
                if (okn[si]) {
                    load_row<EPL>(kbase + row, kn[si]);
                    load_row<EPL>(vbase + row, vn[si]);
                } else {
#pragma unroll
                    for (int w = 0; w < EPL / 2; ++w) kn[si][w] = vn[si][w] = 0u;
                }
            }
        };
        if (s_begin < s_end) fetch(s_begin);
        for (int64_t s0 = s_begin; s0 < s_end; s0 += S) {
            uint32_t kw[S][EPL / 2], vw[S][EPL / 2];
            bool ok[S];
#pragma unroll
            for (int si = 0; si < S; ++si) {
                ok[si] = okn[si];
#pragma unroll
                for (int w = 0; w < EPL / 2; ++w) {
                    kw[si][w] = kn[si][w];
                    vw[si][w] = vn[si][w];
                }
            }
            if (s0 + S < s_end) fetch(s0 + S);
            // partial dot products of this lane's dimensions, index h * S + si
            float val[32];
#pragma unroll
            for (int h = 0; h < GP; ++h)
#pragma unroll
                for (int si = 0; si < S; ++si) {
                    float d = 0.0f;
#pragma unroll
                    for (int w = 0; w < EPL / 2; ++w) {
                        d = fmaf(qf[h][2 * w], bf16_lo(kw[si][w]), d);
                        d = fmaf(qf[h][2 * w + 1], bf16_hi(kw[si][w]), d);
                    }
                    val[h * S + si] = d;
                }
            // butterfly transpose-reduction: lane l ends with the full sum of index l
#pragma unroll
            for (int k = 16; k >= 1; k >>= 1) {
                const bool upper = (lane & k) != 0;
#pragma unroll
                for (int i = 0; i < k; ++i) {
                    const float send = upper ? val[i] : val[i + k];
                    const float keep = upper ? val[i + k] : val[i];
                    val[i] = keep + __shfl_xor_sync(kFull, send, k);
                }
            }
            bool my_ok = false;
#pragma unroll
            for (int si = 0; si < S; ++si)
                if (si == my_si) my_ok = ok[si];
            const float logit = (my_h < g && my_ok) ? val[0] : -INFINITY;

            // online softmax per head (each head's S lanes form an aligned segment)
            float mx = logit;
#pragma unroll
            for (int o = 1; o < S; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
            float mnew[GP], alpha[GP];
            float my_m = -INFINITY;
#pragma unroll
            for (int h = 0; h < GP; ++h) {
                const float cm = __shfl_sync(kFull, mx, h * S);
                mnew[h] = fmaxf(m[h], cm);
                alpha[h] = mnew[h] == -INFINITY ? 1.0f : expf(m[h] - mnew[h]);
                if (h == my_h) my_m = mnew[h];
            }
            const float pl = logit == -INFINITY ? 0.0f : expf(logit - my_m);
            float ps = pl;
#pragma unroll
            for (int o = 1; o < S; o <<= 1) ps += __shfl_xor_sync(kFull, ps, o);
#pragma unroll
            for (int h = 0; h < GP; ++h) {
                const float hs = __shfl_sync(kFull, ps, h * S);
                lsum[h] = lsum[h] * alpha[h] + hs;
                m[h] = mnew[h];
#pragma unroll
                for (int e = 0; e < EPL; ++e) acc[h][e] *= alpha[h];
            }
#pragma unroll
            for (int h = 0; h < GP; ++h)
#pragma unroll
                for (int si = 0; si < S; ++si) {
                    const float pw = __shfl_sync(kFull, pl, h * S + si);
#pragma unroll
                    for (int w = 0; w < EPL / 2; ++w) {
                        acc[h][2 * w] = fmaf(pw, bf16_lo(vw[si][w]), acc[h][2 * w]);
                        acc[h][2 * w + 1] = fmaf(pw, bf16_hi(vw[si][w]), acc[h][2 * w + 1]);
                    }
                }
        }

#pragma unroll
        for (int h = 0; h < GP; ++h) {
            if (h >= g) break;
            const int hq = kh * g + h;
            const int64_t o_idx = (int64_t(b) * a.n_layers + l) * Hq + hq;
            if (a.splits == 1) {
                const float inv = lsum[h] > 0.0f ? 1.0f / lsum[h] : 0.0f;
#pragma unroll
                for (int e = 0; e < EPL; ++e) a.out[o_idx * D + lane * EPL + e] = acc[h][e] * inv;
            } else {
                float* part = a.partial + (o_idx * a.splits + split) * (D + 2);
#pragma unroll
                for (int e = 0; e < EPL; ++e) part[lane * EPL + e] = acc[h][e];
                if (lane == 0) {
                    part[D] = m[h];
                    part[D + 1] = lsum[h];
                }
            }
        }
    }
}

// Merge the chunks of one (sequence, layer, query head): thread d owns one dimension.
__global__ void __launch_bounds__(256) decode_merge_kernel(const __grid_constant__ DecodeArgs a) {
    const int D = a.head_dim;
    const int64_t o_idx = blockIdx.x;
    const float* part = a.partial + o_idx * a.splits * (D + 2);
    float M = -INFINITY;
    for (int s = 0; s < a.splits; ++s) M = fmaxf(M, part[s * (D + 2) + D]);
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
        float num = 0.0f, den = 0.0f;
        for (int s = 0; s < a.splits; ++s) {
            const float ms = part[s * (D + 2) + D];
            if (ms == -INFINITY) continue;
            const float w = expf(ms - M);
            num = fmaf(w, part[s * (D + 2) + d], num);
            den = fmaf(w, part[s * (D + 2) + D + 1], den);
        }
        a.out[o_idx * D + d] = den > 0.0f ? num / den : 0.0f;
    }
}

template <int GP>
cudaError_t launch_gp(const DecodeArgs& a, dim3 grid, size_t smem, cudaStream_t stream) {
    switch (a.head_dim) {
        case 64: decode_kernel<GP, 2><<<grid, kDecodeThreads, smem, stream>>>(a); break;
        case 128: decode_kernel<GP, 4><<<grid, kDecodeThreads, smem, stream>>>(a); break;
        default: decode_kernel<GP, 8><<<grid, kDecodeThreads, smem, stream>>>(a); break;
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs& a, int gp, dim3 grid, size_t smem,
                          cudaStream_t stream) {
    // groups of 1, 2 and 4 query heads run as 4 (padded) heads x 8 slots per
    // warp iteration, groups of 5..8 as 8 heads x 4 slots
    const cudaError_t e = gp <= 4 ? launch_gp<4>(a, grid, smem, stream)
                                  : launch_gp<8>(a, grid, smem, stream);
    if (e != cudaSuccess || a.splits == 1) return e;
    const unsigned n = unsigned(int64_t(grid.z) * a.n_layers * a.n_q_heads);
    decode_merge_kernel<<<n, a.head_dim < 256 ? a.head_dim : 256, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
