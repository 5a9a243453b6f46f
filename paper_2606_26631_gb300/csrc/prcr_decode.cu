// First decode step over the active cache (Sec. 3.3, Eq.
// "decode_with_active_cache"): for every sequence, layer and query head,
//   o = softmax(RoPE(q_raw, (p, p, p)) K_act^T / sqrt(D)) V_act
// over the sequence's cache slots [0, len), the revisited rows included.
//
// Work layout (memory-bound: every cached K/V row is read once per step).
// A CTA owns (sequence, layer, slot chunk). Its prologue rotates the layer's
// query heads at the text position (angle reduced modulo a turn in fixed
// point, float32 sincos), pre-scales them by 1/sqrt(D) into shared memory, and
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

#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kDecodeThreads = 128;


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
    pdl_allow();
    pdl_wait();

    int64_t len = a.seq_len[b];
    if (len < 0 || len > a.capacity) {
        err |= PRCR_ST_CAPACITY;
        len = len < 0 ? 0 : a.capacity;
    }
    if (len > int64_t(a.splits) * a.chunk) {  // above the host's max_len: past the split
        err |= PRCR_ST_CAPACITY;
        len = int64_t(a.splits) * a.chunk;
    }
    // A query position beyond the fixed-point angle reduction (|p| >= 2^31)
    // is reported and the sequence attends to nothing: its output is zeros.
    const int64_t p = a.q_pos[b];
    if (p <= -2147483648LL || p >= 2147483648LL) {
        err |= PRCR_ST_POS_RANGE;
        len = 0;
    }
    const int64_t s_begin = int64_t(split) * a.chunk;
    const int64_t s_end = min(len, s_begin + a.chunk);

    // Query heads of (b, l), rotated at (p, p, p) and scaled by 1/sqrt(D).
    // With the same position on every axis, pair i turns by p * inv_freq_i
    // whatever its band, so each pair's cos/sin serves all heads.
    __shared__ float s_cos[kMaxPairs], s_sin[kMaxPairs];
    for (int i = threadIdx.x; i < P; i += blockDim.x) {
        sincos_turns(double(p), a.turn_freq[i], &s_sin[i], &s_cos[i]);
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
                        d = fmaf(qf[h][2 * w], lo_f32(kw[si][w]), d);
                        d = fmaf(qf[h][2 * w + 1], hi_f32(kw[si][w]), d);
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
                        acc[h][2 * w] = fmaf(pw, lo_f32(vw[si][w]), acc[h][2 * w]);
                        acc[h][2 * w + 1] = fmaf(pw, hi_f32(vw[si][w]), acc[h][2 * w + 1]);
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

// ---------------------------------------------------------------------------
// Tensor-core variant (head_dim 64 and 128), mma.sync m16n8k16 bf16 -> fp32.
//
// A warp serves one KV head and its group of g <= 8 query heads over 16 slots
// per iteration; the next 16 slots' K rows (registers) and V rows (shared
// memory) are requested right after the current QK, so they are in flight
// during the softmax and P V of the current slots.
//   QK:  S^T (16 slots x 8 heads, columns >= g zero) = K (16 slots x 16 dims)
//        x Q^T, D/16 k-steps: the slots fill all 16 MMA rows (with the heads
//        as rows only g of 16 would be used, and two n-tiles of 8 slots take
//        twice the MMAs). The dot product does not depend on the order of the
//        dimensions, so k-step j of lane group t uses the four dimensions
//        t*D/4 + 4j .. +3: each lane then loads its two slots' (g and g + 8)
//        64 contiguous bytes (D = 128) straight into A fragments, and the
//        query's fragments are the B operand. Lane (g, t) holds slots g and
//        g + 8 of heads 2t, 2t+1, so it keeps those two heads' online-softmax
//        state (reduced over the eight lanes of one t).
//   PV:  O^T (16 dims x 8 heads) += V^T (16 dims x 16 slots) x P^T (16 slots x
//        8 heads): P^T's B fragments are S^T's 8 x 8 blocks transposed in
//        registers (movmatrix); O^T's columns are the lane's own heads 2t,
//        2t+1. V tiles are staged in shared memory with cp.async
//        (double-buffered) and read as A fragments with ldmatrix.trans.
// bf16 operands hold only 8 significant bits, so the float32 query and the
// float32 probabilities are each split into a bf16 head and a bf16 remainder
// (two MMAs each): products stay exact and the result keeps ~16 bits per
// operand, float32-accumulated. K and V are bf16 already and enter exactly.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}

// Transpose of an 8 x 8 matrix of 16-bit values held as mma fragments
// (lane 4 r + c holds row r, columns 2c and 2c + 1): afterwards the lane holds
// row r, columns 2c and 2c + 1 of the transpose.
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

// One CTA per (sequence, layer, chunk) takes all KV heads of the layer, its
// warps looping over them (small batches take decode_ring_kernel below).
template <int D>
__global__ void __launch_bounds__(kDecodeThreads, 3)
    decode_mma_kernel(const __grid_constant__ DecodeArgs a) {
    constexpr int KS = D / 16;     // k-steps of QK, m-tiles of PV
    constexpr int LV = D / 32;     // 16-byte K loads per lane per slot
    constexpr int PITCH = D + 8;   // bf16 per staged V row (pad: conflict-free ldmatrix)
    constexpr int VCH = D / 8;     // 16-byte chunks per V row
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int Hq = a.n_q_heads;
    const int P = D / 2;
    float* q_s = reinterpret_cast<float*>(smem_raw);
    uint16_t* vbuf = reinterpret_cast<uint16_t*>(smem_raw + size_t(Hq) * D * sizeof(float));
    const int b = blockIdx.z;
    const int l = blockIdx.y;
    const int split = blockIdx.x, kh0 = 0, kh1 = a.n_kv_heads;
    uint32_t err = 0;
    pdl_allow();

    // Requests that do not depend on the sequence length go out first: this
    // CTA's query rows, and (contiguous caches) its first tile's K and V rows,
    // are prefetched to L2 while the length and position load.
    {
        const char* qrow = reinterpret_cast<const char*>(
            a.q + ((int64_t(b) * a.n_layers + l) * Hq + kh0 * a.group) * D);
        const int qbytes = (kh1 - kh0) * a.group * D * 2;
        for (int o = threadIdx.x * 128; o < qbytes; o += blockDim.x * 128) prefetch_l2(qrow + o);
        if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
            const int64_t s = int64_t(split) * a.chunk + (threadIdx.x & 15);
            const int kh = kh0 + ((threadIdx.x >> 4) & 3);
            if (s < a.capacity && kh < kh1) {
                const int64_t row = int64_t(b) * a.seq_stride + s * a.slot_stride +
                                    int64_t(l) * a.layer_stride + int64_t(kh) * D;
                const uint16_t* base = (threadIdx.x & 64) ? a.cache_v : a.cache_k;
#pragma unroll
                for (int c = 0; c < D * 2; c += 128) prefetch_l2(base + row + c / 2);
            }
        }
    }

    pdl_wait();
    const int64_t p = a.q_pos[b];  // requested together with the length
    int64_t len = a.seq_len[b];
    if (len < 0 || len > a.capacity) {
        err |= PRCR_ST_CAPACITY;
        len = len < 0 ? 0 : a.capacity;
    }
    if (len > int64_t(a.splits) * a.chunk) {  // above the host's max_len: past the split
        err |= PRCR_ST_CAPACITY;
        len = int64_t(a.splits) * a.chunk;
    }
    // A query position beyond the fixed-point angle reduction (|p| >= 2^31)
    // is reported and the sequence attends to nothing: its output is zeros.
    if (p <= -2147483648LL || p >= 2147483648LL) {
        err |= PRCR_ST_POS_RANGE;
        len = 0;
    }
    const int64_t s_begin = int64_t(split) * a.chunk;
    const int64_t s_end = min(len, s_begin + a.chunk);
    __shared__ __align__(16) float s_cos[kMaxPairs];
    __shared__ __align__(16) float s_sin[kMaxPairs];
    for (int i = threadIdx.x; i < P; i += blockDim.x) {
        sincos_turns(double(p), a.turn_freq[i], &s_sin[i], &s_cos[i]);
    }
    __syncthreads();
    const uint16_t* qb = a.q + (int64_t(b) * a.n_layers + l) * Hq * D;
    // the query heads of this CTA's KV heads, eight rotation pairs per thread
    // (two 16-byte loads when the query rows are 16-byte aligned)
    const int e_beg = 0, e_end = Hq * P;
    const bool q16 = (reinterpret_cast<uintptr_t>(a.q) & 15) == 0;
    for (int e = e_beg + 8 * threadIdx.x; e < e_end; e += 8 * blockDim.x) {
        const int hq = e / P;
        const int i = e - hq * P;  // a multiple of 8: P is 32 or 64
        const uint16_t* qx = qb + hq * D + i;
        uint32_t wx[4], wy[4];
        if (q16) {
            const uint4 x4 = __ldg(reinterpret_cast<const uint4*>(qx));
            const uint4 y4 = __ldg(reinterpret_cast<const uint4*>(qx + P));
            wx[0] = x4.x; wx[1] = x4.y; wx[2] = x4.z; wx[3] = x4.w;
            wy[0] = y4.x; wy[1] = y4.y; wy[2] = y4.z; wy[3] = y4.w;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                wx[u] = uint32_t(qx[2 * u]) | (uint32_t(qx[2 * u + 1]) << 16);
                wy[u] = uint32_t(qx[P + 2 * u]) | (uint32_t(qx[P + 2 * u + 1]) << 16);
            }
        }
        float rx[8], ry[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const float x = __uint_as_float((u & 1) ? (wx[u >> 1] & 0xffff0000u) : (wx[u >> 1] << 16));
            const float y = __uint_as_float((u & 1) ? (wy[u >> 1] & 0xffff0000u) : (wy[u >> 1] << 16));
            const float sn = s_sin[i + u], cs = s_cos[i + u];
            rx[u] = fmaf(x, cs, -y * sn) * a.scale;
            ry[u] = fmaf(y, cs, x * sn) * a.scale;
        }
        float4* ox = reinterpret_cast<float4*>(q_s + hq * D + i);
        float4* oy = reinterpret_cast<float4*>(q_s + hq * D + i + P);
        ox[0] = make_float4(rx[0], rx[1], rx[2], rx[3]);
        ox[1] = make_float4(rx[4], rx[5], rx[6], rx[7]);
        oy[0] = make_float4(ry[0], ry[1], ry[2], ry[3]);
        oy[1] = make_float4(ry[4], ry[5], ry[6], ry[7]);
    }
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int gid = lane >> 2;
    const int t = lane & 3;
    const int g = a.group;
    const int64_t lstride = int64_t(l) * a.layer_stride;
    uint16_t* wv = vbuf + size_t(warp) * 2 * 16 * PITCH;
    const uint32_t wv_s = uint32_t(__cvta_generic_to_shared(wv));

    for (int kh = kh0 + warp; kh < kh1; kh += nwarps) {
        // the query B fragments (columns = heads of the group; columns >= g are zero)
        uint32_t qh[KS][2], ql[KS][2];
        {
            const bool hv = gid < g;
            const float* qr = q_s + (kh * g + (hv ? gid : 0)) * D + t * (D / 4);
#pragma unroll
            for (int j = 0; j < KS; ++j) {
                const float x0 = hv ? qr[4 * j] : 0.0f, x1 = hv ? qr[4 * j + 1] : 0.0f;
                const float x2 = hv ? qr[4 * j + 2] : 0.0f, x3 = hv ? qr[4 * j + 3] : 0.0f;
                split_bf16x2(x0, x1, qh[j][0], ql[j][0]);
                split_bf16x2(x2, x3, qh[j][1], ql[j][1]);
            }
        }
        float o[KS][4];
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.0f;
        float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.0f, 0.0f};  // heads 2t, 2t + 1
        const uint16_t* kbase = a.cache_k + lstride + int64_t(kh) * D;
        const uint16_t* vbase = a.cache_v + lstride + int64_t(kh) * D;

        uint4 kn[2][LV];
        uint32_t mask_n = 0u;
        // Block id of slot s0 + (lane & 15) (paged caches), requested before
        // the current tile's QK so that its latency hides behind the MMAs.
        auto block_of = [&](int64_t s0) -> int32_t {
            const int64_t s = s0 + (lane & 15);
            if (a.cache_kind != PRCR_CACHE_PAGED || s >= s_end) return 0;
            return a.block_table[int64_t(b) * a.bt_stride + s / a.block_size];
        };
        // Requests tile s0 (16 slots): K rows into registers, V rows into stage st.
        auto fetch = [&](int64_t s0, int st, int32_t blk) {
            const int64_t s = s0 + (lane & 15);
            int64_t row = -1;
            if (s < s_end) {
                if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
                    row = int64_t(b) * a.seq_stride + s * a.slot_stride;
                } else if (blk < 0 || blk >= a.n_blocks) {
                    err |= PRCR_ST_NO_BLOCK;
                } else {
                    const int64_t lb = s / a.block_size;
                    row = int64_t(blk) * a.block_stride + (s - lb * a.block_size) * a.slot_stride;
                }
            }
            mask_n = __ballot_sync(kFull, row >= 0) & 0xffffu;
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const int64_t rr = __shfl_sync(kFull, row, nt * 8 + gid);
#pragma unroll
                for (int u = 0; u < LV; ++u)
                    kn[nt][u] = rr >= 0 ? __ldg(reinterpret_cast<const uint4*>(kbase + rr + t * (D / 4) + 8 * u))
                                        : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int i = 0; i < (16 * VCH) / 32; ++i) {
                const int c = lane + 32 * i;
                const int slot = c / VCH;
                const int piece = c - slot * VCH;
                const int64_t rr = __shfl_sync(kFull, row, slot);
                const uint32_t dst = wv_s + uint32_t(((st * 16 + slot) * PITCH + piece * 8) * 2);
                cp_async16(dst, rr >= 0 ? vbase + rr + piece * 8 : vbase, rr >= 0 ? 16 : 0);
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
        };

        int st = 0;
        if (s_begin < s_end) fetch(s_begin, 0, block_of(s_begin));
        for (int64_t s0 = s_begin; s0 < s_end; s0 += 16, st ^= 1) {
            const uint32_t mask = mask_n;
            const bool more = s0 + 16 < s_end;
            const int32_t blk_next = more ? block_of(s0 + 16) : 0;

            // S^T (16 slots x 8 columns = the group's query heads, columns >= g
            // zero) = K Q^T: this lane's slots gid (kn[0]) and 8 + gid (kn[1])
            // are the A rows, the query fragments the B operand unchanged; the
            // query's head and remainder products in two chains
            float sh[4] = {0.0f, 0.0f, 0.0f, 0.0f}, sl_[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int j = 0; j < KS; ++j) {
                const uint4& w0 = kn[0][j >> 1];
                const uint4& w1 = kn[1][j >> 1];
                const uint32_t a0 = (j & 1) ? w0.z : w0.x, a2 = (j & 1) ? w0.w : w0.y;
                const uint32_t a1 = (j & 1) ? w1.z : w1.x, a3 = (j & 1) ? w1.w : w1.y;
                mma_16816(sh, a0, a1, a2, a3, qh[j][0], qh[j][1]);
                mma_16816(sl_, a0, a1, a2, a3, ql[j][0], ql[j][1]);
            }
            // the next tile's K and V are in flight during the softmax and P V
            if (more) fetch(s0 + 16, st ^ 1, blk_next);

            // online softmax of this lane's heads 2t, 2t + 1 (columns) over the
            // 16 slots: the eight lanes of one t hold them, two slots each
            const bool oka = (mask >> gid) & 1u, okb = (mask >> (8 + gid)) & 1u;
            float pa[2], pb[2], alpha[2];
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const float va = oka ? sh[hh] + sl_[hh] : -INFINITY;
                const float vb = okb ? sh[2 + hh] + sl_[2 + hh] : -INFINITY;
                float mx = fmaxf(va, vb);
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 4));
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 8));
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 16));
                const float m_new = fmaxf(m_run[hh], mx);
                // arguments are <= 0: __expf's error (a few ulp) is far inside
                // the float32 accumulation's
                alpha[hh] = m_new == -INFINITY ? 1.0f : __expf(m_run[hh] - m_new);
                pa[hh] = va == -INFINITY ? 0.0f : __expf(va - m_new);
                pb[hh] = vb == -INFINITY ? 0.0f : __expf(vb - m_new);
                float ps = pa[hh] + pb[hh];
                ps += __shfl_xor_sync(kFull, ps, 4);
                ps += __shfl_xor_sync(kFull, ps, 8);
                ps += __shfl_xor_sync(kFull, ps, 16);
                l_run[hh] = l_run[hh] * alpha[hh] + ps;
                m_run[hh] = m_new;
            }
            // O^T columns are heads 2t, 2t + 1: this lane's own factors
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                o[mt][0] *= alpha[0]; o[mt][1] *= alpha[1]; o[mt][2] *= alpha[0]; o[mt][3] *= alpha[1];
            }
            // P^T as B fragments: the 8 x 8 blocks (slots 0..7 | 8..15) x heads
            // held as (slot gid; heads 2t, 2t + 1) are transposed in registers
            uint32_t m1h, m1l, m2h, m2l;
            split_bf16x2(pa[0], pa[1], m1h, m1l);
            split_bf16x2(pb[0], pb[1], m2h, m2l);
            const uint32_t pb0h = movmatrix_trans(m1h), pb1h = movmatrix_trans(m2h);
            const uint32_t pb0l = movmatrix_trans(m1l), pb1l = movmatrix_trans(m2l);

            // O^T += V^T P^T
            if (more) asm volatile("cp.async.wait_group 1;" ::: "memory");
            else asm volatile("cp.async.wait_group 0;" ::: "memory");
            __syncwarp();
            const int lslot = (lane & 7) + ((lane >> 4) & 1) * 8;
            const int ldim = ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                uint32_t r0, r1, r2, r3;
                const uint32_t addr = wv_s + uint32_t(((st * 16 + lslot) * PITCH + mt * 16 + ldim) * 2);
                asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                             : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                             : "r"(addr));
                mma_16816(o[mt], r0, r1, r2, r3, pb0h, pb1h);
                mma_16816(o[mt], r0, r1, r2, r3, pb0l, pb1l);
            }
            __syncwarp();
        }

        // heads 2t, 2t+1 of this lane's O^T columns
        const float l0 = l_run[0], l1 = l_run[1], m0 = m_run[0], m1 = m_run[1];
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int h = 2 * t + hh;
            if (h >= g) continue;
            const int64_t o_idx = (int64_t(b) * a.n_layers + l) * Hq + kh * g + h;
            const float lh = hh ? l1 : l0;
            if (a.splits == 1) {
                const float inv = lh > 0.0f ? 1.0f / lh : 0.0f;
                float* out = a.out + o_idx * D;
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    out[mt * 16 + gid] = o[mt][hh] * inv;
                    out[mt * 16 + gid + 8] = o[mt][2 + hh] * inv;
                }
            } else {
                float* part = a.partial + (o_idx * a.splits + split) * (D + 2);
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    part[mt * 16 + gid] = o[mt][hh];
                    part[mt * 16 + gid + 8] = o[mt][2 + hh];
                }
                if (gid == 0) {
                    part[D] = hh ? m1 : m0;
                    part[D + 1] = lh;
                }
            }
        }
    }
    if (err) atomicOr(a.status, err);
}

// Small batches (a grid that would not fill the GPU a few times over): a CTA
// of kRingWarps warps takes one (sequence, layer, chunk) and up to kRingWarps
// KV heads, one per warp, and the chunk is sized so that the grid runs as
// about one wave of kDecodeRingCtasPerSm CTAs per SM. Each warp streams its
// chunk's tiles of 16 slots through a ring of kRingStages stages in shared
// memory: K and V are both staged by cp.async, kRingStages - 1 tiles ahead
// of the one being computed, and the first of them are requested before the
// prologue's barriers (a barrier waits for a thread's plain loads in flight,
// not for its async copies). Two stages keep the CTA's shared memory at
// 66 KB (three CTAs, twelve warps per SM); more warps per SM hide more of
// each warp's latency chain than a deeper ring would.
// The arithmetic is that of decode_mma_kernel (S^T = K Q^T, O^T += V^T P^T,
// the same online softmax); the key dimensions are permuted per lane group as
// there, here with lane group t reading 16-byte chunks t, t + 4, ... of its
// slot's K row, and chunk c of slot s is stored at c ^ 4 (s & 1) so that
// those reads are free of bank conflicts.
constexpr int kRingWarps = kDecodeRingWarps;
constexpr int kRingStages = 2;
// rounds of eight query pairs per thread: the CTA's query heads are at most
// kRingWarps * 8 (a GQA group of 8), i.e. kRingWarps * 8 * D / 2 pairs
constexpr int kRingQRounds = 2;

template <int D>
__global__ void __launch_bounds__(kRingWarps * 32, kDecodeRingCtasPerSm)
    decode_ring_kernel(const __grid_constant__ DecodeArgs a) {
    constexpr int KS = D / 16;      // k-steps of QK, m-tiles of PV
    constexpr int LV = D / 32;      // 16-byte K chunks per lane per slot
    constexpr int NCH = D / 8;      // 16-byte chunks per row
    constexpr int PITCH = D + 8;    // bf16 per staged V row (pad: conflict-free ldmatrix)
    constexpr int KT = 16 * D;      // bf16 per staged K tile
    constexpr int VT = 16 * PITCH;  // bf16 per staged V tile
    constexpr int NS = kRingStages;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ __align__(16) float s_cos[kMaxPairs];
    __shared__ __align__(16) float s_sin[kMaxPairs];
    __shared__ uint32_t s_mask[kRingWarps][NS];
    const int P = D / 2;
    const int g = a.group;
    const int H = a.n_kv_heads;
    const int b = blockIdx.z;
    const int l = blockIdx.y;
    const int n_hg = (H + kRingWarps - 1) / kRingWarps;
    const int split = int(blockIdx.x) / n_hg;
    const int kh0 = (int(blockIdx.x) - split * n_hg) * kRingWarps;
    const int kh1 = min(H, kh0 + kRingWarps);
    const int nq = (kh1 - kh0) * g;  // this CTA's query heads
    // the ring, stage-major: stage st of warp w holds a K tile then a V tile
    // at ring + (st * kRingWarps + w) * (KT + VT); the rotated queries
    // ([nq][D] float32, needed only until every warp holds its fragments)
    // share the last stage, which is first filled after that
    uint16_t* ring = reinterpret_cast<uint16_t*>(smem_raw);
    float* q_s = reinterpret_cast<float*>(ring + size_t(NS - 1) * kRingWarps * (KT + VT));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int gid = lane >> 2;
    const int t = lane & 3;
    const int kh = kh0 + warp;
    const bool wact = kh < kh1;
    const uint16_t* wk = ring + size_t(warp) * (KT + VT);  // this warp's stage 0
    const uint32_t wk_s = uint32_t(__cvta_generic_to_shared(wk));
    const uint32_t wv_s = wk_s + uint32_t(KT * 2);
    constexpr uint32_t kStageBytes = uint32_t(kRingWarps * (KT + VT) * 2);  // one stage of all warps
    uint32_t err = 0;
    pdl_allow();
    {
        // this CTA's query rows into L2 while the preceding grid drains
        const char* qrow = reinterpret_cast<const char*>(
            a.q + ((int64_t(b) * a.n_layers + l) * a.n_q_heads + kh0 * g) * D);
        for (int o = threadIdx.x * 128; o < nq * D * 2; o += blockDim.x * 128) prefetch_l2(qrow + o);
    }
    pdl_wait();
    const int64_t p = a.q_pos[b];
    int64_t len = a.seq_len[b];
    // this thread's query words (eight rotation pairs of a head per round,
    // at most kRingQRounds rounds), requested with the length so that they
    // do not queue behind the ring's first copies
    const uint16_t* qb = a.q + ((int64_t(b) * a.n_layers + l) * a.n_q_heads + kh0 * g) * D;
    const bool q16 = (reinterpret_cast<uintptr_t>(a.q) & 15) == 0;
    uint32_t wx[kRingQRounds][4], wy[kRingQRounds][4];
#pragma unroll
    for (int r = 0; r < kRingQRounds; ++r) {
        const int e = 8 * (threadIdx.x + r * kRingWarps * 32);
        if (e < nq * P) {
            const int hq = e / P;
            const uint16_t* qx = qb + hq * D + (e - hq * P);
            if (q16) {
                const uint4 x4 = __ldg(reinterpret_cast<const uint4*>(qx));
                const uint4 y4 = __ldg(reinterpret_cast<const uint4*>(qx + P));
                wx[r][0] = x4.x; wx[r][1] = x4.y; wx[r][2] = x4.z; wx[r][3] = x4.w;
                wy[r][0] = y4.x; wy[r][1] = y4.y; wy[r][2] = y4.z; wy[r][3] = y4.w;
            } else {
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    wx[r][u] = uint32_t(qx[2 * u]) | (uint32_t(qx[2 * u + 1]) << 16);
                    wy[r][u] = uint32_t(qx[P + 2 * u]) | (uint32_t(qx[P + 2 * u + 1]) << 16);
                }
            }
        }
    }
    if (len < 0 || len > a.capacity) {
        err |= PRCR_ST_CAPACITY;
        len = len < 0 ? 0 : a.capacity;
    }
    if (len > int64_t(a.splits) * a.chunk) {  // above the host's max_len: past the split
        err |= PRCR_ST_CAPACITY;
        len = int64_t(a.splits) * a.chunk;
    }
    // A query position beyond the fixed-point angle reduction (|p| >= 2^31)
    // is reported and the sequence attends to nothing: its output is zeros.
    if (p <= -2147483648LL || p >= 2147483648LL) {
        err |= PRCR_ST_POS_RANGE;
        len = 0;
    }
    const int64_t s_begin = int64_t(split) * a.chunk;
    const int64_t s_end = min(len, s_begin + a.chunk);
    const int n_tiles = s_end > s_begin ? int((s_end - s_begin + 15) / 16) : 0;
    const int64_t lstride = int64_t(l) * a.layer_stride;
    const uint16_t* kbase = a.cache_k + lstride + int64_t(wact ? kh : kh0) * D;
    const uint16_t* vbase = a.cache_v + lstride + int64_t(wact ? kh : kh0) * D;

    // block id of this lane's slot (lane & 15) of tile n (paged caches)
    auto block_id = [&](int n) -> int32_t {
        const int64_t s = s_begin + 16 * int64_t(n) + (lane & 15);
        if (a.cache_kind != PRCR_CACHE_PAGED || n >= n_tiles || s >= s_end) return 0;
        return a.block_table[int64_t(b) * a.bt_stride + s / a.block_size];
    };
    // copies of tile n into stage n % NS (one commit group per call, empty
    // past the last tile or for a warp without a KV head)
    auto issue = [&](int n, int32_t blk) {
        if (wact && n < n_tiles) {
            const int st = n % NS;
            const int64_t s = s_begin + 16 * int64_t(n) + (lane & 15);
            int64_t row = -1;
            if (s < s_end) {
                if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
                    row = int64_t(b) * a.seq_stride + s * a.slot_stride;
                } else if (blk < 0 || blk >= a.n_blocks) {
                    err |= PRCR_ST_NO_BLOCK;
                } else {
                    const int64_t lb = s / a.block_size;
                    row = int64_t(blk) * a.block_stride + (s - lb * a.block_size) * a.slot_stride;
                }
            }
            const uint32_t m = __ballot_sync(kFull, row >= 0) & 0xffffu;
            if (lane == 0) s_mask[warp][st] = m;
            const uint32_t ks_ = wk_s + uint32_t(st) * kStageBytes;
            const uint32_t vs_ = wv_s + uint32_t(st) * kStageBytes;
#pragma unroll
            for (int i = 0; i < (16 * NCH) / 32; ++i) {
                const int c = lane + 32 * i;
                const int slot = c / NCH;
                const int ch = c - slot * NCH;
                const int64_t rr = __shfl_sync(kFull, row, slot);
                const bool ok = rr >= 0;
                cp_async16(ks_ + uint32_t((slot * D + ((ch ^ ((slot & 1) << 2)) * 8)) * 2),
                           ok ? kbase + rr + ch * 8 : kbase, ok ? 16 : 0);
                cp_async16(vs_ + uint32_t((slot * PITCH + ch * 8) * 2),
                           ok ? vbase + rr + ch * 8 : vbase, ok ? 16 : 0);
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    // the first NS - 1 tiles are requested now, before the prologue
    {
        int32_t blk[NS - 1];
#pragma unroll
        for (int i = 0; i < NS - 1; ++i) blk[i] = block_id(i);
#pragma unroll
        for (int i = 0; i < NS - 1; ++i) issue(i, blk[i]);
    }
    int32_t blk_next = block_id(NS - 1);

    // query heads of this CTA rotated at (p, p, p), scaled by 1/sqrt(D): with
    // the same position on every axis, pair i turns by p * inv_freq_i
    // whatever its band, so each pair's cos/sin serves all heads
    for (int i = threadIdx.x; i < P; i += blockDim.x)
        sincos_turns(double(p), a.turn_freq[i], &s_sin[i], &s_cos[i]);
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kRingQRounds; ++r) {
        const int e = 8 * (threadIdx.x + r * kRingWarps * 32);
        if (e >= nq * P) break;
        const int hq = e / P;
        const int i = e - hq * P;  // a multiple of 8: P is 32 or 64
        float rx[8], ry[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const float x = __uint_as_float((u & 1) ? (wx[r][u >> 1] & 0xffff0000u) : (wx[r][u >> 1] << 16));
            const float y = __uint_as_float((u & 1) ? (wy[r][u >> 1] & 0xffff0000u) : (wy[r][u >> 1] << 16));
            const float sn = s_sin[i + u], cs = s_cos[i + u];
            rx[u] = fmaf(x, cs, -y * sn) * a.scale;
            ry[u] = fmaf(y, cs, x * sn) * a.scale;
        }
        float4* ox = reinterpret_cast<float4*>(q_s + hq * D + i);
        float4* oy = reinterpret_cast<float4*>(q_s + hq * D + i + P);
        ox[0] = make_float4(rx[0], rx[1], rx[2], rx[3]);
        ox[1] = make_float4(rx[4], rx[5], rx[6], rx[7]);
        oy[0] = make_float4(ry[0], ry[1], ry[2], ry[3]);
        oy[1] = make_float4(ry[4], ry[5], ry[6], ry[7]);
    }
    __syncthreads();

    // the query B fragments (columns = heads of the group; columns >= g are
    // zero); k-step j of lane group t covers dimensions
    // 8 (t + 4 (j / 2)) + 4 (j % 2) + 0..3, as the K chunks it reads
    uint32_t qh[KS][2], ql[KS][2];
    {
        const bool hv = wact && gid < g;
        const float* qr = q_s + (hv ? (kh - kh0) * g + gid : 0) * D;
#pragma unroll
        for (int j = 0; j < KS; ++j) {
            const int base = 8 * (t + 4 * (j >> 1)) + 4 * (j & 1);
            const float x0 = hv ? qr[base] : 0.0f, x1 = hv ? qr[base + 1] : 0.0f;
            const float x2 = hv ? qr[base + 2] : 0.0f, x3 = hv ? qr[base + 3] : 0.0f;
            split_bf16x2(x0, x1, qh[j][0], ql[j][0]);
            split_bf16x2(x2, x3, qh[j][1], ql[j][1]);
        }
    }
    __syncthreads();  // the queries' stage may now be filled

    if (wact) {
        float o[KS][4];
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.0f;
        float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.0f, 0.0f};  // heads 2t, 2t + 1
        const int lslot = (lane & 7) + ((lane >> 4) & 1) * 8;
        const int ldim = ((lane >> 3) & 1) * 8;

        for (int n = 0; n < n_tiles; ++n) {
            const int st = n % NS;
            // this lane's copies of tile n are complete; after the warp
            // barrier every lane's are visible
            asm volatile("cp.async.wait_group %0;" ::"n"(NS - 2) : "memory");
            __syncwarp();
            // the tile NS - 1 ahead into the stage tile n - 1 used
            {
                const int32_t bn = blk_next;
                blk_next = block_id(n + NS);
                issue(n + NS - 1, bn);
            }
            const uint32_t mask = s_mask[warp][st];

            const uint16_t* kt = wk + size_t(st) * kRingWarps * (KT + VT);
            // S^T (16 slots x 8 columns = the group's query heads, columns >= g
            // zero) = K Q^T: this lane's slots gid (kv[0]) and 8 + gid (kv[1])
            // are the A rows, the query fragments the B operand unchanged; the
            // query's head and remainder products in two chains
            uint4 kv[2][LV];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const int slot = nt * 8 + gid;
#pragma unroll
                for (int u = 0; u < LV; ++u)
                    kv[nt][u] = *reinterpret_cast<const uint4*>(kt + slot * D + (((t + 4 * u) ^ ((slot & 1) << 2)) * 8));
            }
            float sh[4] = {0.0f, 0.0f, 0.0f, 0.0f}, sl_[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int j = 0; j < KS; ++j) {
                const uint4& w0 = kv[0][j >> 1];
                const uint4& w1 = kv[1][j >> 1];
                const uint32_t a0 = (j & 1) ? w0.z : w0.x, a2 = (j & 1) ? w0.w : w0.y;
                const uint32_t a1 = (j & 1) ? w1.z : w1.x, a3 = (j & 1) ? w1.w : w1.y;
                mma_16816(sh, a0, a1, a2, a3, qh[j][0], qh[j][1]);
                mma_16816(sl_, a0, a1, a2, a3, ql[j][0], ql[j][1]);
            }

            // online softmax of this lane's heads 2t, 2t + 1 (columns) over the
            // 16 slots: the eight lanes of one t hold them, two slots each
            const bool oka = (mask >> gid) & 1u, okb = (mask >> (8 + gid)) & 1u;
            float pa[2], pb[2], alpha[2];
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const float va = oka ? sh[hh] + sl_[hh] : -INFINITY;
                const float vb = okb ? sh[2 + hh] + sl_[2 + hh] : -INFINITY;
                float mx = fmaxf(va, vb);
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 4));
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 8));
                mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 16));
                const float m_new = fmaxf(m_run[hh], mx);
                // arguments are <= 0: __expf's error (a few ulp) is far inside
                // the float32 accumulation's
                alpha[hh] = m_new == -INFINITY ? 1.0f : __expf(m_run[hh] - m_new);
                pa[hh] = va == -INFINITY ? 0.0f : __expf(va - m_new);
                pb[hh] = vb == -INFINITY ? 0.0f : __expf(vb - m_new);
                float ps = pa[hh] + pb[hh];
                ps += __shfl_xor_sync(kFull, ps, 4);
                ps += __shfl_xor_sync(kFull, ps, 8);
                ps += __shfl_xor_sync(kFull, ps, 16);
                l_run[hh] = l_run[hh] * alpha[hh] + ps;
                m_run[hh] = m_new;
            }
            // O^T columns are heads 2t, 2t + 1: this lane's own factors
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                o[mt][0] *= alpha[0]; o[mt][1] *= alpha[1]; o[mt][2] *= alpha[0]; o[mt][3] *= alpha[1];
            }
            // P^T as B fragments: the 8 x 8 blocks (slots 0..7 | 8..15) x heads
            // held as (slot gid; heads 2t, 2t + 1) are transposed in registers
            uint32_t m1h, m1l, m2h, m2l;
            split_bf16x2(pa[0], pa[1], m1h, m1l);
            split_bf16x2(pb[0], pb[1], m2h, m2l);
            const uint32_t pb0h = movmatrix_trans(m1h), pb1h = movmatrix_trans(m2h);
            const uint32_t pb0l = movmatrix_trans(m1l), pb1l = movmatrix_trans(m2l);

            // O^T += V^T P^T
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                uint32_t r0, r1, r2, r3;
                const uint32_t addr = wv_s + uint32_t(st) * kStageBytes + uint32_t((lslot * PITCH + mt * 16 + ldim) * 2);
                asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                             : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                             : "r"(addr));
                mma_16816(o[mt], r0, r1, r2, r3, pb0h, pb1h);
                mma_16816(o[mt], r0, r1, r2, r3, pb0l, pb1l);
            }
            __syncwarp();  // stage st is refilled at the next iteration
        }

        // heads 2t, 2t+1 of this lane's O^T columns
        const float l0 = l_run[0], l1 = l_run[1], m0 = m_run[0], m1 = m_run[1];
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int h = 2 * t + hh;
            if (h >= g) continue;
            const int64_t o_idx = (int64_t(b) * a.n_layers + l) * a.n_q_heads + kh * g + h;
            const float lh = hh ? l1 : l0;
            if (a.splits == 1) {
                const float inv = lh > 0.0f ? 1.0f / lh : 0.0f;
                float* out = a.out + o_idx * D;
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    out[mt * 16 + gid] = o[mt][hh] * inv;
                    out[mt * 16 + gid + 8] = o[mt][2 + hh] * inv;
                }
            } else {
                float* part = a.partial + (o_idx * a.splits + split) * (D + 2);
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    part[mt * 16 + gid] = o[mt][hh];
                    part[mt * 16 + gid + 8] = o[mt][2 + hh];
                }
                if (gid == 0) {
                    part[D] = hh ? m1 : m0;
                    part[D + 1] = lh;
                }
            }
        }
    }
    // every copy this thread issued has landed before the CTA may end
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (err) atomicOr(a.status, err);
}

// Merge the chunks of one (sequence, layer, query head). The chunks' maxima
// and sums are reduced by the whole CTA, their weights exp(m_s - M) staged in
// shared memory 256 at a time, and thread d accumulates dimension d over the
// chunks with eight partial rows requested at once.
__global__ void __launch_bounds__(256) decode_merge_kernel(const __grid_constant__ DecodeArgs a) {
    __shared__ float s_red[8];
    __shared__ float s_w[256];
    const int D = a.head_dim, S = a.splits, R = D + 2;
    pdl_allow();
    pdl_wait();  // the decode grid's partials
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    const int64_t o_idx = blockIdx.x;
    const float* part = a.partial + o_idx * S * R;
    float M = -INFINITY;
    for (int sp = threadIdx.x; sp < S; sp += blockDim.x) M = fmaxf(M, part[int64_t(sp) * R + D]);
#pragma unroll
    for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if (lane == 0) s_red[warp] = M;
    __syncthreads();
    M = s_red[0];
    for (int w = 1; w < nw; ++w) M = fmaxf(M, s_red[w]);
    __syncthreads();
    float den = 0.0f;
    for (int sp = threadIdx.x; sp < S; sp += blockDim.x) {
        const float ms = part[int64_t(sp) * R + D];
        if (ms != -INFINITY) den = fmaf(expf(ms - M), part[int64_t(sp) * R + D + 1], den);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) den += __shfl_xor_sync(0xffffffffu, den, o);
    if (lane == 0) s_red[warp] = den;
    __syncthreads();
    den = 0.0f;
    for (int w = 0; w < nw; ++w) den += s_red[w];
    float num[2] = {0.0f, 0.0f};  // dimensions threadIdx.x and threadIdx.x + blockDim.x (D <= 2 x 256)
    for (int s0 = 0; s0 < S; s0 += 256) {
        const int n = min(256, S - s0);
        __syncthreads();
        for (int q = threadIdx.x; q < n; q += blockDim.x) {
            const float ms = part[int64_t(s0 + q) * R + D];
            s_w[q] = ms == -INFINITY ? 0.0f : expf(ms - M);
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int d = threadIdx.x + k * blockDim.x;
            if (d >= D) break;
            const float* col = part + int64_t(s0) * R + d;
            float acc = num[k];
            int q = 0;
            for (; q + 8 <= n; q += 8) {
                float x[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) x[u] = col[int64_t(q + u) * R];
#pragma unroll
                for (int u = 0; u < 8; ++u) acc = fmaf(s_w[q + u], x[u], acc);
            }
            for (; q < n; ++q) acc = fmaf(s_w[q], col[int64_t(q) * R], acc);
            num[k] = acc;
        }
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int d = threadIdx.x + k * blockDim.x;
        if (d < D) a.out[o_idx * D + d] = den > 0.0f ? num[k] / den : 0.0f;
    }
}

// Merge for at most 32 chunks: one warp per (sequence, layer, query head).
// Lane s holds chunk s's maximum and sum (one round trip), the maximum, the
// weights exp(m_s - M) and the denominator stay in registers (shuffles), and
// lane i accumulates dimensions 2i, 2i + 1 (+ 64 j) over the chunks' rows
// with eight rows requested at a time.
__global__ void __launch_bounds__(128) decode_merge_warp_kernel(const __grid_constant__ DecodeArgs a,
                                                                int64_t n_out) {
    pdl_allow();
    pdl_wait();  // the decode grid's partials
    const int D = a.head_dim, S = a.splits, R = D + 2;
    const int lane = threadIdx.x & 31;
    const int64_t o_idx = int64_t(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (o_idx >= n_out) return;
    const float* part = a.partial + o_idx * S * R;
    const float ms = lane < S ? part[int64_t(lane) * R + D] : -INFINITY;
    const float ls = lane < S ? part[int64_t(lane) * R + D + 1] : 0.0f;
    float M = ms;
#pragma unroll
    for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, o));
    const float w = ms == -INFINITY ? 0.0f : expf(ms - M);
    float den = w * ls;
#pragma unroll
    for (int o = 16; o; o >>= 1) den += __shfl_xor_sync(kFull, den, o);
    const float inv = den > 0.0f ? 1.0f / den : 0.0f;
    for (int d0 = 2 * lane; d0 < D; d0 += 64) {
        float2 acc = make_float2(0.0f, 0.0f);
        for (int s0 = 0; s0 < S; s0 += 8) {
            float2 x[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
                x[u] = s0 + u < S ? *reinterpret_cast<const float2*>(part + int64_t(s0 + u) * R + d0)
                                  : make_float2(0.0f, 0.0f);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const float wu = __shfl_sync(kFull, w, (s0 + u) & 31);
                acc.x = fmaf(wu, x[u].x, acc.x);
                acc.y = fmaf(wu, x[u].y, acc.y);
            }
        }
        *reinterpret_cast<float2*>(a.out + o_idx * D + d0) = make_float2(acc.x * inv, acc.y * inv);
    }
}

template <int GP>
cudaError_t launch_gp(const DecodeArgs& a, dim3 grid, size_t smem, cudaStream_t stream) {
    const dim3 block(kDecodeThreads);
    switch (a.head_dim) {
        case 64: return launch_pdl(decode_kernel<GP, 2>, grid, block, smem, stream, a);
        case 128: return launch_pdl(decode_kernel<GP, 4>, grid, block, smem, stream, a);
        default: return launch_pdl(decode_kernel<GP, 8>, grid, block, smem, stream, a);
    }
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs& a, int gp, dim3 grid, size_t smem,
                          cudaStream_t stream) {
    cudaError_t e;
    if (a.ring) {
        // small batch: KV heads split over CTAs, K and V streamed through a
        // shared-memory ring per warp
        const int n_hg = (a.n_kv_heads + kRingWarps - 1) / kRingWarps;
        const int D = a.head_dim;
        // the ring (the rotated queries share its last stage)
        const size_t sm = size_t(kRingWarps) * kRingStages * 16 * (D + D + 8) * sizeof(uint16_t);
        static_assert(8 * 128 * sizeof(float) <= 16 * (2 * 128 + 8) * sizeof(uint16_t) &&
                          8 * 64 * sizeof(float) <= 16 * (2 * 64 + 8) * sizeof(uint16_t),
                      "a GQA group's rotated queries fit in one warp's share of a ring stage");
        dim3 g2 = grid;
        g2.x *= unsigned(n_hg);
        auto k = D == 64 ? decode_ring_kernel<64> : decode_ring_kernel<128>;
        e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(sm));
        if (e == cudaSuccess) e = launch_pdl(k, g2, dim3(kRingWarps * 32), sm, stream, a);
    } else if (a.head_dim == 64 || a.head_dim == 128) {
        // tensor-core kernel: rotated queries + two staged V tiles per warp
        const size_t sm = size_t(a.n_q_heads) * a.head_dim * sizeof(float) +
                          size_t(kDecodeThreads / 32) * 2 * 16 * (a.head_dim + 8) * sizeof(uint16_t);
        auto k = a.head_dim == 64 ? decode_mma_kernel<64> : decode_mma_kernel<128>;
        e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(sm));
        if (e == cudaSuccess) e = launch_pdl(k, grid, dim3(kDecodeThreads), sm, stream, a);
    } else {
        // groups of 1, 2 and 4 query heads run as 4 (padded) heads x 8 slots per
        // warp iteration, groups of 5..8 as 8 heads x 4 slots
        e = gp <= 4 ? launch_gp<4>(a, grid, smem, stream) : launch_gp<8>(a, grid, smem, stream);
    }
    if (e != cudaSuccess || a.splits == 1) return e;
    const int64_t n_out = int64_t(grid.z) * a.n_layers * a.n_q_heads;
    if (a.splits <= 32)
        return launch_pdl(decode_merge_warp_kernel, dim3(unsigned((n_out + 3) / 4)), dim3(128), 0,
                          stream, a, n_out);
    return launch_pdl(decode_merge_kernel, dim3(unsigned(n_out)),
                      dim3(a.head_dim < 256 ? a.head_dim : 256), 0, stream, a);
}

}  // namespace prcr
