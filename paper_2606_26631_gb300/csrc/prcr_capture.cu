// Prefill capture kernel (Sec. 3.1, Eq. "raw_kv" and "global_raw_memory",
// with the position-bound cache entry of Eq. "historical_position_bound_kv").
//
// During multimodal prefill each visual token's pre-rotation key and value
// rows exist once, per layer. This kernel reads them once and writes them
// twice: unchanged into the raw visual memory (with the token's original
// (t, h, w) coordinate), and as the ordinary decoder-cache entry the model
// itself would store: the key rotated with M-RoPE at the original
// coordinate, the value unchanged, at consecutive cache slots.
//
// Work layout as in the rebind kernel: a CTA owns T tokens x G layers; its
// prologue resolves each token's cache row (block-table lookup for paged
// caches) and the float32 cos/sin of every (token, pair) from the angle
// reduced modulo a turn in fixed point; each thread then owns one (token, head, 16-byte
// vector) and its rotate-half partner, for all G layers.
#include <cmath>

#include <cuda_bf16.h>

#include "prcr_internal.h"

namespace prcr {
namespace {

__device__ __forceinline__ uint4 ld_stream(const uint16_t* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ void st_row(uint16_t* p, const uint4& v) {
    asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};"
                 :
                 : "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ uint32_t rot_pack(float x0, float y0, float c0, float s0, float x1,
                                             float y1, float c1, float s1, bool first) {
    const float a0 = first ? fmaf(x0, c0, -y0 * s0) : fmaf(y0, c0, x0 * s0);
    const float a1 = first ? fmaf(x1, c1, -y1 * s1) : fmaf(y1, c1, x1 * s1);
    const __nv_bfloat162 v = __floats2bfloat162_rn(a0, a1);
    return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ void rotate(const uint4& x, const uint4& y, const float* c,
                                       const float* s, uint4& xo, uint4& yo) {
    const uint32_t xs[4] = {x.x, x.y, x.z, x.w};
    const uint32_t ys[4] = {y.x, y.y, y.z, y.w};
    uint32_t xr[4], yr[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const float x0 = __uint_as_float(xs[w] << 16), x1 = __uint_as_float(xs[w] & 0xffff0000u);
        const float y0 = __uint_as_float(ys[w] << 16), y1 = __uint_as_float(ys[w] & 0xffff0000u);
        xr[w] = rot_pack(x0, y0, c[2 * w], s[2 * w], x1, y1, c[2 * w + 1], s[2 * w + 1], true);
        yr[w] = rot_pack(x0, y0, c[2 * w], s[2 * w], x1, y1, c[2 * w + 1], s[2 * w + 1], false);
    }
    xo = make_uint4(xr[0], xr[1], xr[2], xr[3]);
    yo = make_uint4(yr[0], yr[1], yr[2], yr[3]);
}

__device__ __forceinline__ int pair_axis(int i, int layout, int st, int sh, int sw) {
    if (layout == PRCR_LAYOUT_SECTIONED) return i < st ? 0 : (i < st + sh ? 1 : 2);
    const int r = i % 3;
    if (r == 1 && i < 3 * sh) return 1;
    if (r == 2 && i < 3 * sw) return 2;
    return 0;
}

__global__ void __launch_bounds__(512) capture_kernel(const __grid_constant__ CaptureArgs a) {
    extern __shared__ float smem[];
    const int D = a.head_dim;
    const int P = D >> 1;
    const int T = a.tok_per_cta;
    float* cos_s = smem;
    float* sin_s = smem + T * P;
    int64_t* dst_s = reinterpret_cast<int64_t*>(sin_s + T * P);
    const int tok0 = blockIdx.x * T;
    uint32_t err = 0;

    for (int t = threadIdx.x; t < T; t += blockDim.x) {
        const int j = tok0 + t;
        int64_t dst = -1;
        if (j < a.m_count) {
            const int64_t slot = a.slot_begin + j;
            if (slot >= a.capacity) {
                err |= PRCR_ST_CAPACITY;
            } else if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
                dst = a.cache_seq_off + slot * a.slot_stride;
            } else {
                const int64_t lb = slot / a.block_size;
                const int32_t blk = a.bt_row[lb];
                if (blk < 0 || blk >= a.n_blocks) err |= PRCR_ST_NO_BLOCK;
                else dst = int64_t(blk) * a.block_stride + (slot - lb * a.block_size) * a.slot_stride;
            }
            if (a.store_coords && blockIdx.y == 0) {
                a.store_coords[3 * int64_t(j) + 0] = a.coords[3 * int64_t(j) + 0];
                a.store_coords[3 * int64_t(j) + 1] = a.coords[3 * int64_t(j) + 1];
                a.store_coords[3 * int64_t(j) + 2] = a.coords[3 * int64_t(j) + 2];
            }
        }
        dst_s[t] = dst;
    }
    for (int q = threadIdx.x; q < T * P; q += blockDim.x) {
        const int t = q / P;
        const int i = q - t * P;
        const int j = tok0 + t;
        float c = 1.0f, s = 0.0f;
        if (j < a.m_count) {
            const int ax = pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w);
            sincos_turns(double(a.coords[3 * int64_t(j) + ax]), a.turn_freq[i], &s, &c);
        }
        cos_s[q] = c;
        sin_s[q] = s;
    }
    if (err && blockIdx.y == 0) atomicOr(a.status, err);
    __syncthreads();

    const int lanes = a.lanes;
    const int t = threadIdx.x / lanes;
    const int lane = threadIdx.x - t * lanes;
    const int j = tok0 + t;
    if (t >= T || j >= a.m_count) return;
    const int64_t dst = dst_s[t];
    const int vph = D >> 4;
    const int h = lane / vph;
    const int v = lane - h * vph;
    const int64_t off = int64_t(h) * D + v * 8;
    float c[8], s[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        c[e] = cos_s[t * P + v * 8 + e];
        s[e] = sin_s[t * P + v * 8 + e];
    }
    const int l0 = blockIdx.y * a.layers_per_cta;
    const int l1 = min(l0 + a.layers_per_cta, a.n_layers);
    const uint16_t* sk = a.src_k + int64_t(l0) * a.src_layer_stride + int64_t(j) * a.src_token_stride + off;
    const uint16_t* sv = a.src_v + int64_t(l0) * a.src_layer_stride + int64_t(j) * a.src_token_stride + off;
    uint16_t* rk = a.store_k + int64_t(l0) * a.store_layer_stride + int64_t(j) * a.store_token_stride + off;
    uint16_t* rv = a.store_v + int64_t(l0) * a.store_layer_stride + int64_t(j) * a.store_token_stride + off;
    const int64_t dst_row = dst < 0 ? 0 : dst;  // rows with dst < 0 are never written
    uint16_t* ck = a.cache_k + dst_row + int64_t(l0) * a.cache_layer_stride + off;
    uint16_t* cv = a.cache_v + dst_row + int64_t(l0) * a.cache_layer_stride + off;
    for (int l = l0; l < l1; ++l) {
        const uint4 k0 = ld_stream(sk), k1 = ld_stream(sk + P);
        const uint4 v0 = ld_stream(sv), v1 = ld_stream(sv + P);
        st_row(rk, k0);
        st_row(rk + P, k1);
        st_row(rv, v0);
        st_row(rv + P, v1);
        if (dst >= 0) {
            uint4 o0, o1;
            rotate(k0, k1, c, s, o0, o1);
            st_row(ck, o0);
            st_row(ck + P, o1);
            st_row(cv, v0);
            st_row(cv + P, v1);
        }
        sk += a.src_layer_stride; sv += a.src_layer_stride;
        rk += a.store_layer_stride; rv += a.store_layer_stride;
        ck += a.cache_layer_stride; cv += a.cache_layer_stride;
    }
}

}  // namespace

cudaError_t capture_blocks_per_sm(int block, size_t smem, int* out) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, capture_kernel, block, smem);
}

cudaError_t launch_capture(const CaptureArgs& a, dim3 grid, int block, size_t smem,
                           cudaStream_t stream) {
    capture_kernel<<<grid, block, smem, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
