// Rebind + inject kernel (Sec. 3.3, Eq. "cache_reconstruction" and
// "active_cache"; Algorithm 1, the loop over layers).
//
// For every selected token, every layer and every KV head, the raw key row
// is gathered from the store, rotated with M-RoPE at the token's reassigned
// (t, h, w) position, rounded to bf16 and written to the token's cache slot;
// the raw value row is copied unchanged next to it.
//
// Work layout. A CTA owns T tokens x G layers. Its threads first build the
// float32 cos/sin of every (token, rotation pair) of the tile in shared
// memory, once for all G layers and all heads: the angle modulo a turn is
// formed exactly in fixed-point integers (sincos_turns) and only then handed
// to float32 sincosf, so a position near 3e4 keeps a ~2e-7 rad angle error
// instead of the ~2e-3 of a float32 product.
// Then each thread owns one (token, head, 16-byte vector v) slot of the row:
// it loads the 8 bf16 of the first half at v and the 8 bf16 of the second
// half at v + D/2 (the rotate-half partners), for K and V, and walks the G
// layers. Consecutive threads cover consecutive 16-byte vectors of a row, so
// every warp-wide load and store is a set of whole 128-byte lines.
//
// The kernel is launched with programmatic dependent launch behind the plan
// kernel and waits on it (griddepcontrol.wait) before touching the plan.
#include <cmath>

#include <cuda_bf16.h>

#include "prcr_device.cuh"

namespace prcr {
namespace {

__global__ void __launch_bounds__(512) rebind_kernel(const __grid_constant__ RebindArgs a) {
    extern __shared__ float smem[];
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (*reinterpret_cast<const volatile uint32_t*>(a.status) & PRCR_ST_CSR) return;

    const int D = a.head_dim;
    const int P = D >> 1;
    const int T = a.tok_per_cta;
    float* cos_s = smem;
    float* sin_s = smem + T * P;
    const int64_t tok0 = int64_t(blockIdx.x) * T;

    for (int q = threadIdx.x; q < T * P; q += blockDim.x) {
        const int t = q / P;
        const int i = q - t * P;
        const int64_t tok = tok0 + t;
        float c = 1.0f, s = 0.0f;
        if (tok < a.total_k) {
            const int ax = pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w);
            sincos_turns(a.plan_pos[3 * tok + ax], a.turn_freq[i], &s, &c);
        }
        cos_s[q] = c;
        sin_s[q] = s;
    }
    __syncthreads();

    const int lanes = a.lanes;
    const int t = threadIdx.x / lanes;
    const int lane = threadIdx.x - t * lanes;
    const int64_t tok = tok0 + t;
    if (t >= T || tok >= a.total_k) return;
    const int64_t dst = a.plan_dst[tok];
    if (dst < 0) return;
    const int64_t src = a.plan_src[tok];

    const int vph = D >> 4;  // 16-byte vectors per half row of one head
    const int h = lane / vph;
    const int v = lane - h * vph;
    const int half = P;      // elements between rotate-half partners
    const int64_t off = int64_t(h) * D + v * 8;

    float c[8], s[8];
    {
        const float4* cp = reinterpret_cast<const float4*>(cos_s + t * P + v * 8);
        const float4* sp = reinterpret_cast<const float4*>(sin_s + t * P + v * 8);
        const float4 c0 = cp[0], c1 = cp[1], s0 = sp[0], s1 = sp[1];
        c[0] = c0.x; c[1] = c0.y; c[2] = c0.z; c[3] = c0.w;
        c[4] = c1.x; c[5] = c1.y; c[6] = c1.z; c[7] = c1.w;
        s[0] = s0.x; s[1] = s0.y; s[2] = s0.z; s[3] = s0.w;
        s[4] = s1.x; s[5] = s1.y; s[6] = s1.z; s[7] = s1.w;
    }

    const int l0 = blockIdx.y * a.layers_per_cta;
    const int l1 = min(l0 + a.layers_per_cta, a.n_layers);
    const int64_t sls = a.store_layer_stride;
    const int64_t cls = a.cache_layer_stride;
    const uint16_t* sk = a.store_k + src + int64_t(l0) * sls + off;
    const uint16_t* sv = a.store_v + src + int64_t(l0) * sls + off;
    uint16_t* ck = a.cache_k + dst + int64_t(l0) * cls + off;
    uint16_t* cv = a.cache_v + dst + int64_t(l0) * cls + off;

    stream_layers(sk, sv, ck, cv, sls, cls, half, l1 - l0, c, s);
}

}  // namespace

cudaError_t rebind_blocks_per_sm(int block, size_t smem, int* out) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, rebind_kernel, block, smem);
}

cudaError_t launch_rebind(const RebindArgs& a, dim3 grid, int block, size_t smem,
                          cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(block, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, rebind_kernel, a);
}

}  // namespace prcr
