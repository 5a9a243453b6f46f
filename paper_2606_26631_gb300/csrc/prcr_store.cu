// Raw visual memory fill (Sec. 3.1, Eq. "raw_kv" and "global_raw_memory"):
// a strided, 16-byte vectorised copy of pre-rotation K/V rows and of the
// tokens' original coordinates into the store.
#include "prcr_internal.h"

namespace prcr {
namespace {

__global__ void __launch_bounds__(256) store_kernel(const __grid_constant__ StoreArgs a) {
    const int64_t per_layer = int64_t(a.m_count) * a.row_vecs;
    const int64_t total = per_layer * a.n_layers;
    const int64_t stride = int64_t(gridDim.x) * blockDim.x;
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t l = i / per_layer;
        const int64_t rem = i - l * per_layer;
        const int64_t m = rem / a.row_vecs;
        const int64_t v = rem - m * a.row_vecs;
        const int64_t so = l * a.src_layer_stride + m * a.src_token_stride + v * 8;
        const int64_t d = l * a.dst_layer_stride + m * a.dst_token_stride + v * 8;
        *reinterpret_cast<uint4*>(a.dst_k + d) = *reinterpret_cast<const uint4*>(a.src_k + so);
        *reinterpret_cast<uint4*>(a.dst_v + d) = *reinterpret_cast<const uint4*>(a.src_v + so);
    }
    if (a.dst_coords) {
        for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < 3 * int64_t(a.m_count);
             i += stride)
            a.dst_coords[i] = a.src_coords[i];
    }
}

}  // namespace

cudaError_t launch_store(const StoreArgs& a, cudaStream_t stream) {
    const int64_t total = int64_t(a.m_count) * a.row_vecs * a.n_layers;
    int64_t blocks = (total + 255) / 256;
    if (blocks < 1) blocks = 1;
    if (blocks > 152 * 32) blocks = 152 * 32;
    store_kernel<<<int(blocks), 256, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
