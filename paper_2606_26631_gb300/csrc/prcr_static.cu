// prcr_rebind_inject_static: the revisit call without a caller workspace.
//
// Some callers cannot allocate device memory themselves: a plugin that runs
// inside a host framework which owns every byte of device memory through its
// own pool and forbids raw cudaMalloc, or a latency-critical decode loop where
// a cudaMalloc/cudaFree (which may synchronise the device) is not allowed.
// For them this entry point keeps the per-token plan (the scratch the plan
// kernel writes and the rebind kernel reads) in a fixed device array that
// belongs to the library: every GPU that loads libprcr.so holds it until the
// process exits. The caller still passes (and owns) every input and output.
//
// The array is a host-side stand-in in host code, not a device address; its
// device address is looked up once per device (cudaGetSymbolAddress, with
// that device current) on the first call made on that device, and passed to
// the kernels as their workspace. That first call therefore does set-up work
// and should come before any stream capture. The address is kept for the
// life of the process: after a reset of the device (cudaDeviceReset, or its
// primary context released and created again) the library's module is
// loaded anew and the kept address is stale, so this entry point must not be
// called on a device after such a reset.
//
// All calls share the one array and it keeps whatever the last call left:
// calls whose work overlaps on the GPU (different streams, or several host
// threads at once) race on it. Nothing in it has to start at zero: for a
// well-formed batch the plan kernel rewrites every entry the rebind kernel
// then reads, and for a malformed one the rebind kernel reads none.
#include <mutex>

#include "prcr_internal.h"

namespace {

constexpr size_t kStaticTokens = size_t(PRCR_STATIC_MAX_TOKENS);
constexpr size_t kStaticBytes =
    2 * ((8 * kStaticTokens + 255) & ~size_t(255)) + ((24 * kStaticTokens + 255) & ~size_t(255));
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (set up once).
int scratch_address(void** out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PRCR_ECUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
            return PRCR_ECUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return PRCR_OK;
}

}  // namespace

extern "C" PRCR_API int prcr_rebind_inject_static(const prcr_rope_cfg* cfg,
                                                  const prcr_store_desc* store,
                                                  const prcr_cache_desc* cache,
                                                  const prcr_revisit_batch* batch,
                                                  const prcr_outputs* out, int32_t mode,
                                                  int32_t L, int32_t flags, void* stream) {
    // the call's own checks first, so that a malformed call gets the code
    // prcr_rebind_inject would return and does no set-up
    const int rc0 = prcr::check_revisit_args(cfg, store, cache, batch, out, mode, L, flags);
    if (rc0 != PRCR_OK || batch->n_seqs == 0) return rc0;
    if (batch->total_k > PRCR_STATIC_MAX_TOKENS) return PRCR_EWORKSPACE;
    if (prcr::workspace_bytes(batch->total_k) > kStaticBytes) return PRCR_EWORKSPACE;
    void* ws = nullptr;
    if (batch->total_k > 0) {
        const int rc = scratch_address(&ws);
        if (rc != PRCR_OK) return rc;
    }
    return prcr_rebind_inject(cfg, store, cache, batch, out, mode, L, flags, ws, kStaticBytes,
                              stream);
}
