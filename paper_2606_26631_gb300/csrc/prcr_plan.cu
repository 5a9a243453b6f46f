// Plan kernel: position reassignment and cache slots (Sec. 3.2, Algorithm 1).
//
// One CTA per revisit I_tau. It reduces the stored coordinates of the
// selected tokens to their per-axis range (Eq. "selected_coord_range"), then
// gives each token its reassigned position (Eq. "normalized_coord" and
// "image_range_fractional_reinsert", or the rule the mode selects), its
// cache slot (the existing cache length plus its rank among the sequence's
// appended tokens: the Concat of Eq. "active_cache") and the store / cache
// row offsets the rebind kernel streams through. Threads of the whole grid
// also fill the per-sequence outputs (cache length, next text position).
//
// Positions are exact: the PCR value is the rational N/Q with
//   Q = (K+1) * (hi - lo),
//   N = (p - L) * Q + (L+1) * ((hi - lo) + (K-1) * (c - lo)),
// formed in 64-bit integers and rounded once by an IEEE float64 division
// (both operands exactly representable while |N| <= (|p-L| + L + 1) * Q < 2^52).
#include <climits>
#include <cmath>

#include "prcr_internal.h"

namespace prcr {
namespace {

constexpr double kExactLimit = 4503599627370496.0;  // 2^52

// True when every integer formed for p_hat = ((p - L) * Q + tail) / Q with
// 0 <= tail <= (L+1) * Q stays below 2^52 in magnitude, so that the integer
// products cannot overflow and the float64 division sees exact operands.
__device__ __forceinline__ bool exact_ok(int64_t p_minus_l, int32_t L, double Q) {
    return (fabs(double(p_minus_l)) + double(L) + 1.0) * Q < kExactLimit;
}

__device__ __forceinline__ double pcr_position(int64_t p, int32_t L, int64_t K, int32_t c,
                                               int32_t lo, int32_t hi, bool center,
                                               uint32_t& err) {
    const int64_t span = int64_t(hi) - int64_t(lo);
    const int64_t pl = p - L;
    if (span > 0) {
        if (exact_ok(pl, L, double(K + 1) * double(span))) {
            const int64_t Q = (K + 1) * span;
            const int64_t tail = int64_t(L + 1) * (span + (K - 1) * (int64_t(c) - lo));
            return double(pl * Q + tail) / double(Q);
        }
        err |= PRCR_ST_POS_RANGE;
        const double u = double(int64_t(c) - lo) / double(span);
        return double(pl) + double(L + 1) * (1.0 + double(K - 1) * u) / double(K + 1);
    }
    // degenerate axis: u = 0, or u = 1/2 with the centre reading
    const int64_t Q = center ? 2 * (K + 1) : K + 1;
    const int64_t tail = center ? int64_t(L + 1) * (K + 1) : int64_t(L + 1);
    if (exact_ok(pl, L, double(Q))) return double(pl * Q + tail) / double(Q);
    err |= PRCR_ST_POS_RANGE;
    return double(pl) + double(tail) / double(Q);
}

// p + num / (K + 1), exact while representable (UIR).
__device__ __forceinline__ double uir_position(int64_t p, int64_t num, int64_t K, uint32_t& err) {
    if (exact_ok(p, 0, double(K + 1))) return double(p * (K + 1) + num) / double(K + 1);
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

__device__ void plan_revisit(const PlanArgs& a, int r, int* s_part, uint32_t& err) {
    const int beg = a.rev_tok_off[r];
    const int end = a.rev_tok_off[r + 1];
    // sequence owning revisit r: last b with seq_rev_off[b] <= r
    int lo = 0, hi = a.n_seqs;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (a.seq_rev_off[mid] <= r) lo = mid; else hi = mid;
    }
    const int b = lo;
    const int r_first = a.seq_rev_off[b];
    bool ok = beg >= 0 && beg <= end && int64_t(end) <= a.total_k &&
              r_first <= r && r < a.seq_rev_off[b + 1] && r_first >= 0;
    const int t0 = ok ? a.rev_tok_off[r_first] : 0;
    ok = ok && t0 >= 0 && t0 <= beg;
    if (!ok) {  // uniform over the CTA
        err |= PRCR_ST_CSR;
        return;
    }
    const int64_t K = end - beg;
    const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride;

    int mn[3] = {INT_MAX, INT_MAX, INT_MAX};
    int mx[3] = {INT_MIN, INT_MIN, INT_MIN};
    if (a.mode == PRCR_MODE_PCR) {
        for (int j = beg + threadIdx.x; j < end; j += blockDim.x) {
            const int m = a.idx[j];
            if (m >= 0 && m < a.n_tokens) {
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    const int c = crd[3 * int64_t(m) + ax];
                    mn[ax] = min(mn[ax], c);
                    mx[ax] = max(mx[ax], c);
                }
            }
        }
        block_minmax(mn, mx, s_part);
    }

    const int64_t p = a.p_txt[b];
    const int64_t clen = a.cache_len_in[b];
    const bool center = (a.flags & PRCR_FLAG_DEGENERATE_CENTER) != 0;
    const int64_t capacity = a.cache_kind == PRCR_CACHE_CONTIGUOUS
                                 ? int64_t(a.max_slots)
                                 : int64_t(a.bt_stride) * a.block_size;
    for (int j = beg + threadIdx.x; j < end; j += blockDim.x) {
        const int m = a.idx[j];
        const int64_t slot = clen + (j - t0);
        double pos[3];
        int64_t src = 0, dst = -1;
        if (m < 0 || m >= a.n_tokens) {
            err |= PRCR_ST_IDX_RANGE;
            pos[0] = pos[1] = pos[2] = __longlong_as_double(0x7ff8000000000000LL);
        } else {
            const int32_t c[3] = {crd[3 * int64_t(m)], crd[3 * int64_t(m) + 1],
                                  crd[3 * int64_t(m) + 2]};
            switch (a.mode) {
                case PRCR_MODE_PCR:
#pragma unroll
                    for (int ax = 0; ax < 3; ++ax)
                        pos[ax] = pcr_position(p, a.L, K, c[ax], mn[ax], mx[ax], center, err);
                    break;
                case PRCR_MODE_ORIGINAL:
#pragma unroll
                    for (int ax = 0; ax < 3; ++ax) pos[ax] = double(c[ax]);
                    break;
                case PRCR_MODE_UIR: {
                    // p + (j' + 1) / (K + 1), j' the token's rank in its revisit
                    const double v = uir_position(p, int64_t(j - beg + 1), K, err);
                    pos[0] = pos[1] = pos[2] = v;
                    break;
                }
                default: {  // PRCR_MODE_LPA: p + rank in sequence + 1
                    const double v = double(p + (j - t0) + 1);
                    pos[0] = pos[1] = pos[2] = v;
                    break;
                }
            }
            src = int64_t(b) * a.store_seq_stride + int64_t(m) * a.store_token_stride;
            if (clen < 0 || slot >= capacity) {
                err |= PRCR_ST_CAPACITY;
            } else if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
                dst = int64_t(b) * a.cache_seq_stride + slot * a.slot_stride;
            } else {
                const int64_t lb = slot / a.block_size;
                const int32_t blk = a.block_table[int64_t(b) * a.bt_stride + lb];
                if (blk < 0 || blk >= a.n_blocks) {
                    err |= PRCR_ST_NO_BLOCK;
                } else {
                    dst = int64_t(blk) * a.block_stride + (slot - lb * a.block_size) * a.slot_stride;
                }
            }
        }
        a.plan.src[j] = src;
        a.plan.dst[j] = dst;
        a.plan.pos[3 * int64_t(j) + 0] = pos[0];
        a.plan.pos[3 * int64_t(j) + 1] = pos[1];
        a.plan.pos[3 * int64_t(j) + 2] = pos[2];
        if (a.pos_out) {
            a.pos_out[3 * int64_t(j) + 0] = pos[0];
            a.pos_out[3 * int64_t(j) + 1] = pos[1];
            a.pos_out[3 * int64_t(j) + 2] = pos[2];
        }
        if (a.slot_out) a.slot_out[j] = int32_t(slot > INT_MAX ? INT_MAX : slot);
    }
}

__global__ void __launch_bounds__(kPlanThreads) plan_kernel(const __grid_constant__ PlanArgs a) {
    // The rebind grid may start launching now; it waits for this grid to
    // finish (griddepcontrol.wait) before it reads the plan.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ int s_part[33 * 6];
    uint32_t err = 0;

    // Per-sequence outputs and the offsets' structure.
    for (int64_t b = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; b < a.n_seqs;
         b += int64_t(gridDim.x) * blockDim.x) {
        const int r0 = a.seq_rev_off[b];
        const int r1 = a.seq_rev_off[b + 1];
        int64_t k = 0;
        if (r0 < 0 || r1 < r0 || r1 > a.n_revisits) {
            err |= PRCR_ST_CSR;
        } else {
            const int t0 = a.rev_tok_off[r0];
            const int t1 = a.rev_tok_off[r1];
            if (t0 < 0 || t1 < t0 || int64_t(t1) > a.total_k) err |= PRCR_ST_CSR;
            else k = t1 - t0;
        }
        const int64_t len = int64_t(a.cache_len_in[b]) + k;
        if (len > INT_MAX) err |= PRCR_ST_CAPACITY;
        a.cache_len_out[b] = int32_t(len > INT_MAX ? INT_MAX : len);
        const int64_t p = a.p_txt[b];
        a.next_pos_out[b] = a.mode == PRCR_MODE_LPA ? p + k + 1 : p + 1;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        if (a.seq_rev_off[0] != 0 || a.seq_rev_off[a.n_seqs] != a.n_revisits ||
            a.rev_tok_off[0] != 0 || int64_t(a.rev_tok_off[a.n_revisits]) != a.total_k)
            err |= PRCR_ST_CSR;
    }

    for (int r = blockIdx.x; r < a.n_revisits; r += gridDim.x) plan_revisit(a, r, s_part, err);

    if (err) atomicOr(a.status, err);
}

}  // namespace

cudaError_t launch_plan(const PlanArgs& a, cudaStream_t stream) {
    const int seq_ctas = (a.n_seqs + kPlanThreads - 1) / kPlanThreads;
    int grid = a.n_revisits > seq_ctas ? a.n_revisits : seq_ctas;
    if (grid < 1) grid = 1;
    plan_kernel<<<grid, kPlanThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace prcr
