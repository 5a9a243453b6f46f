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
constexpr int kTokPerThread = 4;   // tokens of a revisit each thread keeps in registers
constexpr int kPosTable = 1024;    // exact PCR positions tabulated per axis when span < this

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

// Per-token outputs of one selected token (plan entry, optional position and
// slot outputs). pos[] must already hold the reassigned position.
__device__ __forceinline__ void emit(const PlanArgs& a, int j, int64_t slot, int64_t src,
                                     int64_t dst, const double (&pos)[3]) {
    a.plan.src[j] = src;
    a.plan.dst[j] = dst;
    double* pp = a.plan.pos + 3 * int64_t(j);
    pp[0] = pos[0];
    pp[1] = pos[1];
    pp[2] = pos[2];
    if (a.pos_out) {
        double* po = a.pos_out + 3 * int64_t(j);
        po[0] = pos[0];
        po[1] = pos[1];
        po[2] = pos[2];
    }
    if (a.slot_out) a.slot_out[j] = int32_t(slot > INT_MAX ? INT_MAX : slot);
}

struct RevisitCtx {
    int b, beg, end, t0;
    int64_t K, p, clen, capacity;
    int lo[3], hi[3];
    bool tab[3];
    bool center;
};

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

__device__ __forceinline__ void place_token(const PlanArgs& a, const RevisitCtx& r,
                                            const double (*tab)[kPosTable], int j, int m,
                                            const int (&c)[3], int32_t blk, uint32_t& err) {
    const int64_t slot = r.clen + (j - r.t0);
    double pos[3];
    int64_t src = 0, dst = -1;
    if (m < 0 || m >= a.n_tokens) {
        err |= PRCR_ST_IDX_RANGE;
        pos[0] = pos[1] = pos[2] = __longlong_as_double(0x7ff8000000000000LL);
    } else {
        switch (a.mode) {
            case PRCR_MODE_PCR:
#pragma unroll
                for (int ax = 0; ax < 3; ++ax)
                    pos[ax] = r.tab[ax] ? tab[ax][c[ax] - r.lo[ax]]
                                        : pcr_position(r.p, a.L, r.K, c[ax], r.lo[ax], r.hi[ax],
                                                       r.center, err);
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
        dst = dest_row(a, r, slot, blk, err);
    }
    emit(a, j, slot, src, dst, pos);
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

__device__ void plan_revisit(const PlanArgs& a, int r, int* s_part, double (*s_tab)[kPosTable],
                             uint32_t& err) {
    RevisitCtx x;
    x.beg = a.rev_tok_off[r];
    x.end = a.rev_tok_off[r + 1];
    // sequence owning revisit r: last b with seq_rev_off[b] <= r
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
    if (!ok) {  // uniform over the CTA
        err |= PRCR_ST_CSR;
        return;
    }
    x.K = x.end - x.beg;
    x.p = a.p_txt[x.b];
    x.clen = a.cache_len_in[x.b];
    x.center = (a.flags & PRCR_FLAG_DEGENERATE_CENTER) != 0;
    x.capacity = a.cache_kind == PRCR_CACHE_CONTIGUOUS ? int64_t(a.max_slots)
                                                       : int64_t(a.bt_stride) * a.block_size;
    const int32_t* crd = a.coords + int64_t(x.b) * a.coord_seq_stride;

    // Pass 1: the first kTokPerThread * blockDim tokens stay in registers
    // (index, coordinates, destination block) for pass 2.
    int m_r[kTokPerThread];
    int c_r[kTokPerThread][3];
    int32_t blk_r[kTokPerThread];
#pragma unroll
    for (int u = 0; u < kTokPerThread; ++u) {
        const int j = x.beg + threadIdx.x + u * blockDim.x;
        m_r[u] = j < x.end ? a.idx[j] : -1;
        blk_r[u] = j < x.end ? block_of(a, x, x.clen + (j - x.t0)) : -1;
    }
#pragma unroll
    for (int u = 0; u < kTokPerThread; ++u) load_coords(crd, m_r[u], a.n_tokens, c_r[u]);

    int mn[3] = {INT_MAX, INT_MAX, INT_MAX};
    int mx[3] = {INT_MIN, INT_MIN, INT_MIN};
    if (a.mode == PRCR_MODE_PCR) {
#pragma unroll
        for (int u = 0; u < kTokPerThread; ++u) {
            if (m_r[u] >= 0 && m_r[u] < a.n_tokens) {
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    mn[ax] = min(mn[ax], c_r[u][ax]);
                    mx[ax] = max(mx[ax], c_r[u][ax]);
                }
            }
        }
        for (int j = x.beg + kTokPerThread * blockDim.x + threadIdx.x; j < x.end; j += blockDim.x) {
            int c[3];
            const int m = a.idx[j];
            if (m >= 0 && m < a.n_tokens) {
                load_coords(crd, m, a.n_tokens, c);
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    mn[ax] = min(mn[ax], c[ax]);
                    mx[ax] = max(mx[ax], c[ax]);
                }
            }
        }
        block_minmax(mn, mx, s_part);
    }
#pragma unroll
    for (int ax = 0; ax < 3; ++ax) {
        x.lo[ax] = mn[ax];
        x.hi[ax] = mx[ax];
        const int64_t span = int64_t(mx[ax]) - int64_t(mn[ax]);
        x.tab[ax] = a.mode == PRCR_MODE_PCR && span >= 0 && span < kPosTable;
    }

    // A PCR position depends on the token only through c - lo: tabulate the
    // span + 1 exact values of each axis once (one division each).
    if (a.mode == PRCR_MODE_PCR) {
        const int n0 = x.tab[0] ? x.hi[0] - x.lo[0] + 1 : 0;
        const int n1 = x.tab[1] ? x.hi[1] - x.lo[1] + 1 : 0;
        const int n2 = x.tab[2] ? x.hi[2] - x.lo[2] + 1 : 0;
        for (int e = threadIdx.x; e < n0 + n1 + n2; e += blockDim.x) {
            const int ax = e < n0 ? 0 : (e < n0 + n1 ? 1 : 2);
            const int d = e - (ax == 0 ? 0 : (ax == 1 ? n0 : n0 + n1));
            s_tab[ax][d] = pcr_position(x.p, a.L, x.K, x.lo[ax] + d, x.lo[ax], x.hi[ax], x.center,
                                        err);
        }
        __syncthreads();
    }

    // Pass 2: positions, slots and row offsets.
#pragma unroll
    for (int u = 0; u < kTokPerThread; ++u) {
        const int j = x.beg + threadIdx.x + u * blockDim.x;
        if (j < x.end) place_token(a, x, s_tab, j, m_r[u], c_r[u], blk_r[u], err);
    }
    for (int j = x.beg + kTokPerThread * blockDim.x + threadIdx.x; j < x.end; j += blockDim.x) {
        const int m = a.idx[j];
        int c[3];
        load_coords(crd, m, a.n_tokens, c);
        place_token(a, x, s_tab, j, m, c, block_of(a, x, x.clen + (j - x.t0)), err);
    }
    if (a.mode == PRCR_MODE_PCR) __syncthreads();  // s_tab is reused by the next revisit
}

__global__ void __launch_bounds__(kPlanThreads) plan_kernel(const __grid_constant__ PlanArgs a) {
    // The rebind grid may start launching now; it waits for this grid to
    // finish (griddepcontrol.wait) before it reads the plan.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ int s_part[33 * 6];
    __shared__ double s_tab[3][kPosTable];
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

    for (int r = blockIdx.x; r < a.n_revisits; r += gridDim.x) plan_revisit(a, r, s_part, s_tab, err);

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
