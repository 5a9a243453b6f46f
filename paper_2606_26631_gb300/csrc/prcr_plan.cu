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

#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

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

__device__ __forceinline__ void place_token(const PlanArgs& a, const RevisitCtx& r,
                                            const double (*tab)[kPosTable], int j, int m,
                                            const int (&c)[3], int32_t blk, uint32_t& err) {
    double pos[3];
    int64_t src, dst, slot;
    token_plan(a, r, tab, j, m, c, blk, err, pos, src, dst, slot);
    emit(a, j, slot, src, dst, pos);
}

__device__ void plan_revisit(const PlanArgs& a, int r, int* s_part, double (*s_tab)[kPosTable],
                             uint32_t& err) {
    RevisitCtx x;
    if (!revisit_ctx(a, r, x)) {  // uniform over the CTA
        err |= PRCR_ST_CSR;
        return;
    }
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
    revisit_exactness(a, x);

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
    pdl_allow();
    pdl_wait();
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
    return launch_pdl(plan_kernel, dim3(unsigned(grid)), dim3(kPlanThreads), 0, stream, a);
}

}  // namespace prcr
