// Small-batch revisit path in one kernel (Algorithm 1 end to end).
//
// For a few revisits of modest size the two-kernel path is pure latency: the
// plan kernel, the wait for it, and the rebind kernel's reload of the plan.
// Here every CTA plans the tokens it moves itself. It first checks the whole
// offset structure (small by construction: the host sends only batches of a
// few revisits here), so that a malformed batch is reported and writes
// nothing, exactly as on the two-kernel path; then, for each revisit its
// tokens belong to, it reduces the revisit's coordinate range cooperatively
// and gives its tokens their positions, slots and rows with the same exact
// arithmetic as the plan kernel (token_plan); then it streams the rows as the
// rebind kernel does.
#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

constexpr int kFusedMaxTile = 256;  // tokens per CTA (256 / lanes at most)

__global__ void __launch_bounds__(512) fused_kernel(const __grid_constant__ FusedArgs fa) {
    const PlanArgs& a = fa.plan;
    const RebindArgs& rb = fa.rebind;
    extern __shared__ float smem[];
    __shared__ int64_t s_src[kFusedMaxTile], s_dst[kFusedMaxTile];
    __shared__ double s_pos[3 * kFusedMaxTile];
    __shared__ int s_part[33 * 6];
    __shared__ int s_bad;
    const bool lead = blockIdx.x == 0 && blockIdx.y == 0;

    // 0. the per-sequence inputs are prefetched while the grid this one
    // depends on finishes; this thread's token index is requested before the
    // offsets are checked, so that their latencies overlap
    pdl_allow();
    const int T = rb.tok_per_cta;
    const int64_t tok0 = int64_t(blockIdx.x) * T;
    const int lanes = rb.lanes;
    const int my_t = threadIdx.x / lanes;
    const int64_t my_j = tok0 + my_t;
    const bool my_tok = my_t < T && my_j < a.total_k;
    if (threadIdx.x < a.n_seqs) {
        prefetch_l2(a.cache_len_in + threadIdx.x);
        prefetch_l2(a.p_txt + threadIdx.x);
    }
    pdl_wait();
    const int my_m = my_tok ? a.idx[my_j] : -1;

    // 1. the offsets: monotone, spanning [0, total_k) and [0, n_revisits)
    if (threadIdx.x == 0) s_bad = 0;
    __syncthreads();
    bool bad = false;
    for (int i = threadIdx.x; i < a.n_seqs; i += blockDim.x) {
        const int r0 = a.seq_rev_off[i], r1 = a.seq_rev_off[i + 1];
        bad |= r0 < 0 || r1 < r0 || r1 > a.n_revisits;
    }
    for (int r = threadIdx.x; r < a.n_revisits; r += blockDim.x) {
        const int t0 = a.rev_tok_off[r], t1 = a.rev_tok_off[r + 1];
        bad |= t0 < 0 || t1 < t0 || int64_t(t1) > a.total_k;
    }
    if (threadIdx.x == 0)
        bad |= a.seq_rev_off[0] != 0 || a.seq_rev_off[a.n_seqs] != a.n_revisits ||
               a.rev_tok_off[0] != 0 || int64_t(a.rev_tok_off[a.n_revisits]) != a.total_k;
    if (bad) atomicOr(&s_bad, 1);
    __syncthreads();
    if (s_bad) {
        if (lead && threadIdx.x == 0) atomicOr(a.status, PRCR_ST_CSR);
        return;
    }
    // 1b. with the offsets checked (and in L1): the token's revisit and
    // sequence, then its coordinates and its first layer's rows are
    // prefetched while the revisit ranges are reduced
    if (my_tok && my_m >= 0 && my_m < a.n_tokens) {
        int r0 = 0, r1 = a.n_revisits;  // last revisit starting at or before my_j
        while (r1 - r0 > 1) {
            const int mid = (r0 + r1) >> 1;
            if (a.rev_tok_off[mid] <= my_j) r0 = mid; else r1 = mid;
        }
        int s0 = 0, s1 = a.n_seqs;  // last sequence whose first revisit is at or before r0
        while (s1 - s0 > 1) {
            const int mid = (s0 + s1) >> 1;
            if (a.seq_rev_off[mid] <= r0) s0 = mid; else s1 = mid;
        }
        const int lane = threadIdx.x - my_t * lanes;
        if (lane == 0) prefetch_l2(a.coords + int64_t(s0) * a.coord_seq_stride + 3 * int64_t(my_m));
        if (lane == 1 && a.cache_kind == PRCR_CACHE_PAGED) {
            // the block-table entry of the token's slot (as token_plan finds it)
            const int64_t slot = int64_t(a.cache_len_in[s0]) + (my_j - a.rev_tok_off[a.seq_rev_off[s0]]);
            if (slot >= 0 && slot < int64_t(a.bt_stride) * a.block_size)
                prefetch_l2(a.block_table + int64_t(s0) * a.bt_stride + slot / a.block_size);
        }
        const int vph = rb.head_dim >> 4;
        const int64_t row = int64_t(s0) * a.store_seq_stride + int64_t(my_m) * a.store_token_stride +
                            int64_t(blockIdx.y) * rb.layers_per_cta * rb.store_layer_stride +
                            int64_t(lane / vph) * rb.head_dim + (lane % vph) * 8;
        prefetch_l2(rb.store_k + row);
        prefetch_l2(rb.store_k + row + (rb.head_dim >> 1));
        prefetch_l2(rb.store_v + row);
        prefetch_l2(rb.store_v + row + (rb.head_dim >> 1));
    }
    uint32_t err = 0;
    if (lead) {
        for (int b = threadIdx.x; b < a.n_seqs; b += blockDim.x) {
            const int64_t k = int64_t(a.rev_tok_off[a.seq_rev_off[b + 1]]) - a.rev_tok_off[a.seq_rev_off[b]];
            const int64_t len = int64_t(a.cache_len_in[b]) + k;
            if (len > INT_MAX) err |= PRCR_ST_CAPACITY;
            a.cache_len_out[b] = int32_t(len > INT_MAX ? INT_MAX : len);
            const int64_t p = a.p_txt[b];
            a.next_pos_out[b] = a.mode == PRCR_MODE_LPA ? p + k + 1 : p + 1;
        }
    }

    // 2. plan of this CTA's tokens [tok0, tok1)
    const int64_t tok1 = min(tok0 + T, a.total_k);
    int ra = 0, hi = a.n_revisits;  // last revisit starting at or before tok0
    while (hi - ra > 1) {
        const int mid = (ra + hi) >> 1;
        if (a.rev_tok_off[mid] <= tok0) ra = mid; else hi = mid;
    }
    for (int r = ra; r < a.n_revisits && a.rev_tok_off[r] < tok1; ++r) {
        RevisitCtx x;
        revisit_ctx(a, r, x);  // consistent: checked above
        if (x.K == 0) continue;
        const int32_t* crd = a.coords + int64_t(x.b) * a.coord_seq_stride;
        int mn[3] = {INT_MAX, INT_MAX, INT_MAX};
        int mx[3] = {INT_MIN, INT_MIN, INT_MIN};
        if (a.mode == PRCR_MODE_PCR) {
            for (int j = x.beg + threadIdx.x; j < x.end; j += blockDim.x) {
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
#pragma unroll
        for (int ax = 0; ax < 3; ++ax) {
            x.lo[ax] = mn[ax];
            x.hi[ax] = mx[ax];
            x.tab[ax] = false;
        }
        revisit_exactness(a, x);
        const int64_t j0 = max(int64_t(x.beg), tok0), j1 = min(int64_t(x.end), tok1);
        for (int64_t j = j0 + threadIdx.x; j < j1; j += blockDim.x) {
            const int m = a.idx[j];
            int c[3];
            load_coords(crd, m, a.n_tokens, c);
            double pos[3];
            int64_t src, dst, slot;
            token_plan(a, x, nullptr, int(j), m, c, block_of(a, x, x.clen + (j - x.t0)), err, pos,
                       src, dst, slot);
            const int t = int(j - tok0);
            s_src[t] = src;
            s_dst[t] = dst;
            s_pos[3 * t] = pos[0];
            s_pos[3 * t + 1] = pos[1];
            s_pos[3 * t + 2] = pos[2];
            if (blockIdx.y == 0) {
                if (a.pos_out) {
                    a.pos_out[3 * j] = pos[0];
                    a.pos_out[3 * j + 1] = pos[1];
                    a.pos_out[3 * j + 2] = pos[2];
                }
                if (a.slot_out) a.slot_out[j] = int32_t(slot > INT_MAX ? INT_MAX : slot);
            }
        }
    }
    if (err && blockIdx.y == 0) atomicOr(a.status, err);
    __syncthreads();

    // 3. cos/sin of the tile, then 4. the rows (as in the rebind kernel)
    const int D = rb.head_dim;
    const int P = D >> 1;
    float* cos_s = smem;
    float* sin_s = smem + T * P;
    for (int q = threadIdx.x; q < T * P; q += blockDim.x) {
        const int t = q / P;
        const int i = q - t * P;
        float c = 1.0f, s = 0.0f;
        if (tok0 + t < tok1) {
            const int ax = pair_axis(i, rb.layout, rb.sec_t, rb.sec_h, rb.sec_w);
            sincos_turns(s_pos[3 * t + ax], rb.turn_freq[i], &s, &c);
        }
        cos_s[q] = c;
        sin_s[q] = s;
    }
    __syncthreads();

    const int t = threadIdx.x / lanes;
    const int lane = threadIdx.x - t * lanes;
    if (t >= T || tok0 + t >= tok1) return;
    const int64_t dst = s_dst[t];
    if (dst < 0) return;
    const int64_t src = s_src[t];
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
    const int l0 = blockIdx.y * rb.layers_per_cta;
    const int l1 = min(l0 + rb.layers_per_cta, rb.n_layers);
    const int64_t sls = rb.store_layer_stride;
    const int64_t cls = rb.cache_layer_stride;
    stream_layers(rb.store_k + src + int64_t(l0) * sls + off, rb.store_v + src + int64_t(l0) * sls + off,
                  rb.cache_k + dst + int64_t(l0) * cls + off, rb.cache_v + dst + int64_t(l0) * cls + off,
                  sls, cls, P, l1 - l0, c, s);
}

}  // namespace

cudaError_t fused_blocks_per_sm(int block, size_t smem, int* out) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, fused_kernel, block, smem);
}

cudaError_t launch_fused(const FusedArgs& a, dim3 grid, int block, size_t smem,
                         cudaStream_t stream) {
    return launch_pdl(fused_kernel, grid, dim3(block), smem, stream, a);
}

}  // namespace prcr
