// Small-batch revisit path in one kernel (Algorithm 1 end to end).
//
// For a few revisits of modest size the two-kernel path is pure latency: the
// plan kernel, the wait for it, and the rebind kernel's reload of the plan.
// Here every CTA plans the tokens it moves itself, with as few dependent
// memory round trips as the data allow:
//   A. the offsets, text positions, cache lengths and every selected index of
//      the batch (at most kFusedMaxTokens) are loaded into shared memory in
//      one round trip, and the offsets are checked there: a malformed batch
//      is reported and writes nothing, exactly as on the two-kernel path;
//   B. the first rows of the CTA's own tokens, their block-table entries and
//      coordinates, and the coordinates of every token of the revisits the
//      tile touches are requested together;
//   C. per revisit the coordinate range is reduced (Eq. "selected_coord_range")
//      and the positions of Eq. "image_range_fractional_reinsert" (or the
//      rule the mode selects) are formed with the plan kernel's exact
//      arithmetic, one (token, axis) per lane: GB300's float64 pipe takes
//      many cycles per warp instruction whatever its active lanes, so the
//      divisions of a tile share warp instructions instead of following each
//      other;
//   D. cos/sin of the tile from the positions in 32.32 fixed point;
//   E. the rows already in registers are rotated and stored, and the
//      group's other layers streamed as in the rebind kernel.
// Results are bit-identical to plan + rebind.
#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

constexpr int kFusedMaxTile = 256;  // tokens per CTA (256 / lanes at most)

// Last index r in [0, n) with off[r] <= v (off non-decreasing, off[0] <= v).
__device__ __forceinline__ int last_at_or_before(const int* off, int n, int64_t v) {
    int lo = 0, hi = n;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (off[mid] <= v) lo = mid; else hi = mid;
    }
    return lo;
}

__global__ void __launch_bounds__(512) fused_kernel(const __grid_constant__ FusedArgs fa) {
    const PlanArgs& a = fa.plan;
    const RebindArgs& rb = fa.rebind;
    extern __shared__ float smem[];  // cos / sin of the tile
    __shared__ int s_idx[kFusedMaxTokens];
    __shared__ int s_rto[kFusedMaxRevisits + 1];
    __shared__ int s_sro[kFusedMaxSeqs + 1];
    __shared__ long long s_p[kFusedMaxSeqs];
    __shared__ int s_clen[kFusedMaxSeqs];
    __shared__ long long s_pf[kFusedMaxTile][3];  // positions in 32.32 fixed point
    __shared__ int s_c[kFusedMaxTile][3];         // stored coordinates of the tile's tokens
    __shared__ long long s_dst[kFusedMaxTile];    // cache row (layer term excluded), -1 = skip
    __shared__ int s_skip[kFusedMaxTile];         // position out of range: rows skipped
    __shared__ int s_part[33 * 6];

    const int tid = threadIdx.x, bd = blockDim.x;
    const bool lead = blockIdx.x == 0 && blockIdx.y == 0;
    const int T = rb.tok_per_cta;
    const int lanes = rb.lanes;
    const int64_t tok0 = int64_t(blockIdx.x) * T;
    const int total = int(a.total_k);
    const int64_t tok1 = min(tok0 + T, int64_t(total));
    const int n_seqs = a.n_seqs, n_rev = a.n_revisits;

    // 0. the per-sequence inputs are requested into L2 while the grid this
    // one depends on finishes
    pdl_allow();
    if (tid < n_seqs) {
        prefetch_l2(a.cache_len_in + tid);
        prefetch_l2(a.p_txt + tid);
    }
    pdl_wait();

    // A. offsets, positions, lengths and indices into shared memory, one
    // round trip (loads first, then the shared stores)
    {
        int ro = 0, so = 0, cl = 0;
        long long pt = 0;
        if (tid <= n_rev) ro = a.rev_tok_off[tid];
        if (tid <= n_seqs) so = a.seq_rev_off[tid];
        if (tid < n_seqs) {
            pt = a.p_txt[tid];
            cl = a.cache_len_in[tid];
        }
        for (int base = 0; base < total; base += 8 * bd) {
            int v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = base + tid + u * bd;
                v[u] = i < total ? a.idx[i] : 0;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = base + tid + u * bd;
                if (i < total) s_idx[i] = v[u];
            }
        }
        if (tid <= n_rev) s_rto[tid] = ro;
        if (tid <= n_seqs) s_sro[tid] = so;
        if (tid < n_seqs) {
            s_p[tid] = pt;
            s_clen[tid] = cl;
        }
    }
    __syncthreads();
    // the offsets: monotone, spanning [0, total_k) and [0, n_revisits)
    bool bad = false;
    if (tid < n_seqs) bad = s_sro[tid] < 0 || s_sro[tid + 1] < s_sro[tid] || s_sro[tid + 1] > n_rev;
    if (tid < n_rev) bad |= s_rto[tid] < 0 || s_rto[tid + 1] < s_rto[tid] || s_rto[tid + 1] > total;
    if (tid == 0)
        bad |= s_sro[0] != 0 || s_sro[n_seqs] != n_rev || s_rto[0] != 0 || s_rto[n_rev] != total;
    if (__syncthreads_or(bad)) {
        if (lead && tid == 0) atomicOr(a.status, PRCR_ST_CSR);
        return;
    }

    uint32_t err = 0;
    if (lead) {
        for (int b = tid; b < n_seqs; b += bd) {
            const int64_t k = int64_t(s_rto[s_sro[b + 1]]) - s_rto[s_sro[b]];
            const int64_t len = int64_t(s_clen[b]) + k;
            if (len > INT_MAX) err |= PRCR_ST_CAPACITY;
            a.cache_len_out[b] = int32_t(len > INT_MAX ? INT_MAX : len);
            a.next_pos_out[b] = a.mode == PRCR_MODE_LPA ? s_p[b] + k + 1 : s_p[b] + 1;
        }
    }

    // B. this thread's token: its sequence, index, slot and source row; the
    // first layers' rows go to registers now, the block-table entry and the
    // coordinates (lane 0) to shared memory
    const int D = rb.head_dim;
    const int P = D >> 1;
    const int my_t = tid / lanes;
    const int lane = tid - my_t * lanes;
    const int64_t my_j = tok0 + my_t;
    const bool my_tok = my_t < T && my_j < tok1;
    const int l0 = blockIdx.y * rb.layers_per_cta;
    const int l1 = min(l0 + rb.layers_per_cta, rb.n_layers);
    const int64_t sls = rb.store_layer_stride;
    const int64_t cls = rb.cache_layer_stride;
    const int vph = D >> 4;
    const int64_t off = int64_t(lane / vph) * D + (lane % vph) * 8;
    uint4 k0a = {}, k1a = {}, v0a = {}, v1a = {}, k0b = {}, k1b = {}, v0b = {}, v1b = {};
    int my_m = -1;
    int my_b = 0;
    int64_t my_slot = 0;
    if (my_tok) {
        const int r = last_at_or_before(s_rto, n_rev, my_j);
        my_b = last_at_or_before(s_sro, n_seqs, r);
        my_m = s_idx[my_j];
        my_slot = int64_t(s_clen[my_b]) + (my_j - s_rto[s_sro[my_b]]);
        if (my_m >= 0 && my_m < a.n_tokens) {
            const int64_t src = int64_t(my_b) * a.store_seq_stride + int64_t(my_m) * a.store_token_stride;
            const uint16_t* sk = rb.store_k + src + int64_t(l0) * sls + off;
            const uint16_t* sv = rb.store_v + src + int64_t(l0) * sls + off;
            k0a = ld_stream(sk);
            k1a = ld_stream(sk + P);
            v0a = ld_stream(sv);
            v1a = ld_stream(sv + P);
            if (l0 + 1 < l1) {
                k0b = ld_stream(sk + sls);
                k1b = ld_stream(sk + sls + P);
                v0b = ld_stream(sv + sls);
                v1b = ld_stream(sv + sls + P);
            }
            for (int l = l0 + 2; l < l1 && l < l0 + 4; ++l) {  // the next two layers into L2
                prefetch_l2(sk + int64_t(l - l0) * sls);
                prefetch_l2(sk + int64_t(l - l0) * sls + P);
                prefetch_l2(sv + int64_t(l - l0) * sls);
                prefetch_l2(sv + int64_t(l - l0) * sls + P);
            }
        }
        if (lane == 0) {
            // the token's coordinates and its cache row
            int c[3];
            load_coords(a.coords + int64_t(my_b) * a.coord_seq_stride, my_m, a.n_tokens, c);
            const int64_t capacity = a.cache_kind == PRCR_CACHE_CONTIGUOUS
                                         ? int64_t(a.max_slots)
                                         : int64_t(a.bt_stride) * a.block_size;
            const bool slot_ok = s_clen[my_b] >= 0 && my_slot < capacity;
            int32_t blk = -1;
            if (a.cache_kind == PRCR_CACHE_PAGED && slot_ok)
                blk = a.block_table[int64_t(my_b) * a.bt_stride + my_slot / a.block_size];
            s_c[my_t][0] = c[0];
            s_c[my_t][1] = c[1];
            s_c[my_t][2] = c[2];
            s_skip[my_t] = 0;
            int64_t dst = -1;
            if (my_m < 0 || my_m >= a.n_tokens) {
                err |= PRCR_ST_IDX_RANGE;
            } else if (!slot_ok) {
                err |= PRCR_ST_CAPACITY;
            } else if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
                dst = int64_t(my_b) * a.cache_seq_stride + my_slot * a.slot_stride;
            } else if (blk < 0 || blk >= a.n_blocks) {
                err |= PRCR_ST_NO_BLOCK;
            } else {
                const int64_t lb = my_slot / a.block_size;
                dst = int64_t(blk) * a.block_stride + (my_slot - lb * a.block_size) * a.slot_stride;
            }
            s_dst[my_t] = dst;
            if (blockIdx.y == 0 && a.slot_out)
                a.slot_out[my_j] = int32_t(my_slot > INT_MAX ? INT_MAX : my_slot);
        }
    }

    // C. per revisit the tile touches: its coordinate range, then the
    // positions of its tokens in the tile, one (token, axis) per thread
    const int ra = last_at_or_before(s_rto, n_rev, tok0);
    for (int r = ra; r < n_rev && s_rto[r] < tok1; ++r) {
        const int beg = s_rto[r], end = s_rto[r + 1];
        if (end == beg) continue;
        const int b = last_at_or_before(s_sro, n_seqs, r);
        const int t0s = s_rto[s_sro[b]];  // the sequence's first token in this call
        int mn[3] = {INT_MAX, INT_MAX, INT_MAX};
        int mx[3] = {INT_MIN, INT_MIN, INT_MIN};
        if (a.mode == PRCR_MODE_PCR) {
            const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride;
            for (int j = beg + tid; j < end; j += bd) {
                const int m = s_idx[j];
                if (m >= 0 && m < a.n_tokens) {
#pragma unroll
                    for (int ax = 0; ax < 3; ++ax) {
                        const int c = crd[3 * int64_t(m) + ax];
                        mn[ax] = min(mn[ax], c);
                        mx[ax] = max(mx[ax], c);
                    }
                }
            }
            block_minmax(mn, mx, s_part);  // ends with a barrier: s_c, s_dst are visible
        } else {
            __syncthreads();  // s_c, s_dst are visible
        }
        const int64_t K = end - beg;
        const int64_t p = s_p[b];
        const bool center = (a.flags & PRCR_FLAG_DEGENERATE_CENTER) != 0;
        const int j0 = max(beg, int(tok0)), j1 = min(end, int(tok1));
        for (int q = tid; q < 3 * (j1 - j0); q += bd) {
            const int j = j0 + q / 3, ax = q - (q / 3) * 3;
            const int t = j - int(tok0);
            const int m = s_idx[j];
            double pos;
            uint32_t e = 0;
            if (m < 0 || m >= a.n_tokens) {
                pos = __longlong_as_double(0x7ff8000000000000LL);
            } else {
                switch (a.mode) {
                    case PRCR_MODE_PCR: {
                        // (selects, not an indexed register array: no local memory)
                        const int lo = ax == 0 ? mn[0] : (ax == 1 ? mn[1] : mn[2]);
                        const int hi = ax == 0 ? mx[0] : (ax == 1 ? mx[1] : mx[2]);
                        pos = pcr_position(p, a.L, K, s_c[t][ax], lo, hi, center, e);
                        break;
                    }
                    case PRCR_MODE_ORIGINAL:
                        pos = double(s_c[t][ax]);
                        break;
                    case PRCR_MODE_UIR:
                        pos = uir_position(p, int64_t(j - beg + 1), K, e);
                        break;
                    default:  // PRCR_MODE_LPA: p + rank in sequence + 1
                        pos = double(p + (j - t0s) + 1);
                        break;
                }
                // the angle reduction needs |position| < 2^31, and a position
                // must be the correctly rounded exact value: else the token's
                // rows are skipped
                if (e || !pos_in_range(pos)) {
                    err |= PRCR_ST_POS_RANGE;
                    s_skip[t] = 1;
                }
            }
            s_pf[t][ax] = fixed_32_32(pos);
            if (blockIdx.y == 0 && a.pos_out) a.pos_out[3 * int64_t(j) + ax] = pos;
        }
    }
    if (err && blockIdx.y == 0) atomicOr(a.status, err);
    __syncthreads();

    // D. cos/sin of the tile
    float* cos_s = smem;
    float* sin_s = smem + T * P;
    for (int q = tid; q < T * P; q += bd) {
        const int t = q / P;
        const int i = q - t * P;
        float c = 1.0f, s = 0.0f;
        if (tok0 + t < tok1) {
            const int ax = pair_axis(i, rb.layout, rb.sec_t, rb.sec_h, rb.sec_w);
            sincos_fixed(s_pf[t][ax], rb.turn_freq[i], &s, &c);
        }
        cos_s[q] = c;
        sin_s[q] = s;
    }
    __syncthreads();

    // E. the rows: rotate and store the layers in registers, stream the rest
    if (!my_tok) return;
    const int64_t dst = s_dst[my_t];
    if (dst < 0 || s_skip[my_t]) return;
    const int v = lane % vph;
    float c[8], s[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        c[e] = cos_s[my_t * P + v * 8 + e];
        s[e] = sin_s[my_t * P + v * 8 + e];
    }
    uint16_t* ck = rb.cache_k + dst + int64_t(l0) * cls + off;
    uint16_t* cv = rb.cache_v + dst + int64_t(l0) * cls + off;
    uint4 o0, o1;
    rotate_vec(k0a, k1a, c, s, o0, o1);
    st_row(ck, o0);
    st_row(ck + P, o1);
    st_row(cv, v0a);
    st_row(cv + P, v1a);
    if (l0 + 1 < l1) {
        rotate_vec(k0b, k1b, c, s, o0, o1);
        st_row(ck + cls, o0);
        st_row(ck + cls + P, o1);
        st_row(cv + cls, v0b);
        st_row(cv + cls + P, v1b);
    }
    if (l0 + 2 < l1) {
        const int64_t src = int64_t(my_b) * a.store_seq_stride + int64_t(my_m) * a.store_token_stride;
        stream_layers(rb.store_k + src + int64_t(l0 + 2) * sls + off,
                      rb.store_v + src + int64_t(l0 + 2) * sls + off, ck + 2 * cls, cv + 2 * cls, sls,
                      cls, P, l1 - l0 - 2, c, s);
    }
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
