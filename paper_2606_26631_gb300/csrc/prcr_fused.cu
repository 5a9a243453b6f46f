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
#include <map>
#include <mutex>

#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

constexpr int kFusedMaxTile = 256;  // tokens per CTA (256 / lanes at most)

// 16 bytes global -> shared, asynchronous (L2 only). A barrier does not wait
// for it (it would wait for a plain load in flight): the copying thread waits
// with cp.async.wait_group before it reads the data itself.
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
    const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
}

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
    // dynamic: cos / sin of the tile [2][T][P] floats, then the staged rows
    // [8][blockDim] 16-byte vectors (K, K partner, V, V partner of layers
    // l0 and l0 + 1; vector k of thread tid at k * blockDim + tid)
    extern __shared__ __align__(16) float smem[];
    __shared__ int s_idx[kFusedMaxTokens];
    __shared__ int s_rto[kFusedMaxRevisits + 1];
    __shared__ int s_sro[kFusedMaxSeqs + 1];
    __shared__ long long s_p[kFusedMaxSeqs];
    __shared__ int s_clen[kFusedMaxSeqs];
    __shared__ long long s_pf[kFusedMaxTile][3];  // positions in 32.32 fixed point
    __shared__ int s_c[kFusedMaxTile][3];         // stored coordinates of the tile's tokens
    __shared__ long long s_dst[kFusedMaxTile];    // cache row (layer term excluded), -1 = skip
    __shared__ int s_skip[kFusedMaxTile];         // position out of range: rows skipped
    __shared__ int s_mm[kFusedMaxRevisits][6];    // per touched revisit: min t,h,w, max t,h,w
    __shared__ uint64_t s_tf[kMaxPairs];          // turn rates (read per pair: no divergent
                                                  // constant-bank reads in the cos/sin loop)

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
    // the revisits the tile touches, ra .. rz (meaningful once the offsets
    // are known to be well formed), and their range slots
    const int ra = last_at_or_before(s_rto, n_rev, tok0);
    const int rz = last_at_or_before(s_rto, n_rev, tok1 - 1);
    for (int i = tid; i < 6 * min(rz - ra + 1, kFusedMaxRevisits); i += bd)
        s_mm[i / 6][i % 6] = (i % 6) < 3 ? INT_MAX : INT_MIN;
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

    // B. every load of this phase is issued before any of them is used, the
    // ones that gate the positions first: the coordinates of the touched
    // revisits' tokens (for their ranges, PCR), this thread's token's
    // coordinates and block-table entry (lane 0), then its first layers'
    // rows (registers; needed only at the end)
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
    const int64_t capacity = a.cache_kind == PRCR_CACHE_CONTIGUOUS
                                 ? int64_t(a.max_slots)
                                 : int64_t(a.bt_stride) * a.block_size;
    const bool pcr = a.mode == PRCR_MODE_PCR;
    const int jb = s_rto[ra], je = s_rto[rz + 1];
    // one token of the ranges per thread (the first bd of them)
    int cmn[3] = {INT_MAX, INT_MAX, INT_MAX}, cmx[3] = {INT_MIN, INT_MIN, INT_MIN};
    int rr = -1;
    if (pcr && jb + tid < je) {
        const int j = jb + tid;
        rr = last_at_or_before(s_rto, n_rev, j);
        const int bj = last_at_or_before(s_sro, n_seqs, rr);
        const int m = s_idx[j];
        if (m >= 0 && m < a.n_tokens) {
            const int32_t* q = a.coords + int64_t(bj) * a.coord_seq_stride + 3 * int64_t(m);
#pragma unroll
            for (int ax = 0; ax < 3; ++ax) cmn[ax] = cmx[ax] = q[ax];
        }
    }
    int my_m = -1;
    int my_b = 0;
    int64_t my_slot = 0;
    bool slot_ok = false;
    int c_own[3] = {0, 0, 0};
    int32_t blk = -1;
    uint4* stage = reinterpret_cast<uint4*>(smem + 2 * T * P);
    if (my_tok) {
        const int r = last_at_or_before(s_rto, n_rev, my_j);
        my_b = last_at_or_before(s_sro, n_seqs, r);
        my_m = s_idx[my_j];
        my_slot = int64_t(s_clen[my_b]) + (my_j - s_rto[s_sro[my_b]]);
        slot_ok = s_clen[my_b] >= 0 && my_slot < capacity;
        if (lane == 0) {
            load_coords(a.coords + int64_t(my_b) * a.coord_seq_stride, my_m, a.n_tokens, c_own);
            if (a.cache_kind == PRCR_CACHE_PAGED && slot_ok)
                blk = a.block_table[int64_t(my_b) * a.bt_stride + my_slot / a.block_size];
        }
        if (my_m >= 0 && my_m < a.n_tokens) {
            const int64_t src = int64_t(my_b) * a.store_seq_stride + int64_t(my_m) * a.store_token_stride;
            const uint16_t* sk = rb.store_k + src + int64_t(l0) * sls + off;
            const uint16_t* sv = rb.store_v + src + int64_t(l0) * sls + off;
            cp_async16(stage + 0 * bd + tid, sk);
            cp_async16(stage + 1 * bd + tid, sk + P);
            cp_async16(stage + 2 * bd + tid, sv);
            cp_async16(stage + 3 * bd + tid, sv + P);
            if (l0 + 1 < l1) {
                cp_async16(stage + 4 * bd + tid, sk + sls);
                cp_async16(stage + 5 * bd + tid, sk + sls + P);
                cp_async16(stage + 6 * bd + tid, sv + sls);
                cp_async16(stage + 7 * bd + tid, sv + sls + P);
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
            for (int l = l0 + 2; l < l1 && l < l0 + 4; ++l) {  // the next two layers into L2
                prefetch_l2(sk + int64_t(l - l0) * sls);
                prefetch_l2(sk + int64_t(l - l0) * sls + P);
                prefetch_l2(sv + int64_t(l - l0) * sls);
                prefetch_l2(sv + int64_t(l - l0) * sls + P);
            }
        }
    }
    // coordinate ranges of the touched revisits (Eq. "selected_coord_range"):
    // warp reductions when a warp's tokens share a revisit, then shared atomics
    if (pcr) {
        const int wl = tid & 31;
        for (int base = jb; base < je; base += bd) {
            if (base != jb) {  // tokens beyond the first bd
                const int j = base + tid;
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    cmn[ax] = INT_MAX;
                    cmx[ax] = INT_MIN;
                }
                rr = -1;
                if (j < je) {
                    rr = last_at_or_before(s_rto, n_rev, j);
                    const int bj = last_at_or_before(s_sro, n_seqs, rr);
                    const int m = s_idx[j];
                    if (m >= 0 && m < a.n_tokens) {
                        const int32_t* q = a.coords + int64_t(bj) * a.coord_seq_stride + 3 * int64_t(m);
#pragma unroll
                        for (int ax = 0; ax < 3; ++ax) cmn[ax] = cmx[ax] = q[ax];
                    }
                }
            }
            const int r0 = __shfl_sync(0xffffffffu, rr, 0);
            if (__all_sync(0xffffffffu, rr == r0 || rr < 0)) {
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    cmn[ax] = __reduce_min_sync(0xffffffffu, cmn[ax]);
                    cmx[ax] = __reduce_max_sync(0xffffffffu, cmx[ax]);
                }
                if (wl == 0 && r0 >= 0) {
#pragma unroll
                    for (int ax = 0; ax < 3; ++ax) {
                        atomicMin(&s_mm[r0 - ra][ax], cmn[ax]);
                        atomicMax(&s_mm[r0 - ra][3 + ax], cmx[ax]);
                    }
                }
            } else if (rr >= 0) {
#pragma unroll
                for (int ax = 0; ax < 3; ++ax) {
                    atomicMin(&s_mm[rr - ra][ax], cmn[ax]);
                    atomicMax(&s_mm[rr - ra][3 + ax], cmx[ax]);
                }
            }
        }
    }
    // the turn rates (read per pair in the cos/sin loop; loaded here, where
    // the threads wait for their coordinates anyway)
    if (tid < P) s_tf[tid] = rb.turn_freq[tid];
    // the token's cache row (lane 0)
    if (my_tok && lane == 0) {
        s_c[my_t][0] = c_own[0];
        s_c[my_t][1] = c_own[1];
        s_c[my_t][2] = c_own[2];
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
    __syncthreads();

    // C. positions of the tile's tokens (Eq. "normalized_coord",
    // "image_range_fractional_reinsert", or the rule the mode selects), one
    // (token, axis) per thread
    const bool center = (a.flags & PRCR_FLAG_DEGENERATE_CENTER) != 0;
    for (int q = tid; q < 3 * int(tok1 - tok0); q += bd) {
        const int t = q / 3, ax = q - (q / 3) * 3;
        const int j = int(tok0) + t;
        const int r = last_at_or_before(s_rto, n_rev, j);
        const int b = last_at_or_before(s_sro, n_seqs, r);
        const int beg = s_rto[r];
        const int64_t K = s_rto[r + 1] - beg;
        const int64_t p = s_p[b];
        const int m = s_idx[j];
        double pos;
        uint32_t e = 0;
        if (m < 0 || m >= a.n_tokens) {
            pos = __longlong_as_double(0x7ff8000000000000LL);
        } else {
            switch (a.mode) {
                case PRCR_MODE_PCR:
                    pos = pcr_position(p, a.L, K, s_c[t][ax], s_mm[r - ra][ax], s_mm[r - ra][3 + ax],
                                       center, e);
                    break;
                case PRCR_MODE_ORIGINAL:
                    pos = double(s_c[t][ax]);
                    break;
                case PRCR_MODE_UIR:
                    pos = uir_position(p, int64_t(j - beg + 1), K, e);
                    break;
                default:  // PRCR_MODE_LPA: p + rank in sequence + 1
                    pos = double(p + (j - s_rto[s_sro[b]]) + 1);
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
            sincos_fixed(s_pf[t][ax], s_tf[i], &s, &c);
        }
        cos_s[q] = c;
        sin_s[q] = s;
    }
    __syncthreads();

    // E. the rows: rotate and store the staged layers, stream the rest (a
    // thread waits for its own copies before it may leave: the stage must
    // not be released with copies in flight)
    asm volatile("cp.async.wait_group 0;" ::: "memory");
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
    rotate_vec(stage[0 * bd + tid], stage[1 * bd + tid], c, s, o0, o1);
    st_row(ck, o0);
    st_row(ck + P, o1);
    st_row(cv, stage[2 * bd + tid]);
    st_row(cv + P, stage[3 * bd + tid]);
    if (l0 + 1 < l1) {
        rotate_vec(stage[4 * bd + tid], stage[5 * bd + tid], c, s, o0, o1);
        st_row(ck + cls, o0);
        st_row(ck + cls + P, o1);
        st_row(cv + cls, stage[6 * bd + tid]);
        st_row(cv + cls + P, stage[7 * bd + tid]);
    }
    if (l0 + 2 < l1) {
        const int64_t src = int64_t(my_b) * a.store_seq_stride + int64_t(my_m) * a.store_token_stride;
        stream_layers(rb.store_k + src + int64_t(l0 + 2) * sls + off,
                      rb.store_v + src + int64_t(l0 + 2) * sls + off, ck + 2 * cls, cv + 2 * cls, sls,
                      cls, P, l1 - l0 - 2, c, s);
    }
}

// The kernel's dynamic shared-memory limit raised to `smem` on the current
// device (once per device and size: the attribute is set only when a larger
// size is first needed).
cudaError_t fused_smem_limit(size_t smem) {
    static std::mutex mu;
    static std::map<int, size_t> done;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> g(mu);
    size_t& have = done[dev];
    if (have >= smem) return cudaSuccess;
    e = cudaFuncSetAttribute(fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e == cudaSuccess) have = smem;
    return e;
}

}  // namespace

cudaError_t fused_blocks_per_sm(int block, size_t smem, int* out) {
    const cudaError_t e = fused_smem_limit(smem);
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, fused_kernel, block, smem);
}

cudaError_t launch_fused(const FusedArgs& a, dim3 grid, int block, size_t smem,
                         cudaStream_t stream) {
    const cudaError_t e = fused_smem_limit(smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(fused_kernel, grid, dim3(block), smem, stream, a);
}

size_t fused_stage_bytes(int block) { return size_t(8) * 16 * size_t(block); }

}  // namespace prcr
