// Attention-driven selection of the revisited set (Sec. 2.1, Eq. 3).
//
// The paper names the selection module and what it does (rank the visual
// tokens by relevance to the current decoding context, keep K of them) but
// not its formula. Reading implemented here: relevance of visual token m is
// the trigger query's attention on m at one layer, a softmax over the M
// visual tokens of RoPE(q_h, (p, p, p)) . RoPE(k_m, p_m) / sqrt(D) per query
// head h (GQA: head h reads KV head h / group), averaged over the heads. The
// K most relevant tokens (equal relevance: lower token index first) are
// written in ascending token order, one revisit per sequence, as the offsets
// and indices prcr_rebind_inject takes.
//
// A rotation preserves dot products and composes by adding angles, so
// RoPE(q, (p, p, p)) . RoPE(k, c) = q . R(c - p) k: pair i of the raw key is
// turned by theta_i (c_axis(i) - p) and dotted with the raw query, and the
// 1/sqrt(D) scale is applied to the dot product. The raw bf16 query is then
// exact in any operand format, and nothing is computed per query.
// Kernel 1 (logits, persistent) forms every (token, query head) logit that
// way from the raw key rotated on the fly, and each token tile's per-head
// softmax statistics (max, sum of exp). Kernel 2 (norm) merges the tiles'
// statistics into each head's normaliser; kernel 3 (relevance) averages
// every token's per-head softmax weight; kernel 4 (select), one CTA per
// sequence, finds the K-th largest relevance by counting against thresholds
// two bits at a time on the float bits (relevance >= 0, so bit order is
// value order) and compacts the selection in index order with block-wide
// scans.
#include <cmath>

#include "prcr_device.cuh"
#include "prcr_pdl.cuh"

namespace prcr {
namespace {

// Rotation of an integer position offset: the turn fraction c * rate mod 1
// in 0.32 fixed point is bits 32..63 of the 64-bit product c * rate (rate in
// 0.64 fixed point; the product's wrap mod 2^64 keeps those bits exact for
// any int64 c), then one sin/cos evaluation on [-pi, pi).
__device__ __forceinline__ void sincos_coord(int64_t c, uint64_t turn_freq, float* s, float* co) {
    const uint64_t prod = static_cast<uint64_t>(c) * turn_freq;
    const int frac = static_cast<int>(static_cast<uint32_t>(prod >> 32));
    __sincosf(float(frac) * 1.4629180792671596e-9f, s, co);  // 2 pi / 2^32
}

// 16-byte chunk c of a shared row stored at c ^ bit 3 of c: the 8 lanes of a
// quarter-warp that read chunks 2v (or 2v + 1), v = 0..7, hit 8 distinct
// bank groups.
__device__ __forceinline__ int swz(int c) { return c ^ ((c >> 3) & 1); }

// Logits of every (token, query head). Persistent: CTA c takes a contiguous
// run of the B * n_tiles token tiles (sequence-major), so it reloads the
// rotated queries only when its run enters a new sequence. Per tile of T
// tokens: the tile's cos/sin (one per token and pair) go to shared memory;
// then each row (token, KV head) is taken by L lanes, lane v holding pairs
// 8v..8v+7 (one 16-byte load from each half of the raw key row), which it
// rotates and dots with the group's query heads in packed float2 FMAs; the
// lanes' partial sums are reduced by shuffles. The loads of a lane's next two
// rows are in flight during the current row's arithmetic. The tile's logits are staged
// in shared memory, reduced to per-head (max, sum of exp) and written out
// coalesced.
// L lanes per row (a power of two >= head_dim / 16); G = the GQA group size g
// for g = 1, 2 and 4, else 8 (heads h >= g skipped).
template <int L, int G>
__global__ void __launch_bounds__(256, 3) ads_logits_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    pdl_wait();
    extern __shared__ __align__(16) float sm[];
    const int D = a.head_dim, P = D >> 1, Hq = a.n_q_heads, H = a.n_kv_heads, g = Hq / H;
    const int NV = P >> 3, M = a.n_tokens, T = a.tok_tile;
    const int qrow = D / 4 + 1;  // chunks per row; odd, so adjacent rows fall in other banks
    const int crow = P / 4 + 1;
    float4* q_s = reinterpret_cast<float4*>(sm);  // row h * H + kh holds query head kh * g + h
    float4* c_s = q_s + Hq * qrow;                // [T] cos rows
    float4* s_s = c_s + T * crow;                 // [T] sin rows
    float* lg_s = reinterpret_cast<float*>(s_s + T * crow);  // [Hq][T + 1]
    int* crd_s = reinterpret_cast<int*>(lg_s + Hq * (T + 1));  // [T][3]

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int v = tid & (L - 1), grp = tid / L;
    constexpr int RS = 256 / L;  // rows per pass
    const bool act = v < NV;
    const int t0_r = grp / H, kh0_r = grp - t0_r * H;  // a lane's first row in a tile
    const int dt_r = RS / H, dkh_r = RS - dt_r * H;     // its step between rows
    const int dt_e = 256 / P, di_e = 256 - dt_e * P;    // cos/sin loop step (t, i)
    const int64_t total = int64_t(a.n_seqs) * a.n_tiles;
    const int64_t t_beg = total * blockIdx.x / gridDim.x, t_end = total * (blockIdx.x + 1) / gridDim.x;
    int cur_b = -1;

    for (int64_t tile = t_beg; tile < t_end; ++tile) {
        const int b = int(tile / a.n_tiles), j = int(tile % a.n_tiles);
        const int m0 = j * T, nt = min(T, M - m0);
        if (b != cur_b) {  // the sequence's raw queries as float32 (4-byte loads)
            const uint32_t* src = reinterpret_cast<const uint32_t*>(a.q + int64_t(b) * Hq * D);
            const int nch = D / 4;
            for (int e = tid; e < Hq * nch; e += blockDim.x) {
                const int hq = e / nch, c = e - hq * nch;
                const uint32_t w0 = src[2 * e], w1 = src[2 * e + 1];
                q_s[((hq % g) * H + hq / g) * qrow + swz(c)] =
                    make_float4(lo_f32(w0), hi_f32(w0), lo_f32(w1), hi_f32(w1));
            }
            cur_b = b;
        }
        const int64_t p = a.q_pos[b];
        const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride + 3 * int64_t(m0);
        for (int e = tid; e < 3 * nt; e += blockDim.x) crd_s[e] = crd[e];
        __syncthreads();
        float* cf = reinterpret_cast<float*>(c_s);
        float* sf = reinterpret_cast<float*>(s_s);
        for (int e = tid, t = tid / P, i = tid - (tid / P) * P; e < nt * P;
             e += 256, t += dt_e, i += di_e) {
            if (i >= P) {
                i -= P;
                ++t;
            }
            const int ax = pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w);
            float sn, cn;
            sincos_coord(crd_s[3 * t + ax] - p, a.turn_freq[i], &sn, &cn);
            const int o = (t * crow + swz(i >> 2)) * 4 + (i & 3);
            cf[o] = cn;
            sf[o] = sn;
        }
        __syncthreads();

        const uint16_t* kbase = a.store_k + int64_t(b) * a.store_seq_stride +
                                int64_t(a.layer) * a.store_layer_stride + 8 * v;
        const int rows = nt * H;
        // row r = t * H + kh; a lane's rows advance by RS = dt_r * H + dkh_r.
        // Rows r + RS and r + 2 RS are in flight while row r is computed.
        int t = t0_r, kh = kh0_r;        // the row computed
        int tn = t + dt_r, khn = kh + dkh_r;  // the row two ahead, after the step below
        if (khn >= H) {
            khn -= H;
            ++tn;
        }
        uint4 lo_1 = make_uint4(0, 0, 0, 0), hi_1 = lo_1, lo_2 = lo_1, hi_2 = lo_1;
        if (grp < rows && act) {
            const uint16_t* kr = kbase + int64_t(m0 + t) * a.store_token_stride + kh * D;
            lo_1 = ld_stream(kr);
            hi_1 = ld_stream(kr + P);
        }
        if (grp + RS < rows && act) {
            const uint16_t* kr = kbase + int64_t(m0 + tn) * a.store_token_stride + khn * D;
            lo_2 = ld_stream(kr);
            hi_2 = ld_stream(kr + P);
        }
        for (int r = grp; r - grp < rows; r += RS) {
            const uint4 lo = lo_1, hi = hi_1;
            lo_1 = lo_2;
            hi_1 = hi_2;
            tn += dt_r;
            khn += dkh_r;
            if (khn >= H) {
                khn -= H;
                ++tn;
            }
            if (r + 2 * RS < rows && act) {
                const uint16_t* kr = kbase + int64_t(m0 + tn) * a.store_token_stride + khn * D;
                lo_2 = ld_stream(kr);
                hi_2 = ld_stream(kr + P);
            }
            float acc[G];
#pragma unroll
            for (int h = 0; h < G; ++h) acc[h] = 0.0f;
            if (r < rows && act) {
                const float4* cr = c_s + t * crow;
                const float4* sr = s_s + t * crow;
                const float4 ca = cr[swz(2 * v)], cb = cr[swz(2 * v + 1)];
                const float4 sa = sr[swz(2 * v)], sb = sr[swz(2 * v + 1)];
                const uint32_t lw[4] = {lo.x, lo.y, lo.z, lo.w};
                const uint32_t hw[4] = {hi.x, hi.y, hi.z, hi.w};
                const float2 c2[4] = {make_float2(ca.x, ca.y), make_float2(ca.z, ca.w),
                                      make_float2(cb.x, cb.y), make_float2(cb.z, cb.w)};
                const float2 s2[4] = {make_float2(sa.x, sa.y), make_float2(sa.z, sa.w),
                                      make_float2(sb.x, sb.y), make_float2(sb.z, sb.w)};
                float2 kx[4], ky[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    const float2 x = make_float2(__uint_as_float(lw[w] << 16),
                                                 __uint_as_float(lw[w] & 0xffff0000u));
                    const float2 y = make_float2(__uint_as_float(hw[w] << 16),
                                                 __uint_as_float(hw[w] & 0xffff0000u));
                    const float2 ys = __fmul2_rn(y, s2[w]);
                    const float2 xs = __fmul2_rn(x, s2[w]);
                    kx[w] = __ffma2_rn(x, c2[w], make_float2(-ys.x, -ys.y));
                    ky[w] = __ffma2_rn(y, c2[w], xs);
                }
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    if (G != 8 || h < g) {
                        const float4* qr = q_s + (h * H + kh) * qrow;
                        const float4 qa = qr[swz(2 * v)], qb = qr[swz(2 * v + 1)];
                        const float4 qc = qr[swz(P / 4 + 2 * v)], qd = qr[swz(P / 4 + 2 * v + 1)];
                        float2 s2a = __fmul2_rn(make_float2(qa.x, qa.y), kx[0]);
                        s2a = __ffma2_rn(make_float2(qa.z, qa.w), kx[1], s2a);
                        s2a = __ffma2_rn(make_float2(qb.x, qb.y), kx[2], s2a);
                        s2a = __ffma2_rn(make_float2(qb.z, qb.w), kx[3], s2a);
                        s2a = __ffma2_rn(make_float2(qc.x, qc.y), ky[0], s2a);
                        s2a = __ffma2_rn(make_float2(qc.z, qc.w), ky[1], s2a);
                        s2a = __ffma2_rn(make_float2(qd.x, qd.y), ky[2], s2a);
                        s2a = __ffma2_rn(make_float2(qd.z, qd.w), ky[3], s2a);
                        acc[h] = (s2a.x + s2a.y) * a.scale;
                    }
                }
            }
#pragma unroll
            for (int o = L / 2; o; o >>= 1) {
#pragma unroll
                for (int h = 0; h < G; ++h) acc[h] += __shfl_xor_sync(0xffffffffu, acc[h], o);
            }
            if (r < rows && v == 0) {
#pragma unroll
                for (int h = 0; h < G; ++h)
                    if (G != 8 || h < g) lg_s[(kh * g + h) * (T + 1) + t] = acc[h];
            }
            t += dt_r;
            kh += dkh_r;
            if (kh >= H) {
                kh -= H;
                ++t;
            }
        }
        __syncthreads();

        // per query head: the tile's (max, sum of exp), and its logits written out coalesced
        for (int hq = warp; hq < Hq; hq += blockDim.x >> 5) {
            const float* row = lg_s + hq * (T + 1);
            float mx = -INFINITY;
            for (int t = lane; t < nt; t += 32) mx = fmaxf(mx, row[t]);
#pragma unroll
            for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            float z = 0.0f;
            float* dst = a.logits + (int64_t(b) * Hq + hq) * M + m0;
            for (int t = lane; t < nt; t += 32) {
                z += expf(row[t] - mx);
                dst[t] = row[t];
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
            if (lane == 0) {
                float* ts = a.tile_stats + ((int64_t(b) * Hq + hq) * a.n_tiles + j) * 2;
                ts[0] = mx;
                ts[1] = z;
            }
        }
        // the next tile rewrites the coordinates first, then (after a barrier)
        // the cos/sin rows and logits this tile's warps may still be reading
    }
}

// D += A B on tensor cores: mma.sync m16n8k8 with tf32 operands (the upper
// 19 bits of each float32 register), float32 accumulate. Fragments as the
// PTX ISA lays them out for this shape: a0 (row g, col t), a1 (row g + 8,
// col t), a2 (row g, col t + 4), a3 (row g + 8, col t + 4); b0 (row t, col
// g), b1 (row t + 4, col g); lane = 4 g + t.
__device__ __forceinline__ void mma_1688_tf32(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Tensor-core logits (head_dim 64 and 128). Persistent over work items
// (sequence, group of at most 8 KV heads, 16 NW tokens); warp w of a CTA
// takes tokens 16 w .. 16 w + 15 of the item through the group's KV heads:
//   S (16 rows = the warp's tokens; 8 columns = the GQA group's query heads,
//      columns >= g zero) = K_rot Q^T, D / 8 k-steps of mma.sync m16n8k8 (tf32),
//   K_rot the raw keys turned by the offsets of their coordinates from p.
// The dot product does not depend on the order of the dimensions, so the
// k-slots are permuted: at k-step s, lane group t (= lane & 3) holds pair
// 32 (s / 8) + 8 t + s % 8 of its two tokens (rows g and g + 8), the
// first-half dimension in k-slot t and its rotate-half partner in k-slot
// t + 4. A lane then loads each half of its two rows as 16-byte runs (the
// four lanes of a token cover 64 contiguous bytes) and rotates the two
// tokens' pairs together in packed float2 arithmetic. The cos/sin of a
// lane's (token, pair) are computed once per item into the warp's
// shared-memory table and read back for every KV head. The raw bf16 queries
// are exact tf32 operands (B, kept in shared memory in fragment order per
// (sequence, head group)); each rotated key is split into a tf32 head
// (truncation, one bit operation) and its float32 remainder (< 2^-10 of the
// value, itself truncated by the MMA), and both products are summed in
// float32: ~20 significant bits per product over float32's range. Runs of
// 16-byte loads are double-buffered: the run two ahead is requested as soon
// as a buffer's words are used. Each KV head's logits go straight from the
// accumulators to global memory; the softmax statistics are left to the
// normaliser kernel.
template <int D, int NW>
__global__ void __launch_bounds__(NW * 32, 2) ads_logits_mma_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    constexpr int P = D / 2, KS = D / 8, NR = KS / 8;  // k-steps; 16-byte runs per half row
    constexpr int T = 16 * NW;                         // tokens per work item
    static_assert(NR == 1 || NR == 2, "head_dim 64 or 128");
    extern __shared__ __align__(16) float sm[];
    const int Hq = a.n_q_heads, H = a.n_kv_heads, g = Hq / H, M = a.n_tokens;
    const int KPI = a.kh_per_item, n_khg = (H + KPI - 1) / KPI;
    const int n_it = (M + T - 1) / T;  // work items per (sequence, head group)
    uint4* qf_s = reinterpret_cast<uint4*>(sm);  // [KPI][KS / 2][32] B fragments
    float4* tr_s = reinterpret_cast<float4*>(qf_s + KPI * (KS / 2) * 32);  // [NW][KS][32]
    uint64_t* tf_s = reinterpret_cast<uint64_t*>(tr_s + NW * KS * 32);      // [P] turn rates
    float2* r8_s = reinterpret_cast<float2*>(tf_s + P);  // [P] turn of 8 w-steps; (1, 0) off the w band
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int gid = lane >> 2, tq = lane & 3;
    for (int i = tid; i < P; i += NW * 32) {
        tf_s[i] = a.turn_freq[i];
        float2 r = make_float2(1.0f, 0.0f);
        if (pair_axis(i, a.layout, a.sec_t, a.sec_h, a.sec_w) == 2) sincos_coord(8, a.turn_freq[i], &r.y, &r.x);
        r8_s[i] = r;
    }
    // axis of this lane's pair at each k-step, two bits each
    uint32_t axes = 0u;
#pragma unroll
    for (int s = 0; s < KS; ++s)
        axes |= uint32_t(pair_axis(32 * (s / 8) + 8 * tq + s % 8, a.layout, a.sec_t, a.sec_h,
                                   a.sec_w)) << (2 * s);
    // the tables above come from the arguments alone: they are set up while
    // the grid this one depends on finishes; every global input is read after
    pdl_wait();
    __syncthreads();
    // Schedule: q = total / grid whole items per CTA, a contiguous run. The
    // R = total - q * grid items left over would make R CTAs run q + 1 items;
    // when 2 R <= grid they are split instead into halves by KV heads, one
    // half per CTA, so that no CTA runs more than q + 1/2 items.
    const int64_t total = int64_t(a.n_seqs) * n_khg * n_it;
    const int64_t G = gridDim.x, q = total / G, R = total - q * G;
    const bool halves = R > 0 && 2 * R <= G && KPI > 1;
    const int64_t c = blockIdx.x;
    const int64_t i_beg = halves ? c * q : total * c / G;
    const int64_t i_end = halves ? i_beg + q : total * (c + 1) / G;
    const int n_work = int(i_end - i_beg) + (halves && c < 2 * R ? 1 : 0);
    int cur_b = -1, cur_kh = -1;
    float4* tr_w = tr_s + warp * KS * 32 + lane;
    const int64_t layer_off = int64_t(a.layer) * a.store_layer_stride + 8 * tq;

    for (int w = 0; w < n_work; ++w) {
        const bool half = i_beg + w >= i_end;
        const int64_t item = half ? q * G + c / 2 : i_beg + w;
        const int64_t bg = item / n_it;  // (sequence, KV-head group)
        const int b = int(bg / n_khg), it = int(item - bg * n_it);
        int kh_a = int(bg - int64_t(b) * n_khg) * KPI, nkh = min(KPI, H - kh_a);
        if (half) {  // the first or second half of the group's KV heads
            const int h1 = (nkh + 1) / 2;
            kh_a += (c & 1) ? h1 : 0;
            nkh = (c & 1) ? nkh - h1 : h1;
        }
        const int j = it * NW + warp;  // the warp's 16-token tile
        const int m0 = 16 * j, ntw = min(16, M - m0);
        // this lane's two tokens (rows g and g + 8 of the warp's MMA tile); a
        // token past the end reads the tile's last token (its logits are
        // never written out)
        const int ta = gid, tb = gid + 8;
        const int ma = m0 + min(ta, ntw - 1), mb = m0 + min(tb, ntw - 1);
        const uint16_t* kb = a.store_k + int64_t(b) * a.store_seq_stride + layer_off;
        const uint16_t* ra = kb + int64_t(ma) * a.store_token_stride;
        const uint16_t* rb = kb + int64_t(mb) * a.store_token_stride;
        const int n_runs = nkh * NR;
        // run r = (KV head kh_a + r / NR, 16-byte run r % NR): first-half x and
        // second-half y words of tokens a and b
        uint4 buf0[4], buf1[4];
        // run u of the KV head whose rows start at pa (token a) and pb (token
        // b): compile-time offsets from two pointers advanced by D per head
        const uint16_t* pa = ra + kh_a * D;
        const uint16_t* pb = rb + kh_a * D;
        auto fetch = [&](uint4 (&k)[4], const uint16_t* xa, const uint16_t* xb, int u) {
            k[0] = ld_stream(xa + 32 * u);
            k[1] = ld_stream(xa + 32 * u + P);
            k[2] = ld_stream(xb + 32 * u);
            k[3] = ld_stream(xb + 32 * u + P);
        };
        if (ntw > 0 && n_runs > 0) {
            fetch(buf0, pa, pb, 0);
            if (NR == 2) fetch(buf1, pa, pb, 1);
            else if (n_runs > 1) fetch(buf1, pa + D, pb + D, 0);
        }
        if (b != cur_b || kh_a != cur_kh) {
            // the group's raw queries as B fragments (a bf16 value is an exact
            // tf32 operand): entry (kh, s / 2, lane) holds k-steps s and s + 1
            __syncthreads();  // every warp is done with the previous group's
            const uint16_t* qs = a.q + int64_t(b) * Hq * D;
            for (int e = tid; e < nkh * (KS / 2) * 32; e += NW * 32) {
                const int kk = e / ((KS / 2) * 32), s2 = (e / 32) % (KS / 2), ln = e & 31;
                const int h = ln >> 2, t4 = ln & 3;
                uint4 f = make_uint4(0u, 0u, 0u, 0u);
                if (h < g) {
                    const uint16_t* qr = qs + ((kh_a + kk) * g + h) * D;
                    const int i0 = 32 * ((2 * s2) / 8) + 8 * t4 + (2 * s2) % 8;  // pair of k-step 2 s2
                    f.x = uint32_t(qr[i0]) << 16;
                    f.y = uint32_t(qr[i0 + P]) << 16;
                    f.z = uint32_t(qr[i0 + 1]) << 16;
                    f.w = uint32_t(qr[i0 + 1 + P]) << 16;
                }
                qf_s[e] = f;
            }
            cur_b = b;
            cur_kh = kh_a;
            __syncthreads();
        }
        if (ntw <= 0 || nkh <= 0) continue;  // past the sequence's last token, or no KV head

        // cos/sin of the lane's (token, pair) at each k-step, at the offsets
        // of the tokens' coordinates from the trigger position
        {
            const int32_t* crd = a.coords + int64_t(b) * a.coord_seq_stride;
            const int64_t p = a.q_pos[b];
            const int ca[3] = {crd[3 * ma], crd[3 * ma + 1], crd[3 * ma + 2]};
            const int cb[3] = {crd[3 * mb], crd[3 * mb + 1], crd[3 * mb + 2]};
            const int64_t oa[3] = {ca[0] - p, ca[1] - p, ca[2] - p};
            // Every lane's two tokens on one image row, 8 columns apart (a
            // 16-token tile within a row): token b's angles are token a's
            // turned by 8 w-steps on the w pairs and equal on the others.
            const bool row8 = __all_sync(0xffffffffu, cb[0] == ca[0] && cb[1] == ca[1] &&
                                                          int64_t(cb[2]) == int64_t(ca[2]) + 8);
            if (row8) {
#pragma unroll
                for (int s = 0; s < KS; ++s) {
                    const uint32_t ax = (axes >> (2 * s)) & 3u;
                    const int i = 32 * (s / 8) + 8 * tq + s % 8;
                    float sn, cs;
                    sincos_coord(ax == 0 ? oa[0] : (ax == 1 ? oa[1] : oa[2]), tf_s[i], &sn, &cs);
                    const float2 r = r8_s[i];
                    tr_w[s * 32] = make_float4(cs, fmaf(cs, r.x, -sn * r.y), sn, fmaf(sn, r.x, cs * r.y));
                }
            } else {
                const int64_t ob[3] = {cb[0] - p, cb[1] - p, cb[2] - p};
#pragma unroll
                for (int s = 0; s < KS; ++s) {
                    const uint32_t ax = (axes >> (2 * s)) & 3u;
                    const uint64_t rate = tf_s[32 * (s / 8) + 8 * tq + s % 8];
                    float4 t;
                    sincos_coord(ax == 0 ? oa[0] : (ax == 1 ? oa[1] : oa[2]), rate, &t.z, &t.x);
                    sincos_coord(ax == 0 ? ob[0] : (ax == 1 ? ob[1] : ob[2]), rate, &t.w, &t.y);
                    tr_w[s * 32] = t;
                }
            }
        }
        __syncwarp();

        float acc[4];
        auto clear = [&]() { acc[0] = acc[1] = acc[2] = acc[3] = 0.0f; };
        clear();
        // the eight k-steps of run u of KV head kk (words in k)
        auto run = [&](const uint4 (&k)[4], int kk, int u) {
            const uint4* qf = qf_s + (kk * (KS / 2) + 4 * u) * 32 + lane;
#pragma unroll
            for (int s8 = 0; s8 < 8; ++s8) {
                const int s = 8 * u + s8, w = s8 / 2;
                const bool up = s8 & 1;  // upper bf16 of the word
                const uint32_t wxa = word_of(k[0], w), wya = word_of(k[1], w);
                const uint32_t wxb = word_of(k[2], w), wyb = word_of(k[3], w);
                const float2 X = up ? make_float2(hi_f32(wxa), hi_f32(wxb))
                                    : make_float2(lo_f32(wxa), lo_f32(wxb));
                const float2 Y = up ? make_float2(hi_f32(wya), hi_f32(wyb))
                                    : make_float2(lo_f32(wya), lo_f32(wyb));
                const float4 t = tr_w[s * 32];
                const float2 C = make_float2(t.x, t.y), S = make_float2(t.z, t.w);
                const float2 ys = __fmul2_rn(Y, S), xs = __fmul2_rn(X, S);
                const float2 Xr = __ffma2_rn(X, C, make_float2(-ys.x, -ys.y));
                const float2 Yr = __ffma2_rn(Y, C, xs);
                // tf32 heads by truncation, float32 remainders
                const uint32_t hxa = __float_as_uint(Xr.x) & 0xffffe000u;
                const uint32_t hxb = __float_as_uint(Xr.y) & 0xffffe000u;
                const uint32_t hya = __float_as_uint(Yr.x) & 0xffffe000u;
                const uint32_t hyb = __float_as_uint(Yr.y) & 0xffffe000u;
                // remainders v - head, two per packed FMA with (-1, -1)
                const float2 lx = __ffma2_rn(make_float2(__uint_as_float(hxa), __uint_as_float(hxb)),
                                             make_float2(-1.0f, -1.0f), Xr);
                const float2 ly = __ffma2_rn(make_float2(__uint_as_float(hya), __uint_as_float(hyb)),
                                             make_float2(-1.0f, -1.0f), Yr);
                const float lxa = lx.x, lxb = lx.y, lya = ly.x, lyb = ly.y;
                const uint4 q2 = qf[(s8 / 2) * 32];
                const uint32_t b0 = up ? q2.z : q2.x, b1 = up ? q2.w : q2.y;
                mma_1688_tf32(acc, hxa, hxb, hya, hyb, b0, b1);
                mma_1688_tf32(acc, __float_as_uint(lxa), __float_as_uint(lxb),
                              __float_as_uint(lya), __float_as_uint(lyb), b0, b1);
            }
        };
        // KV head kk done: its logits out (the softmax statistics come from
        // the normaliser kernel, one pass over the logits)
        const bool va = ta < ntw, vb = tb < ntw;
        // columns 2t, 2t + 1 of each KV head's logits; lg advances by g rows per head
        const int h0 = 2 * tq;
        float* lg = a.logits + (int64_t(b) * Hq + kh_a * g + h0) * M + m0;
        const int64_t lg_step = int64_t(g) * M;
        auto finish = [&]() {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                if (h0 + c < g) {
                    if (va) lg[int64_t(c) * M + ta] = acc[c] * a.scale;
                    if (vb) lg[int64_t(c) * M + tb] = acc[2 + c] * a.scale;
                }
            }
            lg += lg_step;
            clear();
        };
        // Each buffer's next run is requested as soon as its words are used:
        // head dim 128, buffer u holds run u of the current KV head; head dim
        // 64 (one run per head), buffers take alternate heads.
        if (NR == 2) {
            for (int kk = 0; kk < nkh; ++kk) {
                run(buf0, kk, 0);
                pa += D;
                pb += D;
                if (kk + 1 < nkh) fetch(buf0, pa, pb, 0);
                run(buf1, kk, 1);
                finish();
                if (kk + 1 < nkh) fetch(buf1, pa, pb, 1);
            }
        } else {
            for (int kk = 0; kk < nkh; kk += 2) {
                run(buf0, kk, 0);
                finish();
                if (kk + 2 < nkh) fetch(buf0, pa + 2 * D, pb + 2 * D, 0);
                if (kk + 1 < nkh) {
                    run(buf1, kk + 1, 0);
                    finish();
                    if (kk + 3 < nkh) fetch(buf1, pa + 3 * D, pb + 3 * D, 0);
                }
                pa += 2 * D;
                pb += 2 * D;
            }
        }
    }
}

// Logits of the selection over the position-bound cache (head_dim 64 or
// 128). The cache already holds each visual token's key rotated at its own
// coordinates, so only the query is turned, once, at (p, p, p); the step is
// then a plain product with the cached rows and runs at memory speed. A
// warp's work item is (sequence b, KV head kh, tile of 16 tokens); items run
// (b, kh) major with tiles fastest and a warp takes a contiguous run of them,
// so it rotates its group's queries once per (b, kh). S^T (16 rows = the
// item's tokens; 8 columns = the group's query heads, columns >= g zero) =
// K Q^T over D/16 k-steps of mma.sync m16n8k16: the bf16 keys are exact
// operands and the float32 query (pre-scaled by 1/sqrt(D)) enters as a bf16
// head and a bf16 remainder (two MMAs per k-step). The key dimensions are
// permuted per lane group so that a lane loads its two tokens' 64 contiguous
// bytes each straight into A fragments. The next item's rows are loaded
// during this item's MMAs (each 16-byte run as soon as the register it goes
// into is used), the rows of the one after that requested into L2. An item
// writes its 16 logits per head (the softmax statistics are left to the
// normaliser kernel); a token without a readable row gets logit -inf.
template <int D>
__global__ void __launch_bounds__(256, D > 128 ? 1 : 2)
    ads_logits_cache_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    constexpr int KS = D / 16, LV = D / 32, P = D / 2;
    extern __shared__ __align__(16) float sm[];
    const int Hq = a.n_q_heads, H = a.n_kv_heads, g = Hq / H, M = a.n_tokens, NT = a.n_tiles;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, gid = lane >> 2, t = lane & 3;
    float* qw = sm + warp * g * D;  // this warp's rotated query rows
    const int64_t n_items = int64_t(a.n_seqs) * H * NT;
    const int64_t n_warps = int64_t(gridDim.x) * (blockDim.x >> 5);
    const int64_t gw = int64_t(blockIdx.x) * (blockDim.x >> 5) + warp;
    const int64_t i_beg = n_items * gw / n_warps, i_end = n_items * (gw + 1) / n_warps;
    uint32_t err = 0;
    pdl_wait();

    // a work item as (sequence, KV head, tile); a warp's items are consecutive,
    // so they are advanced in place rather than divided out of the index
    struct Item {
        int b, kh, j;
    };
    auto advance = [&](Item& x) {
        if (++x.j == NT) {
            x.j = 0;
            if (++x.kh == H) {
                x.kh = 0;
                ++x.b;
            }
        }
    };
    // element offset, without the KV head's D elements, of the key row of
    // token 16 j + (lane & 15) of sequence b, or -1 (past the end, or no
    // readable row). Computed once per item, when its rows are requested.
    const int64_t layer_off = int64_t(a.layer) * a.cache_layer_stride;
    // The row lookup in two halves, one item apart: start() forms the slot of
    // this lane's token and issues its block-table load (paged caches), whose
    // value finish() uses an item later, when the lookup's dependent loads
    // have long returned. The sequence's first image slot is kept per
    // sequence (items run sequence-major).
    struct RowReq {
        int64_t slot;  // -1: no row
        int32_t blk;
    };
    int s0_b = -1;
    int32_t s0_v = 0;
    auto row_start = [&](const Item& x, RowReq& q) {
        q.slot = -1;
        q.blk = 0;
        const int m = 16 * x.j + (lane & 15);
        if (m >= M) return;
        if (x.b != s0_b) {
            s0_b = x.b;
            s0_v = a.img_slot0[x.b];
        }
        const int64_t slot = int64_t(s0_v) + m;
        if (slot < 0 || slot >= a.cache_capacity) {
            err |= PRCR_ST_CAPACITY;
            return;
        }
        q.slot = slot;
        if (a.cache_kind != PRCR_CACHE_CONTIGUOUS) {
            // block index by a 32-bit division when the slot fits in 31 bits
            // (a 64-bit division costs several times as many instructions as
            // the rest of a row lookup)
            const int64_t lb = slot <= INT32_MAX ? int64_t(uint32_t(slot) / uint32_t(a.block_size))
                                                 : slot / a.block_size;
            q.blk = a.block_table[int64_t(x.b) * a.bt_stride + lb];
        }
    };
    auto row_finish = [&](const Item& x, const RowReq& q) -> int64_t {
        if (q.slot < 0) return -1;
        int64_t row;
        if (a.cache_kind == PRCR_CACHE_CONTIGUOUS) {
            row = int64_t(x.b) * a.cache_seq_stride + q.slot * a.cache_slot_stride;
        } else {
            if (q.blk < 0 || q.blk >= a.n_blocks) {
                err |= PRCR_ST_NO_BLOCK;
                return -1;
            }
            const int64_t off = q.slot <= INT32_MAX ? int64_t(uint32_t(q.slot) % uint32_t(a.block_size))
                                                    : q.slot % a.block_size;
            row = int64_t(q.blk) * a.cache_block_stride + off * a.cache_slot_stride;
        }
        return row + layer_off;
    };
    auto row_of = [&](const Item& x) -> int64_t {
        RowReq q;
        row_start(x, q);
        return row_finish(x, q);
    };
    uint4 kn[2][LV];
    uint32_t mask_n = 0u;
    // loads an item's 16 key rows (row: this lane's token, from row_of). A
    // token without a row reads the cache's first row instead: its logit is
    // set to -inf whatever the row holds (tokens are separate MMA rows).
    // this lane's two token rows (tokens gid and gid + 8) of an item, and the
    // item's row mask
    auto rows_of = [&](int64_t row, int kh, const uint16_t* (&kp)[2]) -> uint32_t {
        const uint32_t m = __ballot_sync(0xffffffffu, row >= 0) & 0xffffu;
        const int64_t r0 = (row >= 0 ? row : 0) + int64_t(kh) * D;
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
            kp[nt] = a.cache_k + __shfl_sync(0xffffffffu, r0, nt * 8 + gid) + t * (D / 4);
        return m;
    };
    auto fetch = [&](int64_t row, int kh) {
        const uint16_t* kp[2];
        mask_n = rows_of(row, kh, kp);
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
            for (int u = 0; u < LV; ++u) kn[nt][u] = ld_stream(kp[nt] + 8 * u);
        }
    };
    // the rows of the item after next are requested into L2 (lanes 0..15,
    // one token row each), so that its fetch finds them there
    auto request = [&](int64_t row, int kh) {
        if (lane < 16 && row >= 0) {
            const char* p = reinterpret_cast<const char*>(a.cache_k + row + int64_t(kh) * D);
#pragma unroll
            for (int o = 0; o < D * 2; o += 128) prefetch_l2(p + o);
        }
    };

    uint32_t qh[KS][2], ql[KS][2];
    float* lg_base[2] = {nullptr, nullptr};
    int cur_b = -1, cur_kh = -1;
    bool q_ok = true;  // the sequence's query position is within the angle range
    Item cur, nxt, pf;
    {
        const int64_t bk = i_beg / NT;
        cur.j = int(i_beg - bk * NT);
        cur.b = int(bk / H);
        cur.kh = int(bk - int64_t(cur.b) * H);
    }
    nxt = cur;
    advance(nxt);
    pf = nxt;
    advance(pf);
    int64_t row_nxt = -1, row_pf = -1;
    RowReq req_pf = {-1, 0};  // the started lookup of pf
    if (i_beg < i_end) fetch(row_of(cur), cur.kh);
    if (i_beg + 1 < i_end) {
        row_nxt = row_of(nxt);
        request(row_nxt, nxt.kh);
    }
    if (i_beg + 2 < i_end) row_start(pf, req_pf);
    for (int64_t left = i_end - i_beg; left > 0; --left) {
        const int b = cur.b, kh = cur.kh, j = cur.j;
        if (b != cur_b || kh != cur_kh) {
            // the group's queries turned at (p, p, p), pre-scaled, as A fragments
            // a query position beyond the fixed-point angle reduction is
            // reported and the sequence's logits are all -inf (relevance 0)
            const int64_t p = a.q_pos[b];
            q_ok = p > -2147483648LL && p < 2147483648LL;
            if (!q_ok) err |= PRCR_ST_POS_RANGE;
            const uint16_t* qg = a.q + (int64_t(b) * Hq + kh * g) * D;
            for (int i = lane; i < P; i += 32) {
                float sn, cs;
                sincos_turns(double(p), a.turn_freq[i], &sn, &cs);
                for (int h = 0; h < g; ++h) {
                    const float x = __uint_as_float(uint32_t(qg[h * D + i]) << 16);
                    const float y = __uint_as_float(uint32_t(qg[h * D + i + P]) << 16);
                    qw[h * D + i] = fmaf(x, cs, -y * sn) * a.scale;
                    qw[h * D + i + P] = fmaf(y, cs, x * sn) * a.scale;
                }
            }
            __syncwarp();
            const bool hv = gid < g;
            const float* qr = qw + (hv ? gid : 0) * D + t * (D / 4);
#pragma unroll
            for (int k = 0; k < KS; ++k) {
                const float x0 = hv ? qr[4 * k] : 0.0f, x1 = hv ? qr[4 * k + 1] : 0.0f;
                const float x2 = hv ? qr[4 * k + 2] : 0.0f, x3 = hv ? qr[4 * k + 3] : 0.0f;
                split_bf16x2(x0, x1, qh[k][0], ql[k][0]);
                split_bf16x2(x2, x3, qh[k][1], ql[k][1]);
            }
            __syncwarp();  // qw is rewritten for the next (b, kh)
            cur_b = b;
            cur_kh = kh;
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {  // rows of this lane's heads 2t, 2t + 1
                const int64_t r = int64_t(b) * Hq + kh * g + min(2 * t + hh, g - 1);
                lg_base[hh] = a.logits + r * M;
            }
        }
        // S^T (16 tokens x 8 columns = the group's query heads, columns >= g
        // zero) = K Q^T: rows gid (kn[0]) and gid + 8 (kn[1]) are this lane's
        // tokens, and the query fragments serve as the B operand unchanged
        const uint32_t mask = q_ok ? mask_n : 0u;
        // the next item's rows, each 16-byte run requested as soon as this
        // item's MMAs have used the registers it goes into
        const uint16_t* kp[2] = {a.cache_k, a.cache_k};
        if (left > 1) mask_n = rows_of(row_nxt, nxt.kh, kp);
        float c[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            const uint4& w0 = kn[0][k >> 1];
            const uint4& w1 = kn[1][k >> 1];
            const uint32_t a0 = (k & 1) ? w0.z : w0.x, a2 = (k & 1) ? w0.w : w0.y;
            const uint32_t a1 = (k & 1) ? w1.z : w1.x, a3 = (k & 1) ? w1.w : w1.y;
            mma_16816(c, a0, a1, a2, a3, qh[k][0], qh[k][1]);
            mma_16816(c, a0, a1, a2, a3, ql[k][0], ql[k][1]);
            if ((k & 1) && left > 1) {
                kn[0][k >> 1] = ld_stream(kp[0] + 8 * (k >> 1));
                kn[1][k >> 1] = ld_stream(kp[1] + 8 * (k >> 1));
            }
        }
        Item pf2 = pf;  // the item after pf: its lookup starts now
        advance(pf2);
        if (left > 2) {
            row_pf = row_finish(pf, req_pf);
            request(row_pf, pf.kh);
        }
        if (left > 3) row_start(pf2, req_pf);

        // token gid: heads 2t, 2t + 1 in c[0], c[1]; token gid + 8 in c[2], c[3]
        // (the softmax statistics come from the normaliser kernel, one pass
        // over the logits)
        const bool ok0 = (mask >> gid) & 1u, ok1 = (mask >> (gid + 8)) & 1u;
        float v[4] = {ok0 ? c[0] : -INFINITY, ok0 ? c[1] : -INFINITY, ok1 ? c[2] : -INFINITY,
                      ok1 ? c[3] : -INFINITY};
        const int m0 = 16 * j;
        const bool full = m0 + 16 <= M;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            if (2 * t + hh >= g) continue;
            float* lg = lg_base[hh] + m0;
            if (full) {
                lg[gid] = v[hh];
                lg[gid + 8] = v[2 + hh];
            } else {
                if (m0 + gid < M) lg[gid] = v[hh];
                if (m0 + gid + 8 < M) lg[gid + 8] = v[2 + hh];
            }
        }
        cur = nxt;
        nxt = pf;
        row_nxt = row_pf;
        pf = pf2;
    }
    if (err) atomicOr(a.status, err);
}

// Softmax normaliser of each (sequence, query head) from the tiles' statistics.
__global__ void __launch_bounds__(256) ads_norm_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    pdl_wait();
    __shared__ float s_m[8], s_z[8];
    const int hq = blockIdx.x, b = blockIdx.y;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const float* ts = a.tile_stats + (int64_t(b) * a.n_q_heads + hq) * a.n_tiles * 2;
    float mx = -INFINITY;
    for (int i = threadIdx.x; i < a.n_tiles; i += blockDim.x) mx = fmaxf(mx, ts[2 * i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if (lane == 0) s_m[warp] = mx;
    __syncthreads();
    mx = s_m[0];
    for (int w = 1; w < nw; ++w) mx = fmaxf(mx, s_m[w]);
    float z = 0.0f;
    for (int i = threadIdx.x; i < a.n_tiles; i += blockDim.x) z += ts[2 * i + 1] * expf(ts[2 * i] - mx);
#pragma unroll
    for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) s_z[warp] = z;
    __syncthreads();
    if (threadIdx.x == 0) {
        float zt = 0.0f;
        for (int w = 0; w < nw; ++w) zt += s_z[w];
        float* nrm = a.norm + (int64_t(b) * a.n_q_heads + hq) * 2;
        // no finite logit (no readable token, or a query position out of
        // range): every weight of this head is taken as 0
        nrm[0] = mx == -INFINITY ? 0.0f : mx;
        nrm[1] = mx == -INFINITY ? 0.0f : 1.0f / (zt * float(a.n_q_heads));
    }
}

// Softmax normaliser of each (sequence, query head) straight from its logits
// (the tensor-core and cached-key logits kernels write no tile statistics):
// every thread keeps a running (max, sum of exp) over sixteen logits at a
// time, all of a round's loads requested at once (16-byte loads when the row
// is 16-byte aligned), and the block merges them.
__device__ __forceinline__ void merge_max_sum(float& m, float& s, float m2, float s2) {
    const float mn = fmaxf(m, m2);
    if (mn == -INFINITY) return;
    s = (m == -INFINITY ? 0.0f : s * __expf(m - mn)) + (m2 == -INFINITY ? 0.0f : s2 * __expf(m2 - mn));
    m = mn;
}

__global__ void __launch_bounds__(256) ads_norm_logits_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    pdl_wait();
    __shared__ float s_m[8], s_z[8];
    const int hq = blockIdx.x, b = blockIdx.y, M = a.n_tokens, NT = blockDim.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = NT >> 5;
    const float* lg = a.logits + (int64_t(b) * a.n_q_heads + hq) * M;
    float mx = -INFINITY, z = 0.0f;
    // sixteen logits (-inf past the end) into the running (max, sum of exp)
    auto chunk = [&](const float (&x)[16]) {
        float cm = mx;
#pragma unroll
        for (int u = 0; u < 16; ++u) cm = fmaxf(cm, x[u]);
        if (cm == -INFINITY) return;
        float cz = 0.0f;
#pragma unroll
        for (int u = 0; u < 16; ++u) cz += __expf(x[u] - cm);
        z = (mx == -INFINITY ? 0.0f : z * __expf(mx - cm)) + cz;
        mx = cm;
    };
    if ((M & 3) == 0) {
        // 16-byte loads, eight per thread requested at once (the launch sizes
        // the block so that one round covers the row where it can)
        const float4* l4 = reinterpret_cast<const float4*>(lg);
        const int M4 = M >> 2;
        for (int i4 = 0; i4 < M4; i4 += 8 * NT) {
            float x[2][16];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int j = i4 + u * NT + threadIdx.x;
                const float4 v = j < M4 ? l4[j] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
                x[u >> 2][4 * (u & 3)] = v.x; x[u >> 2][4 * (u & 3) + 1] = v.y;
                x[u >> 2][4 * (u & 3) + 2] = v.z; x[u >> 2][4 * (u & 3) + 3] = v.w;
            }
            chunk(x[0]);
            chunk(x[1]);
        }
    } else {
        for (int i = 0; i < M; i += 16 * NT) {
            float x[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const int t = i + u * NT + threadIdx.x;
                x[u] = t < M ? lg[t] : -INFINITY;
            }
            chunk(x);
        }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, mx, o), z2 = __shfl_xor_sync(0xffffffffu, z, o);
        merge_max_sum(mx, z, m2, z2);
    }
    if (lane == 0) {
        s_m[warp] = mx;
        s_z[warp] = z;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < nw; ++w) merge_max_sum(mx, z, s_m[w], s_z[w]);
        float* nrm = a.norm + (int64_t(b) * a.n_q_heads + hq) * 2;
        nrm[0] = mx == -INFINITY ? 0.0f : mx;
        nrm[1] = mx == -INFINITY ? 0.0f : 1.0f / (z * float(a.n_q_heads));
    }
}

// Relevance of every token: mean over the query heads of its softmax weight,
// the heads accumulated in ascending order (exp of arguments <= 0 by
// __expf, relative error ~1e-6, far inside the relevance's float32 budget). TPT consecutive tokens per thread:
// four (16-byte loads, eight heads' logits requested together) for large
// batches, one (sixteen heads requested together) where the grid would
// otherwise be a few CTAs.
template <int TPT>
__global__ void __launch_bounds__(256) ads_relevance_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    pdl_wait();
    __shared__ float s_n[2 * kSelectMaxQHeads];
    const int b = blockIdx.y;
    const int Hq = a.n_q_heads, M = a.n_tokens;
    for (int i = threadIdx.x; i < 2 * Hq; i += blockDim.x) s_n[i] = a.norm[int64_t(b) * Hq * 2 + i];
    __syncthreads();
    const int m = TPT * (blockIdx.x * blockDim.x + threadIdx.x);
    if (m >= M) return;
    const float* lg = a.logits + int64_t(b) * Hq * M + m;
    float r[TPT];
#pragma unroll
    for (int u = 0; u < TPT; ++u) r[u] = 0.0f;
    if (TPT == 1) {
        int h = 0;
        for (; h + 16 <= Hq; h += 16) {
            float x[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) x[u] = lg[int64_t(h + u) * M];
#pragma unroll
            for (int u = 0; u < 16; ++u) r[0] = fmaf(__expf(x[u] - s_n[2 * (h + u)]), s_n[2 * (h + u) + 1], r[0]);
        }
        for (; h < Hq; ++h) r[0] = fmaf(__expf(lg[int64_t(h) * M] - s_n[2 * h]), s_n[2 * h + 1], r[0]);
    } else if ((M & 3) == 0) {
        int h = 0;
        for (; h + 16 <= Hq; h += 16) {  // sixteen heads' logits requested together
            float4 x[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) x[u] = *reinterpret_cast<const float4*>(lg + int64_t(h + u) * M);
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const float mh = s_n[2 * (h + u)], wh = s_n[2 * (h + u) + 1];
                r[0] = fmaf(__expf(x[u].x - mh), wh, r[0]);
                r[1 % TPT] = fmaf(__expf(x[u].y - mh), wh, r[1 % TPT]);
                r[2 % TPT] = fmaf(__expf(x[u].z - mh), wh, r[2 % TPT]);
                r[3 % TPT] = fmaf(__expf(x[u].w - mh), wh, r[3 % TPT]);
            }
        }
        for (; h < Hq; ++h) {
            const float4 x = *reinterpret_cast<const float4*>(lg + int64_t(h) * M);
            const float mh = s_n[2 * h], wh = s_n[2 * h + 1];
            r[0] = fmaf(__expf(x.x - mh), wh, r[0]);
            r[1 % TPT] = fmaf(__expf(x.y - mh), wh, r[1 % TPT]);
            r[2 % TPT] = fmaf(__expf(x.z - mh), wh, r[2 % TPT]);
            r[3 % TPT] = fmaf(__expf(x.w - mh), wh, r[3 % TPT]);
        }
    } else {
        const int n = min(TPT, M - m);
        for (int h = 0; h < Hq; ++h) {
            const float mh = s_n[2 * h], wh = s_n[2 * h + 1];
#pragma unroll
            for (int u = 0; u < TPT; ++u)
                if (u < n) r[u] = fmaf(__expf(lg[int64_t(h) * M + u] - mh), wh, r[u]);
        }
    }
    const int n = min(TPT, M - m);
#pragma unroll
    for (int u = 0; u < TPT; ++u) {
        if (u < n) {
            a.rel[int64_t(b) * M + m + u] = r[u];
            if (a.score_out) a.score_out[int64_t(b) * M + m + u] = r[u];
        }
    }
}

// Block-wide exclusive scan of one int per thread; returns the total.
__device__ __forceinline__ int block_scan(int v, int* s_warp, int* out_excl) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < nw ? s_warp[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < nw) s_warp[lane] = w;  // inclusive prefix of warp totals
    }
    __syncthreads();
    const int total = s_warp[nw - 1];
    *out_excl = x - v + (warp > 0 ? s_warp[warp - 1] : 0);
    __syncthreads();
    return total;
}

// PER: relevances per thread (a thread keeps its PER consecutive tokens in
// registers; blockDim.x * PER >= n_tokens, blockDim.x a multiple of 32).
template <int PER>
__global__ void __launch_bounds__(1024) ads_select_kernel(const __grid_constant__ SelectArgs a) {
    pdl_allow();
    pdl_wait();
    __shared__ int s_warp[32];
    __shared__ unsigned int s_cnt[3 * 32];
    const int b = blockIdx.x;
    const int M = a.n_tokens;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int beg = threadIdx.x * PER;
    const int nwarp = blockDim.x >> 5;  // a multiple of 32 threads, <= 1024

    // this thread's relevances (from the relevance kernel); tokens past the
    // end read as 0 and are excluded wherever 0 could count
    unsigned int key[PER];
    const float* rs = a.rel + int64_t(b) * M;
#pragma unroll
    for (int i = 0; i < PER; ++i) key[i] = beg + i < M ? __float_as_uint(rs[beg + i]) : 0u;

    // 1. the K-th largest relevance, two bits per round from the top: of the
    // candidates X | d << bit (d = 1, 2, 3) keep the largest that at least K
    // keys reach (relevance >= 0, so float bits order as values; every
    // candidate is >= 1, so the padding never counts). Counting against
    // thresholds needs no histogram, hence no atomics on the few bins that
    // relevances sharing their high bits would all fall into.
    // The search also stops as soon as exactly K keys reach X: the selection
    // is then every key >= X (the compaction below takes all keys above X
    // and, of those equal to X, exactly the K - above that remain).
    const unsigned int K = unsigned(a.k);
    unsigned int X = 0u, cX = 0u;  // cX: keys >= X, once X > 0
    for (int bit = 30; bit >= 0; bit -= 2) {
        const unsigned int x1 = X | (1u << bit), x2 = X | (2u << bit), x3 = X | (3u << bit);
        unsigned int c1 = 0u, c2 = 0u, c3 = 0u;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            c1 += key[i] >= x1;
            c2 += key[i] >= x2;
            c3 += key[i] >= x3;
        }
        c1 = __reduce_add_sync(0xffffffffu, c1);
        c2 = __reduce_add_sync(0xffffffffu, c2);
        c3 = __reduce_add_sync(0xffffffffu, c3);
        if (lane == 0) {
            s_cnt[warp] = c1;
            s_cnt[32 + warp] = c2;
            s_cnt[64 + warp] = c3;
        }
        __syncthreads();
        const bool wl = lane < nwarp;  // this lane reads warp `lane`'s counts
        const unsigned int t1 = __reduce_add_sync(0xffffffffu, wl ? s_cnt[lane] : 0u);
        const unsigned int t2 = __reduce_add_sync(0xffffffffu, wl ? s_cnt[32 + lane] : 0u);
        const unsigned int t3 = __reduce_add_sync(0xffffffffu, wl ? s_cnt[64 + lane] : 0u);
        cX = t3 >= K ? t3 : (t2 >= K ? t2 : (t1 >= K ? t1 : cX));
        X = t3 >= K ? x3 : (t2 >= K ? x2 : (t1 >= K ? x1 : X));
        __syncthreads();
        if (X != 0u && cX == K) break;  // uniform: every thread read the same counts
    }
    // keys strictly above X: all taken; of the keys equal to X, the first ones
    unsigned int above = 0u, n_eq = 0u;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        above += key[i] > X;
        n_eq += beg + i < M && key[i] == X;
    }
    above = __reduce_add_sync(0xffffffffu, above);
    if (lane == 0) s_cnt[warp] = above;
    __syncthreads();
    const int need_eq = int(K - __reduce_add_sync(0xffffffffu, lane < nwarp ? s_cnt[lane] : 0u));

    // 2. ordered compaction: all keys > X, then the first need_eq keys == X
    int eq_before = 0;
    block_scan(int(n_eq), s_warp, &eq_before);
    int n_sel = 0;
    {
        int e = eq_before;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const bool eq = beg + i < M && key[i] == X;
            n_sel += key[i] > X || (eq && e < need_eq);
            e += eq;
        }
    }
    int sel_before = 0;
    block_scan(n_sel, s_warp, &sel_before);
    int32_t* out = a.idx_out + int64_t(b) * a.k;
    {
        int e = eq_before, o = sel_before;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const bool eq = beg + i < M && key[i] == X;
            if (key[i] > X || (eq && e < need_eq)) out[o++] = beg + i;
            e += eq;
        }
    }
    if (threadIdx.x == 0) {
        a.rev_tok_off[b] = b * a.k;
        a.seq_rev_off[b] = b;
        if (b == gridDim.x - 1) {
            a.rev_tok_off[b + 1] = (b + 1) * a.k;
            a.seq_rev_off[b + 1] = b + 1;
        }
    }
}

}  // namespace

size_t select_logits_smem(const SelectArgs& a) {
    const int D = a.head_dim, P = D / 2, T = a.tok_tile;
    return size_t(a.n_q_heads) * (D / 4 + 1) * 16 + 2 * size_t(T) * (P / 4 + 1) * 16 +
           size_t(a.n_q_heads) * (T + 1) * 4 + size_t(T) * 3 * 4;
}

template <int L, int G>
cudaError_t launch_logits_g(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream) {
    const size_t smem = select_logits_smem(a);
    cudaError_t e = cudaFuncSetAttribute(ads_logits_kernel<L, G>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ads_logits_kernel<L, G>, 256, smem);
    if (e != cudaSuccess) return e;
    const int64_t tiles = int64_t(n_seqs) * a.n_tiles;
    const int64_t resident = int64_t(sms) * (per_sm > 0 ? per_sm : 1);
    const unsigned grid = unsigned(tiles < resident ? tiles : resident);
    return launch_pdl(ads_logits_kernel<L, G>, dim3(grid), dim3(256), smem, stream, a);
}

template <int L>
cudaError_t launch_logits(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream) {
    const int g = a.n_q_heads / a.n_kv_heads;
    if (g == 1) return launch_logits_g<L, 1>(a, n_seqs, sms, stream);
    if (g == 2) return launch_logits_g<L, 2>(a, n_seqs, sms, stream);
    if (g == 4) return launch_logits_g<L, 4>(a, n_seqs, sms, stream);
    return launch_logits_g<L, 8>(a, n_seqs, sms, stream);
}

constexpr int kMmaWarps = 8;  // warps per CTA of the tensor-core logits kernel (16 tokens each)

template <int D>
size_t logits_mma_smem(int kpi) {
    return size_t(kpi) * (D / 16) * 32 * 16 + size_t(kMmaWarps) * (D / 8) * 32 * 16 +
           size_t(D / 2) * 16;
}

template <int D>
cudaError_t launch_logits_mma(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream) {
    auto kern = ads_logits_mma_kernel<D, kMmaWarps>;
    const int H = a.n_kv_heads;
    SelectArgs b = a;
    b.kh_per_item = H < 8 ? H : 8;  // KV heads per work item (sizes the query fragments)
    const size_t smem_max = logits_mma_smem<D>(b.kh_per_item);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem_max));
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMmaWarps * 32, smem_max);
    if (e != cudaSuccess) return e;
    const int64_t resident = int64_t(sms) * (per_sm > 0 ? per_sm : 1);
    // Few tokens (a small batch): fewer KV heads per item until there are two
    // items per resident CTA, so that short chains run side by side.
    const int64_t n_it = (a.n_tokens + 16 * kMmaWarps - 1) / (16 * kMmaWarps);
    auto items = [&](int kpi) { return int64_t(n_seqs) * n_it * ((H + kpi - 1) / kpi); };
    while (b.kh_per_item > 1 && items(b.kh_per_item) < 2 * resident)
        b.kh_per_item = (b.kh_per_item + 1) / 2;
    const int64_t n = items(b.kh_per_item);
    const unsigned grid = unsigned(n < resident ? n : resident);
    return launch_pdl(kern, dim3(grid), dim3(kMmaWarps * 32), logits_mma_smem<D>(b.kh_per_item),
                      stream, b);
}

// The normalisers, relevances and selection after a logits kernel.
static cudaError_t launch_select_tail(const SelectArgs& a, int n_seqs, cudaStream_t stream,
                                      bool norm_from_logits = false) {
    // the normaliser from the logits: about 32 logits per thread, one round
    // up to 256 threads (wider blocks would take large grids past one wave)
    int nt = int(((a.n_tokens + 31) / 32 + 31) / 32 * 32);
    nt = nt < 64 ? 64 : (nt > 256 ? 256 : nt);
    cudaError_t e = norm_from_logits
                        ? launch_pdl(ads_norm_logits_kernel, dim3(a.n_q_heads, n_seqs, 1), dim3(nt), 0,
                                     stream, a)
                        : launch_pdl(ads_norm_kernel, dim3(a.n_q_heads, n_seqs, 1), dim3(256), 0, stream, a);
    if (e != cudaSuccess) return e;
    // four tokens per thread once the grid fills the GPU a few times over
    if (int64_t(n_seqs) * a.n_tokens >= (int64_t(1) << 19))
        e = launch_pdl(ads_relevance_kernel<4>, dim3((a.n_tokens + 1023) / 1024, n_seqs, 1), dim3(256),
                       0, stream, a);
    else
        e = launch_pdl(ads_relevance_kernel<1>, dim3((a.n_tokens + 255) / 256, n_seqs, 1), dim3(256), 0,
                       stream, a);
    if (e != cudaSuccess) return e;
    const int M = a.n_tokens;
    // just enough warps for PER tokens per thread: fewer warps, cheaper rounds
    auto threads = [M](int per) { return int(((M + per - 1) / per + 31) / 32 * 32); };
    const dim3 grid(unsigned(n_seqs), 1, 1);
    if (M <= 4096) return launch_pdl(ads_select_kernel<4>, grid, dim3(threads(4)), 0, stream, a);
    if (M <= 8192) return launch_pdl(ads_select_kernel<8>, grid, dim3(threads(8)), 0, stream, a);
    if (M <= 16384) return launch_pdl(ads_select_kernel<16>, grid, dim3(threads(16)), 0, stream, a);
    return launch_pdl(ads_select_kernel<32>, grid, dim3(threads(32)), 0, stream, a);
}

cudaError_t launch_select(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream) {
    cudaError_t e;
    const bool mma = (a.head_dim == 128 || a.head_dim == 64) && a.tok_tile == 16;
    if (a.head_dim == 128 && mma) {
        e = launch_logits_mma<128>(a, n_seqs, sms, stream);
    } else if (a.head_dim == 64 && mma) {
        e = launch_logits_mma<64>(a, n_seqs, sms, stream);
    } else {
        const int L = a.head_dim <= 64 ? 4 : (a.head_dim <= 128 ? 8 : 16);
        e = L == 4 ? launch_logits<4>(a, n_seqs, sms, stream)
                   : (L == 8 ? launch_logits<8>(a, n_seqs, sms, stream)
                             : launch_logits<16>(a, n_seqs, sms, stream));
    }
    if (e != cudaSuccess) return e;
    return launch_select_tail(a, n_seqs, stream, mma);
}

cudaError_t launch_select_cached(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream) {
    const int g = a.n_q_heads / a.n_kv_heads;
    const size_t smem = size_t(8) * g * a.head_dim * sizeof(float);  // 8 warps
    auto k = a.head_dim == 64 ? ads_logits_cache_kernel<64>
             : a.head_dim == 128 ? ads_logits_cache_kernel<128>
                                 : ads_logits_cache_kernel<256>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    int per_sm = 0;
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, 256, smem);
    if (e != cudaSuccess) return e;
    const int64_t items = int64_t(n_seqs) * a.n_kv_heads * a.n_tiles;
    const int64_t ctas = (items + 7) / 8;
    const int64_t resident = int64_t(sms) * (per_sm > 0 ? per_sm : 1);
    e = launch_pdl(k, dim3(unsigned(ctas < resident ? ctas : resident)), dim3(256), smem, stream, a);
    if (e != cudaSuccess) return e;
    return launch_select_tail(a, n_seqs, stream, true);
}

}  // namespace prcr
