// Internal interfaces between the C-ABI layer (prcr_abi.cu) and the kernels.
#pragma once

#include <cstddef>
#include <cmath>
#include <cstdint>

#include <cuda_runtime.h>

#include "prcr.h"

namespace prcr {

constexpr int kPlanThreads = 512;
constexpr int kMaxPairs = PRCR_MAX_HEAD_DIM / 2;
constexpr int kRebindTargetThreads = 256;

// Per-token plan left in the workspace by the plan kernel for the rebind
// kernel (structure of arrays, each array 256-byte aligned).
struct PlanView {
    int64_t* src;  // element offset of the token's store row, layer term excluded
    int64_t* dst;  // element offset of the token's cache row, layer term excluded; -1 = skip
    double*  pos;  // reassigned (t, h, w)
};

inline size_t align256(size_t n) { return (n + 255) & ~size_t(255); }

// Rotation rates of the pairs as fractions of a turn per unit of position,
// in unsigned 0.64 fixed point: round(theta^(-2i/D) / (2 pi) * 2^64) (< 2^63).
inline void fill_turn_freq(const prcr_rope_cfg* cfg, uint64_t* out) {
    const long double two_pi = 6.283185307179586476925286766559005768L;
    const long double two64 = 18446744073709551616.0L;
    const int P = cfg->head_dim / 2;
    for (int i = 0; i < P; ++i) {
        const long double w = powl(static_cast<long double>(cfg->theta),
                                   -2.0L * static_cast<long double>(i) / cfg->head_dim);
        out[i] = static_cast<uint64_t>(llroundl(w / two_pi * two64));
    }
}

#ifdef __CUDACC__
// sin and cos of pos * inv_freq_i. The angle modulo one turn is formed
// exactly in integers: pos in 32.32 fixed point times the 0.64 turn rate is
// the number of turns with 96 fractional bits; the top 32 of those (the low
// half of the 128-bit product's high word, read as signed) are the angle in
// [-pi, pi) to 2^-32 of a turn. Needs |pos| < 2^31. Only the final sin/cos
// runs in float32 (CUDA's sincosf).
// The position in signed 32.32 fixed point, rounded to nearest (ties to
// even), formed from the float64 bits with integer instructions only (GB300's
// float64 pipe is narrow): equal to llrint(pos * 2^32) for |pos| < 2^31, and
// to -2^63 for pos = -2^31 (+2^31 saturates to 2^63 - 1). A larger magnitude,
// infinity or NaN gives 0: such positions are reported and their rows
// skipped wherever they can arise.
__device__ __forceinline__ long long fixed_32_32(double pos) {
    const unsigned long long bits = static_cast<unsigned long long>(__double_as_longlong(pos));
    const int e = int((bits >> 52) & 0x7ff);  // pos * 2^32 = m * 2^(e - 1043)
    if (e == 0 || e > 1054) return 0;         // zero or subnormal (|pos| < 2^-1022), or |pos| > 2^31
    const unsigned long long m = (bits & 0xfffffffffffffull) | (1ull << 52);
    const int sh = e - 1043;
    unsigned long long r;
    if (sh >= 0) {
        r = m << sh;  // < 2^64 (sh <= 11)
    } else if (-sh > 54) {
        r = 0;  // below half a unit
    } else {
        const int s = -sh;
        r = m >> s;
        const unsigned long long rem = m & ((1ull << s) - 1), half = 1ull << (s - 1);
        if (rem > half || (rem == half && (r & 1))) ++r;
    }
    if (bits >> 63) return static_cast<long long>(0ull - r);
    return r > 0x7fffffffffffffffull ? 0x7fffffffffffffffll : static_cast<long long>(r);
}

// Exact float64 of an integer of magnitude below 2^53, from integer
// instructions only.
__device__ __forceinline__ double exact_f64(long long x) {
    if (x == 0) return 0.0;
    const unsigned long long u = x < 0 ? 0ull - static_cast<unsigned long long>(x)
                                       : static_cast<unsigned long long>(x);
    const int sh = __clzll(static_cast<long long>(u)) - 11;  // leading one to bit 52
    const unsigned long long m = u << sh;
    const unsigned long long bits = (static_cast<unsigned long long>(x < 0) << 63) |
                                    (static_cast<unsigned long long>(1075 - sh) << 52) |
                                    (m & 0xfffffffffffffull);
    return __longlong_as_double(static_cast<long long>(bits));
}

// sin and cos from a 32.32 fixed-point position (integer arithmetic up to
// the final float32 sincosf).
__device__ __forceinline__ void sincos_fixed(long long pf, uint64_t turn_freq, float* s, float* c) {
    const long long hi = __mul64hi(pf, static_cast<long long>(turn_freq));
    const int frac = static_cast<int>(static_cast<unsigned int>(static_cast<unsigned long long>(hi)));
    sincosf(static_cast<float>(frac) * 1.46291807926715968e-09f, s, c);  // 2 pi / 2^32
}

__device__ __forceinline__ void sincos_turns(double pos, uint64_t turn_freq, float* s, float* c) {
    sincos_fixed(fixed_32_32(pos), turn_freq, s, c);
}
#endif

inline size_t workspace_bytes(int64_t total_k) {
    if (total_k <= 0) return 0;
    const size_t n = size_t(total_k);
    return 2 * align256(8 * n) + align256(24 * n);
}

inline PlanView plan_view(void* ws, int64_t total_k) {
    char* p = static_cast<char*>(ws);
    const size_t n = size_t(total_k > 0 ? total_k : 0);
    PlanView v;
    v.src = reinterpret_cast<int64_t*>(p);
    v.dst = reinterpret_cast<int64_t*>(p + align256(8 * n));
    v.pos = reinterpret_cast<double*>(p + 2 * align256(8 * n));
    return v;
}

struct PlanArgs {
    // store
    const int32_t* coords;
    int64_t coord_seq_stride;
    int64_t store_seq_stride;
    int64_t store_token_stride;
    int32_t n_tokens;
    // cache
    int32_t cache_kind;
    int32_t block_size;
    int32_t bt_stride;
    int32_t n_blocks;
    int32_t max_slots;
    int64_t cache_seq_stride;
    int64_t block_stride;
    int64_t slot_stride;
    const int32_t* block_table;
    // batch
    const int32_t* seq_rev_off;
    const int32_t* rev_tok_off;
    const int32_t* idx;
    const int64_t* p_txt;
    const int32_t* cache_len_in;
    int32_t n_seqs;
    int32_t n_revisits;
    int64_t total_k;
    // outputs
    int32_t* cache_len_out;
    int64_t* next_pos_out;
    double* pos_out;
    int32_t* slot_out;
    uint32_t* status;
    PlanView plan;
    int32_t mode;
    int32_t L;
    int32_t flags;
};

struct RebindArgs {
    const uint16_t* store_k;
    const uint16_t* store_v;
    uint16_t* cache_k;
    uint16_t* cache_v;
    int64_t store_layer_stride;
    int64_t cache_layer_stride;
    const int64_t* plan_src;
    const int64_t* plan_dst;
    const double* plan_pos;
    const uint32_t* status;
    int64_t total_k;
    int32_t n_layers;
    int32_t head_dim;
    int32_t lanes;           // threads per token: n_kv_heads * head_dim / 16
    int32_t tok_per_cta;     // T
    int32_t layers_per_cta;  // G
    int32_t layout;
    int32_t sec_t;
    int32_t sec_h;
    int32_t sec_w;
    uint64_t turn_freq[kMaxPairs];  // pair i: round(inv_freq_i / (2 pi) * 2^64)
};

struct StoreArgs {
    uint16_t* dst_k;        // store row of (seq, layer_begin, m_begin)
    uint16_t* dst_v;
    const uint16_t* src_k;
    const uint16_t* src_v;
    int64_t dst_layer_stride;
    int64_t dst_token_stride;
    int64_t src_layer_stride;
    int64_t src_token_stride;
    int32_t n_layers;
    int32_t m_count;
    int32_t row_vecs;       // 16-byte vectors per row: H * D / 8
    int32_t* dst_coords;    // store coordinates of (seq, m_begin), or null
    const int32_t* src_coords;
};

struct CaptureArgs {
    const uint16_t* src_k;      // token 0 of layer 0 of the prefill rows
    const uint16_t* src_v;
    int64_t src_layer_stride;
    int64_t src_token_stride;
    uint16_t* store_k;          // store row of (seq, layer_begin, m_begin)
    uint16_t* store_v;
    int64_t store_layer_stride;
    int64_t store_token_stride;
    int32_t* store_coords;      // store coordinates of (seq, m_begin)
    const int32_t* coords;      // [m_count][3] original (t, h, w)
    uint16_t* cache_k;          // cache base shifted to layer_begin
    uint16_t* cache_v;
    int64_t cache_layer_stride;
    int64_t cache_seq_off;      // contiguous: seq * seq_stride
    int64_t block_stride;
    int64_t slot_stride;
    int64_t capacity;           // slots of this sequence
    int64_t slot_begin;
    const int32_t* bt_row;      // paged: block-table row of the sequence
    int32_t cache_kind;
    int32_t block_size;
    int32_t n_blocks;
    uint32_t* status;
    int32_t m_count;
    int32_t n_layers;
    int32_t head_dim;
    int32_t lanes;
    int32_t tok_per_cta;
    int32_t layers_per_cta;
    int32_t layout;
    int32_t sec_t;
    int32_t sec_h;
    int32_t sec_w;
    uint64_t turn_freq[kMaxPairs];  // pair i: round(inv_freq_i / (2 pi) * 2^64)
};

struct DecodeArgs {
    const uint16_t* q;          // [B][n_layers][n_q_heads][D] raw queries
    const int64_t* q_pos;       // [B]
    const int32_t* seq_len;     // [B]
    const uint16_t* cache_k;
    const uint16_t* cache_v;
    int64_t layer_stride;
    int64_t seq_stride;         // contiguous
    int64_t block_stride;       // paged
    int64_t slot_stride;
    int64_t capacity;           // slots per sequence
    const int32_t* block_table;
    int32_t bt_stride;
    int32_t block_size;
    int32_t n_blocks;
    int32_t cache_kind;
    float* out;                 // [B][n_layers][n_q_heads][D]
    float* partial;             // [B][n_layers][n_q_heads][splits][D + 2] when splits > 1
    uint32_t* status;
    int32_t n_layers;
    int32_t n_kv_heads;
    int32_t n_q_heads;
    int32_t head_dim;
    int32_t group;
    int32_t splits;
    int32_t chunk;
    int32_t ring;               // small batch: the ring-staged kernel (head_dim 64, 128)
    float scale;
    uint64_t turn_freq[kMaxPairs];  // pair i: round(inv_freq_i / (2 pi) * 2^64)
};

constexpr int kDecodeMaxChunk = 4096;
constexpr int kDecodeRingWarps = 4;   // KV heads (one per warp) per CTA of the ring kernel
constexpr int kDecodeRingCtasPerSm = 3;

constexpr int kSelectMaxQHeads = 128;
constexpr int kSelectTokTile = 16;   // smallest tile of the logits kernel (sizes the workspace)

inline size_t select_workspace_bytes(int64_t B, int64_t Hq, int64_t M) {
    const int64_t tiles = (M + kSelectTokTile - 1) / kSelectTokTile;
    return align256(size_t(4 * B * Hq * M)) + align256(size_t(8 * B * Hq * tiles)) +
           align256(size_t(8 * B * Hq)) + align256(size_t(4 * B * M));
}

struct SelectArgs {
    const uint16_t* q;          // [B][n_q_heads][D] raw trigger queries
    const int64_t* q_pos;       // [B]
    const uint16_t* store_k;
    int64_t store_seq_stride;
    int64_t store_layer_stride;
    int64_t store_token_stride;
    const int32_t* coords;
    int64_t coord_seq_stride;
    int32_t layer;
    int32_t n_tokens;
    int32_t n_kv_heads;
    int32_t n_q_heads;
    int32_t head_dim;
    int32_t k;
    int32_t layout;
    int32_t sec_t;
    int32_t sec_h;
    int32_t sec_w;
    float scale;
    float* logits;              // workspace [B][n_q_heads][n_tokens]
    float* tile_stats;          // workspace [B][n_q_heads][n_tiles][2] (max, sum of exp)
    float* norm;                // workspace [B][n_q_heads][2] (max, 1 / (sum * n_q_heads))
    float* rel;                 // workspace [B][n_tokens] relevance
    int32_t n_seqs;
    int32_t n_tiles;            // token tiles of the logits kernel per sequence
    int32_t tok_tile;           // tokens per tile
    int32_t kh_per_item;        // tensor-core logits: KV heads per work item
    float* score_out;           // optional [B][n_tokens]
    int32_t* idx_out;           // [B][k]
    int32_t* rev_tok_off;       // [B + 1]
    int32_t* seq_rev_off;       // [B + 1]
    // keys from the position-bound cache (prcr_select_topk_cached)
    const uint16_t* cache_k;
    int64_t cache_seq_stride;   // contiguous
    int64_t cache_layer_stride;
    int64_t cache_block_stride; // paged
    int64_t cache_slot_stride;
    int64_t cache_capacity;     // slots per sequence
    const int32_t* block_table;
    int32_t bt_stride;
    int32_t block_size;
    int32_t n_blocks;
    int32_t cache_kind;
    const int32_t* img_slot0;   // [B] first slot of each sequence's image tokens
    uint32_t* status;
    uint64_t turn_freq[kMaxPairs];  // pair i: round(inv_freq_i / (2 pi) * 2^64)
};

// Every argument check of prcr_rebind_inject except the workspace's: PRCR_OK
// or the negative code that call would return.
int check_revisit_args(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                       const prcr_cache_desc* cache, const prcr_revisit_batch* b,
                       const prcr_outputs* o, int32_t mode, int32_t L, int32_t flags);

cudaError_t launch_select(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream);
// the logits of the cached-key selection, then the same normaliser, relevance
// and selection kernels
cudaError_t launch_select_cached(const SelectArgs& a, int n_seqs, int sms, cudaStream_t stream);

cudaError_t launch_decode(const DecodeArgs& a, int gp, dim3 grid, size_t smem,
                          cudaStream_t stream);
cudaError_t launch_capture(const CaptureArgs& a, dim3 grid, int block, size_t smem,
                           cudaStream_t stream);
cudaError_t capture_blocks_per_sm(int block, size_t smem, int* out);
// Small batches: the whole revisit in one kernel (plan part + rebind part;
// the rebind part's plan pointers are unused).
struct FusedArgs {
    PlanArgs plan;
    RebindArgs rebind;
};
constexpr int64_t kFusedMaxTokens = 2048;
constexpr int kFusedMaxRevisits = 64;
constexpr int kFusedMaxSeqs = 64;

cudaError_t launch_fused(const FusedArgs& a, dim3 grid, int block, size_t smem,
                         cudaStream_t stream);
cudaError_t fused_blocks_per_sm(int block, size_t smem, int* out);
// dynamic shared memory the fused kernel adds to the cos/sin rows: the rows of
// two layers staged per thread
size_t fused_stage_bytes(int block);
cudaError_t launch_plan(const PlanArgs& a, cudaStream_t stream);
cudaError_t launch_rebind(const RebindArgs& a, dim3 grid, int block, size_t smem,
                          cudaStream_t stream);
cudaError_t rebind_blocks_per_sm(int block, size_t smem, int* out);
cudaError_t launch_store(const StoreArgs& a, cudaStream_t stream);

}  // namespace prcr
