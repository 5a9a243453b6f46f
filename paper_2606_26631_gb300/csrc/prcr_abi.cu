// extern "C" entry points of libprcr.so: argument checks, launch planning
// and the two-kernel revisit path (plan, then rebind + inject).
#include <array>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

#include "prcr_internal.h"

namespace prcr {
namespace {

// Turn rates of a (theta, head_dim) pair, computed once (long double pow is
// slow where long double is a software type) and kept for the process.
void copy_turn_freq(const prcr_rope_cfg* cfg, uint64_t* out) {
    static std::mutex mu;
    static std::map<std::pair<uint64_t, int>, std::array<uint64_t, kMaxPairs>> cache;
    uint64_t tbits;
    std::memcpy(&tbits, &cfg->theta, sizeof(tbits));
    const auto key = std::make_pair(tbits, int(cfg->head_dim));
    std::lock_guard<std::mutex> g(mu);
    auto it = cache.find(key);
    if (it == cache.end()) {
        std::array<uint64_t, kMaxPairs> t{};
        fill_turn_freq(cfg, t.data());
        it = cache.emplace(key, t).first;
    }
    std::memcpy(out, it->second.data(), sizeof(uint64_t) * size_t(cfg->head_dim / 2));
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }
inline bool aligned8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }
inline bool mult8(int64_t s) { return s >= 0 && (s & 7) == 0; }

int check_cfg(const prcr_rope_cfg* c) {
    if (!c) return PRCR_EINVAL;
    const int D = c->head_dim;
    if (c->n_layers < 1 || c->n_kv_heads < 1 || D < 16 || D > PRCR_MAX_HEAD_DIM || (D & 15))
        return PRCR_EINVAL;
    if (int64_t(c->n_kv_heads) * D > PRCR_MAX_ROW_ELEMS) return PRCR_EINVAL;
    if (c->sections[0] < 0 || c->sections[1] < 0 || c->sections[2] < 0 ||
        c->sections[0] + c->sections[1] + c->sections[2] != D / 2)
        return PRCR_EINVAL;
    if (c->layout != PRCR_LAYOUT_SECTIONED && c->layout != PRCR_LAYOUT_INTERLEAVED)
        return PRCR_EINVAL;
    if (c->reserved != 0) return PRCR_EINVAL;
    if (!(c->theta > 1.0) || !std::isfinite(c->theta)) return PRCR_EINVAL;
    return PRCR_OK;
}

int check_store(const prcr_rope_cfg* c, const prcr_store_desc* s) {
    if (!s || !s->k || !s->v || !s->coords) return PRCR_EINVAL;
    const int64_t row = int64_t(c->n_kv_heads) * c->head_dim;
    if (s->n_seqs < 1 || s->n_tokens < 1) return PRCR_EINVAL;
    if (s->token_stride < row || s->layer_stride < 0 || s->seq_stride < 0) return PRCR_EINVAL;
    if (s->coord_seq_stride < 3 * int64_t(s->n_tokens) && s->n_seqs > 1) return PRCR_EINVAL;
    if (!aligned16(s->k) || !aligned16(s->v) || !aligned4(s->coords)) return PRCR_EALIGN;
    if (!mult8(s->seq_stride) || !mult8(s->layer_stride) || !mult8(s->token_stride))
        return PRCR_EALIGN;
    return PRCR_OK;
}

int check_cache(const prcr_rope_cfg* c, const prcr_cache_desc* k) {
    if (!k || !k->k || !k->v) return PRCR_EINVAL;
    const int64_t row = int64_t(c->n_kv_heads) * c->head_dim;
    if (k->slot_stride < row || k->layer_stride < 0 || k->n_seqs < 1) return PRCR_EINVAL;
    if (!aligned16(k->k) || !aligned16(k->v)) return PRCR_EALIGN;
    if (!mult8(k->layer_stride) || !mult8(k->slot_stride)) return PRCR_EALIGN;
    if (k->kind == PRCR_CACHE_CONTIGUOUS) {
        if (k->max_slots < 0 || k->seq_stride < 0) return PRCR_EINVAL;
        if (!mult8(k->seq_stride)) return PRCR_EALIGN;
    } else if (k->kind == PRCR_CACHE_PAGED) {
        if (!k->block_table || k->block_size < 1 || k->bt_stride < 0 || k->n_blocks < 0 ||
            k->block_stride < 0)
            return PRCR_EINVAL;
        if (!aligned4(k->block_table)) return PRCR_EALIGN;
        if (!mult8(k->block_stride)) return PRCR_EALIGN;
    } else {
        return PRCR_EINVAL;
    }
    return PRCR_OK;
}

}  // namespace

// Every check of a revisit call except the workspace's.
int check_revisit_args(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                       const prcr_cache_desc* cache, const prcr_revisit_batch* b,
                       const prcr_outputs* o, int32_t mode, int32_t L, int32_t flags) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_store(cfg, store))) return rc;
    if ((rc = check_cache(cfg, cache))) return rc;
    if (!b || !o) return PRCR_EINVAL;
    if (mode < PRCR_MODE_PCR || mode > PRCR_MODE_LPA) return PRCR_EINVAL;
    if (L < 0 || (flags & ~PRCR_FLAG_DEGENERATE_CENTER)) return PRCR_EINVAL;
    if (b->n_seqs < 0 || b->n_revisits < 0 || b->total_k < 0 || b->total_k > INT32_MAX)
        return PRCR_EINVAL;
    if (b->n_seqs == 0) return (b->n_revisits == 0 && b->total_k == 0) ? PRCR_OK : PRCR_EINVAL;
    if (b->n_seqs > store->n_seqs || b->n_seqs > cache->n_seqs) return PRCR_EINVAL;
    if (!b->seq_rev_off || !b->rev_tok_off || !b->p_txt || !b->cache_len_in) return PRCR_EINVAL;
    if (b->total_k > 0 && !b->idx) return PRCR_EINVAL;
    if (!o->cache_len_out || !o->next_pos_out || !o->status) return PRCR_EINVAL;
    if (static_cast<const void*>(o->cache_len_out) == static_cast<const void*>(b->cache_len_in))
        return PRCR_EINVAL;
    if (!aligned4(b->seq_rev_off) || !aligned4(b->rev_tok_off) || !aligned4(b->cache_len_in) ||
        !aligned8(b->p_txt) || (b->idx && !aligned4(b->idx)) || !aligned4(o->cache_len_out) ||
        !aligned8(o->next_pos_out) || !aligned4(o->status) ||
        (o->pos_out && !aligned8(o->pos_out)) || (o->slot_out && !aligned4(o->slot_out)))
        return PRCR_EALIGN;
    return PRCR_OK;
}

namespace {

int check_call(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
               const prcr_cache_desc* cache, const prcr_revisit_batch* b,
               const prcr_outputs* o, int32_t mode, int32_t L, int32_t flags, void* ws,
               size_t ws_bytes) {
    const int rc = check_revisit_args(cfg, store, cache, b, o, mode, L, flags);
    if (rc || b->n_seqs == 0) return rc;
    if (b->total_k > 0) {
        if (!ws || ws_bytes < workspace_bytes(b->total_k)) return PRCR_EWORKSPACE;
        if (!aligned16(ws)) return PRCR_EALIGN;
    }
    return PRCR_OK;
}

PlanArgs make_plan_args(const prcr_store_desc* store, const prcr_cache_desc* cache,
                        const prcr_revisit_batch* b, const prcr_outputs* o, int32_t mode,
                        int32_t L, int32_t flags, void* ws) {
    PlanArgs a = {};
    a.coords = store->coords;
    a.coord_seq_stride = store->coord_seq_stride;
    a.store_seq_stride = store->seq_stride;
    a.store_token_stride = store->token_stride;
    a.n_tokens = store->n_tokens;
    a.cache_kind = cache->kind;
    a.block_size = cache->kind == PRCR_CACHE_PAGED ? cache->block_size : 1;
    a.bt_stride = cache->bt_stride;
    a.n_blocks = cache->n_blocks;
    a.max_slots = cache->max_slots;
    a.cache_seq_stride = cache->seq_stride;
    a.block_stride = cache->block_stride;
    a.slot_stride = cache->slot_stride;
    a.block_table = cache->block_table;
    a.seq_rev_off = b->seq_rev_off;
    a.rev_tok_off = b->rev_tok_off;
    a.idx = b->idx;
    a.p_txt = b->p_txt;
    a.cache_len_in = b->cache_len_in;
    a.n_seqs = b->n_seqs;
    a.n_revisits = b->n_revisits;
    a.total_k = b->total_k;
    a.cache_len_out = o->cache_len_out;
    a.next_pos_out = o->next_pos_out;
    a.pos_out = o->pos_out;
    a.slot_out = o->slot_out;
    a.status = o->status;
    a.plan = plan_view(ws, b->total_k);
    a.mode = mode;
    a.L = L;
    a.flags = flags;
    return a;
}

enum KernelId { kRebind = 0, kCapture = 1, kFused = 2 };

// Resident CTAs per SM of a kernel per (device, kernel, block, smem), cached.
int blocks_per_sm(int dev, int block, size_t smem, int kernel = kRebind) {
    static std::mutex mu;
    static std::map<std::tuple<int, int, int, size_t>, int> cache;
    const auto key = std::make_tuple(dev, kernel, block, smem);
    {
        std::lock_guard<std::mutex> g(mu);
        auto it = cache.find(key);
        if (it != cache.end()) return it->second;
    }
    int n = 0;
    const cudaError_t e = kernel == kRebind    ? rebind_blocks_per_sm(block, smem, &n)
                          : kernel == kCapture ? capture_blocks_per_sm(block, smem, &n)
                                               : fused_blocks_per_sm(block, smem, &n);
    if (e != cudaSuccess || n < 1) n = 1;
    std::lock_guard<std::mutex> g(mu);
    cache[key] = n;
    return n;
}

int sm_count(int dev) {
    static std::mutex mu;
    static std::map<int, int> cache;
    {
        std::lock_guard<std::mutex> g(mu);
        auto it = cache.find(dev);
        if (it != cache.end()) return it->second;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        n = 1;
    std::lock_guard<std::mutex> g(mu);
    cache[dev] = n;
    return n;
}

// Layers each rebind CTA walks. Every CTA of a grid does the same work, so
// the grid runs in ceil(waves) rounds of `slots` resident CTAs: pick the
// group size whose waves are fullest (counting a short last group), charging
// each CTA's cos/sin prologue as about a tenth of one layer's rows, and
// prefer the larger group on ties. A grid that fits in one wave uses one
// layer per CTA (shortest CTAs, lowest latency).
int layers_per_cta(int64_t tiles, int n_layers, int64_t slots) {
    if (tiles * n_layers <= slots) return 1;
    int best = n_layers;
    double best_eff = -1.0;
    for (int G = n_layers; G >= 1; --G) {
        const int64_t groups = (n_layers + G - 1) / G;
        if (groups > 65535) break;
        const double waves = double(tiles * groups) / double(slots);
        const double eff = waves / std::ceil(waves) * double(n_layers) / double(groups * G) /
                           (1.0 + 0.1 / G);
        if (eff > best_eff + 1e-9) {
            best = G;
            best_eff = eff;
        }
    }
    return best;
}

// Arguments and launch shape of the row-moving kernel (rebind or fused).
int rebind_setup(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                 const prcr_cache_desc* cache, const prcr_revisit_batch* b, const prcr_outputs* o,
                 void* ws, RebindArgs& a, dim3& grid, int& block, size_t& smem,
                 KernelId kernel = kRebind) {
    a = RebindArgs{};
    a.store_k = static_cast<const uint16_t*>(store->k);
    a.store_v = static_cast<const uint16_t*>(store->v);
    a.cache_k = static_cast<uint16_t*>(cache->k);
    a.cache_v = static_cast<uint16_t*>(cache->v);
    a.store_layer_stride = store->layer_stride;
    a.cache_layer_stride = cache->layer_stride;
    const PlanView pv = plan_view(ws, b->total_k);
    a.plan_src = pv.src;
    a.plan_dst = pv.dst;
    a.plan_pos = pv.pos;
    a.status = o->status;
    a.total_k = b->total_k;
    a.n_layers = cfg->n_layers;
    a.head_dim = cfg->head_dim;
    a.layout = cfg->layout;
    a.sec_t = cfg->sections[0];
    a.sec_h = cfg->sections[1];
    a.sec_w = cfg->sections[2];
    const int P = cfg->head_dim / 2;
    copy_turn_freq(cfg, a.turn_freq);

    // One thread per (token, head, 16-byte vector of the first half row).
    const int lanes = cfg->n_kv_heads * (cfg->head_dim / 16);
    int T = kRebindTargetThreads / lanes;
    if (T < 1) T = 1;
    block = T * lanes;
    smem = size_t(2) * T * P * sizeof(float);
    a.lanes = lanes;
    a.tok_per_cta = T;
    if (kernel == kFused) smem += fused_stage_bytes(block);

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
    const int64_t tiles = (b->total_k + T - 1) / T;
    const int64_t slots = int64_t(sm_count(dev)) * blocks_per_sm(dev, block, smem, kernel);
    const int G = layers_per_cta(tiles, cfg->n_layers, slots);
    const int64_t groups = (cfg->n_layers + G - 1) / G;
    a.layers_per_cta = G;
    if (tiles > INT32_MAX) return PRCR_EINVAL;
    grid = dim3(unsigned(tiles), unsigned(groups), 1);
    return PRCR_OK;
}

int do_rebind(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
              const prcr_cache_desc* cache, const prcr_revisit_batch* b, const prcr_outputs* o,
              void* ws, cudaStream_t stream) {
    if (b->total_k == 0) return PRCR_OK;
    RebindArgs a;
    dim3 grid;
    int block = 0;
    size_t smem = 0;
    const int rc = rebind_setup(cfg, store, cache, b, o, ws, a, grid, block, smem);
    if (rc) return rc;
    return launch_rebind(a, grid, block, smem, stream) == cudaSuccess ? PRCR_OK : PRCR_ECUDA;
}

int do_plan(const prcr_store_desc* store, const prcr_cache_desc* cache,
            const prcr_revisit_batch* b, const prcr_outputs* o, int32_t mode, int32_t L,
            int32_t flags, void* ws, cudaStream_t stream) {
    const PlanArgs a = make_plan_args(store, cache, b, o, mode, L, flags, ws);
    return launch_plan(a, stream) == cudaSuccess ? PRCR_OK : PRCR_ECUDA;
}

int do_capture(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
               const prcr_cache_desc* cache, int32_t seq, int32_t layer_begin, int32_t n_layers,
               int32_t m_begin, int32_t m_count, int64_t slot_begin, const void* k_src,
               const void* v_src, int64_t src_layer_stride, int64_t src_token_stride,
               const int32_t* coords_src, uint32_t* status, cudaStream_t stream) {
    CaptureArgs a = {};
    const int64_t sbase = int64_t(seq) * store->seq_stride + int64_t(layer_begin) * store->layer_stride +
                          int64_t(m_begin) * store->token_stride;
    a.src_k = static_cast<const uint16_t*>(k_src);
    a.src_v = static_cast<const uint16_t*>(v_src);
    a.src_layer_stride = src_layer_stride;
    a.src_token_stride = src_token_stride;
    a.store_k = static_cast<uint16_t*>(store->k) + sbase;
    a.store_v = static_cast<uint16_t*>(store->v) + sbase;
    a.store_layer_stride = store->layer_stride;
    a.store_token_stride = store->token_stride;
    a.store_coords = store->coords + int64_t(seq) * store->coord_seq_stride + 3 * int64_t(m_begin);
    a.coords = coords_src;
    a.cache_k = static_cast<uint16_t*>(cache->k) + int64_t(layer_begin) * cache->layer_stride;
    a.cache_v = static_cast<uint16_t*>(cache->v) + int64_t(layer_begin) * cache->layer_stride;
    a.cache_layer_stride = cache->layer_stride;
    a.cache_kind = cache->kind;
    a.slot_stride = cache->slot_stride;
    a.slot_begin = slot_begin;
    if (cache->kind == PRCR_CACHE_CONTIGUOUS) {
        a.cache_seq_off = int64_t(seq) * cache->seq_stride;
        a.capacity = cache->max_slots;
        a.block_size = 1;
    } else {
        a.bt_row = cache->block_table + int64_t(seq) * cache->bt_stride;
        a.block_size = cache->block_size;
        a.block_stride = cache->block_stride;
        a.n_blocks = cache->n_blocks;
        a.capacity = int64_t(cache->bt_stride) * cache->block_size;
    }
    a.status = status;
    a.m_count = m_count;
    a.n_layers = n_layers;
    a.head_dim = cfg->head_dim;
    a.layout = cfg->layout;
    a.sec_t = cfg->sections[0];
    a.sec_h = cfg->sections[1];
    a.sec_w = cfg->sections[2];
    const int P = cfg->head_dim / 2;
    copy_turn_freq(cfg, a.turn_freq);
    const int lanes = cfg->n_kv_heads * (cfg->head_dim / 16);
    int T = kRebindTargetThreads / lanes;
    if (T < 1) T = 1;
    const int block = T * lanes;
    const size_t smem = size_t(2) * T * P * sizeof(float) + size_t(T) * sizeof(int64_t);
    a.lanes = lanes;
    a.tok_per_cta = T;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
    const int64_t tiles = (int64_t(m_count) + T - 1) / T;
    const int64_t slots = int64_t(sm_count(dev)) * blocks_per_sm(dev, block, smem, kCapture);
    const int G = layers_per_cta(tiles, n_layers, slots);
    a.layers_per_cta = G;
    const dim3 grid(unsigned(tiles), unsigned((n_layers + G - 1) / G), 1);
    return launch_capture(a, grid, block, smem, stream) == cudaSuccess ? PRCR_OK : PRCR_ECUDA;
}

// dynamic shared memory of the decode kernel: under the 48 KiB default limit
// with room for its 1 KiB of static cos/sin
constexpr size_t kDecodeSmem = 46 * 1024;

// Chunking of the decode step. Sequence lengths differ, so CTAs differ in
// work: aim at ~8 waves of resident CTAs (3 per SM) so that the last wave is
// short, with chunks of at least 256 slots (to amortise each CTA's query
// rotation), a multiple of 32, at most kDecodeMaxChunk, and small enough for
// the chunk's row offsets to fit beside the rotated queries in shared memory.
// A small batch (work for fewer than ~6 waves at 768 slots per chunk) with
// head_dim 64 or 128 takes the ring kernel instead (*ring = 1): its KV heads
// are split over CTAs of kDecodeRingWarps warps and the chunk is sized so that
// the grid is about one wave of kDecodeRingCtasPerSm CTAs per SM, each warp
// streaming its chunk through a shared-memory ring.
void decode_split(int64_t base_ctas, int64_t max_len, int sms, int64_t q_elems, int n_kv_heads,
                  int head_dim, int* splits, int* chunk, int* ring) {
    const bool small = base_ctas * ((max_len + 767) / 768) < int64_t(sms) * 6;
    if (small && (head_dim == 64 || head_dim == 128)) {
        const int64_t units = base_ctas * ((n_kv_heads + kDecodeRingWarps - 1) / kDecodeRingWarps);
        int64_t want = int64_t(sms) * kDecodeRingCtasPerSm / units;
        if (want < 1) want = 1;
        int64_t c = (max_len + want - 1) / want;
        c = (c + 15) / 16 * 16;
        if (c > kDecodeMaxChunk) c = kDecodeMaxChunk;
        *ring = 1;
        *chunk = int(c);
        *splits = int((max_len + c - 1) / c);
        if (*splits < 1) *splits = 1;
        return;
    }
    *ring = 0;
    int64_t want = (int64_t(sms) * 24 + base_ctas - 1) / base_ctas;
    if (want < 1) want = 1;
    int64_t c = (max_len + want - 1) / want;
    c = (c + 31) / 32 * 32;
    // Below ~768 slots a chunk's prologue and its share of the merge outweigh
    // the better balance when there is work for a few waves anyway (measured:
    // 512 -> 768 slots took the qwen25vl-7b shape from 5032 to 5394 GB/s;
    // 1184 -> 768 changed qwen3vl-8b by < 1 %). A small batch at head_dim 256
    // (the CUDA-core kernel) needs the parallelism instead: chunks of 64 slots.
    const int64_t floor_c = small ? 64 : 768;
    if (c < floor_c) c = floor_c;
    if (c > kDecodeMaxChunk) c = kDecodeMaxChunk;
    const int64_t cap = (int64_t(kDecodeSmem) - q_elems * int64_t(sizeof(float))) / 8 / 32 * 32;
    if (c > cap) c = cap;
    *chunk = int(c);
    *splits = int((max_len + c - 1) / c);
    if (*splits < 1) *splits = 1;
}

bool decode_shape_ok(const prcr_rope_cfg* cfg, int32_t n_q_heads) {
    const int D = cfg->head_dim;
    if (D != 64 && D != 128 && D != 256) return false;
    if (int64_t(n_q_heads) * D > PRCR_DECODE_MAX_Q_ELEMS) return false;
    if (n_q_heads < cfg->n_kv_heads || n_q_heads % cfg->n_kv_heads) return false;
    return n_q_heads / cfg->n_kv_heads <= 8;
}

// Checks and fills what both selection entry points share: heads, k, the
// output pointers and the workspace, laid out for token tiles of `tile`.
int select_common(const prcr_rope_cfg* cfg, int32_t n_seqs, int32_t layer, int32_t n_q_heads,
                  int32_t n_tokens, const void* q, const int64_t* q_pos, int32_t k,
                  int32_t* idx_out, int32_t* seq_rev_off, int32_t* rev_tok_off, float* score_out,
                  void* workspace, size_t workspace_bytes, int tile, SelectArgs& a) {
    const int H = cfg->n_kv_heads;
    if (n_seqs < 0 || layer < 0 || layer >= cfg->n_layers || n_q_heads < H || n_q_heads % H ||
        n_q_heads / H > 8 || n_q_heads > kSelectMaxQHeads ||
        int64_t(n_q_heads) * cfg->head_dim > PRCR_DECODE_MAX_Q_ELEMS ||
        n_tokens > PRCR_SELECT_MAX_TOKENS || k < 1 || k > n_tokens)
        return PRCR_EINVAL;
    if (int64_t(n_seqs) * k > INT32_MAX) return PRCR_EINVAL;
    if (n_seqs == 0) return PRCR_OK;
    if (!q || !q_pos || !idx_out || !seq_rev_off || !rev_tok_off) return PRCR_EINVAL;
    if (!aligned4(q) || !aligned8(q_pos) || !aligned4(idx_out) || !aligned4(seq_rev_off) ||
        !aligned4(rev_tok_off) || (score_out && !aligned4(score_out)))
        return PRCR_EALIGN;
    if (!workspace || workspace_bytes < prcr_select_workspace_size(n_seqs, n_q_heads, n_tokens))
        return PRCR_EWORKSPACE;
    if (!aligned16(workspace)) return PRCR_EALIGN;
    a.q = static_cast<const uint16_t*>(q);
    a.q_pos = q_pos;
    a.layer = layer;
    a.n_tokens = n_tokens;
    a.n_kv_heads = H;
    a.n_q_heads = n_q_heads;
    a.head_dim = cfg->head_dim;
    a.k = k;
    a.layout = cfg->layout;
    a.sec_t = cfg->sections[0];
    a.sec_h = cfg->sections[1];
    a.sec_w = cfg->sections[2];
    a.scale = float(1.0 / std::sqrt(double(cfg->head_dim)));
    {
        char* w = static_cast<char*>(workspace);
        const int64_t Bn = n_seqs, Hn = n_q_heads, M = n_tokens;
        a.n_seqs = n_seqs;
        a.tok_tile = tile;
        a.n_tiles = int32_t((M + tile - 1) / tile);
        const int64_t max_tiles = (M + kSelectTokTile - 1) / kSelectTokTile;
        a.logits = reinterpret_cast<float*>(w);
        w += align256(size_t(4 * Bn * Hn * M));
        a.tile_stats = reinterpret_cast<float*>(w);
        w += align256(size_t(8 * Bn * Hn * max_tiles));
        a.norm = reinterpret_cast<float*>(w);
        w += align256(size_t(8 * Bn * Hn));
        a.rel = reinterpret_cast<float*>(w);
    }
    a.score_out = score_out;
    a.idx_out = idx_out;
    a.rev_tok_off = rev_tok_off;
    a.seq_rev_off = seq_rev_off;
    copy_turn_freq(cfg, a.turn_freq);
    return PRCR_OK;
}

}  // namespace
}  // namespace prcr

using namespace prcr;

extern "C" {

size_t prcr_workspace_size(int64_t total_k) { return workspace_bytes(total_k); }

int prcr_plan(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
              const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
              const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags, void* workspace,
              size_t workspace_bytes, void* stream) {
    int rc = check_call(cfg, store, cache, batch, out, mode, L, flags, workspace, workspace_bytes);
    if (rc || batch->n_seqs == 0) return rc;
    return do_plan(store, cache, batch, out, mode, L, flags, workspace,
                   static_cast<cudaStream_t>(stream));
}

int prcr_rebind_apply(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                      const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
                      const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags,
                      void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_call(cfg, store, cache, batch, out, mode, L, flags, workspace, workspace_bytes);
    if (rc || batch->n_seqs == 0) return rc;
    return do_rebind(cfg, store, cache, batch, out, workspace, static_cast<cudaStream_t>(stream));
}

int prcr_rebind_inject(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                       const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
                       const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags,
                       void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_call(cfg, store, cache, batch, out, mode, L, flags, workspace, workspace_bytes);
    if (rc || batch->n_seqs == 0) return rc;
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (batch->total_k > 0 && batch->total_k <= kFusedMaxTokens &&
        batch->n_revisits <= kFusedMaxRevisits && batch->n_seqs <= kFusedMaxSeqs) {
        // a few small revisits: one kernel plans and moves them (no plan round
        // trip), when its grid runs as a single wave, so that every CTA's own
        // planning happens at once instead of wave after wave
        FusedArgs fa;
        dim3 grid;
        int block = 0;
        size_t smem = 0;
        rc = rebind_setup(cfg, store, cache, batch, out, workspace, fa.rebind, grid, block, smem,
                          kFused);
        if (rc) return rc;
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
        const int64_t resident = int64_t(sm_count(dev)) * blocks_per_sm(dev, block, smem, kFused);
        // (its CTA loads the offsets with one thread per entry)
        if (int64_t(grid.x) * grid.y <= resident && block > kFusedMaxRevisits &&
            block > kFusedMaxSeqs) {
            fa.plan = make_plan_args(store, cache, batch, out, mode, L, flags, workspace);
            return launch_fused(fa, grid, block, smem, s) == cudaSuccess ? PRCR_OK : PRCR_ECUDA;
        }
    }
    rc = do_plan(store, cache, batch, out, mode, L, flags, workspace, s);
    if (rc) return rc;
    return do_rebind(cfg, store, cache, batch, out, workspace, s);
}

int prcr_store_raw(const prcr_rope_cfg* cfg, const prcr_store_desc* store, int32_t seq,
                   int32_t layer_begin, int32_t n_layers, int32_t m_begin, int32_t m_count,
                   const void* k_src, const void* v_src, int64_t src_layer_stride,
                   int64_t src_token_stride, const int32_t* coords_src, void* stream) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_store(cfg, store))) return rc;
    if (seq < 0 || seq >= store->n_seqs || layer_begin < 0 || n_layers < 0 ||
        layer_begin + int64_t(n_layers) > cfg->n_layers || m_begin < 0 || m_count < 0 ||
        m_begin + int64_t(m_count) > store->n_tokens)
        return PRCR_EINVAL;
    if (n_layers == 0 || m_count == 0) return PRCR_OK;
    const int64_t row = int64_t(cfg->n_kv_heads) * cfg->head_dim;
    if (!k_src || !v_src || src_token_stride < row || src_layer_stride < 0) return PRCR_EINVAL;
    if (!aligned16(k_src) || !aligned16(v_src) || !mult8(src_layer_stride) ||
        !mult8(src_token_stride) || (coords_src && !aligned4(coords_src)))
        return PRCR_EALIGN;
    StoreArgs a = {};
    const int64_t base = int64_t(seq) * store->seq_stride + int64_t(layer_begin) * store->layer_stride +
                         int64_t(m_begin) * store->token_stride;
    a.dst_k = static_cast<uint16_t*>(store->k) + base;
    a.dst_v = static_cast<uint16_t*>(store->v) + base;
    a.src_k = static_cast<const uint16_t*>(k_src);
    a.src_v = static_cast<const uint16_t*>(v_src);
    a.dst_layer_stride = store->layer_stride;
    a.dst_token_stride = store->token_stride;
    a.src_layer_stride = src_layer_stride;
    a.src_token_stride = src_token_stride;
    a.n_layers = n_layers;
    a.m_count = m_count;
    a.row_vecs = int32_t(row / 8);
    a.dst_coords = coords_src ? store->coords + int64_t(seq) * store->coord_seq_stride +
                                    3 * int64_t(m_begin)
                              : nullptr;
    a.src_coords = coords_src;
    return launch_store(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? PRCR_OK
                                                                             : PRCR_ECUDA;
}

int prcr_prefill_capture(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                         const prcr_cache_desc* cache, int32_t seq, int32_t layer_begin,
                         int32_t n_layers, int32_t m_begin, int32_t m_count, int64_t slot_begin,
                         const void* k_src, const void* v_src, int64_t src_layer_stride,
                         int64_t src_token_stride, const int32_t* coords_src, uint32_t* status,
                         void* stream) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_store(cfg, store))) return rc;
    if ((rc = check_cache(cfg, cache))) return rc;
    if (seq < 0 || seq >= store->n_seqs || seq >= cache->n_seqs || layer_begin < 0 ||
        n_layers < 0 || layer_begin + int64_t(n_layers) > cfg->n_layers || m_begin < 0 ||
        m_count < 0 || m_begin + int64_t(m_count) > store->n_tokens || slot_begin < 0)
        return PRCR_EINVAL;
    if (n_layers == 0 || m_count == 0) return PRCR_OK;
    const int64_t row = int64_t(cfg->n_kv_heads) * cfg->head_dim;
    if (!k_src || !v_src || !coords_src || !status || src_token_stride < row ||
        src_layer_stride < 0)
        return PRCR_EINVAL;
    if (!aligned16(k_src) || !aligned16(v_src) || !mult8(src_layer_stride) ||
        !mult8(src_token_stride) || !aligned4(coords_src) || !aligned4(status))
        return PRCR_EALIGN;
    return do_capture(cfg, store, cache, seq, layer_begin, n_layers, m_begin, m_count, slot_begin,
                      k_src, v_src, src_layer_stride, src_token_stride, coords_src, status,
                      static_cast<cudaStream_t>(stream));
}

size_t prcr_decode_workspace_size(const prcr_rope_cfg* cfg, int32_t n_seqs, int32_t n_q_heads,
                                  int64_t max_len) {
    if (check_cfg(cfg) || n_seqs < 1 || max_len < 1 || !decode_shape_ok(cfg, n_q_heads)) return 0;
    int dev = 0, sms = 1;
    if (cudaGetDevice(&dev) == cudaSuccess) sms = sm_count(dev);
    int splits = 1, chunk = 32, ring = 0;
    decode_split(int64_t(n_seqs) * cfg->n_layers, max_len, sms, int64_t(n_q_heads) * cfg->head_dim,
                 cfg->n_kv_heads, cfg->head_dim, &splits, &chunk, &ring);
    if (splits == 1) return 0;
    return size_t(n_seqs) * cfg->n_layers * n_q_heads * splits * (cfg->head_dim + 2) * sizeof(float);
}

int prcr_decode_attention(const prcr_rope_cfg* cfg, const prcr_cache_desc* cache, int32_t n_seqs,
                          int32_t n_q_heads, const void* q, const int64_t* q_pos,
                          const int32_t* seq_len, int64_t max_len, float* out, uint32_t* status,
                          void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_cache(cfg, cache))) return rc;
    if (!decode_shape_ok(cfg, n_q_heads) || n_seqs < 0 || n_seqs > cache->n_seqs || max_len < 0)
        return PRCR_EINVAL;
    if (n_seqs == 0 || max_len == 0) return PRCR_OK;
    if (!q || !q_pos || !seq_len || !out || !status) return PRCR_EINVAL;
    if (!aligned4(q) || !aligned8(q_pos) || !aligned4(seq_len) || !aligned16(out) ||
        !aligned4(status))
        return PRCR_EALIGN;
    const int64_t capacity = cache->kind == PRCR_CACHE_CONTIGUOUS
                                 ? int64_t(cache->max_slots)
                                 : int64_t(cache->bt_stride) * cache->block_size;
    if (max_len > capacity) return PRCR_EINVAL;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
    DecodeArgs a = {};
    decode_split(int64_t(n_seqs) * cfg->n_layers, max_len, sm_count(dev),
                 int64_t(n_q_heads) * cfg->head_dim, cfg->n_kv_heads, cfg->head_dim, &a.splits,
                 &a.chunk, &a.ring);
    if (n_seqs > 65535 || cfg->n_layers > 65535) return PRCR_EINVAL;  // grid z and y
    if (a.splits > 1) {
        const size_t need = size_t(n_seqs) * cfg->n_layers * n_q_heads * a.splits *
                            (cfg->head_dim + 2) * sizeof(float);
        if (!workspace || workspace_bytes < need) return PRCR_EWORKSPACE;
        if (!aligned16(workspace)) return PRCR_EALIGN;
        a.partial = static_cast<float*>(workspace);
    }
    a.q = static_cast<const uint16_t*>(q);
    a.q_pos = q_pos;
    a.seq_len = seq_len;
    a.cache_k = static_cast<const uint16_t*>(cache->k);
    a.cache_v = static_cast<const uint16_t*>(cache->v);
    a.layer_stride = cache->layer_stride;
    a.seq_stride = cache->seq_stride;
    a.block_stride = cache->block_stride;
    a.slot_stride = cache->slot_stride;
    a.capacity = capacity;
    a.block_table = cache->block_table;
    a.bt_stride = cache->bt_stride;
    a.block_size = cache->kind == PRCR_CACHE_PAGED ? cache->block_size : 1;
    a.n_blocks = cache->n_blocks;
    a.cache_kind = cache->kind;
    a.out = out;
    a.status = status;
    a.n_layers = cfg->n_layers;
    a.n_kv_heads = cfg->n_kv_heads;
    a.n_q_heads = n_q_heads;
    a.head_dim = cfg->head_dim;
    a.group = n_q_heads / cfg->n_kv_heads;
    a.scale = float(1.0 / std::sqrt(double(cfg->head_dim)));
    copy_turn_freq(cfg, a.turn_freq);
    int gp = 1;
    while (gp < a.group) gp <<= 1;
    const size_t smem = size_t(n_q_heads) * cfg->head_dim * sizeof(float) +
                        size_t(a.chunk) * sizeof(int64_t);
    const dim3 grid(unsigned(a.splits), unsigned(cfg->n_layers), unsigned(n_seqs));
    return launch_decode(a, gp, grid, smem, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? PRCR_OK
               : PRCR_ECUDA;
}

size_t prcr_select_workspace_size(int32_t n_seqs, int32_t n_q_heads, int32_t n_tokens) {
    if (n_seqs < 1 || n_q_heads < 1 || n_tokens < 1) return 0;
    return select_workspace_bytes(n_seqs, n_q_heads, n_tokens);
}

int prcr_select_topk(const prcr_rope_cfg* cfg, const prcr_store_desc* store, int32_t n_seqs,
                     int32_t layer, int32_t n_q_heads, const void* q, const int64_t* q_pos,
                     int32_t k, int32_t* idx_out, int32_t* seq_rev_off, int32_t* rev_tok_off,
                     float* score_out, void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_store(cfg, store))) return rc;
    if (n_seqs > store->n_seqs) return PRCR_EINVAL;
    SelectArgs a = {};
    // token tiles of the softmax statistics: 16 tokens (one warp's MMA rows)
    // for the tensor-core logits kernel (head_dim 64, 128); else the CUDA-core
    // kernel's tiles, 64 tokens (32 at head_dim 256, whose cos/sin rows are
    // twice as long)
    const int D = cfg->head_dim;
    rc = select_common(cfg, n_seqs, layer, n_q_heads, store->n_tokens, q, q_pos, k, idx_out,
                       seq_rev_off, rev_tok_off, score_out, workspace, workspace_bytes,
                       D == 64 || D == 128 ? 16 : (D > 128 ? 32 : 64), a);
    if (rc || n_seqs == 0) return rc;
    a.store_k = static_cast<const uint16_t*>(store->k);
    a.store_seq_stride = store->seq_stride;
    a.store_layer_stride = store->layer_stride;
    a.store_token_stride = store->token_stride;
    a.coords = store->coords;
    a.coord_seq_stride = store->coord_seq_stride;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
    return launch_select(a, n_seqs, sm_count(dev), static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? PRCR_OK
               : PRCR_ECUDA;
}

int prcr_select_topk_cached(const prcr_rope_cfg* cfg, const prcr_cache_desc* cache, int32_t n_seqs,
                            int32_t layer, int32_t n_q_heads, int32_t n_tokens,
                            const int32_t* img_slot0, const void* q, const int64_t* q_pos, int32_t k,
                            int32_t* idx_out, int32_t* seq_rev_off, int32_t* rev_tok_off,
                            float* score_out, uint32_t* status, void* workspace,
                            size_t workspace_bytes, void* stream) {
    int rc = check_cfg(cfg);
    if (rc) return rc;
    if ((rc = check_cache(cfg, cache))) return rc;
    if (n_seqs > cache->n_seqs || n_tokens < 1 ||
        (cfg->head_dim != 64 && cfg->head_dim != 128 && cfg->head_dim != 256))
        return PRCR_EINVAL;
    SelectArgs a = {};
    // token tiles of 16: one warp's MMA tile of keys
    rc = select_common(cfg, n_seqs, layer, n_q_heads, n_tokens, q, q_pos, k, idx_out, seq_rev_off,
                       rev_tok_off, score_out, workspace, workspace_bytes, 16, a);
    if (rc || n_seqs == 0) return rc;
    if (!img_slot0 || !status) return PRCR_EINVAL;
    if (!aligned4(img_slot0) || !aligned4(status)) return PRCR_EALIGN;
    a.cache_k = static_cast<const uint16_t*>(cache->k);
    a.cache_seq_stride = cache->seq_stride;
    a.cache_layer_stride = cache->layer_stride;
    a.cache_block_stride = cache->block_stride;
    a.cache_slot_stride = cache->slot_stride;
    a.cache_capacity = cache->kind == PRCR_CACHE_CONTIGUOUS
                           ? int64_t(cache->max_slots)
                           : int64_t(cache->bt_stride) * cache->block_size;
    a.block_table = cache->block_table;
    a.bt_stride = cache->bt_stride;
    a.block_size = cache->kind == PRCR_CACHE_PAGED ? cache->block_size : 1;
    a.n_blocks = cache->n_blocks;
    a.cache_kind = cache->kind;
    a.img_slot0 = img_slot0;
    a.status = status;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PRCR_ECUDA;
    return launch_select_cached(a, n_seqs, sm_count(dev), static_cast<cudaStream_t>(stream)) ==
                   cudaSuccess
               ? PRCR_OK
               : PRCR_ECUDA;
}

int64_t prcr_next_text_pos(int64_t p_txt, int64_t k_seq, int32_t mode) {
    switch (mode) {
        case PRCR_MODE_PCR:
        case PRCR_MODE_ORIGINAL:
        case PRCR_MODE_UIR:
            return p_txt + 1;
        case PRCR_MODE_LPA:
            return p_txt + k_seq + 1;
        default:
            return INT64_MIN;
    }
}

const char* prcr_error_string(int code) {
    switch (code) {
        case PRCR_OK: return "ok";
        case PRCR_EINVAL: return "invalid argument";
        case PRCR_EALIGN: return "pointer or stride not 16-byte aligned";
        case PRCR_EWORKSPACE: return "workspace missing or too small";
        case PRCR_ECUDA: return "CUDA launch failed";
        default: return "unknown error";
    }
}

int prcr_version(void) { return PRCR_VERSION; }

}  // extern "C"
