/*
 * prcr.h - C ABI of the PRCR visual-revisit library (libprcr.so, sm_103a).
 *
 * Position Rebinding Cache Reuse revisits image evidence during decoding
 * without re-running the decoder on it: raw (pre-rotation) visual K/V are
 * kept per layer with each token's original coordinate (Sec. 3.1, Eq.
 * "global_raw_memory"); at a revisit the selected entries are gathered, given
 * new positions that start at the current text position and keep their
 * relative layout (Sec. 3.2, Algorithm 1), their keys are rotated again at
 * those positions and the values reused as they are (Sec. 3.3, Eq.
 * "cache_reconstruction"), and both are appended to the active decoder cache
 * (Eq. "active_cache"). The next text position stays p_txt + 1.
 *
 * Conventions for every entry point:
 *  - All array pointers named "device" point to memory of the current CUDA
 *    device; the caller owns and allocates all of it. The library never
 *    allocates, frees or synchronises; work is enqueued on `stream`
 *    (a cudaStream_t; NULL = the legacy default stream) and runs
 *    asynchronously. Kernels are launched with programmatic stream
 *    serialization: one may become resident while the preceding kernel on
 *    the stream drains, but it reads and writes no memory before that
 *    kernel has completed, so stream order is exactly that of plain launches.
 *  - K/V elements are bf16 (IEEE binary16-brain bit patterns). A token row is
 *    [n_kv_heads][head_dim] contiguous elements; strides between rows,
 *    layers, sequences and blocks are given in elements. Every row start must
 *    be 16-byte aligned (base pointers 16-byte aligned, strides multiples of 8).
 *  - Return value: PRCR_OK (0) or a negative PRCR_E* code. A negative code
 *    means nothing was enqueued. Errors found on the device (bad index,
 *    missing block, full cache, malformed offsets, a position out of range)
 *    are OR-ed as PRCR_ST_* bits into the caller's device status word; the
 *    offending rows are skipped (each entry point states what it outputs
 *    for them), nothing is written out of bounds and no kernel traps.
 *  - Rotation angles: position x theta^(-2i/D) is reduced modulo one turn
 *    exactly in integer fixed point (the position in signed 32.32, the pair's
 *    rate theta^(-2i/D) / (2 pi) in unsigned 0.64, computed once on the host
 *    in long double), giving the angle to 2^-32 of a turn; only the final
 *    sin/cos is float32. This needs |position| < 2^31 (PRCR_ST_POS_RANGE
 *    otherwise).
 *  - State: the outputs of a call depend only on its arguments. The library
 *    keeps process-wide caches that are filled on first use and read-only
 *    afterwards (guarded by a mutex): the turn rates per (theta, head_dim),
 *    the SM count, kernel occupancies and the one-kernel revisit path's
 *    shared-memory limit per device, and, for prcr_rebind_inject_static only,
 *    a fixed scratch array per device and its address. The per-device entries
 *    assume the device is not reset while the process uses the library.
 *    Every entry point except prcr_rebind_inject_static may be called from
 *    several host threads at once.
 */
#ifndef PRCR_H_
#define PRCR_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* 2: adds prcr_select_topk_cached (1: every other entry point) */
#define PRCR_VERSION 2

#if defined(__GNUC__)
#define PRCR_API __attribute__((visibility("default")))
#else
#define PRCR_API
#endif

/* Return codes */
#define PRCR_OK          0
#define PRCR_EINVAL     -1  /* null pointer, bad size, bad config or mode      */
#define PRCR_EALIGN     -2  /* a pointer or stride breaks 16-byte row alignment */
#define PRCR_EWORKSPACE -3  /* workspace missing or smaller than required       */
#define PRCR_ECUDA      -4  /* a CUDA launch or query failed                    */

/* Device status bits (OR-ed into *status) */
#define PRCR_ST_IDX_RANGE  1u  /* a selected index is outside [0, n_tokens)          */
#define PRCR_ST_NO_BLOCK   2u  /* paged: block-table entry < 0 or >= n_blocks         */
#define PRCR_ST_CAPACITY   4u  /* a slot lies beyond the sequence's cache capacity     */
#define PRCR_ST_CSR        8u  /* offsets not monotone / not spanning [0, total_k)     */
#define PRCR_ST_POS_RANGE 16u  /* a reassigned position cannot be formed as a correctly
                                  rounded exact rational (operands of 2^52 or more),
                                  or a position or query position has magnitude 2^31
                                  or more (beyond the exact fixed-point angle
                                  reduction): the rebind skips that token's rows;
                                  decode and cached selection treat that sequence as
                                  having no readable slot                             */

/* Position rules (Sec. 3.2; Table 2) */
#define PRCR_MODE_PCR      0  /* Position-Consistent Reinsertion (the method)        */
#define PRCR_MODE_ORIGINAL 1  /* stored coordinates: the position-bound cache of
                                 Eq. "historical_position_bound_kv" (direct reuse)  */
#define PRCR_MODE_UIR      2  /* uniform interval: p + j/(K+1)                        */
#define PRCR_MODE_LPA      3  /* linear appending: p + r, next position p + K_seq + 1 */

/* flags */
#define PRCR_FLAG_DEGENERATE_CENTER 1  /* u = 1/2 (not 0) on an axis with max == min */

/* M-RoPE band layouts */
#define PRCR_LAYOUT_SECTIONED   0  /* pairs [0,s_t) -> t, [s_t,s_t+s_h) -> h, rest -> w */
#define PRCR_LAYOUT_INTERLEAVED 1  /* pair i -> h if i%3==1 && i<3s_h, w if i%3==2 &&
                                      i<3s_w, else t                                  */

/* Cache kinds */
#define PRCR_CACHE_CONTIGUOUS 0
#define PRCR_CACHE_PAGED      1

#define PRCR_MAX_HEAD_DIM 256
#define PRCR_MAX_ROW_ELEMS 8192   /* n_kv_heads * head_dim */

/* Rotary configuration shared by the store and the cache. */
typedef struct prcr_rope_cfg {
    int32_t n_layers;     /* layers held by the store and the cache (>= 1)             */
    int32_t n_kv_heads;   /* H (>= 1)                                                  */
    int32_t head_dim;     /* D: multiple of 16, <= PRCR_MAX_HEAD_DIM                   */
    int32_t sections[3];  /* rotation pairs driven by t, h, w; sum == D/2, each >= 0   */
    int32_t layout;       /* PRCR_LAYOUT_*                                             */
    int32_t reserved;     /* must be 0                                                 */
    double  theta;        /* RoPE base (> 1); pair i turns at theta^(-2i/D) per unit    */
} prcr_rope_cfg;

/* Raw Visual Evidence Memory (Sec. 3.1, Eq. "global_raw_memory"): per sequence,
 * per layer, per visual token the pre-rotation key and value rows, plus each
 * token's original (t, h, w) coordinate.
 *   key of (seq b, layer l, token m, head h, dim d) is at
 *     k[b*seq_stride + l*layer_stride + m*token_stride + h*D + d]   (same for v)
 *   coordinate axis a of (b, m) is at coords[b*coord_seq_stride + 3*m + a]   */
typedef struct prcr_store_desc {
    void*    k;                 /* device, bf16                                   */
    void*    v;                 /* device, bf16                                   */
    int32_t* coords;            /* device, int32 (t, h, w) per token              */
    int64_t  seq_stride;        /* elements                                       */
    int64_t  layer_stride;      /* elements                                       */
    int64_t  token_stride;      /* elements, >= H*D                               */
    int64_t  coord_seq_stride;  /* int32 elements, >= 3*n_tokens                  */
    int32_t  n_seqs;            /* sequences held                                 */
    int32_t  n_tokens;          /* M: visual tokens per sequence                  */
} prcr_store_desc;

/* Active decoder cache the rebound rows are appended to (Eq. "active_cache").
 * CONTIGUOUS: row (b, l, slot s) at k[b*seq_stride + l*layer_stride + s*slot_stride],
 *             capacity max_slots slots per sequence.
 * PAGED:      slot s of sequence b lives in physical block
 *             blk = block_table[b*bt_stride + s/block_size] at offset o = s % block_size;
 *             row (l, blk, o) at k[l*layer_stride + blk*block_stride + o*slot_stride];
 *             capacity bt_stride*block_size slots per sequence.              */
typedef struct prcr_cache_desc {
    int32_t        kind;          /* PRCR_CACHE_*                                     */
    int32_t        block_size;    /* paged: slots per block (>= 1)                    */
    void*          k;             /* device, bf16                                     */
    void*          v;             /* device, bf16                                     */
    int64_t        seq_stride;    /* contiguous only, elements                        */
    int64_t        layer_stride;  /* elements                                         */
    int64_t        block_stride;  /* paged only, elements                             */
    int64_t        slot_stride;   /* elements between consecutive slots               */
    const int32_t* block_table;   /* paged only, device int32 [n_seqs][bt_stride]     */
    int32_t        bt_stride;     /* paged only: logical blocks per sequence row      */
    int32_t        n_blocks;      /* paged only: physical blocks in the pool          */
    int32_t        max_slots;     /* contiguous only: slots per sequence              */
    int32_t        n_seqs;        /* sequences the cache / block table holds          */
} prcr_cache_desc;

/* One decode step's revisits (Algorithm 1, Require line): for each sequence
 * b, revisits seq_rev_off[b] .. seq_rev_off[b+1]-1; revisit r selects the
 * store tokens idx[rev_tok_off[r] .. rev_tok_off[r+1]-1] (the index set
 * I_tau of Eq. 3, in the order they are appended). Sequence b's latest text
 * token is at position p_txt[b]; its cache holds cache_len_in[b] slots.      */
typedef struct prcr_revisit_batch {
    const int32_t* seq_rev_off;   /* device [n_seqs+1], seq_rev_off[0]=0, [n_seqs]=n_revisits */
    const int32_t* rev_tok_off;   /* device [n_revisits+1], [0]=0, [n_revisits]=total_k       */
    const int32_t* idx;           /* device [total_k], token ids in [0, n_tokens)             */
    const int64_t* p_txt;         /* device [n_seqs]                                           */
    const int32_t* cache_len_in;  /* device [n_seqs], >= 0; must not alias cache_len_out      */
    int32_t        n_seqs;        /* <= store.n_seqs and <= cache.n_seqs                       */
    int32_t        n_revisits;
    int64_t        total_k;       /* < 2^31                                                    */
} prcr_revisit_batch;

/* Outputs of one call. */
typedef struct prcr_outputs {
    int32_t*  cache_len_out;  /* device [n_seqs]: cache_len_in + tokens appended      */
    int64_t*  next_pos_out;   /* device [n_seqs]: next text position                  */
    double*   pos_out;        /* device [total_k][3] reassigned (t,h,w), or NULL       */
    int32_t*  slot_out;       /* device [total_k] cache slot of each token, or NULL    */
    uint32_t* status;         /* device word; must be 0 on entry; PRCR_ST_* bits OR-ed */
} prcr_outputs;

/* Bytes of device workspace prcr_rebind_inject / prcr_plan / prcr_rebind_apply
 * need for total_k selected tokens (the per-token plan: source and
 * destination row offsets and the three reassigned positions). */
PRCR_API size_t prcr_workspace_size(int64_t total_k);

/* prcr_rebind_inject - Algorithm 1 for a batch of sequences, in two kernels
 * on `stream`:
 *  1. plan (Sec. 3.2): per revisit, the coordinate range of Eq.
 *     "selected_coord_range"; per token, u of Eq. "normalized_coord" and the
 *     position of Eq. "image_range_fractional_reinsert" (or the rule `mode`
 *     selects), computed as one correctly rounded float64 division of an
 *     exact integer ratio; the token's cache slot (cache_len_in[b] + its rank
 *     among sequence b's tokens in this call) and source/destination rows.
 *  2. rebind + inject (Sec. 3.3): for every (token, layer, kv head) the raw
 *     key row is gathered, rotated with sectioned/interleaved M-RoPE at the
 *     new positions (angle reduced exactly modulo one turn in fixed point,
 *     then float32 sin/cos and float32 arithmetic, rounded to bf16 to
 *     nearest even), the raw value row is copied bit for bit, and both are
 *     written to the slot.
 * L is the left extension (L >= 0; the paper's default is 2, Sec. 4.4).
 * Rows of tokens with a device error are not written (a token whose position
 * sets PRCR_ST_POS_RANGE included: pos_out / slot_out still receive its
 * computed position and slot); slots outside the appended span are never
 * touched. cache_len_out and next_pos_out count every token of the call. The call is re-runnable: the same inputs
 * give the same outputs. workspace: device, >= prcr_workspace_size(total_k)
 * bytes, 16-byte aligned, not shared with a concurrent call.              */
PRCR_API int prcr_rebind_inject(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                       const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
                       const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags,
                       void* workspace, size_t workspace_bytes, void* stream);

/* prcr_plan - step 1 of prcr_rebind_inject alone (positions, slots,
 * cache_len_out, next_pos_out, status). Same arguments and rules. */
PRCR_API int prcr_plan(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
              const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
              const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags,
              void* workspace, size_t workspace_bytes, void* stream);

/* prcr_rebind_apply - step 2 of prcr_rebind_inject alone: consumes the plan a
 * preceding prcr_plan left in `workspace` (same arguments, same stream order)
 * and moves the rows. It reads out->status and does nothing when the plan
 * reported PRCR_ST_CSR. */
PRCR_API int prcr_rebind_apply(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                      const prcr_cache_desc* cache, const prcr_revisit_batch* batch,
                      const prcr_outputs* out, int32_t mode, int32_t L, int32_t flags,
                      void* workspace, size_t workspace_bytes, void* stream);

/* prcr_rebind_inject_static - prcr_rebind_inject without a caller workspace.
 * The paper has no counterpart to this call; it exists for callers that cannot
 * allocate device memory themselves (a plugin whose host framework owns all
 * device memory through its own pool, or a decode loop where cudaMalloc and
 * cudaFree, which can synchronise the device, are not allowed). It allocates
 * nothing: the per-token plan lives in a fixed array inside the library, of
 * PRCR_STATIC_MAX_TOKENS tokens (2.5 MiB), held on every GPU that loads the
 * library until the process exits. Inputs and outputs are passed and owned by
 * the caller exactly as for prcr_rebind_inject, with the same results.
 *  - total_k > PRCR_STATIC_MAX_TOKENS returns PRCR_EWORKSPACE, nothing enqueued.
 *  - The first call on a device looks up the array's device address (set-up
 *    done once per device); make that first call before any stream capture.
 *    The address is kept for the process: do not call this entry point on a
 *    device after a reset of that device (cudaDeviceReset, or its primary
 *    context released and created again), which leaves the kept address stale.
 *  - Arguments are checked as prcr_rebind_inject checks them (same codes)
 *    before the size limit and before any set-up.
 *  - Every call shares the one array: calls whose work overlaps on the GPU
 *    (other streams, other host threads) race and must be serialised by the
 *    caller. Nothing in the array needs to start at zero.                    */
#define PRCR_STATIC_MAX_TOKENS 65536
PRCR_API int prcr_rebind_inject_static(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                                       const prcr_cache_desc* cache,
                                       const prcr_revisit_batch* batch, const prcr_outputs* out,
                                       int32_t mode, int32_t L, int32_t flags, void* stream);

/* prcr_store_raw - fill the raw visual memory (Sec. 3.1, Eq. "raw_kv" and
 * "global_raw_memory"): copy pre-rotation K/V of tokens m_begin ..
 * m_begin+m_count-1, layers layer_begin .. layer_begin+n_layers-1 of sequence
 * `seq`, and their original coordinates, into the store.
 *   source key of (layer i, token j, head h, dim d):
 *     k_src[i*src_layer_stride + j*src_token_stride + h*D + d]   (device, bf16)
 *   coords_src: device int32 [m_count][3] (t, h, w), or NULL to leave the
 *   store's coordinates unchanged.
 * Ranges outside the store return PRCR_EINVAL. Source and store must not overlap. */
PRCR_API int prcr_store_raw(const prcr_rope_cfg* cfg, const prcr_store_desc* store, int32_t seq,
                   int32_t layer_begin, int32_t n_layers, int32_t m_begin, int32_t m_count,
                   const void* k_src, const void* v_src, int64_t src_layer_stride,
                   int64_t src_token_stride, const int32_t* coords_src, void* stream);

/* prcr_prefill_capture - build the raw visual memory during prefill
 * (Sec. 3.1, Eq. "raw_kv" and "global_raw_memory") in the same pass that
 * writes the model's ordinary cache entries for those tokens (Eq.
 * "historical_position_bound_kv": key rotated at the original coordinate,
 * value unchanged). Tokens m_begin .. m_begin+m_count-1, layers layer_begin ..
 * layer_begin+n_layers-1 of sequence `seq`:
 *   - the pre-rotation rows are read once from k_src / v_src (device bf16;
 *     row of (layer i, token j) at i*src_layer_stride + j*src_token_stride),
 *   - copied unchanged into the store, with coords_src (device int32
 *     [m_count][3], original (t, h, w)) into the store's coordinates,
 *   - and written as RoPE(k, p_m) and v into the cache at slots
 *     slot_begin .. slot_begin+m_count-1 of sequence `seq` (contiguous or
 *     paged through the block table).
 * Host-checked ranges return PRCR_EINVAL; a slot beyond the capacity or an
 * unmapped block sets PRCR_ST_CAPACITY / PRCR_ST_NO_BLOCK in *status (device
 * word) and skips that token's cache rows (its store rows are still written). */
PRCR_API int prcr_prefill_capture(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                                  const prcr_cache_desc* cache, int32_t seq, int32_t layer_begin,
                                  int32_t n_layers, int32_t m_begin, int32_t m_count,
                                  int64_t slot_begin, const void* k_src, const void* v_src,
                                  int64_t src_layer_stride, int64_t src_token_stride,
                                  const int32_t* coords_src, uint32_t* status, void* stream);

/* prcr_decode_attention - the first decode step over the active cache
 * (Sec. 3.3, Eq. "decode_with_active_cache"): for every sequence b, layer l
 * and query head h,
 *   out[b][l][h] = softmax(RoPE(q[b][l][h], (p, p, p)) K^T / sqrt(D)) V,
 * p = q_pos[b], over cache slots [0, seq_len[b]) of sequence b (contiguous, or
 * paged through the block table), the revisited rows included. Query head h
 * reads KV head h / (n_q_heads / n_kv_heads) (grouped-query attention).
 *   q:       device bf16 [n_seqs][n_layers][n_q_heads][D] raw (pre-rotation)
 *   q_pos:   device int64 [n_seqs]  (the next text position, e.g. next_pos_out)
 *   seq_len: device int32 [n_seqs]  (e.g. cache_len_out); max_len >= every
 *            seq_len is a host bound used for the split of the sequence axis
 *   out:     device float32 [n_seqs][n_layers][n_q_heads][D]
 * Limits: D in {64, 128, 256}; n_q_heads a multiple of n_kv_heads, at most 8
 * query heads per KV head and n_q_heads * D <= PRCR_DECODE_MAX_Q_ELEMS;
 * n_seqs and n_layers at most 65535 (launch grid limits).
 * workspace: device, >= prcr_decode_workspace_size(...) bytes (0 when the
 * sequence axis is not split), 16-byte aligned. A seq_len beyond the
 * capacity, or above max_len, sets PRCR_ST_CAPACITY (the slots past the
 * capacity, or past the split made for max_len, are left out); an unmapped
 * block in range sets
 * PRCR_ST_NO_BLOCK and its slots are left out of the softmax. A query
 * position of magnitude 2^31 or more sets PRCR_ST_POS_RANGE and the sequence
 * reads no slot. A sequence with seq_len 0 (or no readable slot) gets an
 * output of zeros.                                                         */
#define PRCR_DECODE_MAX_Q_ELEMS 8192
PRCR_API size_t prcr_decode_workspace_size(const prcr_rope_cfg* cfg, int32_t n_seqs,
                                           int32_t n_q_heads, int64_t max_len);
PRCR_API int prcr_decode_attention(const prcr_rope_cfg* cfg, const prcr_cache_desc* cache,
                                   int32_t n_seqs, int32_t n_q_heads, const void* q,
                                   const int64_t* q_pos, const int32_t* seq_len, int64_t max_len,
                                   float* out, uint32_t* status, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* prcr_select_topk - the revisited index set I_tau (Sec. 2.1, Eq. 3) chosen
 * by attention. The paper names an attention-driven selection (it ranks the
 * visual tokens by relevance to the current decoding context and keeps K);
 * its formula is not in the paper. Reading implemented: for sequence b the
 * relevance of visual token m is the trigger query's attention on m at layer
 * `layer`: per query head h, softmax over the store's M tokens of
 * RoPE(q[b][h], (p, p, p)) . RoPE(k_raw[b][layer][m][h / group], p_m) / sqrt(D),
 * p = q_pos[b], averaged over the heads. The rotation is applied as
 * RoPE(q, (p,p,p)) . RoPE(k, c) = q . R(c - p) k, the integer offset c - p
 * reduced modulo one turn in 64-bit integer arithmetic (to 2^-32 of a turn
 * while |c - p| < 2^31; no status word: larger offsets lose accuracy as
 * |c - p| * 2^-65 of a turn). The k most relevant tokens (equal
 * relevance: lower index first) are written in ascending token order as one
 * revisit per sequence, ready for prcr_rebind_inject:
 *   idx_out     device int32 [n_seqs * k]   selected token ids
 *   seq_rev_off device int32 [n_seqs + 1]   b
 *   rev_tok_off device int32 [n_seqs + 1]   b * k
 *   score_out   optional device float32 [n_seqs][n_tokens] relevance
 *   q           device bf16 [n_seqs][n_q_heads][D] raw trigger queries of `layer`
 * Limits: 1 <= k <= n_tokens <= PRCR_SELECT_MAX_TOKENS; n_q_heads a multiple of
 * n_kv_heads, <= 8 per KV head, n_q_heads * D <= PRCR_DECODE_MAX_Q_ELEMS.
 * workspace: device >= prcr_select_workspace_size(...) bytes (the logits).   */
#define PRCR_SELECT_MAX_TOKENS 32768
PRCR_API size_t prcr_select_workspace_size(int32_t n_seqs, int32_t n_q_heads, int32_t n_tokens);
PRCR_API int prcr_select_topk(const prcr_rope_cfg* cfg, const prcr_store_desc* store,
                              int32_t n_seqs, int32_t layer, int32_t n_q_heads, const void* q,
                              const int64_t* q_pos, int32_t k, int32_t* idx_out,
                              int32_t* seq_rev_off, int32_t* rev_tok_off, float* score_out,
                              void* workspace, size_t workspace_bytes, void* stream);

/* prcr_select_topk_cached - the same selection (Sec. 2.1, Eq. 3) read from
 * the decoder's position-bound cache instead of the raw store: the visual
 * tokens' keys there are already rotated at their own coordinates (Eq.
 * "historical_position_bound_kv"; e.g. the cache rows prcr_prefill_capture
 * wrote), so only the trigger query is rotated. Relevance of visual token m
 * of sequence b: per query head h, softmax over the n_tokens tokens of
 *   RoPE(q[b][h], (p, p, p)) . K_cache[b][layer][img_slot0[b] + m][h / group] / sqrt(D),
 * p = q_pos[b], averaged over the heads (with keys rotated exactly this is
 * prcr_select_topk's relevance; the cache's bf16 rounding of the keys is the
 * only difference). Token m is the image's m-th token in the order its rows
 * occupy slots img_slot0[b] .. img_slot0[b] + n_tokens - 1 (contiguous cache,
 * or paged through the block table), the order prcr_prefill_capture and
 * prcr_store_raw give the same token, so idx_out indexes the raw store too.
 *   img_slot0   device int32 [n_seqs]  first cache slot of sequence b's image
 *   status      device uint32 word: a token whose slot lies beyond the
 *               sequence's capacity sets PRCR_ST_CAPACITY, one in an unmapped
 *               block PRCR_ST_NO_BLOCK; such a token gets relevance 0. A query
 *               position of magnitude 2^31 or more sets PRCR_ST_POS_RANGE and
 *               every token of that sequence gets relevance 0. A sequence
 *               whose tokens all have relevance 0 selects its first k tokens
 *               (equal relevance: lower index first)
 * Other arguments, outputs, limits and the workspace (prcr_select_workspace_size
 * with the same n_seqs, n_q_heads, n_tokens) are those of prcr_select_topk;
 * head_dim must be 64, 128 or 256 (PRCR_EINVAL otherwise).               */
PRCR_API int prcr_select_topk_cached(const prcr_rope_cfg* cfg, const prcr_cache_desc* cache,
                                     int32_t n_seqs, int32_t layer, int32_t n_q_heads,
                                     int32_t n_tokens, const int32_t* img_slot0, const void* q,
                                     const int64_t* q_pos, int32_t k, int32_t* idx_out,
                                     int32_t* seq_rev_off, int32_t* rev_tok_off, float* score_out,
                                     uint32_t* status, void* workspace, size_t workspace_bytes,
                                     void* stream);

/* prcr_next_text_pos - host helper: the position the next text token takes
 * after a revisit appended k_seq tokens to a sequence whose latest text token
 * is at p_txt: p_txt + 1 for PCR, ORIGINAL and UIR (Sec. 3.2, Sec. 3.3);
 * p_txt + k_seq + 1 for LPA. Returns INT64_MIN for an unknown mode. */
PRCR_API int64_t prcr_next_text_pos(int64_t p_txt, int64_t k_seq, int32_t mode);

/* Text for a PRCR_E* return code (static string). */
PRCR_API const char* prcr_error_string(int code);

/* PRCR_VERSION of the built library. */
PRCR_API int prcr_version(void);

#ifdef __cplusplus
}
#endif
#endif /* PRCR_H_ */
