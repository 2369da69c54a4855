/*
 * kvk.h -- C ABI of the GB300-native compressed-KV decode path.
 *
 * The library implements the per-step decode attention that reads a
 * per-layer compressed KV cache, and the append that writes new tokens into
 * it, for the per-layer cache plans of KV-Kaizen (arxiv 2609.37988):
 *
 *   depth      a layer owns a cache (an "anchor") or inherits the nearest
 *              anchor before it and reads it with its own query (Sec. 2.1);
 *   precision  a cache is stored at 16, 8, 4 or 2 bits (Sec. 2.1) with
 *              either quantiser of Appendix C.3: the grouped asymmetric one
 *              (a scale and a zero point per group of channels or
 *              positions) or the paper's symmetric per-vector one (one bf16
 *              scale per token-head row, codes in [-q, q], q = 2^(b-1) - 1);
 *   rank       an MLA latent truncated to its first d coordinates plus the
 *              post-RoPE positional key (Sec. 2.1, Appendix C.2).
 *
 * A plan (one action per layer, eq. (cost)-(action space) in Sec. 2.2) is
 * fixed for the whole generation (Sec. 2.3), so the cache is laid out once.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Ownership: the caller owns every device buffer (arenas, workspace,
 *    inputs, outputs).  The library owns only its host-side cache object.
 *    No entry point allocates device memory.
 *  - Asynchrony: device work is enqueued on the caller's stream and is never
 *    synchronised, except by kvk_get_device_error.
 *  - Validation: arguments are checked on the host before anything is
 *    enqueued; a failed check returns an error status and enqueues nothing.
 *    Device-side bounds violations (for example a kept position past the
 *    sequence length) set a device error word, skip the offending access and
 *    let the kernel finish; they never trap.
 *  - kvk_last_error() returns a thread-local, human-readable message for the
 *    last non-OK status returned on the calling thread.
 *  - Pointers marked "device" must be device-accessible and 16-byte aligned.
 *  - Layer indices are 0-based.
 */
#ifndef KVK_H
#define KVK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same handle as cudaStream_t; declared opaquely so this header needs no
 * CUDA include.  NULL is the legacy default stream. */
typedef struct CUstream_st *kvk_stream;

typedef enum {
  KVK_OK = 0,
  KVK_ERR_INVALID_ARG = 1,     /* null pointer, bad size, misaligned buffer  */
  KVK_ERR_INVALID_CONFIG = 2,  /* plan rejected (e.g. layer 0 inherits)      */
  KVK_ERR_INHERITED_LAYER = 3, /* write to a layer that owns no cache        */
  KVK_ERR_CAPACITY = 4,        /* append would pass max_ctx, or a noalloc
                                  decode needs more partials than its fixed
                                  buffer holds                               */
  KVK_ERR_UNSUPPORTED = 5,     /* valid request this library does not handle */
  KVK_ERR_CUDA = 6,            /* a CUDA runtime call failed                 */
  KVK_ERR_DEVICE = 7           /* the device error word was set              */
} kvk_status;

enum { KVK_KIND_GQA = 0, KVK_KIND_MLA = 1 };
enum { KVK_AXIS_TOKEN = 0, KVK_AXIS_CHANNEL = 1 };
enum { KVK_QUANT_GROUPED = 0, KVK_QUANT_SYMMETRIC = 1 };
enum { KVK_DTYPE_F32 = 0, KVK_DTYPE_BF16 = 1 };

/* Device error word values (kvk_get_device_error). */
enum {
  KVK_DEVERR_NONE = 0,
  KVK_DEVERR_KEPT_RANGE = 1,   /* kept position >= sequence length           */
  KVK_DEVERR_CAPACITY = 2,     /* append position >= capacity                */
  KVK_DEVERR_COUNT = 4,        /* per-sequence append count out of range     */
  KVK_DEVERR_TIMEOUT = 8,      /* a bounded wait on an async copy gave up    */
  KVK_DEVERR_ALIGN = 16        /* shared memory not aligned for a copy; the  */
                               /* call computed nothing                      */
};

/* Model geometry.  GQA: n_q_heads query heads, n_kv_heads KV heads of
 * head_dim (Sec. 2.1, Tab. backbones).  MLA: latent width latent_dim (r),
 * positional key rope_dim (d_R), content/value head width head_dim,
 * n_q_heads heads sharing one latent (Appendix B, C.2). */
typedef struct {
  int32_t kind;        /* KVK_KIND_GQA or KVK_KIND_MLA                      */
  int32_t n_layers;    /* L                                                 */
  int32_t n_q_heads;   /* H_q                                               */
  int32_t n_kv_heads;  /* H_kv (GQA); ignored for MLA                       */
  int32_t head_dim;    /* d_h: 64 or 128 (GQA); 128 (MLA content/value)     */
  int32_t latent_dim;  /* r (MLA); ignored for GQA                          */
  int32_t rope_dim;    /* d_R (MLA, 64); ignored for GQA                    */
  int32_t max_batch;   /* sequences per cache                               */
  int32_t max_ctx;     /* positions per sequence                            */
} kvk_model_desc;

/* One plan action (Sec. 2.2).  inherit=1 is the depth action; otherwise the
 * layer owns a cache at `bits` (16 = bf16; 8, 4 or 2 = quantised codes) and,
 * for MLA, keeps the first `width` latent coordinates (truncate on write,
 * Appendix C.2).
 *  scheme KVK_QUANT_GROUPED: `group` elements per fp32 (scale, zero) pair;
 *    key_axis selects per-token groups (g channels of one token) or
 *    per-channel groups (g positions of one channel, KIVI keys); values are
 *    per-token.  This library: bits 8 or 4, group 32 or 64.
 *  scheme KVK_QUANT_SYMMETRIC: the paper's quantiser (Appendix C.3): one
 *    bf16 scale s = max|x| / q per token-head row of keys and of values,
 *    codes clip(rint(x / s), -q, q) with q = 2^(b-1) - 1 (three levels at
 *    two bits), x = code * s; `group` is ignored and both axes must be
 *    KVK_AXIS_TOKEN.  This library: GQA, head_dim 128, bits 8, 4 or 2.
 *  MLA layers at 8, 4 or 2 bits (all three axes at once): each position's
 *    kept latent c[:width] and its positional key k^R are each quantised as
 *    ONE vector, with one bf16 scale (symmetric; 8/4/2 bits) or one fp32
 *    (scale, zero) pair (grouped, the group spanning the vector; 8/4 bits);
 *    `group` and the axes are ignored.  Decode feeds the codes to the
 *    tensor cores as exact f16 values with the value weights p * s rounded
 *    to f16 hi + lo, so p * s (p <= 256) must stay below 65504: latent
 *    scales below 255.
 * evict_capacity > 0 reserves a kept-position list of that length per
 * sequence (eviction composed with compression, Sec. 3.4). */
typedef struct {
  int32_t inherit;
  int32_t bits;
  int32_t group;
  int32_t key_axis;
  int32_t value_axis;
  int32_t width;
  int32_t evict_capacity;
  int32_t scheme;      /* KVK_QUANT_GROUPED or KVK_QUANT_SYMMETRIC */
} kvk_layer_cfg;

typedef struct kvk_cache kvk_cache;

/* Validate a plan and report the device bytes each layer's arena needs
 * (0 for inheritors).  arena_bytes: host array of n_layers entries.
 * Errors: INVALID_ARG, INVALID_CONFIG (layer 0 inherits, bits not in
 * {16,8,4,2}, unknown scheme, group not dividing head_dim for the grouped
 * scheme, a per-channel axis with the symmetric scheme, MLA width not in
 * r/8..r), and UNSUPPORTED for valid plans outside this library (grouped 2-bit
 * codes, per-channel values, head_dim other than 64/128, the symmetric
 * scheme with GQA head_dim 64, per-channel keys with eviction). */
kvk_status kvk_cache_plan(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                          size_t *arena_bytes);

/* Device workspace bytes for a cache whose decode calls use at most
 * max_splits context splits.  Holds the device error word, split-K partials,
 * and the absorbed MLA query. */
kvk_status kvk_workspace_size(const kvk_model_desc *desc, int32_t max_splits,
                              size_t *ws_bytes);

/* Create a cache over caller-allocated arenas.  arenas: host array of
 * n_layers device pointers (NULL for inheritors), each of at least the size
 * kvk_cache_plan reported; workspace: device buffer of ws_bytes.  The cache
 * starts empty; call kvk_cache_reset (or zero the arenas) before first use.
 * The cache keeps the pointers; the caller keeps the memory alive.
 * INVALID_CONFIG also when a grouped 8- or 4-bit anchor with per-token keys
 * and evict_capacity > 0 holds max_batch x n_kv_heads x capacity >= 2^31
 * records (its kept-list gather addresses records as 31-bit rows). */
kvk_status kvk_cache_create(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                            void *const *arenas, void *workspace, size_t ws_bytes,
                            int32_t max_splits, kvk_cache **out);
kvk_status kvk_cache_destroy(kvk_cache *cache);

/* Zero every sequence length, kept list, merge counter and the device error
 * word, on `stream`. */
kvk_status kvk_cache_reset(kvk_cache *cache, kvk_stream stream);

/* src[layer]: nearest anchor at or before `layer` (Sec. 2.1). */
kvk_status kvk_layer_source(const kvk_cache *cache, int32_t layer, int32_t *src);

/* Device pointer to the int32[max_batch] sequence lengths of the anchor that
 * `layer` reads (advanced by kvk_append). */
kvk_status kvk_layer_lengths(const kvk_cache *cache, int32_t layer,
                             const int32_t **lens_device);

/* Append n_new positions to every sequence of anchor `layer`: quantise (or
 * truncate, for MLA) on write.
 *  GQA: k, v device [B, n_new, H_kv, head_dim] in in_dtype (F32 or BF16).
 *       Per-token groups are quantised immediately; per-channel key groups
 *       are buffered in bf16 until g positions of a group exist, then
 *       quantised along the positions (KIVI keys, Appendix C.3).
 *  MLA: k = latent c device [B, n_new, latent_dim] BF16 (only the first
 *       `width` coordinates are stored, Appendix C.2), v = positional key
 *       k^R device [B, n_new, rope_dim] BF16, post-RoPE.
 *  B = max_batch.  n_new_per_seq: optional device int32[B]; sequence b then
 *  appends only its first n_new_per_seq[b] <= n_new rows (ragged lengths).
 * Errors: INHERITED_LAYER, CAPACITY (host-side bound on the lengths),
 * INVALID_ARG. */
kvk_status kvk_append(kvk_cache *cache, int32_t layer, const void *k, const void *v,
                      int32_t in_dtype, int32_t n_new, const int32_t *n_new_per_seq,
                      kvk_stream stream);

/* Roll back the last n positions of every sequence of every anchor (for
 * example a rejected speculative step), in one launch on `stream`: each
 * length becomes max(0, length - n).  Caches with per-channel key groups
 * return UNSUPPORTED (a quantised group cannot be re-opened). */
kvk_status kvk_rewind(kvk_cache *cache, int32_t n, kvk_stream stream);

/* The split count kvk_decode_attention / kvk_decode_attention_mla would use
 * for `layer` with n_splits = 0 (host only; depends on the host-side bound
 * on the anchor's lengths, the SM count and the decode schedule).  Under the
 * run schedule (kvk_set_decode_schedule) it is the number of partial slots
 * per (sequence, KV head) that kvk_decode_partial with n_splits = 0 writes. */
kvk_status kvk_decode_plan_splits(kvk_cache *cache, int32_t layer, int32_t *n_splits);

/* Install the kept-position list of anchor `layer` (eviction, Sec. 3.4):
 * idx device int32 [B, evict_capacity] sorted ascending, n_kept device
 * int32[B] <= evict_capacity.  Decode then reads only those positions; an
 * entry past the sequence length sets KVK_DEVERR_KEPT_RANGE and is skipped.
 * The list is shared by the sequence's KV heads (kvk_evict_window installs
 * per-head lists).  n_kept == NULL clears the lists (all positions are read
 * again). */
kvk_status kvk_set_kept(kvk_cache *cache, int32_t layer, const int32_t *idx,
                        const int32_t *n_kept, kvk_stream stream);

/* Attention-scored eviction composed with the compressed cache (Sec. 3.4;
 * the paper's evictors sum attention over a 32-query observation window).
 * For every sequence b and KV head j of anchor `layer`, each position t
 * before the last n_win gets the attention mass that the window's queries of
 * the heads of j put on it,
 *   vote[b,j,t] = sum_{w < n_win} sum_{h in group j}
 *                 softmax_{u <= p_w}(softmax_scale <q[b,w,h], k_u>)[t],
 * p_w = len_b - n_win + w (window query w sits at position p_w and sees the
 * positions up to itself; keys dequantised from the cache).  The budget -
 * n_win largest votes (equal votes: the smaller position first) and the
 * window become the kept list of (b, j), sorted; a sequence of at most
 * `budget` positions keeps all of them.  The lists are installed as the
 * anchor's kept lists, one per (sequence, KV head): decode then reads, for
 * KV head j of sequence b, only its own list, until kvk_set_kept replaces or
 * clears it.
 *  q_win:   device [B, n_win, H_q, head_dim] in q_dtype, post-RoPE, the
 *           queries of each sequence's last n_win positions; 1 <= n_win <= 256;
 *  budget:  n_win <= budget <= evict_capacity;
 *  scratch: device, 256-byte aligned, at least kvk_evict_scratch_size bytes.
 *           Once the stream reaches the end of the call it starts with the
 *           votes: float32 vote[b,j,t] at index (b H_kv + j) C + t, C =
 *           max_ctx rounded up to a multiple of 64, for t < len_b - n_win of
 *           the sequences longer than `budget` (the rest unspecified).
 * Errors: INHERITED_LAYER (evict on the anchor), INVALID_CONFIG
 * (evict_capacity 0), UNSUPPORTED (MLA, grouped per-channel keys),
 * INVALID_ARG. */
kvk_status kvk_evict_scratch_size(const kvk_cache *cache, int32_t layer, int32_t n_win,
                                  size_t *scratch_bytes);
kvk_status kvk_evict_window(kvk_cache *cache, int32_t layer, const void *q_win, int32_t q_dtype,
                            int32_t n_win, float softmax_scale, int32_t budget, void *scratch,
                            size_t scratch_bytes, kvk_stream stream);

/* Causal chunk attention (pre-fill) of `layer` over its compressed cache
 * (Sec. 4 times pre-fill over compressed caches): the chunk is the last n_q
 * positions of every sequence, already written with kvk_append; query i of
 * sequence b sits at position len_b - n_q + i and attends to positions
 * 0 .. len_b - n_q + i of the dequantised stored keys and values (the ones
 * decode reads), with its own query heads (an inheriting layer reads its
 * anchor).  Queries before position 0 (len_b < n_q) give zeros.  Kept lists
 * are not used: pre-fill reads every position.  Keys with per-channel groups
 * are read as decode reads them: complete groups of positions from their
 * codes and the group plane, the open group from the bf16 residual.
 *  q:       device [B, n_q, H_q, head_dim] in q_dtype (post-RoPE),
 *           16-byte aligned;
 *  out:     device float32 [B, n_q, H_q, head_dim], 16-byte aligned;
 *  scratch: device, 256-byte aligned, at least kvk_prefill_scratch_size
 *           bytes: the anchor's cache dequantised once into the products'
 *           operand layout (1 KB per position and KV head for quantised
 *           anchors, 512 B for bf16) and a job counter.
 * Errors: UNSUPPORTED (MLA: see kvk_prefill_attention_mla; head_dim != 128),
 * INVALID_ARG (n_q outside [1, max_ctx], null or misaligned pointers,
 * scale not finite and positive, scratch too small). */
kvk_status kvk_prefill_scratch_size(const kvk_cache *cache, int32_t layer, int32_t n_q,
                                    size_t *scratch_bytes);
kvk_status kvk_prefill_attention(kvk_cache *cache, int32_t layer, const void *q, int32_t q_dtype,
                                 int32_t n_q, float softmax_scale, float *out, void *scratch,
                                 size_t scratch_bytes, kvk_stream stream);

/* Causal chunk attention (pre-fill) of MLA layer `layer` over its latent
 * cache (bf16 or quantised, at its kept width d): the chunk is the last n_q
 * positions of every sequence, already written with kvk_append; query i of
 * sequence b, at position len_b - n_q + i, attends to positions 0 .. itself
 * with the absorbed query of each head (Appendix C.2, as
 * kvk_decode_attention_mla: q_lat = W_UK[h][:, :d]^T q_nope, scores
 * sigma (q_lat . c[:d] + q_pe . k^R), output W_UV[h][:, :d] o_lat).  Each
 * query row runs the decode path over its own causal prefix (one CTA per
 * row, or per pair of consecutive rows of a sequence for bf16 latents of
 * width >= 256 when n_q is even).  Queries before position 0 give zeros.
 *  q_nope:  device bf16 [B, n_q, H, head_dim]; q_pe: bf16 [B, n_q, H, rope]
 *           (post-RoPE);
 *  w_uk, w_uv: device bf16 [H, head_dim, latent] as for decode;
 *  out:     device float32 [B, n_q, H, head_dim];
 *  scratch: device, 256-byte aligned, at least kvk_prefill_scratch_size
 *           bytes (which answers for MLA layers too): the rows' absorbed
 *           queries and latent partials;
 * all 16-byte aligned.  Errors: INVALID_ARG (not an MLA cache, n_q outside
 * [1, max_ctx], null or misaligned pointers, scale not finite and positive,
 * scratch too small). */
kvk_status kvk_prefill_attention_mla(kvk_cache *cache, int32_t layer, const void *q_nope,
                                     const void *q_pe, const void *w_uk, const void *w_uv,
                                     int32_t n_q, float softmax_scale, float *out, void *scratch,
                                     size_t scratch_bytes, kvk_stream stream);

/* Copy anchor `layer`'s kept lists out, device to device, on `stream`.
 * *per_head (host) = -1: no list installed (nothing copied); 0: lists per
 * sequence, idx [B, evict_capacity], n_kept [B]; 1: lists per (sequence, KV
 * head), idx [B, H_kv, evict_capacity], n_kept [B, H_kv].  idx and n_kept
 * are device buffers of at least the per-head sizes. */
kvk_status kvk_export_kept(const kvk_cache *cache, int32_t layer, int32_t *idx, int32_t *n_kept,
                           int32_t *per_head, kvk_stream stream);

/* GQA decode attention of `layer` with its own query (inheritors read their
 * source anchor, Sec. 2.1):
 *   out[b,h,:] = sum_t softmax_t(scale * <q[b,h], k_t>) v_t
 * over the positions of sequence b (or its kept list), KV head h / G with
 * G = H_q / H_kv.  q: device [B, H_q, head_dim] in q_dtype; out: device
 * float [B, H_q, head_dim].  softmax_scale: finite and > 0, else
 * KVK_ERR_INVALID_ARG.  n_splits: context splits (0 = chosen from the SM
 * count), at most the max_splits given at creation. */
kvk_status kvk_decode_attention(kvk_cache *cache, int32_t layer, const void *q,
                                int32_t q_dtype, float softmax_scale, float *out,
                                int32_t n_splits, kvk_stream stream);

/* MLA decode attention of `layer` in the absorbed form (Appendix C.2):
 *   q_lat[b,h] = W_UK[h][:, :d]^T q_nope[b,h]
 *   s_t       = scale * (<q_lat, c_t[:d]> + <q_pe, k^R_t>)
 *   out[b,h]  = W_UV[h][:, :d] sum_t softmax_t(s_t) c_t[:d]
 * q_nope device bf16 [B, H, head_dim]; q_pe device bf16 [B, H, rope_dim]
 * (post-RoPE); w_uk, w_uv device bf16 [H, head_dim, latent_dim]; out device
 * float [B, H, head_dim].  softmax_scale: finite and > 0. */
kvk_status kvk_decode_attention_mla(kvk_cache *cache, int32_t layer, const void *q_nope,
                                    const void *q_pe, const void *w_uk, const void *w_uv,
                                    float softmax_scale, float *out, int32_t n_splits,
                                    kvk_stream stream);

/* Split-K pieces of kvk_decode_attention (the seam a context-parallel
 * multi-GPU variant would all-gather across).  kvk_decode_partial writes
 * partials device float [n_splits, B*H_q, head_dim + 2]: per row the
 * unnormalised accumulator sum_t 2^(x_t - m) v_t (head_dim floats), then m,
 * then l = sum_t 2^(x_t - m), with x_t = scale * log2(e) * <q, k_t>.  A split
 * that reads no position stores m = -inf, l = 0.  n_splits >= 2: equal
 * contiguous context splits.  n_splits = 0: the automatic schedule, with
 * kvk_decode_plan_splits slots; under the run schedule each slot holds one
 * piece of a partition of the positions (not an equal split), and merging
 * all slots with kvk_splitk_reduce gives the attention output. */
kvk_status kvk_decode_partial(kvk_cache *cache, int32_t layer, const void *q,
                              int32_t q_dtype, float softmax_scale, float *partials,
                              int32_t n_splits, kvk_stream stream);

/* Decode attention exactly like kvk_decode_attention, for callers that
 * cannot provide scratch device memory: for example a process whose device
 * memory belongs to another allocator or is planned to a fixed budget, which
 * may not call cudaMalloc to size a workspace for its largest split count.
 * (The paper has no counterpart; this is a deployment convenience.)
 *  - Allocates nothing and calls no allocating routine.  The split-K
 *    partials go to one fixed buffer of 16 MiB (4,194,304 floats) compiled
 *    into the library; every GPU that loads the library holds that buffer
 *    until the process exits.
 *  - The partials take S * max_batch * n_q_heads * (head_dim + 2) floats,
 *    where S is the split count the call actually uses: n_splits capped at
 *    the number of 64-position tiles of the context, or with n_splits = 0
 *    the automatic plan's count (kvk_decode_plan_splits: the split count, or
 *    under the run schedule the partial slots per (sequence, KV head)); a
 *    call that resolves to one split of the split grid writes its output
 *    directly and needs no partials.  A call needing more
 *    than 4,194,304 floats returns KVK_ERR_CAPACITY and enqueues nothing;
 *    pass fewer splits or use kvk_decode_attention.
 *  - The cache's device must be the current device (the buffer is per
 *    device); otherwise KVK_ERR_INVALID_ARG and nothing is enqueued.
 *  - All calls on a device share the buffer, and it keeps the last call's
 *    contents.  Each call writes every partial it later reads, so nothing
 *    needs clearing, but calls that overlap on the GPU (different streams,
 *    or different caches at once) race on it: order them.
 *  - The first call on each device looks up the buffer's device address
 *    (with that device current); make that first call before any stream
 *    capture.
 * Arguments, layouts and other errors as kvk_decode_attention. */
kvk_status kvk_decode_attention_noalloc(kvk_cache *cache, int32_t layer, const void *q,
                                        int32_t q_dtype, float softmax_scale, float *out,
                                        int32_t n_splits, kvk_stream stream);

/* Merge split partials in the format above:
 *   out[row] = sum_s 2^(m_s - M) acc_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s.
 * partials device float [n_splits, n_rows, dim + 2]; out device float
 * [n_rows, dim].  Rows where every split is empty are written as zeros. */
kvk_status kvk_splitk_reduce(const float *partials, int32_t n_splits, int32_t n_rows,
                             int32_t dim, float *out, kvk_stream stream);

/* Cost accounting of the cache's plan.
 *  bits_per_token_model: sum over layers of eq. (cost), in bits per token;
 *  bytes_per_token_stored: bytes this library stores per token, summed over
 *      anchors, including the quantisers' metadata (fp32 scale/zero pairs,
 *      or two bf16 scales per row for the symmetric scheme; Tab. realized_bits
 *      counts metadata the same way);
 *  rho: eq. (compression) against the bf16 GQA cache of the same geometry
 *      (for MLA, n_kv_heads * head_dim = latent_dim is used as C0's width,
 *      the conversion rule r = n_kv d_h of Appendix B). */
kvk_status kvk_cost(const kvk_cache *cache, double *bits_per_token_model,
                    double *bytes_per_token_stored, double *rho);

/* The same accounting for a plan before any cache exists (host only, no
 * device call).  Validates the plan like kvk_cache_plan. */
kvk_status kvk_plan_cost(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                         double *bits_per_token_model, double *bytes_per_token_stored,
                         double *rho);

/* Copy anchor `layer`'s stored state out in canonical (unpermuted) form,
 * device to device, on `stream`.  Positions past a sequence's length hold
 * unspecified values.  Shapes (B = max_batch, T = max_ctx, D = head_dim):
 *  bf16 GQA:   k_out, v_out bf16 [B, H_kv, T, D]; the rest unused.
 *  quantised:  k_out, v_out uint8 codes [B, H_kv, T, D] (one code per byte);
 *              v_scale, v_zero float [B, H_kv, T, D/g];
 *              per-token keys: k_scale, k_zero float [B, H_kv, T, D/g];
 *              per-channel keys: k_scale, k_zero float [B, H_kv, T/g, D] and
 *              k_residual bf16 [B, H_kv, g, D] (positions of the open group,
 *              row = position mod g).
 *  symmetric:  k_out, v_out int8 codes in [-q, q] [B, H_kv, T, D];
 *              k_scale, v_scale float [B, H_kv, T] (the stored bf16 scales,
 *              widened); k_zero, v_zero, k_residual unused.
 *  MLA:        k_out bf16 [B, T, width] latent, v_out bf16 [B, T, rope_dim].
 *  quantised MLA: k_out, v_out codes [B, T, width] (latent) and
 *              [B, T, rope_dim] (k^R), one byte each (int8 in [-q, q] for
 *              the symmetric scheme, uint8 for the grouped one); k_scale,
 *              k_zero float [B, T] of the latent vectors, v_scale, v_zero of
 *              the k^R vectors (zeros 0 for the symmetric scheme).
 * Any pointer the format does not use may be NULL. */
kvk_status kvk_export_layer(const kvk_cache *cache, int32_t layer, void *k_out, void *v_out,
                            float *k_scale, float *k_zero, float *v_scale, float *v_zero,
                            void *k_residual, kvk_stream stream);

/* Number of polls a decode kernel's bounded wait on its own asynchronous
 * copies makes, inside the tile loop, before it gives up
 * (kvk_decode_attention, kvk_decode_partial, the no-alloc decode and the
 * MLA decode of quantised latents).  KVK_WAIT_LIMIT_DEFAULT unless changed
 * here; the setting applies to the calls enqueued after it.  A wait that
 * gives up makes its CTA stop consuming tiles, let the copies it has in
 * flight land (with a limit of its own), set KVK_DEVERR_TIMEOUT and return;
 * the outputs of that call are unspecified and later calls are unaffected.
 * 0 makes every such wait give up at its first poll: a way to exercise that
 * path without a fault.  Errors: KVK_ERR_INVALID_ARG for a null cache. */
#define KVK_WAIT_LIMIT_DEFAULT 4194304u
kvk_status kvk_set_wait_limit(kvk_cache *cache, uint32_t polls);

/* How an automatic GQA decode (n_splits = 0) partitions the work over CTAs
 * (a scheduling choice; the paper's method is the same either way):
 *  KVK_SCHEDULE_SPLITS: a grid of (context split, KV head, sequence), every
 *      split the same number of positions;
 *  KVK_SCHEDULE_RUNS: one or a few whole waves of resident CTAs, each taking
 *      an equal run of the flattened (sequence, KV head, tile) grid, a run
 *      meeting at most two (sequence, KV head) units; quantised anchors with
 *      per-token keys or the symmetric scheme read without a kept list
 *      (other anchors use the splits);
 *  KVK_SCHEDULE_AUTO (default): the runs where the split grid would give
 *      each CTA at most 13 tiles and leave its last wave of CTAs less than
 *      90 % full (and every run CTA gets at least four tiles), else the
 *      splits.
 * run_ctas: the number of run CTAs (clamped to [units, tiles], units = B *
 * H_kv, tiles of 64 or 128 positions per unit); 0 = the fewest whole waves
 * of resident CTAs that are at least the units.  run_setup: planned tiles
 * charged to each unit's start (query set-up, first copies, epilogue) in
 * the partition, so that runs that start a second unit carry fewer data
 * tiles; -1 = the library's default, else 0..64.
 * Results agree to rounding (the merge order of partial sums differs).
 * Applies to calls enqueued after it.  Errors: INVALID_ARG for a null cache,
 * an unknown schedule, run_ctas < 0 or run_setup outside [-1, 64]. */
#define KVK_SCHEDULE_AUTO 0
#define KVK_SCHEDULE_SPLITS 1
#define KVK_SCHEDULE_RUNS 2
kvk_status kvk_set_decode_schedule(kvk_cache *cache, int32_t schedule, int32_t run_ctas,
                                   int32_t run_setup);

/* Synchronise `stream`, read the device error word into *code and clear it.
 * Returns KVK_ERR_DEVICE if the word was non-zero.  After a
 * KVK_DEVERR_TIMEOUT the outputs of the affected calls are unspecified. */
kvk_status kvk_get_device_error(kvk_cache *cache, kvk_stream stream, int32_t *code);

const char *kvk_status_string(kvk_status s);
const char *kvk_last_error(void);

/* Library version string ("kvk <major>.<minor> sm_103a"). */
const char *kvk_version(void);

#ifdef __cplusplus
}
#endif
#endif /* KVK_H */
