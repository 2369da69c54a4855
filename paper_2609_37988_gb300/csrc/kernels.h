// kernels.h -- launch interface between the host library and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvk {

// One GQA anchor as the kernels see it.
struct GqaView {
  uint8_t *rec;        // records base
  float2 *gmeta;       // per-channel key (scale, zero) plane, or null
  uint8_t *resid;      // per-channel key residual plane, or null
  int32_t *lens;       // [B]
  int32_t *counter;    // append completion counter
  int32_t *kept_n;     // [B] (shared by the kv heads) or [B * Hkv] (per head)
  int32_t *kept_idx;   // [B * kept_cap] or [B * Hkv * kept_cap]
  uint32_t *scales;    // symmetric scheme: bf16 (K, V) scale pair per (slab, position)
  int64_t cap;         // positions per slab
  int kept_cap;
  int kept_per_head;   // kept lists per (sequence, kv head) instead of per sequence
  int B, Hkv, D, bits, group, key_axis, rec_bytes;
  int scheme;          // kSchemeGrouped or kSchemeSym
};

struct MlaView {
  uint8_t *rec;        // [B][cap][(width + rope) bf16], or quantised codes (layout.h)
  uint8_t *meta;       // quantised: per-position scales (and zeros) plane, else null
  int32_t *lens;
  int32_t *counter;
  int64_t cap;
  int B, width, rope, rec_bytes;
  int bits;            // 16, or 8 / 4 / 2 for quantised latents
  int scheme;          // kSchemeGrouped or kSchemeSym (quantised latents)
  // 0: decode, one query row per sequence.  n > 0: pre-fill, n query rows
  // per sequence: row b n + i is query i of sequence b, at position
  // lens[b] - n + i, attending to positions 0 .. itself
  int n_q = 0;
};
// query rows of an MLA launch, and for row vb its sequence and the positions it reads
__host__ __device__ __forceinline__ int mla_rows(const MlaView &v) { return v.n_q ? v.B * v.n_q : v.B; }
__device__ __forceinline__ int mla_row_seq(const MlaView &v, int vb) { return v.n_q ? vb / v.n_q : vb; }
__device__ __forceinline__ int mla_row_len(const MlaView &v, int vb, int b) {
  const int L = v.lens[b];
  return v.n_q ? max(0, min(L, L - v.n_q + (vb - b * v.n_q) + 1)) : L;
}

struct GqaDecodeArgs {
  GqaView v;
  const void *q;       // [B, Hq, D]
  int q_f32;           // 1: q is float32, 0: bf16
  int Hq, G;
  float sig_log2;      // softmax scale * log2(e)
  int n_splits;
  int items_per_split; // multiple of kTile
  int gather;          // read the kept list
  float *partial;      // [n_splits, B*Hq, D+2], written when out is null
  float *out;          // [B, Hq, D]: normalised output (single split)
  int32_t *err;
  uint32_t wait_limit = 1u << 22;  // polls of a bounded wait on this CTA's copies before it gives up
  // host copy of the anchor's record-table tensor map (gqa_make_rows_tmap),
  // required by the kept-list gather of grouped per-token records
  const void *rows = nullptr;
  // run schedule (quantised formats with per-token keys or the symmetric
  // scheme, contiguous reads, partials only): run_ctas > 0 CTAs take equal
  // runs of the (unit, tile) grid of run_tpu kernel tiles per unit, into
  // run_slots partial slots per unit; 0 = the (split, kv head, sequence) grid.
  // run_tpu counts run_setup planned tiles per unit for its start-up cost
  // before its data tiles; run_q, run_r: the planned tile count W = B Hkv
  // run_tpu as q run_ctas + r.
  int run_ctas = 0, run_tpu = 0, run_slots = 0, run_q = 0, run_r = 0, run_setup = 0;
};

// Returns cudaSuccess or the launch error.  Template dispatch on
// (bits, D, key axis, q dtype) happens inside.
cudaError_t launch_gqa_decode(const GqaDecodeArgs &a, cudaStream_t st);
int gqa_decode_ctas_per_sm(int bits, int D, int key_axis, int group, int scheme);
int gqa_decode_tile(int bits, int D, int key_axis, int group, int scheme);
// Whether the format's kept-list gather copies records by tensor-map rows,
// and the 128-byte tensor map of an anchor's record table for it: rows
// slab * cap + position, one record per row (B * Hkv * cap < 2^31).
bool gqa_decode_row_gather(int bits, int key_axis, int scheme);
cudaError_t gqa_make_rows_tmap(void *out, const GqaView &v);

// cuTensorMapEncodeTiled reached through the runtime's driver entry point
// (no link against the driver library); arguments in the driver's order,
// enums as their integer values.  cudaErrorInvalidValue if it refuses.
cudaError_t encode_tensor_map_tiled(void *map, int dtype, int rank, void *base,
                                    const uint64_t *dims, const uint64_t *strides,
                                    const uint32_t *box, const uint32_t *elem_strides,
                                    int interleave, int swizzle, int l2_promotion, int oob_fill);

struct RewindArgs {
  int32_t *lens[64];
  int n_anchors, B, n;
};
cudaError_t launch_rewind(const RewindArgs &a, cudaStream_t st);

cudaError_t launch_splitk_merge(const float *partials, int n_splits, int n_rows, int dim,
                                float *out, cudaStream_t st);

// Append n_new rows per sequence (per-sequence counts optional).
cudaError_t launch_gqa_append(const GqaView &v, const void *k, const void *vv, int in_f32,
                              int n_new, const int32_t *n_per_seq, int32_t *err,
                              cudaStream_t st);
cudaError_t launch_mla_append(const MlaView &v, const void *c, const void *kr, int latent,
                              int n_new, const int32_t *n_per_seq, int32_t *err,
                              cudaStream_t st);

// Window-vote eviction of one GQA anchor (evict.cu): votes of the positions
// before the last n_win, top budget - n_win of them and the window written
// as per-(sequence, kv head) kept lists into the anchor's arena.  scratch:
// float votes [B * Hkv * cap] then float2 row statistics
// [B * Hkv * rows * tiles] with rows = n_win * G, tiles = cap / 128.
struct EvictArgs {
  GqaView v;
  const void *q;       // [B, n_win, Hq, D]
  int q_f32;
  int Hq, G, n_win, budget;
  float sig_log2;      // softmax scale * log2(e)
  int n_tiles;         // 128-position tiles launched per (sequence, kv head)
  int sc_stride;       // n_tiles * kEvictTile: row stride of the scores
  int stat_sub;        // statistics entries per tile and row (1 or kEvictStatSub)
  float *votes;        // [B * Hkv][cap]
  float2 *stats;       // [B * Hkv][R][n_tiles * stat_sub] per-tile (max, sum)
  float2 *fin;         // [B * Hkv][R] merged (max, sum)
  float *scores;       // [B * Hkv][R][sc_stride] scaled scores (log2 domain)
  int32_t *err;
};
cudaError_t launch_gqa_evict(const EvictArgs &a, cudaStream_t st);

// Causal chunk attention (prefill) over a GQA anchor, head_dim 128.
struct PfArgs {
  GqaView v;
  const void *q;       // [B, n_q, Hq, D]
  int q_f32;
  int Hq, G, n_q;
  float sig_log2;      // softmax scale * log2(e)
  float *out;          // [B, n_q, Hq, D]
  int *counter;        // the job counter, zeroed by the launch
  uint8_t *tiles;      // [B * Hkv][cap / 64] expanded tiles of prefill_tile_bytes(bits)
  int32_t *err;
};
cudaError_t launch_gqa_prefill(const PfArgs &a, cudaStream_t st);
bool prefill_plan_fits(const PfArgs &a);
size_t prefill_tile_bytes(int bits);
constexpr int kEvictTile = 128;
constexpr int kEvictStatSub = 4;  // statistics entries per tile and row, at most
// Whether the evictor scores on the tensor cores (head_dim 128, at most 256
// window query rows per KV head); otherwise it scores on the CUDA cores and
// stores the scores.
inline bool evict_uses_tc(int D, int R) { return D == 128 && R >= 1 && R <= 256; }

cudaError_t launch_gqa_export(const GqaView &v, void *k_out, void *v_out, float *k_scale,
                              float *k_zero, float *v_scale, float *v_zero, void *k_resid,
                              int max_ctx, cudaStream_t st);
cudaError_t launch_mla_export(const MlaView &v, void *c_out, void *kr_out, float *c_scale,
                              float *c_zero, float *kr_scale, float *kr_zero, int max_ctx,
                              cudaStream_t st);

struct MlaDecodeArgs {
  MlaView v;
  const void *q_nope;  // bf16 [B, H, Dn]
  const void *q_pe;    // bf16 [B, H, rope]
  const void *w_uk;    // bf16 [H, Dn, r]
  const void *w_uv;    // bf16 [H, Dv, r]
  int H, Dn, r;
  float sig_log2;
  int n_splits, items_per_split;
  uint16_t *qlat;      // workspace bf16 [B, H, 2*width + rope] (hi | lo | pe)
  float *partial;      // [n_splits, B*H, width+2]
  float *olat;         // [B, H, width]
  float *out;          // [B, H, Dv]
  int32_t *err;
  const void *tmap;    // host copy of the anchor's 128-byte tensor map (mla_make_tmap)
  uint32_t wait_limit = 1u << 22;  // polls of a bounded wait in the tile loop before it gives up
};
cudaError_t launch_mla_decode(const MlaDecodeArgs &a, cudaStream_t st);
// the same for an anchor of quantised latents (mla_q.cu; one CTA per SM)
cudaError_t launch_mla_decode_q(const MlaDecodeArgs &a, cudaStream_t st);
// Encodes the decode kernel's tensor map of an MLA anchor into `out` (128
// bytes, 64-byte aligned).
cudaError_t mla_make_tmap(void *out, const MlaView &v);
int mla_decode_ctas_per_sm(int width, int bits = 16);

}  // namespace kvk
