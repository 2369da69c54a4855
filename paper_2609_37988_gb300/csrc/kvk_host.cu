// kvk_host.cu -- host side of the C ABI declared in include/kvk.h.
//
// Validates plans (Sec. 2.2: one action per layer, layer 0 owns a cache),
// resolves every layer's source anchor (Sec. 2.1: nearest anchor at or
// before it), plans arena layouts, chooses split counts and launches the
// kernels on the caller's stream.  It never allocates device memory.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/kvk.h"
#include "kernels.h"
#include "layout.h"

using namespace kvk;

namespace {

thread_local std::string g_last_error;

kvk_status fail(kvk_status s, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

kvk_status cuda_fail(cudaError_t e, const char *what) {
  return fail(KVK_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

kvk_status check_desc(const kvk_model_desc *d, bool need_support = true) {
  if (!d) return fail(KVK_ERR_INVALID_ARG, "null model descriptor");
  if (d->kind != KVK_KIND_GQA && d->kind != KVK_KIND_MLA)
    return fail(KVK_ERR_INVALID_ARG, "unknown model kind %d", d->kind);
  if (d->n_layers <= 0 || d->n_q_heads <= 0 || d->max_batch <= 0 || d->max_ctx <= 0)
    return fail(KVK_ERR_INVALID_ARG, "layers, heads, batch and context must be positive");
  if (d->max_ctx > (1 << 28)) return fail(KVK_ERR_INVALID_ARG, "max_ctx too large");
  if (d->kind == KVK_KIND_GQA) {
    if (d->n_kv_heads <= 0 || d->n_q_heads % d->n_kv_heads)
      return fail(KVK_ERR_INVALID_ARG, "n_q_heads must be a positive multiple of n_kv_heads");
    if (d->head_dim <= 0) return fail(KVK_ERR_INVALID_ARG, "head_dim must be positive");
    if (need_support && d->head_dim != 64 && d->head_dim != 128)
      return fail(KVK_ERR_UNSUPPORTED, "head_dim %d (supported: 64 and 128)", d->head_dim);
    if (need_support && d->n_q_heads / d->n_kv_heads > 8)
      return fail(KVK_ERR_UNSUPPORTED, "more than 8 query heads per KV head");
  } else {
    if (d->latent_dim < 8 || d->latent_dim % 8 || d->rope_dim < 0)
      return fail(KVK_ERR_INVALID_ARG, "latent_dim must be a positive multiple of 8");
    if (need_support && (d->head_dim != 128 || d->rope_dim != 64))
      return fail(KVK_ERR_UNSUPPORTED, "MLA needs head_dim 128 and rope_dim 64");
    if (need_support && d->n_q_heads > 16)
      return fail(KVK_ERR_UNSUPPORTED, "MLA with more than 16 heads");
  }
  return KVK_OK;
}

kvk_status check_layer(const kvk_model_desc *d, const kvk_layer_cfg *c, int l,
                       bool need_support = true) {
  if (c->inherit) {
    if (l == 0) return fail(KVK_ERR_INVALID_CONFIG, "layer 0 must own a cache (it inherits)");
    return KVK_OK;
  }
  if (c->scheme != KVK_QUANT_GROUPED && c->scheme != KVK_QUANT_SYMMETRIC)
    return fail(KVK_ERR_INVALID_CONFIG, "layer %d: unknown quantisation scheme %d", l, c->scheme);
  if (d->kind == KVK_KIND_MLA) {
    if (c->bits != 16 && c->bits != 8 && c->bits != 4 && c->bits != 2)
      return fail(KVK_ERR_INVALID_CONFIG, "layer %d: bits %d not in {16, 8, 4, 2}", l, c->bits);
    // quantised latents: the kept latent and k^R are each one vector
    // (symmetric: 8/4/2 bits; grouped: 8/4 bits, the group spanning the vector)
    if (need_support && c->bits == 2 && c->scheme == KVK_QUANT_GROUPED)
      return fail(KVK_ERR_UNSUPPORTED,
                  "layer %d: grouped 2-bit latents are not supported (the symmetric scheme has them)", l);
    const int r = d->latent_dim;
    if (c->width != r && c->width != r / 2 && c->width != r / 4 && c->width != r / 8)
      return fail(KVK_ERR_INVALID_CONFIG, "layer %d: width %d not in {r/8, r/4, r/2, r}", l, c->width);
    if (need_support && c->width != 64 && c->width != 128 && c->width != 256 && c->width != 512)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: width %d (supported: 64..512)", l, c->width);
    if (need_support && c->evict_capacity)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: eviction lists on MLA layers", l);
    return KVK_OK;
  }
  if (c->bits != 16 && c->bits != 8 && c->bits != 4 && c->bits != 2)
    return fail(KVK_ERR_INVALID_CONFIG, "layer %d: bits %d not in {16, 8, 4, 2}", l, c->bits);
  if (c->bits != 16 && c->scheme == KVK_QUANT_SYMMETRIC) {
    // one scale per token-head row (Appendix C.3): both axes per token
    if (c->key_axis != KVK_AXIS_TOKEN || c->value_axis != KVK_AXIS_TOKEN)
      return fail(KVK_ERR_INVALID_CONFIG,
                  "layer %d: the symmetric scheme scales whole token-head rows", l);
    if (need_support && d->head_dim != 128)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: symmetric scheme with head_dim %d (supported: 128)",
                  l, d->head_dim);
  } else if (c->bits != 16) {
    if (c->group <= 0 || d->head_dim % c->group)
      return fail(KVK_ERR_INVALID_CONFIG, "layer %d: group %d must divide head_dim", l, c->group);
    if (!need_support) return KVK_OK;
    if (c->bits == 2)
      return fail(KVK_ERR_UNSUPPORTED,
                  "layer %d: grouped 2-bit codes are not supported (the symmetric scheme has them)", l);
    if (c->group != 32 && c->group != 64)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: group %d (supported: 32, 64)", l, c->group);
    if (c->value_axis != KVK_AXIS_TOKEN)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: values are quantised per token", l);
    if (c->key_axis != KVK_AXIS_TOKEN && c->key_axis != KVK_AXIS_CHANNEL)
      return fail(KVK_ERR_INVALID_CONFIG, "layer %d: unknown key axis", l);
    if (c->key_axis == KVK_AXIS_CHANNEL && c->evict_capacity)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d: per-channel keys with an eviction list", l);
  }
  if (c->evict_capacity < 0 || c->evict_capacity > d->max_ctx)
    return fail(KVK_ERR_INVALID_CONFIG, "layer %d: evict_capacity out of range", l);
  return KVK_OK;
}

// Internal scheme and group of a layer: bf16 layers count as grouped with a
// nominal group of 64; symmetric layers scale whole rows (group = head_dim).
int layer_scheme(const kvk_layer_cfg *c) {
  return (c->bits != 16 && c->scheme == KVK_QUANT_SYMMETRIC) ? kSchemeSym : kSchemeGrouped;
}
int layer_group(const kvk_model_desc *d, const kvk_layer_cfg *c) {
  if (c->bits == 16) return 64;
  return layer_scheme(c) == kSchemeSym ? d->head_dim : c->group;
}

ArenaLayout layer_layout(const kvk_model_desc *d, const kvk_layer_cfg *c) {
  const bool mla = d->kind == KVK_KIND_MLA;
  return arena_layout(mla ? 1 : 0, d->max_batch, mla ? 1 : d->n_kv_heads, d->max_ctx, d->head_dim,
                      c->bits, layer_group(d, c), c->key_axis, c->evict_capacity, c->width,
                      d->rope_dim, layer_scheme(c));
}

struct WsLayout {
  size_t err, partial, qlat, olat, total;
};

WsLayout ws_layout(const kvk_model_desc *d, int max_splits) {
  WsLayout w;
  size_t off = 0;
  w.err = off;
  off += 256;
  const bool mla = d->kind == KVK_KIND_MLA;
  const size_t dim = mla ? (size_t)d->latent_dim : (size_t)d->head_dim;
  w.partial = off;
  off += align256((int64_t)max_splits * d->max_batch * d->n_q_heads * (dim + 2) * 4);
  w.qlat = off;
  if (mla) off += align256((int64_t)d->max_batch * d->n_q_heads * (2 * d->latent_dim + 64) * 2);
  w.olat = off;
  if (mla) off += align256((int64_t)d->max_batch * d->n_q_heads * d->latent_dim * 4);
  w.total = off;
  return w;
}

}  // namespace

// planned set-up tiles per unit of a run-schedule decode unless set
// (4: the best of 0..8 measured on int4 and symmetric 4-bit anchors at the
// 14B step shape, B = 20..64)
constexpr int kRunSetupDefault = 4;

struct kvk_cache {
  kvk_model_desc desc;
  std::vector<kvk_layer_cfg> cfg;
  std::vector<int> src;
  std::vector<uint8_t *> arena;
  std::vector<ArenaLayout> lay;
  std::vector<long long> len_hi;  // host upper bound on every sequence's length
  std::vector<int> kept_on;
  uint8_t *ws;
  size_t ws_bytes;
  WsLayout wl;
  int max_splits;
  int sm_count;
  int device;
  std::vector<int> ctas;  // per layer, decode CTAs per SM (0 = not queried)
  uint32_t wait_limit = KVK_WAIT_LIMIT_DEFAULT;  // decode tile-loop waits (kvk_set_wait_limit)
  int schedule = KVK_SCHEDULE_AUTO;              // decode partition (kvk_set_decode_schedule)
  int run_ctas = 0;                              // CTAs of a run-schedule decode (0: whole waves)
  int run_setup = kRunSetupDefault;              // planned set-up tiles per unit of a run decode
  struct alignas(64) Tmap {
    uint8_t bytes[128];
  };
  // per anchor: MLA, the decode kernel's tensor map; GQA with kept lists in
  // a row-gather format, the record table's (gqa_make_rows_tmap)
  std::vector<Tmap> tmap;
  std::vector<char> has_tmap;

  GqaView gqa_view(int l) const {
    const ArenaLayout &A = lay[l];
    const kvk_layer_cfg &c = cfg[l];
    uint8_t *a = arena[l];
    GqaView v;
    v.rec = a + A.rec;
    v.gmeta = A.gmeta >= 0 ? reinterpret_cast<float2 *>(a + A.gmeta) : nullptr;
    v.resid = A.resid >= 0 ? a + A.resid : nullptr;
    v.scales = A.scales >= 0 ? reinterpret_cast<uint32_t *>(a + A.scales) : nullptr;
    v.lens = reinterpret_cast<int32_t *>(a + A.lens);
    v.counter = reinterpret_cast<int32_t *>(a + A.counter);
    v.kept_n = reinterpret_cast<int32_t *>(a + A.kept_n);
    v.kept_idx = reinterpret_cast<int32_t *>(a + A.kept_idx);
    v.cap = A.cap;
    v.kept_cap = c.evict_capacity;
    v.kept_per_head = kept_on[l] == 2;
    v.B = desc.max_batch;
    v.Hkv = desc.n_kv_heads;
    v.D = desc.head_dim;
    v.bits = c.bits;
    v.group = layer_group(&desc, &c);
    v.key_axis = c.bits == 16 ? 0 : c.key_axis;
    v.rec_bytes = A.rec_bytes;
    v.scheme = layer_scheme(&c);
    return v;
  }
  MlaView mla_view(int l) const {
    const ArenaLayout &A = lay[l];
    uint8_t *a = arena[l];
    MlaView v;
    v.rec = a + A.rec;
    v.meta = A.scales >= 0 ? a + A.scales : nullptr;
    v.bits = cfg[l].bits;
    v.scheme = layer_scheme(&cfg[l]);
    v.lens = reinterpret_cast<int32_t *>(a + A.lens);
    v.counter = reinterpret_cast<int32_t *>(a + A.counter);
    v.cap = A.cap;
    v.B = desc.max_batch;
    v.width = cfg[l].width;
    v.rope = desc.rope_dim;
    v.rec_bytes = A.rec_bytes;
    return v;
  }
  int32_t *err() const { return reinterpret_cast<int32_t *>(ws + wl.err); }
};

namespace {

kvk_status check_layer_index(const kvk_cache *c, int layer) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  if (layer < 0 || layer >= c->desc.n_layers)
    return fail(KVK_ERR_INVALID_ARG, "layer %d out of range [0, %d)", layer, c->desc.n_layers);
  return KVK_OK;
}

// Split count of a GQA decode: `tiles` 64-item tiles per (sequence, KV head)
// unit, kernel tiles of `per` such tiles, `slots` resident CTAs.  Cost model
// of a split count s: the launch rounds split boundaries to the kernel tile,
// so each working CTA runs nt kernel tiles plus a fixed cost of about two
// tiles (query set-up, merge of the warps' states, the partial); CTAs run in
// waves of `slots`, and a partial last wave costs at least half a wave (its
// CTAs have the SMs to themselves but run at most ~2x faster).  For the
// bf16 kernel (`full_tail`), bound by HBM rather than by its issue rate and
// running two CTAs per SM with three stages each, a partial last wave costs
// a whole wave and a CTA's fixed cost is about four tiles.  Among choices
// within 1 % the fewer splits win.  Measured on the 7B and 14B step shapes
// and every format, this model's pick is within 1 % of the best split count
// for the quantised kernels; for bf16 at B = 8..64 and T = 2048..16384 it
// is the best or within 1 % except at B = 40 (4 %) (the 14B step: one
// split, 160.5 us); the kept-list gather has a rule of its own (auto_splits).
int choose_splits(int units, int tiles, int per, int slots, int max_splits, bool full_tail) {
  const double F = full_tail ? 4.0 : 2.0, tail = 0.5;
  if (tiles <= 1) return 1;
  per = std::max(1, per);
  const int ktiles = (tiles + per - 1) / per;
  const int smax = std::max(1, std::min(max_splits, ktiles));
  int best = 1;
  double best_t = 1e300;
  for (int s = 1; s <= smax; ++s) {
    const int nt = ((tiles + s - 1) / s + per - 1) / per;  // kernel tiles per CTA
    const int used = (ktiles + nt - 1) / nt;                // splits that get work
    const double w = (double)units * used / slots;
    double t;
    if (w <= 1.0) {
      t = F + nt;
    } else {
      const double fl = std::floor(w), f = w - fl;
      const double last = f <= 1e-9 ? 0.0 : full_tail ? 1.0 : std::max(f, tail);
      t = (F + nt) * (fl + last);
    }
    if (t < best_t * 0.99) {
      best_t = t;
      best = s;
    }
  }
  return best;
}

// Tiles of 64 items (positions, or kept-list entries) an anchor's decode
// covers, from the host-side bound on its lengths.
int layer_tiles(const kvk_cache *c, int a) {
  const long long items = c->kept_on[a] ? c->cfg[a].evict_capacity : c->len_hi[a];
  return (int)std::max<long long>(1, (items + kTile - 1) / kTile);
}

int auto_splits(kvk_cache *c, int a) {
  const bool mla = c->desc.kind == KVK_KIND_MLA;
  if (!c->ctas[a]) {
    if (mla) {
      c->ctas[a] = mla_decode_ctas_per_sm(c->cfg[a].width, c->cfg[a].bits);
    } else {
      const kvk_layer_cfg &L = c->cfg[a];
      c->ctas[a] = gqa_decode_ctas_per_sm(L.bits, c->desc.head_dim, L.bits == 16 ? 0 : L.key_axis,
                                          layer_group(&c->desc, &L), layer_scheme(&L));
    }
  }
  const int units = mla ? c->desc.max_batch : c->desc.max_batch * c->desc.n_kv_heads;
  const int slots = c->sm_count * c->ctas[a];
  if (mla) {
    // Latent partials are as wide as the latent, and a second wave of these
    // long CTAs costs more than it fills: as many splits as keep every CTA
    // resident at once.
    const int s = std::max(1, std::min(slots / std::max(1, units), c->max_splits));
    return std::min(s, std::min(64, layer_tiles(c, a)));
  }
  const kvk_layer_cfg &L = c->cfg[a];
  const int kt = gqa_decode_tile(L.bits, c->desc.head_dim, L.bits == 16 ? 0 : L.key_axis,
                                 layer_group(&c->desc, &L), layer_scheme(&L));
  if (c->kept_on[a]) {
    // Kept-list gathers (random record reads) run best with one wave of
    // CTAs filling at most 85 % of the resident slots: at the 131k-context
    // shape (32 units, int4 g32, 608 slots) 16 splits (512 CTAs) took 32.0
    // us per call against 36.1 with 19 (every slot), 37.4 with 14, 35.5
    // with 20; the same held for the earlier chunked gather (36.9 / 40.4).
    const int ktiles = (layer_tiles(c, a) + kt / kTile - 1) / (kt / kTile);
    const int s = (int)(0.85 * slots) / std::max(1, units);
    return std::max(1, std::min(std::min(s, ktiles), c->max_splits));
  }
  return choose_splits(units, layer_tiles(c, a), kt / kTile, slots, c->max_splits, L.bits == 16);
}

// The run schedule of an automatic decode of anchor a (kernel side in
// decode_gqa.cuh): n CTAs, each an equal run of the (unit, kernel tile)
// grid, n >= units so that a run meets at most two units.  n is the
// smallest whole number of waves of resident CTAs that is at least the
// number of units, or the count set with kvk_set_decode_schedule (clamped
// to [units, tiles]).  Formats: quantised with per-token keys or the
// symmetric scheme, contiguous reads.  Returns false (split grid) when the
// format has no run kernel, the schedule is off, there are fewer tiles than
// CTAs, or the partial slots would exceed max_splits.  The automatic choice
// takes the runs only where the split grid gives each CTA at most 13 kernel
// tiles and leaves its last wave less than 90 % full: the decode is bound
// by HBM even with a partly filled last wave, so what the runs save is the
// per-CTA start-up of many short splits.  Measured at the 14B step shape
// (int4 g32, one anchor): B = 20 (6 splits of 11 tiles) 54.1 -> 48.6 us,
// B = 24 (5 of 13) 58.9 -> 56.5 us; with 16 or more tiles per split the
// runs were 1-4 % slower (B = 32 and 64, symmetric 8-bit at B = 32).
struct RunPlan {
  int ctas = 0, tpu = 0, slots = 0, q = 0, r = 0, setup = 0;
};
bool plan_runs(kvk_cache *c, int a, RunPlan *p) {
  const kvk_layer_cfg &L = c->cfg[a];
  if (c->schedule == KVK_SCHEDULE_SPLITS || c->desc.kind != KVK_KIND_GQA) return false;
  if (L.bits == 16 || c->kept_on[a]) return false;
  if (layer_scheme(&L) != kSchemeSym && L.key_axis != 0) return false;  // per-channel keys
  const int kt = gqa_decode_tile(L.bits, c->desc.head_dim, L.key_axis, layer_group(&c->desc, &L),
                                 layer_scheme(&L));
  const int per = kt / kTile;
  const long long tdata = (layer_tiles(c, a) + per - 1) / per;  // data tiles per unit
  const long long tpu = tdata + c->run_setup;                   // planned tiles per unit
  const long long units = (long long)c->desc.max_batch * c->desc.n_kv_heads;
  const long long total = units * tpu;
  auto_splits(c, a);  // queries the CTAs per SM
  const long long slots = (long long)c->sm_count * c->ctas[a];
  long long n;
  if (c->run_ctas > 0) {
    n = std::min<long long>(std::max<long long>(c->run_ctas, units), total);
  } else {
    n = slots;
    while (n < units) n += slots;
  }
  // the kernel's run arithmetic is 32-bit: W < 2^31, n < 2^16
  if (n > total || total >= (1LL << 31) || n >= (1LL << 16)) return false;
  if (c->schedule == KVK_SCHEDULE_AUTO) {
    if (total < 4 * n) return false;
    const int s = std::min(auto_splits(c, a), layer_tiles(c, a));
    const long long nt = (tdata + s - 1) / s;                 // kernel tiles per split
    const long long grid = units * ((tdata + nt - 1) / nt);   // CTAs that get work
    const double fill = (double)(grid % slots) / (double)slots;
    if (nt > 13 || grid % slots == 0 || fill >= 0.9) return false;
  }
  int kmax = 0;
  for (long long u = 0; u < units; ++u) {
    const long long c0 = ((u * tpu + 1) * n - 1) / total, c1 = ((u + 1) * tpu * n - 1) / total;
    kmax = std::max<int>(kmax, (int)(c1 - c0 + 1));
  }
  if (kmax > c->max_splits) return false;
  p->ctas = (int)n;
  p->tpu = (int)tpu;
  p->slots = kmax;
  p->q = (int)(total / n);
  p->r = (int)(total % n);
  p->setup = c->run_setup;
  return true;
}

}  // namespace

extern "C" {

const char *kvk_status_string(kvk_status s) {
  switch (s) {
    case KVK_OK: return "ok";
    case KVK_ERR_INVALID_ARG: return "invalid argument";
    case KVK_ERR_INVALID_CONFIG: return "invalid configuration";
    case KVK_ERR_INHERITED_LAYER: return "layer inherits its cache";
    case KVK_ERR_CAPACITY: return "capacity exceeded";
    case KVK_ERR_UNSUPPORTED: return "unsupported";
    case KVK_ERR_CUDA: return "CUDA error";
    case KVK_ERR_DEVICE: return "device error word set";
  }
  return "unknown status";
}

const char *kvk_last_error(void) { return g_last_error.c_str(); }

const char *kvk_version(void) { return "kvk 0.1 sm_103a"; }

kvk_status kvk_cache_plan(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                          size_t *arena_bytes) {
  kvk_status s = check_desc(desc);
  if (s) return s;
  if (!cfg || !arena_bytes) return fail(KVK_ERR_INVALID_ARG, "null plan or output");
  for (int l = 0; l < desc->n_layers; ++l) {
    s = check_layer(desc, &cfg[l], l);
    if (s) return s;
  }
  for (int l = 0; l < desc->n_layers; ++l)
    arena_bytes[l] = cfg[l].inherit ? 0 : (size_t)layer_layout(desc, &cfg[l]).total;
  return KVK_OK;
}

kvk_status kvk_workspace_size(const kvk_model_desc *desc, int32_t max_splits, size_t *ws_bytes) {
  kvk_status s = check_desc(desc);
  if (s) return s;
  if (!ws_bytes || max_splits < 1 || max_splits > 256)
    return fail(KVK_ERR_INVALID_ARG, "max_splits must be in [1, 256]");
  *ws_bytes = ws_layout(desc, max_splits).total;
  return KVK_OK;
}

kvk_status kvk_cache_create(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                            void *const *arenas, void *workspace, size_t ws_bytes,
                            int32_t max_splits, kvk_cache **out) {
  if (!out) return fail(KVK_ERR_INVALID_ARG, "null output handle");
  *out = nullptr;
  std::vector<size_t> bytes(desc ? std::max(0, desc->n_layers) : 0);
  kvk_status s = kvk_cache_plan(desc, cfg, bytes.data());
  if (s) return s;
  if (max_splits < 1 || max_splits > 256) return fail(KVK_ERR_INVALID_ARG, "max_splits must be in [1, 256]");
  if (!arenas || !workspace || !aligned16(workspace))
    return fail(KVK_ERR_INVALID_ARG, "null or misaligned arenas/workspace");
  const WsLayout wl = ws_layout(desc, max_splits);
  if (ws_bytes < wl.total)
    return fail(KVK_ERR_INVALID_ARG, "workspace too small: %zu < %zu", ws_bytes, wl.total);
  for (int l = 0; l < desc->n_layers; ++l) {
    if (cfg[l].inherit) continue;
    if (!arenas[l] || (reinterpret_cast<uintptr_t>(arenas[l]) & 255u))
      return fail(KVK_ERR_INVALID_ARG, "arena of layer %d is null or not 256-byte aligned", l);
  }
  kvk_cache *c = new (std::nothrow) kvk_cache();
  if (!c) return fail(KVK_ERR_INVALID_ARG, "out of host memory");
  c->desc = *desc;
  c->cfg.assign(cfg, cfg + desc->n_layers);
  c->src.resize(desc->n_layers);
  c->arena.assign(desc->n_layers, nullptr);
  c->lay.resize(desc->n_layers);
  c->len_hi.assign(desc->n_layers, 0);
  c->kept_on.assign(desc->n_layers, 0);
  c->ctas.assign(desc->n_layers, 0);
  int last = 0;
  for (int l = 0; l < desc->n_layers; ++l) {
    if (!cfg[l].inherit) {
      last = l;
      c->arena[l] = static_cast<uint8_t *>(arenas[l]);
      c->lay[l] = layer_layout(desc, &cfg[l]);
    }
    c->src[l] = last;
  }
  c->ws = static_cast<uint8_t *>(workspace);
  c->ws_bytes = ws_bytes;
  c->wl = wl;
  c->max_splits = max_splits;
  cudaError_t e = cudaGetDevice(&c->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, c->device);
  if (e != cudaSuccess) {
    delete c;
    return cuda_fail(e, "querying the device");
  }
  c->tmap.resize(desc->n_layers);
  c->has_tmap.assign(desc->n_layers, 0);
  for (int l = 0; l < desc->n_layers; ++l) {
    if (cfg[l].inherit) continue;
    if (desc->kind == KVK_KIND_MLA) {
      if (cfg[l].bits != 16) continue;  // quantised tiles use bulk copies
      e = mla_make_tmap(c->tmap[l].bytes, c->mla_view(l));
    } else {
      if (cfg[l].evict_capacity <= 0 ||
          !gqa_decode_row_gather(cfg[l].bits, cfg[l].key_axis, layer_scheme(&cfg[l])))
        continue;
      const GqaView gv = c->gqa_view(l);
      if ((long long)gv.B * gv.Hkv * gv.cap >= (1LL << 31)) {
        delete c;
        return fail(KVK_ERR_INVALID_CONFIG,
                    "layer %d: kept lists on grouped per-token anchors need max_batch x n_kv_heads x "
                    "capacity below 2^31 records",
                    l);
      }
      e = gqa_make_rows_tmap(c->tmap[l].bytes, gv);
    }
    if (e != cudaSuccess) {
      delete c;
      return cuda_fail(e, "encoding an anchor's tensor map");
    }
    c->has_tmap[l] = 1;
  }
  *out = c;
  return KVK_OK;
}

kvk_status kvk_cache_destroy(kvk_cache *cache) {
  delete cache;
  return KVK_OK;
}

kvk_status kvk_set_wait_limit(kvk_cache *c, uint32_t polls) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  c->wait_limit = polls;
  return KVK_OK;
}

kvk_status kvk_set_decode_schedule(kvk_cache *c, int32_t schedule, int32_t run_ctas,
                                   int32_t run_setup) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  if (schedule != KVK_SCHEDULE_AUTO && schedule != KVK_SCHEDULE_SPLITS && schedule != KVK_SCHEDULE_RUNS)
    return fail(KVK_ERR_INVALID_ARG, "unknown decode schedule %d", schedule);
  if (run_ctas < 0) return fail(KVK_ERR_INVALID_ARG, "run_ctas %d < 0", run_ctas);
  if (run_setup < -1 || run_setup > 64)
    return fail(KVK_ERR_INVALID_ARG, "run_setup %d outside [-1, 64]", run_setup);
  c->schedule = schedule;
  c->run_ctas = run_ctas;
  c->run_setup = run_setup < 0 ? kRunSetupDefault : run_setup;
  return KVK_OK;
}

kvk_status kvk_cache_reset(kvk_cache *c, kvk_stream stream) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  for (int l = 0; l < c->desc.n_layers; ++l) {
    if (c->cfg[l].inherit) continue;
    const ArenaLayout &A = c->lay[l];
    // lens, counter and kept_n are the arena's first three 256-byte-aligned slots
    cudaError_t e = cudaMemsetAsync(c->arena[l], 0, (size_t)A.kept_idx, st);
    if (e != cudaSuccess) return cuda_fail(e, "resetting lengths");
    c->len_hi[l] = 0;
    c->kept_on[l] = 0;
  }
  cudaError_t e = cudaMemsetAsync(c->err(), 0, 4, st);
  if (e != cudaSuccess) return cuda_fail(e, "resetting the error word");
  return KVK_OK;
}

kvk_status kvk_layer_source(const kvk_cache *c, int32_t layer, int32_t *src) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (!src) return fail(KVK_ERR_INVALID_ARG, "null output");
  *src = c->src[layer];
  return KVK_OK;
}

kvk_status kvk_layer_lengths(const kvk_cache *c, int32_t layer, const int32_t **lens) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (!lens) return fail(KVK_ERR_INVALID_ARG, "null output");
  const int a = c->src[layer];
  *lens = reinterpret_cast<const int32_t *>(c->arena[a] + c->lay[a].lens);
  return KVK_OK;
}

kvk_status kvk_append(kvk_cache *c, int32_t layer, const void *k, const void *v, int32_t in_dtype,
                      int32_t n_new, const int32_t *n_new_per_seq, kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->cfg[layer].inherit)
    return fail(KVK_ERR_INHERITED_LAYER, "layer %d inherits layer %d's cache", layer, c->src[layer]);
  if (n_new < 0) return fail(KVK_ERR_INVALID_ARG, "n_new < 0");
  if (n_new == 0) return KVK_OK;
  if (!k || !v || !aligned16(k) || !aligned16(v))
    return fail(KVK_ERR_INVALID_ARG, "null or misaligned k/v");
  if (c->len_hi[layer] + n_new > c->desc.max_ctx)
    return fail(KVK_ERR_CAPACITY, "layer %d: %lld + %d positions exceed max_ctx %d", layer,
                c->len_hi[layer], n_new, c->desc.max_ctx);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (c->desc.kind == KVK_KIND_GQA) {
    if (in_dtype != KVK_DTYPE_F32 && in_dtype != KVK_DTYPE_BF16)
      return fail(KVK_ERR_INVALID_ARG, "in_dtype must be F32 or BF16");
    e = launch_gqa_append(c->gqa_view(layer), k, v, in_dtype == KVK_DTYPE_F32, n_new,
                          n_new_per_seq, c->err(), st);
  } else {
    if (in_dtype != KVK_DTYPE_BF16) return fail(KVK_ERR_INVALID_ARG, "MLA appends take BF16");
    e = launch_mla_append(c->mla_view(layer), k, v, c->desc.latent_dim, n_new, n_new_per_seq,
                          c->err(), st);
  }
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  c->len_hi[layer] += n_new;
  return KVK_OK;
}

kvk_status kvk_rewind(kvk_cache *c, int32_t n, kvk_stream stream) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  if (n < 0) return fail(KVK_ERR_INVALID_ARG, "n < 0");
  RewindArgs r;
  r.B = c->desc.max_batch;
  r.n = n;
  r.n_anchors = 0;
  for (int l = 0; l < c->desc.n_layers; ++l) {
    const kvk_layer_cfg &L = c->cfg[l];
    if (L.inherit) continue;
    if (c->desc.kind == KVK_KIND_GQA && L.bits != 16 && L.key_axis == KVK_AXIS_CHANNEL)
      return fail(KVK_ERR_UNSUPPORTED, "layer %d has per-channel key groups", l);
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  for (int l = 0; l < c->desc.n_layers; ++l) {
    if (c->cfg[l].inherit) continue;
    r.lens[r.n_anchors++] = reinterpret_cast<int32_t *>(c->arena[l] + c->lay[l].lens);
    c->len_hi[l] = std::max<long long>(0, c->len_hi[l] - n);
    if (r.n_anchors == 64) {
      cudaError_t e = launch_rewind(r, st);
      if (e != cudaSuccess) return cuda_fail(e, "rewind launch");
      r.n_anchors = 0;
    }
  }
  if (r.n_anchors) {
    cudaError_t e = launch_rewind(r, st);
    if (e != cudaSuccess) return cuda_fail(e, "rewind launch");
  }
  return KVK_OK;
}

kvk_status kvk_decode_plan_splits(kvk_cache *c, int32_t layer, int32_t *n_splits) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (!n_splits) return fail(KVK_ERR_INVALID_ARG, "null output");
  RunPlan rp;
  *n_splits = plan_runs(c, c->src[layer], &rp)
                  ? rp.slots
                  : std::min(auto_splits(c, c->src[layer]), layer_tiles(c, c->src[layer]));
  return KVK_OK;
}

kvk_status kvk_set_kept(kvk_cache *c, int32_t layer, const int32_t *idx, const int32_t *n_kept,
                        kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->cfg[layer].inherit)
    return fail(KVK_ERR_INHERITED_LAYER, "layer %d inherits; set the list on layer %d", layer,
                c->src[layer]);
  const int cap = c->cfg[layer].evict_capacity;
  if (!n_kept) {
    c->kept_on[layer] = 0;
    return KVK_OK;
  }
  if (cap <= 0) return fail(KVK_ERR_INVALID_CONFIG, "layer %d has evict_capacity 0", layer);
  if (!idx) return fail(KVK_ERR_INVALID_ARG, "null kept index list");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const ArenaLayout &A = c->lay[layer];
  const size_t B = c->desc.max_batch;
  cudaError_t e = cudaMemcpyAsync(c->arena[layer] + A.kept_idx, idx, B * cap * 4,
                                  cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(c->arena[layer] + A.kept_n, n_kept, B * 4, cudaMemcpyDeviceToDevice, st);
  if (e != cudaSuccess) return cuda_fail(e, "copying the kept list");
  c->kept_on[layer] = 1;
  return KVK_OK;
}

namespace {
struct EvictScratch {
  size_t votes, stats, scores, total;  // region sizes: votes, statistics, scores
  int n_tiles;
};
EvictScratch evict_scratch(const kvk_cache *c, int layer, int n_win) {
  EvictScratch e;
  const size_t units = (size_t)c->desc.max_batch * c->desc.n_kv_heads;
  const size_t cap = (size_t)c->lay[layer].cap;
  const size_t R = (size_t)n_win * (c->desc.n_q_heads / c->desc.n_kv_heads);
  e.n_tiles = (int)((cap + kEvictTile - 1) / kEvictTile);
  e.votes = align256((int64_t)(units * cap * 4));
  e.stats = align256((int64_t)((units * R * kEvictStatSub * e.n_tiles + units * R) * 8));
  e.scores = evict_uses_tc(c->desc.head_dim, (int)R)
                 ? 0
                 : align256((int64_t)(units * R * e.n_tiles * kEvictTile * 4));
  e.total = e.votes + e.stats + e.scores;
  return e;
}

kvk_status check_evict(const kvk_cache *c, int32_t layer, int32_t n_win) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_GQA) return fail(KVK_ERR_UNSUPPORTED, "eviction scoring on an MLA cache");
  const kvk_layer_cfg &L = c->cfg[layer];
  if (L.inherit)
    return fail(KVK_ERR_INHERITED_LAYER, "layer %d inherits; evict on layer %d", layer, c->src[layer]);
  if (L.evict_capacity <= 0) return fail(KVK_ERR_INVALID_CONFIG, "layer %d has evict_capacity 0", layer);
  if (L.bits != 16 && L.key_axis == KVK_AXIS_CHANNEL && L.scheme != KVK_QUANT_SYMMETRIC)
    return fail(KVK_ERR_UNSUPPORTED, "layer %d: eviction with per-channel keys", layer);
  if (n_win < 1 || n_win > 256) return fail(KVK_ERR_INVALID_ARG, "n_win %d outside [1, 256]", n_win);
  return KVK_OK;
}
}  // namespace

kvk_status kvk_evict_scratch_size(const kvk_cache *c, int32_t layer, int32_t n_win, size_t *bytes) {
  kvk_status s = check_evict(c, layer, n_win);
  if (s) return s;
  if (!bytes) return fail(KVK_ERR_INVALID_ARG, "null output");
  *bytes = evict_scratch(c, layer, n_win).total;
  return KVK_OK;
}

kvk_status kvk_evict_window(kvk_cache *c, int32_t layer, const void *q_win, int32_t q_dtype,
                            int32_t n_win, float softmax_scale, int32_t budget, void *scratch,
                            size_t scratch_bytes, kvk_stream stream) {
  kvk_status s = check_evict(c, layer, n_win);
  if (s) return s;
  const kvk_layer_cfg &L = c->cfg[layer];
  if (budget < n_win || budget > L.evict_capacity)
    return fail(KVK_ERR_INVALID_ARG, "budget %d outside [n_win %d, evict_capacity %d]", budget, n_win,
                L.evict_capacity);
  if (!q_win || !aligned16(q_win)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned q_win");
  if (q_dtype != KVK_DTYPE_F32 && q_dtype != KVK_DTYPE_BF16)
    return fail(KVK_ERR_INVALID_ARG, "q_dtype must be F32 or BF16");
  if (!std::isfinite(softmax_scale) || !(softmax_scale > 0.f))
    return fail(KVK_ERR_INVALID_ARG, "softmax scale must be finite and positive");
  const EvictScratch es = evict_scratch(c, layer, n_win);
  if (!scratch || (reinterpret_cast<uintptr_t>(scratch) & 255u) || scratch_bytes < es.total)
    return fail(KVK_ERR_INVALID_ARG, "scratch null, not 256-byte aligned or smaller than %zu bytes",
                es.total);
  EvictArgs a;
  a.v = c->gqa_view(layer);
  a.v.kept_per_head = 1;
  a.q = q_win;
  a.q_f32 = q_dtype == KVK_DTYPE_F32;
  a.Hq = c->desc.n_q_heads;
  a.G = c->desc.n_q_heads / c->desc.n_kv_heads;
  a.n_win = n_win;
  a.budget = budget;
  a.sig_log2 = softmax_scale * 1.4426950408889634f;
  a.n_tiles = es.n_tiles;
  a.sc_stride = es.n_tiles * kEvictTile;
  a.stat_sub = evict_uses_tc(c->desc.head_dim, n_win * a.G) ? kEvictStatSub : 1;
  a.votes = static_cast<float *>(scratch);
  a.stats = reinterpret_cast<float2 *>(static_cast<uint8_t *>(scratch) + es.votes);
  a.fin = a.stats + (size_t)c->desc.max_batch * c->desc.n_kv_heads * n_win * a.G * kEvictStatSub *
                        es.n_tiles;
  a.scores = es.scores ? reinterpret_cast<float *>(static_cast<uint8_t *>(scratch) + es.votes + es.stats)
                       : nullptr;
  a.err = c->err();
  cudaError_t e = launch_gqa_evict(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "eviction launch");
  c->kept_on[layer] = 2;  // per-(sequence, kv head) lists from now on
  return KVK_OK;
}

namespace {
kvk_status check_prefill(const kvk_cache *c, int32_t layer, int32_t n_q) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_GQA) return fail(KVK_ERR_UNSUPPORTED, "pre-fill on an MLA cache");
  if (c->desc.head_dim != 128) return fail(KVK_ERR_UNSUPPORTED, "pre-fill needs head_dim 128");
  if (n_q < 1 || n_q > c->desc.max_ctx)
    return fail(KVK_ERR_INVALID_ARG, "n_q %d outside [1, max_ctx]", n_q);
  return KVK_OK;
}
// Pre-fill scratch: the job counter, then the expanded tiles (every
// 64-position tile of every unit, dequantised once).
struct PrefillScratch {
  size_t counters, tiles, total;
};
PrefillScratch prefill_scratch(const kvk_cache *c, int32_t layer, int32_t n_q) {
  (void)n_q;
  PrefillScratch p;
  const int a = c->src[layer];
  p.counters = 0;
  p.tiles = 1024;
  const size_t units = (size_t)c->desc.max_batch * c->desc.n_kv_heads;
  p.total = p.tiles + units * (size_t)(c->lay[a].cap / 64) * prefill_tile_bytes(c->cfg[a].bits);
  return p;
}
}  // namespace

namespace {
// MLA pre-fill scratch: the absorbed queries of every query row, then the
// rows' latent partials (one split)
struct MlaPrefillScratch {
  size_t qlat, partial, total;
};
MlaPrefillScratch mla_prefill_scratch(const kvk_cache *c, int32_t layer, int32_t n_q) {
  const int a = c->src[layer];
  const size_t rows = (size_t)c->desc.max_batch * n_q * c->desc.n_q_heads;
  const int W = c->cfg[a].width;
  MlaPrefillScratch p;
  p.qlat = 0;
  p.partial = (size_t)align256((int64_t)(rows * (2 * W + c->desc.rope_dim) * 2));
  p.total = p.partial + rows * (W + 2) * 4;
  return p;
}
kvk_status check_prefill_mla(const kvk_cache *c, int32_t layer, int32_t n_q) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_MLA) return fail(KVK_ERR_INVALID_ARG, "cache is not MLA");
  if (n_q < 1 || n_q > c->desc.max_ctx)
    return fail(KVK_ERR_INVALID_ARG, "n_q %d outside [1, max_ctx]", n_q);
  return KVK_OK;
}
}  // namespace

kvk_status kvk_prefill_scratch_size(const kvk_cache *c, int32_t layer, int32_t n_q, size_t *bytes) {
  if (c && c->desc.kind == KVK_KIND_MLA) {
    kvk_status s = check_prefill_mla(c, layer, n_q);
    if (s) return s;
    if (!bytes) return fail(KVK_ERR_INVALID_ARG, "null output");
    *bytes = mla_prefill_scratch(c, layer, n_q).total;
    return KVK_OK;
  }
  kvk_status s = check_prefill(c, layer, n_q);
  if (s) return s;
  if (!bytes) return fail(KVK_ERR_INVALID_ARG, "null output");
  *bytes = prefill_scratch(c, layer, n_q).total;
  return KVK_OK;
}

kvk_status kvk_prefill_attention(kvk_cache *c, int32_t layer, const void *q, int32_t q_dtype, int32_t n_q,
                                 float softmax_scale, float *out, void *scratch, size_t scratch_bytes,
                                 kvk_stream stream) {
  kvk_status s = check_prefill(c, layer, n_q);
  if (s) return s;
  if (!q || !aligned16(q)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned q");
  if (!out || !aligned16(out)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned out");
  if (q_dtype != KVK_DTYPE_F32 && q_dtype != KVK_DTYPE_BF16)
    return fail(KVK_ERR_INVALID_ARG, "q_dtype must be F32 or BF16");
  if (!std::isfinite(softmax_scale) || !(softmax_scale > 0.f))
    return fail(KVK_ERR_INVALID_ARG, "softmax scale must be finite and positive");
  const PrefillScratch ps = prefill_scratch(c, layer, n_q);
  if (!scratch || (reinterpret_cast<uintptr_t>(scratch) & 255u) || scratch_bytes < ps.total)
    return fail(KVK_ERR_INVALID_ARG, "scratch null, not 256-byte aligned or smaller than %zu bytes",
                ps.total);
  PfArgs a;
  a.v = c->gqa_view(c->src[layer]);
  a.q = q;
  a.q_f32 = q_dtype == KVK_DTYPE_F32;
  a.Hq = c->desc.n_q_heads;
  a.G = c->desc.n_q_heads / c->desc.n_kv_heads;
  a.n_q = n_q;
  a.sig_log2 = softmax_scale * 1.4426950408889634f;
  a.counter = reinterpret_cast<int *>(static_cast<uint8_t *>(scratch) + ps.counters);
  a.tiles = static_cast<uint8_t *>(scratch) + ps.tiles;
  a.out = out;
  a.err = c->err();
  if (!prefill_plan_fits(a)) return fail(KVK_ERR_UNSUPPORTED, "pre-fill plan does not fit shared memory");
  cudaError_t e = launch_gqa_prefill(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "pre-fill launch");
  return KVK_OK;
}

kvk_status kvk_export_kept(const kvk_cache *c, int32_t layer, int32_t *idx, int32_t *n_kept,
                           int32_t *per_head, kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->cfg[layer].inherit)
    return fail(KVK_ERR_INHERITED_LAYER, "layer %d inherits layer %d's lists", layer, c->src[layer]);
  if (!idx || !n_kept || !per_head) return fail(KVK_ERR_INVALID_ARG, "null output");
  const int cap = c->cfg[layer].evict_capacity;
  *per_head = c->kept_on[layer] == 2 ? 1 : (c->kept_on[layer] == 1 ? 0 : -1);
  if (cap <= 0 || c->kept_on[layer] == 0) return KVK_OK;
  const size_t units = (size_t)c->desc.max_batch * (c->kept_on[layer] == 2 ? c->desc.n_kv_heads : 1);
  const ArenaLayout &A = c->lay[layer];
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(idx, c->arena[layer] + A.kept_idx, units * cap * 4,
                                  cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(n_kept, c->arena[layer] + A.kept_n, units * 4, cudaMemcpyDeviceToDevice, st);
  if (e != cudaSuccess) return cuda_fail(e, "copying the kept lists");
  return KVK_OK;
}

static kvk_status gqa_decode_common(kvk_cache *c, int32_t layer, const void *q, int32_t q_dtype,
                                    float scale, float *out, float *partial, int32_t n_splits,
                                    bool merge, kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_GQA) return fail(KVK_ERR_INVALID_ARG, "cache is not GQA");
  if (!q || !aligned16(q)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned q");
  if (q_dtype != KVK_DTYPE_F32 && q_dtype != KVK_DTYPE_BF16)
    return fail(KVK_ERR_INVALID_ARG, "q_dtype must be F32 or BF16");
  if (n_splits < 0 || n_splits > c->max_splits)
    return fail(KVK_ERR_INVALID_ARG, "n_splits %d outside [0, %d]", n_splits, c->max_splits);
  if (!std::isfinite(scale) || !(scale > 0.f))
    return fail(KVK_ERR_INVALID_ARG, "softmax scale must be finite and positive");
  const int a = c->src[layer];
  GqaDecodeArgs args;
  args.v = c->gqa_view(a);
  args.gather = c->kept_on[a];
  const int tiles = layer_tiles(c, a);
  RunPlan rp;
  const bool runs = n_splits == 0 && plan_runs(c, a, &rp);
  if (runs) n_splits = rp.slots;
  if (n_splits == 0) n_splits = auto_splits(c, a);
  // a partial-only call keeps the caller's split count (extra splits are
  // empty and write m = -inf, l = 0); a full call never uses more splits
  // than tiles.
  if (merge && !runs) n_splits = std::min(n_splits, tiles);
  args.q = q;
  args.q_f32 = q_dtype == KVK_DTYPE_F32;
  args.Hq = c->desc.n_q_heads;
  args.G = c->desc.n_q_heads / c->desc.n_kv_heads;
  args.sig_log2 = scale * 1.4426950408889634f;
  args.n_splits = n_splits;
  // split boundaries fall on the kernel's tile height (64 or 128 positions)
  const int kt =
      gqa_decode_tile(args.v.bits, args.v.D, args.v.key_axis, args.v.group, args.v.scheme);
  const int per = kt / kTile;
  const int tps = ((tiles + n_splits - 1) / n_splits + per - 1) / per * per;
  args.items_per_split = tps * kTile;
  args.err = c->err();
  args.wait_limit = c->wait_limit;
  args.rows = c->has_tmap[a] ? c->tmap[a].bytes : nullptr;
  if (runs) {
    args.run_ctas = rp.ctas;
    args.run_tpu = rp.tpu;
    args.run_slots = rp.slots;
    args.run_q = rp.q;
    args.run_r = rp.r;
    args.run_setup = rp.setup;
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (merge && n_splits == 1 && !runs) {
    args.out = out;  // one split: the kernel normalises and writes the output
    args.partial = nullptr;
  } else {
    args.out = nullptr;
    args.partial = partial ? partial : reinterpret_cast<float *>(c->ws + c->wl.partial);
  }
  cudaError_t e = launch_gqa_decode(args, st);
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  if (merge && (n_splits > 1 || runs)) {
    e = launch_splitk_merge(args.partial, n_splits, c->desc.max_batch * c->desc.n_q_heads,
                            c->desc.head_dim, out, st);
    if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  }
  return KVK_OK;
}

}  // extern "C"

// Records a failed CUDA call as the thread's last error (for noalloc.cu).
kvk_status kvk_internal_cuda_error(cudaError_t e, const char *what) { return cuda_fail(e, what); }

// INVALID_ARG unless the calling thread's current device is the one the cache
// was created on (for noalloc.cu, whose fixed buffer is per device).
kvk_status kvk_internal_check_current_device(const kvk_cache *c) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  int dev = -1;
  const cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "querying the current device");
  if (dev != c->device)
    return fail(KVK_ERR_INVALID_ARG,
                "current device %d is not the cache's device %d: make the cache's device current",
                dev, c->device);
  return KVK_OK;
}

// Decode with the split-K partials in device memory the caller of this
// function chose (`partial`, `partial_floats` floats) instead of the cache's
// workspace.  Rejects a call whose partials would not fit.  Used by the
// fixed-scratch entry point in noalloc.cu; not part of the C ABI.
kvk_status kvk_internal_decode_with_partials(kvk_cache *c, int32_t layer, const void *q,
                                             int32_t q_dtype, float scale, float *out,
                                             int32_t n_splits, float *partial,
                                             size_t partial_floats, kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_GQA) return fail(KVK_ERR_INVALID_ARG, "cache is not GQA");
  if (!out || !aligned16(out)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned out");
  if (n_splits < 0 || n_splits > c->max_splits)
    return fail(KVK_ERR_INVALID_ARG, "n_splits %d outside [0, %d]", n_splits, c->max_splits);
  const int a = c->src[layer];
  const int tiles = layer_tiles(c, a);
  RunPlan rp;
  const bool runs = n_splits == 0 && plan_runs(c, a, &rp);
  int ns = runs ? rp.slots : std::min(n_splits == 0 ? auto_splits(c, a) : n_splits, tiles);
  const size_t need = (ns > 1 || runs) ? (size_t)ns * c->desc.max_batch * c->desc.n_q_heads *
                                   ((size_t)c->desc.head_dim + 2)
                             : 0;
  if (need > partial_floats)
    return fail(KVK_ERR_CAPACITY,
                "layer %d: %d splits x %d rows need %zu partial floats; the fixed buffer "
                "holds %zu (use fewer splits or kvk_decode_attention)",
                layer, ns, c->desc.max_batch * c->desc.n_q_heads, need, partial_floats);
  return gqa_decode_common(c, layer, q, q_dtype, scale, out, partial, runs ? 0 : ns, true, stream);
}

extern "C" {

kvk_status kvk_decode_attention(kvk_cache *c, int32_t layer, const void *q, int32_t q_dtype,
                                float softmax_scale, float *out, int32_t n_splits,
                                kvk_stream stream) {
  if (!out || !aligned16(out)) return fail(KVK_ERR_INVALID_ARG, "null or misaligned out");
  return gqa_decode_common(c, layer, q, q_dtype, softmax_scale, out, nullptr, n_splits, true,
                           stream);
}

kvk_status kvk_decode_partial(kvk_cache *c, int32_t layer, const void *q, int32_t q_dtype,
                              float softmax_scale, float *partials, int32_t n_splits,
                              kvk_stream stream) {
  if (!partials || !aligned16(partials))
    return fail(KVK_ERR_INVALID_ARG, "null or misaligned partials");
  if (n_splits == 1 || n_splits < 0)
    return fail(KVK_ERR_INVALID_ARG, "kvk_decode_partial needs n_splits 0 (automatic) or >= 2");
  return gqa_decode_common(c, layer, q, q_dtype, softmax_scale, nullptr, partials, n_splits,
                           false, stream);
}

kvk_status kvk_splitk_reduce(const float *partials, int32_t n_splits, int32_t n_rows, int32_t dim,
                             float *out, kvk_stream stream) {
  if (!partials || !out) return fail(KVK_ERR_INVALID_ARG, "null partials or out");
  if (n_splits < 1 || n_splits > 256 || n_rows < 1 || dim < 1)
    return fail(KVK_ERR_INVALID_ARG, "bad sizes");
  cudaError_t e = launch_splitk_merge(partials, n_splits, n_rows, dim, out,
                                      reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  return KVK_OK;
}

kvk_status kvk_decode_attention_mla(kvk_cache *c, int32_t layer, const void *q_nope,
                                    const void *q_pe, const void *w_uk, const void *w_uv,
                                    float softmax_scale, float *out, int32_t n_splits,
                                    kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->desc.kind != KVK_KIND_MLA) return fail(KVK_ERR_INVALID_ARG, "cache is not MLA");
  if (!q_nope || !q_pe || !w_uk || !w_uv || !out || !aligned16(q_nope) || !aligned16(q_pe) ||
      !aligned16(w_uk) || !aligned16(w_uv) || !aligned16(out))
    return fail(KVK_ERR_INVALID_ARG, "null or misaligned MLA operand");
  if (n_splits < 0 || n_splits > c->max_splits)
    return fail(KVK_ERR_INVALID_ARG, "n_splits %d outside [0, %d]", n_splits, c->max_splits);
  if (!std::isfinite(softmax_scale) || !(softmax_scale > 0.f))
    return fail(KVK_ERR_INVALID_ARG, "softmax scale must be finite and positive");
  const int a = c->src[layer];
  MlaDecodeArgs args;
  args.v = c->mla_view(a);
  args.tmap = c->tmap[a].bytes;
  const int tiles = layer_tiles(c, a);
  if (n_splits == 0) n_splits = auto_splits(c, a);
  n_splits = std::min(std::min(n_splits, tiles), 64);
  args.q_nope = q_nope;
  args.q_pe = q_pe;
  args.w_uk = w_uk;
  args.w_uv = w_uv;
  args.H = c->desc.n_q_heads;
  args.Dn = c->desc.head_dim;
  args.r = c->desc.latent_dim;
  args.sig_log2 = softmax_scale * 1.4426950408889634f;
  args.n_splits = n_splits;
  args.items_per_split = ((tiles + n_splits - 1) / n_splits) * kTile;
  args.qlat = reinterpret_cast<uint16_t *>(c->ws + c->wl.qlat);
  args.partial = reinterpret_cast<float *>(c->ws + c->wl.partial);
  args.olat = reinterpret_cast<float *>(c->ws + c->wl.olat);
  args.out = out;
  args.err = c->err();
  args.wait_limit = c->wait_limit;
  cudaError_t e = launch_mla_decode(args, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "MLA decode launch");
  return KVK_OK;
}


kvk_status kvk_prefill_attention_mla(kvk_cache *c, int32_t layer, const void *q_nope,
                                     const void *q_pe, const void *w_uk, const void *w_uv,
                                     int32_t n_q, float softmax_scale, float *out, void *scratch,
                                     size_t scratch_bytes, kvk_stream stream) {
  kvk_status s = check_prefill_mla(c, layer, n_q);
  if (s) return s;
  if (!q_nope || !q_pe || !w_uk || !w_uv || !out || !aligned16(q_nope) || !aligned16(q_pe) ||
      !aligned16(w_uk) || !aligned16(w_uv) || !aligned16(out))
    return fail(KVK_ERR_INVALID_ARG, "null or misaligned MLA operand");
  if (!std::isfinite(softmax_scale) || !(softmax_scale > 0.f))
    return fail(KVK_ERR_INVALID_ARG, "softmax scale must be finite and positive");
  const MlaPrefillScratch ps = mla_prefill_scratch(c, layer, n_q);
  if (!scratch || (reinterpret_cast<uintptr_t>(scratch) & 255u) || scratch_bytes < ps.total)
    return fail(KVK_ERR_INVALID_ARG, "scratch null, not 256-byte aligned or smaller than %zu bytes",
                ps.total);
  const int a = c->src[layer];
  MlaDecodeArgs args;
  args.v = c->mla_view(a);
  args.v.n_q = n_q;  // query row b n_q + i: query i of sequence b over its causal prefix
  args.tmap = c->tmap[a].bytes;
  args.q_nope = q_nope;
  args.q_pe = q_pe;
  args.w_uk = w_uk;
  args.w_uv = w_uv;
  args.H = c->desc.n_q_heads;
  args.Dn = c->desc.head_dim;
  args.r = c->desc.latent_dim;
  args.sig_log2 = softmax_scale * 1.4426950408889634f;
  args.n_splits = 1;  // every row's prefix in one CTA (rows are plentiful)
  args.items_per_split = layer_tiles(c, a) * kTile;
  args.qlat = reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(scratch) + ps.qlat);
  args.partial = reinterpret_cast<float *>(static_cast<uint8_t *>(scratch) + ps.partial);
  args.olat = nullptr;
  args.out = out;
  args.err = c->err();
  args.wait_limit = c->wait_limit;
  cudaError_t e = launch_mla_decode(args, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "MLA pre-fill launch");
  return KVK_OK;
}

kvk_status kvk_plan_cost(const kvk_model_desc *desc, const kvk_layer_cfg *cfg,
                         double *bits_model, double *bytes_stored, double *rho) {
  kvk_status s = check_desc(desc, false);
  if (s) return s;
  if (!cfg) return fail(KVK_ERR_INVALID_ARG, "null plan");
  for (int l = 0; l < desc->n_layers; ++l) {
    s = check_layer(desc, &cfg[l], l, false);
    if (s) return s;
  }
  const kvk_model_desc &d = *desc;
  const bool mla = d.kind == KVK_KIND_MLA;
  double bits = 0.0, bytes = 0.0;
  for (int l = 0; l < d.n_layers; ++l) {
    const kvk_layer_cfg &a = cfg[l];
    if (a.inherit) continue;  // eq. (cost): inheriting costs nothing
    if (mla) {
      bits += (double)(a.width + d.rope_dim) * a.bits;
      // codes, plus per position the two vectors' metadata: a bf16 scale
      // each (symmetric) or an fp32 scale and zero each (grouped)
      bytes += (double)(a.width + d.rope_dim) * a.bits / 8.0 +
               (a.bits == 16 ? 0.0 : (a.scheme == KVK_QUANT_SYMMETRIC ? 4.0 : 16.0));
    } else {
      bits += 2.0 * d.n_kv_heads * d.head_dim * a.bits;
      double per;
      if (a.bits == 16) {
        per = 4.0 * d.head_dim;
      } else if (a.scheme == KVK_QUANT_SYMMETRIC) {
        // codes + one bf16 scale per row, K and V
        per = 2.0 * d.head_dim * a.bits / 8.0 + 2.0 * 2.0;
      } else {
        // codes + one fp32 (scale, zero) pair per group, K and V
        per = 2.0 * d.head_dim * a.bits / 8.0 + 2.0 * 8.0 * d.head_dim / a.group;
      }
      bytes += per * d.n_kv_heads;
    }
  }
  // eq. (compression): against the bf16 GQA cache; for MLA the conversion
  // width r = n_kv d_h of Appendix B stands for n_kv d_h.
  const double width = mla ? (double)d.latent_dim : (double)d.n_kv_heads * d.head_dim;
  const double c0 = d.n_layers * 2.0 * width * 16.0;
  if (bits_model) *bits_model = bits;
  if (bytes_stored) *bytes_stored = bytes;
  if (rho) *rho = c0 / bits;
  return KVK_OK;
}

kvk_status kvk_cost(const kvk_cache *c, double *bits_model, double *bytes_stored, double *rho) {
  if (!c) return fail(KVK_ERR_INVALID_ARG, "null cache");
  return kvk_plan_cost(&c->desc, c->cfg.data(), bits_model, bytes_stored, rho);
}

kvk_status kvk_export_layer(const kvk_cache *c, int32_t layer, void *k_out, void *v_out,
                            float *k_scale, float *k_zero, float *v_scale, float *v_zero,
                            void *k_residual, kvk_stream stream) {
  kvk_status s = check_layer_index(c, layer);
  if (s) return s;
  if (c->cfg[layer].inherit)
    return fail(KVK_ERR_INHERITED_LAYER, "layer %d inherits layer %d's cache", layer, c->src[layer]);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (c->desc.kind == KVK_KIND_GQA)
    e = launch_gqa_export(c->gqa_view(layer), k_out, v_out, k_scale, k_zero, v_scale, v_zero,
                          k_residual, c->desc.max_ctx, st);
  else
    e = launch_mla_export(c->mla_view(layer), k_out, v_out, k_scale, k_zero, v_scale, v_zero,
                          c->desc.max_ctx, st);
  if (e != cudaSuccess) return cuda_fail(e, "export launch");
  return KVK_OK;
}

kvk_status kvk_get_device_error(kvk_cache *c, kvk_stream stream, int32_t *code) {
  if (!c || !code) return fail(KVK_ERR_INVALID_ARG, "null cache or output");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t h = 0;
  cudaError_t e = cudaMemcpyAsync(&h, c->err(), 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->err(), 0, 4, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "reading the device error word");
  *code = h;
  if (h) return fail(KVK_ERR_DEVICE, "device error word 0x%x", h);
  return KVK_OK;
}

}  // extern "C"
