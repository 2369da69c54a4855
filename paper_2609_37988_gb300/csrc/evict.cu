// evict.cu -- window-vote eviction composed with a compressed GQA cache
// (Sec. 3.3: an evictor runs on the same cache and the reduction factors
// multiply; the evictors sum attention over an observation window of the
// last queries, Appendix "Eviction implementations").
//
// For sequence b, KV head j, the window queries w < n_win (at positions
// p_w = len - n_win + w, each seeing positions 0..p_w) of the G query heads
// of j vote for every position t before the window:
//     vote[t] = sum_{w, h} 2^(x_{w,h}(t) - M_{w,h}) / L_{w,h}
// with x = scale log2(e) <q_{w,h}, k_t> on the dequantised key and (M, L)
// the row's maximum and sum over its causal range.  The budget - n_win
// largest votes (ties: the smaller position) and the window become the
// anchor's kept list for (b, j), sorted.  Four launches: row statistics per
// 128-position tile, their merge per row, the votes, the selection.
//
// The scores run on the CUDA cores in fp32: the evictor runs once per
// prefill, not per decode step, and fp32 dot products keep the votes within
// ~1e-6 of the fp64 definition.
#include <math.h>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {
namespace {

constexpr int kT = kEvictTile;  // positions per CTA (one per thread)
constexpr int kRC = 32;         // query rows per chunk

// Dequantised channel ch of the key of position t from its record (the
// scale word of the symmetric scheme passed in).
__device__ __forceinline__ float key_elem(const GqaView &v, const RecLayout &L, const uint8_t *rec,
                                          int t, uint32_t sc_word, int ch) {
  const int D = v.D;
  if (v.bits == 16) {
    int byte, hi;
    k_pos(ch, 16, D, &byte, &hi);
    return bf16_to_f32(*reinterpret_cast<const uint16_t *>(rec + byte));
  }
  if (v.scheme == kSchemeSym) {
    const int lb = sym_k_bit(ch, v.bits, D);
    const int u = (rec[sym_phys(lb >> 3, t, v.rec_bytes)] >> (lb & 7)) & ((1 << v.bits) - 1);
    const float s = __uint_as_float(sc_word << 16);
    return s * (float)(u - sym_levels(v.bits));
  }
  int byte, hi;
  k_pos(ch, v.bits, D, &byte, &hi);
  const int x = rec[byte];
  const int code = v.bits == 8 ? x : (hi ? x >> 4 : x & 15);
  const float2 m = reinterpret_cast<const float2 *>(rec + L.km_off)[ch / v.group];
  return fmaf((float)code, m.x, m.y);
}

// Shared memory of the two scoring passes: dequantised keys [kT][D + 4]
// (rows padded by 16 bytes: the 16-byte loads of eight consecutive threads,
// one row each, fall in distinct banks), the query rows of one chunk
// [kRC][D], the tile's raw records.
template <int D>
constexpr int evict_kstride() { return D + 4; }
template <int D>
constexpr int evict_smem(int rec_bytes) {
  return kT * evict_kstride<D>() * 4 + kRC * D * 4 + kT * rec_bytes;
}

// VOTES = false: row statistics (M, L) of this tile per window query row;
// VOTES = true: the tile's votes from the merged statistics.
template <int D, bool VOTES>
__global__ void __launch_bounds__(kT) evict_pass_kernel(const EvictArgs a) {
  pdl_wait();
  pdl_trigger();
  const GqaView &v = a.v;
  const int tile = blockIdx.x, j = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int len = v.lens[b];
  if (len <= a.budget) return;  // the sequence keeps every position
  const int P = len - a.n_win;
  const int t0 = tile * kT;
  if (t0 >= (VOTES ? P : len)) return;
  const int unit = b * v.Hkv + j;
  const int R = a.n_win * a.G;
  extern __shared__ __align__(16) uint8_t smem[];
  float *kf = reinterpret_cast<float *>(smem);
  constexpr int KS = evict_kstride<D>();
  float *qs = kf + kT * KS;
  uint8_t *recs = reinterpret_cast<uint8_t *>(qs + kRC * D);

  // the tile's records (contiguous in the slab), then one key row per thread
  const size_t slab = (size_t)b * v.Hkv + j;
  const int nrow = min(kT, len - t0);
  {
    const uint4 *src = reinterpret_cast<const uint4 *>(v.rec + (slab * v.cap + t0) * v.rec_bytes);
    uint4 *dst = reinterpret_cast<uint4 *>(recs);
    const int n = nrow * v.rec_bytes / 16;
    for (int q = tid; q < n; q += kT) dst[q] = src[q];
  }
  __syncthreads();
  const int t = t0 + tid;
  const bool live = tid < nrow;
  if (live) {
    const RecLayout L = rec_layout(v.bits, D, v.group, v.key_axis);
    const uint8_t *rec = recs + tid * v.rec_bytes;
    const uint32_t sw = v.scheme == kSchemeSym ? v.scales[slab * v.cap + t] : 0u;
    for (int ch = 0; ch < D; ++ch) kf[tid * KS + ch] = key_elem(v, L, rec, t, sw, ch);
  }
  float vote = 0.f;
  float2 *stats = a.stats + (size_t)unit * R * a.n_tiles;          // [R][n_tiles]
  const float2 *fin = a.stats + (size_t)gridDim.z * v.Hkv * R * a.n_tiles + (size_t)unit * R;
  for (int rc0 = 0; rc0 < R; rc0 += kRC) {
    const int nr = min(kRC, R - rc0);
    __syncthreads();  // the previous chunk's rows are consumed (and the keys are written)
    for (int e = tid; e < kRC * D; e += kT) {  // rows past the last are zero
      const int rr = e / D, ch = e % D;
      const int r = rc0 + rr, w = r / a.G, h = j * a.G + r % a.G;
      const size_t qi = (((size_t)b * a.n_win + w) * a.Hq + h) * D + ch;
      qs[rr * D + ch] = rr >= nr ? 0.f
                        : a.q_f32 ? static_cast<const float *>(a.q)[qi]
                                  : bf16_to_f32(static_cast<const uint16_t *>(a.q)[qi]);
    }
    __syncthreads();
    // x[rr] = <q_rr, k_t>: eight key channels in registers against every
    // row's eight (broadcast) query channels
    float x[kRC];
#pragma unroll
    for (int rr = 0; rr < kRC; ++rr) x[rr] = 0.f;
    if (live) {
      const float *kr = kf + tid * KS;
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 8) {
        const float4 k0 = *reinterpret_cast<const float4 *>(kr + c0);
        const float4 k1 = *reinterpret_cast<const float4 *>(kr + c0 + 4);
#pragma unroll
        for (int rr = 0; rr < kRC; ++rr) {
          const float4 q0 = *reinterpret_cast<const float4 *>(qs + rr * D + c0);
          const float4 q1 = *reinterpret_cast<const float4 *>(qs + rr * D + c0 + 4);
          float s = x[rr];
          s = fmaf(k0.x, q0.x, s); s = fmaf(k0.y, q0.y, s);
          s = fmaf(k0.z, q0.z, s); s = fmaf(k0.w, q0.w, s);
          s = fmaf(k1.x, q1.x, s); s = fmaf(k1.y, q1.y, s);
          s = fmaf(k1.z, q1.z, s); s = fmaf(k1.w, q1.w, s);
          x[rr] = s;
        }
      }
    }
#pragma unroll
    for (int rr = 0; rr < kRC; ++rr) x[rr] *= a.sig_log2;
    if constexpr (VOTES) {
      // positions before the window: every window query sees them
#pragma unroll
      for (int rr = 0; rr < kRC; ++rr) {
        if (rr >= nr) break;
        const float2 ml = fin[rc0 + rr];
        if (live && t < P && ml.y > 0.f) vote += exp2f(x[rr] - ml.x) / ml.y;
      }
    } else {
      // per row: maximum and sum over this tile's positions in its causal
      // range (block reductions over the 128 threads)
      __shared__ float red[4][kRC];
      __shared__ float rowm[kRC];
#pragma unroll
      for (int rr = 0; rr < kRC; ++rr) {
        const int w = (rc0 + rr) / a.G;
        const bool ok = live && rr < nr && t <= P + w;
        float m = ok ? x[rr] : -INFINITY;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
        if (lane == 0) red[warp][rr] = m;
      }
      __syncthreads();
      if (tid < kRC) rowm[tid] = fmaxf(fmaxf(red[0][tid], red[1][tid]), fmaxf(red[2][tid], red[3][tid]));
      __syncthreads();
#pragma unroll
      for (int rr = 0; rr < kRC; ++rr) {
        const int w = (rc0 + rr) / a.G;
        const bool ok = live && rr < nr && t <= P + w;
        const float m = rowm[rr];
        float l = (ok && m != -INFINITY) ? exp2f(x[rr] - m) : 0.f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
        if (lane == 0) red[warp][rr] = l;
      }
      __syncthreads();
      if (tid < nr)
        stats[(size_t)(rc0 + tid) * a.n_tiles + tile] =
            make_float2(rowm[tid], red[0][tid] + red[1][tid] + red[2][tid] + red[3][tid]);
    }
  }
  if constexpr (VOTES) {
    if (live && t < P) a.votes[(size_t)unit * v.cap + t] = vote;
  }
}

// Merged (M, L) of every window query row over its tiles.
__global__ void __launch_bounds__(128) evict_merge_stats_kernel(const EvictArgs a) {
  pdl_wait();
  pdl_trigger();
  const GqaView &v = a.v;
  const int R = a.n_win * a.G;
  const int units = v.B * v.Hkv;
  const int id = blockIdx.x * blockDim.x + threadIdx.x;
  if (id >= units * R) return;
  const int unit = id / R, r = id % R, b = unit / v.Hkv;
  const int len = v.lens[b];
  if (len <= a.budget) return;
  const int nt = min((len + kT - 1) / kT, a.n_tiles);
  const float2 *st = a.stats + ((size_t)unit * R + r) * a.n_tiles;
  float M = -INFINITY;
  for (int i = 0; i < nt; ++i) M = fmaxf(M, st[i].x);
  float L = 0.f;
  if (M != -INFINITY)
    for (int i = 0; i < nt; ++i)
      if (st[i].x != -INFINITY) L += st[i].y * exp2f(st[i].x - M);
  float2 *fin = a.stats + (size_t)units * R * a.n_tiles;
  fin[id] = make_float2(M, L);
}

// Block-wide exclusive scan of one int per thread (1024 threads); returns the
// thread's exclusive prefix and writes the block total to *total.
__device__ __forceinline__ int block_scan_1024(int x, int *wsum, int *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int inc = x;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += y;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    int s = wsum[lane];
    int si = s;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, si, off);
      if (lane >= off) si += y;
    }
    wsum[lane] = si - s;  // exclusive prefix of the warp totals
    if (lane == 31) *total = si;
  }
  __syncthreads();
  const int r = wsum[warp] + inc - x;
  __syncthreads();  // wsum is reused by the next scan
  return r;
}

// Kept list of one (sequence, kv head): the budget - n_win largest votes by
// a radix select on their bit patterns (votes are >= 0, so the patterns
// order as the values), then the chosen positions in increasing order and
// the window.
__global__ void __launch_bounds__(1024) evict_select_kernel(const EvictArgs a) {
  pdl_wait();
  pdl_trigger();
  const GqaView &v = a.v;
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int unit = b * v.Hkv + j;
  const int len = v.lens[b];
  int32_t *out = v.kept_idx + (size_t)unit * v.kept_cap;
  if (len <= a.budget) {  // everything is kept
    for (int t = tid; t < len; t += 1024) out[t] = t;
    if (tid == 0) v.kept_n[unit] = len;
    return;
  }
  const int P = len - a.n_win, k = a.budget - a.n_win;
  const uint32_t *key = reinterpret_cast<const uint32_t *>(a.votes + (size_t)unit * v.cap);
  __shared__ int hist[256];
  __shared__ uint32_t s_prefix;
  __shared__ int s_rank;
  __shared__ int wsum[32];
  __shared__ int s_total;
  uint32_t prefix = 0, mask = 0;
  int rank = k;  // 1-based rank (from the top) of the wanted key among the matches
  if (k > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int d = tid; d < 256; d += 1024) hist[d] = 0;
      __syncthreads();
      for (int t = tid; t < P; t += 1024) {
        const uint32_t kk = key[t];
        if ((kk & mask) == prefix) atomicAdd(&hist[(kk >> shift) & 255], 1);
      }
      __syncthreads();
      if (tid == 0) {
        int cum = 0, sel = 0;
        for (int d = 255; d >= 0; --d) {
          if (cum + hist[d] >= rank) { sel = d; break; }
          cum += hist[d];
        }
        s_prefix = prefix | ((uint32_t)sel << shift);
        s_rank = rank - cum;
      }
      __syncthreads();
      prefix = s_prefix;
      rank = s_rank;
      mask |= 0xFFu << shift;
      __syncthreads();
    }
  }
  // positions above the threshold key, and the first `rank` equal to it
  const uint32_t theta = prefix;
  int eq_carry = 0, out_carry = 0;
  for (int c0 = 0; c0 < P && k > 0; c0 += 1024) {
    const int t = c0 + tid;
    const uint32_t kk = t < P ? key[t] : 0u;
    const bool gt = t < P && kk > theta, eq = t < P && kk == theta;
    const int eq_before = eq_carry + block_scan_1024(eq ? 1 : 0, wsum, &s_total);
    const int eq_tot = s_total;
    const bool take = gt || (eq && eq_before < rank);
    const int pos = out_carry + block_scan_1024(take ? 1 : 0, wsum, &s_total);
    const int take_tot = s_total;
    if (take && pos < k) out[pos] = t;
    eq_carry += eq_tot;
    out_carry += take_tot;
  }
  for (int i = tid; i < a.n_win; i += 1024) out[k + i] = P + i;
  if (tid == 0) v.kept_n[unit] = a.budget;
}

template <int D>
cudaError_t launch_evict_d(const EvictArgs &a, cudaStream_t st) {
  const int smem = evict_smem<D>(a.v.rec_bytes);
  cudaError_t e = cudaFuncSetAttribute(evict_pass_kernel<D, false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(evict_pass_kernel<D, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem);
  if (e != cudaSuccess) return e;
  const dim3 grid(a.n_tiles, a.v.Hkv, a.v.B);
  e = launch_pdl(evict_pass_kernel<D, false>, grid, dim3(kT), smem, st, a);
  if (e == cudaSuccess) {
    const int rows = a.v.B * a.v.Hkv * a.n_win * a.G;
    e = launch_pdl(evict_merge_stats_kernel, dim3((rows + 127) / 128), dim3(128), 0, st, a);
  }
  if (e == cudaSuccess) e = launch_pdl(evict_pass_kernel<D, true>, grid, dim3(kT), smem, st, a);
  if (e == cudaSuccess)
    e = launch_pdl(evict_select_kernel, dim3(a.v.Hkv, a.v.B), dim3(1024), 0, st, a);
  return e;
}

}  // namespace

cudaError_t launch_gqa_evict(const EvictArgs &a, cudaStream_t st) {
  switch (a.v.D) {
    case 128: return launch_evict_d<128>(a, st);
    case 64: return launch_evict_d<64>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace kvk
