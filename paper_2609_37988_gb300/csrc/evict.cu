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
// anchor's kept list for (b, j), sorted.  Four launches: scores and row
// statistics per 128-position tile, the statistics merged per row, the votes
// (streaming the stored scores), the selection.
//
// The scores run on the CUDA cores in fp32: the evictor runs once per
// prefill, not per decode step, and fp32 dot products keep the votes within
// ~1e-6 of the fp64 definition.  Storing the scores (R x 4 bytes per
// position) costs less than computing them twice (R x D products).
#include <math.h>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {
namespace {

constexpr int kT = kEvictTile;  // positions per scoring tile

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

// Scores of one 128-position tile against every window query row of its
// (sequence, KV head): X[r][t] = sig_log2 <q_r, k_t>, an fp32 contraction of
// [R x D] by [D x 128] on the CUDA cores, register-tiled: thread (tx, ty)
// holds rows ty*4 .. ty*4+3 of a 64-row chunk against positions tx*4 ..
// tx*4+3 and 64 + tx*4 .. 64 + tx*4+3 of the tile (32 products per pair of
// key loads and one query load).  The dequantised keys sit channel-major in
// shared memory [D][128], the chunk's query rows [D][64].  Each row's
// (max, sum 2^(x - max)) over the tile's positions in its causal range goes
// to the per-tile statistics, and the scores of the positions before the
// window go to the score buffer, which the vote pass streams instead of
// recomputing them.
constexpr int kRC = 64;        // window query rows per chunk
constexpr int kThreads = 256;  // 16 position groups x 16 row groups

template <int D>
constexpr int evict_smem() {
  return (D * kT + D * kRC) * 4;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2) evict_scores_kernel(const EvictArgs a) {
  pdl_wait();
  const GqaView &v = a.v;
  const int tile = blockIdx.x, j = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x;
  const int len = v.lens[b];
  const int t0 = tile * kT;
  if (len <= a.budget || t0 >= len) {  // the sequence keeps everything / tile past the end
    pdl_trigger();
    return;
  }
  const int P = len - a.n_win;
  const int unit = b * v.Hkv + j;
  const int R = a.n_win * a.G;
  extern __shared__ __align__(16) float evict_sm[];
  float *kt = evict_sm;          // [D][kT]
  float *qt = evict_sm + D * kT; // [D][kRC]
  const size_t slab = (size_t)b * v.Hkv + j;
  {
    // two threads per position, half of the channels each
    const int p = tid & (kT - 1), half = tid / kT;
    const int t = t0 + p;
    const bool live = t < len;
    const RecLayout L = rec_layout(v.bits, D, v.group, v.key_axis);
    const uint8_t *rec = v.rec + (slab * v.cap + (live ? t : t0)) * v.rec_bytes;
    const uint32_t sw = (live && v.scheme == kSchemeSym) ? v.scales[slab * v.cap + t] : 0u;
    for (int ch = half * (D / 2); ch < (half + 1) * (D / 2); ++ch)
      kt[ch * kT + p] = live ? key_elem(v, L, rec, t, sw, ch) : 0.f;
  }
  const int tx = tid & 15, ty = tid >> 4;
  float2 *stats = a.stats + (size_t)unit * R * a.n_tiles;
  float *scores = a.scores + (size_t)unit * R * a.sc_stride;
  for (int rc0 = 0; rc0 < R; rc0 += kRC) {
    __syncthreads();  // keys written; the previous chunk's query rows consumed
    // the chunk's query rows, channel-major (rows past R are zero)
    for (int e = tid; e < kRC * (D / 4); e += kThreads) {
      const int rr = e & (kRC - 1), c4 = e / kRC;
      const int r = rc0 + rr;
      float4 x4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (r < R) {
        const int w = r / a.G, h = j * a.G + r % a.G;
        const size_t qi = (((size_t)b * a.n_win + w) * a.Hq + h) * D + 4 * c4;
        if (a.q_f32) {
          x4 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + qi);
        } else {
          const uint2 u = *reinterpret_cast<const uint2 *>(static_cast<const uint16_t *>(a.q) + qi);
          x4 = make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                           __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
        }
      }
      qt[(4 * c4 + 0) * kRC + rr] = x4.x;
      qt[(4 * c4 + 1) * kRC + rr] = x4.y;
      qt[(4 * c4 + 2) * kRC + rr] = x4.z;
      qt[(4 * c4 + 3) * kRC + rr] = x4.w;
    }
    __syncthreads();
    float acc[4][8];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[i][c] = 0.f;
#pragma unroll 4
    for (int k = 0; k < D; ++k) {
      const float4 k0 = *reinterpret_cast<const float4 *>(kt + k * kT + tx * 4);
      const float4 k1 = *reinterpret_cast<const float4 *>(kt + k * kT + 64 + tx * 4);
      const float4 q4 = *reinterpret_cast<const float4 *>(qt + k * kRC + ty * 4);
      const float kk[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
      const float qq[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int c = 0; c < 8; ++c) acc[i][c] = fmaf(qq[i], kk[c], acc[i][c]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int r = rc0 + ty * 4 + i;
      const int last = P + r / a.G;  // the last position row r sees
      float m = -INFINITY;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const int t = t0 + (c >> 2) * 64 + tx * 4 + (c & 3);
        acc[i][c] *= a.sig_log2;
        if (t <= last) m = fmaxf(m, acc[i][c]);
      }
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
      float l = 0.f;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const int t = t0 + (c >> 2) * 64 + tx * 4 + (c & 3);
        if (t <= last) l += exp2f(acc[i][c] - m);  // m is finite: this row sees t
      }
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
      if (r < R) {
        if (tx == 0) stats[(size_t)r * a.n_tiles + tile] = make_float2(m, l);
        float *row = scores + (size_t)r * a.sc_stride + t0 + tx * 4;
        if (t0 + tx * 4 < P) *reinterpret_cast<float4 *>(row) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        if (t0 + 64 + tx * 4 < P)
          *reinterpret_cast<float4 *>(row + 64) = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
      }
    }
  }
  pdl_trigger();
}

// Votes of 256 positions before the window: sum over the rows of
// 2^(x - M - log2 L) with the rows' merged statistics, streaming the scores.
constexpr int kVoteT = 256;
constexpr int kVoteRows = 1024;  // merged statistics staged per round

__global__ void __launch_bounds__(kVoteT) evict_votes_kernel(const EvictArgs a) {
  pdl_wait();
  const GqaView &v = a.v;
  const int j = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int len = v.lens[b];
  const int P = len - a.n_win;
  const int t = blockIdx.x * kVoteT + tid;
  if (len <= a.budget || (int)blockIdx.x * kVoteT >= P) {
    pdl_trigger();
    return;
  }
  const int unit = b * v.Hkv + j;
  const int R = a.n_win * a.G;
  const float2 *fin = a.stats + (size_t)gridDim.z * v.Hkv * R * a.n_tiles + (size_t)unit * R;
  const float *x = a.scores + (size_t)unit * R * a.sc_stride + t;
  __shared__ float norm[kVoteRows];
  float vote = 0.f;
  for (int r0 = 0; r0 < R; r0 += kVoteRows) {
    const int nr = min(kVoteRows, R - r0);
    __syncthreads();
    for (int i = tid; i < nr; i += kVoteT) {
      const float2 ml = fin[r0 + i];
      norm[i] = ml.x + log2f(ml.y);
    }
    __syncthreads();
    if (t < P) {
#pragma unroll 8
      for (int r = 0; r < nr; ++r) vote += exp2f(x[(size_t)(r0 + r) * a.sc_stride] - norm[r]);
    }
  }
  if (t < P) a.votes[(size_t)unit * v.cap + t] = vote;
  pdl_trigger();
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
  constexpr int smem = evict_smem<D>();
  cudaError_t e = cudaFuncSetAttribute(evict_scores_kernel<D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(evict_scores_kernel<D>, dim3(a.n_tiles, a.v.Hkv, a.v.B), dim3(kThreads), smem, st, a);
  if (e == cudaSuccess) {
    const int rows = a.v.B * a.v.Hkv * a.n_win * a.G;
    e = launch_pdl(evict_merge_stats_kernel, dim3((rows + 127) / 128), dim3(128), 0, st, a);
  }
  if (e == cudaSuccess)
    e = launch_pdl(evict_votes_kernel, dim3((a.v.cap + kVoteT - 1) / kVoteT, a.v.Hkv, a.v.B),
                   dim3(kVoteT), 0, st, a);
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
