// evict.cu -- window-vote eviction composed with a compressed GQA cache
// (Sec. 3.4: an evictor runs on the same cache and the reduction factors
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

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"
#include "umma.cuh"
#include "window_tc.cuh"

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
  const float2 *fin = a.fin + (size_t)unit * R;
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
// One warp per (unit, row): lanes stride over the row's tile entries
// (coalesced), then warp reductions of the maximum and of the rescaled sums.
constexpr int kMergeWarps = 8;
__global__ void __launch_bounds__(32 * kMergeWarps) evict_merge_stats_kernel(const EvictArgs a) {
  pdl_wait();
  pdl_trigger();
  const GqaView &v = a.v;
  const int R = a.n_win * a.G;
  const int units = v.B * v.Hkv;
  const int id = blockIdx.x * kMergeWarps + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (id >= units * R) return;
  const int unit = id / R, r = id % R, b = unit / v.Hkv;
  const int len = v.lens[b];
  if (len <= a.budget) return;
  const int nt = min((len + kT - 1) / kT, a.n_tiles) * a.stat_sub;
  const float2 *st = a.stats + ((size_t)unit * R + r) * a.n_tiles * a.stat_sub;
  float M = -INFINITY;
  for (int i = lane; i < nt; i += 32) M = fmaxf(M, st[i].x);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float L = 0.f;
  if (M != -INFINITY)
    for (int i = lane; i < nt; i += 32) {
      const float2 e = st[i];
      if (e.x != -INFINITY) L += e.y * exp2f(e.x - M);
    }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
  if (lane == 0) a.fin[id] = make_float2(M, L);
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

// keys t0 .. t0+7 (zero past n); t0 is a multiple of 8 and the array
// 32-byte aligned
__device__ __forceinline__ void load8(const uint32_t *key, int t0, int n, uint32_t (&kk)[8]) {
  if (t0 + 8 <= n) {
    const uint4 u0 = *reinterpret_cast<const uint4 *>(key + t0);
    const uint4 u1 = *reinterpret_cast<const uint4 *>(key + t0 + 4);
    kk[0] = u0.x; kk[1] = u0.y; kk[2] = u0.z; kk[3] = u0.w;
    kk[4] = u1.x; kk[5] = u1.y; kk[6] = u1.z; kk[7] = u1.w;
  } else {
#pragma unroll
    for (int u = 0; u < 8; ++u) kk[u] = t0 + u < n ? key[t0 + u] : 0u;
  }
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
      // votes of similar size share their leading bytes, so most lanes of a
      // warp hit the bin of lane 0: those are counted with one atomic, the
      // others one by one.  Eight consecutive votes per thread per round
      // keep eight loads in flight.
      for (int c0 = 0; c0 < P; c0 += 8 * 1024) {
        uint32_t kk[8];
        load8(key, c0 + 8 * tid, P, kk);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const bool hit = c0 + 8 * tid + u < P && (kk[u] & mask) == prefix;
          const uint32_t bin = hit ? (kk[u] >> shift) & 255 : 256u;
          const uint32_t bin0 = __shfl_sync(0xffffffffu, bin, 0);
          const uint32_t same = __ballot_sync(0xffffffffu, bin == bin0);
          if (bin == bin0) {
            if ((threadIdx.x & 31) == 0 && bin0 < 256u) atomicAdd(&hist[bin0], __popc(same));
          } else if (hit) {
            atomicAdd(&hist[bin], 1);
          }
        }
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
  // (one scan of the packed counts: greater in the high half, equal in the
  // low half; a taken position's slot is the greater ones before it plus
  // the equal ones before it, at most `rank`)
  const uint32_t theta = prefix;
  int gt_carry = 0, eq_carry = 0;
  for (int c0 = 0; c0 < P && k > 0; c0 += 8 * 1024) {
    const int tb = c0 + 8 * tid;  // this thread's eight consecutive positions
    uint32_t kk[8];
    load8(key, tb, P, kk);
    int ngt = 0, neq = 0;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      ngt += tb + u < P && kk[u] > theta;
      neq += tb + u < P && kk[u] == theta;
    }
    const int ex = block_scan_1024((ngt << 16) | neq, wsum, &s_total);
    const int tot = s_total;
    int gt_before = gt_carry + (ex >> 16), eq_before = eq_carry + (ex & 0xFFFF);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const bool gt = tb + u < P && kk[u] > theta, eq = tb + u < P && kk[u] == theta;
      const int pos = gt_before + min(eq_before, rank);
      if ((gt || (eq && eq_before < rank)) && pos < k) out[pos] = tb + u;
      gt_before += gt;
      eq_before += eq;
    }
    gt_carry += tot >> 16;
    eq_carry += tot & 0xFFFF;
  }
  for (int i = tid; i < a.n_win; i += 1024) out[k + i] = P + i;
  if (tid == 0) v.kept_n[unit] = a.budget;
}

// ---------------------------------------------------------------------------
// Tensor-core scoring (tcgen05; head_dim 128, at most 256 window rows).
//
// The scores of a 128-position tile are one UMMA chain over K = 128
// channels.  The dequantised keys, split into bf16 hi + lo, and the window
// query rows (split likewise when they arrive in fp32; bf16 queries have no
// lo part) sit in shared memory in the K-major 128-byte-swizzled layout
// (two 64-channel boxes of 128-byte rows, 16-byte chunk c of row r stored at
// chunk c ^ (r & 7)).  hi*hi + hi*lo + lo*hi keeps ~16 significant bits of
// each factor (the dropped lo*lo term is below 2^-16 of the product); the
// tensor cores accumulate in fp32 in TMEM.
//  * statistics pass: A = query rows (M = 128 per chunk), B = keys (N = 128
//    positions): TMEM lane = row, so each thread reduces its row over the
//    positions without shuffles (two entries per tile and row, one per
//    64-position half);
//  * vote pass: A = keys (M = 128 positions), B = query rows (N = R rounded
//    up to 16): TMEM lane = position, so each thread sums its position's
//    weights over the rows.
// The vote pass recomputes the scores: on the tensor cores that is cheaper
// than a round trip through HBM.  A CTA (one per SM) walks a contiguous range
// of (unit, tile) items; with two key stages the keys of the next item are
// dequantised while the tensor cores run the current one, and the epilogue
// of an item reads one TMEM buffer while the next item's chain fills the
// other.  Query rows past R are zero; in the statistics pass the last row
// chunk may read rows past the query buffer (lanes that are never used).
constexpr int kTcWorkers = 512;              // dequantise and run the epilogues
constexpr int kTcThreads = kTcWorkers + 32;  // + the MMA warp
static_assert(kEvictStatSub == kTcWorkers / 128, "one statistics entry per worker column slice");

struct TcPlan {
  int items_per_cta, n_items;
  int R16, nch, q_lo, k_lo, nst, nstg, fmt;  // nst key stages, nstg staging buffers
  int kb_nch, kb_stride, stg_bytes;  // staged 16-byte chunks per position, their stride
  int nc_magic;                      // ceil(2^16 / kb_nch): e / kb_nch = (e nc_magic) >> 16 here
  int stage, off_q, off_ql, off_k, off_stg, off_norm, off_pv, off_bar, smem;
};

template <bool VOTES>
__global__ void __launch_bounds__(kTcThreads, 1) evict_tc_kernel(const EvictArgs a, const TcPlan p) {
  extern __shared__ uint8_t evict_tc_raw[];
  uint8_t *sm = evict_tc_raw + ((1024u - (smem_u32(evict_tc_raw) & 1023u)) & 1023u);
  // bar[0], [1]: the chain of TMEM buffer 0 / 1 done; [2]: drain; [3], [4]:
  // the keys of an even / odd item staged (one arrival per worker warp)
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm + p.off_bar);
  uint32_t *tbase = reinterpret_cast<uint32_t *>(sm + p.off_bar + 40);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + p.off_bar + 44);
  float *norm = reinterpret_cast<float *>(sm + p.off_norm);
  float *pv = reinterpret_cast<float *>(sm + p.off_pv);
  uint8_t *qh = sm + p.off_q, *ql = sm + p.off_ql;
  const GqaView &v = a.v;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int R = a.n_win * a.G;
  constexpr uint32_t kLimit = 1u << 22;
  constexpr uint32_t kSleepyLimit = 1u << 20;  // polls of up to 2 us each
  constexpr int D = 128;
  constexpr int KBOX = 128 * 128;  // bytes of one 64-channel box of a 128-row key tile

  if (tid == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(&bar[i], i < 3 ? 1 : kTcWorkers / 32);
    *abort_flag = 0;
    fence_mbar_init();
  }
  pdl_wait();  // the cache, lengths and (vote pass) merged statistics are complete
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tbase)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tbase;

  const int it0 = blockIdx.x * p.items_per_cta;
  const int it1 = min(it0 + p.items_per_cta, p.n_items);
  // worker warp w reads TMEM lanes 32 (w % 4) .. + 31; slice = w / 4
  const int quarter = warp & 3, slice = warp >> 2;
  const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
  uint32_t phases = 0u;  // bit tb: parity of TMEM buffer tb's next completion
  bool failed = false;

  const int gshift = v.group == 64 ? 6 : 5;  // grouped layers: groups of 32 or 64 channels
  // rows of this thread in the statistics epilogue, divided by G (the row's
  // window query), once
  int rdiv[2];
#pragma unroll
  for (int c = 0; c < 2; ++c) rdiv[c] = (128 * c + 32 * quarter + lane) / a.G;
  // (unit, tile) of item `it` and the unit's length, advanced without divisions
  struct Cursor {
    int it, unit, tile, len;
  };
  const int units = v.B * v.Hkv;
  auto at = [&](int it) {
    Cursor c;
    c.it = it;
    c.unit = it / a.n_tiles;
    c.tile = it - c.unit * a.n_tiles;
    c.len = c.unit < units ? v.lens[c.unit / v.Hkv] : 0;
    return c;
  };
  auto next_valid = [&](Cursor c) {  // c or the first valid item after it (c.it == it1: none)
    while (c.it < it1) {
      if (c.len > a.budget && c.tile * kT < (VOTES ? c.len - a.n_win : c.len)) break;
      // an invalid item has no valid successor in its unit: on to the next unit
      c.it += a.n_tiles - c.tile;
      c.tile = 0;
      ++c.unit;
      c.len = c.unit < units ? v.lens[c.unit / v.Hkv] : 0;
    }
    c.it = min(c.it, it1);
    return c;
  };
  auto after = [&](Cursor c) {  // the item after c
    ++c.it;
    if (++c.tile == a.n_tiles) {
      c.tile = 0;
      ++c.unit;
      c.len = c.unit < units ? v.lens[c.unit / v.Hkv] : 0;
    }
    return c;
  };

  // query rows of `unit` (and, for the votes, the rows' log-normalisers;
  // +inf for the padding rows, whose weights are then 0)
  auto load_q = [&](int unit) {
    const int b = unit / v.Hkv, j = unit % v.Hkv;
    const int box = p.R16 * 128;
    for (int e = tid; e < p.R16 * (D / 8); e += kTcWorkers) {
      const int r = e >> 4, c8 = e & 15;
      float x[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] = 0.f;
      if (r < R) {
        const int w = r / a.G, h = j * a.G + r % a.G;
        const size_t qi = (((size_t)b * a.n_win + w) * a.Hq + h) * D + 8 * c8;
        if (a.q_f32) {
          const float4 u0 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + qi);
          const float4 u1 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + qi + 4);
          x[0] = u0.x; x[1] = u0.y; x[2] = u0.z; x[3] = u0.w;
          x[4] = u1.x; x[5] = u1.y; x[6] = u1.z; x[7] = u1.w;
        } else {
          const uint4 u = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.q) + qi);
          const uint32_t ww[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(ww[i] << 16);
            x[2 * i + 1] = __uint_as_float(ww[i] & 0xFFFF0000u);
          }
        }
      }
      put8(qh, ql, p.q_lo != 0, r, 8 * c8, box, x);
    }
    if constexpr (VOTES) {
      for (int r = tid; r < p.R16; r += kTcWorkers) {
        if (r < R) {
          const float2 f = a.fin[(size_t)unit * R + r];
          norm[r] = f.x + log2f(f.y);
        } else {
          norm[r] = INFINITY;
        }
      }
    }
    fence_proxy_async();
    workers_sync<kTcWorkers>();
  };

  // asynchronous copy of the K bundles of item `it` (K section in logical
  // order, then the group metadata or the symmetric scale word) into staging
  // buffer g; one commit group per call
  auto stage_copy = [&](const Cursor &cu, int g) {
    const int unit = cu.unit, t0 = cu.tile * kT, len = cu.len;
    uint8_t *dst0 = sm + p.off_stg + g * p.stg_bytes;
    const int NC = p.kb_nch;
    const int ks16 = TcFmtKs16(p.fmt);
    const bool sym = p.fmt >= kFmtS8;
    const int nrec = v.rec_bytes >> 4;
    const int km = ks16 * 32;  // grouped: key metadata follows the K and V sections
    const uint8_t *base = v.rec + (size_t)unit * v.cap * v.rec_bytes;
    for (int e = tid; e < kT * NC; e += kTcWorkers) {
      const int pos = (e * p.nc_magic) >> 16, c = e - pos * NC;
      const int t = t0 + pos;
      const bool ok = t < len;
      const int so = sym ? 16 * ((c + sym_rot(t, nrec)) & (nrec - 1)) : c < ks16 ? 16 * c : km + 16 * (c - ks16);
      cp_async16(dst0 + pos * p.kb_stride + 16 * c, base + (size_t)(ok ? t : t0) * v.rec_bytes + so, ok);
    }
    if (sym)
      for (int pos = tid; pos < kT; pos += kTcWorkers) {
        const int t = t0 + pos;
        const bool ok = t < len;
        cp_async4(dst0 + pos * p.kb_stride + 16 * ks16,
                  v.scales + (size_t)unit * v.cap + (ok ? t : t0), ok);
      }
    cp_async_commit();
  };

  // dequantised keys of the item staged in buffer g into key stage s
  auto dequant = [&](int g, int s) {
    const int pidx = tid & 127, hf = tid >> 7;  // position, channel quarter
    const uint8_t *bundle = sm + p.off_stg + g * p.stg_bytes + pidx * p.kb_stride;
    uint8_t *kh = sm + p.off_k + s * p.stage, *kl = kh + 2 * KBOX;
    switch (p.fmt) {
      case kFmtBf16: tc_dequant<kFmtBf16>(bundle, bundle + TcFmtKs16(kFmtBf16) * 16, pidx, hf, gshift, kh, kl); break;
      case kFmtG8: tc_dequant<kFmtG8>(bundle, bundle + TcFmtKs16(kFmtG8) * 16, pidx, hf, gshift, kh, kl); break;
      case kFmtG4: tc_dequant<kFmtG4>(bundle, bundle + TcFmtKs16(kFmtG4) * 16, pidx, hf, gshift, kh, kl); break;
      case kFmtS8: tc_dequant<kFmtS8>(bundle, bundle + TcFmtKs16(kFmtS8) * 16, pidx, hf, gshift, kh, kl); break;
      case kFmtS4: tc_dequant<kFmtS4>(bundle, bundle + TcFmtKs16(kFmtS4) * 16, pidx, hf, gshift, kh, kl); break;
      default: tc_dequant<kFmtS2>(bundle, bundle + TcFmtKs16(kFmtS2) * 16, pidx, hf, gshift, kh, kl); break;
    }
  };

  // one MMA chain for the tile in key stage s into TMEM buffer tb (thread 0)
  auto issue = [&](int s, int tb) {
    tc_fence_after();
    const uint32_t kh = smem_u32(sm + p.off_k + s * p.stage), kl = kh + 2 * KBOX;
    const uint32_t qa = smem_u32(qh), qb = smem_u32(ql);
    const uint32_t qbox = (uint32_t)p.R16 * 128;
    const uint32_t d0 = tmem + 256u * tb;
    auto dsc = [](uint32_t addr) { return umma_desc(addr, 16, 1024, 2); };
    if constexpr (!VOTES) {
      const uint32_t id = umma_idesc(128, 128, false, false);
      for (int c = 0; c < p.nch; ++c) {
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const uint32_t ko = (ks >> 2) * KBOX + (ks & 3) * 32;
          const uint32_t qo = (ks >> 2) * qbox + c * 16384 + (ks & 3) * 32;
          umma_f16(d0 + 128 * c, dsc(qa + qo), dsc(kh + ko), id, ks > 0);
          if (p.k_lo) umma_f16(d0 + 128 * c, dsc(qa + qo), dsc(kl + ko), id, true);
          if (p.q_lo) umma_f16(d0 + 128 * c, dsc(qb + qo), dsc(kh + ko), id, true);
        }
      }
    } else {
      const uint32_t id = umma_idesc(128, p.R16, false, false);
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
        const uint32_t ko = (ks >> 2) * KBOX + (ks & 3) * 32;
        const uint32_t qo = (ks >> 2) * qbox + (ks & 3) * 32;
        umma_f16(d0, dsc(kh + ko), dsc(qa + qo), id, ks > 0);
        if (p.k_lo) umma_f16(d0, dsc(kl + ko), dsc(qa + qo), id, true);
        if (p.q_lo) umma_f16(d0, dsc(kh + ko), dsc(qb + qo), id, true);
      }
    }
    umma_commit(&bar[tb]);
  };

  // epilogue of item `it` from TMEM buffer tb
  auto epilogue = [&](const Cursor &cu, int tb) {
    const int unit = cu.unit, tile = cu.tile, len = cu.len;
    const int P = len - a.n_win;
    const int t0 = tile * kT;
    const float sg = a.sig_log2;
    if constexpr (!VOTES) {
      float2 *st = a.stats + (size_t)unit * R * (kEvictStatSub * a.n_tiles);
      for (int c = 0; c < p.nch; ++c) {
        if (128 * c + 32 * quarter >= R) continue;  // the warp's rows are all padding
        const int r = 128 * c + 32 * quarter + lane;
        const int last = P + (c == 0 ? rdiv[0] : rdiv[1]);  // the last position row r sees
        float y[32];
        const uint32_t ta = tmem + 256u * tb + 128 * c + 32 * slice + lane_off;
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          float z[16];
          tmem_ld16(ta + 16 * q, z);
#pragma unroll
          for (int i = 0; i < 16; ++i) y[16 * q + i] = z[i];
        }
        const int tb0 = t0 + 32 * slice;
        const int nv = min(32, last - tb0 + 1);  // positions of the slice row r sees
        float m = -INFINITY, l = 0.f;
        if (nv >= 32) {  // four independent chains each
          float mm[4] = {y[0], y[1], y[2], y[3]}, ll[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int i = 4; i < 32; ++i) mm[i & 3] = fmaxf(mm[i & 3], y[i]);
          const float ms = fmaxf(fmaxf(mm[0], mm[1]), fmaxf(mm[2], mm[3])) * sg;
#pragma unroll
          for (int i = 0; i < 32; ++i) ll[i & 3] += fast_exp2(fmaf(y[i], sg, -ms));
          m = ms;
          l = (ll[0] + ll[1]) + (ll[2] + ll[3]);
        } else if (nv > 0) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nv) m = fmaxf(m, y[i]);
          const float ms = m * sg;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nv) l += fast_exp2(fmaf(y[i], sg, -ms));
          m = ms;
        }
        if (r < R)
          st[(size_t)r * (kEvictStatSub * a.n_tiles) + kEvictStatSub * tile + slice] = make_float2(m, l);
      }
    } else {
      const int pos = 32 * quarter + lane, t = t0 + pos;
      const int n16 = p.R16 / 16, per = (n16 + 3) / 4;
      const int bk0 = min(n16, slice * per), bk1 = min(n16, bk0 + per);
      float vv[4] = {0.f, 0.f, 0.f, 0.f};  // four independent chains
      for (int bk = bk0; bk < bk1; ++bk) {
        float y[16];
        tmem_ld16(tmem + 256u * tb + 16 * bk + lane_off, y);
        const float4 *nr = reinterpret_cast<const float4 *>(norm + 16 * bk);
#pragma unroll
        for (int i4 = 0; i4 < 4; ++i4) {
          const float4 c4 = nr[i4];
          vv[0] += fast_exp2(fmaf(y[4 * i4], sg, -c4.x));
          vv[1] += fast_exp2(fmaf(y[4 * i4 + 1], sg, -c4.y));
          vv[2] += fast_exp2(fmaf(y[4 * i4 + 2], sg, -c4.z));
          vv[3] += fast_exp2(fmaf(y[4 * i4 + 3], sg, -c4.w));
        }
      }
      const float vote = (vv[0] + vv[1]) + (vv[2] + vv[3]);
      if (slice) pv[(slice - 1) * 128 + pos] = vote;
      workers_sync<kTcWorkers>();
      if (!slice && t < P) a.votes[(size_t)unit * v.cap + t] = vote + pv[pos] + pv[128 + pos] + pv[256 + pos];
    }
  };

  // waits for the chain in TMEM buffer tb, runs its epilogue, frees the buffers
  auto finish = [&](const Cursor &it, int tb) -> bool {
    const bool ok = mbar_wait_sleepy(&bar[tb], (phases >> tb) & 1u, kSleepyLimit, abort_flag, 2000);
    phases ^= 1u << tb;
    if (workers_sync_or<kTcWorkers>(!ok)) return false;
    tc_fence_after();
    epilogue(it, tb);
    tc_fence_before();
    workers_sync<kTcWorkers>();
    return true;
  };

  if (warp == kTcWorkers / 32) {
    // ======================= MMA warp =====================================
    // the same item sequence as the workers; each chain once its keys are staged
    int kk = 0;
    for (Cursor cu = next_valid(at(it0)); cu.it < it1; cu = next_valid(after(cu)), ++kk) {
      if (!mbar_wait_sleepy(&bar[3 + (kk & 1)], (kk >> 1) & 1, kSleepyLimit, abort_flag, 2000)) {
        if (lane == 0) *abort_flag = 1;
        break;
      }
      if (lane == 0) issue(kk % p.nst, kk & 1);
      __syncwarp();
    }
    // every chain issued lands before TMEM is released (bounded)
    if (lane == 0 && kk > 0) {
      umma_commit(&bar[2]);
      mbar_wait(&bar[2], 0, kLimit);
    }
    __syncwarp();
  } else {
    // ======================= workers ======================================
    int cur_unit = -1, pend_tb = 0, k = 0;
    bool has_pend = false;
    Cursor pend;
    Cursor it = next_valid(at(it0));
    if (it.it < it1) stage_copy(it, 0);
    while (it.it < it1 && !failed) {
      const int unit = it.unit;
      const Cursor nxt = next_valid(after(it));
      if (p.nstg == 2) {
        if (nxt.it < it1)
          stage_copy(nxt, (k + 1) & 1);  // overwrites the staging of item k - 1, already dequantised
        else
          cp_async_commit();  // an empty group keeps the wait count below uniform
      }
      if (unit != cur_unit) {
        if (has_pend) {
          failed = !finish(pend, pend_tb);
          has_pend = false;
          if (failed) break;
        }
        load_q(unit);
        cur_unit = unit;
      }
      if (p.nst == 1 && has_pend) {  // the single key stage must be free
        failed = !finish(pend, pend_tb);
        has_pend = false;
        if (failed) break;
      }
      if (p.nstg == 2)
        cp_async_wait<1>();  // this item's bundles landed (the next item's may be in flight)
      else
        cp_async_wait<0>();
      workers_sync<kTcWorkers>();
      dequant(p.nstg == 2 ? (k & 1) : 0, k % p.nst);
      fence_proxy_async();  // the keys, written here, are read by the tensor cores
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar[3 + (k & 1)]);
      if (p.nstg == 1 && nxt.it < it1) {  // the staging is consumed once every worker is done
        workers_sync<kTcWorkers>();
        stage_copy(nxt, 0);
      }
      if (has_pend) {
        failed = !finish(pend, pend_tb);
        if (failed) break;
      }
      pend = it; pend_tb = k & 1; has_pend = true;
      ++k;
      it = nxt;
    }
    if (!failed && has_pend) failed = !finish(pend, pend_tb);
    cp_async_wait<0>();  // no copy outlives the CTA
    if (failed) {
      *abort_flag = 1;
      if (tid == 0) set_err(a.err, 8);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512)
                 : "memory");
  pdl_trigger();
}

// Shared-memory plan of the tensor-core kernels: the query rows first (hi,
// then lo), so that the statistics pass's reads past the last query row
// (at most 112 rows of 128 bytes per box) stay inside the key stages that
// follow; two key stages when they fit, else one; two staging buffers of
// the K bundles.  Bundle strides are odd multiples of 16 bytes, so the
// 16-byte loads of eight consecutive positions fall in distinct banks.
TcPlan tc_plan(const EvictArgs &a, int sms) {
  TcPlan p;
  const int R = a.n_win * a.G;
  p.R16 = (R + 15) / 16 * 16;
  p.nch = (p.R16 + 127) / 128;
  p.q_lo = a.q_f32 ? 1 : 0;
  p.k_lo = a.v.bits != 16 ? 1 : 0;
  p.fmt = a.v.bits == 16 ? kFmtBf16
          : a.v.scheme == kSchemeSym ? (a.v.bits == 8 ? kFmtS8 : a.v.bits == 4 ? kFmtS4 : kFmtS2)
                                     : (a.v.bits == 8 ? kFmtG8 : kFmtG4);
  const int ks16 = TcFmtKs16(p.fmt);
  const int extra = a.v.bits == 16 ? 0 : a.v.scheme == kSchemeSym ? 1 : meta_bytes(128, a.v.group) / 16;
  p.kb_nch = ks16 + (a.v.scheme == kSchemeSym ? 0 : extra);  // the scale word is copied apart
  const int kb = ks16 + extra;
  p.kb_stride = 16 * (kb % 2 ? kb : kb + 1);
  p.nc_magic = (65536 + p.kb_nch - 1) / p.kb_nch;
  p.stg_bytes = kT * p.kb_stride;
  p.stage = p.k_lo ? 4 * 128 * 128 : 2 * 128 * 128;
  p.off_q = 0;
  p.off_ql = p.R16 * 256;
  const int qbytes = p.R16 * 256 * (p.q_lo ? 2 : 1);
  p.off_k = (qbytes + 1023) / 1024 * 1024;
  auto fits = [&](int nst, int nstg) {
    return p.off_k + nst * p.stage + nstg * p.stg_bytes + 256 * 4 + 3 * 128 * 4 + 64 + 1024 <= 232448;
  };
  p.nst = fits(2, 2) ? 2 : 1;
  p.nstg = fits(p.nst, 2) ? 2 : 1;
  p.off_stg = p.off_k + p.nst * p.stage;
  p.off_norm = p.off_stg + p.nstg * p.stg_bytes;
  p.off_pv = p.off_norm + 256 * 4;
  p.off_bar = p.off_pv + 3 * 128 * 4;
  p.smem = p.off_bar + 64 + 1024;  // + alignment of the base to 1024 bytes
  p.n_items = a.v.B * a.v.Hkv * a.n_tiles;
  const int grid = std::max(1, std::min(p.n_items, sms));
  p.items_per_cta = (p.n_items + grid - 1) / grid;
  return p;
}

cudaError_t launch_evict_tc(const EvictArgs &a, cudaStream_t st) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const TcPlan p = tc_plan(a, sms);
  cudaError_t e = cudaFuncSetAttribute(evict_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       p.smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(evict_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, p.smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((p.n_items + p.items_per_cta - 1) / p.items_per_cta);
  e = launch_pdl(evict_tc_kernel<false>, grid, dim3(kTcThreads), p.smem, st, a, p);
  if (e == cudaSuccess) {
    const int rows = a.v.B * a.v.Hkv * a.n_win * a.G;
    e = launch_pdl(evict_merge_stats_kernel, dim3((rows + kMergeWarps - 1) / kMergeWarps),
                   dim3(32 * kMergeWarps), 0, st, a);
  }
  if (e == cudaSuccess) e = launch_pdl(evict_tc_kernel<true>, grid, dim3(kTcThreads), p.smem, st, a, p);
  if (e == cudaSuccess)
    e = launch_pdl(evict_select_kernel, dim3(a.v.Hkv, a.v.B), dim3(1024), 0, st, a);
  return e;
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
    e = launch_pdl(evict_merge_stats_kernel, dim3((rows + kMergeWarps - 1) / kMergeWarps),
                   dim3(32 * kMergeWarps), 0, st, a);
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
  if (evict_uses_tc(a.v.D, a.n_win * a.G)) return launch_evict_tc(a, st);
  switch (a.v.D) {
    case 128: return launch_evict_d<128>(a, st);
    case 64: return launch_evict_d<64>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace kvk
