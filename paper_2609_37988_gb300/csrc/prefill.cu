// prefill.cu -- causal chunk attention over a compressed GQA cache
// (head_dim 128) on the tensor cores: the queries of each sequence's last n_q
// positions attend to the dequantised cache up to their own position (the
// pre-fill the paper times over compressed caches, Sec. 4; the chunk's keys
// and values are written with kvk_append first, so the chunk reads the same
// stored keys and values the decode steps then read).
//
// Rows: row r = i G + h of a (sequence, KV head) unit is chunk query i and
// head h of the KV head's group; query i sits at position len - n_q + i and
// sees positions 0 .. len - n_q + i.  A job is 128 consecutive rows of one
// unit.  Two launches:
//  * expand: every 64-position tile of the cache is dequantised once into
//    the layout the products read (bf16 hi and lo halves, K-major
//    128-byte-swizzled boxes), in caller scratch;
//  * attention, one pass over the tiles: per tile, S = Q K^T (TMEM lane =
//    row) with x = sigma log2(e) <q, k>; each row's maximum over the tile
//    (its four slices' maxima through shared memory) against the row's
//    reference m, which moves only when a score rises more than 8 above it
//    (O and the row's sums then rescaled by 2^(m_old - m_new) in place);
//    P = 2^(x - m) (zero past the row's limit, at most 2^8) as bf16 hi and
//    lo pairs into TMEM, O += P V (P the A operand from TMEM, the value
//    tile an MN-major B operand); after the job's last tile O (TMEM lane =
//    row) is divided by the row's sum of P and written out.
// The attention kernel runs one persistent CTA per SM: a copy warp
// brings each job's tiles in with bulk copies, three MMA warps issue the
// tcgen05 products (one thread issues at most one product per ~45 cycles:
// the scores of even and of odd tiles, and the value products, are three
// streams), 16 worker warps stage the query rows into TMEM (the A operand
// of the score products) and run the epilogues.  Products are hi*hi +
// hi*lo + lo*hi (no lo part for bf16 caches or bf16 queries), fp32
// accumulation in TMEM.  Jobs are handed out from a counter in bands of
// units whose tiles stay in L2, the longest row blocks first.
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"
#include "umma.cuh"
#include "window_tc.cuh"

namespace kvk {
namespace {

constexpr int kPfWorkers = 512;
constexpr int kPfThreads = kPfWorkers + 128;  // + three MMA warps and the copy warp
constexpr int kPfRows = 128;                 // rows per job
constexpr int kPfT = 64;                     // positions per tile
constexpr int kPfBox = kPfT * 128;           // one 64-channel box of a tile (8 KB)
constexpr int kPfMaxStages = 6;              // key (and value) stages at most
constexpr int kPfBarBytes = 320;             // barriers and the CTA's shared words

struct PfPlan {
  int n_rb, n_jobs, grid, n_t64;
  int q_lo, k_lo, fmt, gshift;
  int kpc;            // keys with per-channel groups (codes + group plane + residual)
  int ks16, nrec;
  uint32_t nc_magic;  // expand: ceil(2^32 / nrec), e / nrec = umulhi(e, nc_magic)
  int b_stride;       // expand: staged record stride (odd multiple of 16 bytes)
  int kbytes, tbytes; // a tile's keys (hi, lo); the whole tile (keys, values)
  int ns;             // key stages of the attention kernels
  int nv;             // value stages (output pass)
  int band;           // units per band of the job order
  int off_v, off_red, off_bar, smem, smem_x;  // key stages at offset 0
};

// Tiles a job reads: positions up to that of the job's last row.
__device__ __forceinline__ int pf_tiles(int len, int n_q, int G, int r_last) {
  const int p_max = len - n_q + r_last / G;
  return p_max >= 0 ? p_max / kPfT + 1 : 0;
}

// Expand: the keys and values of one 64-position tile of one unit, staged
// raw (rotations undone), dequantised per (position, channel quarter) into
// [K hi | K lo | V hi | V lo] (8 KB boxes; no lo halves for bf16 caches)
// and stored for every job of the unit to copy.  Positions past the length
// are zero.
__global__ void __launch_bounds__(kPfWorkers) prefill_expand_kernel(const PfArgs a, const PfPlan p) {
  extern __shared__ uint8_t pf_raw[];
  uint8_t *sm = pf_raw + ((1024u - (smem_u32(pf_raw) & 1023u)) & 1023u);
  const GqaView &v = a.v;
  const int tile = blockIdx.x, unit = blockIdx.y, tid = threadIdx.x;
  pdl_wait();
  const int len = v.lens[unit / v.Hkv];
  const int t0 = tile * kPfT;
  if (t0 >= len) {
    pdl_trigger();
    return;
  }
  uint8_t *stg = sm + p.tbytes;
  const uint8_t *base = v.rec + (size_t)unit * v.cap * v.rec_bytes;
  const bool sym = p.fmt >= kFmtS8, bf = p.fmt == kFmtBf16;
  for (int e = tid; e < kPfT * p.nrec; e += kPfWorkers) {
    const int pos = (int)__umulhi((uint32_t)e, p.nc_magic), c = e - pos * p.nrec;
    const int t = t0 + pos;
    const bool ok = t < len;
    int so;
    if (sym)
      so = (c + sym_rot(t, p.nrec)) & (p.nrec - 1);
    else if (!bf && c >= p.ks16 && c < 2 * p.ks16)
      so = p.ks16 + ((c - p.ks16 + v_rot(t, v.rec_bytes, p.ks16)) & (p.ks16 - 1));
    else
      so = c;
    cp_async16(stg + pos * p.b_stride + 16 * c, base + (size_t)(ok ? t : t0) * v.rec_bytes + 16 * so, ok);
  }
  if (sym)
    for (int pos = tid; pos < kPfT; pos += kPfWorkers) {
      const int t = t0 + pos;
      const bool ok = t < len;
      cp_async4(stg + pos * p.b_stride + v.rec_bytes, v.scales + (size_t)unit * v.cap + (ok ? t : t0), ok);
    }
  // per-channel keys: the (scale, zero) rows of the tile's complete groups
  // of positions (kPfT >> gshift groups of 128 channels; rows of the open
  // group are zero and unused: those positions come from the residual)
  const int g0 = t0 >> p.gshift, full = (len >> p.gshift) << p.gshift;
  float2 *mrows = reinterpret_cast<float2 *>(stg + kPfT * p.b_stride);
  if (p.kpc) {
    const int ng = kPfT >> p.gshift;
    for (int i = tid; i < ng * 128 * 8 / 16; i += kPfWorkers) {
      const int gi = i / 64, c = i - gi * 64;  // 64 chunks of 16 bytes per row
      const bool ok = ((g0 + gi) << p.gshift) < full;
      const float2 *src = v.gmeta + ((size_t)unit * (v.cap >> p.gshift) + (ok ? g0 + gi : 0)) * 128;
      cp_async16(reinterpret_cast<uint8_t *>(mrows) + 16 * i, reinterpret_cast<const uint8_t *>(src) + 16 * c, ok);
    }
  }
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();
  // threads [0, 256): key quarters; [256, 512): value quarters
  const int pidx = tid & (kPfT - 1), part = tid / kPfT;
  const uint8_t *bundle = stg + pidx * p.b_stride;
  const int ks = 16 * p.ks16;
  const int mb = (p.nrec * 16 - 2 * ks) / 2;  // grouped: one metadata block
  uint8_t *kh = sm, *kl = sm + 2 * kPfBox;
  if (part < 4 && p.kpc) {
    // per-channel keys: complete groups from codes and the group rows, the
    // open group from the bf16 residual (row t mod g), zero past the length
    const int t = t0 + pidx;
    if (t < full) {
      const float2 *mr = mrows + ((t >> p.gshift) - g0) * 128;
      if (p.fmt == kFmtG8)
        tc_dequant_kpc<8, kPfBox>(bundle, mr, pidx, part, kh, kl);
      else
        tc_dequant_kpc<4, kPfBox>(bundle, mr, pidx, part, kh, kl);
    } else {
      const uint4 z = make_uint4(0, 0, 0, 0);
      if (t < len) {
        const uint8_t *res = v.resid + ((size_t)unit * ((size_t)1 << p.gshift) + (t & ((1 << p.gshift) - 1))) * 256;
        tc_dequant<kFmtBf16, kPfBox>(res, nullptr, pidx, part, p.gshift, kh, kl);
      } else {
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) put_chunk(kh, pidx, 32 * part + 8 * cc, kPfBox, z);
      }
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) put_chunk(kl, pidx, 32 * part + 8 * cc, kPfBox, z);
    }
  } else if (part < 4) {
    const uint8_t *kmeta = sym ? bundle + v.rec_bytes : bundle + 2 * ks;
    switch (p.fmt) {
      case kFmtBf16: tc_dequant<kFmtBf16, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
      case kFmtG8: tc_dequant<kFmtG8, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
      case kFmtG4: tc_dequant<kFmtG4, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
      case kFmtS8: tc_dequant<kFmtS8, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
      case kFmtS4: tc_dequant<kFmtS4, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
      default: tc_dequant<kFmtS2, kPfBox>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
    }
  } else {
    const int qc = part - 4;
    uint8_t *vh = sm + p.kbytes, *vl = vh + 2 * kPfBox;
    const uint8_t *vsec = bundle + ks, *vmeta = bundle + 2 * ks + (p.kpc ? 0 : mb);
    const float svs =
        sym ? __uint_as_float(*reinterpret_cast<const uint32_t *>(bundle + v.rec_bytes) & 0xFFFF0000u) : 0.f;
    switch (p.fmt) {
      case kFmtBf16: tc_dequant_v<kFmtBf16, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
      case kFmtG8: tc_dequant_v<kFmtG8, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
      case kFmtG4: tc_dequant_v<kFmtG4, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
      case kFmtS8: tc_dequant_v<kFmtS8, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
      case kFmtS4: tc_dequant_v<kFmtS4, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
      default: tc_dequant_v<kFmtS2, kPfBox>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
    }
  }
  __syncthreads();
  uint4 *dst = reinterpret_cast<uint4 *>(a.tiles + ((size_t)unit * p.n_t64 + tile) * p.tbytes);
  const uint4 *src = reinterpret_cast<const uint4 *>(sm);
  for (int i = tid; i < p.tbytes / 16; i += kPfWorkers) dst[i] = src[i];
  pdl_trigger();
}

// S = Q K^T of one tile into TMEM columns d0.., Q (bf16 pairs, hi then lo
// 64 columns on) from TMEM at t_q, the keys (hi, then lo 2 boxes on) K-major
// in shared memory at kh: 16 channels per k-step.
template <bool KLO, bool QLO>
__device__ __forceinline__ void pf_issue_scores(uint32_t d0, uint32_t t_q, uint32_t kh) {
  constexpr uint32_t id = umma_idesc(128, kPfT, false, false);
  constexpr uint32_t hi = umma_desc_hi_sw128(1024);
  const uint32_t lo_h = umma_desc_lo(kh, 16), lo_l = lo_h + (2 * kPfBox >> 4);
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const uint32_t ko = ((ks >> 2) * kPfBox + (ks & 3) * 32) >> 4;
    umma_f16_ts_w(d0, t_q + 8 * ks, lo_h + ko, hi, id, ks > 0);
    if (KLO) umma_f16_ts_w(d0, t_q + 8 * ks, lo_l + ko, hi, id, true);
    if (QLO) umma_f16_ts_w(d0, t_q + 64 + 8 * ks, lo_h + ko, hi, id, true);
  }
}
// O += P V of one tile: P (bf16 pairs, hi then lo 32 columns on) from TMEM
// at pa, the values (hi, then lo 2 boxes on) MN-major in shared memory at vh
// (64-channel boxes kPfBox apart), 16 positions per k-step.
template <bool KLO>
__device__ __forceinline__ void pf_issue_values(uint32_t t_o, uint32_t pa, uint32_t vh, bool acc) {
  constexpr uint32_t id = umma_idesc(128, 128, false, true);
  constexpr uint32_t hi = umma_desc_hi_sw128(1024);
  const uint32_t lo_h = umma_desc_lo(vh, kPfBox), lo_l = lo_h + (2 * kPfBox >> 4);
#pragma unroll
  for (int ks = 0; ks < kPfT / 16; ++ks) {
    umma_f16_ts_w(t_o, pa + 8 * ks, lo_h + 128 * ks, hi, id, acc || ks > 0);
    if (KLO) umma_f16_ts_w(t_o, pa + 8 * ks, lo_l + 128 * ks, hi, id, true);
    umma_f16_ts_w(t_o, pa + 32 + 8 * ks, lo_h + 128 * ks, hi, id, true);
  }
}

__global__ void __launch_bounds__(kPfThreads, 1) prefill_kernel(const PfArgs a, const PfPlan p) {
  constexpr int D = 128;
  constexpr uint32_t kLimit = 1u << 20;  // polls of up to 2 us each
  extern __shared__ uint8_t pf_raw[];
  uint8_t *sm = pf_raw + ((1024u - (smem_u32(pf_raw) & 1023u)) & 1023u);
  // barriers: kfull[6] keys of a stage landed, kfree[6] its score product
  // done, vfull[6] / vfree[6] the same for values; per tile parity: sdone[2]
  // scores done, epi[2] the workers' epilogue done (16 arrivals), pvdone[2]
  // value product done; qready the job's query rows staged (16 arrivals),
  // drain[3] (one per MMA warp).  A barrier per parity completes every other tile, and the next
  // completion of one always depends on the wait for its previous one, so
  // no wait can fall two phases behind.
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm + p.off_bar);
  constexpr int S6 = kPfMaxStages;
  uint64_t *kfull = bar, *kfree = bar + S6, *vfull = bar + 2 * S6, *vfree = bar + 3 * S6;
  uint64_t *sdone = bar + 4 * S6, *epi = sdone + 2, *pvdone = sdone + 4, *qready = sdone + 6, *drain = sdone + 7;
  constexpr int kBars = 4 * S6 + 10;
  static_assert(kBars * 8 + 12 <= kPfBarBytes, "barrier region");
  uint32_t *tbase = reinterpret_cast<uint32_t *>(sm + p.off_bar + kBars * 8);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + p.off_bar + kBars * 8 + 4);
  volatile int *s_job = reinterpret_cast<volatile int *>(sm + p.off_bar + kBars * 8 + 8);
  const GqaView &v = a.v;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int R = a.n_q * a.G;
  const int quarter = warp & 3, slice = warp >> 2;
  const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
  const float sg = a.sig_log2;
  const int vbytes = p.tbytes - p.kbytes;

  if (tid == 0) {
    for (int i = 0; i < kBars; ++i) {
      uint64_t *b = &bar[i];
      mbar_init(b, (b == epi || b == epi + 1 || b == qready) ? kPfWorkers / 32 : 1);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  pdl_wait();  // the expanded tiles, lengths and (output pass) statistics are complete
  constexpr uint32_t kCols = 512;
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tbase)),
                 "n"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tbase;
  // TMEM columns (lane = the job's row in every region): scores of tile k
  // at 64 (k & 1), fp32; the job's query rows as bf16 pairs (hi 64 columns,
  // then lo), the A operand of the score products; output pass: O at 128
  // (fp32, 128 channels) and P of tile k at 256 + 64 (k & 1) (bf16 pairs,
  // hi 32 columns, then lo), the A operand of the value products.
  const uint32_t t_o = tmem + 128;
  const uint32_t t_q = tmem + 384;
  auto t_p = [&](int k) { return tmem + 256 + 64 * (k & 1); };

  // Jobs are handed out one at a time from a counter, so CTAs finish
  // together although jobs differ in length.  Order: bands of p.band units
  // (whose tiles the band's jobs share in L2), in each band the longest row
  // blocks first.
  // Every thread of the CTA takes part in each hand-out; a role that gave up
  // keeps taking jobs (and skips them) until none is left, so no barrier
  // waits for threads that left.
  const int units = v.B * v.Hkv;
  int *counter = a.counter;
  auto next_job = [&]() -> int {
    asm volatile("bar.sync 2, %0;" ::"n"(kPfThreads) : "memory");  // the previous id is read
    if (tid == 0) *s_job = atomicAdd(counter, 1);
    asm volatile("bar.sync 2, %0;" ::"n"(kPfThreads) : "memory");
    return *s_job;
  };
  struct Job {
    int unit, b, j, r0, nr, len, n_t;
  };
  auto job_at = [&](int job) {
    Job J;
    const int per = p.band * p.n_rb;
    const int g = job / per, w = job - g * per;
    const int ub = min(p.band, units - g * p.band);  // units in this band
    const int step = w / ub;
    J.unit = g * p.band + (w - step * ub);
    const int rb = p.n_rb - 1 - step;
    J.b = J.unit / v.Hkv;
    J.j = J.unit - J.b * v.Hkv;
    J.r0 = rb * kPfRows;
    J.nr = min(kPfRows, R - J.r0);
    J.len = v.lens[J.b];
    J.n_t = pf_tiles(J.len, a.n_q, a.G, J.r0 + J.nr - 1);
    return J;
  };
  auto sleepy = [&](uint64_t *b, uint32_t parity) {
    return mbar_wait_sleepy(b, parity, kLimit, abort_flag, 2000);
  };

  if (warp == kPfWorkers / 32 + 1) {
    // ======================= copy warp ====================================
    // lane 0 copies each tile's keys (and values) into the next stage once
    // the products that read the stage's previous tile are done
    int kk = 0;
    bool ok = true;
    for (int job = next_job(); job < p.n_jobs; job = next_job()) {
      if (ok && lane == 0) {
        const Job J = job_at(job);
        const uint8_t *src0 = a.tiles + (size_t)J.unit * p.n_t64 * p.tbytes;
        for (int k = 0; k < J.n_t && ok; ++k, ++kk) {
          const int s = kk % p.ns, u = kk / p.ns;
          if (u > 0) ok = sleepy(&kfree[s], (u - 1) & 1);
          // the stage is written only by bulk copies and read only by the
          // products (both async proxy, ordered by the commit's release of
          // kfree): no proxy fence
          if (ok) {
            mbar_expect_tx(&kfull[s], p.kbytes);
            bulk_g2s(sm + s * p.kbytes, src0 + (size_t)k * p.tbytes, p.kbytes, &kfull[s]);
          }
          if (ok) {
            const int sv = kk % p.nv, uv = kk / p.nv;
            if (uv > 0) ok = sleepy(&vfree[sv], (uv - 1) & 1);
            if (ok) {
              mbar_expect_tx(&vfull[sv], vbytes);
              bulk_g2s(sm + p.off_v + sv * vbytes, src0 + (size_t)k * p.tbytes + p.kbytes, vbytes, &vfull[sv]);
            }
          }
        }
        if (!ok) *abort_flag = 1;
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    // the last copies land before the CTA leaves (bounded; at once when
    // they were consumed)
    if (lane == 0)
      for (int c = max(0, kk - max(p.ns, p.nv)); c < kk; ++c) {
        if (c >= kk - p.ns) mbar_wait(&kfull[c % p.ns], (c / p.ns) & 1, 1u << 22);
        if (c >= kk - p.nv) mbar_wait(&vfull[c % p.nv], (c / p.nv) & 1, 1u << 22);
      }
    __syncwarp();
  } else if (warp >= kPfWorkers / 32) {
    // ======================= MMA warps ====================================
    // Each warp's lane 0 issues a stream of products (one thread issues at
    // most one product per ~45 cycles, so several streams keep the tensor
    // cores busy): warps 16 and 18 the score products of the even and the
    // odd tiles, warp 19 (output pass) the value products.  A commit covers
    // the products its own thread issued.
    const int role = warp == kPfWorkers / 32 ? 0 : warp == kPfWorkers / 32 + 2 ? 1 : 2;
    auto issue_s = [&](int kk, int s) {  // S = Q K^T of the tile in key stage s
      tc_fence_after();
      const uint32_t kh = smem_u32(sm + s * p.kbytes), d0 = tmem + 64u * (kk & 1);
      if (p.k_lo) {
        if (p.q_lo) pf_issue_scores<true, true>(d0, t_q, kh);
        else pf_issue_scores<true, false>(d0, t_q, kh);
      } else {
        if (p.q_lo) pf_issue_scores<false, true>(d0, t_q, kh);
        else pf_issue_scores<false, false>(d0, t_q, kh);
      }
      umma_commit(&sdone[kk & 1]);
      umma_commit(&kfree[s]);
    };
    auto issue_pv = [&](int c, int s, bool acc) {  // O += P V of tile c, values in stage s
      tc_fence_after();
      const uint32_t vh = smem_u32(sm + p.off_v + s * vbytes);
      if (p.k_lo) pf_issue_values<true>(t_o, t_p(c), vh, acc);
      else pf_issue_values<false>(t_o, t_p(c), vh, acc);
      umma_commit(&pvdone[c & 1]);
      umma_commit(&vfree[s]);
    };
    auto wait_epi = [&](int c) -> bool {  // the workers' epilogue of tile c
      return c < 0 || sleepy(&epi[c & 1], (c >> 1) & 1);
    };
    auto pv = [&](int c, bool acc) -> bool {  // value product of tile c once its P is written
      const int s = c % p.nv;
      bool ok = wait_epi(c);
      if (ok) ok = sleepy(&vfull[s], (c / p.nv) & 1);
      if (ok) issue_pv(c, s, acc);
      return ok;
    };
    // Barrier phases: a score warp waits for epi(c) (its parity's previous
    // phase) before S(c + 2), and epi[c & 1] completes for tile c + 2 only
    // after S(c + 2); the value warp waits for every epi(c) in order before
    // PV(c), which the workers await before the epilogue of c + 2.  So every
    // wait is for the phase after the one its warp last saw.
    int kk = 0, njob = 0, issued = 0;
    bool ok = true;
    for (int job = next_job(); job < p.n_jobs; job = next_job()) {
      if (ok && lane == 0) {
        const Job J = job_at(job);
        // this job's query rows are staged (and the last job's O was read)
        ok = sleepy(qready, njob & 1);
        ++njob;
        for (int k = 0; k < J.n_t && ok; ++k, ++kk) {
          if ((kk & 1) == role) {
            const int s = kk % p.ns;
            if (kk >= 2) ok = wait_epi(kk - 2);  // the score buffer of tile kk - 2 is read
            if (ok) ok = sleepy(&kfull[s], (kk / p.ns) & 1);
            if (ok) issue_s(kk, s);
            ++issued;
          } else if (role == 2) {
            ok = pv(kk, k > 0);
            ++issued;
          }
        }
        if (!ok) *abort_flag = 1;
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    // every product this warp issued lands before TMEM is released (bounded)
    if (lane == 0 && issued > 0) {
      umma_commit(&drain[role]);
      mbar_wait(&drain[role], 0, 1u << 22);  // drain[0..2]
    }
    __syncwarp();
  } else {
    // ======================= workers ======================================
    bool failed = false;
    auto wait_pv = [&](int c) -> bool {  // completion of tile c's value product
      return c < 0 || sleepy(&pvdone[c & 1], (c >> 1) & 1);
    };
    // query rows r0 .. r0 + 127 of the unit (zero past R) into TMEM, this
    // thread's row and quarter of the channels; output pass: the rows'
    // log-normalisers (+inf for rows that see no position)
    auto load_q = [&](const Job &J) {
      const int rl = 32 * quarter + lane;
      float x[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) x[i] = 0.f;
      if (rl < J.nr) {
        const int r = J.r0 + rl;
        const int qi = r / a.G, h = J.j * a.G + (r - qi * a.G);
        const size_t off = (((size_t)J.b * a.n_q + qi) * a.Hq + h) * D + 32 * slice;
        if (a.q_f32) {
          const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + off);
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const float4 u = src[c];
            x[4 * c] = u.x; x[4 * c + 1] = u.y; x[4 * c + 2] = u.z; x[4 * c + 3] = u.w;
          }
        } else {
          const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.q) + off);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const uint4 u = src[c];
            const uint32_t ww[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              x[8 * c + 2 * i] = __uint_as_float(ww[i] << 16);
              x[8 * c + 2 * i + 1] = __uint_as_float(ww[i] & 0xFFFF0000u);
            }
          }
        }
      }
      uint32_t hw[16], lw[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) split2<true>(x[2 * i], x[2 * i + 1], hw[i], lw[i]);
      tmem_st16_nw(t_q + 16 * slice + lane_off, hw);
      if (p.q_lo) tmem_st16_nw(t_q + 64 + 16 * slice + lane_off, lw);
      tmem_wait_st();
      tc_fence_before();  // the rows, stored here, are read by the tensor cores
      workers_sync<kPfWorkers>();
    };

    int kk = 0;
    float *smax = reinterpret_cast<float *>(sm + p.off_red);  // [4 slices][128 rows]
    for (int job = next_job(); job < p.n_jobs; job = next_job()) {
      if (failed) continue;
      const Job J = job_at(job);
      const int base = J.len - a.n_q;  // position of chunk query 0
      load_q(J);
      __syncwarp();
      if (lane == 0) mbar_arrive(qready);
      // this thread's row of the job (and slice of each tile's positions)
      const int rl = 32 * quarter + lane;
      const bool row_live = rl < J.nr;
      const int last = base + (J.r0 + rl) / a.G;  // the last position the row sees
      // The row's reference maximum (scaled scores, base 2) and this slice's
      // sum of weights.  The reference stays while no score of the row rises
      // more than 8 above it (P <= 2^8); when one does, the row's four
      // threads move it and rescale their channels of O (in TMEM, after the
      // value product of the previous tile) and their sums.  The weights
      // are not normalised: O is divided by the row's sum at the end.
      float c_ref = -INFINITY, l_run = 0.f;
      for (int k = 0; k < J.n_t; ++k, ++kk) {
        // scores of this tile, and its P buffer free
        bool ok = !failed && sleepy(&sdone[kk & 1], (kk >> 1) & 1);
        if (ok) ok = wait_pv(kk - 2);
        if (workers_sync_or<kPfWorkers>(!ok)) {
          failed = true;
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const int tb = k * kPfT + 16 * slice;  // first position of this thread's slice
        const int nv = row_live ? min(16, last - tb + 1) : 0;  // live positions (<= 0: none)
        float y[16];
        tmem_ld16(tmem + 64u * (kk & 1) + 16 * slice + lane_off, y);
        float mx = -INFINITY;
        if (nv >= 16) {  // the whole slice is in the row's range (most tiles)
          float mm[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) mm[i] = fmaxf(fmaxf(y[i], y[4 + i]), fmaxf(y[8 + i], y[12 + i]));
          mx = fmaxf(fmaxf(mm[0], mm[1]), fmaxf(mm[2], mm[3]));
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (i < nv) mx = fmaxf(mx, y[i]);
        }
        smax[slice * kPfRows + rl] = mx;
        workers_sync<kPfWorkers>();  // the row's four slice maxima
        const float M = sg * fmaxf(fmaxf(smax[rl], smax[kPfRows + rl]),
                                   fmaxf(smax[2 * kPfRows + rl], smax[3 * kPfRows + rl]));
        if (M > c_ref + 8.f) {  // the same decision on the row's four threads
          if (c_ref != -INFINITY) {
            // O holds this job's earlier tiles: rescale this thread's 32
            // channels once the previous tile's value product is done
            if (!wait_pv(kk - 1)) {
              failed = true;
              *abort_flag = 1;
            } else {
              tc_fence_after();
              const float f = fast_exp2(c_ref - M);
              float z[16];
              uint32_t zw[16];
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                tmem_ld16(t_o + 32 * slice + 16 * h + lane_off, z);
#pragma unroll
                for (int i = 0; i < 16; ++i) zw[i] = __float_as_uint(z[i] * f);
                tmem_st16_nw(t_o + 32 * slice + 16 * h + lane_off, zw);
              }
              l_run *= f;
            }
          }
          c_ref = M;
        }
        // P of this row over the slice's 16 positions, hi and lo halves
        float x0[8], x1[8];
        if (nv >= 16) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            x0[i] = fast_exp2(fmaf(y[i], sg, -c_ref));
            x1[i] = fast_exp2(fmaf(y[8 + i], sg, -c_ref));
          }
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            x0[i] = i < nv ? fast_exp2(fmaf(y[i], sg, -c_ref)) : 0.f;
            x1[i] = 8 + i < nv ? fast_exp2(fmaf(y[8 + i], sg, -c_ref)) : 0.f;
          }
        }
        // positions 16 slice .. 16 slice + 15 of the tile: 8 columns of
        // bf16 pairs (hi), the same 32 columns on (lo)
        uint32_t hw[8], lw[8];
        float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          split2<true>(x0[2 * i], x0[2 * i + 1], hw[i], lw[i]);
          split2<true>(x1[2 * i], x1[2 * i + 1], hw[4 + i], lw[4 + i]);
          ls[i] += (x0[2 * i] + x0[2 * i + 1]) + (x1[2 * i] + x1[2 * i + 1]);
        }
        l_run += (ls[0] + ls[1]) + (ls[2] + ls[3]);
        tmem_st8_nw(t_p(kk) + 8 * slice + lane_off, hw);
        tmem_st8_nw(t_p(kk) + 32 + 8 * slice + lane_off, lw);
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&epi[kk & 1]);
      }
      // a rescale's wait that gave up on the last tile is seen by every worker
      if (workers_sync_or<kPfWorkers>(failed)) {
        failed = true;
        *abort_flag = 1;
        continue;
      }
      // O: lane = the job's row, 32 channels per slice, divided by the sum
      // of the row's weights (the four slices' sums, same reference)
      float o[32];
      if (J.n_t > 0) {
        const bool ok = wait_pv(kk - 1);
        if (workers_sync_or<kPfWorkers>(!ok)) {
          failed = true;
          *abort_flag = 1;
          continue;
        }
        tc_fence_after();
        float z[16];
        tmem_ld16(t_o + 32 * slice + lane_off, z);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] = z[i];
        tmem_ld16(t_o + 32 * slice + 16 + lane_off, z);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[16 + i] = z[i];
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = 0.f;
      }
      smax[slice * kPfRows + rl] = l_run;
      workers_sync<kPfWorkers>();
      const float L = (smax[rl] + smax[kPfRows + rl]) + (smax[2 * kPfRows + rl] + smax[3 * kPfRows + rl]);
      const float inv = L > 0.f ? 1.f / L : 0.f;
      if (row_live) {
        const int r = J.r0 + rl;
        const int qi = r / a.G, h = J.j * a.G + (r - qi * a.G);
        float4 *dst = reinterpret_cast<float4 *>(a.out + (((size_t)J.b * a.n_q + qi) * a.Hq + h) * D + 32 * slice);
#pragma unroll
        for (int c = 0; c < 8; ++c)
          dst[c] = make_float4(o[4 * c] * inv, o[4 * c + 1] * inv, o[4 * c + 2] * inv, o[4 * c + 3] * inv);
      }
      tc_fence_before();
      workers_sync<kPfWorkers>();  // O and the sums read before the next job's first products
    }
    if (failed && tid == 0) set_err(a.err, 8);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kCols)
                 : "memory");
  pdl_trigger();
}

// Shared-memory plan.  Attention kernel: the key stages, the value stages,
// the rows' slice maxima (and at a job's end their sums of weights),
// barriers; the query rows, S, P and O live in TMEM.  Expand kernel: one
// tile and its staged records.
PfPlan pf_plan(const PfArgs &a, int sms) {
  PfPlan p;
  const int R = a.n_q * a.G;
  p.n_rb = (R + kPfRows - 1) / kPfRows;
  p.n_jobs = a.v.B * a.v.Hkv * p.n_rb;
  p.n_t64 = a.v.cap / kPfT;
  p.q_lo = a.q_f32 ? 1 : 0;
  p.k_lo = a.v.bits != 16 ? 1 : 0;
  p.fmt = a.v.bits == 16 ? kFmtBf16
          : a.v.scheme == kSchemeSym ? (a.v.bits == 8 ? kFmtS8 : a.v.bits == 4 ? kFmtS4 : kFmtS2)
                                     : (a.v.bits == 8 ? kFmtG8 : kFmtG4);
  p.gshift = a.v.group == 64 ? 6 : 5;
  p.kpc = a.v.bits != 16 && a.v.key_axis == 1 ? 1 : 0;
  p.ks16 = TcFmtKs16(p.fmt);
  p.nrec = a.v.rec_bytes / 16;
  p.nc_magic = (uint32_t)((0x100000000ull + p.nrec - 1) / p.nrec);
  const bool sym = p.fmt >= kFmtS8;
  const int bchunks = p.nrec + (sym ? 1 : 0);
  p.b_stride = 16 * (bchunks % 2 ? bchunks : bchunks + 1);
  p.kbytes = 2 * kPfBox * (p.k_lo ? 2 : 1);
  p.tbytes = 2 * p.kbytes;
  // + the (scale, zero) rows of the tile's position groups (per-channel keys)
  p.smem_x = p.tbytes + kPfT * p.b_stride + (p.kpc ? 2 * 128 * 8 : 0) + 1024;
  const int vb = p.tbytes - p.kbytes;
  const int rbytes = 4 * kPfRows * 4;
  // the most stages that fit.  Value tiles wait for the value product three
  // tiles back, key tiles only for the score product, so values get the
  // larger share (int4: 2 key and 5 value stages of 32 KB); keys keep at
  // least two (a score warp's wait for the stage it skipped relies on ns >= 2).
  const int avail = 232448 - (rbytes + kPfBarBytes + 1024);
  const int T = avail / p.kbytes;  // key and value tiles are the same size
  p.ns = std::min(kPfMaxStages, std::max(2, T / 3));
  p.nv = std::max(1, std::min(kPfMaxStages, T - p.ns));
  // bands of units whose tiles take up to 32 MB (L2 holds two bands)
  const long long unit_bytes = (long long)p.n_t64 * p.tbytes;
  p.band = (int)std::max(1LL, std::min<long long>(a.v.B * a.v.Hkv, (32LL << 20) / std::max(1LL, unit_bytes)));
  p.off_v = p.ns * p.kbytes;
  p.off_red = p.off_v + p.nv * vb;
  p.off_bar = p.off_red + rbytes;
  // + alignment of the base to 1024 bytes; at least half the SM's shared
  // memory, so that one CTA (holding its TMEM columns) runs per SM
  p.smem = std::max(p.off_bar + kPfBarBytes + 1024, 116 * 1024);
  p.grid = std::max(1, std::min(p.n_jobs, sms));
  return p;
}

}  // namespace

size_t prefill_tile_bytes(int bits) { return (size_t)2 * 2 * kPfBox * (bits != 16 ? 2 : 1); }

bool prefill_plan_fits(const PfArgs &a) {
  const PfPlan o = pf_plan(a, 1);
  return o.smem <= 232448 && o.ns >= 2 && o.nv >= 2;
}

cudaError_t launch_gqa_prefill(const PfArgs &a, cudaStream_t st) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const PfPlan po = pf_plan(a, sms);
  cudaError_t e = cudaFuncSetAttribute(prefill_expand_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       po.smem_x);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, po.smem);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(a.counter, 0, sizeof(int), st);  // the job counter
  if (e == cudaSuccess)
    e = launch_pdl(prefill_expand_kernel, dim3(po.n_t64, a.v.B * a.v.Hkv), dim3(kPfWorkers), po.smem_x, st,
                   a, po);
  if (e == cudaSuccess)
    e = launch_pdl(prefill_kernel, dim3(po.grid), dim3(kPfThreads), po.smem, st, a, po);
  return e;
}

}  // namespace kvk
