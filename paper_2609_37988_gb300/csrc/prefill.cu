// prefill.cu -- causal chunk attention over a compressed GQA cache
// (head_dim 128) on the tensor cores: the queries of each sequence's last n_q
// positions attend to the dequantised cache up to their own position (the
// pre-fill the paper times over compressed caches, Sec. 5; the chunk's keys
// and values are written with kvk_append first, so the chunk reads the same
// stored keys and values the decode steps then read).
//
// Rows: row r = i G + h of a (sequence, KV head) unit is chunk query i and
// head h of the KV head's group; query i sits at position len - n_q + i and
// sees positions 0 .. len - n_q + i.  A job is 128 consecutive rows of one
// unit.  Two kernels over jobs, one persistent CTA per SM (16 worker warps,
// one MMA warp):
//  * statistics: per row, the maximum M and the sum L of 2^(x - M) of its
//    scaled scores x = sigma log2(e) <q, k> over its causal range, online
//    over 128-position tiles (S = Q K^T with TMEM lane = row, so a thread
//    updates its row's running pair);
//  * output: per 64-position tile, S = Q K^T, P = 2^(x - M - log2 L) (zero
//    past the row's limit) into shared memory, O^T += V^T P^T; after the last
//    tile O^T (TMEM lane = channel) is written out.  The normalisers being
//    final, the output pass never rescales O.
// Keys and values are dequantised into bf16 hi + lo halves in the K-major
// 128-byte-swizzled layout (rows = positions); the value MMA reads the value
// tile as an MN-major operand of that same layout.  Products are
// hi*hi + hi*lo + lo*hi (no lo part for bf16 caches or bf16 queries), fp32
// accumulation in TMEM.
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
constexpr int kPfThreads = kPfWorkers + 32;
constexpr int kPfRows = 128;  // rows per job
constexpr int kQBox = kPfRows * 128;  // one 64-channel box of the job's query rows

struct PfPlan {
  int n_rb, n_jobs, grid;
  int q_lo, k_lo, fmt, gshift;
  int ks16, nrec, ncopy;  // K-section chunks, record chunks, chunks staged per position
  uint32_t nc_magic;      // ceil(2^32 / ncopy): e / ncopy = umulhi(e, nc_magic)
  int b_stride, stg_bytes, stage, nst, nstg;
  int off_ql, off_k, off_stg, off_p, off_norm, off_red, off_bar, smem;
};

// Tiles a job reads: positions up to that of the job's last row.
__device__ __forceinline__ int pf_tiles(int len, int n_q, int G, int r_last, int tt) {
  const int p_max = len - n_q + r_last / G;
  return p_max >= 0 ? p_max / tt + 1 : 0;
}

template <bool OUT>
__global__ void __launch_bounds__(kPfThreads, 1) prefill_kernel(const PfArgs a, const PfPlan p) {
  constexpr int TT = OUT ? 64 : 128;     // positions per tile
  constexpr int KBOX = TT * 128;         // one 64-channel box of a key (value) tile
  constexpr int D = 128;
  constexpr uint32_t kLimit = 1u << 20;  // polls of up to 2 us each
  extern __shared__ uint8_t pf_raw[];
  uint8_t *sm = pf_raw + ((1024u - (smem_u32(pf_raw) & 1023u)) & 1023u);
  // bar: [0], [1] keys (and values) of an even / odd tile staged (16
  // arrivals); [2], [3] scores of an even / odd tile done; [4] P of a tile
  // written (16 arrivals); [5] its value product done; [6] drain
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm + p.off_bar);
  uint32_t *tbase = reinterpret_cast<uint32_t *>(sm + p.off_bar + 56);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + p.off_bar + 60);
  volatile int *s_job = reinterpret_cast<volatile int *>(sm + p.off_bar + 64);
  float *norm = reinterpret_cast<float *>(sm + p.off_norm);  // [128] log-normaliser per job row
  float2 *red = reinterpret_cast<float2 *>(sm + p.off_red);  // [4][128] slice statistics
  uint8_t *qh = sm, *ql = sm + p.off_ql;
  uint8_t *ph = sm + p.off_p, *pl = ph + kPfRows * 128;
  const GqaView &v = a.v;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int R = a.n_q * a.G;
  const int quarter = warp & 3, slice = warp >> 2;
  const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
  const float sg = a.sig_log2;

  if (tid == 0) {
    for (int i = 0; i < 7; ++i) mbar_init(&bar[i], (i == 0 || i == 1 || i == 4) ? kPfWorkers / 32 : 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  pdl_wait();
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tbase)),
                 "r"(256)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tbase;
  // TMEM: statistics: scores of tile k at column 128 (k & 1); output: scores
  // at 64 (k & 1), O^T at 128
  const uint32_t t_o = tmem + 128;

  // Jobs are handed out one at a time from a counter (the longest row
  // blocks first), so CTAs finish together although jobs differ in length.
  // Every thread of the CTA takes part in each hand-out; a CTA that gave up
  // keeps taking jobs (and skips them) until none is left, so no barrier
  // waits for threads that left.
  const int units = v.B * v.Hkv;
  int *counter = a.counter + (OUT ? 1 : 0);
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
    const int step = job / units;
    J.unit = job - step * units;
    const int rb = p.n_rb - 1 - step;
    J.b = J.unit / v.Hkv;
    J.j = J.unit - J.b * v.Hkv;
    J.r0 = rb * kPfRows;
    J.nr = min(kPfRows, R - J.r0);
    J.len = v.lens[J.b];
    J.n_t = pf_tiles(J.len, a.n_q, a.G, J.r0 + J.nr - 1, TT);
    return J;
  };

  if (warp == kPfWorkers / 32) {
    // ======================= MMA warp =====================================
    auto dsc = [](uint32_t addr) { return umma_desc(addr, 16, 1024, 2); };
    const uint32_t qa = smem_u32(qh), qb = smem_u32(ql);
    auto issue_s = [&](int kk) {  // S = Q K^T of the tile in stage kk % nst
      tc_fence_after();
      const uint32_t kh = smem_u32(sm + p.off_k + (kk % p.nst) * p.stage), kl = kh + 2 * KBOX;
      const uint32_t d0 = OUT ? tmem + 64u * (kk & 1) : tmem + 128u * (kk & 1);
      constexpr uint32_t id = umma_idesc(128, TT, false, false);
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
        const uint32_t ko = (ks >> 2) * KBOX + (ks & 3) * 32;
        const uint32_t qo = (ks >> 2) * kQBox + (ks & 3) * 32;
        umma_f16(d0, dsc(qa + qo), dsc(kh + ko), id, ks > 0);
        if (p.k_lo) umma_f16(d0, dsc(qa + qo), dsc(kl + ko), id, true);
        if (p.q_lo) umma_f16(d0, dsc(qb + qo), dsc(kh + ko), id, true);
      }
      umma_commit(&bar[2 + (kk & 1)]);
    };
    auto issue_pv = [&](int kk, bool acc) {  // O^T += V^T P^T of tile kk
      tc_fence_after();
      const uint32_t vh = smem_u32(sm + p.off_k + (kk % p.nst) * p.stage) + 2 * (p.k_lo ? 2 : 1) * KBOX;
      const uint32_t vl = vh + 2 * KBOX;
      const uint32_t pa = smem_u32(ph), pb = smem_u32(pl);
      constexpr uint32_t id = umma_idesc(128, kPfRows, true, false);
#pragma unroll
      for (int ks = 0; ks < TT / 16; ++ks) {
        // values MN-major: channels in 64-wide boxes KBOX apart, 16 positions per k-step
        const uint64_t va = umma_desc(vh + ks * 2048, KBOX, 1024, 2);
        const uint64_t vb = umma_desc(vl + ks * 2048, KBOX, 1024, 2);
        umma_f16(t_o, va, dsc(pa + ks * 32), id, acc || ks > 0);
        if (p.k_lo) umma_f16(t_o, vb, dsc(pa + ks * 32), id, true);
        umma_f16(t_o, va, dsc(pb + ks * 32), id, true);
      }
      umma_commit(&bar[5]);
    };
    int kk = 0;
    bool ok = true;
    for (int job = next_job(); job < p.n_jobs; job = next_job()) {
      if (!ok) continue;
      const Job J = job_at(job);
      for (int k = 0; k < J.n_t && ok; ++k, ++kk) {
        // with one stage the previous tile's values are read before the
        // workers overwrite them with this tile; with two, this tile's scores
        // go first so that they overlap the previous tile's P
        const bool pv_first = OUT && p.nst == 1;
        if (pv_first && k > 0) {
          ok = mbar_wait_sleepy(&bar[4], (kk - 1) & 1, kLimit, abort_flag, 2000);
          if (ok && lane == 0) issue_pv(kk - 1, k > 1);
        }
        if (ok) ok = mbar_wait_sleepy(&bar[kk & 1], (kk >> 1) & 1, kLimit, abort_flag, 2000);
        if (ok && lane == 0) issue_s(kk);
        if (OUT && !pv_first && ok && k > 0) {
          ok = mbar_wait_sleepy(&bar[4], (kk - 1) & 1, kLimit, abort_flag, 2000);
          if (ok && lane == 0) issue_pv(kk - 1, k > 1);
        }
        __syncwarp();
      }
      if (!ok && lane == 0) *abort_flag = 1;
      if constexpr (OUT) {
        if (ok && J.n_t > 0) {
          ok = mbar_wait_sleepy(&bar[4], (kk - 1) & 1, kLimit, abort_flag, 2000);
          if (ok && lane == 0) issue_pv(kk - 1, J.n_t > 1);
          __syncwarp();
        }
      }
    }
    if (!ok && lane == 0) *abort_flag = 1;
    // every MMA this warp issued lands before TMEM is released (bounded)
    if (lane == 0 && kk > 0) {
      umma_commit(&bar[6]);
      mbar_wait(&bar[6], 0, 1u << 22);
    }
    __syncwarp();
  } else {
    // ======================= workers ======================================
    const int pidx = tid & (TT - 1), part = tid / TT;  // staging/dequant: position, part
    bool failed = false;
    uint32_t pv_seen = 0;  // value products whose completion the workers have waited for
    auto wait_pv = [&](int kk) -> bool {  // completion of tile kk's value product
      bool ok = true;
      while (ok && (int)pv_seen <= kk) {
        ok = mbar_wait_sleepy(&bar[5], pv_seen & 1, kLimit, abort_flag, 2000);
        ++pv_seen;
      }
      return ok;
    };

    // query rows r0 .. r0 + 127 of the unit (zero past R); output pass: the
    // rows' log-normalisers (+inf for rows that see no position)
    auto load_q = [&](const Job &J) {
      for (int e = tid; e < kPfRows * (D / 8); e += kPfWorkers) {
        const int rl = e >> 4, c8 = e & 15;
        const int r = J.r0 + rl;
        float x[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = 0.f;
        if (rl < J.nr) {
          const int qi = r / a.G, h = J.j * a.G + (r - qi * a.G);
          const size_t off = (((size_t)J.b * a.n_q + qi) * a.Hq + h) * D + 8 * c8;
          if (a.q_f32) {
            const float4 u0 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + off);
            const float4 u1 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.q) + off + 4);
            x[0] = u0.x; x[1] = u0.y; x[2] = u0.z; x[3] = u0.w;
            x[4] = u1.x; x[5] = u1.y; x[6] = u1.z; x[7] = u1.w;
          } else {
            const uint4 u = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.q) + off);
            const uint32_t ww[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              x[2 * i] = __uint_as_float(ww[i] << 16);
              x[2 * i + 1] = __uint_as_float(ww[i] & 0xFFFF0000u);
            }
          }
        }
        put8(qh, ql, p.q_lo != 0, rl, 8 * c8, kQBox, x);
      }
      if constexpr (OUT) {
        for (int rl = tid; rl < kPfRows; rl += kPfWorkers) {
          float nv = INFINITY;
          if (rl < J.nr) {
            const float2 f = a.stats[(size_t)J.unit * R + J.r0 + rl];
            if (f.y > 0.f) nv = f.x + log2f(f.y);
          }
          norm[rl] = nv;
        }
      }
      fence_proxy_async();
      workers_sync<kPfWorkers>();
    };

    // asynchronous copy of tile k's records (rotation undone; statistics:
    // the K section and key metadata only) into staging buffer g
    auto stage_copy = [&](const Job &J, int k, int g) {
      const int t0 = k * TT;
      uint8_t *dst0 = sm + p.off_stg + g * p.stg_bytes;
      const uint8_t *base = v.rec + (size_t)J.unit * v.cap * v.rec_bytes;
      const bool sym = p.fmt >= kFmtS8, bf = p.fmt == kFmtBf16;
      for (int e = tid; e < TT * p.ncopy; e += kPfWorkers) {
        const int pos = (int)__umulhi((uint32_t)e, p.nc_magic), c = e - pos * p.ncopy;
        const int t = t0 + pos;
        const bool ok = t < J.len;
        // logical chunk cl of the record, and where it is stored
        const int cl = OUT ? c : (c < p.ks16 ? c : 2 * p.ks16 + (c - p.ks16));
        int so;
        if (sym) {
          so = (cl + sym_rot(t, p.nrec)) & (p.nrec - 1);
        } else if (!bf && cl >= p.ks16 && cl < 2 * p.ks16) {
          so = p.ks16 + ((cl - p.ks16 + v_rot(t, v.rec_bytes, p.ks16)) & (p.ks16 - 1));
        } else {
          so = cl;
        }
        // output pass: the whole logical record; statistics: K section and
        // key metadata back to back
        cp_async16(dst0 + pos * p.b_stride + 16 * (OUT ? cl : c),
                   base + (size_t)(ok ? t : t0) * v.rec_bytes + 16 * so, ok);
      }
      if (sym)
        for (int pos = tid; pos < TT; pos += kPfWorkers) {
          const int t = t0 + pos;
          const bool ok = t < J.len;
          cp_async4(dst0 + pos * p.b_stride + (OUT ? v.rec_bytes : 16 * p.ks16),
                    v.scales + (size_t)J.unit * v.cap + (ok ? t : t0), ok);
        }
      cp_async_commit();
    };

    // dequantised keys (and values) of the tile staged in buffer g into
    // stage s: threads [0, 4 TT) the keys by (position, channel quarter),
    // the output pass's other threads the values
    auto dequant = [&](int g, int s) {
      const uint8_t *bundle = sm + p.off_stg + g * p.stg_bytes + pidx * p.b_stride;
      uint8_t *kh = sm + p.off_k + s * p.stage, *kl = kh + 2 * KBOX;
      const int ks = 16 * p.ks16;  // K-section bytes
      const int mb = (p.nrec * 16 - 2 * ks) / 2;  // grouped: bytes of one metadata block
      const bool sym = p.fmt >= kFmtS8;
      if (part < 4) {
        const uint8_t *kmeta = !OUT ? bundle + ks : sym ? bundle + v.rec_bytes : bundle + 2 * ks;
        switch (p.fmt) {
          case kFmtBf16: tc_dequant<kFmtBf16, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
          case kFmtG8: tc_dequant<kFmtG8, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
          case kFmtG4: tc_dequant<kFmtG4, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
          case kFmtS8: tc_dequant<kFmtS8, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
          case kFmtS4: tc_dequant<kFmtS4, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
          default: tc_dequant<kFmtS2, KBOX>(bundle, kmeta, pidx, part, p.gshift, kh, kl); break;
        }
      } else if constexpr (OUT) {
        const int qc = part - 4;
        uint8_t *vh = kh + 2 * (p.k_lo ? 2 : 1) * KBOX, *vl = vh + 2 * KBOX;
        const uint8_t *vsec = bundle + ks;
        const uint8_t *vmeta = bundle + 2 * ks + mb;
        const float svs =
            sym ? __uint_as_float(*reinterpret_cast<const uint32_t *>(bundle + v.rec_bytes) & 0xFFFF0000u) : 0.f;
        switch (p.fmt) {
          case kFmtBf16: tc_dequant_v<kFmtBf16, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
          case kFmtG8: tc_dequant_v<kFmtG8, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
          case kFmtG4: tc_dequant_v<kFmtG4, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
          case kFmtS8: tc_dequant_v<kFmtS8, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
          case kFmtS4: tc_dequant_v<kFmtS4, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
          default: tc_dequant_v<kFmtS2, KBOX>(vsec, vmeta, svs, pidx, qc, p.gshift, vh, vl); break;
        }
      }
    };

    int kk = 0;
    for (int job = next_job(); job < p.n_jobs; job = next_job()) {
      if (failed) continue;
      const Job J = job_at(job);
      const int base = J.len - a.n_q;  // position of chunk query 0
      load_q(J);
      // this thread's row of the job in the score epilogues
      const int rl = 32 * quarter + lane;
      const bool row_live = rl < J.nr;
      const int last = base + (J.r0 + rl) / a.G;  // the last position the row sees
      const bool warp_live = 32 * quarter < J.nr;
      float m_run = -INFINITY, l_run = 0.f;  // statistics: this slice's running pair
      const bool pipe = p.nst == 2;
      // Stage tile kn (tile counter kkn): its records have landed; the values
      // the stage held are read (the value product of tile kkn - nst);
      // dequantised and announced to the MMA warp.  With two stages the next
      // tile is staged before this tile's scores are awaited, so that the
      // dequantisation overlaps the score product.
      auto stage_tile = [&](int kn, int kkn) -> bool {
        if (p.nstg == 2) {
          if (kn + 1 < J.n_t)
            stage_copy(J, kn + 1, (kkn + 1) & 1);  // the staging of tile kkn - 1, consumed
          else
            cp_async_commit();  // keeps the wait count uniform
          cp_async_wait<1>();
        } else {
          cp_async_wait<0>();
        }
        const bool ok = OUT ? wait_pv(kkn - p.nst) : true;
        if (workers_sync_or<kPfWorkers>(!ok)) return false;
        if (OUT || part < 4) dequant(kkn & (p.nstg - 1), kkn % p.nst);
        fence_proxy_async();  // the stage, written here, is read by the tensor cores
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar[kkn & 1]);
        if (p.nstg == 1 && kn + 1 < J.n_t) {
          workers_sync<kPfWorkers>();  // the one staging buffer is consumed
          stage_copy(J, kn + 1, 0);
        }
        return true;
      };
      if (J.n_t > 0) {
        stage_copy(J, 0, kk & (p.nstg - 1));
        if (!stage_tile(0, kk)) failed = true;
      }
      for (int k = 0; k < J.n_t && !failed; ++k, ++kk) {
        if (pipe && k + 1 < J.n_t && !stage_tile(k + 1, kk + 1)) { failed = true; break; }
        // scores of this tile; output pass: the P buffer is free
        bool ok = mbar_wait_sleepy(&bar[2 + (kk & 1)], (kk >> 1) & 1, kLimit, abort_flag, 2000);
        if (OUT && ok) ok = wait_pv(kk - 1);
        if (workers_sync_or<kPfWorkers>(!ok)) { failed = true; break; }
        tc_fence_after();
        const int t0 = k * TT;
        if constexpr (!OUT) {
          // online (max, sum) of this row over the slice's 32 positions
          if (warp_live) {
            float y[32];
            const uint32_t ta = tmem + 128u * (kk & 1) + 32 * slice + lane_off;
            {
              float z[16];
              tmem_ld16(ta, z);
#pragma unroll
              for (int i = 0; i < 16; ++i) y[i] = z[i];
              tmem_ld16(ta + 16, z);
#pragma unroll
              for (int i = 0; i < 16; ++i) y[16 + i] = z[i];
            }
            const int nv = min(32, last - (t0 + 32 * slice) + 1);
            if (row_live && nv > 0) {
              float mm = -INFINITY;
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < nv) mm = fmaxf(mm, y[i]);
              const float mn = fmaxf(m_run, mm * sg);
              float ll[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < nv) ll[i & 3] += fast_exp2(fmaf(y[i], sg, -mn));
              l_run = l_run * fast_exp2(m_run - mn) + ((ll[0] + ll[1]) + (ll[2] + ll[3]));
              m_run = mn;
            }
          }
        } else {
          // P of this row over the slice's 16 positions, hi and lo halves
          float y[16];
          tmem_ld16(tmem + 64u * (kk & 1) + 16 * slice + lane_off, y);
          const float c = norm[rl];
          const int tb = t0 + 16 * slice;
          float x0[8], x1[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            x0[i] = tb + i <= last ? fast_exp2(fmaf(y[i], sg, -c)) : 0.f;
            x1[i] = tb + 8 + i <= last ? fast_exp2(fmaf(y[8 + i], sg, -c)) : 0.f;
          }
          put8(ph, pl, true, rl, 16 * slice, kPfRows * 128, x0);
          put8(ph, pl, true, rl, 16 * slice + 8, kPfRows * 128, x1);
          fence_proxy_async();  // P, written here, is read by the tensor cores
        }
        tc_fence_before();
        __syncwarp();
        if (OUT && lane == 0) mbar_arrive(&bar[4]);
        // one stage: the next tile after this one's epilogue (and, in the
        // output pass, its value product)
        if (!pipe && k + 1 < J.n_t && !stage_tile(k + 1, kk + 1)) { failed = true; break; }
      }
      if (failed) {
        *abort_flag = 1;
        continue;
      }
      if constexpr (!OUT) {
        // the four slices' pairs of each row, combined
        red[slice * kPfRows + rl] = make_float2(m_run, l_run);
        workers_sync<kPfWorkers>();
        if (slice == 0 && row_live) {
          float M = -INFINITY;
#pragma unroll
          for (int s2 = 0; s2 < 4; ++s2) M = fmaxf(M, red[s2 * kPfRows + rl].x);
          float L = 0.f;
          if (M != -INFINITY)
#pragma unroll
            for (int s2 = 0; s2 < 4; ++s2) {
              const float2 e = red[s2 * kPfRows + rl];
              if (e.x != -INFINITY) L += e.y * fast_exp2(e.x - M);
            }
          a.stats[(size_t)J.unit * R + J.r0 + rl] = make_float2(M, L);
        }
        workers_sync<kPfWorkers>();
      } else {
        // O^T: lane = channel 32 quarter + lane, columns = the job's rows
        float o[32];
        if (J.n_t > 0) {
          if (!wait_pv(kk - 1)) failed = true;
          if (workers_sync_or<kPfWorkers>(failed)) { failed = true; *abort_flag = 1; continue; }
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
        const int d = 32 * quarter + lane;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int rr = 32 * slice + i;
          if (rr < J.nr) {
            const int r = J.r0 + rr;
            const int qi = r / a.G, h = J.j * a.G + (r - qi * a.G);
            a.out[(((size_t)J.b * a.n_q + qi) * a.Hq + h) * D + d] = o[i];
          }
        }
        tc_fence_before();
        workers_sync<kPfWorkers>();  // O^T read before the next job's first value product
      }
    }
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
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256)
                 : "memory");
  pdl_trigger();
}

// Shared-memory plan: the job's query rows (hi, then lo), the key (and
// value) stages, the staging buffers of raw records (strides odd multiples
// of 16 bytes), P (output pass), normalisers and slice statistics, barriers.
PfPlan pf_plan(const PfArgs &a, bool out, int sms) {
  PfPlan p;
  const int R = a.n_q * a.G;
  const int TT = out ? 64 : 128;
  p.n_rb = (R + kPfRows - 1) / kPfRows;
  p.n_jobs = a.v.B * a.v.Hkv * p.n_rb;
  p.q_lo = a.q_f32 ? 1 : 0;
  p.k_lo = a.v.bits != 16 ? 1 : 0;
  p.fmt = a.v.bits == 16 ? kFmtBf16
          : a.v.scheme == kSchemeSym ? (a.v.bits == 8 ? kFmtS8 : a.v.bits == 4 ? kFmtS4 : kFmtS2)
                                     : (a.v.bits == 8 ? kFmtG8 : kFmtG4);
  p.gshift = a.v.group == 64 ? 6 : 5;
  p.ks16 = TcFmtKs16(p.fmt);
  p.nrec = a.v.rec_bytes / 16;
  const bool sym = p.fmt >= kFmtS8;
  const int kmeta16 = (p.fmt == kFmtBf16 || sym) ? 0 : (p.nrec - 2 * p.ks16) / 2;
  p.ncopy = out ? p.nrec : p.ks16 + kmeta16;
  p.nc_magic = (uint32_t)((0x100000000ull + p.ncopy - 1) / p.ncopy);
  const int bchunks = (out ? p.nrec : p.ncopy) + (sym ? 1 : 0);
  p.b_stride = 16 * (bchunks % 2 ? bchunks : bchunks + 1);
  p.stg_bytes = TT * p.b_stride;
  const int kbox = TT * 128;
  p.stage = 2 * kbox * ((p.k_lo ? 2 : 1) * (out ? 2 : 1));
  p.off_ql = kPfRows * 256;
  const int qbytes = kPfRows * 256 * (p.q_lo ? 2 : 1);
  p.off_k = (qbytes + 1023) / 1024 * 1024;
  const int pbytes = out ? 2 * kPfRows * 128 : 0;
  const int tail = pbytes + kPfRows * 4 + 4 * kPfRows * 8 + 128 + 1024;
  auto fits = [&](int nst, int nstg) { return p.off_k + nst * p.stage + nstg * p.stg_bytes + tail <= 232448; };
  p.nst = fits(2, 1) ? 2 : 1;
  p.nstg = fits(p.nst, 2) ? 2 : 1;
  p.off_stg = p.off_k + p.nst * p.stage;
  p.off_p = (p.off_stg + p.nstg * p.stg_bytes + 1023) / 1024 * 1024;
  p.off_norm = p.off_p + pbytes;
  p.off_red = p.off_norm + kPfRows * 4;
  p.off_bar = p.off_red + 4 * kPfRows * 8;
  p.smem = p.off_bar + 128 + 1024;
  p.grid = std::max(1, std::min(p.n_jobs, sms));
  return p;
}

}  // namespace

bool prefill_plan_fits(const PfArgs &a) {
  const PfPlan s = pf_plan(a, false, 1), o = pf_plan(a, true, 1);
  return s.smem <= 232448 && o.smem <= 232448;
}

cudaError_t launch_gqa_prefill(const PfArgs &a, cudaStream_t st) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const PfPlan ps = pf_plan(a, false, sms), po = pf_plan(a, true, sms);
  cudaError_t e = cudaFuncSetAttribute(prefill_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       ps.smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(prefill_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, po.smem);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(a.counter, 0, 2 * sizeof(int), st);  // the job counters
  if (e == cudaSuccess)
    e = launch_pdl(prefill_kernel<false>, dim3(ps.grid), dim3(kPfThreads), ps.smem, st, a, ps);
  if (e == cudaSuccess)
    e = launch_pdl(prefill_kernel<true>, dim3(po.grid), dim3(kPfThreads), po.smem, st, a, po);
  return e;
}

}  // namespace kvk
