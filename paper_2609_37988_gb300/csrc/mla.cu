// mla.cu -- decode attention over a truncated MLA latent cache (Appendix C.2).
//
// The cache stores, per (sequence, position), the latent c[:d] (d = the
// layer's kept width, truncated on write) and the post-RoPE positional key
// k^R, both bf16.  With the content-key up-projection absorbed into the
// query, one decode step of head h is
//     q_lat = W_UK[h][:, :d]^T q_nope                      (absorb)
//     s_t   = sigma (<q_lat, c_t[:d]> + <q_pe, k^R_t>)      (latent scores)
//     o_lat = sum_t softmax_t(s) c_t[:d]                    (latent values)
//     out   = W_UV[h][:, :d] o_lat                          (up-projection)
// All heads of a sequence share the latent, so every cache byte is read once
// for all H heads and both contractions are dense enough for the tensor
// cores: the latent decode issues tcgen05.mma (operands staged by TMA tensor
// copies in shared memory, accumulators in TMEM); the small absorb and the
// merge + up-projection use mma.m16n8k16.  bf16 operands, fp32 accumulate;
// fp32 operands that must enter a bf16 product (q_lat, softmax weights,
// o_lat) are split into hi + lo bf16 halves, so products keep ~16
// significant bits.
#include <math.h>

#include <algorithm>

#include <cuda.h>  // CUtensorMap and its enums (the encoder is reached through the runtime)

#include "common.cuh"
#include "kernels.h"
#include "layout.h"
#include "mla_common.cuh"
#include "umma.cuh"

namespace kvk {
namespace {

// Latent split-K decode on the 5th-generation tensor cores.  Grid (split,
// query row / R); 8 warps: warps 0-3 run the softmax and the epilogue,
// warps 4, 6 and 7 issue the UMMAs, warp 5 the TMA copies.  Below, the
// operands are described for R = 1 (decode); with R = 2 (pairs of pre-fill
// rows) the query operand, S, P and O carry the two rows' 32 columns side by
// side.  Tiles of TR positions of [c[:W] | k^R] (TR = 48 for W = 512, so
// that three stages fit (two with R = 2), 128 for W = 64, else 64).
//
// Shared memory per stage: the tile as (W + 64)/64 boxes of TR positions x
// 64 coordinates, each box TR rows of 128 bytes in the 128-byte swizzled
// layout, written by TMA tensor copies (TR/BR per box, completing on the
// stage's mbarrier).  The same bytes serve both products:
//   scores  S[pos x 32] = C[pos x (W+64)] [Q_hi ; Q_lo]^T
//           (UMMA M=64 (rows past TR are ignored; M=128 for TR = 128),
//           N=32: columns 0-15 are the heads' q_lat hi (+ q_pe) parts,
//           16-31 their q_lat lo parts; A = the tile K-major);
//   values  O^T[W x 32] += C^T[W x TR pos] [P_hi | P_lo]
//           (UMMA M=128 latent rows (64 for W = 64), N = 16 heads hi + 16
//           heads lo, A = the tile read MN-major); O = columns h + 16+h.
// Score rows come back with tcgen05.ld (M=64 accumulator: row r in TMEM
// lane 32 (r/16) + r%16, so lane r%16 of softmax warp r/16 owns position r;
// M=128: lane r%32 of warp r/32):
// its 16 scores stay in registers; the online softmax is base 2 with a stale
// maximum kept within 2^8 (one vote per tile; maxima are reduced only when
// one rises).  The weights go hi/lo in bf16 into the P operand; O stays in
// TMEM until the end (rescaled in place on the rare tiles that raise a
// maximum).  Two score warps issue a tile's score products as soon as it
// has landed, each half of the K-steps into its own accumulator (the softmax
// adds the two), so a stage's chain (landing, scores, softmax, values) is
// short; the value warp issues values(t) as soon as P(t) is written; the
// copy warp refills a stage as soon as the values that read it completed.
// Every wait is bounded (an abort flag stops the other role); the CTA frees
// its TMEM on every path.
// rows of one TMA box (the anchor's tensor map) for kept width w
__host__ __device__ constexpr int mla_box_rows(int w) { return w == 512 ? 48 : 64; }
// positions per tile: 48 at d = 512 (three stages fit), 128 at d = 64 (M =
// 128 score products, every softmax lane owning a position, two CTAs per SM
// with two stages each), 64 otherwise.  Measured (B = 64, T = 4096 decode
// call; 4 x 1024-row pre-fill): 128-position tiles took d = 64 from 29.2 to
// 28.4 us per call and 0.63 to 0.54 ms per pre-fill; at d = 128 and 256 the
// calls were unchanged and the d = 128 pre-fill went 0.74 -> 0.80 ms.
__host__ __device__ constexpr int mla_tile_rows(int w, int r) {
  return w == 512 ? 48 : (r == 1 && w == 64) ? 128 : 64;
}

// R: query rows per CTA (pre-fill rows of one sequence share every tile;
// decode: R = 1).  The query operand, S, P and O have NQ = 32 R columns:
// row rho of the CTA, head h at 32 rho + h (hi part, with q_pe) and
// 32 rho + 16 + h (lo part).
template <int W, int R = 1>
struct MlaCfg {
  static constexpr int NQ = 32 * R;                   // Q rows; S, P, O columns
  static constexpr int NH = 16 * R;                   // (row, head) pairs of a CTA
  static constexpr int TR = mla_tile_rows(W, R);      // positions per tile
  static constexpr int BR = mla_box_rows(W);          // rows per TMA copy
  static constexpr int MS = TR > 64 ? 128 : 64;       // score UMMA M
  static constexpr int PNS = TR > 64 ? 2048 : 1024;   // P operand: bytes between 8-column blocks
  static constexpr int KH = W + kRope;                // hi extent: latent + rope
  static constexpr int BOXES = KH / 64;               // 64-coordinate boxes per tile
  static constexpr int BOX = TR * 128;                // bytes per box
  static constexpr int STAGE = BOXES * BOX;
  // stages: the decode is bound by the bytes in flight per SM, so as many
  // as shared memory holds beside the rest at the CTAs per SM each width
  // runs: four at d = 256 (the call 49.1 -> 45.5 us), three at d = 512 (two
  // with R = 2, whose query operand takes the room), three at d = 128 and
  // two at d = 64 (two CTAs per SM; one CTA per SM with eight or six stages
  // took the d = 128 call 33.9 -> 34.8 us and both pre-fills 15-45 % longer)
  static constexpr int NST = (R > 1 && W == 512) ? 2 : W == 256 ? 4 : TR > 64 ? 2 : 3;
  static constexpr int QB = NQ * KH * 2;              // [Q_hi ; Q_lo] operand (NQ rows)
  static constexpr int PB = 4 * PNS * R;              // [P_hi | P_lo] operand, 4 R column blocks
  static constexpr int OFF_Q = NST * STAGE;
  static constexpr int OFF_P = OFF_Q + QB;            // two buffers
  static constexpr int OFF_RED = OFF_P + 2 * PB;      // float [4][NH] maxima, [4][NH] sums
  static constexpr int OFF_BAR = OFF_RED + 512 * R;   // full[NST], sbar[2], pbar[2], obar[NST], dbar[3]
  static constexpr int NBAR = 2 * NST + 7;
  static constexpr int OFF_TB = OFF_BAR + 8 * NBAR;   // TMEM base address, abort flag
  static constexpr int SMEM = OFF_TB + 16 + 1024;     // + slack to align the base to 1024
  static constexpr int MV = W >= 128 ? 128 : 64;      // value UMMA M
  static constexpr int MB = W / MV;                   // value M-blocks
  static constexpr int OCOLS = NQ * MB;               // TMEM columns of O
  static constexpr int SCOLS = 4 * NQ;                // two S buffers of two K-halves
  static constexpr int TCOLS = OCOLS + SCOLS <= 128 ? 128 : OCOLS + SCOLS <= 256 ? 256 : 512;
  static_assert(KH % 64 == 0 && W % 64 == 0, "whole boxes");
  static_assert(TR % 16 == 0 && TR % BR == 0 && (TR <= 64 || TR == 128), "tile rows");
  static_assert(OCOLS + SCOLS <= TCOLS, "TMEM columns");
  static_assert(SMEM <= 232448, "shared memory");
  static_assert(R == 1 || R == 2, "one or two query rows per CTA");
};

// 2-D TMA tile load (x = coordinate, y = row) completing on `bar`
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *tmap, int x, int y,
                                            uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// warps: 0-3 softmax, 4 and 7 the score products of even and odd tiles, 5
// copies, 6 value products (one thread issues at most one tcgen05 product
// per ~45 cycles: the products come as three streams)
constexpr int kMlaThreads = 256;

template <int W, int R>
__global__ void __launch_bounds__(kMlaThreads, 1)
    mla_decode_kernel(const __grid_constant__ CUtensorMap tmap, const MlaView v,
                      const uint16_t *__restrict__ qlat, const uint16_t *__restrict__ q_pe, int H,
                      float sig, int items_per_split, int n_splits, float *__restrict__ partial,
                      int32_t *err) {
  using C = MlaCfg<W, R>;
  constexpr int NQ = C::NQ, NH = C::NH;
  constexpr int TR = C::TR;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  // full[s]: tile landed in stage s; sbar[i]: scores of a tile with parity i
  // done; pbar[i]: its weights written (4 arrivals); obar[s]: the values of
  // the tile in stage s done; dbar[3]: everything each MMA warp issued done
  uint64_t *full = reinterpret_cast<uint64_t *>(sm + C::OFF_BAR);
  uint64_t *sbar = full + C::NST, *pbar = sbar + 2, *obar = pbar + 2, *dbar = obar + C::NST;
  uint32_t *tbase = reinterpret_cast<uint32_t *>(sm + C::OFF_TB);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + C::OFF_TB + 4);
  float *red = reinterpret_cast<float *>(sm + C::OFF_RED);  // [4 warps][NH]
  float *lsum = red + 4 * NH;                               // [4 warps][NH]
  uint8_t *q_s = sm + C::OFF_Q;

  // query rows vb0 .. vb0 + R - 1 (decode: the sequence; pre-fill: R
  // consecutive chunk rows of one sequence, the last seeing the most)
  const int split = blockIdx.x, vb0 = blockIdx.y * R;
  const int b = mla_row_seq(v, vb0);             // the sequence whose cache it reads
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int len = mla_row_len(v, vb0 + R - 1, b);
  const int i0 = split * items_per_split;
  const int i1 = (split == n_splits - 1) ? len : min(i0 + items_per_split, len);
  const int n_tiles = i1 > i0 ? (i1 - i0 + TR - 1) / TR : 0;
  const int row0 = b * (int)v.cap + i0;  // tensor-map row of the split's first position
  constexpr uint32_t kLimit = 1u << 22;

  if (tid == 0) {
    for (int i = 0; i < C::NBAR; ++i) {
      const bool sb = i >= C::NST && i < C::NST + 2;      // both score warps commit
      const bool pb = i >= C::NST + 2 && i < C::NST + 4;  // the four softmax warps
      mbar_init(&full[i], pb ? 4 : sb ? 2 : 1);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tbase)),
                 "r"(C::TCOLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();  // barriers initialised, TMEM address published
  tc_fence_after();
  // The copy warp streams the cache at once: this kernel's CTAs start only
  // after every CTA of the absorb kernel passed its own wait for the work
  // enqueued before the call (which wrote the cache and the lengths).  The
  // other warps wait for the absorb itself before reading its q_lat.
  // Query operand, K-major core layout: row n, coordinate k at
  // (n/8) SBO + (k/8) 128 + (n%8) 16 + (k%8) 2 with SBO = (W+64)/8 128.
  // Rows 32 rho + h: [q_lat hi | q_pe] of head h of query row vb0 + rho;
  // rows 32 rho + 16 + h: [q_lat lo | 0].
  if (warp < 5 || warp == 7) {
    pdl_wait();
    constexpr int QROW = 2 * W + kRope;  // qlat row: [hi(W) | (unused 64) | lo(W)]
    // warps 0-4 stage it; the second score warp only waits for it
    for (int q = tid; warp < 5 && q < NQ * (C::KH / 8); q += 160) {  // 16-byte cp.async, zero-filled
      const int n = q / (C::KH / 8), c = q % (C::KH / 8);
      const int vb = vb0 + n / 32, nn = n & 31, h = nn & 15;
      const uint16_t *qb = qlat + (size_t)vb * H * QROW;
      const uint16_t *src = qb;
      const bool valid = h < H && (nn < 16 || c < W / 8);
      if (valid)
        src = nn >= 16    ? qb + (size_t)h * QROW + C::KH + 8 * c
              : c < W / 8 ? qb + (size_t)h * QROW + 8 * c
                          : q_pe + ((size_t)vb * H + h) * kRope + 8 * (c - W / 8);
      cp_async16(q_s + (n / 8) * (C::KH / 8 * 128) + c * 128 + (n % 8) * 16, src, valid);
    }
    cp_async_commit();
    cp_async_wait<0>();
    fence_proxy_async();
    tc_fence_before();
    asm volatile("bar.sync 2, 192;" ::: "memory");  // warps 0-4 and 7: the query is staged
    tc_fence_after();
  }
  const uint32_t tmem = *tbase;
  const uint32_t t_o = tmem, t_s = tmem + C::OCOLS;  // O columns, then two S buffers
  auto stage = [&](int s) { return sm + s * C::STAGE; };
  auto pbuf = [&](int ps) { return sm + C::OFF_P + ps * C::PB; };
  bool failed = false;

  if (warp == 5) {
    // ======================= copy warp ====================================
    int issued = 0;
    if (lane == 0) {
      for (; issued < n_tiles; ++issued) {
        const int s = issued % C::NST;
        // the stage's previous tile was read by its values
        if (issued >= C::NST &&
            !mbar_wait_or_abort(&obar[s], ((issued - C::NST) / C::NST) & 1, kLimit, abort_flag)) {
          *abort_flag = 1;
          set_err(err, 8);
          break;
        }
        fence_proxy_async();
        mbar_expect_tx(&full[s], C::STAGE);
#pragma unroll
        for (int j = 0; j < C::BOXES; ++j)
#pragma unroll
          for (int h = 0; h < TR / C::BR; ++h)
            tma_load_2d(stage(s) + j * C::BOX + h * C::BR * 128, &tmap, 64 * j,
                        row0 + issued * TR + h * C::BR, &full[s]);
      }
      // the last copies land before the CTA leaves (bounded; done at once
      // when they were consumed)
      for (int u = max(0, issued - C::NST); u < issued; ++u)
        mbar_wait(&full[u % C::NST], (u / C::NST) & 1, kLimit);
    }
    __syncwarp();
    pdl_trigger();
  } else if (warp == 4 || warp == 7) {
    // ======================= score warps ==================================
    // Both warps take every tile: warp 4 the first half of the K-steps into
    // its own accumulator, warp 7 the second half into another (the softmax
    // adds the two), so that a tile's scores take half the issue time.
    // Before tile t a warp waits for softmax(t-2) (the S buffer is free),
    // then for the tile's landing; both waits are for consecutive phases.
    const int role = warp == 4 ? 0 : 1;
    constexpr uint32_t ID_S = umma_idesc(C::MS, NQ, false, false);
    constexpr int KS = C::KH / 16, KHALF = KS / 2;
    static_assert(KS % 2 == 0, "K-steps split evenly over the two score warps");
    for (int t = 0; t < n_tiles && !failed; ++t) {
      const int s = t % C::NST;
      bool ok = true;
      if (t >= 2) ok = mbar_wait_or_abort(&pbar[t & 1], ((t - 2) >> 1) & 1, kLimit, abort_flag);
      if (ok) ok = mbar_wait_or_abort(&full[s], (t / C::NST) & 1, kLimit, abort_flag);
      // rows past the split's end: zero them (the cache may hold anything)
      const int nval = min(TR, i1 - (i0 + t * TR));
      if (ok && nval < TR) {
        for (int q = lane; q < C::BOXES * (TR - nval) * 8; q += 32) {
          const int j = q / ((TR - nval) * 8), rem = q % ((TR - nval) * 8);
          const int r = nval + rem / 8, u = rem % 8;
          *reinterpret_cast<uint4 *>(stage(s) + j * C::BOX + r * 128 + 16 * u) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async();
        __syncwarp();
      }
      if (ok && lane == 0) {  // this warp's half of scores(t) -> S[t & 1][role]
        tc_fence_after();
        const uint64_t dc = umma_desc(smem_u32(stage(s)), 16, 1024, 2);
        const uint64_t dq = umma_desc(smem_u32(q_s), 128, C::KH / 8 * 128, 0);
#pragma unroll
        for (int kk = 0; kk < KHALF; ++kk) {
          const int ks = role * KHALF + kk;
          umma_f16(t_s + NQ * (2 * (t & 1) + role),
                   dc + (uint64_t)(((ks / 4) * C::BOX + (ks % 4) * 32) >> 4), dq + (uint64_t)(ks * 16),
                   ID_S, kk > 0);
        }
        umma_commit(&sbar[t & 1]);  // one of the two arrivals
      }
      failed = !__all_sync(0xffffffffu, ok);
    }
    if (failed && lane == 0) {
      *abort_flag = 1;
      set_err(err, 8);
    }
    // every UMMA this warp issued lands before the CTA leaves (bounded)
    if (lane == 0) {
      umma_commit(&dbar[2 * role]);
      mbar_wait(&dbar[2 * role], 0, kLimit);
    }
    __syncwarp();
    pdl_trigger();
  } else if (warp == 6) {
    // ======================= value warp ===================================
    // values(t) once P(t) is written; it waits for every pbar phase in
    // order, and pbar(t + 2) needs obar(t), committed after values(t)
    constexpr uint32_t ID_V = umma_idesc(C::MV, NQ, true, true);
    for (int t = 0; t < n_tiles && !failed; ++t) {
      const bool ok = mbar_wait_or_abort(&pbar[t & 1], (t >> 1) & 1, kLimit, abort_flag);
      if (ok && lane == 0) {  // O^T[:, hi | lo] += C^T [P_hi | P_lo]
        tc_fence_after();
        const uint64_t da = umma_desc(smem_u32(stage(t % C::NST)), C::BOX, 1024, 2);
        const uint64_t dp = umma_desc(smem_u32(pbuf(t & 1)), 128, C::PNS, 0);
#pragma unroll
        for (int ks = 0; ks < TR / 16; ++ks)
#pragma unroll
          for (int mb = 0; mb < C::MB; ++mb)
            umma_f16(t_o + NQ * mb, da + (uint64_t)(((2 * mb) * C::BOX + ks * 2048) >> 4),
                     dp + (uint64_t)(ks * 16), ID_V, t > 0 || ks > 0);
        umma_commit(&obar[t % C::NST]);
      }
      failed = !__all_sync(0xffffffffu, ok);
    }
    if (failed && lane == 0) {
      *abort_flag = 1;
      set_err(err, 8);
    }
    if (lane == 0) {
      umma_commit(&dbar[1]);
      mbar_wait(&dbar[1], 0, kLimit);
    }
    __syncwarp();
    pdl_trigger();
  } else {
    // ======================= softmax warps ================================
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    // this lane's tile position: M = 128 scores put position r in TMEM lane
    // r; M = 64 in lane 32 (r/16) + r%16 (lanes 0-15 of each warp)
    constexpr bool ALL = C::MS == 128;
    constexpr int RL = ALL ? 32 : 16;  // lanes holding positions
    const int prow = ALL ? 32 * warp + lane : 16 * warp + lane;
    // each row's own end: row rho sees the positions below its causal limit
    int i1r[R];
#pragma unroll
    for (int r = 0; r < R; ++r) i1r[r] = R == 1 ? i1 : min(i1, mla_row_len(v, vb0 + r, b));
    float m_run[NH], l_part[NH];  // (row, head) pair j = 16 rho + h
#pragma unroll
    for (int j = 0; j < NH; ++j) { m_run[j] = -1e30f; l_part[j] = 0.f; }
    for (int t = 0; t < n_tiles; ++t) {
      const int base = i0 + t * TR;
      bool ok = mbar_wait_or_abort(&sbar[t & 1], (t >> 1) & 1, kLimit, abort_flag);
      // P buffer (t & 1) was read by values(t-2)
      if (ok && t >= 2)
        ok = mbar_wait_or_abort(&obar[(t - 2) % C::NST], ((t - 2) / C::NST) & 1, kLimit, abort_flag);
      if (softmax_sync_or(!ok)) { failed = true; break; }
      tc_fence_after();
      float x[NH];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        // hi and lo columns of both K-halves
        float hi[16], lo[16], hi2[16], lo2[16];
        const uint32_t sa = t_s + 2 * NQ * (t & 1) + 32 * r + lane_off;
        tmem_ld16(sa, hi);
        tmem_ld16(sa + 16, lo);
        tmem_ld16(sa + NQ, hi2);
        tmem_ld16(sa + NQ + 16, lo2);
        const bool live = (ALL || lane < 16) && prow < min(TR, i1r[r] - base);
#pragma unroll
        for (int h = 0; h < 16; ++h) x[16 * r + h] = live ? (hi[h] + hi2[h]) + (lo[h] + lo2[h]) : -INFINITY;
      }
      bool need = false;
#pragma unroll
      for (int j = 0; j < NH; ++j) need |= x[j] * sig > m_run[j] + 8.f;
      if (softmax_sync_or(need)) {
        // new maxima: reduce over the 16 rows of each warp, then the 4 warps
#pragma unroll
        for (int j = 0; j < NH; ++j) {
          float mx = x[j];
#pragma unroll
          for (int off = 1; off < RL; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
          if (lane == 0) red[warp * NH + j] = mx;
        }
        softmax_sync();
        float alpha[NH];
        bool any = false;
#pragma unroll
        for (int j = 0; j < NH; ++j) {
          const float mt = fmaxf(fmaxf(red[j], red[NH + j]), fmaxf(red[2 * NH + j], red[3 * NH + j])) * sig;
          alpha[j] = 1.f;
          if (mt > m_run[j] + 8.f) {  // stale maximum kept while within 2^8
            alpha[j] = fast_exp2(m_run[j] - mt);
            m_run[j] = mt;
            any = true;
          }
          l_part[j] *= alpha[j];
        }
        if (t >= 1 && any) {
          // O holds values up to t-1: wait for them, scale per head in TMEM
          ok = mbar_wait_or_abort(&obar[(t - 1) % C::NST], ((t - 1) / C::NST) & 1, kLimit, abort_flag);
          if (softmax_sync_or(!ok)) { failed = true; break; }
          tc_fence_after();
#pragma unroll
          for (int mb = 0; mb < C::MB; ++mb)
#pragma unroll
            for (int c = 0; c < 2 * R; ++c) {  // column block c: row c/2, hi or lo
              float o[16];
              tmem_ld16(t_o + NQ * mb + 16 * c + lane_off, o);
#pragma unroll
              for (int h = 0; h < 16; ++h) o[h] *= alpha[16 * (c / 2) + h];
              tmem_st16(t_o + NQ * mb + 16 * c + lane_off, o);
            }
        }
        softmax_sync();  // `red` is reused by the next vote
      }
      // weights hi/lo in bf16 into the MN-major P operand: position k, column
      // n (32 rho + h hi, 32 rho + 16 + h lo) at (k/8) 128 + (n/8) PNS +
      // (k%8) 16 + (n%8) 2
      if ((ALL || lane < 16) && prow < TR) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
          uint32_t hw[8], lw[8];
#pragma unroll
          for (int h = 0; h < 16; h += 2) {
            const int j = 16 * r + h;
            const float p0 = fast_exp2(fmaf(x[j], sig, -m_run[j]));
            const float p1 = fast_exp2(fmaf(x[j + 1], sig, -m_run[j + 1]));
            l_part[j] += p0;
            l_part[j + 1] += p1;
            split2<true>(p0, p1, hw[h / 2], lw[h / 2]);
          }
          uint8_t *pp = pbuf(t & 1) + 4 * C::PNS * r + (prow / 8) * 128 + (prow % 8) * 16;
          *reinterpret_cast<uint4 *>(pp) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *reinterpret_cast<uint4 *>(pp + C::PNS) = make_uint4(hw[4], hw[5], hw[6], hw[7]);
          *reinterpret_cast<uint4 *>(pp + 2 * C::PNS) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
          *reinterpret_cast<uint4 *>(pp + 3 * C::PNS) = make_uint4(lw[4], lw[5], lw[6], lw[7]);
        }
      }
      fence_proxy_async();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pbar[t & 1]);  // one of the four arrivals
    }
    pdl_trigger();
    // ---- partial of this split: O^T columns 32 rho + h + 32 rho + 16 + h, m, l
    if (!failed && n_tiles > 0) {
      const int t = n_tiles - 1;
      const bool ok = mbar_wait_or_abort(&obar[t % C::NST], (t / C::NST) & 1, kLimit, abort_flag);
      failed = softmax_sync_or(!ok);
    }
    if (failed && tid == 0) {
      *abort_flag = 1;
      set_err(err, 8);
    }
    if (!failed) {
      tc_fence_after();
      const size_t RS = (size_t)W + 2;
      const size_t prow_base = ((size_t)split * mla_rows(v) + vb0) * H;  // + rho H: row rho
#pragma unroll
      for (int j = 0; j < NH; ++j) {
        float sum = l_part[j];
#pragma unroll
        for (int off = 1; off < RL; off <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
        if (lane == 0) lsum[warp * NH + j] = sum;
      }
#pragma unroll
      for (int mb = 0; mb < C::MB; ++mb)
#pragma unroll
        for (int rho = 0; rho < R; ++rho) {
          float o[16];
          if (n_tiles > 0) {
            float lo[16];
            tmem_ld16(t_o + NQ * mb + 32 * rho + lane_off, o);
            tmem_ld16(t_o + NQ * mb + 32 * rho + 16 + lane_off, lo);
#pragma unroll
            for (int h = 0; h < 16; ++h) o[h] += lo[h];
          } else {
#pragma unroll
            for (int h = 0; h < 16; ++h) o[h] = 0.f;
          }
          // latent row of this lane: M=128 blocks use every lane; the M=64
          // block (W = 64) holds row 16 warp + lane in lanes 0-15
          const int r = C::MV == 128 ? 128 * mb + 32 * warp + lane : 16 * warp + lane;
          if (C::MV == 128 || lane < 16) {
#pragma unroll
            for (int h = 0; h < 16; ++h)
              if (h < H) partial[(prow_base + (size_t)rho * H + h) * RS + r] = o[h];
          }
        }
      softmax_sync();
      if (tid < H * R) {
        const int rho = R == 1 ? 0 : tid / H, j = 16 * rho + tid - rho * H;
        const float L = lsum[j] + lsum[NH + j] + lsum[2 * NH + j] + lsum[3 * NH + j];
        float mh = m_run[0];
#pragma unroll
        for (int jj = 1; jj < NH; ++jj) mh = (j == jj) ? m_run[jj] : mh;
        float *pr = partial + (prow_base + tid) * RS;
        pr[W] = (L > 0.f) ? mh : -INFINITY;
        pr[W + 1] = L;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 4)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TCOLS)
                 : "memory");
}

// ---------------------------------------------------------------------------
// Kernel attributes of the latent decode: its dynamic shared memory, and the
// largest shared-memory carveout (with no preference the occupancy query
// sizes the carveout for one CTA per SM, although two CTAs of the narrower
// widths fit).
template <int W, int R = 1>
cudaError_t mla_decode_attrs() {
  auto k = mla_decode_kernel<W, R>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, MlaCfg<W, R>::SMEM);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

// R = 2 (two query rows per CTA) for pre-fill calls whose sequences hold an
// even number of query rows, so that the pairs never straddle two sequences:
// every tile then serves both rows (the score product's N = 64, one issue).
template <int W, int R>
cudaError_t launch_mla_t(const MlaDecodeArgs &a, cudaStream_t st) {
  using C = MlaCfg<W, R>;
  if (a.n_splits > 64) return cudaErrorInvalidValue;  // merge weights hold 64 splits
  const int B = mla_rows(a.v);  // query rows
  if (R > 1 && (a.v.n_q % R != 0)) return cudaErrorInvalidValue;
  auto k = mla_decode_kernel<W, R>;
  constexpr int MU_SMEM = (64 * (W + 8)) * 2 + (2 * 64 * 16 + 16) * 4;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = mla_decode_attrs<W, R>();
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(mla_merge_upv_kernel<W>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               MU_SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaError_t e = launch_pdl(mla_absorb_kernel<W>, dim3(W / 64, a.H, (B + 15) / 16), dim3(128), 0,
                             st, static_cast<const uint16_t *>(a.q_nope),
                             static_cast<const uint16_t *>(a.q_pe),
                             static_cast<const uint16_t *>(a.w_uk), B, a.H, a.r, a.qlat);
  if (e == cudaSuccess)
    e = launch_pdl(k, dim3(a.n_splits, B / R), dim3(kMlaThreads), C::SMEM, st,
                   *static_cast<const CUtensorMap *>(a.tmap), a.v,
                   static_cast<const uint16_t *>(a.qlat), static_cast<const uint16_t *>(a.q_pe),
                   a.H, a.sig_log2, a.items_per_split, a.n_splits, a.partial, a.err);
  if (e == cudaSuccess)
    e = launch_pdl(mla_merge_upv_kernel<W>, dim3(a.H, (B + 15) / 16, 4), dim3(128), MU_SMEM, st,
                   static_cast<const float *>(a.partial), a.n_splits,
                   static_cast<const uint16_t *>(a.w_uv), B, a.H, a.r, a.out);
  return e;
}

// Latent decode CTAs that fit on one SM, from the kernel's registers and
// shared memory and its TMEM columns (the runtime's occupancy query answers
// one for this kernel at any size, while two CTAs of the narrower widths do
// run side by side).
template <int W>
int mla_ctas_t() {
  using C = MlaCfg<W>;
  auto k = mla_decode_kernel<W, 1>;
  if (mla_decode_attrs<W>() != cudaSuccess) return 1;
  cudaFuncAttributes fa;
  int dev = 0, smem_sm = 0, regs_sm = 0, resv = 0;
  if (cudaFuncGetAttributes(&fa, k) != cudaSuccess || cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&resv, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess)
    return 1;
  const int warp_regs = (fa.numRegs * 32 + 255) / 256 * 256;  // allocation unit: 256
  const int by_regs = regs_sm / (kMlaThreads / 32 * warp_regs);
  const int by_smem = smem_sm / (C::SMEM + resv);
  const int by_tmem = 512 / C::TCOLS;
  const int n = std::min(std::min(by_regs, by_smem), std::min(by_tmem, 2048 / kMlaThreads));
  return n > 0 ? n : 1;
}

}  // namespace

// Tensor map of an MLA anchor's records for the decode kernel: a 2-D view
// [B cap rows x (width + rope) bf16], boxes of 64 x 64 with the 128-byte
// swizzle (the UMMA operand layout).  The encoder is the driver's
// cuTensorMapEncodeTiled, reached through the runtime's entry-point query so
// the library links the static runtime only.
cudaError_t mla_make_tmap(void *out, const MlaView &v) {
  const uint64_t dims[2] = {(uint64_t)(v.width + v.rope), (uint64_t)v.B * (uint64_t)v.cap};
  const uint64_t strides[1] = {(uint64_t)v.rec_bytes};
  const uint32_t box[2] = {64, (uint32_t)mla_box_rows(v.width)};
  const uint32_t estr[2] = {1, 1};
  return encode_tensor_map_tiled(out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, v.rec, dims, strides, box,
                                 estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

cudaError_t launch_mla_decode(const MlaDecodeArgs &a, cudaStream_t st) {
  if (a.v.bits != 16) return launch_mla_decode_q(a, st);
  if (!a.tmap) return cudaErrorInvalidValue;
  // pre-fill rows in pairs where the score products bound a tile (d >= 256:
  // 2.75 -> 2.19 ms at d = 512, 1.54 -> 1.01 ms at d = 256 for 4 x 1024
  // rows); at d <= 128 the softmax bounds it and pairs gain nothing
  const bool pairs = a.v.n_q > 0 && a.v.n_q % 2 == 0;
  switch (a.v.width) {
    case 512: return pairs ? launch_mla_t<512, 2>(a, st) : launch_mla_t<512, 1>(a, st);
    case 256: return pairs ? launch_mla_t<256, 2>(a, st) : launch_mla_t<256, 1>(a, st);
    case 128: return launch_mla_t<128, 1>(a, st);
    case 64: return launch_mla_t<64, 1>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

int mla_decode_ctas_per_sm(int width, int bits) {
  if (bits != 16) return 1;  // quantised latents: 16 warps and up to 227 KB of shared memory
  switch (width) {
    case 512: return mla_ctas_t<512>();
    case 256: return mla_ctas_t<256>();
    case 128: return mla_ctas_t<128>();
    case 64: return mla_ctas_t<64>();
    default: return 1;
  }
}

}  // namespace kvk
