// mla_q.cu -- MLA decode over a quantised latent cache: the three axes of a
// layer's plan together (Sec. 2.1: a kept latent width, codes of 8, 4 or 2
// bits, and sharing by later layers; Appendix C.2 truncation with the
// quantisers of Appendix C.3).
//
// Each position stores its kept latent c[:W] and its positional key k^R as
// one quantised vector each: x = s u + z with unsigned codes u and, per
// vector, a scale s and an offset z (symmetric scheme: z = -q s; grouped
// scheme: z = the vector's minimum); the decode reads them centred, x =
// s (u - C0) + (z + C0 s).  A vector's (s, z) are constant over its
// coordinates, so both products keep the (centred) codes as operands:
//   score_t  = sigma ( s_t <q_lat, u_t> + z_t sum(q_lat)
//                    + s^R_t <q_pe, u^R_t> + z^R_t sum(q_pe) )
//   o_lat    = sum_t p_t (s_t u_t + z_t) / sum_t p_t
//            = ( sum_t (p_t s_t) u_t + sum_t p_t z_t ) / sum_t p_t .
// The codes enter the tcgen05 products as exact f16 subnormals (the bit
// pattern u is the half u 2^-24), the query and the value weights p s as f16
// hi + lo halves, fp32 accumulation in TMEM; the latent and positional parts
// of the score accumulate in separate TMEM columns so that each gets its
// own scale.  The tensor-core work per position equals the bf16 latent
// decode's (mla.cu): the quantisation only changes the bytes read and adds
// an expansion of the codes into the operand layout in shared memory.
#include <math.h>

#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"
#include "mla_common.cuh"
#include "umma.cuh"

namespace kvk {
namespace {

// Grid (split, query row); 16 warps:
//   0-3   softmax and epilogue (TMEM lane = tile position, as in mla.cu);
//   4, 7  score products (each tile's k-steps split between the two);
//   5     idle (keeps the warpgroups aligned);
//   6     value products;
//   8-15  expansion of a tile's codes, read from global memory (L2
//         prefetched a few tiles ahead), into the f16 operand layout.
// NST operand stages (the f16 tile as (W + 64) / 64 boxes of TR rows x 128
// bytes in the 128-byte swizzled K-major layout, plus the tile's
// per-position (s, z', s^R, z'^R)): tiles of 128 positions (score products
// M = 128, TMEM lane = position) where two stages fit, else 64 (M = 64,
// lanes 0-15 of each lane quarter), and as many stages (up to 4) as shared
// memory holds beside the query and the weights (a tile's stage is busy
// from its expansion through its value products, so the stage count bounds
// how many tiles are in that chain at once).
constexpr int kMlaQThreads = 512;
constexpr int kExpWarps = 8;                 // warps 8-15
constexpr int kExpThreads = 32 * kExpWarps;
constexpr uint32_t kSleepNs = 256;           // suspend hint of the role loops' barrier waits
constexpr int kMlaQSmemMax = 232448;

template <int W, int BITS, bool SYM>
struct MlaQTile {
  static constexpr int KH = W + kRope;
  static constexpr int pns(int TR) { return TR * 16 > 1024 ? TR * 16 : 1024; }
  // shared memory besides the stages: query, weights, sums, barriers
  static constexpr int fixed(int TR) { return 32 * KH * 2 + 2 * 4 * pns(TR) + 128 + 768 + 8 * 24 + 16 + 1024; }
  static constexpr int stage(int TR) { return (KH / 64) * TR * 128 + TR * 16; }
  static constexpr int nst(int TR) { return (kMlaQSmemMax - fixed(TR)) / stage(TR); }
  static constexpr int TR = nst(128) >= 2 ? 128 : 64;
  static constexpr int NST = nst(TR) < 4 ? nst(TR) : 4;
};

template <int W, int BITS, bool SYM>
struct MlaQCfg {
  static constexpr int TR = MlaQTile<W, BITS, SYM>::TR;  // positions per tile
  static constexpr int SM = TR == 128 ? 128 : 64;       // score product M
  static constexpr int KH = W + kRope;
  static constexpr int BOXES = KH / 64;
  static constexpr int BOX = TR * 128;
  static constexpr int OSTAGE = BOXES * BOX;          // f16 operand tile
  static constexpr int NST = MlaQTile<W, BITS, SYM>::NST;
  static constexpr int REC = KH * BITS / 8;           // stored record bytes
  static constexpr int MB = SYM ? 4 : 16;             // metadata bytes per position
  static constexpr int PF = 4;                        // tiles prefetched into L2 ahead
  static constexpr int OMETA = TR * 16;               // float4 (s, z, s^R, z^R) per position
  static constexpr int QB = 32 * KH * 2;
  static constexpr int PNS = TR * 16 > 1024 ? TR * 16 : 1024;  // P: stride of 8-column groups
  static constexpr int PB = 4 * PNS;
  static constexpr int OFF_OM = NST * OSTAGE;
  static constexpr int OFF_Q = OFF_OM + NST * OMETA;
  static constexpr int OFF_P = OFF_Q + QB;
  static constexpr int OFF_QS = OFF_P + 2 * PB;       // float [2][16] query sums (latent, rope)
  static constexpr int OFF_RED = OFF_QS + 128;        // float [4][16] maxima, sums, zero sums
  static constexpr int OFF_BAR = OFF_RED + 3 * 256;
  static constexpr int NSB = 4;                       // score buffers in TMEM
  // full[NST], sbar[NSB], pbar[2], obar[NST], dbar[3], sfree[NSB]
  static constexpr int NBAR = 2 * NST + 2 * NSB + 5;
  static constexpr int OFF_TB = OFF_BAR + 8 * NBAR;
  static constexpr int SMEM = OFF_TB + 16 + 1024;
  static constexpr int MV = W >= 128 ? 128 : 64;
  static constexpr int MBL = W / MV;                  // value M-blocks
  static constexpr int OCOLS = 32 * MBL;
  // the score k-steps of a tile split between the two score warps: warp 4
  // takes latent k-steps [0, KA), warp 7 the rest and the positional ones,
  // each into accumulators of its own (32 columns: 16 heads hi | lo)
  static constexpr int KL = W / 16, KA = (KL + kRope / 16) / 2, KB = KL - KA;
  static constexpr int SBUF = KB > 0 ? 96 : 64;      // [A | B | rope] columns per buffer
  static constexpr int SCOLS = SBUF * NSB;
  static constexpr int TCOLS = 512;
  static_assert(NST >= 2, "operand stages");
  static_assert(OCOLS + SCOLS <= TCOLS, "TMEM columns");
  static_assert(REC % 16 == 0 && (TR * MB) % 16 == 0, "prefetch sizes");
  static_assert(OSTAGE % 1024 == 0 && OFF_Q % 16 == 0 && OFF_P % 16 == 0, "alignment");
  static_assert(SMEM <= kMlaQSmemMax, "shared memory");
  static_assert(BITS == 8 || BITS == 4 || (BITS == 2 && SYM), "code widths");
};


// The stored bytes of one chunk of 8 codes (BITS bytes) and their f16 pairs
// (code 2p, code 2p + 1) * 2^-24.
template <int BITS>
struct RawChunk {
  using T = typename std::conditional<BITS == 8, uint2, uint32_t>::type;
};
// one chunk's stored bytes, from global memory through the read-only path
template <int BITS>
__device__ __forceinline__ typename RawChunk<BITS>::T ldg_chunk(const uint8_t *src) {
  if constexpr (BITS == 8) return __ldg(reinterpret_cast<const uint2 *>(src));
  else if constexpr (BITS == 4) return __ldg(reinterpret_cast<const unsigned int *>(src));
  else return __ldg(reinterpret_cast<const unsigned short *>(src));
}
// prefetch `bytes` (a multiple of 16, from a 16-byte aligned address) into L2
__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}
template <int BITS>
__device__ __forceinline__ uint4 expand_chunk(typename RawChunk<BITS>::T w) {
  if constexpr (BITS == 8) {
    return make_uint4(__byte_perm(w.x, 0u, 0x4140), __byte_perm(w.x, 0u, 0x4342),
                      __byte_perm(w.y, 0u, 0x4140), __byte_perm(w.y, 0u, 0x4342));
  } else if constexpr (BITS == 4) {
    return make_uint4(w & 0x000F000Fu, (w >> 4) & 0x000F000Fu, (w >> 8) & 0x000F000Fu,
                      (w >> 12) & 0x000F000Fu);
  } else {
    const uint32_t z = __byte_perm(w, 0u, 0x4140);  // byte 1 to bits 16..23
    return make_uint4(z & 0x00030003u, (z >> 2) & 0x00030003u, (z >> 4) & 0x00030003u,
                      (z >> 6) & 0x00030003u);
  }
}

template <int W, int BITS, bool SYM>
__global__ void __launch_bounds__(kMlaQThreads, 1)
    mla_decode_q_kernel(const MlaView v, const uint16_t *__restrict__ qlat,
                        const uint16_t *__restrict__ q_pe, int H, float sig, int items_per_split,
                        int n_splits, float *__restrict__ partial, int32_t *err, uint32_t wait_limit) {
  using C = MlaQCfg<W, BITS, SYM>;
  constexpr int TR = C::TR, KH = C::KH;
  constexpr float kCodeScale = 16777216.f;  // codes enter the products as u * 2^-24
  extern __shared__ uint8_t smem_raw[];
  uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t *full = reinterpret_cast<uint64_t *>(sm + C::OFF_BAR);
  uint64_t *sbar = full + C::NST, *pbar = sbar + C::NSB, *obar = pbar + 2, *dbar = obar + C::NST;
  uint64_t *sfree = dbar + 3;
  uint32_t *tbase = reinterpret_cast<uint32_t *>(sm + C::OFF_TB);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + C::OFF_TB + 4);
  float *red = reinterpret_cast<float *>(sm + C::OFF_RED);  // [4 warps][16] maxima
  float *lsum = red + 4 * kHeads;                           // [4 warps][16] sums
  float *zsum = lsum + 4 * kHeads;                          // [4 warps][16] value zero terms
  float *qsum = reinterpret_cast<float *>(sm + C::OFF_QS);  // [latent, rope][16]
  uint8_t *q_s = sm + C::OFF_Q;

  const int split = blockIdx.x, vb = blockIdx.y;  // vb: the query row (decode: sequence)
  const int b = mla_row_seq(v, vb);              // the sequence whose cache it reads
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int len = mla_row_len(v, vb, b);
  const int i0 = split * items_per_split;
  const int i1 = (split == n_splits - 1) ? len : min(i0 + items_per_split, len);
  const int n_tiles = i1 > i0 ? (i1 - i0 + TR - 1) / TR : 0;
  const size_t pos0 = (size_t)b * v.cap;  // slab of sequence b
  // waits in the tile loops poll at most wait_limit times; the final waits
  // for a role's own copies and products (before the CTA leaves) kLimit
  constexpr uint32_t kLimit = 1u << 22;

  if (tid == 0) {
    for (int i = 0; i < C::NBAR; ++i) {
      // full: one arrival per expansion warp; pbar and sfree: per softmax
      // warp; sbar: per score warp; the rest: one (a commit)
      const int o_pbar = C::NST + C::NSB, o_sfree = 2 * C::NST + C::NSB + 5;
      const bool exp = i < C::NST;
      const bool four = (i >= o_pbar && i < o_pbar + 2) || i >= o_sfree;
      const bool two = i >= C::NST && i < C::NST + C::NSB;  // sbar: both score warps commit
      mbar_init(&full[i], exp ? kExpWarps : four ? 4 : two ? 2 : 1);
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
  // Query operand (f16), K-major core layout: row n, coordinate k at
  // (n/8) SBO + (k/8) 128 + (n%8) 16 + (k%8) 2, SBO = KH/8 128.  Rows 0-15:
  // [q_lat hi | q_pe hi] of head n; rows 16-31: [q_lat lo | q_pe lo] of head
  // n - 16.  The latent halves come from the absorb (f16 hi/lo); q_pe (bf16)
  // is split here.  Warps 0-4 stage it; the second score warp waits for it.
  if (warp < 5 || warp == 7) {
    pdl_wait();
    constexpr int QROW = 2 * W + kRope;  // qlat row: [hi(W) | (64 unused) | lo(W)]
    const uint16_t *qb = qlat + (size_t)vb * H * QROW;
    auto qdst = [&](int n, int c) { return q_s + (n / 8) * (KH / 8 * 128) + c * 128 + (n % 8) * 16; };
    if (warp < 5) {
      for (int q = tid; q < 32 * (W / 8); q += 160) {  // latent parts: 16-byte cp.async
        const int n = q / (W / 8), c = q % (W / 8), h = n & 15;
        const bool valid = h < H;
        const uint16_t *src = valid ? qb + (size_t)h * QROW + (n >= 16 ? KH : 0) + 8 * c : qb;
        cp_async16(qdst(n, c), src, valid);
      }
      for (int q = tid; q < 16 * (kRope / 8); q += 160) {  // positional parts: hi and lo rows
        const int h = q / (kRope / 8), c = q % (kRope / 8);
        uint4 hi = make_uint4(0, 0, 0, 0), lo = hi;
        if (h < H) {
          const uint4 w = *reinterpret_cast<const uint4 *>(q_pe + ((size_t)vb * H + h) * kRope + 8 * c);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
          uint32_t hs[4], ls[4];
#pragma unroll
          for (int i = 0; i < 4; ++i)
            split2<false>(__uint_as_float(ws[i] << 16), __uint_as_float(ws[i] & 0xffff0000u), hs[i], ls[i]);
          hi = make_uint4(hs[0], hs[1], hs[2], hs[3]);
          lo = make_uint4(ls[0], ls[1], ls[2], ls[3]);
        }
        *reinterpret_cast<uint4 *>(qdst(h, W / 8 + c)) = hi;
        *reinterpret_cast<uint4 *>(qdst(16 + h, W / 8 + c)) = lo;
      }
    }
    cp_async_commit();
    cp_async_wait<0>();
    fence_proxy_async();
    tc_fence_before();
    asm volatile("bar.sync 2, 192;" ::: "memory");  // warps 0-4 and 7: the query is staged
    tc_fence_after();
  }
  const uint32_t tmem = *tbase;
  const uint32_t t_o = tmem, t_s = tmem + C::OCOLS;  // O columns, then NSB S buffers of 64
  auto ostage = [&](int s) { return sm + s * C::OSTAGE; };
  auto ometa = [&](int s) { return reinterpret_cast<float4 *>(sm + C::OFF_OM + s * C::OMETA); };
  auto pbuf = [&](int ps) { return sm + C::OFF_P + ps * C::PB; };
  bool failed = false;

  // Register split over the warpgroups (launched with 128 per thread, 65536
  // in all): expansion 80 + 80, products 96, softmax 256, in all
  // (80 + 80 + 96 + 256) x 128 = 65536; each warpgroup's role begins with its
  // own (the softmax increase waits for the decreases).
  if (warp >= 8) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 80;\n" ::: "memory");
    // ======================= expansion warps ==============================
    // tile t -> operand stage t % NST (free once the values of tile t - NST
    // were computed); rows past the split's end are zero, with zero scales
    const int et = tid - 256;  // 0 .. kExpThreads - 1
    // codes are centred on C0 (symmetric: q, so the operand is the signed
    // code itself and the offset term vanishes; grouped: the mid code), by an
    // exact f16 subtraction of subnormals: u - C0 with the offset moved into
    // z' = z + C0 s, which keeps the fp32 accumulations free of a large
    // common offset that would cancel at the end
    constexpr int kC0 = SYM ? (1 << (BITS - 1)) - 1 : 1 << (BITS - 1);
    constexpr uint32_t kC0Pair = (uint32_t)kC0 * 0x00010001u;
    // chunk q = et + 256 i of a tile (8 codes): row q / (KH / 8), chunk
    // q % (KH / 8); its raw and operand offsets are the same in every tile
    // (threads past the last chunk repeat it: the same bytes, written twice)
    constexpr int kCpr = KH / 8, kJobs = TR * kCpr;
    constexpr int kPer = (kJobs + kExpThreads - 1) / kExpThreads;
    // offsets of chunk i of this thread, recomputed where used (registers go
    // to the loads in flight)
    auto roff = [&](int i) {
      const int q = min(et + kExpThreads * i, kJobs - 1), row = q / kCpr;
      return row * C::REC + (q - row * kCpr) * BITS;
    };
    auto soff = [&](int i) {
      const int q = min(et + kExpThreads * i, kJobs - 1), row = q / kCpr, c8 = q - row * kCpr;
      return (c8 / 8) * C::BOX + row * 128 + 16 * ((c8 % 8) ^ (row % 8));
    };
    // the split's records and metadata rows in global memory; tiles are
    // prefetched into L2 PF ahead of the expansion (a hint, no completion)
    const uint8_t *grec = v.rec + (pos0 + i0) * C::REC;
    const uint8_t *gmeta = v.meta + (pos0 + i0) * C::MB;
    auto prefetch = [&](int u) {
      if (et == 0 && u < n_tiles) {
        const int nv = min(TR, i1 - (i0 + u * TR));
        prefetch_l2(grec + (size_t)u * TR * C::REC, (uint32_t)(nv * C::REC));
        prefetch_l2(gmeta + (size_t)u * TR * C::MB, (uint32_t)(((nv * C::MB + 15) / 16) * 16));
      }
    };
    for (int u = 0; u < C::PF; ++u) prefetch(u);
    for (int t = 0; t < n_tiles; ++t) {
      const int s = t % C::NST;
      prefetch(t + C::PF);
      bool ok = true;
      if (t >= C::NST)
        ok = mbar_wait_sleepy(&obar[s], ((t - C::NST) / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
      if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
      const int nval = min(TR, i1 - (i0 + t * TR));
      const uint8_t *raw = grec + (size_t)t * TR * C::REC;
      const uint8_t *rmeta = gmeta + (size_t)t * TR * C::MB;
      uint8_t *ost = ostage(s);
      // this thread's metadata row (at most one: TR <= 256), loaded first
      const int mrow = et;
      uint4 mw = make_uint4(0, 0, 0, 0);
      if (mrow < nval) {
        if constexpr (SYM) mw.x = __ldg(reinterpret_cast<const uint32_t *>(rmeta) + mrow);
        else mw = __ldg(reinterpret_cast<const uint4 *>(rmeta) + mrow);
      }
      if (nval == TR) {
        // every load of the tile before the first use
        typename RawChunk<BITS>::T w[kPer];
#pragma unroll
        for (int i = 0; i < kPer; ++i) w[i] = ldg_chunk<BITS>(raw + roff(i));
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
          const uint4 x = expand_chunk<BITS>(w[i]);
          *reinterpret_cast<uint4 *>(ost + soff(i)) =
              make_uint4(hsub2_u32(x.x, kC0Pair), hsub2_u32(x.y, kC0Pair), hsub2_u32(x.z, kC0Pair),
                         hsub2_u32(x.w, kC0Pair));
        }
      } else {
        // the split's last, partial tile: rows past its end are zero
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
          uint4 x = make_uint4(0, 0, 0, 0);
          if ((int)(roff(i) / C::REC) < nval) {
            x = expand_chunk<BITS>(ldg_chunk<BITS>(raw + roff(i)));
            x = make_uint4(hsub2_u32(x.x, kC0Pair), hsub2_u32(x.y, kC0Pair), hsub2_u32(x.z, kC0Pair),
                           hsub2_u32(x.w, kC0Pair));
          }
          *reinterpret_cast<uint4 *>(ost + soff(i)) = x;
        }
      }
      if (mrow < TR) {
        float4 m = make_float4(0.f, 0.f, 0.f, 0.f);
        if (mrow < nval) {
          if constexpr (SYM) {
            // x = s (u - q): centred on q, no offset
            m = make_float4(__uint_as_float(mw.x << 16), 0.f, __uint_as_float(mw.x & 0xffff0000u), 0.f);
          } else {
            m = make_float4(__uint_as_float(mw.x), __uint_as_float(mw.y), __uint_as_float(mw.z),
                            __uint_as_float(mw.w));
            m.y = fmaf((float)kC0, m.x, m.y);
            m.w = fmaf((float)kC0, m.z, m.w);
          }
        }
        ometa(s)[mrow] = m;
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&full[s]);
      }
    }
    if (failed && lane == 0) {
      *abort_flag = 1;
      set_err(err, 8);
    }
    __syncwarp();
    pdl_trigger();
  } else if (warp >= 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 96;\n" ::: "memory");
    if (warp == 5) {
      // no role: the tiles come from global memory (see the expansion warps)
      pdl_trigger();
    } else if (warp == 4 || warp == 7) {
      // ======================= score warps ==================================
      // both warps work on every tile, warp 4 the latent k-steps [0, KA)
      // into S columns [0, 32), warp 7 the latent ones [KA, KL) into
      // [32, 64) and the positional ones into the last 32 columns; each
      // waits for the tile's expansion and for softmax(t - NSB) to have read
      // the buffer, and commits to the buffer's barrier (two arrivals)
      const int role = warp == 4 ? 0 : 1;
      constexpr uint32_t ID_S = umma_idesc_f16(C::SM, 32, false, false);
      for (int t = 0; t < n_tiles && !failed; ++t) {
        const int s = t % C::NST;
        bool ok = true;
        if (t >= C::NSB)
          ok = mbar_wait_sleepy(&sfree[t % C::NSB], ((t - C::NSB) / C::NSB) & 1, wait_limit, abort_flag, kSleepNs);
        if (ok) ok = mbar_wait_sleepy(&full[s], (t / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
        if (ok && lane == 0) {
          tc_fence_after();
          const uint64_t dc = umma_desc(smem_u32(ostage(s)), 16, 1024, 2);
          const uint64_t dq = umma_desc(smem_u32(q_s), 128, KH / 8 * 128, 0);
          const uint32_t S = t_s + C::SBUF * (t % C::NSB);
          auto mma = [&](uint32_t d, int ks, bool acc) {
            umma_f16(d, dc + (uint64_t)(((ks / 4) * C::BOX + (ks % 4) * 32) >> 4), dq + (uint64_t)(ks * 16),
                     ID_S, acc);
          };
          if (role == 0) {
#pragma unroll
            for (int ks = 0; ks < C::KA; ++ks) mma(S, ks, ks > 0);
          } else {
#pragma unroll
            for (int ks = C::KA; ks < C::KL; ++ks) mma(S + 32, ks, ks > C::KA);
#pragma unroll
            for (int ks = C::KL; ks < KH / 16; ++ks) mma(S + C::SBUF - 32, ks, ks > C::KL);
          }
          umma_commit(&sbar[t % C::NSB]);
        }
        failed = !__all_sync(0xffffffffu, ok);
      }
      if (failed && lane == 0) {
        *abort_flag = 1;
        set_err(err, 8);
      }
      if (lane == 0) {
        umma_commit(&dbar[2 * role]);
        mbar_wait(&dbar[2 * role], 0, kLimit);
      }
      __syncwarp();
      pdl_trigger();
    } else {
      // ======================= value warp ===================================
      constexpr uint32_t ID_V = umma_idesc_f16(C::MV, 32, true, true);
      for (int t = 0; t < n_tiles && !failed; ++t) {
        const bool ok = mbar_wait_sleepy(&pbar[t & 1], (t >> 1) & 1, wait_limit, abort_flag, kSleepNs);
        if (ok && lane == 0) {  // O^T[:, hi | lo] += U^T [P'_hi | P'_lo]
          tc_fence_after();
          const uint64_t da = umma_desc(smem_u32(ostage(t % C::NST)), C::BOX, 1024, 2);
          const uint64_t dp = umma_desc(smem_u32(pbuf(t & 1)), 128, C::PNS, 0);
  #pragma unroll
          for (int ks = 0; ks < TR / 16; ++ks)
  #pragma unroll
            for (int mb = 0; mb < C::MBL; ++mb)
              umma_f16(t_o + 32 * mb, da + (uint64_t)(((2 * mb) * C::BOX + ks * 2048) >> 4),
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
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 256;\n" ::: "memory");
    // ======================= softmax warps ================================
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    // this lane's tile position: M = 128 puts row r in lane r; M = 64 puts
    // row r in lane 32 (r / 16) + r % 16 (lanes 0-15 of each quarter)
    constexpr int kRowLanes = C::SM == 128 ? 32 : 16;
    const int prow = kRowLanes * warp + lane;
    // per-head sums of the query halves as the products use them: thread
    // (h = tid / 8, j = tid % 8) adds chunks j, j + 8, ... of rows h and 16 + h
    {
      const int h = tid >> 3, j = tid & 7;
      float sl = 0.f, sr = 0.f;
      for (int c = j; c < KH / 8; c += 8) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int n = h + 16 * half;
          const uint4 w = *reinterpret_cast<const uint4 *>(q_s + (n / 8) * (KH / 8 * 128) + c * 128 + (n % 8) * 16);
          const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
          float acc = 0.f;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float2 f = unpack2<false>(ws[i]);
            acc += f.x + f.y;
          }
          if (c < W / 8) sl += acc; else sr += acc;
        }
      }
#pragma unroll
      for (int off = 1; off < 8; off <<= 1) {
        sl += __shfl_xor_sync(0xffffffffu, sl, off);
        sr += __shfl_xor_sync(0xffffffffu, sr, off);
      }
      if (j == 0) {
        qsum[h] = sl;
        qsum[kHeads + h] = sr;
      }
      softmax_sync();
    }
    float qsl[kHeads], qsr[kHeads];
#pragma unroll
    for (int h = 0; h < kHeads; ++h) { qsl[h] = qsum[h]; qsr[h] = qsum[kHeads + h]; }
    float m_run[kHeads], l_part[kHeads], z_part[kHeads];
#pragma unroll
    for (int h = 0; h < kHeads; ++h) { m_run[h] = -1e30f; l_part[h] = 0.f; z_part[h] = 0.f; }
    for (int t = 0; t < n_tiles; ++t) {
      const int base = i0 + t * TR, nval = min(TR, i1 - base);
      bool ok = mbar_wait_sleepy(&sbar[t % C::NSB], (t / C::NSB) & 1, wait_limit, abort_flag, kSleepNs);
      // the tile's scales were written before its operand was published:
      // acquire them (the phase of tile t is complete, the next cannot be)
      if (ok) ok = mbar_wait_sleepy(&full[t % C::NST], (t / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
      // P buffer (t & 1) was read by values(t-2)
      if (ok && t >= 2)
        ok = mbar_wait_sleepy(&obar[(t - 2) % C::NST], ((t - 2) / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
      if (softmax_sync_or(!ok)) { failed = true; break; }
      tc_fence_after();
      const bool live = lane < kRowLanes && prow < nval;
      const float4 md = live ? ometa(t % C::NST)[prow] : make_float4(0.f, 0.f, 0.f, 0.f);
      float x[kHeads];
      {
        // [A hi | A lo | (B hi | B lo |) rope hi | rope lo] of the 16 heads
        float sv[64], sr[32];
        const uint32_t S = t_s + C::SBUF * (t % C::NSB) + lane_off;
        tmem_ld64(S, sv);
        if constexpr (C::KB > 0) tmem_ld32(S + 64, sr);
        // the score buffer is free for tile t + NSB
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sfree[t % C::NSB]);
        const float scl = md.x * kCodeScale, scr = md.z * kCodeScale;
#pragma unroll
        for (int h = 0; h < kHeads; ++h) {
          // latent and positional parts (with one accumulator pair each
          // when the latent k-steps were not split)
          const float lat = C::KB > 0 ? (sv[h] + sv[16 + h]) + (sv[32 + h] + sv[48 + h]) : sv[h] + sv[16 + h];
          const float rp = C::KB > 0 ? sr[h] + sr[16 + h] : sv[32 + h] + sv[48 + h];
          x[h] = live ? fmaf(lat, scl, fmaf(rp, scr, fmaf(md.y, qsl[h], md.w * qsr[h]))) : -INFINITY;
        }
      }
      bool need = false;
#pragma unroll
      for (int h = 0; h < kHeads; ++h) need |= x[h] * sig > m_run[h] + 8.f;
      if (softmax_sync_or(need)) {
#pragma unroll
        for (int h = 0; h < kHeads; ++h) {
          float mx = x[h];
#pragma unroll
          for (int off = 1; off < kRowLanes; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
          if (lane == 0) red[warp * kHeads + h] = mx;
        }
        softmax_sync();
        float alpha[kHeads];
        bool any = false;
#pragma unroll
        for (int h = 0; h < kHeads; ++h) {
          const float mt =
              fmaxf(fmaxf(red[h], red[kHeads + h]), fmaxf(red[2 * kHeads + h], red[3 * kHeads + h])) * sig;
          alpha[h] = 1.f;
          if (mt > m_run[h] + 8.f) {
            alpha[h] = fast_exp2(m_run[h] - mt);
            m_run[h] = mt;
            any = true;
          }
          l_part[h] *= alpha[h];
          z_part[h] *= alpha[h];
        }
        if (t >= 1 && any) {
          ok = mbar_wait_sleepy(&obar[(t - 1) % C::NST], ((t - 1) / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
          if (softmax_sync_or(!ok)) { failed = true; break; }
          tc_fence_after();
#pragma unroll
          for (int mb = 0; mb < C::MBL; ++mb)
#pragma unroll
            for (int half = 0; half < 2; ++half) {
              float o[16];
              tmem_ld16(t_o + 32 * mb + 16 * half + lane_off, o);
#pragma unroll
              for (int h = 0; h < 16; ++h) o[h] *= alpha[h];
              tmem_st16(t_o + 32 * mb + 16 * half + lane_off, o);
            }
        }
        softmax_sync();
      }
      // value weights P' = p s (the latent scale of the position) as f16 hi
      // + lo into the MN-major P operand: position k, column n (0-15 hi,
      // 16-31 lo) at (k/8) 128 + (n/8) PNS + (k%8) 16 + (n%8) 2
      if (lane < kRowLanes && prow < TR) {
        uint32_t hw[8], lw[8];
#pragma unroll
        for (int h = 0; h < kHeads; h += 2) {
          const float p0 = fast_exp2(fmaf(x[h], sig, -m_run[h]));
          const float p1 = fast_exp2(fmaf(x[h + 1], sig, -m_run[h + 1]));
          l_part[h] += p0;
          l_part[h + 1] += p1;
          z_part[h] = fmaf(p0, md.y, z_part[h]);
          z_part[h + 1] = fmaf(p1, md.y, z_part[h + 1]);
          split2<false>(p0 * md.x, p1 * md.x, hw[h / 2], lw[h / 2]);
        }
        uint8_t *pp = pbuf(t & 1) + (prow / 8) * 128 + (prow % 8) * 16;
        *reinterpret_cast<uint4 *>(pp) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4 *>(pp + C::PNS) = make_uint4(hw[4], hw[5], hw[6], hw[7]);
        *reinterpret_cast<uint4 *>(pp + 2 * C::PNS) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        *reinterpret_cast<uint4 *>(pp + 3 * C::PNS) = make_uint4(lw[4], lw[5], lw[6], lw[7]);
      }
      fence_proxy_async();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&pbar[t & 1]);
    }
    pdl_trigger();
    // ---- partial of this split: o_lat rows, m, l ----------------------------
    if (!failed && n_tiles > 0) {
      const int t = n_tiles - 1;
      const bool ok = mbar_wait_sleepy(&obar[t % C::NST], (t / C::NST) & 1, wait_limit, abort_flag, kSleepNs);
      failed = softmax_sync_or(!ok);
    }
    if (failed && tid == 0) {
      *abort_flag = 1;
      set_err(err, 8);
    }
    if (!failed) {
      tc_fence_after();
      const size_t RS = (size_t)W + 2;
      const size_t prow_base = ((size_t)split * mla_rows(v) + vb) * H;
#pragma unroll
      for (int h = 0; h < kHeads; ++h) {
        float sum = l_part[h], zs = z_part[h];
#pragma unroll
        for (int off = 1; off < kRowLanes; off <<= 1) {
          sum += __shfl_xor_sync(0xffffffffu, sum, off);
          zs += __shfl_xor_sync(0xffffffffu, zs, off);
        }
        if (lane == 0) {
          lsum[warp * kHeads + h] = sum;
          zsum[warp * kHeads + h] = zs;
        }
      }
      softmax_sync();
      float zt[kHeads];
#pragma unroll
      for (int h = 0; h < kHeads; ++h)
        zt[h] = zsum[h] + zsum[kHeads + h] + zsum[2 * kHeads + h] + zsum[3 * kHeads + h];
#pragma unroll
      for (int mb = 0; mb < C::MBL; ++mb) {
        float o[16];
        if (n_tiles > 0) {
          float lo[16];
          tmem_ld16(t_o + 32 * mb + lane_off, o);
          tmem_ld16(t_o + 32 * mb + 16 + lane_off, lo);
#pragma unroll
          for (int h = 0; h < 16; ++h) o[h] = fmaf(o[h] + lo[h], kCodeScale, zt[h]);
        } else {
#pragma unroll
          for (int h = 0; h < 16; ++h) o[h] = 0.f;
        }
        const int r = C::MV == 128 ? 128 * mb + 32 * warp + lane : 16 * warp + lane;
        if (C::MV == 128 || lane < 16) {
#pragma unroll
          for (int h = 0; h < kHeads; ++h)
            if (h < H) partial[(prow_base + h) * RS + r] = o[h];
        }
      }
      if (tid < H) {
        const float L = lsum[tid] + lsum[kHeads + tid] + lsum[2 * kHeads + tid] + lsum[3 * kHeads + tid];
        float mh = m_run[0];
#pragma unroll
        for (int h = 1; h < kHeads; ++h) mh = (tid == h) ? m_run[h] : mh;
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

template <int W, int BITS, bool SYM>
cudaError_t launch_mla_q_t(const MlaDecodeArgs &a, cudaStream_t st) {
  using C = MlaQCfg<W, BITS, SYM>;
  if (a.n_splits > 64) return cudaErrorInvalidValue;  // merge weights hold 64 splits
  const int B = mla_rows(a.v);  // query rows
  auto k = mla_decode_q_kernel<W, BITS, SYM>;
  constexpr int MU_SMEM = (64 * (W + 8)) * 2 + (2 * 64 * 16 + 16) * 4;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(mla_merge_upv_kernel<W>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               MU_SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  cudaError_t e = launch_pdl(mla_absorb_kernel<W, true>, dim3(W / 64, a.H, (B + 15) / 16),
                             dim3(128), 0, st, static_cast<const uint16_t *>(a.q_nope),
                             static_cast<const uint16_t *>(a.q_pe),
                             static_cast<const uint16_t *>(a.w_uk), B, a.H, a.r, a.qlat);
  if (e == cudaSuccess)
    e = launch_pdl(k, dim3(a.n_splits, B), dim3(kMlaQThreads), C::SMEM, st, a.v,
                   static_cast<const uint16_t *>(a.qlat), static_cast<const uint16_t *>(a.q_pe),
                   a.H, a.sig_log2, a.items_per_split, a.n_splits, a.partial, a.err, a.wait_limit);
  if (e == cudaSuccess)
    e = launch_pdl(mla_merge_upv_kernel<W>, dim3(a.H, (B + 15) / 16, 4), dim3(128), MU_SMEM, st,
                   static_cast<const float *>(a.partial), a.n_splits,
                   static_cast<const uint16_t *>(a.w_uv), B, a.H, a.r, a.out);
  return e;
}

template <int W>
cudaError_t launch_mla_q_w(const MlaDecodeArgs &a, cudaStream_t st) {
  const bool sym = a.v.scheme == kSchemeSym;
  switch (a.v.bits) {
    case 8: return sym ? launch_mla_q_t<W, 8, true>(a, st) : launch_mla_q_t<W, 8, false>(a, st);
    case 4: return sym ? launch_mla_q_t<W, 4, true>(a, st) : launch_mla_q_t<W, 4, false>(a, st);
    case 2: return sym ? launch_mla_q_t<W, 2, true>(a, st) : cudaErrorInvalidValue;
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

// MLA decode over a quantised latent anchor: absorb (f16 halves), the
// latent decode above, then the merge fused with the up-projection.
cudaError_t launch_mla_decode_q(const MlaDecodeArgs &a, cudaStream_t st) {
  if (a.v.rope != kRope || !a.v.meta) return cudaErrorInvalidValue;
  switch (a.v.width) {
    case 512: return launch_mla_q_w<512>(a, st);
    case 256: return launch_mla_q_w<256>(a, st);
    case 128: return launch_mla_q_w<128>(a, st);
    case 64: return launch_mla_q_w<64>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace kvk
