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
// cores (mma.m16n8k16, bf16 operands, fp32 accumulate).  fp32 operands that
// must enter a bf16 MMA (q_lat, softmax weights, o_lat) are split into
// hi + lo bf16 halves, so products keep ~16 significant bits.
#include <math.h>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {
namespace {

constexpr int kRope = 64;
constexpr int kHeads = 16;

__device__ __forceinline__ int swz8(int row, int chunk) { return chunk ^ (row & 7); }

// ---------------------------------------------------------------------------
// Absorb: q_lat[b,h,i] = sum_j q_nope[b,h,j] W_UK[h,j,i], i < d.  Grid
// (64-coordinate block, head, 16-sequence block): M = 16 sequences, N = 64
// latent coordinates (16 per warp), K = Dn = 128.  Small CTAs, many of them:
// the operands arrive in one round trip.  Output qlat[b][h] =
// [hi(d) | pe(64) | lo(d)].
template <int W>
__global__ void __launch_bounds__(128)
    mla_absorb_kernel(const uint16_t *__restrict__ q_nope, const uint16_t *__restrict__ q_pe,
                      const uint16_t *__restrict__ w_uk, int B, int H, int r,
                      uint16_t *__restrict__ qlat) {
  constexpr int Dn = 128;
  __shared__ __align__(16) uint16_t a_s[16 * Dn];  // [b][j], swizzled 16B chunks
  __shared__ __align__(16) uint16_t w_s[Dn * 64];  // [j][i], swizzled
  const int h = blockIdx.y, i0 = blockIdx.x * 64, b0 = blockIdx.z * 16;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  constexpr int QROW = 2 * W + kRope;
  for (int q = tid; q < 16 * Dn / 8; q += 128) {
    const int row = q / (Dn / 8), u = q % (Dn / 8);
    const int b = b0 + row;
    uint4 x = make_uint4(0, 0, 0, 0);
    if (b < B) x = *reinterpret_cast<const uint4 *>(q_nope + ((size_t)b * H + h) * Dn + 8 * u);
    *reinterpret_cast<uint4 *>(a_s + row * Dn + 8 * swz8(row, u)) = x;
  }
  for (int q = tid; q < Dn * 8; q += 128) {
    const int j = q / 8, u = q % 8;
    const uint4 x = *reinterpret_cast<const uint4 *>(w_uk + ((size_t)h * Dn + j) * r + i0 + 8 * u);
    *reinterpret_cast<uint4 *>(w_s + j * 64 + 8 * swz8(j, u)) = x;
  }
  __syncthreads();
  float acc[2][4] = {};
  const int mat = lane >> 3, rr = lane & 7;
#pragma unroll
  for (int ks = 0; ks < Dn / 16; ++ks) {
    uint32_t a0, a1, a2, a3, b0r, b1r, b2r, b3r;
    {
      const int row = rr + ((mat & 1) ? 8 : 0);
      ldmatrix_x4(a0, a1, a2, a3, a_s + row * Dn + 8 * swz8(row, 2 * ks + (mat >> 1)));
    }
    {
      const int j = 16 * ks + rr + ((mat & 1) ? 8 : 0);
      ldmatrix_x4_t(b0r, b1r, b2r, b3r, w_s + j * 64 + 8 * swz8(j, 2 * warp + (mat >> 1)));
    }
    mma_bf16(acc[0], a0, a1, a2, a3, b0r, b1r);
    mma_bf16(acc[1], a0, a1, a2, a3, b2r, b3r);
  }
#pragma unroll
  for (int n = 0; n < 2; ++n) {
    const int i = i0 + 16 * warp + 8 * n + 2 * c;
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
      const int b = b0 + g + 8 * hr;
      if (b >= B) continue;
      uint32_t hi, lo;
      split2<true>(acc[n][2 * hr], acc[n][2 * hr + 1], hi, lo);
      uint16_t *dst = qlat + ((size_t)b * H + h) * QROW;
      *reinterpret_cast<uint32_t *>(dst + i) = hi;
      *reinterpret_cast<uint32_t *>(dst + W + kRope + i) = lo;
    }
  }
}

// ---------------------------------------------------------------------------
// Latent split-K decode.  Grid (split, sequence); 8 warps.  Tile = 64
// positions of [c[:W] | k^R] streamed through a cp.async ring.
//   score phase: warp (mb, nb) = (warp/2, warp%2): 16 positions x 8 heads,
//                K = W (q_lat hi and lo) + 64 (q_pe);
//   value phase: warp w owns (16 latent rows x 8 heads) units w, w+8, ...
//                of O^T[W x 16], K = the tile's 64 positions (P hi and lo).
template <int W>
struct MlaCfg {
  static constexpr int RB = (W + kRope) * 2;      // record bytes
  static constexpr int NCH = RB / 16;             // 16-byte chunks per record
  static constexpr int STAGE = kTile * RB;
  static constexpr int NST = W >= 512 ? 2 : (W >= 256 ? 3 : 4);
  static constexpr int QH_ROW = (W + kRope) * 2;  // bytes: hi q_lat | q_pe
  static constexpr int QL_ROW = W * 2;            // bytes: lo q_lat
  static constexpr int Q_BYTES = kHeads * (QH_ROW + QL_ROW);
  static constexpr int P_BYTES = 4 * 2 * 4 * 32 * 4;
  static constexpr int X_BYTES = 4 * kHeads * 4 * 2;  // tile maxima, row sums
  static constexpr int SMEM = Q_BYTES + P_BYTES + X_BYTES + NST * STAGE;
  static constexpr int UNITS = W / 8;              // (16 rows x 8 heads) value units
  static constexpr int UPW = (UNITS + 7) / 8;      // units per warp
  static_assert(NCH % 8 == 0, "swizzle needs 8-chunk multiples");
};

template <int W>
__global__ void __launch_bounds__(256)
    mla_decode_kernel(const MlaView v, const uint16_t *__restrict__ qlat,
                      const uint16_t *__restrict__ q_pe, int H, float sig_log2,
                      int items_per_split, int n_splits, float *__restrict__ partial,
                      int32_t *err) {
  using C = MlaCfg<W>;
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t *qh_s = smem;
  uint8_t *ql_s = smem + kHeads * C::QH_ROW;
  uint32_t *p_s = reinterpret_cast<uint32_t *>(smem + C::Q_BYTES);
  float *tmax_s = reinterpret_cast<float *>(smem + C::Q_BYTES + C::P_BYTES);  // [4][16]
  float *lsum_s = tmax_s + 4 * kHeads;                                         // [4][16]
  uint8_t *stages = smem + C::Q_BYTES + C::P_BYTES + C::X_BYTES;

  const int split = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  const int len = v.lens[b];
  const int i0 = split * items_per_split;
  const int i1 = (split == n_splits - 1) ? len : min(i0 + items_per_split, len);
  const int n_tiles = i1 > i0 ? (i1 - i0 + kTile - 1) / kTile : 0;
  const uint8_t *rec = v.rec + (size_t)b * v.cap * C::RB;

  // absorbed query [hi | pe] and [lo] into shared memory, swizzled rows;
  // q_pe comes straight from the caller's tensor
  {
    constexpr int QROW = 2 * W + kRope;
    const uint16_t *qb = qlat + (size_t)b * H * QROW;
    for (int q = tid; q < kHeads * (C::QH_ROW / 16); q += 256) {
      const int h = q / (C::QH_ROW / 16), u = q % (C::QH_ROW / 16);
      uint4 x = make_uint4(0, 0, 0, 0);
      if (h < H) {
        x = (u < W / 8) ? *reinterpret_cast<const uint4 *>(qb + (size_t)h * QROW + 8 * u)
                        : *reinterpret_cast<const uint4 *>(q_pe + ((size_t)b * H + h) * kRope +
                                                           8 * (u - W / 8));
      }
      *reinterpret_cast<uint4 *>(qh_s + h * C::QH_ROW + 16 * swz8(h, u)) = x;
    }
    for (int q = tid; q < kHeads * (C::QL_ROW / 16); q += 256) {
      const int h = q / (C::QL_ROW / 16), u = q % (C::QL_ROW / 16);
      uint4 x = make_uint4(0, 0, 0, 0);
      if (h < H) x = *reinterpret_cast<const uint4 *>(qb + (size_t)h * QROW + W + kRope + 8 * u);
      *reinterpret_cast<uint4 *>(ql_s + h * C::QL_ROW + 16 * swz8(h, u)) = x;
    }
  }

  auto issue = [&](int t, int s) {
    const int base = i0 + t * kTile;
    uint8_t *st = stages + s * C::STAGE;
    for (int q = tid; q < kTile * C::NCH; q += 256) {
      const int row = q / C::NCH, u = q - row * C::NCH;
      const int item = base + row;
      const bool valid = item < i1;
      const uint8_t *src = rec + (size_t)(valid ? item : 0) * C::RB + 16 * u;
      cp_async16(st + row * C::RB + 16 * swz8(row, u), src, valid);
    }
  };

  const int mb = warp >> 1, nb = warp & 1;
  float m_run[2][2] = {{-INFINITY, -INFINITY}, {-INFINITY, -INFINITY}};  // [nb][hh]
  float l_part[2] = {0.f, 0.f};  // this warp's rows, heads nb*8 + 2c + hh
  float acc[C::UPW][4];
#pragma unroll
  for (int u = 0; u < C::UPW; ++u) acc[u][0] = acc[u][1] = acc[u][2] = acc[u][3] = 0.f;

#pragma unroll
  for (int s = 0; s < C::NST - 1; ++s) {
    if (s < n_tiles) issue(s, s);
    cp_async_commit();
  }
  for (int t = 0; t < n_tiles; ++t) {
    cp_async_wait<C::NST - 2>();
    __syncthreads();
    {
      const int nt = t + C::NST - 1;
      if (nt < n_tiles) issue(nt, nt % C::NST);
      cp_async_commit();
    }
    const uint8_t *st = stages + (t % C::NST) * C::STAGE;
    const int base = i0 + t * kTile;

    // ---- scores: 16 positions x 8 heads per warp -------------------------
    // four independent accumulators (hi/lo x even/odd k-steps) so the MMA
    // chain is not one long dependency
    float dacc[4][4] = {};
    const int mat = lane >> 3, rr = lane & 7;
    const int hrow = 8 * nb + rr;
#pragma unroll 4
    for (int ks = 0; ks < W / 16; ++ks) {
      uint32_t a0, a1, a2, a3;
      {
        const int row = 16 * mb + rr + ((mat & 1) ? 8 : 0);
        ldmatrix_x4(a0, a1, a2, a3, st + row * C::RB + 16 * swz8(row, 2 * ks + (mat >> 1)));
      }
      uint32_t b0, b1, b2, b3;  // hi (2 chunks) then lo (2 chunks)
      const uint8_t *base_q = (mat < 2) ? qh_s + hrow * C::QH_ROW : ql_s + hrow * C::QL_ROW;
      ldmatrix_x4(b0, b1, b2, b3, base_q + 16 * swz8(hrow, 2 * ks + (mat & 1)));
      mma_bf16(dacc[(ks & 1) * 2], a0, a1, a2, a3, b0, b1);
      mma_bf16(dacc[(ks & 1) * 2 + 1], a0, a1, a2, a3, b2, b3);
    }
#pragma unroll
    for (int ks = W / 16; ks < (W + kRope) / 16; ++ks) {
      uint32_t a0, a1, a2, a3;
      {
        const int row = 16 * mb + rr + ((mat & 1) ? 8 : 0);
        ldmatrix_x4(a0, a1, a2, a3, st + row * C::RB + 16 * swz8(row, 2 * ks + (mat >> 1)));
      }
      uint32_t b0, b1;
      ldmatrix_x2(b0, b1, qh_s + hrow * C::QH_ROW + 16 * swz8(hrow, 2 * ks + (mat & 1)));
      mma_bf16(dacc[ks & 3], a0, a1, a2, a3, b0, b1);
    }
    float d[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) d[k] = (dacc[0][k] + dacc[1][k]) + (dacc[2][k] + dacc[3][k]);
    const bool vA = base + 16 * mb + g < i1, vB = base + 16 * mb + g + 8 < i1;
    float x[4];
    x[0] = vA ? d[0] * sig_log2 : -INFINITY;
    x[1] = vA ? d[1] * sig_log2 : -INFINITY;
    x[2] = vB ? d[2] * sig_log2 : -INFINITY;
    x[3] = vB ? d[3] * sig_log2 : -INFINITY;
    float mt0 = fmaxf(x[0], x[2]), mt1 = fmaxf(x[1], x[3]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      mt0 = fmaxf(mt0, __shfl_xor_sync(0xffffffffu, mt0, off));
      mt1 = fmaxf(mt1, __shfl_xor_sync(0xffffffffu, mt1, off));
    }
    if (g == 0) {
      tmax_s[mb * kHeads + 8 * nb + 2 * c] = mt0;
      tmax_s[mb * kHeads + 8 * nb + 2 * c + 1] = mt1;
    }
    __syncthreads();

    // ---- running maxima: every thread derives the same values -------------
    float alpha[2][2];
#pragma unroll
    for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int h = 8 * n2 + 2 * c + hh;
        float mt = fmaxf(fmaxf(tmax_s[h], tmax_s[kHeads + h]),
                         fmaxf(tmax_s[2 * kHeads + h], tmax_s[3 * kHeads + h]));
        alpha[n2][hh] = 1.f;
        if (mt > m_run[n2][hh] + 8.f) {  // lazy: keep a stale max within 2^8
          alpha[n2][hh] = (m_run[n2][hh] == -INFINITY) ? 0.f : fast_exp2(m_run[n2][hh] - mt);
          m_run[n2][hh] = mt;
        }
      }
    // ---- weights of this warp's 16 positions -> P^T fragments -------------
    {
      // this warp's head block nb (selects, not indexing: no local memory)
      const float ma = nb ? m_run[1][0] : m_run[0][0], mb2 = nb ? m_run[1][1] : m_run[0][1];
      l_part[0] *= nb ? alpha[1][0] : alpha[0][0];
      l_part[1] *= nb ? alpha[1][1] : alpha[0][1];
      float p[4];
      p[0] = (ma == -INFINITY) ? 0.f : fast_exp2(x[0] - ma);
      p[1] = (mb2 == -INFINITY) ? 0.f : fast_exp2(x[1] - mb2);
      p[2] = (ma == -INFINITY) ? 0.f : fast_exp2(x[2] - ma);
      p[3] = (mb2 == -INFINITY) ? 0.f : fast_exp2(x[3] - mb2);
      l_part[0] += p[0] + p[2];
      l_part[1] += p[1] + p[3];
      uint32_t ht, lt, hb, lb;
      split2<true>(p[0], p[1], ht, lt);
      split2<true>(p[2], p[3], hb, lb);
      uint32_t *pf = p_s + ((mb * 2 + nb) * 4) * 32;
      pf[0 * 32 + lane] = movmatrix_t(ht);
      pf[1 * 32 + lane] = movmatrix_t(hb);
      pf[2 * 32 + lane] = movmatrix_t(lt);
      pf[3 * 32 + lane] = movmatrix_t(lb);
    }
    // rescale the value accumulators of this warp's units
#pragma unroll
    for (int u = 0; u < C::UPW; ++u) {
      const int unit = warp + 8 * u;
      if (unit < C::UNITS) {
        const int un = unit & 1;
        const float a0 = un ? alpha[1][0] : alpha[0][0], a1 = un ? alpha[1][1] : alpha[0][1];
        acc[u][0] *= a0; acc[u][2] *= a0;
        acc[u][1] *= a1; acc[u][3] *= a1;
      }
    }
    __syncthreads();

    // ---- values: O^T[16 latent x 8 heads] += C^T[16 x 64 pos] P^T -----------
#pragma unroll
    for (int u = 0; u < C::UPW; ++u) {
      const int unit = warp + 8 * u;
      if (unit < C::UNITS) {
        const int mblk = unit >> 1, un = unit & 1;
#pragma unroll
        for (int kb = 0; kb < 4; ++kb) {
          uint32_t a0, a1, a2, a3;
          const int row = 16 * kb + rr + ((mat >> 1) ? 8 : 0);
          ldmatrix_x4_t(a0, a1, a2, a3, st + row * C::RB + 16 * swz8(row, 2 * mblk + (mat & 1)));
          const uint32_t *pf = p_s + ((kb * 2 + un) * 4) * 32;
          mma_bf16(acc[u], a0, a1, a2, a3, pf[lane], pf[32 + lane]);
          mma_bf16(acc[u], a0, a1, a2, a3, pf[64 + lane], pf[96 + lane]);
        }
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();

  // ---- row sums across the four position blocks ----------------------------
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l_part[0] += __shfl_xor_sync(0xffffffffu, l_part[0], off);
    l_part[1] += __shfl_xor_sync(0xffffffffu, l_part[1], off);
  }
  if (g == 0) {
    lsum_s[mb * kHeads + 8 * nb + 2 * c] = l_part[0];
    lsum_s[mb * kHeads + 8 * nb + 2 * c + 1] = l_part[1];
  }
  __syncthreads();

  const size_t RS = (size_t)W + 2;
  const size_t prow0 = ((size_t)split * v.B + b) * H;
#pragma unroll
  for (int u = 0; u < C::UPW; ++u) {
    const int unit = warp + 8 * u;
    if (unit < C::UNITS) {
      const int mblk = unit >> 1, un = unit & 1;
      const int r0 = 16 * mblk + g;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int h = 8 * un + 2 * c + hh;
        if (h < H) {
          float *pr = partial + (prow0 + h) * RS;
          pr[r0] = acc[u][hh];
          pr[r0 + 8] = acc[u][2 + hh];
        }
      }
    }
  }
  // publish m and l: lane (g == 0, c) of warp 0 holds m for heads 2c+hh and
  // 8+2c+hh (all threads agree on m_run).
  if (warp == 0 && g == 0) {
#pragma unroll
    for (int n2 = 0; n2 < 2; ++n2)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int h = 8 * n2 + 2 * c + hh;
        if (h < H) {
          float *pr = partial + (prow0 + h) * RS;
          pr[W] = m_run[n2][hh];
          pr[W + 1] = lsum_s[h] + lsum_s[kHeads + h] + lsum_s[2 * kHeads + h] +
                      lsum_s[3 * kHeads + h];
        }
      }
  }
  (void)err;
}

// ---------------------------------------------------------------------------
// Split-K merge fused with the up-projection: out[b,h,o] = sum_i o_lat[b,h,i]
// W_UV[h,o,i] with o_lat the LSE merge of the splits' partials.  Grid (head,
// 16-sequence block, quarter of the 128 outputs); 4 warps.  The CTA's 32
// W_UV rows are prefetched into shared memory (cp.async) while phase 1
// merges the 16 rows into o_lat (split hi/lo bf16, shared memory); phase 2:
// warp w computes 16 sequences x 8 outputs over K = d on the tensor cores.
template <int W>
__global__ void __launch_bounds__(128)
    mla_merge_upv_kernel(const float *__restrict__ partial, int n_splits,
                         const uint16_t *__restrict__ w_uv, int B, int H, int r,
                         float *__restrict__ out) {
  constexpr int Dv = 128;
  constexpr int OST = W + 8;  // padded rows (bf16): conflict-free ldmatrix
  extern __shared__ __align__(128) uint8_t dyn_smem[];
  uint16_t *oh_s = reinterpret_cast<uint16_t *>(dyn_smem);  // [16][OST]
  uint16_t *ol_s = oh_s + 16 * OST;                         // [16][OST]
  uint16_t *w_s = ol_s + 16 * OST;                          // [32][OST]
  float *wt_s = reinterpret_cast<float *>(w_s + 32 * OST);  // [64][16]
  float *linv_s = wt_s + 64 * 16;                           // [16]
  const int h = blockIdx.x, b0 = blockIdx.y * 16, o0 = blockIdx.z * 32;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  // prefetch this CTA's 32 rows of W_UV[h][:, :W]
  for (int q = tid; q < 32 * (W / 8); q += 128) {
    const int o = q / (W / 8), u = q % (W / 8);
    cp_async16(w_s + o * OST + 8 * u, w_uv + ((size_t)h * Dv + o0 + o) * r + 8 * u, true);
  }
  cp_async_commit();
  const size_t RS = (size_t)W + 2;
  const size_t pstride = (size_t)B * H * RS;
  // merge weights: every split's (m, l) of the 16 rows loaded at once
  float *l_s = linv_s + 16;  // [64][16] split sums, then 1/L
  for (int q = tid; q < n_splits * 16; q += 128) {
    const int sp = q >> 4, row = q & 15, b = b0 + row;
    float ms = -INFINITY, ls = 0.f;
    if (b < B) {
      const float *pr = partial + sp * pstride + ((size_t)b * H + h) * RS;
      ms = pr[W];
      ls = pr[W + 1];
    }
    wt_s[q] = ms;
    l_s[q] = ls;
  }
  __syncthreads();
  if (tid < 16) {
    float M = -INFINITY, L = 0.f;
    for (int sp = 0; sp < n_splits; ++sp) M = fmaxf(M, wt_s[sp * 16 + tid]);
    for (int sp = 0; sp < n_splits; ++sp) {
      const float ms = wt_s[sp * 16 + tid];
      const float wt = (ms == -INFINITY || M == -INFINITY) ? 0.f : exp2f(ms - M);
      wt_s[sp * 16 + tid] = wt;
      L += wt * l_s[sp * 16 + tid];
    }
    linv_s[tid] = (L > 0.f) ? 1.f / L : 0.f;
  }
  __syncthreads();
  // o_lat = sum_s w_s acc_s / L, (row, pair) elements of the 16 rows: each
  // thread keeps its PER elements in registers and issues a split's loads
  // together, one memory round trip per split
  constexpr int PER = 16 * (W / 2) / 128;
  constexpr int SG = PER >= 16 ? 1 : 16 / PER;  // splits whose loads are in flight together
  float2 oacc[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) oacc[k] = make_float2(0.f, 0.f);
  for (int sp0 = 0; sp0 < n_splits; sp0 += SG) {
    float2 x[SG][PER];
#pragma unroll
    for (int g2 = 0; g2 < SG; ++g2) {
      const int sp = sp0 + g2;
#pragma unroll
      for (int k = 0; k < PER; ++k) {
        const int e = tid + 128 * k, row = e / (W / 2), i = 2 * (e % (W / 2));
        const int b = b0 + row;
        x[g2][k] = (sp < n_splits && b < B)
                       ? *reinterpret_cast<const float2 *>(partial + sp * pstride +
                                                           ((size_t)b * H + h) * RS + i)
                       : make_float2(0.f, 0.f);
      }
    }
#pragma unroll
    for (int g2 = 0; g2 < SG; ++g2) {
      const int sp = sp0 + g2;
      if (sp >= n_splits) break;
#pragma unroll
      for (int k = 0; k < PER; ++k) {
        const int row = (tid + 128 * k) / (W / 2);
        const float wt = wt_s[sp * 16 + row];
        oacc[k].x = fmaf(wt, x[g2][k].x, oacc[k].x);
        oacc[k].y = fmaf(wt, x[g2][k].y, oacc[k].y);
      }
    }
  }
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int e = tid + 128 * k, row = e / (W / 2), i = 2 * (e % (W / 2));
    const float li = linv_s[row];
    uint32_t hi, lo;
    split2<true>(oacc[k].x * li, oacc[k].y * li, hi, lo);
    *reinterpret_cast<uint32_t *>(oh_s + row * OST + i) = hi;
    *reinterpret_cast<uint32_t *>(ol_s + row * OST + i) = lo;
  }
  cp_async_wait<0>();
  __syncthreads();
  const int mat = lane >> 3, rr = lane & 7;
  float acc[4] = {0.f, 0.f, 0.f, 0.f}, acc2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
  for (int ks = 0; ks < W / 16; ++ks) {
    uint32_t a0, a1, a2, a3, l0, l1, l2, l3, b0r, b1r;
    const int row = rr + ((mat & 1) ? 8 : 0);
    const int col = 16 * ks + 8 * (mat >> 1);
    ldmatrix_x4(a0, a1, a2, a3, oh_s + row * OST + col);
    ldmatrix_x4(l0, l1, l2, l3, ol_s + row * OST + col);
    ldmatrix_x2(b0r, b1r, w_s + (8 * warp + rr) * OST + 16 * ks + 8 * (mat & 1));
    mma_bf16(acc, a0, a1, a2, a3, b0r, b1r);
    mma_bf16(acc2, l0, l1, l2, l3, b0r, b1r);
  }
#pragma unroll
  for (int hr = 0; hr < 2; ++hr) {
    const int b = b0 + g + 8 * hr;
    if (b < B) {
      float *dst = out + ((size_t)b * H + h) * Dv + o0 + 8 * warp + 2 * c;
      dst[0] = acc[2 * hr] + acc2[2 * hr];
      dst[1] = acc[2 * hr + 1] + acc2[2 * hr + 1];
    }
  }
}

template <int W>
cudaError_t launch_mla_t(const MlaDecodeArgs &a, cudaStream_t st) {
  using C = MlaCfg<W>;
  if (a.n_splits > 64) return cudaErrorInvalidValue;  // merge weights hold 64 splits
  const int B = a.v.B;
  mla_absorb_kernel<W><<<dim3(W / 64, a.H, (B + 15) / 16), 128, 0, st>>>(
      static_cast<const uint16_t *>(a.q_nope), static_cast<const uint16_t *>(a.q_pe),
      static_cast<const uint16_t *>(a.w_uk), B, a.H, a.r, a.qlat);
  auto k = mla_decode_kernel<W>;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k<<<dim3(a.n_splits, B), 256, C::SMEM, st>>>(a.v, a.qlat,
                                                static_cast<const uint16_t *>(a.q_pe), a.H,
                                                a.sig_log2, a.items_per_split,
                                                a.n_splits, a.partial, a.err);
  constexpr int MU_SMEM = (64 * (W + 8)) * 2 + (2 * 64 * 16 + 16) * 4;
  static bool mu_attr = false;
  if (!mu_attr) {
    cudaError_t e2 = cudaFuncSetAttribute(mla_merge_upv_kernel<W>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, MU_SMEM);
    if (e2 != cudaSuccess) return e2;
    mu_attr = true;
  }
  mla_merge_upv_kernel<W><<<dim3(a.H, (B + 15) / 16, 4), 128, MU_SMEM, st>>>(
      a.partial, a.n_splits, static_cast<const uint16_t *>(a.w_uv), B, a.H, a.r, a.out);
  return cudaGetLastError();
}

template <int W>
int mla_ctas_t() {
  using C = MlaCfg<W>;
  auto k = mla_decode_kernel<W>;
  cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k, 256, C::SMEM) != cudaSuccess) n = 1;
  return n > 0 ? n : 1;
}

}  // namespace

cudaError_t launch_mla_decode(const MlaDecodeArgs &a, cudaStream_t st) {
  switch (a.v.width) {
    case 512: return launch_mla_t<512>(a, st);
    case 256: return launch_mla_t<256>(a, st);
    case 128: return launch_mla_t<128>(a, st);
    case 64: return launch_mla_t<64>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

int mla_decode_ctas_per_sm(int width) {
  switch (width) {
    case 512: return mla_ctas_t<512>();
    case 256: return mla_ctas_t<256>();
    case 128: return mla_ctas_t<128>();
    case 64: return mla_ctas_t<64>();
    default: return 1;
  }
}

}  // namespace kvk
