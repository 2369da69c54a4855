// mla_common.cuh -- pieces shared by the MLA latent decodes (bf16 and
// quantised latents): the query absorption, the split merge fused with
// the up-projection, and the named barrier of the four softmax warps.
#pragma once
#include <math.h>

#include "common.cuh"

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
// F16: q_lat hi/lo as f16 halves (the operand type of the quantised
// latent decode) instead of bf16.
template <int W, bool F16 = false>
__global__ void __launch_bounds__(128)
    mla_absorb_kernel(const uint16_t *__restrict__ q_nope, const uint16_t *__restrict__ q_pe,
                      const uint16_t *__restrict__ w_uk, int B, int H, int r,
                      uint16_t *__restrict__ qlat) {
  pdl_wait();
  constexpr int Dn = 128;
  __shared__ __align__(16) uint16_t a_s[16 * Dn];  // [b][j], swizzled 16B chunks
  __shared__ __align__(16) uint16_t w_s[Dn * 64];  // [j][i], swizzled
  const int h = blockIdx.y, i0 = blockIdx.x * 64, b0 = blockIdx.z * 16;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  constexpr int QROW = 2 * W + kRope;
  // every operand chunk in flight at once (asynchronous 16-byte copies;
  // rows past the batch are zero-filled)
#pragma unroll
  for (int q = tid; q < 16 * Dn / 8; q += 128) {
    const int row = q / (Dn / 8), u = q % (Dn / 8);
    const int b = b0 + row;
    cp_async16(a_s + row * Dn + 8 * swz8(row, u),
               q_nope + ((size_t)(b < B ? b : 0) * H + h) * Dn + 8 * u, b < B);
  }
#pragma unroll
  for (int q = tid; q < Dn * 8; q += 128) {
    const int j = q / 8, u = q % 8;
    cp_async16(w_s + j * 64 + 8 * swz8(j, u), w_uk + ((size_t)h * Dn + j) * r + i0 + 8 * u, true);
  }
  cp_async_commit();
  cp_async_wait<0>();
  pdl_trigger();
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
      split2<!F16>(acc[n][2 * hr], acc[n][2 * hr + 1], hi, lo);
      uint16_t *dst = qlat + ((size_t)b * H + h) * QROW;
      *reinterpret_cast<uint32_t *>(dst + i) = hi;
      *reinterpret_cast<uint32_t *>(dst + W + kRope + i) = lo;
    }
  }
}

// ---------------------------------------------------------------------------
// Split-K merge fused with the up-projection: out[b,h,o] = sum_i o_lat[b,h,i]
// W_UV[h,o,i] with o_lat the LSE merge of the splits' partials.  Grid (head,
// 16-sequence block, quarter of the 128 outputs); 4 warps.  The CTA's 32
// W_UV rows are prefetched into shared memory (cp.async) while phase 1
// merges the 16 rows into o_lat (split hi/lo bf16, shared memory); phase 2:
// warp w computes 16 sequences x 8 outputs over K = d on the tensor cores.
// `partial` is written by the decode kernel this launch overlaps
// (programmatic dependent launch): it is read with coherent loads after the
// grid-dependency wait, never through the read-only path (no __restrict__),
// whose loads may be scheduled as if the data were constant for the whole
// kernel.
template <int W>
__global__ void __launch_bounds__(128)
    mla_merge_upv_kernel(const float *partial, int n_splits,
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
  // prefetch this CTA's 32 rows of W_UV[h][:, :W].  Issued before the wait
  // for the decode kernel: this kernel's CTAs start only after the decode's
  // CTAs passed their own wait, which followed the absorb, whose CTAs in turn
  // waited for everything the caller enqueued before the call; the partials,
  // the decode's output, are read after the wait.
  for (int q = tid; q < 32 * (W / 8); q += 128) {
    const int o = q / (W / 8), u = q % (W / 8);
    cp_async16(w_s + o * OST + 8 * u, w_uv + ((size_t)h * Dv + o0 + o) * r + 8 * u, true);
  }
  cp_async_commit();
  pdl_wait();
  const size_t RS = (size_t)W + 2;
  const size_t pstride = (size_t)B * H * RS;
  // o_lat = sum_s w_s acc_s / L, (row, pair) elements of the 16 rows: each
  // thread keeps its PER elements in registers and issues a split group's
  // loads together; the first group's loads go out with the (m, l) loads
  // below, so that a merge of up to SG splits takes one memory round trip
  constexpr int PER = 16 * (W / 2) / 128;
  // splits whose loads are in flight together: 32 elements per thread, and
  // both splits of the widest latent (64 registers of loads there)
  constexpr int SG = PER >= 32 ? 2 : 32 / PER;
  float2 x[SG][PER];
  auto load_group = [&](int sp0) {
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
  };
  load_group(0);
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
  float2 oacc[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) oacc[k] = make_float2(0.f, 0.f);
  for (int sp0 = 0; sp0 < n_splits; sp0 += SG) {
    if (sp0 > 0) load_group(sp0);
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
  pdl_trigger();
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

// barrier over the four softmax warps (named barrier 1, 128 threads); the
// reduction form returns whether any thread passed true
__device__ __forceinline__ void softmax_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
__device__ __forceinline__ bool softmax_sync_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, 128, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"(v ? 1u : 0u)
      : "memory");
  return r != 0;
}

}  // namespace
}  // namespace kvk
