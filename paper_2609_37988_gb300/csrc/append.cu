// append.cu -- quantise / truncate on write (Appendix C.2, C.3).
//
// GQA rows: one warp per (sequence, new position, KV head).  Values, and keys
// with per-token groups, are quantised at once with the grouped asymmetric
// quantiser as an exact binary32 operation sequence (round-to-nearest
// subtract and divide, rint = round half to even, no contraction):
//     scale = (max - min) / (2^b - 1),  zero = min,
//     code  = clamp(rint((x - min) / scale), 0, 2^b - 1)   (scale 0 -> 0).
// Keys with per-channel groups (KIVI) are kept in bf16 in a residual plane
// until `group` positions of a group exist; then the group is quantised
// along positions, one (scale, zero) per channel.
//
// The sequence lengths advance after every row has been written: the last
// CTA to finish (completion counter) updates them, so no extra launch and no
// waiting are needed.
#include <math.h>

#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {
namespace {

__device__ __forceinline__ float load_in(const void *p, size_t i, int f32) {
  return f32 ? static_cast<const float *>(p)[i] : bf16_to_f32(static_cast<const uint16_t *>(p)[i]);
}

__device__ __forceinline__ int seq_count(const int32_t *n_per_seq, int b, int n_new,
                                         int32_t *err) {
  if (!n_per_seq) return n_new;
  const int n = n_per_seq[b];
  if (n < 0 || n > n_new) {
    set_err(err, 4);
    return 0;
  }
  return n;
}

// Quantise one lane's E elements belonging to groups of GS channels spread
// over GS/E consecutive lanes.  Returns codes, writes the group's scale and
// zero into (sc, zr) on every lane of the group.
template <int E>
__device__ __forceinline__ void quant_lane(const float (&x)[E], int GS, int levels,
                                           uint32_t (&code)[E], float &sc, float &zr) {
  float mn = x[0], mx = x[0];
#pragma unroll
  for (int e = 1; e < E; ++e) { mn = fminf(mn, x[e]); mx = fmaxf(mx, x[e]); }
  const int lanes = GS / E;
  for (int off = 1; off < lanes; off <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  }
  const float lev = (float)levels;
  const float scale = __fdiv_rn(__fsub_rn(mx, mn), lev);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (scale == 0.f) {
      code[e] = 0;
    } else {
      float r = rintf(__fdiv_rn(__fsub_rn(x[e], mn), scale));
      r = fminf(fmaxf(r, 0.f), lev);
      code[e] = (uint32_t)r;
    }
  }
  sc = scale;
  zr = mn;
}

// Symmetric per-vector quantiser (Appendix C.3) of one warp's row, lane
// holding E channels: s = bf16(max|x| / q) (one binary32 division, then
// round to nearest even), code = clip(rint(x / s), -q, q) with the stored
// scale, returned offset by q (u = code + q).  A zero row stores s = 0 and
// code 0.  Returns the bf16 bits of s.
template <int E>
__device__ __forceinline__ uint16_t quant_sym_lane(const float (&x)[E], int bits,
                                                   uint32_t (&u)[E]) {
  float am = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e) am = fmaxf(am, fabsf(x[e]));
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, off));
  const float q = (float)sym_levels(bits);
  const uint16_t sb = f32_to_bf16_bits(__fdiv_rn(am, q));
  const float s = bf16_to_f32(sb);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    float r = 0.f;
    if (s != 0.f) r = fminf(fmaxf(rintf(__fdiv_rn(x[e], s)), -q), q);
    u[e] = (uint32_t)(int)(r + q);
  }
  return sb;
}

// Symmetric record of (sequence b, position t, KV head kvh): both sections
// assembled in the per-warp buffer in physical (rotated) order, stored as
// whole 16-byte chunks; the two scales go to the scale plane.
template <int D>
__device__ void append_row_sym(const GqaView &v, const float (&xk)[D / 32],
                               const float (&xv)[D / 32], int b, int kvh, int t, uint32_t *buf,
                               int lane) {
  constexpr int E = D / 32;
  const int rb = v.rec_bytes;
  const int kb = D * v.bits / 8;
  const size_t row = ((size_t)b * v.Hkv + kvh) * v.cap + t;
  uint32_t uk[E], uv[E];
  const uint32_t sk = quant_sym_lane<E>(xk, v.bits, uk);
  const uint32_t sv = quant_sym_lane<E>(xv, v.bits, uv);
  for (int w = lane; w < rb / 4; w += 32) buf[w] = 0;
  __syncwarp();
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int ch = lane * E + e;
    const int lk = sym_k_bit(ch, v.bits, D);
    const int pk = 8 * sym_phys(lk >> 3, t, rb) + (lk & 7);
    atomicOr(buf + (pk >> 5), uk[e] << (pk & 31));
    const int lv = sym_v_bit(ch, v.bits, D) + 8 * kb;
    const int pv = 8 * sym_phys(lv >> 3, t, rb) + (lv & 7);
    atomicOr(buf + (pv >> 5), uv[e] << (pv & 31));
  }
  __syncwarp();
  uint4 *rec = reinterpret_cast<uint4 *>(v.rec + row * rb);
  for (int q = lane; q < rb / 16; q += 32) rec[q] = reinterpret_cast<const uint4 *>(buf)[q];
  if (lane == 0) v.scales[row] = sk | (sv << 16);
  __syncwarp();
}

// Writes one section (K or V) of a record through a per-warp shared buffer
// so the global stores are whole 16-byte chunks.
template <int D>
__device__ void put_section(uint32_t *buf, int bits, bool is_k, const uint32_t (&val)[D / 32],
                            int t, int rec_bytes, int lane) {
  constexpr int E = D / 32;
  const int words = D * bits / 32;
  for (int w = lane; w < words; w += 32) buf[w] = 0;
  __syncwarp();
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int ch = lane * E + e;
    int byte, hi;
    if (is_k)
      k_pos(ch, bits, D, &byte, &hi);
    else
      v_pos(ch, bits, D, t, rec_bytes, &byte, &hi);
    uint32_t v = val[e];
    int shift = (byte & 3) * 8;
    if (bits == 4) shift += hi * 4;
    atomicOr(buf + (byte >> 2), v << shift);
  }
  __syncwarp();
}

template <int D>
__device__ __forceinline__ void load_row(const void *kin, const void *vin, int in_f32,
                                         size_t ibase, int lane, float (&xk)[D / 32],
                                         float (&xv)[D / 32]) {
#pragma unroll
  for (int e = 0; e < D / 32; ++e) {
    xk[e] = load_in(kin, ibase + lane * (D / 32) + e, in_f32);
    xv[e] = load_in(vin, ibase + lane * (D / 32) + e, in_f32);
  }
}

// Quantises and writes one (sequence b, position t, KV head kvh) record from
// the warp's inputs (lane holds channels [lane E, lane E + E)).
template <int D>
__device__ void append_row(const GqaView &v, const float (&xk)[D / 32], const float (&xv)[D / 32],
                           int b, int kvh, int t, uint32_t *buf, int lane) {
  constexpr int E = D / 32;
  if (v.scheme == kSchemeSym) {
    append_row_sym<D>(v, xk, xv, b, kvh, t, buf, lane);
    return;
  }
  const RecLayout L = rec_layout(v.bits, D, v.group, v.key_axis);
  uint8_t *rec = v.rec + (((size_t)b * v.Hkv + kvh) * v.cap + t) * L.rec;
  const bool kq = v.bits != 16 && v.key_axis == 0;
  const bool kres = v.bits != 16 && v.key_axis == 1;
  // ---- K section ----
  if (!kres) {
    uint32_t val[E];
    float sc = 0.f, zr = 0.f;
    if (kq) {
      quant_lane<E>(xk, v.group, (1 << v.bits) - 1, val, sc, zr);
    } else {
#pragma unroll
      for (int e = 0; e < E; ++e) val[e] = f32_to_bf16_bits(xk[e]);
    }
    put_section<D>(buf, kq ? v.bits : 16, true, val, t, L.rec, lane);
    const int kb = D * v.bits / 8;
    for (int q = lane; q < kb / 16; q += 32)
      reinterpret_cast<uint4 *>(rec + L.k_off)[q] = reinterpret_cast<uint4 *>(buf)[q];
    if (kq && (lane * E) % v.group == 0)
      reinterpret_cast<float2 *>(rec + L.km_off)[(lane * E) / v.group] = make_float2(sc, zr);
    __syncwarp();
  }
  // ---- V section ----
  {
    uint32_t val[E];
    float sc = 0.f, zr = 0.f;
    const bool vq = v.bits != 16;
    if (vq) {
      quant_lane<E>(xv, v.group, (1 << v.bits) - 1, val, sc, zr);
    } else {
#pragma unroll
      for (int e = 0; e < E; ++e) val[e] = f32_to_bf16_bits(xv[e]);
    }
    put_section<D>(buf, v.bits, false, val, t, L.rec, lane);
    const int vb = D * v.bits / 8;
    for (int q = lane; q < vb / 16; q += 32)
      reinterpret_cast<uint4 *>(rec + L.v_off)[q] = reinterpret_cast<uint4 *>(buf)[q];
    if (vq && (lane * E) % v.group == 0)
      reinterpret_cast<float2 *>(rec + L.vm_off)[(lane * E) / v.group] = make_float2(sc, zr);
  }
}

template <int D>
__global__ void __launch_bounds__(128)
    gqa_append_rows(const GqaView v, const void *kin, const void *vin, int in_f32, int n_new,
                    const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  constexpr int E = D / 32;
  __shared__ __align__(16) uint32_t sbuf[4][(2 * D * 2 + 2 * 64) / 4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t wid = (size_t)blockIdx.x * 4 + warp;
  const size_t total = (size_t)v.B * n_new * v.Hkv;
  if (wid < total) {
    const int kvh = (int)(wid % v.Hkv);
    const int i = (int)((wid / v.Hkv) % n_new);
    const int b = (int)(wid / ((size_t)v.Hkv * n_new));
    const int nb = seq_count(n_per_seq, b, n_new, err);
    const int t = v.lens[b] + i;
    bool ok = i < nb;
    if (ok && t >= v.cap) {
      if (lane == 0) set_err(err, 2);
      ok = false;
    }
    if (ok) {
      float xk[E], xv[E];
      load_row<D>(kin, vin, in_f32, (((size_t)b * n_new + i) * v.Hkv + kvh) * D, lane, xk, xv);
      append_row<D>(v, xk, xv, b, kvh, t, sbuf[warp], lane);
    }
  }
  // The last CTA advances the lengths (per-token layouts only; per-channel
  // keys advance them in the residual kernel, which runs last).
  if (v.bits == 16 || v.key_axis == 0) {
    __syncthreads();
    __shared__ int last;
    if (threadIdx.x == 0) {
      __threadfence();
      last = (atomicAdd(v.counter, 1) == (int)gridDim.x - 1);
    }
    __syncthreads();
    if (last) {
      for (int b = threadIdx.x; b < v.B; b += blockDim.x) {
        const int nb = seq_count(n_per_seq, b, n_new, nullptr);
        v.lens[b] = min((long long)v.lens[b] + nb, (long long)v.cap);
      }
      if (threadIdx.x == 0) *v.counter = 0;
    }
  }
}

// Short appends (a decode step: n_new x H_kv <= 64 rows per sequence,
// per-token layouts): one CTA of 8 warps per sequence.  The CTA reads the
// length once while the warps' first input loads are in flight, writes all
// rows of its sequence and then advances the length itself -- no other CTA
// reads it, so no completion counter or fence is needed.
template <int D>
__global__ void __launch_bounds__(256)
    gqa_append_seq(const GqaView v, const void *kin, const void *vin, int in_f32, int n_new,
                   const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  constexpr int E = D / 32;
  __shared__ __align__(16) uint32_t sbuf[8][(2 * D * 2 + 2 * 64) / 4];
  __shared__ int s_len, s_nb;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x;
  const int rows = n_new * v.Hkv;
  float xk[E], xv[E];
  if (warp < rows)
    load_row<D>(kin, vin, in_f32, ((size_t)b * n_new * v.Hkv + warp) * D, lane, xk, xv);
  if (threadIdx.x == 0) {
    s_nb = seq_count(n_per_seq, b, n_new, err);
    s_len = v.lens[b];
  }
  __syncthreads();
  const int len = s_len, nb = s_nb;
  for (int r = warp; r < rows; r += 8) {
    const int i = r / v.Hkv, kvh = r - i * v.Hkv;
    if (r != warp)
      load_row<D>(kin, vin, in_f32, ((size_t)b * n_new * v.Hkv + r) * D, lane, xk, xv);
    if (i >= nb) continue;
    const int t = len + i;
    if (t >= v.cap) {
      if (lane == 0) set_err(err, 2);
      continue;
    }
    append_row<D>(v, xk, xv, b, kvh, t, sbuf[warp], lane);
  }
  __syncthreads();
  if (threadIdx.x == 0) v.lens[b] = min((long long)len + nb, (long long)v.cap);
}

// Per-channel key groups completed by this append: one thread per
// (sequence, kv head, group, channel pair {ch, ch+8} sharing 4-bit bytes).
template <int D>
__global__ void __launch_bounds__(128)
    gqa_append_kgroups(const GqaView v, const void *kin, int in_f32, int n_new,
                       const int32_t *n_per_seq, int32_t *err, int max_groups) {
  pdl_wait();
  pdl_trigger();
  const int pairs = D / 2;
  const size_t id = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t total = (size_t)v.B * v.Hkv * max_groups * pairs;
  if (id >= total) return;
  const int pr = (int)(id % pairs);
  const int gidx = (int)((id / pairs) % max_groups);
  const int kvh = (int)((id / ((size_t)pairs * max_groups)) % v.Hkv);
  const int b = (int)(id / ((size_t)pairs * max_groups * v.Hkv));
  const int GS = v.group;
  const int nb = seq_count(n_per_seq, b, n_new, nullptr);
  const int len0 = v.lens[b];
  const int G = len0 / GS + gidx;  // candidate group
  if ((G + 1) * GS > len0 + nb || (G + 1) * GS > v.cap) return;  // not completed now
  const int ch0 = (pr / 8) * 16 + (pr % 8);  // channels ch0 and ch0 + 8
  const size_t slab = (size_t)b * v.Hkv + kvh;
  const RecLayout L = rec_layout(v.bits, D, GS, 1);
  const uint8_t *res = v.resid + slab * (size_t)GS * D * 2;
  const int levels = (1 << v.bits) - 1;
  uint32_t codes[2][64];
  float scs[2], zrs[2];
  for (int h = 0; h < 2; ++h) {
    const int ch = ch0 + 8 * h;
    int kb, khi;
    k_pos(ch, 16, D, &kb, &khi);
    float mn = INFINITY, mx = -INFINITY;
    float xs[64];
    for (int r = 0; r < GS; ++r) {
      const int p = G * GS + r;
      float x;
      if (p < len0) {
        x = bf16_to_f32(*reinterpret_cast<const uint16_t *>(res + (size_t)r * D * 2 + kb));
      } else {
        const size_t ii = (((size_t)b * n_new + (p - len0)) * v.Hkv + kvh) * D + ch;
        x = bf16_to_f32(f32_to_bf16_bits(load_in(kin, ii, in_f32)));  // keys buffer as bf16
      }
      xs[r] = x;
      mn = fminf(mn, x);
      mx = fmaxf(mx, x);
    }
    const float scale = __fdiv_rn(__fsub_rn(mx, mn), (float)levels);
    for (int r = 0; r < GS; ++r) {
      if (scale == 0.f) {
        codes[h][r] = 0;
      } else {
        float q = rintf(__fdiv_rn(__fsub_rn(xs[r], mn), scale));
        codes[h][r] = (uint32_t)fminf(fmaxf(q, 0.f), (float)levels);
      }
    }
    scs[h] = scale;
    zrs[h] = mn;
  }
  for (int h = 0; h < 2; ++h)
    v.gmeta[(slab * (v.cap / GS) + G) * D + ch0 + 8 * h] = make_float2(scs[h], zrs[h]);
  for (int r = 0; r < GS; ++r) {
    uint8_t *rec = v.rec + (slab * v.cap + (size_t)G * GS + r) * L.rec + L.k_off;
    int b0, h0, b1, h1;
    k_pos(ch0, v.bits, D, &b0, &h0);
    k_pos(ch0 + 8, v.bits, D, &b1, &h1);
    if (v.bits == 8) {
      rec[b0] = (uint8_t)codes[0][r];
      rec[b1] = (uint8_t)codes[1][r];
    } else {
      // 4-bit: channels ch0 and ch0+8 share one byte (low and high nibble)
      rec[b0] = (uint8_t)(codes[0][r] | (codes[1][r] << 4));
    }
  }
  (void)err;
}

// Positions of the group left open after this append go to the residual
// plane; block b then advances sequence b's length.
template <int D>
__global__ void __launch_bounds__(128)
    gqa_append_kresid(const GqaView v, const void *kin, int in_f32, int n_new,
                      const int32_t *n_per_seq) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  const int GS = v.group;
  const int nb = seq_count(n_per_seq, b, n_new, nullptr);
  const int len0 = v.lens[b];
  const int len1 = min(len0 + nb, (int)v.cap);
  const int open0 = (len1 / GS) * GS;  // first position of the open group
  const int first = max(open0, len0);
  const int rows = len1 - first;
  const int work = rows * v.Hkv * D;
  for (int q = threadIdx.x; q < work; q += blockDim.x) {
    const int ch = q % D;
    const int kvh = (q / D) % v.Hkv;
    const int p = first + q / (D * v.Hkv);
    const size_t ii = (((size_t)b * n_new + (p - len0)) * v.Hkv + kvh) * D + ch;
    int kb, khi;
    k_pos(ch, 16, D, &kb, &khi);
    uint8_t *res = v.resid + ((size_t)b * v.Hkv + kvh) * GS * D * 2 + (size_t)(p % GS) * D * 2;
    *reinterpret_cast<uint16_t *>(res + kb) = f32_to_bf16_bits(load_in(kin, ii, in_f32));
  }
  __syncthreads();
  if (threadIdx.x == 0) v.lens[b] = len1;
}

__global__ void __launch_bounds__(128)
    mla_append_rows(const MlaView v, const uint16_t *c, const uint16_t *kr, int latent, int n_new,
                    const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t wid = (size_t)blockIdx.x * 4 + warp;
  if (wid < (size_t)v.B * n_new) {
    const int i = (int)(wid % n_new), b = (int)(wid / n_new);
    const int nb = seq_count(n_per_seq, b, n_new, err);
    const int t = v.lens[b] + i;
    bool ok = i < nb;
    if (ok && t >= v.cap) {
      if (lane == 0) set_err(err, 2);
      ok = false;
    }
    if (ok) {
      uint16_t *rec = reinterpret_cast<uint16_t *>(v.rec + ((size_t)b * v.cap + t) * v.rec_bytes);
      const uint16_t *cs = c + ((size_t)b * n_new + i) * latent;
      const uint16_t *ks = kr + ((size_t)b * n_new + i) * v.rope;
      for (int e = lane; e < v.width; e += 32) rec[e] = cs[e];  // first `width` coordinates
      for (int e = lane; e < v.rope; e += 32) rec[v.width + e] = ks[e];
    }
  }
  __syncthreads();
  __shared__ int last;
  if (threadIdx.x == 0) {
    __threadfence();
    last = (atomicAdd(v.counter, 1) == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (last) {
    for (int b = threadIdx.x; b < v.B; b += blockDim.x) {
      const int nb = seq_count(n_per_seq, b, n_new, nullptr);
      v.lens[b] = min((long long)v.lens[b] + nb, (long long)v.cap);
    }
    if (threadIdx.x == 0) *v.counter = 0;
  }
}

// Quantised MLA append (the layout in layout.h): one warp per (sequence,
// new position); the kept latent c[:W] and the positional key are each
// quantised as one vector (symmetric: one bf16 scale; grouped: one fp32
// scale and zero), codes staged in shared memory and stored chunk by chunk.
template <int W>
__global__ void __launch_bounds__(128)
    mla_append_q(const MlaView v, const uint16_t *c, const uint16_t *kr, int latent, int n_new,
                 const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  constexpr int R = 64, KH = W + R, EC = W / 32, ER = R / 32;
  __shared__ uint8_t buf[4][KH];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t wid = (size_t)blockIdx.x * 4 + warp;
  if (wid < (size_t)v.B * n_new) {
    const int i = (int)(wid % n_new), b = (int)(wid / n_new);
    const int nb = seq_count(n_per_seq, b, n_new, err);
    const int t = v.lens[b] + i;
    bool ok = i < nb;
    if (ok && t >= v.cap) {
      if (lane == 0) set_err(err, 2);
      ok = false;
    }
    if (ok) {
      const uint16_t *cs = c + ((size_t)b * n_new + i) * latent;
      const uint16_t *ks = kr + ((size_t)b * n_new + i) * R;
      float xc[EC], xr[ER];
#pragma unroll
      for (int e = 0; e < EC; ++e) xc[e] = bf16_to_f32(cs[lane + 32 * e]);
#pragma unroll
      for (int e = 0; e < ER; ++e) xr[e] = bf16_to_f32(ks[lane + 32 * e]);
      uint32_t uc[EC], ur[ER];
      if (v.scheme == kSchemeSym) {
        const uint16_t sc = quant_sym_lane<EC>(xc, v.bits, uc);
        const uint16_t sr = quant_sym_lane<ER>(xr, v.bits, ur);
        if (lane == 0)
          reinterpret_cast<uint32_t *>(v.meta)[(size_t)b * v.cap + t] = (uint32_t)sc | ((uint32_t)sr << 16);
      } else {
        const int lev = (1 << v.bits) - 1;
        float sc, zc, sr, zr;
        quant_lane<EC>(xc, W, lev, uc, sc, zc);
        quant_lane<ER>(xr, R, lev, ur, sr, zr);
        if (lane == 0)
          reinterpret_cast<float4 *>(v.meta)[(size_t)b * v.cap + t] = make_float4(sc, zc, sr, zr);
      }
#pragma unroll
      for (int e = 0; e < EC; ++e) buf[warp][lane + 32 * e] = (uint8_t)uc[e];
#pragma unroll
      for (int e = 0; e < ER; ++e) buf[warp][W + lane + 32 * e] = (uint8_t)ur[e];
      __syncwarp();
      uint8_t *rec = v.rec + ((size_t)b * v.cap + t) * v.rec_bytes;
      for (int j = lane; j < KH / 8; j += 32) {
        const uint8_t *cd = buf[warp] + 8 * j;
        if (v.bits == 8) {
          uint2 w;
          w.x = cd[0] | (cd[1] << 8) | (cd[2] << 16) | ((uint32_t)cd[3] << 24);
          w.y = cd[4] | (cd[5] << 8) | (cd[6] << 16) | ((uint32_t)cd[7] << 24);
          reinterpret_cast<uint2 *>(rec)[j] = w;
        } else if (v.bits == 4) {
          uint32_t w = 0;
#pragma unroll
          for (int k = 0; k < 8; ++k) w |= (uint32_t)cd[k] << mla_q_bit(k, 4);
          reinterpret_cast<uint32_t *>(rec)[j] = w;
        } else {
          uint32_t w = 0;
#pragma unroll
          for (int k = 0; k < 8; ++k) w |= (uint32_t)cd[k] << mla_q_bit(k, 2);
          reinterpret_cast<uint16_t *>(rec)[j] = (uint16_t)w;
        }
      }
    }
  }
  __syncthreads();
  __shared__ int last;
  if (threadIdx.x == 0) {
    __threadfence();
    last = (atomicAdd(v.counter, 1) == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (last) {
    for (int b = threadIdx.x; b < v.B; b += blockDim.x) {
      const int nb = seq_count(n_per_seq, b, n_new, nullptr);
      v.lens[b] = min((long long)v.lens[b] + nb, (long long)v.cap);
    }
    if (threadIdx.x == 0) *v.counter = 0;
  }
}

}  // namespace

cudaError_t launch_gqa_append(const GqaView &v, const void *k, const void *vv, int in_f32,
                              int n_new, const int32_t *n_per_seq, int32_t *err,
                              cudaStream_t st) {
  const size_t rows = (size_t)v.B * n_new * v.Hkv;
  const unsigned blocks = (unsigned)((rows + 3) / 4);
  const bool kpc = v.bits != 16 && v.key_axis == 1;
  const bool d128 = v.D == 128;
  cudaError_t e = cudaSuccess;
  if (kpc) {
    // groups first (they read residual rows the open group may overwrite)
    const int max_groups = (n_new + v.group - 1) / v.group + 1;
    const size_t thr = (size_t)v.B * v.Hkv * max_groups * (v.D / 2);
    const dim3 grid((unsigned)((thr + 127) / 128));
    e = launch_pdl(d128 ? gqa_append_kgroups<128> : gqa_append_kgroups<64>, grid, dim3(128), 0, st,
                   v, k, in_f32, n_new, n_per_seq, err, max_groups);
  }
  if (e == cudaSuccess) {
    if (!kpc && (size_t)n_new * v.Hkv <= 64)
      e = launch_pdl(d128 ? gqa_append_seq<128> : gqa_append_seq<64>, dim3(v.B), dim3(256), 0, st,
                     v, k, vv, in_f32, n_new, n_per_seq, err);
    else
      e = launch_pdl(d128 ? gqa_append_rows<128> : gqa_append_rows<64>, dim3(blocks), dim3(128), 0,
                     st, v, k, vv, in_f32, n_new, n_per_seq, err);
  }
  if (e == cudaSuccess && kpc)
    e = launch_pdl(d128 ? gqa_append_kresid<128> : gqa_append_kresid<64>, dim3(v.B), dim3(128), 0,
                   st, v, k, in_f32, n_new, n_per_seq);
  return e;
}

cudaError_t launch_mla_append(const MlaView &v, const void *c, const void *kr, int latent,
                              int n_new, const int32_t *n_per_seq, int32_t *err,
                              cudaStream_t st) {
  const size_t rows = (size_t)v.B * n_new;
  const dim3 grid((unsigned)((rows + 3) / 4));
  const uint16_t *cc = static_cast<const uint16_t *>(c), *kk = static_cast<const uint16_t *>(kr);
  if (v.bits != 16) {
    if (v.rope != 64) return cudaErrorInvalidValue;
    switch (v.width) {
      case 512: return launch_pdl(mla_append_q<512>, grid, dim3(128), 0, st, v, cc, kk, latent, n_new, n_per_seq, err);
      case 256: return launch_pdl(mla_append_q<256>, grid, dim3(128), 0, st, v, cc, kk, latent, n_new, n_per_seq, err);
      case 128: return launch_pdl(mla_append_q<128>, grid, dim3(128), 0, st, v, cc, kk, latent, n_new, n_per_seq, err);
      case 64: return launch_pdl(mla_append_q<64>, grid, dim3(128), 0, st, v, cc, kk, latent, n_new, n_per_seq, err);
      default: return cudaErrorInvalidValue;
    }
  }
  return launch_pdl(mla_append_rows, grid, dim3(128), 0, st, v, cc, kk, latent, n_new, n_per_seq, err);
}

}  // namespace kvk
