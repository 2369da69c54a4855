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

// rint(fl(d / s)) for s > 0 and |d / s| at most a few hundred, without a
// division in the common case.  rs is the fast reciprocal of s
// (__fdividef(1, s): within 2 ulp of 1/s for normal s), so y = fl(d rs) is
// within 1.8e-7 |d/s| of d/s, and fl(d/s) within 6e-8 |d/s|: for |d/s| <=
// 300 the two differ by less than 7.2e-5, and when y is further than 1e-4
// from the nearest half-integer both round to the same integer.  Otherwise
// (or when y is not finite, as for a scale whose reciprocal overflows) the
// correctly rounded division decides.  `near` reports that case.
__device__ __forceinline__ float rint_quot_fast(float d, float rs, bool &near) {
  const float y = __fmul_rn(d, rs);
  const float r = rintf(y);
  near = !(fabsf(__fsub_rn(y, r)) < 0.4999f);
  return r;
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
  const float rs = scale == 0.f ? 0.f : __fdividef(1.f, scale);
  float r[E];
  bool any_near = false;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    bool near;
    r[e] = rint_quot_fast(__fsub_rn(x[e], mn), rs, near);
    any_near |= near;
  }
  if (__any_sync(0xffffffffu, any_near && scale != 0.f)) {
#pragma unroll
    for (int e = 0; e < E; ++e)
      if (scale != 0.f) r[e] = rintf(__fdiv_rn(__fsub_rn(x[e], mn), scale));
  }
#pragma unroll
  for (int e = 0; e < E; ++e) code[e] = scale == 0.f ? 0u : (uint32_t)fminf(fmaxf(r[e], 0.f), lev);
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
  const float rs = s == 0.f ? 0.f : __fdividef(1.f, s);
  float rq[E];
  bool any_near = false;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    bool near;
    rq[e] = rint_quot_fast(x[e], rs, near);
    any_near |= near;
  }
  if (__any_sync(0xffffffffu, any_near && s != 0.f)) {
#pragma unroll
    for (int e = 0; e < E; ++e)
      if (s != 0.f) rq[e] = rintf(__fdiv_rn(x[e], s));
  }
#pragma unroll
  for (int e = 0; e < E; ++e) {
    float r = 0.f;
    if (s != 0.f) r = fminf(fmaxf(rq[e], -q), q);
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

// E = D / 32 consecutive elements of one lane, one vector load (inputs are
// 16-byte aligned and rows are D elements long)
template <int E>
__device__ __forceinline__ void load_lane(const void *in, size_t i, int f32, float (&x)[E]) {
  static_assert(E == 2 || E == 4, "two or four elements per lane");
  if (f32) {
    const float *p = static_cast<const float *>(in) + i;
    if constexpr (E == 4) {
      const float4 w = *reinterpret_cast<const float4 *>(p);
      x[0] = w.x; x[1] = w.y; x[2] = w.z; x[3] = w.w;
    } else {
      const float2 w = *reinterpret_cast<const float2 *>(p);
      x[0] = w.x; x[1] = w.y;
    }
  } else {
    const uint16_t *p = static_cast<const uint16_t *>(in) + i;
    uint32_t w[E / 2];
    if constexpr (E == 4) {
      const uint2 u = *reinterpret_cast<const uint2 *>(p);
      w[0] = u.x; w[1] = u.y;
    } else {
      w[0] = *reinterpret_cast<const uint32_t *>(p);
    }
#pragma unroll
    for (int j = 0; j < E / 2; ++j) {
      x[2 * j] = __uint_as_float(w[j] << 16);
      x[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
  }
}

template <int D>
__device__ __forceinline__ void load_row(const void *kin, const void *vin, int in_f32,
                                         size_t ibase, int lane, float (&xk)[D / 32],
                                         float (&xv)[D / 32]) {
  load_lane<D / 32>(kin, ibase + lane * (D / 32), in_f32, xk);
  load_lane<D / 32>(vin, ibase + lane * (D / 32), in_f32, xv);
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

// Row wid = (b n_new + i) Hkv + kvh of an append, tracked as (b, i, kvh)
// and advanced by a fixed stride with carries instead of divided per row:
// the stride's own decomposition is computed once.
struct RowIdx {
  uint32_t b, i, kvh;
};
struct RowStep {
  uint32_t Hkv, n_new, db, di, dk;
  __device__ RowStep(uint32_t step, uint32_t Hkv_, uint32_t n_new_) : Hkv(Hkv_), n_new(n_new_) {
    const uint32_t q = step / Hkv;
    dk = step - q * Hkv;
    db = q / n_new;
    di = q - db * n_new;
  }
  __device__ RowIdx at(uint32_t w) const {
    const uint32_t q = w / Hkv, b = q / n_new;
    return RowIdx{b, q - b * n_new, w - q * Hkv};
  }
  __device__ RowIdx next(RowIdx r) const {  // the row `step` further on
    r.kvh += dk;
    const uint32_t c = r.kvh >= Hkv;
    r.kvh -= c ? Hkv : 0u;
    r.i += di + c;
    const uint32_t c2 = r.i >= n_new;
    r.i -= c2 ? n_new : 0u;
    r.b += db + c2;
    return r;
  }
};

template <int D>
__global__ void __launch_bounds__(128)
    gqa_append_rows(const GqaView v, const void *kin, const void *vin, int in_f32, int n_new,
                    const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  constexpr int E = D / 32;
  __shared__ __align__(16) uint32_t sbuf[4][(2 * D * 2 + 2 * 64) / 4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t total = (size_t)v.B * n_new * v.Hkv;
  // rows wid, wid + 4 gridDim.x, ...: a bounded grid, so that the completion
  // counter below takes one atomic per CTA, not one per four rows
  // (the grid stride and the first row fit 32 bits; the row index itself
  // stays 64-bit, its (b, i, kvh) advance by the stride)
  const RowStep rstep((uint32_t)gridDim.x * 4u, (uint32_t)v.Hkv, (uint32_t)n_new);
  RowIdx ridx = rstep.at((uint32_t)min((size_t)blockIdx.x * 4 + warp, total));
  for (size_t wid = (size_t)blockIdx.x * 4 + warp; wid < total; wid += (size_t)gridDim.x * 4) {
    const int kvh = (int)ridx.kvh, i = (int)ridx.i, b = (int)ridx.b;
    ridx = rstep.next(ridx);
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
    __syncwarp();  // the row buffer is free again
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

// ---- bulk appends, head_dim 128, per-token layouts -------------------------
// One warp per (sequence, new position, KV head) row over a bounded grid,
// lane L holding channels 4L .. 4L+3.  Each lane packs its codes into one
// register per section; the record's 32-bit words are then gathered from
// the lanes that hold their channels by warp shuffles (the channel order of
// layout.h, derived per format below) and stored as whole words, the 128-
// to 512-byte record in one to four coalesced store instructions.

// 4-bit codes (grouped int4 or symmetric 4-bit): p = K codes | V codes << 16.
// Lanes 0-15 build K word T = lane (lane column c = T / 4, word w = T % 4
// holds k-steps 2w, 2w+1: nibble h + 2 jj from lane 4 (2w + jj) + c/2 + 2h
// element 2 (c%2), nibble 4 + h + 2 jj from its element 2 (c%2) + 1).
// Lanes 16-31 build logical V word U = lane - 16 (chunk k = U / 4, word
// wd = U % 4: M-blocks 2k + mm, rows g = 2 wd + gg, g + 8 e: bits
// 8 (2 gg + mm) + 4 e from lane 4 (2k + mm) + 2e + wd/2, element
// 2 (wd%2) + gg).
struct Gather4 {
  int src[4], sh, dlo[4], dhi[4];
  __device__ explicit Gather4(int lane) {
    if (lane < 16) {
      const int c = lane >> 2, w = lane & 3;
      sh = 8 * (c & 1);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int jj = q >> 1, h = q & 1;
        src[q] = 4 * (2 * w + jj) + (c >> 1) + 2 * h;
        dlo[q] = 4 * (h + 2 * jj);
        dhi[q] = 4 * (4 + h + 2 * jj);
      }
    } else {
      const int u = lane - 16, k = u >> 2, wd = u & 3;
      sh = 16 + 8 * (wd & 1);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int mm = q >> 1, e = q & 1;
        src[q] = 4 * (2 * k + mm) + 2 * e + (wd >> 1);
        dlo[q] = 8 * mm + 4 * e;
        dhi[q] = 16 + 8 * mm + 4 * e;
      }
    }
  }
  __device__ __forceinline__ uint32_t word(uint32_t p) const {
    uint32_t x = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t b = __shfl_sync(0xffffffffu, p, src[q]) >> sh;
      x |= ((b & 0xFu) << dlo[q]) | (((b >> 4) & 0xFu) << dhi[q]);
    }
    return x;
  }
};

// 8-bit codes: every lane builds K word T = lane (chunk T / 4 = 4 (bp / 16)
// + c, k-step j = 4 (chunk / 4) + T % 4: bytes 0-1 from lane 4j + c/2,
// bytes 2-3 from lane 4j + c/2 + 2, each lane's elements 2 (c%2), +1) and
// logical V word U = lane (M-block m = U / 4, word wd = U % 4: bytes 2 gg + e
// from lane 4m + 2e + wd/2, element 2 (wd%2) + gg).
struct Gather8 {
  int ks0, ks1, ksh, vs0, vs1, vsh;
  __device__ explicit Gather8(int lane) {
    const int chunk = lane >> 2, c = chunk & 3, j = 4 * (chunk >> 2) + (lane & 3);
    ks0 = 4 * j + (c >> 1);
    ks1 = ks0 + 2;
    ksh = 16 * (c & 1);
    const int m = lane >> 2, wd = lane & 3;
    vs0 = 4 * m + (wd >> 1);
    vs1 = vs0 + 2;
    vsh = 16 * (wd & 1);
  }
  __device__ __forceinline__ uint32_t kword(uint32_t pk) const {
    const uint32_t a = (__shfl_sync(0xffffffffu, pk, ks0) >> ksh) & 0xFFFFu;
    const uint32_t b = (__shfl_sync(0xffffffffu, pk, ks1) >> ksh) & 0xFFFFu;
    return a | (b << 16);
  }
  __device__ __forceinline__ uint32_t vword(uint32_t pv) const {
    const uint32_t a = __shfl_sync(0xffffffffu, pv, vs0) >> vsh;
    const uint32_t b = __shfl_sync(0xffffffffu, pv, vs1) >> vsh;
    return __byte_perm(a, b, 0x5140);
  }
};

// bf16 values: lane owns K words T = lane, lane + 32 (chunk T / 4, c =
// chunk % 4, j = 2 (chunk / 4) + (T % 4) / 2, h = T % 2: the bf16 pair of
// elements 2 (c%2), +1 of lane 4j + c/2 + 2h) and V words W = lane, lane + 32
// (row g = W / 8, M-block m = W % 8: element g % 4 of lanes 4m + g/4 (low
// half) and 4m + g/4 + 2 (high half)).
struct Gather16 {
  int ks[2], kreg, vs[2], vreg, vhalf;
  __device__ explicit Gather16(int lane) {
    const int c = (lane >> 2) & 3;
    kreg = c & 1;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int T = lane + 32 * i, chunk = T >> 2;
      const int j = 2 * (chunk >> 2) + ((T & 3) >> 1);
      ks[i] = 4 * j + (c >> 1) + 2 * (T & 1);
    }
    const int g0 = lane >> 3;  // rows g0 (W = lane) and g0 + 4 (W = lane + 32)
    const int m = lane & 7;
    vs[0] = 4 * m + (g0 >> 2);
    vs[1] = 4 * m + ((g0 + 4) >> 2);
    vreg = ((g0 & 3) >> 1);  // the same for g0 + 4
    vhalf = 16 * (g0 & 1);
  }
  __device__ __forceinline__ uint32_t kword(uint32_t k0, uint32_t k1, int i) const {
    const uint32_t a = __shfl_sync(0xffffffffu, k0, ks[i]);
    const uint32_t b = __shfl_sync(0xffffffffu, k1, ks[i]);
    return kreg ? b : a;
  }
  __device__ __forceinline__ uint32_t vword(uint32_t v0, uint32_t v1, int i) const {
    const uint32_t a0 = __shfl_sync(0xffffffffu, v0, vs[i]);
    const uint32_t a1 = __shfl_sync(0xffffffffu, v1, vs[i]);
    const uint32_t b0 = __shfl_sync(0xffffffffu, v0, vs[i] + 2);
    const uint32_t b1 = __shfl_sync(0xffffffffu, v1, vs[i] + 2);
    const uint32_t lo = ((vreg ? a1 : a0) >> vhalf) & 0xFFFFu;
    const uint32_t hi = ((vreg ? b1 : b0) >> vhalf) & 0xFFFFu;
    return lo | (hi << 16);
  }
};

// Codes of one lane's four channels in one register (code e at bits BITS e).
template <int BITS>
__device__ __forceinline__ uint32_t pack_codes(const uint32_t (&c)[4]) {
  return c[0] | (c[1] << BITS) | (c[2] << (2 * BITS)) | (c[3] << (3 * BITS));
}

// KPC: keys with per-channel groups -- the kernel writes the value section
// and its metadata only (the key codes are written when a group of
// positions completes, by gqa_append_kgroups) and leaves the lengths to the
// residual kernel, which runs last.
template <int BITS, int GS, bool SYM, bool KPC = false>
__global__ void __launch_bounds__(256)
    gqa_append_bulk(const GqaView v, const void *kin, const void *vin, int in_f32, int n_new,
                    const int32_t *n_per_seq, int32_t *err) {
  pdl_wait();
  pdl_trigger();
  static_assert(!KPC || (!SYM && BITS != 16), "per-channel keys: grouped codes");
  constexpr int D = 128, E = 4;
  constexpr int SEC = D * BITS / 8;                       // bytes per section
  constexpr int MBY = ((D / GS) * 8 + 15) & ~15;          // one section's group metadata
  constexpr int REC = SYM ? 2 * SEC : BITS == 16 ? 2 * SEC : 2 * SEC + (KPC ? 1 : 2) * MBY;
  constexpr int KM = 2 * SEC, VM = KPC ? 2 * SEC : KM + MBY;
  constexpr int NC = SEC / 16;                            // chunks per code section
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  const size_t total = (size_t)v.B * n_new * v.Hkv;
  Gather4 g4(lane);
  Gather8 g8(lane);
  Gather16 g16(lane);
  (void)g4; (void)g8; (void)g16;
  // two rows per iteration, their loads issued together and their
  // arithmetic independent (rows past the end compute on row 0's inputs and
  // store nothing)
  auto process = [&](const float (&xk)[E], const float (&xv)[E], bool ok, size_t row, int t) {
    uint8_t *rec = v.rec + row * REC;
    if constexpr (BITS == 16) {
      uint32_t k0 = pack2<true>(xk[0], xk[1]), k1 = pack2<true>(xk[2], xk[3]);
      uint32_t v0 = pack2<true>(xv[0], xv[1]), v1 = pack2<true>(xv[2], xv[3]);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const uint32_t kw = g16.kword(k0, k1, h), vw = g16.vword(v0, v1, h);
        if (ok) {
          reinterpret_cast<uint32_t *>(rec)[lane + 32 * h] = kw;
          reinterpret_cast<uint32_t *>(rec + SEC)[lane + 32 * h] = vw;
        }
      }
    } else {
      uint32_t ck[E], cv[E];
      if constexpr (SYM) {
        const uint32_t sk = quant_sym_lane<E>(xk, BITS, ck);
        const uint32_t sv = quant_sym_lane<E>(xv, BITS, cv);
        if (ok && lane == 0) v.scales[row] = sk | (sv << 16);
      } else {
        float ks = 0.f, kz = 0.f, vs, vz;
        if constexpr (!KPC) quant_lane<E>(xk, GS, (1 << BITS) - 1, ck, ks, kz);
        else for (int e = 0; e < E; ++e) ck[e] = 0u;
        quant_lane<E>(xv, GS, (1 << BITS) - 1, cv, vs, vz);
        if (ok && (lane * E) % GS == 0) {
          if constexpr (!KPC) reinterpret_cast<float2 *>(rec + KM)[(lane * E) / GS] = make_float2(ks, kz);
          reinterpret_cast<float2 *>(rec + VM)[(lane * E) / GS] = make_float2(vs, vz);
        }
      }
      const uint32_t pk = pack_codes<BITS>(ck), pv = pack_codes<BITS>(cv);
      // logical chunk of this lane's word(s) and its physical 16-byte slot:
      // symmetric records rotate all chunks by sym_rot(t), grouped ones the
      // V chunks by v_rot(t)
      if constexpr (BITS == 4) {
        const uint32_t w = g4.word(pk | (pv << 16));
        int off;
        if (lane < 16) {
          off = SYM ? 16 * (((lane >> 2) + sym_rot(t, REC / 16)) & (REC / 16 - 1)) + 4 * (lane & 3)
                    : 4 * lane;
        } else {
          const int u = lane - 16, k = u >> 2;
          off = SYM ? 16 * ((NC + k + sym_rot(t, REC / 16)) & (REC / 16 - 1)) + 4 * (u & 3)
                    : SEC + 16 * ((k + v_rot(t, REC, NC)) & (NC - 1)) + 4 * (u & 3);
        }
        if (ok && (!KPC || lane >= 16)) *reinterpret_cast<uint32_t *>(rec + off) = w;
      } else {
        const uint32_t kw = g8.kword(pk), vw = g8.vword(pv);
        const int kc = lane >> 2;
        const int koff = SYM ? 16 * ((kc + sym_rot(t, REC / 16)) & (REC / 16 - 1)) + 4 * (lane & 3)
                             : 4 * lane;
        const int voff = SYM ? 16 * ((NC + kc + sym_rot(t, REC / 16)) & (REC / 16 - 1)) + 4 * (lane & 3)
                             : SEC + 16 * ((kc + v_rot(t, REC, NC)) & (NC - 1)) + 4 * (lane & 3);
        if (ok) {
          if constexpr (!KPC) *reinterpret_cast<uint32_t *>(rec + koff) = kw;
          *reinterpret_cast<uint32_t *>(rec + voff) = vw;
        }
      }
    }
  };
  const size_t step = (size_t)gridDim.x * wpb;
  // 32-bit index arithmetic (the launcher sends fewer than 2^31 rows)
  const RowStep rstep((uint32_t)step, (uint32_t)v.Hkv, (uint32_t)n_new);
  RowIdx ridx = rstep.at((uint32_t)min((size_t)blockIdx.x * wpb + warp, total));
  for (size_t w0 = (size_t)blockIdx.x * wpb + warp; w0 < total; w0 += 2 * step) {
    bool ok[2];
    size_t row[2];
    int tt[2];
    float xk[2][E], xv[2][E];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const size_t wid = w0 + u * step;
      const RowIdx r = ridx;
      ridx = rstep.next(ridx);  // row wid + step
      ok[u] = false;
      row[u] = 0;
      tt[u] = 0;
      size_t in_off = 0;
      if (wid < total) {
        const int kvh = (int)r.kvh, i = (int)r.i, b = (int)r.b;
        in_off = wid * D;  // inputs are [B, n_new, H_kv, D], row wid
        const int nb = seq_count(n_per_seq, b, n_new, err);
        const int t = v.lens[b] + i;
        if (i < nb) {
          if (t >= v.cap) {
            if (lane == 0) set_err(err, 2);
          } else {
            ok[u] = true;
            row[u] = ((size_t)b * v.Hkv + kvh) * v.cap + t;
            tt[u] = t;
          }
        }
      }
      load_row<D>(kin, vin, in_f32, in_off, lane, xk[u], xv[u]);
    }
    process(xk[0], xv[0], ok[0], row[0], tt[0]);
    process(xk[1], xv[1], ok[1], row[1], tt[1]);
  }
  // the last CTA advances the lengths (per-channel keys: the residual
  // kernel does, after this one)
  if constexpr (KPC) return;
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

// Per-channel key groups completed by this append: one warp per (sequence,
// KV head, group of GS positions).  The group's keys (residual rows for
// positions already stored, the appended rows for new ones, rounded to
// bf16 as the residual holds them) are staged in natural channel order in
// shared memory; lane L quantises the channel pairs {c, c + 8} of pairs L
// (and L + 32 when D = 128; c = 16 (p / 8) + p % 8: the two channels of one
// 4-bit byte)
// over the group's positions: scale = fl((max - min) / levels) correctly
// rounded, codes rint((x - min) / scale) through the fast reciprocal with
// the rounding check of rint_quot_fast (the correctly rounded division
// where it cannot decide), the codes packed into the positions' key
// sections in shared memory and stored as whole 16-byte chunks.
constexpr int kKgWarps = 4;
// dynamic shared memory of gqa_append_kgroups: per warp the staged keys
// (GS rows of D + 8 bf16) and the key sections (GS rows of D bits / 8 bytes)
__host__ __device__ constexpr int kg_warp_bytes(int D, int GS, int bits) {
  return ((GS * (D + 8) * 2 + GS * D * bits / 8) + 15) & ~15;
}
template <int D>
__global__ void __launch_bounds__(32 * kKgWarps)
    gqa_append_kgroups(const GqaView v, const void *kin, int in_f32, int n_new,
                       const int32_t *n_per_seq, int32_t *err, int max_groups) {
  pdl_wait();
  pdl_trigger();
  constexpr int PAD = D + 8;                      // bf16 per staged row (conflict-free columns)
  extern __shared__ __align__(16) uint8_t kg_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t wid = (size_t)blockIdx.x * kKgWarps + warp;
  const size_t total = (size_t)v.B * v.Hkv * max_groups;
  if (wid >= total) return;
  const int gidx = (int)(wid % max_groups);
  const int kvh = (int)((wid / max_groups) % v.Hkv);
  const int b = (int)(wid / ((size_t)max_groups * v.Hkv));
  const int GS = v.group;
  const int nb = seq_count(n_per_seq, b, n_new, nullptr);
  const int len0 = v.lens[b];
  const int G = len0 / GS + gidx;  // candidate group
  if ((G + 1) * GS > len0 + nb || (G + 1) * GS > v.cap) return;  // not completed now (warp-uniform)
  const size_t slab = (size_t)b * v.Hkv + kvh;
  const RecLayout L = rec_layout(v.bits, D, GS, 1);
  const int sec = D * v.bits / 8;
  const uint8_t *res = v.resid + slab * (size_t)GS * D * 2;
  uint8_t *wbase = kg_smem + warp * kg_warp_bytes(D, GS, v.bits);
  uint16_t *xs = reinterpret_cast<uint16_t *>(wbase);
  uint8_t *ks = wbase + GS * PAD * 2;
  // ---- the group's keys, natural channel order ----
  constexpr int CPR = D / 8;  // 8-channel pieces per row
  for (int q = lane; q < GS * CPR; q += 32) {
    const int r = q / CPR, c8 = 8 * (q - r * CPR);
    const int p = G * GS + r;
    uint16_t h[8];
    if (p < len0) {
      // residual row r: bf16 in the key fragment order
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        int kb, khi;
        k_pos(c8 + e, 16, D, &kb, &khi);
        h[e] = *reinterpret_cast<const uint16_t *>(res + (size_t)r * D * 2 + kb);
      }
    } else {
      const size_t ii = (((size_t)b * n_new + (p - len0)) * v.Hkv + kvh) * D + c8;
      if (in_f32) {
        const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(kin) + ii);
        const float4 u0 = src[0], u1 = src[1];
        const float f[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) h[e] = f32_to_bf16_bits(f[e]);
      } else {
        const uint4 u = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(kin) + ii);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) { h[2 * e] = (uint16_t)(w[e] & 0xffffu); h[2 * e + 1] = (uint16_t)(w[e] >> 16); }
      }
    }
    uint4 o;
    o.x = h[0] | ((uint32_t)h[1] << 16); o.y = h[2] | ((uint32_t)h[3] << 16);
    o.z = h[4] | ((uint32_t)h[5] << 16); o.w = h[6] | ((uint32_t)h[7] << 16);
    *reinterpret_cast<uint4 *>(xs + r * PAD + c8) = o;
  }
  for (int q = lane; q < GS * sec / 16; q += 32) reinterpret_cast<uint4 *>(ks)[q] = make_uint4(0, 0, 0, 0);
  __syncwarp();
  // ---- per channel: scale, zero, codes ----
  const float lev = (float)((1 << v.bits) - 1);
#pragma unroll
  for (int pp = 0; pp < D / 64; ++pp) {  // D / 2 channel pairs, 32 per pass
    const int pr = lane + 32 * pp;
    const int ch0 = (pr >> 3) * 16 + (pr & 7);
    float sc[2], zr[2], rs[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int ch = ch0 + 8 * h;
      float mn = INFINITY, mx = -INFINITY;
      for (int r = 0; r < GS; ++r) {
        const float x = bf16_to_f32(xs[r * PAD + ch]);
        mn = fminf(mn, x);
        mx = fmaxf(mx, x);
      }
      sc[h] = __fdiv_rn(__fsub_rn(mx, mn), lev);
      zr[h] = mn;
      rs[h] = sc[h] == 0.f ? 0.f : __fdividef(1.f, sc[h]);
      v.gmeta[(slab * (v.cap / GS) + G) * D + ch] = make_float2(sc[h], mn);
    }
    int kb0, kh0, kb1, kh1;
    k_pos(ch0, v.bits, D, &kb0, &kh0);
    k_pos(ch0 + 8, v.bits, D, &kb1, &kh1);
    for (int r = 0; r < GS; ++r) {
      uint32_t c[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (sc[h] == 0.f) {
          c[h] = 0u;
        } else {
          const float d = __fsub_rn(bf16_to_f32(xs[r * PAD + ch0 + 8 * h]), zr[h]);
          bool near;
          float q = rint_quot_fast(d, rs[h], near);
          if (near) q = rintf(__fdiv_rn(d, sc[h]));
          c[h] = (uint32_t)fminf(fmaxf(q, 0.f), lev);
        }
      }
      if (v.bits == 8) {
        ks[r * sec + kb0] = (uint8_t)c[0];
        ks[r * sec + kb1] = (uint8_t)c[1];
      } else {
        // channels ch0 and ch0 + 8 share one byte (low and high nibble)
        ks[r * sec + kb0] = (uint8_t)(c[0] | (c[1] << 4));
      }
    }
  }
  __syncwarp();
  // ---- the group's key sections, whole 16-byte chunks ----
  const int cps = sec / 16;
  for (int q = lane; q < GS * cps; q += 32) {
    const int r = q / cps, u = q - r * cps;
    uint8_t *rec = v.rec + (slab * v.cap + (size_t)G * GS + r) * L.rec + L.k_off;
    reinterpret_cast<uint4 *>(rec)[u] = reinterpret_cast<const uint4 *>(ks + r * sec)[u];
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
  for (size_t wid = (size_t)blockIdx.x * 4 + warp; wid < (size_t)v.B * n_new;
       wid += (size_t)gridDim.x * 4) {
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
  for (size_t wid = (size_t)blockIdx.x * 4 + warp; wid < (size_t)v.B * n_new;
       wid += (size_t)gridDim.x * 4) {
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
    __syncwarp();  // the row buffer is free again
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

// CTAs of `wpc` row warps for `rows` rows: one per wpc rows, up to 2048
// threads per SM of the current device; the kernels loop over the rest
unsigned row_blocks(size_t rows, int wpc = 4) {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
      sms = 148;
  }
  const size_t need = (rows + wpc - 1) / wpc, cap = (size_t)sms * (64 / wpc);
  return (unsigned)(need < cap ? (need > 0 ? need : 1) : cap);
}

}  // namespace

cudaError_t launch_gqa_append(const GqaView &v, const void *k, const void *vv, int in_f32,
                              int n_new, const int32_t *n_per_seq, int32_t *err,
                              cudaStream_t st) {
  const size_t rows = (size_t)v.B * n_new * v.Hkv;
  const unsigned blocks = row_blocks(rows);
  const bool kpc = v.bits != 16 && v.key_axis == 1;
  const bool d128 = v.D == 128;
  cudaError_t e = cudaSuccess;
  if (kpc) {
    // groups first (they read residual rows the open group may overwrite)
    const int max_groups = (n_new + v.group - 1) / v.group + 1;
    const size_t warps = (size_t)v.B * v.Hkv * max_groups;
    const dim3 grid((unsigned)((warps + kKgWarps - 1) / kKgWarps));
    auto kern = d128 ? gqa_append_kgroups<128> : gqa_append_kgroups<64>;
    const int smem = kKgWarps * kg_warp_bytes(v.D, v.group, v.bits);
    static bool attr_set = false;
    if (!attr_set) {
      // the largest need: head_dim 128, groups of 64, 8-bit codes
      const int most = kKgWarps * kg_warp_bytes(128, 64, 8);
      e = cudaFuncSetAttribute(gqa_append_kgroups<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(gqa_append_kgroups<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
      if (e != cudaSuccess) return e;
      attr_set = true;
    }
    e = launch_pdl(kern, grid, dim3(32 * kKgWarps), (size_t)smem, st, v, k, in_f32, n_new, n_per_seq, err,
                   max_groups);
  }
  if (e == cudaSuccess) {
    const dim3 bg(row_blocks(rows, 8));
    if (kpc && (size_t)n_new * v.Hkv > 64 && d128 && rows < (1u << 31) && (v.bits == 8 || v.bits == 4)) {
      // bulk appends of the values beside per-channel keys (head_dim 128)
      auto bulk = [&](auto kern) {
        return launch_pdl(kern, bg, dim3(256), 0, st, v, k, vv, in_f32, n_new, n_per_seq, err);
      };
      if (v.bits == 8) e = v.group == 32 ? bulk(gqa_append_bulk<8, 32, false, true>) : bulk(gqa_append_bulk<8, 64, false, true>);
      else e = v.group == 32 ? bulk(gqa_append_bulk<4, 32, false, true>) : bulk(gqa_append_bulk<4, 64, false, true>);
    } else if (!kpc && (size_t)n_new * v.Hkv > 64 && d128 && rows < (1u << 31) &&
        (v.bits == 16 || v.bits == 8 || v.bits == 4)) {
      // bulk appends of the per-token layouts with head_dim 128
      const bool sym = v.scheme == kSchemeSym;
      auto bulk = [&](auto kern) {
        return launch_pdl(kern, bg, dim3(256), 0, st, v, k, vv, in_f32, n_new, n_per_seq, err);
      };
      if (v.bits == 16) e = bulk(gqa_append_bulk<16, 64, false>);
      else if (sym) e = v.bits == 8 ? bulk(gqa_append_bulk<8, 64, true>) : bulk(gqa_append_bulk<4, 64, true>);
      else if (v.bits == 8) e = v.group == 32 ? bulk(gqa_append_bulk<8, 32, false>) : bulk(gqa_append_bulk<8, 64, false>);
      else e = v.group == 32 ? bulk(gqa_append_bulk<4, 32, false>) : bulk(gqa_append_bulk<4, 64, false>);
    } else if (!kpc && (size_t)n_new * v.Hkv <= 64)
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
  const dim3 grid(row_blocks(rows));
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
