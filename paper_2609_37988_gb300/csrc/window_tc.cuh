// window_tc.cuh -- pieces shared by the tensor-core kernels that score a
// block of query rows against a compressed GQA cache (the window-vote
// evictor and chunk attention): key formats, the bf16 hi/lo split into the
// K-major 128-byte-swizzled shared-memory layout the tcgen05 MMA reads, the
// per-quarter key dequantiser, worker barriers.  Head dim 128.
#pragma once

#include <stdint.h>

#include "common.cuh"
#include "layout.h"

namespace kvk {

// named barrier 1 over the first N threads (the worker warps; an MMA warp
// after them runs on its own)
template <int N>
__device__ __forceinline__ void workers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(N) : "memory");
}
template <int N>
__device__ __forceinline__ bool workers_sync_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, %2, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(N)
      : "memory");
  return r != 0;
}

// 16-byte chunks of a head_dim-128 K section per key format
__host__ __device__ constexpr int TcFmtKs16(int fmt) {
  return fmt == 0 ? 16 : (fmt == 1 || fmt == 3) ? 8 : (fmt == 2 || fmt == 4) ? 4 : 2;
}

// key formats of the tensor-core dequantiser
enum { kFmtBf16 = 0, kFmtG8, kFmtG4, kFmtS8, kFmtS4, kFmtS2 };

template <int FMT>
struct TcFmt {
  static constexpr int BITS = FMT == kFmtBf16                   ? 16
                              : (FMT == kFmtG8 || FMT == kFmtS8) ? 8
                              : (FMT == kFmtG4 || FMT == kFmtS4) ? 4
                                                                 : 2;
  static constexpr bool SYM = FMT >= kFmtS8;
  static constexpr int KS = 128 * BITS / 8;  // K-section bytes
};

// hi (and lo) bf16 words of 8 channels -> one swizzled 16-byte chunk of row
// `row` holding channels ch0 .. ch0 + 7 (box stride `box` bytes)
__device__ __forceinline__ void put_chunk(uint8_t *buf, int row, int ch0, int box, uint4 w) {
  const int off = (ch0 >> 6) * box + row * 128 + ((((ch0 & 63) >> 3) ^ (row & 7)) << 4);
  *reinterpret_cast<uint4 *>(buf + off) = w;
}
__device__ __forceinline__ void put8(uint8_t *hi, uint8_t *lo, bool with_lo, int row, int ch0,
                                     int box, const float (&x)[8]) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) split2<true>(x[2 * i], x[2 * i + 1], h[i], l[i]);
  put_chunk(hi, row, ch0, box, make_uint4(h[0], h[1], h[2], h[3]));
  if (with_lo) put_chunk(lo, row, ch0, box, make_uint4(l[0], l[1], l[2], l[3]));
}
// exact float of a small unsigned integer (< 2^23) on the FMA/ALU pipes
__device__ __forceinline__ float u2f(uint32_t u) {
  return __uint_as_float(0x4B000000u | u) - 8388608.f;
}

// Channels 32 qc .. 32 qc + 31 of one position's key, from its staged K
// section (logical order) and `kmeta` (the key group metadata, or the
// symmetric scale word), dequantised into the key stage (hi, and lo unless
// bf16).
// Every layout places quarter qc at a fixed offset from quarter 0 with the
// same pattern (bf16: +64 bytes per quarter; 8-bit: +64 (qc >> 1) + 8 (qc &
// 1) bytes; 4-bit: +4 qc bytes; 2-bit: +32 (qc >> 1) + 8 (qc & 1) bits), so
// the quarter's words are loaded at a run-time offset and the channels are
// picked out at the compile-time positions of quarter 0.
template <int FMT, int KBOX = 128 * 128>
__device__ __forceinline__ void tc_dequant(const uint8_t *bundle, const uint8_t *kmeta, int row,
                                           int qc, int gshift, uint8_t *kh, uint8_t *kl) {
  using F = TcFmt<FMT>;
  constexpr int D = 128;
  const uint32_t *bw = reinterpret_cast<const uint32_t *>(bundle);
  if constexpr (F::BITS == 16) {
    static_assert(!F::SYM && F::KS == 256, "bf16 keys: 256 bytes, no scale");
    // bf16 keys are exact: gather them into channel order, no lo part
    uint32_t w[16];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const uint4 u = reinterpret_cast<const uint4 *>(bundle)[4 * qc + c];
      w[4 * c] = u.x; w[4 * c + 1] = u.y; w[4 * c + 2] = u.z; w[4 * c + 3] = u.w;
    }
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
      uint32_t o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        int b0, b1, h0, h1;
        k_pos(8 * cc + 2 * i, 16, D, &b0, &h0);
        k_pos(8 * cc + 2 * i + 1, 16, D, &b1, &h1);
        const uint32_t sel = (uint32_t)((b0 & 3) | (((b0 & 3) + 1) << 4) | ((4 + (b1 & 3)) << 8) |
                                        ((5 + (b1 & 3)) << 12));
        o[i] = __byte_perm(w[b0 >> 2], w[b1 >> 2], sel);
      }
      put_chunk(kh, row, 32 * qc + 8 * cc, KBOX, make_uint4(o[0], o[1], o[2], o[3]));
    }
  } else {
    constexpr int QL = (1 << (F::BITS - 1)) - 1;  // symmetric code offset
    // the quarter's words; channel l of quarter 0 sits in word W(l) at bit S(l)
    constexpr int NW = F::BITS == 8 ? 8 : 4;
    uint32_t w[NW];
    if constexpr (F::BITS == 8) {
      const int ob = 16 * (qc >> 1) + 2 * (qc & 1);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const uint2 u = *reinterpret_cast<const uint2 *>(bw + 4 * c + ob);
        w[2 * c] = u.x; w[2 * c + 1] = u.y;
      }
    } else if constexpr (F::BITS == 4) {
#pragma unroll
      for (int c = 0; c < 4; ++c) w[c] = bw[4 * c + qc];
    } else {
#pragma unroll
      for (int c = 0; c < 4; ++c) w[c] = bw[2 * c + (qc >> 1)] >> (8 * (qc & 1));
    }
    const float sym_s = F::SYM ? __uint_as_float(*reinterpret_cast<const uint32_t *>(kmeta) << 16) : 0.f;
    // groups of 32 or 64 channels: the quarter lies in one group
    float2 m = make_float2(0.f, 0.f);
    if constexpr (!F::SYM) m = *reinterpret_cast<const float2 *>(kmeta + 8 * ((32 * qc) >> gshift));
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
      const int ch0 = 32 * qc + 8 * cc;
      float x[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int l = 8 * cc + i;  // channel of quarter 0
        int wi, sh;
        if constexpr (F::BITS == 2) {
          const int bit = sym_k_bit(l, 2, D);
          wi = bit >> 6;
          sh = bit & 63;
        } else {
          int byte, hi;
          k_pos(l, F::BITS, D, &byte, &hi);
          wi = F::BITS == 8 ? 2 * (byte >> 4) + ((byte & 15) >> 2) : byte >> 4;
          sh = 8 * (byte & 3) + 4 * hi;
        }
        const uint32_t u = (w[wi] >> sh) & ((1u << F::BITS) - 1u);
        x[i] = F::SYM ? sym_s * (u2f(u) - (float)QL) : fmaf(u2f(u), m.x, m.y);
      }
      put8(kh, kl, true, row, ch0, KBOX, x);
    }
  }
}

// The same for keys with per-channel groups (KIVI layout): the position's
// codes (K section in the same channel order as per-token codes) and the
// (scale, zero) of each channel for the position's group of positions, mrow
// [128] float2.
template <int BITS, int KBOX = 128 * 128>
__device__ __forceinline__ void tc_dequant_kpc(const uint8_t *bundle, const float2 *mrow, int row,
                                               int qc, uint8_t *kh, uint8_t *kl) {
  static_assert(BITS == 8 || BITS == 4, "per-channel keys: 8- or 4-bit codes");
  constexpr int D = 128;
  const uint32_t *bw = reinterpret_cast<const uint32_t *>(bundle);
  constexpr int NW = BITS == 8 ? 8 : 4;
  uint32_t w[NW];
  if constexpr (BITS == 8) {
    const int ob = 16 * (qc >> 1) + 2 * (qc & 1);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const uint2 u = *reinterpret_cast<const uint2 *>(bw + 4 * c + ob);
      w[2 * c] = u.x; w[2 * c + 1] = u.y;
    }
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c) w[c] = bw[4 * c + qc];
  }
#pragma unroll
  for (int cc = 0; cc < 4; ++cc) {
    const int ch0 = 32 * qc + 8 * cc;
    float x[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int l = 8 * cc + i;  // channel of quarter 0
      int byte, hi;
      k_pos(l, BITS, D, &byte, &hi);
      const int wi = BITS == 8 ? 2 * (byte >> 4) + ((byte & 15) >> 2) : byte >> 4;
      const int sh = 8 * (byte & 3) + 4 * hi;
      const uint32_t u = (w[wi] >> sh) & ((1u << BITS) - 1u);
      const float2 m = mrow[ch0 + i];
      x[i] = fmaf(u2f(u), m.x, m.y);
    }
    put8(kh, kl, true, row, ch0, KBOX, x);
  }
}

// Channels 32 qc .. 32 qc + 31 of one position's value, from the V section
// of its staged record (logical order, rotation undone) and its metadata
// (grouped: the (scale, zero) pairs of the value groups; symmetric: the
// value scale), dequantised into a value stage with the key stage's layout
// (rows = positions, 64-channel boxes of `VBOX` bytes).  As for keys, every
// value layout places quarter qc at a fixed offset from quarter 0 (bf16: +8
// bytes in each 32-byte row of 16 channels; 8-bit: +32 qc bytes; 4-bit: +16
// qc bytes; 2-bit: +16 (qc >> 1) + (qc & 1) bytes).
template <int FMT, int VBOX>
__device__ __forceinline__ void tc_dequant_v(const uint8_t *vsec, const uint8_t *vmeta, float sym_s,
                                             int row, int qc, int gshift, uint8_t *vh, uint8_t *vl) {
  using F = TcFmt<FMT>;
  const uint32_t *vw = reinterpret_cast<const uint32_t *>(vsec);
  if constexpr (F::BITS == 16) {
    // channel l of quarter 0: 16-bit half e = (l >> 3) & 1 of word
    // 2 (l & 7) + (l >> 4) of the quarter's words w[2g + e'] = vw[8g + 2qc + e']
    uint32_t w[16];
#pragma unroll
    for (int g = 0; g < 8; ++g) {
      const uint2 u = *reinterpret_cast<const uint2 *>(vw + 8 * g + 2 * qc);
      w[2 * g] = u.x; w[2 * g + 1] = u.y;
    }
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
      uint32_t o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int l0 = 8 * cc + 2 * i, l1 = l0 + 1;
        const int b0 = 4 * (2 * (l0 & 7) + (l0 >> 4)) + 2 * ((l0 >> 3) & 1);
        const int b1 = 4 * (2 * (l1 & 7) + (l1 >> 4)) + 2 * ((l1 >> 3) & 1);
        const uint32_t sel = (uint32_t)((b0 & 3) | (((b0 & 3) + 1) << 4) | ((4 + (b1 & 3)) << 8) |
                                        ((5 + (b1 & 3)) << 12));
        o[i] = __byte_perm(w[b0 >> 2], w[b1 >> 2], sel);
      }
      put_chunk(vh, row, 32 * qc + 8 * cc, VBOX, make_uint4(o[0], o[1], o[2], o[3]));
    }
  } else {
    constexpr int QL = (1 << (F::BITS - 1)) - 1;
    constexpr int NW = F::BITS == 8 ? 8 : 4;
    uint32_t w[NW];
    if constexpr (F::BITS == 8) {
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const uint4 u = *reinterpret_cast<const uint4 *>(vw + 8 * qc + 4 * i);
        w[4 * i] = u.x; w[4 * i + 1] = u.y; w[4 * i + 2] = u.z; w[4 * i + 3] = u.w;
      }
    } else if constexpr (F::BITS == 4) {
      const uint4 u = *reinterpret_cast<const uint4 *>(vw + 4 * qc);
      w[0] = u.x; w[1] = u.y; w[2] = u.z; w[3] = u.w;
    } else {
      const uint4 u = *reinterpret_cast<const uint4 *>(vw + 4 * (qc >> 1));
      const int sh = 8 * (qc & 1);
      w[0] = u.x >> sh; w[1] = u.y >> sh; w[2] = u.z >> sh; w[3] = u.w >> sh;
    }
    float2 m = make_float2(0.f, 0.f);
    if constexpr (!F::SYM) m = *reinterpret_cast<const float2 *>(vmeta + 8 * ((32 * qc) >> gshift));
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
      float x[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int l = 8 * cc + i;  // channel of quarter 0
        const int g = l & 7, e = (l >> 3) & 1, hh = l >> 4;
        int wi, sh;
        if constexpr (F::BITS == 8) {
          const int bl = 16 * hh + 2 * g + e;
          wi = bl >> 2;
          sh = 8 * (bl & 3);
        } else if constexpr (F::BITS == 4) {
          const int bl = 2 * g + hh;
          wi = bl >> 2;
          sh = 8 * (bl & 3) + 4 * e;
        } else {
          wi = g >> 1;
          sh = 16 * (g & 1) + 2 * (2 * hh + e);
        }
        const uint32_t u = (w[wi] >> sh) & ((1u << F::BITS) - 1u);
        x[i] = F::SYM ? sym_s * (u2f(u) - (float)QL) : fmaf(u2f(u), m.x, m.y);
      }
      put8(vh, vl, true, row, 32 * qc + 8 * cc, VBOX, x);
    }
  }
}

}  // namespace kvk
