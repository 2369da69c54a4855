// export.cu -- copy an anchor's stored state out in canonical order.
//
// Reverses the fragment-order permutation of layout.h so that a caller (or a
// test) sees codes as [batch, kv head, position, channel], one per byte,
// with the float (scale, zero) metadata beside them.
#include "common.cuh"
#include "kernels.h"
#include "layout.h"

namespace kvk {
namespace {

__global__ void gqa_export_kernel(const GqaView v, uint8_t *k_out, uint8_t *v_out, float *k_scale,
                                  float *k_zero, float *v_scale, float *v_zero, int max_ctx) {
  const int D = v.D;
  const size_t total = (size_t)v.B * v.Hkv * max_ctx * D;
  const RecLayout L = rec_layout(v.bits, D, v.group, v.key_axis);
  const int esz = v.bits == 16 ? 2 : 1;
  for (size_t id = (size_t)blockIdx.x * blockDim.x + threadIdx.x; id < total;
       id += (size_t)gridDim.x * blockDim.x) {
    const int ch = (int)(id % D);
    const size_t row = id / D;  // (slab, t)
    const int t = (int)(row % max_ctx);
    const size_t slab = row / max_ctx;
    if (v.scheme == kSchemeSym) {
      // signed codes in [-q, q] and the two bf16 scales, widened
      const uint8_t *rec = v.rec + (slab * v.cap + t) * v.rec_bytes;
      const int q = sym_levels(v.bits), mask = (1 << v.bits) - 1;
      for (int kv = 0; kv < 2; ++kv) {
        uint8_t *dst = kv ? v_out : k_out;
        if (!dst) continue;
        const int lb = kv ? sym_v_bit(ch, v.bits, D) + D * v.bits : sym_k_bit(ch, v.bits, D);
        const int pb = sym_phys(lb >> 3, t, v.rec_bytes);
        const int u = (rec[pb] >> (lb & 7)) & mask;
        dst[id] = (uint8_t)(int8_t)(u - q);
      }
      if (ch == 0) {
        const uint32_t w = v.scales[slab * v.cap + t];
        if (k_scale) k_scale[row] = bf16_to_f32((uint16_t)(w & 0xffffu));
        if (v_scale) v_scale[row] = bf16_to_f32((uint16_t)(w >> 16));
      }
      continue;
    }
    const uint8_t *rec = v.rec + (slab * v.cap + t) * L.rec;
    for (int kv = 0; kv < 2; ++kv) {
      uint8_t *dst = kv ? v_out : k_out;
      if (!dst) continue;
      int byte, hi;
      if (kv)
        v_pos(ch, v.bits, D, t, L.rec, &byte, &hi);
      else
        k_pos(ch, v.bits, D, &byte, &hi);
      const uint8_t *sec = rec + (kv ? L.v_off : L.k_off);
      if (esz == 2) {
        reinterpret_cast<uint16_t *>(dst)[id] = *reinterpret_cast<const uint16_t *>(sec + byte);
      } else if (v.bits == 8) {
        dst[id] = sec[byte];
      } else {
        dst[id] = hi ? (sec[byte] >> 4) : (sec[byte] & 15);
      }
    }
    if (v.bits != 16 && ch % v.group == 0) {
      const int gi = ch / v.group;
      const size_t mi = row * (D / v.group) + gi;
      const float2 vm = reinterpret_cast<const float2 *>(rec + L.vm_off)[gi];
      if (v_scale) v_scale[mi] = vm.x;
      if (v_zero) v_zero[mi] = vm.y;
      if (v.key_axis == 0) {
        const float2 km = reinterpret_cast<const float2 *>(rec + L.km_off)[gi];
        if (k_scale) k_scale[mi] = km.x;
        if (k_zero) k_zero[mi] = km.y;
      }
    }
  }
}

// Per-channel key metadata [slab][G][D] and residual rows [slab][g][D].
__global__ void gqa_export_kgroups(const GqaView v, float *k_scale, float *k_zero,
                                   uint16_t *k_resid, int max_ctx) {
  const int D = v.D, GS = v.group;
  const int nG = max_ctx / GS;
  const size_t slabs = (size_t)v.B * v.Hkv;
  const size_t n1 = slabs * nG * D, n2 = slabs * GS * D;
  for (size_t id = (size_t)blockIdx.x * blockDim.x + threadIdx.x; id < n1 + n2;
       id += (size_t)gridDim.x * blockDim.x) {
    if (id < n1) {
      const int ch = (int)(id % D);
      const int G = (int)((id / D) % nG);
      const size_t slab = id / ((size_t)D * nG);
      const float2 m = v.gmeta[(slab * (v.cap / GS) + G) * D + ch];
      if (k_scale) k_scale[id] = m.x;
      if (k_zero) k_zero[id] = m.y;
    } else if (k_resid) {
      const size_t j = id - n1;
      const int ch = (int)(j % D);
      const size_t rowi = j / D;  // slab * GS + r
      int byte, hi;
      k_pos(ch, 16, D, &byte, &hi);
      k_resid[j] = *reinterpret_cast<const uint16_t *>(v.resid + rowi * D * 2 + byte);
    }
  }
}

__global__ void mla_export_kernel(const MlaView v, uint16_t *c_out, uint16_t *kr_out,
                                  int max_ctx) {
  const int W = v.width + v.rope;
  const size_t total = (size_t)v.B * max_ctx * W;
  for (size_t id = (size_t)blockIdx.x * blockDim.x + threadIdx.x; id < total;
       id += (size_t)gridDim.x * blockDim.x) {
    const int e = (int)(id % W);
    const size_t row = id / W;
    const int t = (int)(row % max_ctx);
    const size_t b = row / max_ctx;
    const uint16_t x = reinterpret_cast<const uint16_t *>(v.rec + (b * v.cap + t) * v.rec_bytes)[e];
    if (e < v.width) {
      if (c_out) c_out[row * v.width + e] = x;
    } else if (kr_out) {
      kr_out[row * v.rope + (e - v.width)] = x;
    }
  }
}

// Quantised MLA anchor: codes of the latent [B, T, width] and of k^R [B, T,
// rope] (signed codes for the symmetric scheme, unsigned for the grouped
// one), one byte each, and the per-position scales (and zeros).
__global__ void mla_export_q_kernel(const MlaView v, uint8_t *c_out, uint8_t *kr_out,
                                    float *c_scale, float *c_zero, float *kr_scale, float *kr_zero,
                                    int max_ctx) {
  const int KH = v.width + v.rope;
  const int off = v.scheme == kSchemeSym ? sym_levels(v.bits) : 0;
  const size_t total = (size_t)v.B * max_ctx * KH;
  for (size_t id = (size_t)blockIdx.x * blockDim.x + threadIdx.x; id < total;
       id += (size_t)gridDim.x * blockDim.x) {
    const int k = (int)(id % KH);
    const size_t row = id / KH;
    const int t = (int)(row % max_ctx);
    const size_t b = row / max_ctx;
    const size_t pos = b * v.cap + t;
    const uint8_t *rec = v.rec + pos * v.rec_bytes;
    uint32_t chunk;
    if (v.bits == 8) chunk = reinterpret_cast<const uint32_t *>(rec)[(k >> 3) * 2 + ((k & 7) >> 2)] >>
                             (8 * (k & 3));
    else if (v.bits == 4) chunk = reinterpret_cast<const uint32_t *>(rec)[k >> 3] >> mla_q_bit(k & 7, 4);
    else chunk = (uint32_t)reinterpret_cast<const uint16_t *>(rec)[k >> 3] >> mla_q_bit(k & 7, 2);
    const int u = (int)(chunk & ((1u << v.bits) - 1));
    const uint8_t code = (uint8_t)(int8_t)(u - off);
    if (k < v.width) {
      if (c_out) c_out[row * v.width + k] = code;
    } else if (kr_out) {
      kr_out[row * v.rope + (k - v.width)] = code;
    }
    if (k == 0) {
      float sc, zc, sr, zr;
      if (v.scheme == kSchemeSym) {
        const uint32_t w = reinterpret_cast<const uint32_t *>(v.meta)[pos];
        sc = __uint_as_float(w << 16);
        sr = __uint_as_float(w & 0xffff0000u);
        zc = zr = 0.f;
      } else {
        const float4 m = reinterpret_cast<const float4 *>(v.meta)[pos];
        sc = m.x; zc = m.y; sr = m.z; zr = m.w;
      }
      if (c_scale) c_scale[row] = sc;
      if (c_zero) c_zero[row] = zc;
      if (kr_scale) kr_scale[row] = sr;
      if (kr_zero) kr_zero[row] = zr;
    }
  }
}

}  // namespace

cudaError_t launch_gqa_export(const GqaView &v, void *k_out, void *v_out, float *k_scale,
                              float *k_zero, float *v_scale, float *v_zero, void *k_resid,
                              int max_ctx, cudaStream_t st) {
  gqa_export_kernel<<<1024, 256, 0, st>>>(v, static_cast<uint8_t *>(k_out),
                                          static_cast<uint8_t *>(v_out), k_scale, k_zero,
                                          v_scale, v_zero, max_ctx);
  if (v.bits != 16 && v.key_axis == 1)
    gqa_export_kgroups<<<1024, 256, 0, st>>>(v, k_scale, k_zero,
                                             static_cast<uint16_t *>(k_resid), max_ctx);
  return cudaGetLastError();
}

cudaError_t launch_mla_export(const MlaView &v, void *c_out, void *kr_out, float *c_scale,
                              float *c_zero, float *kr_scale, float *kr_zero, int max_ctx,
                              cudaStream_t st) {
  if (v.bits != 16)
    mla_export_q_kernel<<<1024, 256, 0, st>>>(v, static_cast<uint8_t *>(c_out),
                                              static_cast<uint8_t *>(kr_out), c_scale, c_zero,
                                              kr_scale, kr_zero, max_ctx);
  else
    mla_export_kernel<<<1024, 256, 0, st>>>(v, static_cast<uint16_t *>(c_out),
                                            static_cast<uint16_t *>(kr_out), max_ctx);
  return cudaGetLastError();
}

}  // namespace kvk
