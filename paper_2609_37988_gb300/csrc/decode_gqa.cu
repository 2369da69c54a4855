// decode_gqa.cu -- dispatch of the GQA decode kernel by cache format, and
// the tensor maps its kept-list gather reads.
#include <cuda.h>  // CUtensorMap and its enums (the encoder is reached through the runtime)

#include "kernels.h"
#include "layout.h"

namespace kvk {

cudaError_t launch_gqa_decode_b16(const GqaDecodeArgs &a, cudaStream_t st);
cudaError_t launch_gqa_decode_b8(const GqaDecodeArgs &a, cudaStream_t st);
cudaError_t launch_gqa_decode_b4(const GqaDecodeArgs &a, cudaStream_t st);
int gqa_ctas_b16(int D, int kax, int gs);
int gqa_ctas_b8(int D, int kax, int gs);
int gqa_ctas_b4(int D, int kax, int gs);
cudaError_t launch_gqa_decode_sym(const GqaDecodeArgs &a, cudaStream_t st);
int gqa_ctas_sym(int bits);
int gqa_tile_sym(int bits);

cudaError_t launch_gqa_decode(const GqaDecodeArgs &a, cudaStream_t st) {
  if (a.v.bits != 16 && a.v.scheme == kSchemeSym) return launch_gqa_decode_sym(a, st);
  switch (a.v.bits) {
    case 16: return launch_gqa_decode_b16(a, st);
    case 8: return launch_gqa_decode_b8(a, st);
    case 4: return launch_gqa_decode_b4(a, st);
    default: return cudaErrorInvalidValue;
  }
}

// positions per decode tile: 128 for per-token 4-bit keys and symmetric
// 4- and 2-bit caches, else 64
int gqa_decode_tile(int bits, int D, int key_axis, int group, int scheme) {
  (void)D; (void)group;
  if (bits != 16 && scheme == kSchemeSym) return gqa_tile_sym(bits);
  return (bits == 4 && key_axis == 0) ? 128 : 64;
}

// grouped int8/int4 with per-token keys gather whole records by tensor-map
// rows (GqaCfg::GTMA); the other formats copy 16-byte chunks
bool gqa_decode_row_gather(int bits, int key_axis, int scheme) {
  return (bits == 8 || bits == 4) && key_axis == 0 && scheme != kSchemeSym;
}

cudaError_t encode_tensor_map_tiled(void *map, int dtype, int rank, void *base,
                                    const uint64_t *dims, const uint64_t *strides,
                                    const uint32_t *box, const uint32_t *elem_strides,
                                    int interleave, int swizzle, int l2_promotion, int oob_fill) {
  using Encode = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                              const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                              const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  static Encode encode = nullptr;
  if (!encode) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    const cudaError_t e =
        cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    encode = reinterpret_cast<Encode>(fn);
  }
  const CUresult r = encode(static_cast<CUtensorMap *>(map), (CUtensorMapDataType)dtype,
                            (cuuint32_t)rank, base, reinterpret_cast<const cuuint64_t *>(dims),
                            reinterpret_cast<const cuuint64_t *>(strides),
                            reinterpret_cast<const cuuint32_t *>(box),
                            reinterpret_cast<const cuuint32_t *>(elem_strides),
                            (CUtensorMapInterleave)interleave, (CUtensorMapSwizzle)swizzle,
                            (CUtensorMapL2promotion)l2_promotion, (CUtensorMapFloatOOBfill)oob_fill);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// The record table of a GQA anchor as a 2-D tensor of 32-bit words: row
// slab * cap + position (slab = b * Hkv + kvh), rec_bytes / 4 words per
// row; one box is one record (a row copy fetches four).
cudaError_t gqa_make_rows_tmap(void *out, const GqaView &v) {
  const uint64_t rows = (uint64_t)v.B * (uint64_t)v.Hkv * (uint64_t)v.cap;
  if (rows >= (1ull << 31) || v.rec_bytes % 16 != 0 || v.rec_bytes / 4 > 256) return cudaErrorInvalidValue;
  const uint64_t dims[2] = {(uint64_t)v.rec_bytes / 4, rows};
  const uint64_t strides[1] = {(uint64_t)v.rec_bytes};
  const uint32_t box[2] = {(uint32_t)v.rec_bytes / 4, 1};
  const uint32_t estr[2] = {1, 1};
  return encode_tensor_map_tiled(out, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, v.rec, dims, strides, box,
                                 estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                                 CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

int gqa_decode_ctas_per_sm(int bits, int D, int key_axis, int group, int scheme) {
  if (bits != 16 && scheme == kSchemeSym) return gqa_ctas_sym(bits);
  switch (bits) {
    case 16: return gqa_ctas_b16(D, key_axis, group);
    case 8: return gqa_ctas_b8(D, key_axis, group);
    case 4: return gqa_ctas_b4(D, key_axis, group);
    default: return 1;
  }
}

}  // namespace kvk
