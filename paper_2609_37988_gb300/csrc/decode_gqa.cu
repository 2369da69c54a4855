// decode_gqa.cu -- dispatch of the GQA decode kernel by cache format.
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
