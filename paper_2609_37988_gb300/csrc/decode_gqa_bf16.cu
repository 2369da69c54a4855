// decode_gqa_bf16.cu -- instantiations of the GQA decode kernel for
// 16-bit caches (one translation unit per bit-width so they build in parallel).
#include "decode_gqa.cuh"

namespace kvk {

cudaError_t launch_gqa_decode_b16(const GqaDecodeArgs &a, cudaStream_t st) {
  if (a.v.D == 128) return launch_gqa_decode_t<16, 128, 0, 32>(a, st);
  if (a.v.D == 64) return launch_gqa_decode_t<16, 64, 0, 32>(a, st);
  return cudaErrorInvalidValue;
}

int gqa_ctas_b16(int D, int, int) {
  if (D == 128) return gqa_ctas_per_sm_t<16, 128, 0, 32>();
  return gqa_ctas_per_sm_t<16, 64, 0, 32>();
}
}  // namespace kvk
