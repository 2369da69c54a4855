// decode_gqa_q4.cu -- instantiations of the GQA decode kernel for
// 4-bit caches (one translation unit per bit-width so they build in parallel).
#include "decode_gqa.cuh"

namespace kvk {

cudaError_t launch_gqa_decode_b4(const GqaDecodeArgs &a, cudaStream_t st) {
#define KVK_CASE(D_, KAX_, GS_) \
  if (a.v.D == D_ && a.v.key_axis == KAX_ && a.v.group == GS_) \
    return launch_gqa_decode_t<4, D_, KAX_, GS_>(a, st);
  KVK_CASE(128, 0, 32) KVK_CASE(128, 0, 64) KVK_CASE(128, 1, 32) KVK_CASE(128, 1, 64)
  KVK_CASE(64, 0, 32) KVK_CASE(64, 0, 64) KVK_CASE(64, 1, 32) KVK_CASE(64, 1, 64)
#undef KVK_CASE
  return cudaErrorInvalidValue;
}

int gqa_ctas_b4(int D, int kax, int gs) {
#define KVK_CASE(D_, KAX_, GS_) \
  if (D == D_ && kax == KAX_ && gs == GS_) return gqa_ctas_per_sm_t<4, D_, KAX_, GS_>();
  KVK_CASE(128, 0, 32) KVK_CASE(128, 0, 64) KVK_CASE(128, 1, 32) KVK_CASE(128, 1, 64)
  KVK_CASE(64, 0, 32) KVK_CASE(64, 0, 64) KVK_CASE(64, 1, 32) KVK_CASE(64, 1, 64)
#undef KVK_CASE
  return 1;
}
}  // namespace kvk
