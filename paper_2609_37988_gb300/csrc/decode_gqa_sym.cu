// decode_gqa_sym.cu -- instantiations of the GQA decode kernel for caches
// quantised with the symmetric per-vector scheme (one bf16 scale per
// token-head row, Appendix C.3): 8, 4 and 2 bits, head_dim 128.
#include "decode_gqa.cuh"

namespace kvk {

cudaError_t launch_gqa_decode_sym(const GqaDecodeArgs &a, cudaStream_t st) {
  if (a.v.D != 128) return cudaErrorInvalidValue;
  switch (a.v.bits) {
    case 8: return launch_gqa_decode_t<8, 128, kKaxSym, 128>(a, st);
    case 4: return launch_gqa_decode_t<4, 128, kKaxSym, 128>(a, st);
    case 2: return launch_gqa_decode_t<2, 128, kKaxSym, 128>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

int gqa_ctas_sym(int bits) {
  switch (bits) {
    case 8: return gqa_ctas_per_sm_t<8, 128, kKaxSym, 128>();
    case 4: return gqa_ctas_per_sm_t<4, 128, kKaxSym, 128>();
    case 2: return gqa_ctas_per_sm_t<2, 128, kKaxSym, 128>();
    default: return 1;
  }
}

int gqa_tile_sym(int bits) {
  switch (bits) {
    case 8: return gqa_tile_t<8, 128, kKaxSym, 128>();
    case 4: return gqa_tile_t<4, 128, kKaxSym, 128>();
    case 2: return gqa_tile_t<2, 128, kKaxSym, 128>();
    default: return kTile;
  }
}

}  // namespace kvk
