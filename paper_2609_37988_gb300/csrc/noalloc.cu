// noalloc.cu -- decode attention that allocates nothing and needs no
// caller-provided scratch.
//
// Some callers cannot hand the library device memory for scratch: their
// device memory is owned by another allocator or planned up front to a fixed
// budget, and they cannot (or may not) call cudaMalloc to size a workspace
// for the largest split count they will use.  kvk_decode_attention_noalloc
// serves them: the split-K partials of the GQA decode live in one fixed
// array inside this library, so a call needs only the cache, the query and
// the output.
//
// The array is file-scope device memory: every GPU that loads the library
// holds it until the process exits, and every call on a device shares it.
// Its host-side name is only a stand-in for the device symbol, so its device
// address is looked up once per device with cudaGetSymbolAddress (with that
// device current) the first time a call runs there.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/kvk.h"

// host side of this library (kvk_host.cu)
kvk_status kvk_internal_cuda_error(cudaError_t e, const char *what);
kvk_status kvk_internal_check_current_device(const kvk_cache *c);
kvk_status kvk_internal_decode_with_partials(kvk_cache *c, int32_t layer, const void *q,
                                             int32_t q_dtype, float scale, float *out,
                                             int32_t n_splits, float *partial,
                                             size_t partial_floats, kvk_stream stream);

namespace {

// 16 MiB of fp32 split-K partials: e.g. 8 splits x 32 sequences x 40 query
// heads x (128 + 2) floats = 5.3 MiB fits; larger requests are rejected.
constexpr size_t kScratchFloats = size_t(4) << 20;
static __device__ __align__(256) float g_scratch[kScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float *g_dev_ptr[kMaxDevices] = {};

// Device address of g_scratch on the current device (looked up once).
cudaError_t scratch_for_current_device(float **ptr) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_dev_ptr[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return e;
    g_dev_ptr[dev] = static_cast<float *>(p);
  }
  *ptr = g_dev_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" kvk_status kvk_decode_attention_noalloc(kvk_cache *cache, int32_t layer,
                                                   const void *q, int32_t q_dtype,
                                                   float softmax_scale, float *out,
                                                   int32_t n_splits, kvk_stream stream) {
  // The buffer looked up below belongs to the current device; the cache's
  // arenas to the device it was created on.  Refuse a mismatch up front.
  const kvk_status ds = kvk_internal_check_current_device(cache);
  if (ds != KVK_OK) return ds;
  float *scratch = nullptr;
  const cudaError_t e = scratch_for_current_device(&scratch);
  if (e != cudaSuccess) return kvk_internal_cuda_error(e, "looking up the fixed scratch buffer");
  // Each split writes every partial row it owns (empty splits write m = -inf,
  // l = 0) before the merge reads it, so the shared buffer needs no clearing.
  return kvk_internal_decode_with_partials(cache, layer, q, q_dtype, softmax_scale, out, n_splits,
                                           scratch, kScratchFloats, stream);
}
