// merge.cu -- split-K merge of decode partials.
//
// Partial rows hold [acc (dim) | m | l] with acc = sum_t 2^(x_t - m) v_t and
// l = sum_t 2^(x_t - m) over one split's positions.  The merged row is
//   out = sum_s 2^(m_s - M) acc_s / sum_s 2^(m_s - M) l_s,   M = max_s m_s,
// the log-sum-exp identity that makes softmax attention decomposable over a
// partition of the context.
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace kvk {
namespace {

__global__ void __launch_bounds__(128)
    splitk_merge_kernel(const float *__restrict__ P, int S, int n_rows, int dim,
                        float *__restrict__ out) {
  const int row = blockIdx.x;
  const size_t RS = (size_t)dim + 2;
  __shared__ float w_s[256];
  __shared__ float L_s;
  if (threadIdx.x < 32) {
    float M = -INFINITY;
    for (int s = threadIdx.x; s < S; s += 32) M = fmaxf(M, P[((size_t)s * n_rows + row) * RS + dim]);
    for (int off = 16; off; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float L = 0.f;
    for (int s = threadIdx.x; s < S; s += 32) {
      const float *pr = P + ((size_t)s * n_rows + row) * RS;
      const float ms = pr[dim];
      const float w = (ms == -INFINITY || M == -INFINITY) ? 0.f : exp2f(ms - M);
      w_s[s] = w;
      L += w * pr[dim + 1];
    }
    for (int off = 16; off; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
    if (threadIdx.x == 0) L_s = L;
  }
  __syncthreads();
  const float L = L_s;
  for (int ch = threadIdx.x; ch < dim; ch += blockDim.x) {
    float A = 0.f;
    for (int s = 0; s < S; ++s) {
      const float w = w_s[s];
      if (w != 0.f) A += w * P[((size_t)s * n_rows + row) * RS + ch];
    }
    out[(size_t)row * dim + ch] = (L > 0.f) ? A / L : 0.f;
  }
}

__global__ void rewind_kernel(const RewindArgs a) {
  for (int i = threadIdx.x; i < a.n_anchors * a.B; i += blockDim.x) {
    int32_t *l = a.lens[i / a.B] + (i % a.B);
    *l = max(0, *l - a.n);
  }
}

}  // namespace

cudaError_t launch_rewind(const RewindArgs &a, cudaStream_t st) {
  rewind_kernel<<<1, 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_splitk_merge(const float *partials, int n_splits, int n_rows, int dim,
                                float *out, cudaStream_t st) {
  if (n_splits > 256) return cudaErrorInvalidValue;
  splitk_merge_kernel<<<n_rows, 128, 0, st>>>(partials, n_splits, n_rows, dim, out);
  return cudaGetLastError();
}

}  // namespace kvk
