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

// P is written by the decode this launch overlaps (programmatic dependent
// launch), so it is read with coherent loads after the grid-dependency wait,
// not through the read-only path (no __restrict__).
// One thread per output element: every load of the row's partials (the S
// maxima, sums and this element's accumulators) is issued before any is
// used, so the merge costs one memory round trip.  Rows per CTA: 128 / dim
// (dim <= 128), else one row with a channel loop.
template <int SB>
__global__ void __launch_bounds__(128)
    splitk_merge_kernel(const float *P, int S, int n_rows, int dim,
                        float *__restrict__ out) {
  pdl_wait();
  pdl_trigger();
  const int width = dim >= 128 ? 128 : dim;  // threads per row
  const int rpc = 128 / width, r_in = (int)threadIdx.x / width;
  const int row = blockIdx.x * rpc + r_in;
  if (r_in >= rpc || row >= n_rows) return;
  const int ch0 = (int)threadIdx.x % width;
  const size_t RS = (size_t)dim + 2;
  const size_t SS = (size_t)n_rows * RS;  // split stride
  const float *pr = P + (size_t)row * RS;
  float m[SB], l[SB];
#pragma unroll
  for (int s = 0; s < SB; ++s) {
    m[s] = s < S ? pr[s * SS + dim] : -INFINITY;
    l[s] = s < S ? pr[s * SS + dim + 1] : 0.f;
  }
  for (int ch = ch0; ch < dim; ch += 128) {
    float x[SB];
#pragma unroll
    for (int s = 0; s < SB; ++s) x[s] = s < S ? pr[s * SS + ch] : 0.f;
    float M = -INFINITY;
#pragma unroll
    for (int s = 0; s < SB; ++s) M = fmaxf(M, m[s]);
    float L = 0.f, A = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int s = 0; s < SB; ++s) {
        const float w = m[s] == -INFINITY ? 0.f : exp2f(m[s] - M);
        L = fmaf(w, l[s], L);
        A = fmaf(w, x[s], A);
      }
    }
    out[(size_t)row * dim + ch] = (L > 0.f) ? A / L : 0.f;
  }
}

// more than 16 splits: the same, with the split loop not unrolled
__global__ void __launch_bounds__(128)
    splitk_merge_kernel_n(const float *P, int S, int n_rows, int dim,
                          float *__restrict__ out) {
  pdl_wait();
  pdl_trigger();
  const int width = dim >= 128 ? 128 : dim;  // threads per row
  const int rpc = 128 / width, r_in = (int)threadIdx.x / width;
  const int row = blockIdx.x * rpc + r_in;
  if (r_in >= rpc || row >= n_rows) return;
  const int ch0 = (int)threadIdx.x % width;
  const size_t RS = (size_t)dim + 2;
  const size_t SS = (size_t)n_rows * RS;
  const float *pr = P + (size_t)row * RS;
  float M = -INFINITY;
  for (int s = 0; s < S; ++s) M = fmaxf(M, pr[s * SS + dim]);
  for (int ch = ch0; ch < dim; ch += 128) {
    float L = 0.f, A = 0.f;
    if (M != -INFINITY) {
      for (int s = 0; s < S; ++s) {
        const float ms = pr[s * SS + dim];
        const float w = ms == -INFINITY ? 0.f : exp2f(ms - M);
        L = fmaf(w, pr[s * SS + dim + 1], L);
        A = fmaf(w, pr[s * SS + ch], A);
      }
    }
    out[(size_t)row * dim + ch] = (L > 0.f) ? A / L : 0.f;
  }
}

__global__ void rewind_kernel(const RewindArgs a) {
  pdl_wait();
  pdl_trigger();
  for (int i = threadIdx.x; i < a.n_anchors * a.B; i += blockDim.x) {
    int32_t *l = a.lens[i / a.B] + (i % a.B);
    *l = max(0, *l - a.n);
  }
}

}  // namespace

cudaError_t launch_rewind(const RewindArgs &a, cudaStream_t st) {
  return launch_pdl(rewind_kernel, dim3(1), dim3(256), 0, st, a);
}

cudaError_t launch_splitk_merge(const float *partials, int n_splits, int n_rows, int dim,
                                float *out, cudaStream_t st) {
  if (n_splits < 1 || n_rows < 0 || dim < 1) return cudaErrorInvalidValue;
  if (n_rows == 0) return cudaSuccess;
  const int rpc = dim >= 128 ? 1 : 128 / dim;
  const int grid = (n_rows + rpc - 1) / rpc;
  if (n_splits <= 8)
    return launch_pdl(splitk_merge_kernel<8>, grid, dim3(128), 0, st, partials, n_splits, n_rows, dim, out);
  else if (n_splits <= 16)
    return launch_pdl(splitk_merge_kernel<16>, grid, dim3(128), 0, st, partials, n_splits, n_rows, dim, out);
  else
    return launch_pdl(splitk_merge_kernel_n, grid, dim3(128), 0, st, partials, n_splits, n_rows, dim, out);
}

}  // namespace kvk
