// Gradient-conflict statistics of Figure 1 from the per-bucket Gram
// matrices: pairwise cosines cos_ij = G_ij / sqrt(G_ii G_jj) (a pair
// conflicts when its cosine is negative, Definition A.4 / Eq. 2), their mean,
// population standard deviation and minimum over the K(K-1)/2 pairs, and a
// flag for "at least one pair conflicts" (the per-step event whose frequency
// Figure 1 plots per layer).  A pair involving a zero-norm gradient has
// cosine 0 and does not conflict.  One thread per bucket.
#include <cuda_runtime.h>

#include "common.cuh"

namespace bkmoo {
namespace {

__global__ void conflicts_kernel(const double* gram, int K, int64_t B, float* out_cos,
                                 float* out_stats, int32_t* out_conflict) {
  const int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const double* G = gram + b * K * K;
  double r[kMaxK];
  for (int i = 0; i < K; ++i) {
    const double d = G[i * K + i];
    r[i] = d > 0.0 ? 1.0 / sqrt(d) : 0.0;
  }
  double sum = 0.0, sum2 = 0.0, mn = 1.0;
  int conflict = 0;
  for (int i = 0; i < K; ++i) {
    for (int j = 0; j < K; ++j) {
      double c = (i == j) ? (r[i] > 0.0 ? 1.0 : 0.0) : G[i * K + j] * r[i] * r[j];
      if (i < j) {
        sum += c;
        sum2 += c * c;
        mn = c < mn ? c : mn;
        if (c < 0.0) conflict = 1;
      }
      if (out_cos) out_cos[b * K * K + i * K + j] = (float)c;
    }
  }
  const double np = 0.5 * K * (K - 1);
  const double mean = sum / np;
  const double var = sum2 / np - mean * mean;
  if (out_stats) {
    out_stats[b * 3 + 0] = (float)mean;
    out_stats[b * 3 + 1] = (float)sqrt(var > 0.0 ? var : 0.0);
    out_stats[b * 3 + 2] = (float)mn;
  }
  if (out_conflict) out_conflict[b] = conflict;
}

}  // namespace
}  // namespace bkmoo

extern "C" int bkmoo_conflicts(const double* gram, int32_t K, int64_t n_buckets, float* out_cos,
                               float* out_stats, int32_t* out_conflict, void* stream) {
  if (K < 2 || K > bkmoo::kMaxK || n_buckets < 0 || (n_buckets > 0 && !gram))
    return BKMOO_ERR_INVALID;
  if (n_buckets == 0) return BKMOO_OK;
  const int threads = 128;
  const int64_t grid = (n_buckets + threads - 1) / threads;
  bkmoo::conflicts_kernel<<<(unsigned)grid, threads, 0, static_cast<cudaStream_t>(stream)>>>(
      gram, K, n_buckets, out_cos, out_stats, out_conflict);
  return cudaGetLastError() == cudaSuccess ? BKMOO_OK : BKMOO_ERR_CUDA;
}
