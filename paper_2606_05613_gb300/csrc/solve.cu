// Solve pass: one warp per bucket.  The warp reduces the bucket's per-chunk
// Gram partials in a fixed order (lane p owns entry p of the triangle and adds
// the chunks in ascending order, in fp64) into G in shared memory, then solves
// the bucket's rule (solver.cuh) and writes beta and the bucket's status.
#include "solver.cuh"

namespace bkmoo {
namespace {

using namespace solver;

__global__ void __launch_bounds__(32 * kSolveWarpsPerBlock)
    solve_kernel(const PlanView v, const SolveParams p, float* out_weights,
                 int32_t* out_status) {
  __shared__ double Gs[kSolveWarpsPerBlock][kMaxK * kMaxK];
  __shared__ double Bs[kSolveWarpsPerBlock][kMaxK];
  __shared__ float Fs[kSolveWarpsPerBlock][kMaxK * kMaxK];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int64_t b = v.b_lo + (int64_t)blockIdx.x * kSolveWarpsPerBlock + wi;
  if (b >= v.b_hi) return;
  const int K = v.K;
  if (!header_ok(v)) {
    if (lane == 0 && out_status) out_status[b] = BKMOO_ERR_WORKSPACE;
    return;
  }
  double* G = Gs[wi];
  double* beta = Bs[wi];
  reduce_bucket(v, b, G, lane);
  const int st = solve_bucket_warp<0>(K, G, Fs[wi], p, b, beta, lane);
  for (int k = lane; k < K; k += 32) {
    const float f = (float)beta[k];
    v.beta[b * K + k] = f;
    if (out_weights) out_weights[b * K + k] = f;
  }
  if (lane == 0 && out_status) out_status[b] = st;
}

__global__ void __launch_bounds__(32 * kSolveWarpsPerBlock)
    gram_finalize_kernel(const PlanView v, double* out_gram) {
  __shared__ double Gs[kSolveWarpsPerBlock][kMaxK * kMaxK];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int64_t b = (int64_t)blockIdx.x * kSolveWarpsPerBlock + wi;
  if (b >= v.n_buckets) return;
  if (!header_ok(v)) return;
  const int K = v.K;
  double* G = Gs[wi];
  reduce_bucket(v, b, G, lane);
  for (int i = lane; i < K * K; i += 32) out_gram[b * K * K + i] = G[i];
}

}  // namespace

cudaError_t launch_solve(const PlanView& v, const SolveParams& p, float* out_weights,
                         int32_t* out_status, cudaStream_t s) {
  if (v.b_hi <= v.b_lo) return cudaSuccess;
  const int64_t grid = (v.b_hi - v.b_lo + kSolveWarpsPerBlock - 1) / kSolveWarpsPerBlock;
  solve_kernel<<<(unsigned)grid, 32 * kSolveWarpsPerBlock, 0, s>>>(v, p, out_weights, out_status);
  return cudaGetLastError();
}

cudaError_t launch_gram_finalize(const PlanView& v, double* out_gram, cudaStream_t s) {
  if (v.n_buckets == 0) return cudaSuccess;
  const int64_t grid = (v.n_buckets + kSolveWarpsPerBlock - 1) / kSolveWarpsPerBlock;
  gram_finalize_kernel<<<(unsigned)grid, 32 * kSolveWarpsPerBlock, 0, s>>>(v, out_gram);
  return cudaGetLastError();
}

}  // namespace bkmoo
