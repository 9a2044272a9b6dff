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

// Block (x = group j, y-stride over buckets b): for a bucket of more than
// kGroupMinChunks chunks, thread p < K(K+1)/2 sums entry p over the chunks
// [c0 + 512 j, c0 + 512 (j+1)) of the bucket (eight interleaved fp64 sums,
// fixed tree) and writes the result into the group's first row.  Each
// (row, entry) is read and written by one thread only.
__global__ void __launch_bounds__(256) group_reduce_kernel(const PlanView v) {
  if (!header_ok(v)) return;
  const int P = tri(v.K);
  const int p = threadIdx.x;
  if (p >= P) return;
  for (int64_t b = v.b_lo + blockIdx.y; b < v.b_hi; b += gridDim.y) {
    const int64_t cb0 = v.chunk_prefix[b], cb1 = v.chunk_prefix[b + 1];
    if (cb1 - cb0 <= kGroupMinChunks) continue;
    const int64_t c0 = cb0 + (int64_t)blockIdx.x * kGroupChunks;
    if (c0 >= cb1) continue;
    const int64_t c1 = min(c0 + kGroupChunks, cb1);
    double t[8] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
    const double* src = v.partials + c0 * P + p;
    int64_t c = c0;
    for (; c + 8 <= c1; c += 8, src += 8 * P) {
#pragma unroll
      for (int j = 0; j < 8; ++j) t[j] += src[j * P];
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (c + j < c1) t[j] += src[j * P];
    v.partials[c0 * P + p] = ((t[0] + t[1]) + (t[2] + t[3])) + ((t[4] + t[5]) + (t[6] + t[7]));
  }
}

// Element i of the fp64 division / square-root helpers of the fast solvers
// (op 0: a[i] / b[i] by div_nr, op 1: sqrt(a[i]) by sqrt_nr); grid-stride.
__global__ void selftest_fp64_kernel(int op, const double* a, const double* b, double* out,
                                     int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = op == 0 ? div_nr(a[i], b[i]) : sqrt_nr(a[i]);
}

}  // namespace

cudaError_t launch_selftest_fp64(int op, const double* a, const double* b, double* out, int64_t n,
                                 cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  int64_t grid = (n + 255) / 256;
  if (grid > 4096) grid = 4096;
  selftest_fp64_kernel<<<(unsigned)grid, 256, 0, s>>>(op, a, b, out, n);
  return cudaGetLastError();
}

cudaError_t launch_group_reduce(const PlanView& v, cudaStream_t s) {
  if (v.max_chunks <= kGroupMinChunks || v.b_hi <= v.b_lo) return cudaSuccess;
  const int64_t gx = (v.max_chunks + kGroupChunks - 1) / kGroupChunks;
  int64_t gy = v.b_hi - v.b_lo;
  if (gy > 65535) gy = 65535;
  group_reduce_kernel<<<dim3((unsigned)gx, (unsigned)gy), 256, 0, s>>>(v);
  return cudaGetLastError();
}

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
