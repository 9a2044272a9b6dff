// Combination pass with a per-thread prefetch into shared memory: the
// arithmetic, element order and stores of combine_kernel (combine_impl.cuh),
// with each thread copying its next positions' K vectors into its own
// shared-memory slots by cp.async, S stages ahead, instead of loading them
// into registers just before use.  Each element is still read and written by
// one thread only, and read before it is written, so in-place use (out ==
// one of the gradients) stays race-free.
#pragma once

#include "combine_impl.cuh"
#include "gram_prefetch.cuh"

namespace bkmoo {

#ifndef BKMOO_COMBINE_PREFETCH_STAGES
#define BKMOO_COMBINE_PREFETCH_STAGES 4
#endif
constexpr int kCombinePrefetchStages = BKMOO_COMBINE_PREFETCH_STAGES;

// Stages per thread (measured on GB300): 2 for K <= 4 (Qwen3-8B K=4 bf16
// combination 11.96 -> 11.83 ms against 4 stages; sweep K=2 1.80 -> 1.77 ms),
// 4 for K = 5..8 (Llama-3.2-1B K=8: 3.11 ms, 3.20 with 2 stages), 3 above
// (K = 16: 192 KB of slots, one CTA per SM with 128 KB of copies in flight).
__host__ __device__ constexpr int combine_prefetch_stages(int K) {
  return K <= 4 ? 2 : K <= 8 ? kCombinePrefetchStages : 3;
}
__host__ __device__ constexpr int combine_prefetch_smem_bytes(int K) {
  return combine_prefetch_stages(K) * K * kThreads * 16;
}

template <int K, int DTI, int DTO>
__global__ void __launch_bounds__(kThreads)
    combine_prefetch_kernel(const GradPtrs g, const PlanView v, void* out) {
  constexpr int EPV = elems_per_vec(DTI);
  constexpr int IB = 16 / EPV;
  constexpr int S = combine_prefetch_stages(K);
  extern __shared__ __align__(16) unsigned char cpf_smem[];
  uint4* slots = reinterpret_cast<uint4*>(cpf_smem);
  auto slot = [&](int s, int k) -> uint4* { return slots + ((s * K + k) * kThreads + threadIdx.x); };
  if (!header_ok(v)) return;    // the Gram pass already recorded the error

  VecCursor<EPV> pc;
  pc.begin(v);
  int issued = 0;
  auto issue = [&]() {
    const int s = issued % S;
    if (pc.more(v)) {
      const int64_t off = (pc.vs + (int64_t)pc.i * EPV) * IB;
#pragma unroll
      for (int k = 0; k < K; ++k) cp_async16(slot(s, k), static_cast<const char*>(g.p[k]) + off);
      pc.next(v);
    }
    cp_async_commit();
    ++issued;
  };
#pragma unroll
  for (int j = 0; j < S - 1; ++j) issue();

  int consumed = 0;
  int64_t b = v.b_lo;
  for (int64_t w = v.c_lo + blockIdx.x; w < v.c_hi; w += gridDim.x) {
    b = find_bucket(v.chunk_prefix, v.n_buckets, w, b);
    float beta[K];
#pragma unroll
    for (int k = 0; k < K; ++k) beta[k] = v.beta[b * K + k];
    const int64_t be = v.offsets[b + 1];
    const int64_t s0 = v.offsets[b] + (w - v.chunk_prefix[b]) * v.chunk_elems;
    const int64_t e = min(s0 + v.chunk_elems, be);
    int64_t vs = (s0 + EPV - 1) / EPV * EPV;
    if (vs > e) vs = e;
    int64_t ve = e / EPV * EPV;
    if (ve < vs) ve = vs;
    const int nv = (int)((ve - vs) / EPV);

    for (int i = threadIdx.x; i < nv; i += kThreads) {
      issue();
      cp_async_wait<S - 1>();
      const int s = consumed % S;
      const int64_t el = vs + (int64_t)i * EPV;
      uint4 r[K];
#pragma unroll
      for (int k = 0; k < K; ++k) r[k] = *slot(s, k);
      float y[EPV];
#pragma unroll
      for (int q = 0; q < EPV; ++q) {
        float t = 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) t = fmaf(beta[k], vec_elem<DTI>(r[k], q), t);
        y[q] = t;
      }
      store_out<DTO>(out, el, y, EPV);
      ++consumed;
    }
    const int nh = (int)(vs - s0), nt = (int)(e - ve);
    if ((int)threadIdx.x < nh + nt) {
      const int64_t idx = (int)threadIdx.x < nh ? s0 + threadIdx.x : ve + (threadIdx.x - nh);
      float t = 0.0f;
#pragma unroll
      for (int k = 0; k < K; ++k) t = fmaf(beta[k], load_scalar<DTI>(g.p[k], idx), t);
      store_scalar<DTO>(out, idx, t);
    }
  }
  cp_async_wait<0>();
}

}  // namespace bkmoo
