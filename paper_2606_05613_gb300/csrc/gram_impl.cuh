// Gram pass: per-chunk partial Gram matrices of the K gradients.
//
// Every rule of the method depends on a bucket's gradients only through the
// inner products <g_i, g_j> over the bucket (Eq. 3 / Eq. 6 are a quadratic in
// them, Eq. 4's dual and Eq. 5's projections are built from them), so the
// bucket's data is streamed once and reduced to K(K+1)/2 numbers.
//
// Work unit: a chunk of chunk_elems elements of one bucket (the last chunk of
// a bucket may be short).  A CTA of 256 threads loads one 16-byte vector of
// each of the K gradients per thread per step (coalesced, read-only path,
// no L1 allocation), widens bf16 to fp32 exactly, and accumulates the upper
// triangle of x x^T in fp32 registers: each thread sums at most 16 vectors
// (64 fp32 or 128 bf16 elements) of a chunk.  The CTA then reduces the
// triangle with a fixed warp-shuffle tree (fp32) and a fixed sum over its 8
// warps (fp64), and writes the chunk's partials as fp64.  No atomics: the
// result depends only on the data, never on scheduling.
//
// Vector loads need 16-byte aligned addresses: the gradient bases are 16-byte
// aligned (checked on the host) and the head / tail elements of a chunk that
// fall before / after the first / last aligned vector take a scalar path.
#pragma once

#include "common.cuh"

namespace bkmoo {

// Whether a row's products are issued as paired fp32 FMAs (__ffma2_rn: the
// entries (i, j) and (i, j+1) in one instruction, each rounded exactly as
// fmaf rounds it, so the sums are bit-identical either way).  Measured on
// GB300: bf16 K=8 Gram 6 % faster, fp32 K=16 5 % faster; fp32 K=8 and K=12
// slower (the pair (x_j, x_j+1) comes from two different loads and costs
// moves, where bf16 values are produced by the widening into fresh pairs).
template <int K, int DT>
__host__ __device__ constexpr bool pair_fma() {
  return (DT == BKMOO_BF16 && K >= 2 && K <= 8) || (DT == BKMOO_F32 && K == 16);
}

template <int K, int DT>
__device__ __forceinline__ void triangle_update(float (&acc)[tri(K)], const float (&x)[K]) {
  int p = 0;
#pragma unroll
  for (int i = 0; i < K; ++i) {
    if (pair_fma<K, DT>()) {
      int j = i;
      if (i & 1) {  // pairs start at even columns: (x_j, x_j+1) is one register pair
        acc[p] = fmaf(x[i], x[i], acc[p]);
        ++p;
        ++j;
      }
#pragma unroll
      for (; j + 1 < K; j += 2) {
        const float2 t = __ffma2_rn(make_float2(x[i], x[i]), make_float2(x[j], x[j + 1]),
                                    make_float2(acc[p], acc[p + 1]));
        acc[p] = t.x;
        acc[p + 1] = t.y;
        p += 2;
      }
      if (j < K) {
        acc[p] = fmaf(x[i], x[j], acc[p]);
        ++p;
      }
    } else {
#pragma unroll
      for (int j = i; j < K; ++j) {
        acc[p] = fmaf(x[i], x[j], acc[p]);
        ++p;
      }
    }
  }
}

template <int K, int DT>
__device__ __forceinline__ void gram_accumulate(float (&acc)[tri(K)], const uint4 (&r)[K]) {
  constexpr int EPV = elems_per_vec(DT);
#pragma unroll
  for (int e = 0; e < EPV; ++e) {
    float x[K];
#pragma unroll
    for (int k = 0; k < K; ++k) x[k] = vec_elem<DT>(r[k], e);
    triangle_update<K, DT>(acc, x);
  }
}

template <int K, int DT>
__device__ __forceinline__ void gram_accumulate_scalar(float (&acc)[tri(K)], const GradPtrs& g,
                                                       int64_t i) {
  float x[K];
#pragma unroll
  for (int k = 0; k < K; ++k) x[k] = load_scalar<DT>(g.p[k], i);
  int p = 0;
#pragma unroll
  for (int a = 0; a < K; ++a) {
#pragma unroll
    for (int b = a; b < K; ++b) {
      acc[p] = fmaf(x[a], x[b], acc[p]);
      ++p;
    }
  }
}

// Fixed-order CTA reduction of the per-thread triangles; writes P doubles.
template <int P>
__device__ __forceinline__ void cta_reduce_store(float (&acc)[P], float (*red)[P], double* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int p = 0; p < P; ++p) {
    float v = acc[p];
    v += __shfl_down_sync(0xffffffffu, v, 16);
    v += __shfl_down_sync(0xffffffffu, v, 8);
    v += __shfl_down_sync(0xffffffffu, v, 4);
    v += __shfl_down_sync(0xffffffffu, v, 2);
    v += __shfl_down_sync(0xffffffffu, v, 1);
    if (lane == 0) red[warp][p] = v;
  }
  __syncthreads();
  for (int p = threadIdx.x; p < P; p += kThreads) {
    double s = 0.0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += (double)red[w][p];
    out[p] = s;
  }
  __syncthreads();
}

template <int K, int DT>
__global__ void __launch_bounds__(kThreads) gram_partials_kernel(const GradPtrs g,
                                                                  const PlanView v) {
  constexpr int P = tri(K);
  constexpr int EPV = elems_per_vec(DT);
  constexpr int UNROLL = (K <= 8) ? 2 : 1;
  __shared__ float red[kWarps][P];

  if (!header_ok(v)) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
    return;
  }
  int64_t b = v.b_lo;
  for (int64_t w = v.c_lo + blockIdx.x; w < v.c_hi; w += gridDim.x) {
    b = find_bucket(v.chunk_prefix, v.n_buckets, w, b);
    const int64_t be = v.offsets[b + 1];
    const int64_t s = v.offsets[b] + (w - v.chunk_prefix[b]) * v.chunk_elems;
    const int64_t e = min(s + v.chunk_elems, be);
    int64_t vs = (s + EPV - 1) / EPV * EPV;
    if (vs > e) vs = e;
    int64_t ve = e / EPV * EPV;
    if (ve < vs) ve = vs;
    const int nv = (int)((ve - vs) / EPV);

    float acc[P];
#pragma unroll
    for (int p = 0; p < P; ++p) acc[p] = 0.0f;

    int i = threadIdx.x;
    if (UNROLL == 2) {
      for (; i + kThreads < nv; i += 2 * kThreads) {
        uint4 r0[K], r1[K];
#pragma unroll
        for (int k = 0; k < K; ++k) {
          const char* base = static_cast<const char*>(g.p[k]) + (vs + (int64_t)i * EPV) * (16 / EPV);
          r0[k] = ld16_nc(base);
          r1[k] = ld16_nc(base + (size_t)kThreads * 16);
        }
        gram_accumulate<K, DT>(acc, r0);
        gram_accumulate<K, DT>(acc, r1);
      }
    }
    for (; i < nv; i += kThreads) {
      uint4 r0[K];
#pragma unroll
      for (int k = 0; k < K; ++k)
        r0[k] = ld16_nc(static_cast<const char*>(g.p[k]) + (vs + (int64_t)i * EPV) * (16 / EPV));
      gram_accumulate<K, DT>(acc, r0);
    }
    const int nh = (int)(vs - s), nt = (int)(e - ve);
    if ((int)threadIdx.x < nh + nt) {
      const int64_t idx = (int)threadIdx.x < nh ? s + threadIdx.x : ve + (threadIdx.x - nh);
      gram_accumulate_scalar<K, DT>(acc, g, idx);
    }
    cta_reduce_store<P>(acc, red, v.partials + w * P);
  }
}

#define BKMOO_GRAM_TABLE(DT)                                                              \
  static const void* const kGramTable[kMaxK] = {                                          \
      (const void*)gram_partials_kernel<1, DT>,  (const void*)gram_partials_kernel<2, DT>,  \
      (const void*)gram_partials_kernel<3, DT>,  (const void*)gram_partials_kernel<4, DT>,  \
      (const void*)gram_partials_kernel<5, DT>,  (const void*)gram_partials_kernel<6, DT>,  \
      (const void*)gram_partials_kernel<7, DT>,  (const void*)gram_partials_kernel<8, DT>,  \
      (const void*)gram_partials_kernel<9, DT>,  (const void*)gram_partials_kernel<10, DT>, \
      (const void*)gram_partials_kernel<11, DT>, (const void*)gram_partials_kernel<12, DT>, \
      (const void*)gram_partials_kernel<13, DT>, (const void*)gram_partials_kernel<14, DT>, \
      (const void*)gram_partials_kernel<15, DT>, (const void*)gram_partials_kernel<16, DT>}

}  // namespace bkmoo
