// Combination pass: d = sum_k beta_{b,k} g_k over every bucket b.
//
// Every rule's resolved update is a linear combination of the bucket's K
// gradients (Algorithm 1: d_(k) = sum_t alpha_t g_(k),t for MGDA, the CAGrad
// maximiser g0 + c||g0|| g_w / ||g_w||, and the sum of projected gradients
// for PCGrad), and the global update is the concatenation of the buckets'
// directions (Section 3.2).  The coefficients beta were written by the solve
// kernel into the workspace.
//
// Same chunking as the Gram pass.  Each thread reads one 16-byte vector of
// every gradient, forms sum_k beta_k x_k in fp32 (k ascending), rounds to the
// output type (bf16: round to nearest even) and writes it.  Reads use the
// coherent evict-first path because out may be one of the inputs (in-place):
// each element is read by the thread that later overwrites it, and by no one
// else, so in-place use is race-free.
#pragma once

#include <cuda_bf16.h>

#include "common.cuh"

namespace bkmoo {

template <int DTO>
__device__ __forceinline__ void store_out(void* out, int64_t i, const float* y, int n) {
  if (DTO == BKMOO_F32) {
    float* o = static_cast<float*>(out) + i;
    if (n == 4) {
      st16_cs(o, make_uint4(__float_as_uint(y[0]), __float_as_uint(y[1]), __float_as_uint(y[2]),
                            __float_as_uint(y[3])));
    } else {  // n == 8
      st16_cs(o, make_uint4(__float_as_uint(y[0]), __float_as_uint(y[1]), __float_as_uint(y[2]),
                            __float_as_uint(y[3])));
      st16_cs(o + 4, make_uint4(__float_as_uint(y[4]), __float_as_uint(y[5]),
                                __float_as_uint(y[6]), __float_as_uint(y[7])));
    }
  } else {
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(out) + i;
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (2 * q < n) {
        __nv_bfloat162 h = __floats2bfloat162_rn(y[2 * q], y[2 * q + 1]);
        w[q] = *reinterpret_cast<uint32_t*>(&h);
      }
    }
    if (n == 8) st16_cs(o, make_uint4(w[0], w[1], w[2], w[3]));
    else st8_cs(o, make_uint2(w[0], w[1]));  // n == 4
  }
}

template <int DTO>
__device__ __forceinline__ void store_scalar(void* out, int64_t i, float y) {
  if (DTO == BKMOO_F32) static_cast<float*>(out)[i] = y;
  else static_cast<__nv_bfloat16*>(out)[i] = __float2bfloat16_rn(y);
}

template <int K, int DTI, int DTO>
__global__ void __launch_bounds__(kThreads) combine_kernel(const GradPtrs g, const PlanView v,
                                                            void* out) {
  constexpr int EPV = elems_per_vec(DTI);
  constexpr int IB = 16 / EPV;  // input bytes per element
  if (!header_ok(v)) return;    // the Gram pass already recorded the error

  int64_t b = v.b_lo;
  for (int64_t w = v.c_lo + blockIdx.x; w < v.c_hi; w += gridDim.x) {
    b = find_bucket(v.chunk_prefix, v.n_buckets, w, b);
    float beta[K];
#pragma unroll
    for (int k = 0; k < K; ++k) beta[k] = v.beta[b * K + k];
    const int64_t be = v.offsets[b + 1];
    const int64_t s = v.offsets[b] + (w - v.chunk_prefix[b]) * v.chunk_elems;
    const int64_t e = min(s + v.chunk_elems, be);
    int64_t vs = (s + EPV - 1) / EPV * EPV;
    if (vs > e) vs = e;
    int64_t ve = e / EPV * EPV;
    if (ve < vs) ve = vs;
    const int nv = (int)((ve - vs) / EPV);

    int i = threadIdx.x;
    // K >= 9: two vectors per thread in flight (measured 8 % faster at K = 16;
    // no change at K = 4 and 8, where the occupancy already hides the latency)
    if (K >= 9) {
      for (; i + kThreads < nv; i += 2 * kThreads) {
        const int64_t el0 = vs + (int64_t)i * EPV, el1 = el0 + (int64_t)kThreads * EPV;
        uint4 r0[K], r1[K];
#pragma unroll
        for (int k = 0; k < K; ++k) {
          r0[k] = ld16_cs(static_cast<const char*>(g.p[k]) + el0 * IB);
          r1[k] = ld16_cs(static_cast<const char*>(g.p[k]) + el1 * IB);
        }
        float y0[EPV], y1[EPV];
#pragma unroll
        for (int q = 0; q < EPV; ++q) {
          float t0 = 0.0f, t1 = 0.0f;
#pragma unroll
          for (int k = 0; k < K; ++k) {
            t0 = fmaf(beta[k], vec_elem<DTI>(r0[k], q), t0);
            t1 = fmaf(beta[k], vec_elem<DTI>(r1[k], q), t1);
          }
          y0[q] = t0;
          y1[q] = t1;
        }
        store_out<DTO>(out, el0, y0, EPV);
        store_out<DTO>(out, el1, y1, EPV);
      }
    }
    for (; i < nv; i += kThreads) {
      const int64_t el = vs + (int64_t)i * EPV;
      uint4 r[K];
#pragma unroll
      for (int k = 0; k < K; ++k) r[k] = ld16_cs(static_cast<const char*>(g.p[k]) + el * IB);
      float y[EPV];
#pragma unroll
      for (int q = 0; q < EPV; ++q) {
        float t = 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) t = fmaf(beta[k], vec_elem<DTI>(r[k], q), t);
        y[q] = t;
      }
      store_out<DTO>(out, el, y, EPV);
    }
    const int nh = (int)(vs - s), nt = (int)(e - ve);
    if ((int)threadIdx.x < nh + nt) {
      const int64_t idx = (int)threadIdx.x < nh ? s + threadIdx.x : ve + (threadIdx.x - nh);
      float t = 0.0f;
#pragma unroll
      for (int k = 0; k < K; ++k) t = fmaf(beta[k], load_scalar<DTI>(g.p[k], idx), t);
      store_scalar<DTO>(out, idx, t);
    }
  }
}

#define BKMOO_COMBINE_ROW(K, DTI)                                        \
  {(const void*)combine_kernel<K, DTI, BKMOO_F32>,                       \
   (const void*)combine_kernel<K, DTI, BKMOO_BF16>}

#define BKMOO_COMBINE_TABLE(DTI)                                                            \
  static const void* const kCombineTable[kMaxK][2] = {                                      \
      BKMOO_COMBINE_ROW(1, DTI),  BKMOO_COMBINE_ROW(2, DTI),  BKMOO_COMBINE_ROW(3, DTI),    \
      BKMOO_COMBINE_ROW(4, DTI),  BKMOO_COMBINE_ROW(5, DTI),  BKMOO_COMBINE_ROW(6, DTI),    \
      BKMOO_COMBINE_ROW(7, DTI),  BKMOO_COMBINE_ROW(8, DTI),  BKMOO_COMBINE_ROW(9, DTI),    \
      BKMOO_COMBINE_ROW(10, DTI), BKMOO_COMBINE_ROW(11, DTI), BKMOO_COMBINE_ROW(12, DTI),   \
      BKMOO_COMBINE_ROW(13, DTI), BKMOO_COMBINE_ROW(14, DTI), BKMOO_COMBINE_ROW(15, DTI),   \
      BKMOO_COMBINE_ROW(16, DTI)}

}  // namespace bkmoo
