// Fused resolve: one persistent, co-resident grid resolves bucket after
// bucket (Algorithm 1's inner loop over buckets) so that a bucket's
// gradients are read from HBM once, by the Gram pass, and read again by the
// combination while they are still in L2.
//
// Roles.  CTAs 0 .. n_stream-1 stream; CTA n_stream solves.
//  streamer i works on two buckets at once, in small steps (2 vectors per
//  thread per step), so that HBM reads of the next bucket overlap the solve
//  and the L2-served combination of the previous one:
//    Gram of its slice of bucket gb (slice i of n_stream equal, 16-byte-
//      aligned pieces), loads marked L2 evict_last so that the bucket stays
//      in L2; the slice's triangle (fp32 per thread over at most 16 vectors,
//      fixed warp-shuffle tree, fp64 across warps and sub-slices) goes to the
//      ring of partials, then arrive[gb] += 1 (release).  gb runs at most one
//      bucket ahead of cb.
//    combination of its slice of bucket cb once ready[cb] is seen (acquire),
//      loads marked evict_first (each line is read for the last time),
//      stores evict_first.  It only blocks (bounded) on ready[cb] when no
//      Gram step is left to overlap.
//  solver: for each bucket b, wait until arrive[b] == n_stream (bounded),
//    reduce the n_stream partials in a fixed order (fp64), solve the rule
//    (solver.cuh), write beta_b, out_weights, out_status, then ready[b] = 1
//    (release).
// A streamer writes the partials of bucket b+2 only after it has seen
// ready[b], i.e. after the solver has read bucket b's, so two ring slots of
// partials suffice.  No wait closes a cycle: a streamer blocks on ready[cb]
// only after arriving for cb and cb+1, and the solver waits only for
// arrivals.  Every wait gives up after about a second,
// records BKMOO_ERR_TIMEOUT in the workspace status word and ends the kernel;
// any recorded error makes every other wait end at once.
//
// The grid must be co-resident (cooperative launch).  Results are
// deterministic for a given grid size; the chunking differs from the
// three-pass path, so the two agree to rounding, not bit for bit.
#pragma once

#include <cuda_bf16.h>

#include "combine_impl.cuh"
#include "gram_impl.cuh"
#include "solver.cuh"

namespace bkmoo {

constexpr uint64_t kFusedWaitNs = 1000000000ull;  // deadline of one wait: 1 s

// L2 eviction-priority policies (createpolicy) and 16-byte loads carrying them.
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint4 ld16_policy_nc(const void* p, uint64_t pol) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p), "l"(pol));
  return r;
}
__device__ __forceinline__ uint4 ld16_policy(const void* p, uint64_t pol) {
  uint4 r;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p), "l"(pol));
  return r;
}

__device__ __forceinline__ int ld_acquire(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait until *p >= target: gives up 1 s after it started.  False on
// timeout (recorded as BKMOO_ERR_TIMEOUT) or as soon as any error is
// recorded in the workspace status word.
__device__ __forceinline__ bool fused_wait(const int32_t* p, int target, WsHeader* h) {
  const uint64_t t0 = global_ns();
  for (unsigned it = 0;; ++it) {
    if (ld_acquire(p) >= target) return true;
    if ((it & 31u) == 31u) {
      if (*(volatile int32_t*)&h->status != 0) return false;
      if (global_ns() - t0 > kFusedWaitNs) break;
    }
    __nanosleep(64);
  }
  record_error(h, BKMOO_ERR_TIMEOUT);
  return false;
}

// Slice [lo, hi) of bucket b for streamer i.
template <int EPV>
__device__ __forceinline__ void fused_slice(const PlanView& v, int64_t b, int i, int n,
                                            int64_t* lo, int64_t* hi) {
  const int64_t bo = v.offsets[b], be = v.offsets[b + 1];
  int64_t S = (be - bo + n - 1) / n;
  S = (S + EPV - 1) / EPV * EPV;
  int64_t a = bo + (int64_t)i * S;
  if (a > be) a = be;
  int64_t z = a + S;
  if (z > be) z = be;
  *lo = a;
  *hi = z;
}

template <int K>
__device__ __noinline__ void fused_solver_cta(const FusedView& f, const SolveParams& prm) {
  constexpr int P = tri(K);
  __shared__ double G[K * K];
  __shared__ double part[kThreads];
  __shared__ double beta_sh[K];
  __shared__ int go;
  const PlanView& v = f.v;
  const int n = f.n_stream;
  // thread t sums stripe t / P of entry t % P over the CTAs of that stripe
  constexpr int STRIPES = kThreads / P > 0 ? kThreads / P : 1;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t b = 0; b < v.n_buckets; ++b) {
    if (threadIdx.x == 0) go = fused_wait(f.arrive + b, n, v.hdr) ? 1 : 0;
    __syncthreads();
    if (!go) return;
    const double* ring = f.ring + (size_t)(b & 1) * kFusedMaxCtas * P;
    if ((int)threadIdx.x < STRIPES * P) {
      const int e = threadIdx.x % P, st = threadIdx.x / P;
      const int c0 = (int)((int64_t)n * st / STRIPES), c1 = (int)((int64_t)n * (st + 1) / STRIPES);
      double t = 0.0;
      for (int c = c0; c < c1; ++c) t += __ldcg(ring + (size_t)c * P + e);
      part[threadIdx.x] = t;
    }
    __syncthreads();
    if ((int)threadIdx.x < P) {
      double t = 0.0;
      for (int st = 0; st < STRIPES; ++st) t += part[st * P + threadIdx.x];
      int i = 0, r = threadIdx.x;
      while (r >= K - i) {
        r -= K - i;
        ++i;
      }
      G[i * K + i + r] = t;
      G[(i + r) * K + i] = t;
    }
    __syncthreads();
    if (warp == 0) {
      const int st = solver::solve_bucket_warp(K, G, prm, b, beta_sh, lane);
      if (lane < K) {
        const float fb = (float)beta_sh[lane];
        v.beta[b * K + lane] = fb;
        if (f.out_weights) f.out_weights[b * K + lane] = fb;
        __threadfence();
      }
      if (lane == 0 && f.out_status) f.out_status[b] = st;
      __syncwarp();
      if (lane == 0) {
        __threadfence();
        atomicExch(f.ready + b, 1);
      }
    }
    __syncthreads();
  }
}

// Resident CTAs per SM the register budget is capped for: the streaming
// loops need about 48 (K <= 4) and 128 (K <= 8) registers per thread; the
// solver code shares the kernel and spills instead of lowering occupancy.
template <int K>
struct FusedMinBlocks {
  static constexpr int value = K <= 4 ? 4 : (K <= 8 ? 2 : 1);
};

template <int K, int DT, int DTO>
__global__ void __launch_bounds__(kThreads, FusedMinBlocks<K>::value)
    fused_resolve_kernel(const GradPtrs g, const FusedView f, const SolveParams prm, void* out) {
  constexpr int P = tri(K);
  constexpr int EPV = elems_per_vec(DT);
  constexpr int IB = 16 / EPV;
  constexpr int STEP = 2;                 // vectors per thread per Gram / combine step
  __shared__ float red[kWarps][P];
  __shared__ float beta_sh[K];
  __shared__ int s_go;
  const PlanView& v = f.v;
  if (!header_ok(v)) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
    if ((int)blockIdx.x == f.n_stream && f.out_status)
      for (int64_t b = threadIdx.x; b < v.n_buckets; b += kThreads)
        f.out_status[b] = BKMOO_ERR_WORKSPACE;
    return;
  }
  if ((int)blockIdx.x == f.n_stream) {
    fused_solver_cta<K>(f, prm);
    return;
  }
  const int cta = blockIdx.x, n = f.n_stream;
  const int64_t B = v.n_buckets;
  const uint64_t keep = policy_evict_last(), last_use = policy_evict_first();

  // Gram stepper over bucket gb (this CTA's slice)
  int64_t gb = 0, g_lo = 0, g_vs = 0, g_nv = 0, g_next = 0;
  int g_pend = 0;
  bool g_open = false;
  float acc[P];
#pragma unroll
  for (int p = 0; p < P; ++p) acc[p] = 0.0f;
  double acc64 = 0.0;
  // combination stepper over bucket cb
  int64_t cb = 0, c_lo = 0, c_hi = 0, c_vs = 0, c_nv = 0, c_next = 0;
  bool c_open = false;
  float beta[K];

  while (cb < B) {
    // one Gram step, at most one bucket ahead of the combination
    const bool can_gram = gb < B && gb <= cb + 1;
    if (can_gram) {
      if (!g_open) {
        int64_t hi;
        fused_slice<EPV>(v, gb, cta, n, &g_lo, &hi);
        g_vs = (g_lo + EPV - 1) / EPV * EPV;
        if (g_vs > hi) g_vs = hi;
        int64_t ve = hi / EPV * EPV;
        if (ve < g_vs) ve = g_vs;
        g_nv = (ve - g_vs) / EPV;
        const int nh = (int)(g_vs - g_lo), nt = (int)(hi - ve);
        if ((int)threadIdx.x < nh + nt) {
          const int64_t idx = (int)threadIdx.x < nh ? g_lo + threadIdx.x : ve + (threadIdx.x - nh);
          gram_accumulate_scalar<K, DT>(acc, g, idx);
        }
        g_next = 0;
        g_pend = 0;
        acc64 = 0.0;
        g_open = true;
      }
      {
        uint4 r[STEP][K];
#pragma unroll
        for (int j = 0; j < STEP; ++j) {
          const int64_t idx = g_next + threadIdx.x + (int64_t)j * kThreads;
          if (idx < g_nv) {
#pragma unroll
            for (int k = 0; k < K; ++k)
              r[j][k] = ld16_policy_nc(static_cast<const char*>(g.p[k]) + (g_vs + idx * EPV) * IB, keep);
          }
        }
#pragma unroll
        for (int j = 0; j < STEP; ++j)
          if (g_next + threadIdx.x + (int64_t)j * kThreads < g_nv) gram_accumulate<K, DT>(acc, r[j]);
      }
      g_next += (int64_t)STEP * kThreads;
      g_pend += STEP;
      const bool done = g_next >= g_nv;
      if (done || g_pend >= kVecPerThread) {   // fixed-order reduction of the sub-slice
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
        for (int p = 0; p < P; ++p) {
          float x = acc[p];
          x += __shfl_down_sync(0xffffffffu, x, 16);
          x += __shfl_down_sync(0xffffffffu, x, 8);
          x += __shfl_down_sync(0xffffffffu, x, 4);
          x += __shfl_down_sync(0xffffffffu, x, 2);
          x += __shfl_down_sync(0xffffffffu, x, 1);
          if (lane == 0) red[warp][p] = x;
          acc[p] = 0.0f;
        }
        __syncthreads();
        if ((int)threadIdx.x < P) {
          double t = 0.0;
#pragma unroll
          for (int w = 0; w < kWarps; ++w) t += (double)red[w][threadIdx.x];
          acc64 += t;
        }
        g_pend = 0;
        if (done) {
          double* ring = f.ring + (size_t)(gb & 1) * kFusedMaxCtas * P + (size_t)cta * P;
          if ((int)threadIdx.x < P) {
            ring[threadIdx.x] = acc64;
            __threadfence();
          }
        }
        __syncthreads();
        if (done) {
          if (threadIdx.x == 0) atomicAdd(f.arrive + gb, 1);
          ++gb;
          g_open = false;
        }
      }
    }

    // combination of bucket cb once its beta is ready
    if (cb < gb) {
      if (!c_open) {
        if (threadIdx.x == 0) {
          int go;
          if (can_gram && gb <= cb + 1 && gb < B) {   // more Gram work to overlap: just look
            go = ld_acquire(f.ready + cb) >= 1 ? 1 : 0;
            if (!go && *(volatile int32_t*)&v.hdr->status != 0) go = -1;
          } else {
            go = fused_wait(f.ready + cb, 1, v.hdr) ? 1 : -1;
          }
          if (go == 1) {
#pragma unroll
            for (int k = 0; k < K; ++k) beta_sh[k] = __ldcg(v.beta + cb * K + k);
          }
          s_go = go;
        }
        __syncthreads();
        const int go = s_go;
        if (go < 0) return;
        if (go == 1) {
#pragma unroll
          for (int k = 0; k < K; ++k) beta[k] = beta_sh[k];
          fused_slice<EPV>(v, cb, cta, n, &c_lo, &c_hi);
          c_vs = (c_lo + EPV - 1) / EPV * EPV;
          if (c_vs > c_hi) c_vs = c_hi;
          int64_t ve = c_hi / EPV * EPV;
          if (ve < c_vs) ve = c_vs;
          c_nv = (ve - c_vs) / EPV;
          const int nh = (int)(c_vs - c_lo), nt = (int)(c_hi - ve);
          if ((int)threadIdx.x < nh + nt) {
            const int64_t idx = (int)threadIdx.x < nh ? c_lo + threadIdx.x : ve + (threadIdx.x - nh);
            float t = 0.0f;
#pragma unroll
            for (int k = 0; k < K; ++k) t = fmaf(beta[k], load_scalar<DT>(g.p[k], idx), t);
            store_scalar<DTO>(out, idx, t);
          }
          c_next = 0;
          c_open = true;
        }
        __syncthreads();
      }
      if (c_open) {
        uint4 r[STEP][K];
#pragma unroll
        for (int j = 0; j < STEP; ++j) {
          const int64_t idx = c_next + threadIdx.x + (int64_t)j * kThreads;
          if (idx < c_nv) {
#pragma unroll
            for (int k = 0; k < K; ++k)
              r[j][k] = ld16_policy(static_cast<const char*>(g.p[k]) + (c_vs + idx * EPV) * IB, last_use);
          }
        }
#pragma unroll
        for (int j = 0; j < STEP; ++j) {
          const int64_t idx = c_next + threadIdx.x + (int64_t)j * kThreads;
          if (idx < c_nv) {
            float y[EPV];
#pragma unroll
            for (int q = 0; q < EPV; ++q) {
              float t = 0.0f;
#pragma unroll
              for (int k = 0; k < K; ++k) t = fmaf(beta[k], vec_elem<DT>(r[j][k], q), t);
              y[q] = t;
            }
            store_out<DTO>(out, c_vs + idx * EPV, y, EPV);
          }
        }
        c_next += (int64_t)STEP * kThreads;
        if (c_next >= c_nv) {
          c_open = false;
          ++cb;
        }
      }
    }
  }
}

#define BKMOO_FUSED_ROW(K, DTI)                                               \
  {(const void*)fused_resolve_kernel<K, DTI, BKMOO_F32>,                      \
   (const void*)fused_resolve_kernel<K, DTI, BKMOO_BF16>}

// Eight values of K per translation unit (compiled in parallel).
#define BKMOO_FUSED_TABLE8(DTI, K0)                                                        \
  static const void* const kFusedTable[8][2] = {                                           \
      BKMOO_FUSED_ROW(K0 + 0, DTI), BKMOO_FUSED_ROW(K0 + 1, DTI),                          \
      BKMOO_FUSED_ROW(K0 + 2, DTI), BKMOO_FUSED_ROW(K0 + 3, DTI),                          \
      BKMOO_FUSED_ROW(K0 + 4, DTI), BKMOO_FUSED_ROW(K0 + 5, DTI),                          \
      BKMOO_FUSED_ROW(K0 + 6, DTI), BKMOO_FUSED_ROW(K0 + 7, DTI)}

}  // namespace bkmoo
