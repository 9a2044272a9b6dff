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
// A poll that does not order later loads (so it can be issued before a
// streaming step and read after it); pair a positive poll with fence_acquire.
__device__ __forceinline__ int ld_relaxed(const int32_t* p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ void fence_acquire() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
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
  constexpr int STRIPES = kThreads / P > 0 ? kThreads / P : 1;
  __shared__ double G[K * K];
  __shared__ float Gf[K * K];
  __shared__ double part[kThreads];
  __shared__ double beta_sh[K];
  __shared__ int go;
  const PlanView& v = f.v;
  const int n = f.n_stream;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t b = 0; b < v.n_buckets; ++b) {
    if (threadIdx.x == 0) go = fused_wait(f.arrive + b, n, v.hdr) ? 1 : 0;
    __syncthreads();
    if (!go) return;
    // fixed-order reduction of the n CTA partials: thread t sums entry t % P
    // over stripe t / P of the CTAs with four interleaved accumulators, then
    // thread e adds its STRIPES stripe sums in order
    const double* ring = f.ring + (size_t)(b & 1) * kFusedMaxCtas * P;
    if ((int)threadIdx.x < STRIPES * P) {
      const int e = threadIdx.x % P, st = threadIdx.x / P;
      const int c0 = (int)((int64_t)n * st / STRIPES), c1 = (int)((int64_t)n * (st + 1) / STRIPES);
      double t0 = 0.0, t1 = 0.0, t2 = 0.0, t3 = 0.0;
      int c = c0;
      for (; c + 3 < c1; c += 4) {
        t0 += __ldcg(ring + (size_t)c * P + e);
        t1 += __ldcg(ring + (size_t)(c + 1) * P + e);
        t2 += __ldcg(ring + (size_t)(c + 2) * P + e);
        t3 += __ldcg(ring + (size_t)(c + 3) * P + e);
      }
      for (; c < c1; ++c) t0 += __ldcg(ring + (size_t)c * P + e);
      part[threadIdx.x] = (t0 + t1) + (t2 + t3);
    }
    __syncthreads();
    if ((int)threadIdx.x < P) {
      double t0 = 0.0, t1 = 0.0;
      int st = 0;
      for (; st + 1 < STRIPES; st += 2) {
        t0 += part[st * P + threadIdx.x];
        t1 += part[(st + 1) * P + threadIdx.x];
      }
      if (st < STRIPES) t0 += part[st * P + threadIdx.x];
      const double t = t0 + t1;
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
      const int st = solver::solve_bucket_warp<K>(K, G, Gf, prm, b, beta_sh, lane);
      if (lane < K) {
        const float fb = (float)beta_sh[lane];
        v.beta[b * K + lane] = fb;
        if (f.out_weights) f.out_weights[b * K + lane] = fb;
        __threadfence();
      }
      if (lane == 0 && f.out_status) f.out_status[b] = st;
      __syncwarp();
      // BKMOO_FLAG_TEST_WITHHOLD: bucket 0 is never published, so every
      // wait on it runs out (the failure-detection test)
      if (lane == 0 && !(b == 0 && (prm.flags & BKMOO_FLAG_TEST_WITHHOLD))) {
        __threadfence();
        atomicExch(f.ready + b, 1);
      }
    }
    __syncthreads();
  }
}

// Resident CTAs per SM the register budget is capped for: the streaming
// loops need up to 128 (K <= 4) and 255 (K > 4) registers per thread; the
// solver code shares the kernel and spills instead of lowering occupancy.
template <int K>
struct FusedMinBlocks {
  static constexpr int value = K <= 4 ? 2 : 1;
};

// Piece of bucket b streamed by warp w of CTA cta: the CTA's slice cut in
// kWarps equal, 16-byte-aligned pieces.
template <int EPV>
__device__ __forceinline__ void warp_piece(const PlanView& v, int64_t b, int cta, int n, int w,
                                           int64_t* lo, int64_t* hi) {
  int64_t a, z;
  fused_slice<EPV>(v, b, cta, n, &a, &z);
  int64_t ps = (z - a + kWarps - 1) / kWarps;
  ps = (ps + EPV - 1) / EPV * EPV;
  int64_t l = a + (int64_t)w * ps;
  if (l > z) l = z;
  int64_t h = l + ps;
  if (h > z) h = z;
  *lo = l;
  *hi = h;
}

template <int K, int DT, int DTO>
__global__ void __launch_bounds__(kThreads, FusedMinBlocks<K>::value)
    fused_resolve_kernel(const GradPtrs g, const FusedView f, const SolveParams prm, void* out) {
  constexpr int P = tri(K);
  constexpr int NP = (P + 31) / 32;       // fp64 accumulators per lane
  constexpr int EPV = elems_per_vec(DT);
  constexpr int IB = 16 / EPV;
  constexpr int STEP = K <= 2 ? 4 : 2;    // vectors per lane per Gram / combination step
  __shared__ double part_sm[2][kWarps][P];
  __shared__ int cnt_sm[2];
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
  if (threadIdx.x < 2) cnt_sm[threadIdx.x] = 0;
  __syncthreads();   // the only CTA-wide barrier; every warp runs on its own below

  const int cta = blockIdx.x, n = f.n_stream;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t B = v.n_buckets;
  const uint64_t keep = policy_evict_last(), last_use = policy_evict_first();

  int64_t gb = 0, g_vs = 0, g_nv = 0, g_next = 0;
  int g_pend = 0;
  bool g_open = false;
  float acc[P];
#pragma unroll
  for (int p = 0; p < P; ++p) acc[p] = 0.0f;
  double acc64[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) acc64[i] = 0.0;

  int64_t cb = 0, c_vs = 0, c_nv = 0, c_next = 0;
  bool c_open = false;
  float beta[K];
#pragma unroll
  for (int k = 0; k < K; ++k) beta[k] = 0.0f;

  while (cb < B) {
    // poll for beta of bucket cb now; read the answer after the Gram step
    const bool want = !c_open && cb < gb;
    int flag = 0;
    if (want && lane == 0) flag = ld_relaxed(f.ready + cb);

    // ---- one Gram step of bucket gb: at most one bucket ahead of cb, and
    // when ahead, at most `lookahead` of a piece ahead of the combination
    // of cb, so that both buckets' unconsumed lines fit in L2
    bool gram_ok = gb < B && gb <= cb + 1;
    if (gram_ok && gb == cb + 1 && g_open) {
      const int64_t lead = (g_nv * f.lookahead) >> 10;
      const int64_t follow = c_open ? (c_next * g_nv) / (c_nv > 0 ? c_nv : 1) : 0;
      gram_ok = g_next < follow + lead;
    }
    if (gram_ok) {
      if (!g_open) {
        int64_t lo, hi;
        warp_piece<EPV>(v, gb, cta, n, wid, &lo, &hi);
        g_vs = (lo + EPV - 1) / EPV * EPV;
        if (g_vs > hi) g_vs = hi;
        int64_t ve = hi / EPV * EPV;
        if (ve < g_vs) ve = g_vs;
        g_nv = (ve - g_vs) / EPV;
        const int nh = (int)(g_vs - lo), nt = (int)(hi - ve);
        if (lane < nh + nt) {
          const int64_t idx = lane < nh ? lo + lane : ve + (lane - nh);
          gram_accumulate_scalar<K, DT>(acc, g, idx);
        }
        g_next = 0;
        g_pend = 0;
        g_open = true;
      }
      uint4 r[STEP][K];
#pragma unroll
      for (int j = 0; j < STEP; ++j) {
        const int64_t idx = g_next + lane + 32 * j;
        if (idx < g_nv) {
#pragma unroll
          for (int k = 0; k < K; ++k)
            r[j][k] = ld16_policy_nc(static_cast<const char*>(g.p[k]) + (g_vs + idx * EPV) * IB, keep);
        }
      }
#pragma unroll
      for (int j = 0; j < STEP; ++j)
        if (g_next + lane + 32 * j < g_nv) gram_accumulate<K, DT>(acc, r[j]);
      g_next += 32 * STEP;
      g_pend += STEP;
      const bool done = g_next >= g_nv;
      if (done || g_pend >= kVecPerThread) {
        // fixed butterfly over the warp; lane p % 32 keeps entry p in fp64
#pragma unroll
        for (int p = 0; p < P; ++p) {
          float x = acc[p];
          x += __shfl_xor_sync(0xffffffffu, x, 16);
          x += __shfl_xor_sync(0xffffffffu, x, 8);
          x += __shfl_xor_sync(0xffffffffu, x, 4);
          x += __shfl_xor_sync(0xffffffffu, x, 2);
          x += __shfl_xor_sync(0xffffffffu, x, 1);
          if ((p & 31) == lane) acc64[p >> 5] += (double)x;
          acc[p] = 0.0f;
        }
        g_pend = 0;
      }
      if (done) {
        // combine the CTA's 8 warp partials in a fixed order; the last warp
        // to finish publishes the CTA's partial and arrives
        const int slot = (int)(gb & 1);
#pragma unroll
        for (int i = 0; i < NP; ++i)
          if (lane + 32 * i < P) part_sm[slot][wid][lane + 32 * i] = acc64[i];
        __threadfence_block();
        __syncwarp();
        int last = 0;
        if (lane == 0) last = (atomicAdd(&cnt_sm[slot], 1) == kWarps - 1) ? 1 : 0;
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          __threadfence_block();
          double* ring = f.ring + (size_t)slot * kFusedMaxCtas * P + (size_t)cta * P;
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            const int p = lane + 32 * i;
            if (p < P) {
              double t = 0.0;
#pragma unroll
              for (int w = 0; w < kWarps; ++w) t += ((volatile double*)part_sm[slot][w])[p];
              ring[p] = t;
            }
          }
          __threadfence();
          __syncwarp();
          if (lane == 0) {
            cnt_sm[slot] = 0;
            __threadfence();
            atomicAdd(f.arrive + gb, 1);
          }
        }
#pragma unroll
        for (int i = 0; i < NP; ++i) acc64[i] = 0.0;
        ++gb;
        g_open = false;
      }
    }

    // ---- open the combination of bucket cb once its beta is ready
    if (want) {
      flag = __shfl_sync(0xffffffffu, flag, 0);
      bool more = gb < B && gb <= cb + 1;
      if (more && gb == cb + 1 && g_open) more = g_next < ((g_nv * f.lookahead) >> 10);
      if (!flag && !more) {   // nothing left to overlap: wait
        int ok = 0;
        if (lane == 0) ok = fused_wait(f.ready + cb, 1, v.hdr) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, ok, 0)) return;
        flag = 1;
      }
      if (flag) {
        fence_acquire();
        float bl = lane < K ? __ldcg(v.beta + cb * K + lane) : 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) beta[k] = __shfl_sync(0xffffffffu, bl, k);
        int64_t lo, hi;
        warp_piece<EPV>(v, cb, cta, n, wid, &lo, &hi);
        c_vs = (lo + EPV - 1) / EPV * EPV;
        if (c_vs > hi) c_vs = hi;
        int64_t ve = hi / EPV * EPV;
        if (ve < c_vs) ve = c_vs;
        c_nv = (ve - c_vs) / EPV;
        const int nh = (int)(c_vs - lo), nt = (int)(hi - ve);
        if (lane < nh + nt) {
          const int64_t idx = lane < nh ? lo + lane : ve + (lane - nh);
          float t = 0.0f;
#pragma unroll
          for (int k = 0; k < K; ++k) t = fmaf(beta[k], load_scalar<DT>(g.p[k], idx), t);
          store_scalar<DTO>(out, idx, t);
        }
        c_next = 0;
        c_open = true;
      } else if (*(volatile int32_t*)&v.hdr->status != 0) {
        return;
      }
    }

    // ---- one combination step of bucket cb, from the end of the piece back
    // to its start: the lines the Gram pass read last are read first, so
    // an LRU L2 still holds them even when the bucket and its output
    // together slightly exceed the cache
    if (c_open) {
      uint4 r[STEP][K];
#pragma unroll
      for (int j = 0; j < STEP; ++j) {
        const int64_t idx = c_nv - 1 - (c_next + lane + 32 * j);
        if (idx >= 0) {
#pragma unroll
          for (int k = 0; k < K; ++k)
            r[j][k] = ld16_policy(static_cast<const char*>(g.p[k]) + (c_vs + idx * EPV) * IB, last_use);
        }
      }
#pragma unroll
      for (int j = 0; j < STEP; ++j) {
        const int64_t idx = c_nv - 1 - (c_next + lane + 32 * j);
        if (idx >= 0) {
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
      c_next += 32 * STEP;
      if (c_next >= c_nv) {
        c_open = false;
        ++cb;
      }
    }
  }
}

#define BKMOO_FUSED_ROW(K, DTI)                                               \
  {(const void*)fused_resolve_kernel<K, DTI, BKMOO_F32>,                      \
   (const void*)fused_resolve_kernel<K, DTI, BKMOO_BF16>}

// A few values of K per translation unit (compiled in parallel).
#define BKMOO_FUSED_TABLE4(DTI, K0)                                                        \
  static const void* const kFusedTable[4][2] = {                                           \
      BKMOO_FUSED_ROW(K0 + 0, DTI), BKMOO_FUSED_ROW(K0 + 1, DTI),                          \
      BKMOO_FUSED_ROW(K0 + 2, DTI), BKMOO_FUSED_ROW(K0 + 3, DTI)}
#define BKMOO_FUSED_TABLE2(DTI, K0)                                                        \
  static const void* const kFusedTable[2][2] = {BKMOO_FUSED_ROW(K0 + 0, DTI),               \
                                                BKMOO_FUSED_ROW(K0 + 1, DTI)}

}  // namespace bkmoo
