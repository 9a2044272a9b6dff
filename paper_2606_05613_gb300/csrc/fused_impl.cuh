// Fused resolve: one persistent, co-resident grid runs Gram -> solve ->
// combination bucket by bucket (Algorithm 1 resolves each bucket as soon as
// it is full), so that a bucket's gradients come from HBM once, for the Gram
// pass, and are read again by the combination while they are still in L2.
//
// Why groups.  Between the Gram read of a byte and its re-read, HBM keeps
// streaming other data; the re-read hits L2 only if everything read in
// between still fits.  That interval is the bucket's own streaming time plus
// the latency of its solve and hand-offs, so the grid is split into
// n_groups groups of CTAs: group g resolves buckets g, g + n_groups, ... one
// after the other, each bucket spread over the group's CTAs, and the host
// chooses n_groups so that (lookahead + 1) buckets per group fit the L2
// budget.  Many small buckets are then in flight at once, each handled by a
// few dozen CTAs, and every group streams its next bucket(s) while its
// current one is being solved.
//
// CTA layout.  Warps 0..10 stream, warp 11 solves.
//  A streaming warp owns piece (c_local * 11 + warp) of every bucket of its
//  group (the bucket's 16-byte vectors cut into group_size * 11 equal
//  pieces; the unaligned head and tail elements go to the first and last
//  piece) and walks a fixed schedule of segments: Gram(0) .. Gram(L-1),
//  then Gram(j + L), Comb(j) for j = 0, 1, ... (L = lookahead).  Each lane
//  keeps S stages of its next items (the K 16-byte vectors of one position)
//  in flight with cp.async into its own shared-memory slots, across segment
//  boundaries: a combination's inputs are prefetched before its beta is
//  known, since beta is only needed to consume them.
//    Gram segment: fp32 sums per lane over at most 16 items, fixed butterfly
//      into fp64 lane-owned entries; at the end the warp stores them in
//      shared memory, and the last of the 11 warps to finish adds them in a
//      fixed order, writes the CTA's partial to the group's ring slot and
//      arrives on arrive[b] (after a fence).  The CTA whose arrival
//      completes the bucket queues b for its own solver warp.
//    Comb segment: wait (bounded) for ready[b] (acquire), read beta, then
//      d = sum_k beta_k g_k over the piece, positions taken from the end of
//      the piece backwards (the lines read last are reused first).
//  The solver warp takes queued buckets: it sums the group's CTA partials
//  in a fixed order (fp64), solves the rule (solver.cuh), writes beta,
//  out_weights and out_status, fences and sets ready[b]; ready[B] counts the
//  buckets published.  It leaves when the CTA's streaming warps are done.
//
// Ring slots: bucket j of a group uses slot j % kFusedRing.  A warp writes
// bucket j's partial only while j <= (its next combination) + lookahead, so
// bucket j - kFusedRing (< j - lookahead - 1) was combined, hence solved,
// hence its partials were read: kFusedRing > lookahead + 1 suffices.
//
// Waits.  Streaming warps wait only for ready flags, the solver warp only
// for its queue; neither wait closes a cycle (a bucket is queued once all
// its Gram pieces arrived, and Gram work never waits for a combination).
// Every wait ends after about a second without progress, records
// BKMOO_ERR_TIMEOUT in the workspace status word and leaves the kernel; any
// recorded error ends every other wait at once.
//
// The grid must be co-resident (cooperative launch).  Results are
// deterministic for a given grid and group count; the pieces differ from
// the three-pass path's chunks, so the two agree to rounding, not bit for
// bit.
#pragma once

#include <cuda_bf16.h>

#include "combine_impl.cuh"
#include "gram_prefetch.cuh"
#include "solver.cuh"

namespace bkmoo {

constexpr uint64_t kFusedWaitNs = 1000000000ull;  // a wait gives up after 1 s
constexpr int kFusedQueue = 16;                    // solver queue entries per CTA

// L2 eviction-priority policies (createpolicy).
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
// cp.async of 16 bytes carrying an L2 eviction policy.
__device__ __forceinline__ void cp_async16_policy(void* smem_dst, const void* src, uint64_t pol) {
  asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(smem_dst)),
               "l"(src), "l"(pol)
               : "memory");
}

__device__ __forceinline__ int ld_acquire(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// A poll that does not order later loads (issued before a streaming step and
// read after it); pair a positive poll with fence_acquire.
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

// Piece q of W of bucket b: vectors [vlo, vhi) (in vector units from the
// bucket's first aligned element vs), plus the bucket's unaligned head
// [bo, vs) for q == 0 and tail [ve, be) for q == W - 1.
struct Piece {
  int64_t bo, be, vs, ve;  // bucket bounds and its aligned vector span (elements)
  int64_t vlo, vhi;        // this piece's vectors
};

template <int EPV>
__device__ __forceinline__ Piece fused_piece(const PlanView& v, int64_t b, int q, int W) {
  Piece p;
  p.bo = v.offsets[b];
  p.be = v.offsets[b + 1];
  p.vs = (p.bo + EPV - 1) / EPV * EPV;
  if (p.vs > p.be) p.vs = p.be;
  p.ve = p.be / EPV * EPV;
  if (p.ve < p.vs) p.ve = p.vs;
  const int64_t nv = (p.ve - p.vs) / EPV;
  p.vlo = nv * q / W;
  p.vhi = nv * (q + 1) / W;
  return p;
}

// Fixed-order sum of the M CTA partials (rows of P doubles) of one bucket
// into the symmetric G (shared).  For P <= 16 the rows are split into
// S = 32 / P stripes (lane l: entry l % P, rows l / P, l / P + S, ...) and the
// stripe sums are then added in stripe order; for P > 16 lane l owns entries
// l and l + 32 over all rows.  Each lane adds its rows in increasing order,
// loading them eight at a time so that the L2 round trips (the rows were
// written by other CTAs) overlap instead of following one another.
template <int P, int STRIDE>
__device__ __forceinline__ double fused_rows_sum(const double* rows, int c0, int M, int p) {
  double t = 0.0;
  for (int c = c0; c < M; c += 8 * STRIDE) {
    double x[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      x[i] = c + i * STRIDE < M ? __ldcg(rows + (size_t)(c + i * STRIDE) * P + p) : 0.0;
#pragma unroll
    for (int i = 0; i < 8; ++i) t += x[i];
  }
  return t;
}

template <int K>
__device__ __forceinline__ void fused_reduce(const double* rows, int M, double* G, int lane) {
  constexpr int P = tri(K);
  auto put = [&](int p, double t) {
    int i = 0, r = p;
    while (r >= K - i) {
      r -= K - i;
      ++i;
    }
    G[i * K + i + r] = t;
    G[(i + r) * K + i] = t;
  };
  if constexpr (P <= 16) {
    constexpr int S = 32 / P;
    const double part = lane < S * P ? fused_rows_sum<P, S>(rows, lane / P, M, lane % P) : 0.0;
    double tot = 0.0;
#pragma unroll
    for (int s = 0; s < S; ++s) tot += __shfl_sync(0xffffffffu, part, s * P + (lane % P));
    if (lane < P) put(lane, tot);
  } else {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int p = lane + 32 * h;
      if (p < P) put(p, fused_rows_sum<P, 1>(rows, 0, M, p));
    }
  }
}

// The solver warp of a CTA: takes the buckets its CTA completed from the
// shared-memory queue, reduces, solves and publishes them.
template <int K>
__device__ __noinline__ void fused_solver_warp(const FusedView& f, const SolveParams& prm,
                                               volatile int* queue, volatile int* done_warps) {
  constexpr int P = tri(K);
  __shared__ double G[K * K];
  __shared__ float Gf[K * K];
  __shared__ double beta_sh[K];
  const PlanView& v = f.v;
  const int lane = threadIdx.x & 31;
  const int64_t B = v.n_buckets;
  int head = 0;
  uint64_t t0 = global_ns();
  int seen = -1;
  for (unsigned it = 0;; ++it) {
    const int b32 = queue[head % kFusedQueue];
    __syncwarp();
    if (b32 >= 0) {
      const int64_t b = b32;
      if (lane == 0) queue[head % kFusedQueue] = -1;
      ++head;
      __threadfence();
      const int64_t grp = b % f.n_groups, j = b / f.n_groups;
      const int M = (int)((gridDim.x - grp + f.n_groups - 1) / f.n_groups);
      const double* rows =
          f.ring + ((size_t)grp * kFusedRing + (size_t)(j % kFusedRing)) * f.group_ctas * P;
      fused_reduce<K>(rows, M, G, lane);
      __syncwarp();
      const int st = solver::solve_bucket_warp<K>(K, G, Gf, prm, b, beta_sh, lane);
      if (lane < K) {
        const float fb = (float)beta_sh[lane];
        v.beta[b * K + lane] = fb;
        if (f.out_weights) f.out_weights[b * K + lane] = fb;
      }
      if (lane == 0 && f.out_status) f.out_status[b] = st;
      __threadfence();
      __syncwarp();
      // BKMOO_FLAG_TEST_WITHHOLD: bucket 0 is never published, so every
      // wait on it runs out (the failure-detection test)
      if (lane == 0 && !(b == 0 && (prm.flags & BKMOO_FLAG_TEST_WITHHOLD))) {
        atomicExch(f.ready + b, 1);
        atomicAdd(f.ready + B, 1);
      }
      __syncwarp();
      t0 = global_ns();
      continue;
    }
    if ((it & 15u) == 15u) {
      if (*done_warps == kFusedStreamWarps) return;
      if (*(volatile int32_t*)&v.hdr->status != 0) return;
      const int pub = ld_relaxed(f.ready + B);
      const uint64_t now = global_ns();
      if (pub != seen) {
        seen = pub;
        t0 = now;
      } else if (now - t0 > kFusedWaitNs) {
        if (lane == 0) record_error(v.hdr, BKMOO_ERR_TIMEOUT);
        return;
      }
    }
    __nanosleep(32);
  }
}

// A warp's schedule over the J buckets of its group with look-ahead L:
// Gram(0) .. Gram(L-1), then for j = 0 .. J-1: Gram(j + L) (when
// j + L < J) and Comb(j).  seg_at(s) gives segment s's (comb, j).
struct FusedSched {
  int64_t J;
  int L;
  __device__ int64_t prologue() const { return J < L ? J : L; }
  __device__ int64_t pairs() const { return J > L ? J - L : 0; }
  __device__ int64_t total() const { return prologue() + J + pairs(); }
  __device__ void seg_at(int64_t s, bool* comb, int64_t* j) const {
    const int64_t p0 = prologue(), np = pairs();
    if (s < p0) {
      *comb = false;
      *j = s;
      return;
    }
    const int64_t t = s - p0;
    if (t < 2 * np) {
      *comb = (t & 1) != 0;
      *j = *comb ? t / 2 : t / 2 + L;
      return;
    }
    *comb = true;
    *j = np + (t - 2 * np);
  }
};

// Per-thread producer: walks the same segments as the consumer and copies
// the K vectors of its next item into stage (issued % S) with cp.async;
// every call commits one group (empty once the schedule is exhausted).  A
// piece is shared by STRIDE threads (a warp here; a whole CTA in the
// cluster kernel).  Items of a segment: n = ceil(piece vectors / STRIDE) per
// thread (uniform over the STRIDE threads); item i is vector
// lo + lane + STRIDE i of a Gram piece, hi - 1 - (lane + STRIDE i) of a
// combination piece (read backwards), valid when inside [lo, hi).
template <int K, int DT, int STRIDE = 32>
struct FusedProducer {
  FusedSched sch;
  int64_t seg, total;
  int grp, ng, q, W, lane;   // lane: this thread's index among the STRIDE that share a piece
  const char* src[K];        // this thread's next item in each gradient
  int64_t step;              // bytes to its following item (negative: backwards)
  int left, valid;           // items left in the segment, and how many of them are valid
  uint64_t pol;
  __device__ void begin(const PlanView& v, const GradPtrs& g) {
    total = sch.total();
    seg = 0;
    open(v, g);
  }
  __device__ void open(const PlanView& v, const GradPtrs& g) {
    constexpr int EPV = elems_per_vec(DT);
    constexpr int IB = 16 / EPV;
    while (seg < total) {
      bool comb;
      int64_t j;
      sch.seg_at(seg, &comb, &j);
      const Piece pc = fused_piece<EPV>(v, grp + j * ng, q, W);
      const int64_t n = pc.vhi - pc.vlo;
      left = (int)((n + STRIDE - 1) / STRIDE);
      valid = n > lane ? (int)((n - lane + STRIDE - 1) / STRIDE) : 0;
      // pointers are only dereferenced for the `valid` first items
      const int64_t first = comb ? pc.vhi - 1 - lane : pc.vlo + lane;
      step = (comb ? -(int64_t)STRIDE : (int64_t)STRIDE) * 16;
#pragma unroll
      for (int k = 0; k < K; ++k)
        src[k] = static_cast<const char*>(g.p[k]) + (pc.vs + first * EPV) * IB;
      // Gram reads stay in L2 for the re-read (evict_last); the re-read is
      // the last use (evict_first)
      pol = comb ? policy_evict_first() : policy_evict_last();
      if (left > 0) return;
      ++seg;
    }
  }
  template <typename Slot>
  __device__ __forceinline__ void issue(const PlanView& v, const GradPtrs& g, Slot slot,
                                        int stage) {
    if (seg < total) {
      if (valid > 0) {
#pragma unroll
        for (int k = 0; k < K; ++k) {
          cp_async16_policy(slot(stage, k), src[k], pol);
          src[k] += step;
        }
        --valid;
      }
      if (--left == 0) {
        ++seg;
        open(v, g);
      }
    }
    cp_async_commit();
  }
};

template <int K, int DT, int DTO>
__global__ void __launch_bounds__(kFusedThreads, 1)
    fused_resolve_kernel(const GradPtrs g, const FusedView f, const SolveParams prm, void* out) {
  constexpr int P = tri(K);
  constexpr int NP = (P + 31) / 32;       // fp64 accumulators per lane
  constexpr int EPV = elems_per_vec(DT);
  constexpr int S = fused_stages(K);
  __shared__ double part_sm[kFusedRing][kFusedStreamWarps][P];
  __shared__ int cnt_sm[kFusedRing];
  __shared__ int queue_sm[kFusedQueue];
  __shared__ int q_tail, done_warps;
  extern __shared__ __align__(16) unsigned char fused_smem[];
  const PlanView& v = f.v;
  if (!header_ok(v)) {
    if (blockIdx.x == 0) {
      if (threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
      if (f.out_status)
        for (int64_t b = threadIdx.x; b < v.n_buckets; b += blockDim.x)
          f.out_status[b] = BKMOO_ERR_WORKSPACE;
    }
    return;
  }
  if (threadIdx.x < kFusedRing) cnt_sm[threadIdx.x] = 0;
  if (threadIdx.x < kFusedQueue) queue_sm[threadIdx.x] = -1;
  if (threadIdx.x == 0) {
    q_tail = 0;
    done_warps = 0;
  }
  __syncthreads();   // the only CTA-wide barrier; every warp runs on its own below

  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (wid == kFusedStreamWarps) {
    fused_solver_warp<K>(f, prm, queue_sm, &done_warps);
    return;
  }

  // stage slots [S][K][streaming threads] of 16-byte vectors: neighbouring
  // lanes use neighbouring 16-byte words (no shared-memory bank conflicts)
  uint4* slots = reinterpret_cast<uint4*>(fused_smem);
  constexpr int NT = 32 * kFusedStreamWarps;
  auto slot = [&](int st, int k) -> uint4* { return slots + (st * K + k) * NT + threadIdx.x; };

  const int ng = f.n_groups;
  const int cta = blockIdx.x, grp = cta % ng, c_loc = cta / ng;
  const int M = (int)((gridDim.x - grp + ng - 1) / ng);
  const int W = M * kFusedStreamWarps, q = c_loc * kFusedStreamWarps + wid;
  const int64_t B = v.n_buckets;
  const FusedSched sch{grp < B ? (B - grp + ng - 1) / ng : 0, f.lookahead};

  FusedProducer<K, DT> pr;
  pr.sch = sch;
  pr.grp = grp;
  pr.ng = ng;
  pr.q = q;
  pr.W = W;
  pr.lane = lane;
  pr.begin(v, g);
  int issued = 0;
#pragma unroll 1
  for (int j = 0; j < S - 1; ++j) pr.issue(v, g, slot, issued++ % S);
  int consumed = 0;

  float acc[P];
#pragma unroll
  for (int p = 0; p < P; ++p) acc[p] = 0.0f;
  double acc64[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) acc64[i] = 0.0;
  auto flush = [&]() {
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
  };

  bool failed = false;
  const int64_t total = sch.total();
  for (int64_t seg = 0; seg < total && !failed; ++seg) {
    bool comb;
    int64_t j;
    sch.seg_at(seg, &comb, &j);
    const int64_t b = grp + j * ng;
    const Piece pc = fused_piece<EPV>(v, b, q, W);
    const int64_t n_items = (pc.vhi - pc.vlo + 31) / 32;
    if (!comb) {
      // ---- Gram of this warp's piece of bucket b
      const int nh = q == 0 ? (int)(pc.vs - pc.bo) : 0;
      const int nt = q == W - 1 ? (int)(pc.be - pc.ve) : 0;
      if (lane < nh + nt) {
        const int64_t idx = lane < nh ? pc.bo + lane : pc.ve + (lane - nh);
        gram_accumulate_scalar<K, DT>(acc, g, idx);
      }
      for (int64_t i = 0; i < n_items; ++i) {
        pr.issue(v, g, slot, issued++ % S);
        cp_async_wait<S - 1>();
        const int st = consumed++ % S;
        if (pc.vlo + lane + 32 * i < pc.vhi) {
          uint4 r[K];
#pragma unroll
          for (int k = 0; k < K; ++k) r[k] = *slot(st, k);
          gram_accumulate<K, DT>(acc, r);
        }
        if ((i & (kVecPerThread - 1)) == kVecPerThread - 1) flush();
      }
      flush();
      // the CTA's warp partials, added in a fixed order by the last warp to
      // finish, which writes the CTA partial and arrives
      const int rs = (int)(j % kFusedRing);
#pragma unroll
      for (int i = 0; i < NP; ++i)
        if (lane + 32 * i < P) part_sm[rs][wid][lane + 32 * i] = acc64[i];
      __threadfence_block();
      __syncwarp();
      int last = 0;
      if (lane == 0) last = (atomicAdd(&cnt_sm[rs], 1) == kFusedStreamWarps - 1) ? 1 : 0;
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence_block();
        double* row = f.ring + (((size_t)grp * kFusedRing + rs) * f.group_ctas + c_loc) * P;
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          const int p = lane + 32 * i;
          if (p < P) {
            double t = 0.0;
#pragma unroll
            for (int w = 0; w < kFusedStreamWarps; ++w) t += ((volatile double*)part_sm[rs][w])[p];
            __stcg(row + p, t);
          }
        }
        __threadfence();
        __syncwarp();
        if (lane == 0) {
          cnt_sm[rs] = 0;
          if (atomicAdd(f.arrive + b, 1) == M - 1) {
            // this CTA completed bucket b: hand it to the solver warp
            __threadfence();
            const int pos = atomicAdd(&q_tail, 1);
            ((volatile int*)queue_sm)[pos % kFusedQueue] = (int)b;
            __threadfence_block();
          }
        }
      }
#pragma unroll
      for (int i = 0; i < NP; ++i) acc64[i] = 0.0;
    } else {
      // ---- combination of this warp's piece of bucket b, backwards
      int ok = 0;
      if (lane == 0) ok = fused_wait(f.ready + b, 1, v.hdr) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        failed = true;
        break;
      }
      fence_acquire();
      float beta[K];
      {
        const float bl = lane < K ? __ldcg(v.beta + b * K + lane) : 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) beta[k] = __shfl_sync(0xffffffffu, bl, k);
      }
      const int nh = q == 0 ? (int)(pc.vs - pc.bo) : 0;
      const int nt = q == W - 1 ? (int)(pc.be - pc.ve) : 0;
      if (lane < nh + nt) {
        const int64_t idx = lane < nh ? pc.bo + lane : pc.ve + (lane - nh);
        float t = 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) t = fmaf(beta[k], load_scalar<DT>(g.p[k], idx), t);
        store_scalar<DTO>(out, idx, t);
      }
      for (int64_t i = 0; i < n_items; ++i) {
        pr.issue(v, g, slot, issued++ % S);
        cp_async_wait<S - 1>();
        const int st = consumed++ % S;
        const int64_t idx = pc.vhi - 1 - (lane + 32 * i);
        if (idx >= pc.vlo) {
          float y[EPV];
#pragma unroll
          for (int e = 0; e < EPV; ++e) {
            float t = 0.0f;
#pragma unroll
            for (int k = 0; k < K; ++k) t = fmaf(beta[k], vec_elem<DT>(*slot(st, k), e), t);
            y[e] = t;
          }
          store_out<DTO>(out, pc.vs + idx * EPV, y, EPV);
        }
      }
    }
  }
  cp_async_wait<0>();
  __syncwarp();
  if (lane == 0) atomicAdd(&done_warps, 1);
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
