// Fused resolve, one thread-block cluster per bucket: Gram -> solve ->
// combination for a bucket on the W SMs of one cluster, with no grid-wide
// synchronisation, so that the bucket's gradients are read from HBM once and
// re-read from L2 a few microseconds later (Algorithm 1 resolves each bucket
// as soon as it is complete).
//
// The grid is n_clusters clusters of W = 8 CTAs, one CTA per SM (15 clusters
// fit on a 152-SM part; 9-CTA clusters cover more SMs but measured slower).
// Cluster c resolves buckets c, c + n_clusters, ... in turn.  A bucket's
// 16-byte vectors are cut into W equal pieces, one per CTA (the unaligned
// head and tail elements go to the first and last piece).  A CTA has 15
// streaming warps and one solver warp; streaming thread t takes vectors t,
// t + 480, ... of the piece, items 0, 1, ... in that order (a CTA step reads
// 7.5 KB of each gradient contiguously).
//
// Streaming warps walk a fixed schedule of segments,
//   G(0), H(1), C(0), R(1), H(2), C(1), R(2), ..., C(J - 1),
// G = a bucket's whole Gram, H = its first `head` items per thread, R = the
// rest, C = the combination (read backwards: the lines read last first).
// Every thread keeps S stages of its next items (the K vectors of one
// position) in flight with cp.async into its own shared-memory slots, across
// segment boundaries (a combination's inputs do not depend on beta), with L2
// policies evict_last on Gram reads and evict_first on the re-read.  Gram
// sums are fp32 per thread over at most 16 items, then a fixed butterfly into
// fp64 lane-owned entries.  At the end of a bucket's Gram (G or R) each warp
// stores its partial in shared memory and arrives on named barrier 1 without
// waiting; at the start of a combination it waits on named barrier 2 for
// beta.  The H segment keeps the SM streaming while the bucket before it is
// solved, at the cost of holding `head` items per thread more in L2.
//
// The solver warp, per bucket j of the cluster:
//   1. waits on named barrier 1 for the 15 warp partials, adds them in warp
//      order into the CTA's partial,
//   2. stores the CTA's partial into slot [j % 2][rank] of every CTA of the
//      cluster (distributed shared memory) and arrives, with release
//      semantics at cluster scope, on that CTA's exchange barrier of slot
//      j % 2 (an mbarrier expecting W arrivals),
//   3. waits (acquire, bounded) for its own exchange barrier, adds the W
//      partials in rank order into G -- every CTA computes the same sums in
//      the same order, so every CTA solves for the same beta -- and solves
//      the rule (solver.cuh); CTA rank 0 writes beta, out_weights and
//      out_status,
//   4. publishes beta in shared memory and arrives on named barrier 2.
//
// Slot reuse: a peer writes slot j % 2 for bucket j only after it solved
// bucket j - 1, which needed this CTA's partial of bucket j - 1, which this
// CTA sent after its solver had finished bucket j - 2 (the last reader of
// the slot); the same argument orders the mbarrier phases (bucket j is phase
// j / 2 of slot j % 2) and the warp partial slots.  The named barriers never
// see two buckets' arrivals at once: warps arrive on barrier 1 for bucket
// j + 1 only after passing barrier 2 for bucket j, and the solver arrives on
// barrier 2 for bucket j + 1 only after passing barrier 1 for it.
// Only the exchange waits poll; each gives up after about a second without
// completion, or at once when any wait of the grid already gave up
// (BKMOO_ERR_TIMEOUT in the workspace status word), and the solver then
// carries on with what it has so that every barrier is still reached; the
// test flag BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE exercises this path.  A last
// cluster barrier keeps every CTA's shared memory alive until its peers are
// done with it.  Clusters never wait for one another, so they need not be
// co-resident.
//
// Results are deterministic for a given cluster shape and count; the pieces
// differ from the three-pass path's chunks, so the two agree to rounding.
#pragma once

#include <cooperative_groups.h>

#include "fused_impl.cuh"

namespace bkmoo {

// stages of the per-thread cp.async ring: 24 / K, i.e. 180 KiB of slots for
// K = 1..4 (measured faster than 28 / K, the most that fits)
__host__ __device__ constexpr int cluster_stages(int K) { return K >= 12 ? 2 : 24 / K; }
__host__ __device__ constexpr int cluster_smem_bytes(int K) {
  return cluster_stages(K) * K * 16 * kClusterStreamThreads;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
// Arrive on the barrier at the same shared-memory offset in CTA `rank` of
// the cluster; release at cluster scope (orders this thread's earlier
// stores, local or remote, before the arrival).
__device__ __forceinline__ void mbar_arrive_remote(uint64_t* bar, unsigned rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(remote)
               : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, unsigned parity) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2; "
      "selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Named barriers 1 and 2 (barrier 0 is __syncthreads): arrive without
// waiting, or wait for the count.
__device__ __forceinline__ void named_arrive(int id, int count) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void named_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Whole-warp bounded wait for phase `parity` of an exchange barrier: every
// lane's own try_wait must succeed (so every lane acquires).  False after
// about a second, or at once when a wait elsewhere already gave up.
__device__ bool cluster_exchange_wait(uint64_t* bar, unsigned parity, WsHeader* h, int lane) {
  const uint64_t t0 = global_ns();
  for (unsigned it = 0;; ++it) {
    if (__all_sync(0xffffffffu, mbar_try_wait_cluster(bar, parity))) return true;
    if ((it & 15u) == 15u) {
      bool give_up = *(volatile int32_t*)&h->status != 0 || global_ns() - t0 > kFusedWaitNs;
      if (__shfl_sync(0xffffffffu, give_up, 0)) break;
    }
  }
  if (lane == 0) record_error(h, BKMOO_ERR_TIMEOUT);
  return false;
}

// Segment s of a cluster's schedule over its J buckets (see above): kind
// 0 = G, 1 = H, 2 = C, 3 = R, and the bucket index j within the cluster.
struct ClusterSched {
  int64_t J;
  __device__ int64_t total() const { return J > 0 ? 3 * J - 1 : 0; }
  __device__ void at(int64_t s, int* kind, int64_t* j) const {
    if (s == 0) {
      *kind = 0;
      *j = 0;
      return;
    }
    if (s == 3 * J - 2) {
      *kind = 2;
      *j = J - 1;
      return;
    }
    const int64_t m = (s - 1) / 3;
    const int r = (int)((s - 1) - 3 * m);
    *kind = r == 0 ? 1 : r == 1 ? 2 : 3;
    *j = r == 1 ? m : m + 1;
  }
};

// Items [i0, i1) of thread t in segment (kind, piece): n = ceil(vectors / T)
// items per thread, H takes the first min(head, n), R the rest.
struct ClusterRange {
  int i0, i1, n_valid;
};
template <int T>
__device__ __forceinline__ ClusterRange cluster_range(int kind, const Piece& pc, int t, int head) {
  const int64_t npc = pc.vhi - pc.vlo;
  const int n = (int)((npc + T - 1) / T);
  const int h = head < 0 ? 0 : head < n ? head : n;
  ClusterRange r;
  r.i0 = kind == 3 ? h : 0;
  r.i1 = kind == 1 ? h : n;
  r.n_valid = npc > t ? (int)((npc - t + T - 1) / T) : 0;
  return r;
}

// Per-thread producer over the same segments as the consumer: copies the K
// vectors of its next item into stage (issued % S); every call commits one
// group (empty once the schedule is exhausted).  Item i is vector
// vlo + t + T i of a Gram piece, vhi - 1 - (t + T i) of a combination piece,
// valid when inside [vlo, vhi) -- the valid items of a range come first.
template <int K, int DT>
struct ClusterProducer {
  static constexpr int T = kClusterStreamThreads;
  ClusterSched sch;
  int64_t seg, total;
  int cid, ncl, q, t, head;
  const char* src[K];  // this thread's next item in each gradient
  int64_t step;        // bytes to its following item (negative: backwards)
  int left, valid;     // items left in the segment, and how many of them are valid
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
      int kind;
      int64_t j;
      sch.at(seg, &kind, &j);
      const Piece pc = fused_piece<EPV>(v, cid + j * ncl, q, kClusterCtas);
      const ClusterRange r = cluster_range<T>(kind, pc, t, head);
      left = r.i1 - r.i0;
      const int vend = r.n_valid < r.i1 ? r.n_valid : r.i1;
      valid = vend > r.i0 ? vend - r.i0 : 0;
      const bool comb = kind == 2;
      // pointers are only dereferenced for the `valid` first items
      const int64_t first = comb ? pc.vhi - 1 - t : pc.vlo + t + (int64_t)T * r.i0;
      step = (comb ? -(int64_t)T : (int64_t)T) * 16;
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

// The solver warp of a CTA (see above).
template <int K>
__device__ void cluster_solver_warp(const PlanView& v, const SolveParams& prm, float* out_weights,
                                    int32_t* out_status, int64_t J, int cid, int ncl, int rank,
                                    double (*part_sm)[kClusterStreamWarps][tri(K)],
                                    double* cta_sm, double (*xch)[kClusterCtas][tri(K)],
                                    uint64_t* xbar, double* G, float* Gf, double* beta_tmp,
                                    double (*beta_sh)[K]) {
  namespace cg = cooperative_groups;
  constexpr int P = tri(K);
  constexpr int W = kClusterCtas;
  const int lane = threadIdx.x & 31;
  cg::cluster_group cluster = cg::this_cluster();
  for (int64_t j = 0; j < J; ++j) {
    const int64_t b = cid + j * ncl;
    const int sl = (int)(j & 1);
    // 1. this CTA's warp partials, in warp order
    named_sync(1, kClusterThreads);
    for (int p = lane; p < P; p += 32) {
      double t = 0.0;
#pragma unroll
      for (int w = 0; w < kClusterStreamWarps; ++w) t += part_sm[sl][w][p];
      cta_sm[p] = t;
    }
    __syncwarp();
    // 2. to every CTA of the cluster: lane r writes CTA r's copy and arrives
    // (BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE: CTA 0 withholds its first one)
    const bool withhold =
        (prm.flags & BKMOO_FLAG_TEST_WITHHOLD_EXCHANGE) != 0u && rank == 0 && j == 0;
    if (lane < W && !withhold) {
      double* dst = cluster.map_shared_rank(&xch[sl][rank][0], lane);
#pragma unroll
      for (int p = 0; p < P; ++p) dst[p] = cta_sm[p];
      mbar_arrive_remote(&xbar[sl], (unsigned)lane);
    }
    // 3. the W partials in rank order, then the rule
    const bool ok = cluster_exchange_wait(&xbar[sl], (unsigned)((j >> 1) & 1), v.hdr, lane);
    for (int p = lane; p < P; p += 32) {
      double t = 0.0;
#pragma unroll
      for (int r = 0; r < W; ++r) t += xch[sl][r][p];
      int i = 0, rr = p;
      while (rr >= K - i) {
        rr -= K - i;
        ++i;
      }
      G[i * K + i + rr] = t;
      G[(i + rr) * K + i] = t;
    }
    __syncwarp();
    int st = solver::solve_bucket_warp<K>(K, G, Gf, prm, b, beta_tmp, lane);
    if (!ok) st = BKMOO_ERR_TIMEOUT;
    // 4. beta for the streaming warps; rank 0 writes the bucket's results
    if (lane < K) {
      beta_sh[sl][lane] = beta_tmp[lane];
      if (rank == 0) {
        const float fb = (float)beta_tmp[lane];
        v.beta[b * K + lane] = fb;
        if (out_weights) out_weights[b * K + lane] = fb;
      }
    }
    if (lane == 0 && rank == 0 && out_status) out_status[b] = st;
    __syncwarp();
    __threadfence_block();
    named_arrive(2, kClusterThreads);
  }
}

template <int K, int DT, int DTO>
__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kClusterThreads, 1)
    fused_cluster_kernel(const GradPtrs g, const PlanView v, const SolveParams prm,
                         float* out_weights, int32_t* out_status, void* out, int head) {
  namespace cg = cooperative_groups;
  constexpr int P = tri(K);
  constexpr int NP = (P + 31) / 32;
  constexpr int EPV = elems_per_vec(DT);
  constexpr int S = cluster_stages(K);
  constexpr int T = kClusterStreamThreads;
  __shared__ double part_sm[2][kClusterStreamWarps][P];
  __shared__ double cta_sm[P];
  __shared__ double xch[2][kClusterCtas][P];
  __shared__ __align__(8) uint64_t xbar[2];
  __shared__ double G[K * K];
  __shared__ float Gf[K * K];
  __shared__ double beta_tmp[K];
  __shared__ double beta_sh[2][K];
  extern __shared__ __align__(16) unsigned char cl_smem[];

  // uniform across the grid: every CTA leaves before any barrier
  if (!header_ok(v)) {
    if (blockIdx.x == 0) {
      if (threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
      if (out_status)
        for (int64_t b = threadIdx.x; b < v.n_buckets; b += blockDim.x)
          out_status[b] = BKMOO_ERR_WORKSPACE;
    }
    return;
  }
  cg::cluster_group cluster = cg::this_cluster();
  constexpr int W = kClusterCtas;
  const int rank = (int)cluster.block_rank();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int ncl = (int)(gridDim.x / W), cid = (int)(blockIdx.x / W);
  const int64_t B = v.n_buckets;
  const int64_t J = cid < B ? (B - cid + ncl - 1) / ncl : 0;
  if (threadIdx.x == 0) {
    mbar_init(&xbar[0], (unsigned)W);
    mbar_init(&xbar[1], (unsigned)W);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // every exchange barrier of the cluster is initialised before any arrival
  cluster.sync();

  if (wid == kClusterStreamWarps) {
    cluster_solver_warp<K>(v, prm, out_weights, out_status, J, cid, ncl, rank, part_sm,
                           cta_sm, xch, xbar, G, Gf, beta_tmp, beta_sh);
  } else {
    const int t = threadIdx.x;
    // stage slots [S][K][threads] of 16-byte vectors: neighbouring threads
    // use neighbouring 16-byte words (no shared-memory bank conflicts)
    uint4* slots = reinterpret_cast<uint4*>(cl_smem);
    auto slot = [&](int st, int k) -> uint4* { return slots + (st * K + k) * T + t; };

    ClusterProducer<K, DT> pr;
    pr.sch = ClusterSched{J};
    pr.cid = cid;
    pr.ncl = ncl;
    pr.q = rank;
    pr.t = t;
    pr.head = head;
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

    const ClusterSched sch{J};
    const int64_t total = sch.total();
    for (int64_t seg = 0; seg < total; ++seg) {
      int kind;
      int64_t j;
      sch.at(seg, &kind, &j);
      const int64_t b = cid + j * ncl;
      const Piece pc = fused_piece<EPV>(v, b, rank, W);
      const ClusterRange rg = cluster_range<T>(kind, pc, t, head);
      const int nh = rank == 0 ? (int)(pc.vs - pc.bo) : 0;
      const int nt = rank == W - 1 ? (int)(pc.be - pc.ve) : 0;
      if (kind != 2) {
        // ---- Gram items [i0, i1) of the piece; the unaligned elements with
        // the bucket's first Gram segment
        if (kind != 3 && t < nh + nt) {
          const int64_t idx = t < nh ? pc.bo + t : pc.ve + (t - nh);
          gram_accumulate_scalar<K, DT>(acc, g, idx);
        }
        for (int i = rg.i0; i < rg.i1; ++i) {
          pr.issue(v, g, slot, issued++ % S);
          cp_async_wait<S - 1>();
          const int st = consumed++ % S;
          if (i < rg.n_valid) {
            uint4 r[K];
#pragma unroll
            for (int k = 0; k < K; ++k) r[k] = *slot(st, k);
            gram_accumulate<K, DT>(acc, r);
          }
          if ((i & (kVecPerThread - 1)) == kVecPerThread - 1) flush();
        }
        if (kind != 1) {
          // the bucket's Gram is complete: publish this warp's partial
          flush();
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            if (lane + 32 * i < P) part_sm[j & 1][wid][lane + 32 * i] = acc64[i];
            acc64[i] = 0.0;
          }
          __syncwarp();
          __threadfence_block();
          named_arrive(1, kClusterThreads);
        }
      } else {
        // ---- combination of the piece, backwards, once beta is published
        named_sync(2, kClusterThreads);
        float beta[K];
#pragma unroll
        for (int k = 0; k < K; ++k) beta[k] = (float)beta_sh[j & 1][k];
        if (t < nh + nt) {
          const int64_t idx = t < nh ? pc.bo + t : pc.ve + (t - nh);
          float y = 0.0f;
#pragma unroll
          for (int k = 0; k < K; ++k) y = fmaf(beta[k], load_scalar<DT>(g.p[k], idx), y);
          store_scalar<DTO>(out, idx, y);
        }
        int64_t oel = pc.vs + (pc.vhi - 1 - t) * EPV;  // output element of item i
        for (int i = rg.i0; i < rg.i1; ++i, oel -= (int64_t)T * EPV) {
          pr.issue(v, g, slot, issued++ % S);
          cp_async_wait<S - 1>();
          const int st = consumed++ % S;
          if (i < rg.n_valid) {
            float y[EPV];
#pragma unroll
            for (int e = 0; e < EPV; ++e) {
              float s = 0.0f;
#pragma unroll
              for (int k = 0; k < K; ++k) s = fmaf(beta[k], vec_elem<DT>(*slot(st, k), e), s);
              y[e] = s;
            }
            store_out<DTO>(out, oel, y, EPV);
          }
        }
      }
    }
    cp_async_wait<0>();
  }
  // peers may still write into this CTA's shared memory until they pass here
  cluster.sync();
}

}  // namespace bkmoo
