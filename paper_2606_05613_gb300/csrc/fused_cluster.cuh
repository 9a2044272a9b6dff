// Fused resolve, one thread-block cluster per bucket: Gram -> solve ->
// combination for a bucket on the 8 SMs of one cluster, with no global
// synchronisation at all, so that the bucket's gradients are read from HBM
// once and re-read from L2 a few microseconds later.
//
// The grid is n_clusters clusters of kClusterCtas CTAs (one CTA of 8 warps
// per SM).  Cluster c resolves buckets c, c + n_clusters, ... in turn; a
// bucket's 16-byte vectors are cut into kClusterCtas equal pieces, one per
// CTA (the unaligned head and tail elements go to the first and last
// piece), thread t of a CTA taking vectors t, t + 256, ... of its piece (a
// CTA step reads 4 KB of each gradient contiguously).  For each bucket
// every CTA
//   1. streams the Gram of its piece (fp32 per thread over at most 16
//      items, a fixed butterfly into fp64 lane-owned entries, the 8 warp
//      partials added in warp order into the CTA's partial in shared
//      memory),
//   2. waits at the cluster barrier (release / acquire: every CTA's partial
//      is then visible to every other CTA),
//   3. on warp 0: adds the kClusterCtas CTA partials, read from the peers'
//      shared memory in rank order, into G and solves the rule
//      (solver.cuh) -- every CTA computes the same beta from the same sums
//      in the same order, so no broadcast is needed -- and CTA rank 0 writes
//      beta, out_weights and out_status,
//   4. combines its pieces, re-read backwards (the lines read last first).
// Each lane keeps S stages of its next items (K vectors of one position)
// in flight with cp.async into its own shared-memory slots, across the
// Gram / combination boundary (a combination's inputs do not depend on
// beta), with L2 policies evict_last on Gram reads and evict_first on the
// re-read.
//
// The CTA partial of bucket j sits in slot j % 2: it is rewritten at bucket
// j + 2, after every CTA of the cluster has passed the barrier of bucket
// j + 1, i.e. after every CTA finished reading it.  A last barrier keeps
// every CTA's shared memory alive until its peers are done with it.  There
// is no spin-wait: every CTA of a cluster goes through the same sequence of
// barriers (one per bucket of the cluster, plus the last).  Clusters never
// wait for one another, so they need not be co-resident.
//
// Results are deterministic for a given cluster count; the pieces differ
// from the three-pass path's chunks, so the two agree to rounding.
#pragma once

#include <cooperative_groups.h>

#include "fused_impl.cuh"

namespace bkmoo {

__host__ __device__ constexpr int cluster_stages(int K) {
  return K <= 1 ? 16 : K == 2 ? 12 : K == 3 ? 8 : 6;
}
__host__ __device__ constexpr int cluster_smem_bytes(int K) {
  return cluster_stages(K) * K * 16 * kClusterThreads;
}

template <int K, int DT, int DTO>
__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kClusterThreads, 1)
    fused_cluster_kernel(const GradPtrs g, const PlanView v, const SolveParams prm,
                         float* out_weights, int32_t* out_status, void* out) {
  namespace cg = cooperative_groups;
  constexpr int P = tri(K);
  constexpr int NP = (P + 31) / 32;
  constexpr int EPV = elems_per_vec(DT);
  constexpr int S = cluster_stages(K);
  __shared__ double part_sm[kClusterWarps][P];
  __shared__ double cta_part[2][P];
  __shared__ double G[K * K];
  __shared__ float Gf[K * K];
  __shared__ double beta_sh[K];
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
  const int rank = (int)cluster.block_rank();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int ncl = (int)(gridDim.x / kClusterCtas), cid = (int)(blockIdx.x / kClusterCtas);
  // piece q = rank of W = kClusterCtas, shared by the CTA's threads
  const int W = kClusterCtas, q = rank;
  const int T = kClusterThreads, t = threadIdx.x;
  const int64_t B = v.n_buckets;
  const FusedSched sch{cid < B ? (B - cid + ncl - 1) / ncl : 0, 0};

  // stage slots [S][K][threads] of 16-byte vectors: neighbouring threads use
  // neighbouring 16-byte words (no shared-memory bank conflicts)
  uint4* slots = reinterpret_cast<uint4*>(cl_smem);
  auto slot = [&](int st, int k) -> uint4* {
    return slots + (st * K + k) * kClusterThreads + threadIdx.x;
  };

  FusedProducer<K, DT, kClusterThreads> pr;
  pr.sch = sch;
  pr.grp = cid;
  pr.ng = ncl;
  pr.q = q;
  pr.W = W;
  pr.lane = t;
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

  const int64_t total = sch.total();
  for (int64_t seg = 0; seg < total; ++seg) {
    bool comb;
    int64_t j;
    sch.seg_at(seg, &comb, &j);
    const int64_t b = cid + j * ncl;
    const Piece pc = fused_piece<EPV>(v, b, q, W);
    const int64_t npc = pc.vhi - pc.vlo;
    const int n_items = (int)((npc + T - 1) / T);
    const int n_valid = npc > t ? (int)((npc - t + T - 1) / T) : 0;
    const int nh = q == 0 ? (int)(pc.vs - pc.bo) : 0;
    const int nt = q == W - 1 ? (int)(pc.be - pc.ve) : 0;
    if (!comb) {
      // ---- 1. Gram of this warp's piece
      if (t < nh + nt) {
        const int64_t idx = t < nh ? pc.bo + t : pc.ve + (t - nh);
        gram_accumulate_scalar<K, DT>(acc, g, idx);
      }
      for (int i = 0; i < n_items; ++i) {
        pr.issue(v, g, slot, issued++ % S);
        cp_async_wait<S - 1>();
        const int st = consumed++ % S;
        if (i < n_valid) {
          uint4 r[K];
#pragma unroll
          for (int k = 0; k < K; ++k) r[k] = *slot(st, k);
          gram_accumulate<K, DT>(acc, r);
        }
        if ((i & (kVecPerThread - 1)) == kVecPerThread - 1) flush();
      }
      flush();
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        if (lane + 32 * i < P) part_sm[wid][lane + 32 * i] = acc64[i];
        acc64[i] = 0.0;
      }
      __syncthreads();
      const int sl = (int)(j & 1);
      for (int p = threadIdx.x; p < P; p += kClusterThreads) {
        double t = 0.0;
#pragma unroll
        for (int w = 0; w < kClusterWarps; ++w) t += part_sm[w][p];
        cta_part[sl][p] = t;
      }
      // ---- 2. every CTA partial of the bucket is written
      cluster.sync();
      // ---- 3. the same sums, in the same order, in every CTA; solve
      if (wid == 0) {
        for (int p = lane; p < P; p += 32) {
          double t = 0.0;
#pragma unroll
          for (int r = 0; r < kClusterCtas; ++r) t += cluster.map_shared_rank(&cta_part[sl][0], r)[p];
          int i = 0, rr = p;
          while (rr >= K - i) {
            rr -= K - i;
            ++i;
          }
          G[i * K + i + rr] = t;
          G[(i + rr) * K + i] = t;
        }
        __syncwarp();
        const int st = solver::solve_bucket_warp<K>(K, G, Gf, prm, b, beta_sh, lane);
        if (rank == 0) {
          if (lane < K) {
            const float fb = (float)beta_sh[lane];
            v.beta[b * K + lane] = fb;
            if (out_weights) out_weights[b * K + lane] = fb;
          }
          if (lane == 0 && out_status) out_status[b] = st;
        }
      }
      __syncthreads();
    } else {
      // ---- 4. combination of this warp's piece, backwards
      float beta[K];
#pragma unroll
      for (int k = 0; k < K; ++k) beta[k] = (float)beta_sh[k];
      if (t < nh + nt) {
        const int64_t idx = t < nh ? pc.bo + t : pc.ve + (t - nh);
        float y = 0.0f;
#pragma unroll
        for (int k = 0; k < K; ++k) y = fmaf(beta[k], load_scalar<DT>(g.p[k], idx), y);
        store_scalar<DTO>(out, idx, y);
      }
      int64_t oel = pc.vs + (pc.vhi - 1 - t) * EPV;   // output element of item i
      for (int i = 0; i < n_items; ++i, oel -= (int64_t)T * EPV) {
        pr.issue(v, g, slot, issued++ % S);
        cp_async_wait<S - 1>();
        const int st = consumed++ % S;
        if (i < n_valid) {
          float y[EPV];
#pragma unroll
          for (int e = 0; e < EPV; ++e) {
            float t = 0.0f;
#pragma unroll
            for (int k = 0; k < K; ++k) t = fmaf(beta[k], vec_elem<DT>(*slot(st, k), e), t);
            y[e] = t;
          }
          store_out<DTO>(out, oel, y, EPV);
        }
      }
    }
  }
  cp_async_wait<0>();
  // peers may still read this CTA's partials of the last bucket
  cluster.sync();
}

}  // namespace bkmoo
