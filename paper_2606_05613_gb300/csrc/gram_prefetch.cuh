// Gram pass for large K with a per-thread prefetch into shared memory.
//
// At K >= 12 a thread's K(K+1)/2 fp32 accumulators (136 at K = 16) leave
// room for 8 warps per SM, and a thread that loads its K vectors into
// registers and then computes keeps one load batch in flight at a time.
// Here each thread copies its next vector sets into its own shared-memory
// slots with cp.async (16-byte LDGSTS, no register cost), S stages ahead,
// and computes from the oldest stage; a thread reads only slots it wrote
// itself, so cp.async.wait_group is the only synchronisation.  The chunks,
// the per-thread element order, the fp32 sums and the fixed reduction are
// those of gram_partials_kernel (gram_impl.cuh), so the partials are
// bit-identical to it.
#pragma once

#include "gram_impl.cuh"

namespace bkmoo {

#ifndef BKMOO_GRAM_PREFETCH_MIN_K
#define BKMOO_GRAM_PREFETCH_MIN_K 12
#endif
constexpr int kPrefetchMinK = BKMOO_GRAM_PREFETCH_MIN_K;
constexpr int kPrefetchStages = 3;

__host__ __device__ constexpr int prefetch_smem_bytes(int K) {
  return kPrefetchStages * K * kThreads * 16;
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(smem_dst)),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// The bucket of a CTA's current chunk with its chunk and element bounds in
// registers.  A CTA's next chunk lies gridDim.x chunks on, with one CTA per
// SM often many small buckets away; a plain search then costs several
// dependent global loads on the path of the copies this kernel issues.
// seek() guesses the bucket from the current bucket's chunk count (exact
// when the buckets have equal chunk counts, as one tensor cut into equal
// buckets does) and loads the guess's four bounds in one round trip; a wrong
// guess falls back to find_bucket.  (The other kernels keep the plain
// search: these registers would cost them occupancy.)
struct BucketTracker {
  int64_t b, c0, c1, o0, o1;
  __device__ void load(const PlanView& v, int64_t bb) {
    b = bb;
    c0 = v.chunk_prefix[bb];
    c1 = v.chunk_prefix[bb + 1];
    o0 = v.offsets[bb];
    o1 = v.offsets[bb + 1];
  }
  __device__ void init(const PlanView& v) { load(v, v.b_lo < v.n_buckets ? v.b_lo : 0); }
  __device__ void seek(const PlanView& v, int64_t w) {
    if (c0 <= w && w < c1) return;
    if (c0 <= w) {
      const int64_t g = b + (w - c0) / (c1 - c0);
      if (g < v.n_buckets) {
        const int64_t g0 = v.chunk_prefix[g], g1 = v.chunk_prefix[g + 1];
        const int64_t h0 = v.offsets[g], h1 = v.offsets[g + 1];
        if (g0 <= w && w < g1) {
          b = g;
          c0 = g0;
          c1 = g1;
          o0 = h0;
          o1 = h1;
          return;
        }
      }
    }
    load(v, find_bucket(v.chunk_prefix, v.n_buckets, w, b));
  }
  // chunk w's element range [s, e) and vector range [vs, vs + nv * EPV)
  template <int EPV>
  __device__ void range(const PlanView& v, int64_t w, int64_t* s, int64_t* e, int64_t* vs,
                        int* nv) const {
    *s = o0 + (w - c0) * v.chunk_elems;
    *e = min(*s + v.chunk_elems, o1);
    int64_t a = (*s + EPV - 1) / EPV * EPV;
    if (a > *e) a = *e;
    int64_t z = *e / EPV * EPV;
    if (z < a) z = a;
    *vs = a;
    *nv = (int)((z - a) / EPV);
  }
};

// This thread's sequence of 16-byte positions: chunk w = c_lo + blockIdx.x,
// + gridDim.x, ...; within a chunk the vectors i = t, t + 256, ... < nv.
// On entering a chunk the cursor also issues the loads of the bounds of the
// bucket its next chunk is guessed to fall in (from the current bucket's
// chunk count), so that the next move finds them in registers instead of
// waiting a round trip on the path of the copies; a wrong guess falls back
// to BucketTracker::seek.
template <int EPV>
struct VecCursor {
  BucketTracker bt;
  int64_t w, vs;
  int nv, i;
  int64_t nb, n0, n1, p0, p1;   // preloaded guess for the next chunk (nb < 0: none)
  __device__ void preload(const PlanView& v) {
    nb = -1;
    const int64_t wn = w + gridDim.x;
    if (wn < bt.c1 || wn >= v.c_hi) return;
    const int64_t g = bt.b + (wn - bt.c0) / (bt.c1 - bt.c0);
    if (g >= v.n_buckets) return;
    nb = g;
    n0 = v.chunk_prefix[g];
    n1 = v.chunk_prefix[g + 1];
    p0 = v.offsets[g];
    p1 = v.offsets[g + 1];
  }
  __device__ void move(const PlanView& v) {
    if (!(bt.c0 <= w && w < bt.c1)) {
      if (nb >= 0 && n0 <= w && w < n1) {
        bt.b = nb;
        bt.c0 = n0;
        bt.c1 = n1;
        bt.o0 = p0;
        bt.o1 = p1;
      } else {
        bt.seek(v, w);
      }
    }
    preload(v);
  }
  __device__ void settle(const PlanView& v) {
    while (w < v.c_hi) {
      move(v);
      int64_t s, e;
      bt.range<EPV>(v, w, &s, &e, &vs, &nv);
      if (i < nv) return;
      w += gridDim.x;
      i = threadIdx.x;
    }
  }
  __device__ void begin(const PlanView& v) {
    w = v.c_lo + blockIdx.x;
    bt.init(v);
    nb = -1;
    i = threadIdx.x;
    settle(v);
  }
  __device__ bool more(const PlanView& v) const { return w < v.c_hi; }
  __device__ void next(const PlanView& v) {
    i += kThreads;
    if (i >= nv) {
      w += gridDim.x;
      i = threadIdx.x;
      settle(v);
    }
  }
};

template <int K, int DT>
__global__ void __launch_bounds__(kThreads) gram_prefetch_kernel(const GradPtrs g,
                                                                 const PlanView v) {
  constexpr int P = tri(K);
  constexpr int EPV = elems_per_vec(DT);
  constexpr int IB = 16 / EPV;
  constexpr int S = kPrefetchStages;
  extern __shared__ __align__(16) unsigned char pf_smem[];
  __shared__ float red[kWarps][P];
  // slot (stage s, gradient k) of thread t
  uint4* slots = reinterpret_cast<uint4*>(pf_smem);
  auto slot = [&](int s, int k) -> uint4* { return slots + ((s * K + k) * kThreads + threadIdx.x); };

  if (!header_ok(v)) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
    return;
  }
  // the producer cursor runs S - 1 positions ahead of the consumer
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
    cp_async_commit();   // empty groups keep the group count in step
    ++issued;
  };
#pragma unroll
  for (int j = 0; j < S - 1; ++j) issue();

  int consumed = 0;
  BucketTracker ct;
  ct.init(v);
  for (int64_t w = v.c_lo + blockIdx.x; w < v.c_hi; w += gridDim.x) {
    // the producer is usually still on this chunk: take its bucket bounds
    if (pc.w == w) ct = pc.bt;
    else ct.seek(v, w);
    int64_t s0, e, vs;
    int nv;
    ct.range<EPV>(v, w, &s0, &e, &vs, &nv);
    const int64_t ve = vs + (int64_t)nv * EPV;

    float acc[P];
#pragma unroll
    for (int p = 0; p < P; ++p) acc[p] = 0.0f;
    for (int i = threadIdx.x; i < nv; i += kThreads) {
      issue();                       // position consumed + S - 1
      cp_async_wait<S - 1>();        // the oldest group (this position) has landed
      const int s = consumed % S;
      uint4 r[K];
#pragma unroll
      for (int k = 0; k < K; ++k) r[k] = *slot(s, k);
      gram_accumulate<K, DT>(acc, r);
      ++consumed;
    }
    const int nh = (int)(vs - s0), nt = (int)(e - ve);
    if ((int)threadIdx.x < nh + nt) {
      const int64_t idx = (int)threadIdx.x < nh ? s0 + threadIdx.x : ve + (threadIdx.x - nh);
      gram_accumulate_scalar<K, DT>(acc, g, idx);
    }
    cta_reduce_store<P>(acc, red, v.partials + w * P);
  }
  cp_async_wait<0>();
}

#define BKMOO_GRAM_PREFETCH_TABLE(DT)                                                       \
  static const void* const kGramPrefetchTable[kMaxK] = {                                    \
      (const void*)gram_prefetch_kernel<1, DT>,  (const void*)gram_prefetch_kernel<2, DT>,  \
      (const void*)gram_prefetch_kernel<3, DT>,  (const void*)gram_prefetch_kernel<4, DT>,  \
      (const void*)gram_prefetch_kernel<5, DT>,  (const void*)gram_prefetch_kernel<6, DT>,  \
      (const void*)gram_prefetch_kernel<7, DT>,  (const void*)gram_prefetch_kernel<8, DT>,  \
      (const void*)gram_prefetch_kernel<9, DT>,  (const void*)gram_prefetch_kernel<10, DT>, \
      (const void*)gram_prefetch_kernel<11, DT>, (const void*)gram_prefetch_kernel<12, DT>, \
      (const void*)gram_prefetch_kernel<13, DT>, (const void*)gram_prefetch_kernel<14, DT>, \
      (const void*)gram_prefetch_kernel<15, DT>, (const void*)gram_prefetch_kernel<16, DT>}

}  // namespace bkmoo
