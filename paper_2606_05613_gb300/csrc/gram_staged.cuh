// Gram pass, shared-memory-staged variant: the same per-chunk partial Gram
// matrices as gram_partials_kernel (gram_impl.cuh), with the gradients
// brought into shared memory by the bulk-copy (TMA) engine instead of by
// the computing threads.
//
// Why: the K(K+1)/2 fp32 accumulators of a thread grow with K (136 at
// K = 16), which caps the register-file occupancy at 8 warps per SM; with
// the loads issued by those same warps, each warp alternates between
// waiting for HBM and computing, and the SM cannot keep enough bytes in
// flight.  Here the bulk-copy engine keeps NS - 1 stages in flight per CTA
// (a ring of NS shared-memory stages with a full/empty mbarrier pair per
// stage) while the 8 warps compute from shared memory, so the HBM stream
// does not wait for the arithmetic.  Thread 0 issues the copies (one
// 4 KiB bulk copy per gradient per stage), NS - 1 stages ahead.
//
// CTA = 8 warps (256 threads; a separate producer warp would make 9 and cut
// the register budget per thread to 168), one CTA per SM, persistent over
// the chunks w = blockIdx.x, blockIdx.x + gridDim.x, ...
// A stage holds 4 KiB of each of the K gradients (1024 fp32 / 2048 bf16
// elements); a chunk (kVecPerThread x 256 vectors of 16 bytes per
// gradient) is 16 stages.  Consumer thread t takes the 32-bit words
// t, t + 256, t + 512, t + 768 of each stage (bank-conflict-free), i.e. at
// most 64 fp32 or 128 bf16 elements per chunk, summed in fp32; the CTA then
// reduces the triangle with the fixed warp-shuffle tree (fp32) and the fixed
// sum over the 8 warps (fp64), as in gram_impl.cuh.  Head and tail elements
// of a chunk outside its 16-byte-aligned vector range are read directly
// from global memory.  No atomics: deterministic.
//
// Every mbarrier wait is bounded (about one second of globaltimer): on
// expiry the thread records BKMOO_ERR_TIMEOUT in the workspace status word,
// and every thread then stops waiting and reading shared memory but keeps to
// the common loop (so the CTA barriers stay matched); thread 0 finally waits
// (bounded again) for the copies it issued, so no copy lands in shared
// memory of a finished CTA.
#pragma once

#include "gram_impl.cuh"

namespace bkmoo {

constexpr int kStagedConsumers = kThreads;              // 8 warps
constexpr int kStagedThreads = kStagedConsumers;
constexpr int kStageBytesPerGrad = 4096;
constexpr int kStageVecs = kStageBytesPerGrad / 16;     // 256 vectors
constexpr uint64_t kStagedWaitNs = 1000000000ull;

// Stages in the ring: about 192 KiB of shared memory, 2 to 8 stages.
__host__ __device__ constexpr int staged_stages(int K) {
  return (196608 / (K * kStageBytesPerGrad)) < 2   ? 2
         : (196608 / (K * kStageBytesPerGrad)) > 8 ? 8
                                                    : 196608 / (K * kStageBytesPerGrad);
}
__host__ __device__ constexpr int staged_smem_bytes(int K) {
  return staged_stages(K) * K * kStageBytesPerGrad + 2 * 8 * staged_stages(K);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t staged_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait for the phase of the given parity to complete; false on
// expiry, or once the wait has lasted over a millisecond and an error is
// recorded in the workspace status word.  A normal wait touches only the
// mbarrier (and the timer every 64 polls), never global memory: hundreds of
// warps polling one global word would contend in its L2 slice.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, const WsHeader* h) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = staged_ns();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 63u) == 0) {
      const uint64_t dt = staged_ns() - t0;
      if (dt > kStagedWaitNs) return false;
      if (dt > 1000000ull && *(volatile const int32_t*)&h->status != 0) return false;
    }
  }
}
// Bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// The vector range [vs, ve) and head/tail of chunk w (as in gram_impl.cuh).
struct ChunkRange {
  int64_t s, e, vs, ve;
  int nv;
};
template <int EPV>
__device__ __forceinline__ ChunkRange chunk_range(const PlanView& v, int64_t b, int64_t w) {
  ChunkRange c;
  const int64_t be = v.offsets[b + 1];
  c.s = v.offsets[b] + (w - v.chunk_prefix[b]) * v.chunk_elems;
  c.e = min(c.s + v.chunk_elems, be);
  c.vs = (c.s + EPV - 1) / EPV * EPV;
  if (c.vs > c.e) c.vs = c.e;
  c.ve = c.e / EPV * EPV;
  if (c.ve < c.vs) c.ve = c.vs;
  c.nv = (int)((c.ve - c.vs) / EPV);
  return c;
}

// Cursor over the (chunk, stage) sequence of one CTA: the chunks
// w = c_lo + blockIdx.x, + gridDim.x, ... and the stages of each chunk's
// vector range (chunks without whole vectors have none).
template <int EPV>
struct StageCursor {
  int64_t w, b;
  ChunkRange c;
  int st;
  __device__ void begin(const PlanView& v) {
    w = v.c_lo + blockIdx.x;
    b = v.b_lo;
    st = 0;
    settle(v);
  }
  // move to the first stage at or after (w, st)
  __device__ void settle(const PlanView& v) {
    while (w < v.c_hi) {
      b = find_bucket(v.chunk_prefix, v.n_buckets, w, b);
      c = chunk_range<EPV>(v, b, w);
      if (st * kStageVecs < c.nv) return;
      w += gridDim.x;
      st = 0;
    }
  }
  __device__ bool more(const PlanView& v) const { return w < v.c_hi; }
  __device__ void next(const PlanView& v) {
    ++st;
    settle(v);
  }
};

template <int K, int DT>
__global__ void __launch_bounds__(kStagedThreads, 1)
    gram_staged_kernel(const GradPtrs g, const PlanView v) {
  constexpr int P = tri(K);
  constexpr int EPV = elems_per_vec(DT);
  constexpr int NS = staged_stages(K);
  constexpr int STAGE = K * kStageBytesPerGrad;
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + NS * STAGE);
  uint64_t* empty = full + NS;
  __shared__ float red[kWarps][P];

  if (!header_ok(v)) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(v.hdr, BKMOO_ERR_WORKSPACE);
    return;
  }
  const int t = threadIdx.x;
  const int warp = t >> 5, lane = t & 31;
  if (t == 0) {
    for (int i = 0; i < NS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  // Thread 0 issues the bulk copies, NS - 1 stages ahead of consumption:
  // before it issues stage j into slot j % NS it waits until every warp has
  // released stage j - NS from that slot.
  StageCursor<EPV> pc;
  uint32_t pit = 0;   // stages issued (thread 0)
  bool dead = false;  // an error was recorded: stop waiting and reading
  auto issue = [&]() {
    const int slot = (int)(pit % NS);
    if (pit >= (uint32_t)NS && !mbar_wait(&empty[slot], ((pit / NS) + 1) & 1, v.hdr)) {
      record_error(v.hdr, BKMOO_ERR_TIMEOUT);
      dead = true;
      return;
    }
    const int nvs = min(kStageVecs, pc.c.nv - pc.st * kStageVecs);
    const uint32_t bytes = (uint32_t)nvs * 16u;
    mbar_arrive_expect_tx(&full[slot], bytes * K);
    unsigned char* dst = smem + slot * STAGE;
    const int64_t el = pc.c.vs + (int64_t)pc.st * kStageVecs * EPV;
#pragma unroll
    for (int k = 0; k < K; ++k)
      bulk_g2s(dst + k * kStageBytesPerGrad, static_cast<const char*>(g.p[k]) + el * (16 / EPV),
               bytes, &full[slot]);
    ++pit;
    pc.next(v);
  };
  if (t == 0) {
    pc.begin(v);
    for (int i = 0; i < NS - 1 && pc.more(v) && !dead; ++i) issue();
  }

  uint32_t it = 0;    // stages consumed
  int64_t b = v.b_lo;
  for (int64_t w = v.c_lo + blockIdx.x; w < v.c_hi; w += gridDim.x) {
    b = find_bucket(v.chunk_prefix, v.n_buckets, w, b);
    const ChunkRange c = chunk_range<EPV>(v, b, w);
    float acc[P];
#pragma unroll
    for (int p = 0; p < P; ++p) acc[p] = 0.0f;
    for (int st = 0; st * kStageVecs < c.nv; ++st, ++it) {
      if (t == 0 && !dead && pc.more(v)) issue();
      const int slot = (int)(it % NS);
      if (!dead && !mbar_wait(&full[slot], (it / NS) & 1, v.hdr)) {
        record_error(v.hdr, BKMOO_ERR_TIMEOUT);
        dead = true;
      }
      const int nwords = dead ? 0 : min(kStageVecs, c.nv - st * kStageVecs) * 4;
      const unsigned char* src = smem + slot * STAGE;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int wd = t + j * kStagedConsumers;
        if (wd < nwords) {
          uint32_t x[K];
#pragma unroll
          for (int k = 0; k < K; ++k)
            x[k] = reinterpret_cast<const uint32_t*>(src + k * kStageBytesPerGrad)[wd];
          if (DT == BKMOO_F32) {
            int p = 0;
#pragma unroll
            for (int i = 0; i < K; ++i)
#pragma unroll
              for (int jj = i; jj < K; ++jj) {
                acc[p] = fmaf(__uint_as_float(x[i]), __uint_as_float(x[jj]), acc[p]);
                ++p;
              }
          } else {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              int p = 0;
#pragma unroll
              for (int i = 0; i < K; ++i) {
                const float xi = h ? __uint_as_float(x[i] & 0xffff0000u)
                                   : __uint_as_float(x[i] << 16);
#pragma unroll
                for (int jj = i; jj < K; ++jj) {
                  const float xj = h ? __uint_as_float(x[jj] & 0xffff0000u)
                                     : __uint_as_float(x[jj] << 16);
                  acc[p] = fmaf(xi, xj, acc[p]);
                  ++p;
                }
              }
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[slot]);
    }
    const int nh = (int)(c.vs - c.s), nt = (int)(c.e - c.ve);
    if (t < nh + nt) {
      const int64_t idx = t < nh ? c.s + t : c.ve + (t - nh);
      gram_accumulate_scalar<K, DT>(acc, g, idx);
    }
    // fixed-order reduction over the warps (as cta_reduce_store)
#pragma unroll
    for (int p = 0; p < P; ++p) {
      float x = acc[p];
      x += __shfl_down_sync(0xffffffffu, x, 16);
      x += __shfl_down_sync(0xffffffffu, x, 8);
      x += __shfl_down_sync(0xffffffffu, x, 4);
      x += __shfl_down_sync(0xffffffffu, x, 2);
      x += __shfl_down_sync(0xffffffffu, x, 1);
      if (lane == 0) red[warp][p] = x;
    }
    __syncthreads();
    for (int p = t; p < P; p += kStagedConsumers) {
      double s = 0.0;
#pragma unroll
      for (int q = 0; q < kWarps; ++q) s += (double)red[q][p];
      v.partials[w * P + p] = s;
    }
    __syncthreads();
  }
  if (t == 0 && dead) {
    // wait (bounded, ignoring the status word) for the copies this CTA may
    // still have in flight: at most the last NS stages issued
    for (uint32_t j = pit > (uint32_t)NS ? pit - NS : 0; j < pit; ++j) {
      const uint64_t t0 = staged_ns();
      while (!mbar_try_wait(&full[j % NS], (j / NS) & 1) && staged_ns() - t0 <= kStagedWaitNs) {
      }
    }
  }
}

#define BKMOO_GRAM_STAGED_TABLE(DT)                                                     \
  static const void* const kGramStagedTable[kMaxK] = {                                  \
      (const void*)gram_staged_kernel<1, DT>,  (const void*)gram_staged_kernel<2, DT>,  \
      (const void*)gram_staged_kernel<3, DT>,  (const void*)gram_staged_kernel<4, DT>,  \
      (const void*)gram_staged_kernel<5, DT>,  (const void*)gram_staged_kernel<6, DT>,  \
      (const void*)gram_staged_kernel<7, DT>,  (const void*)gram_staged_kernel<8, DT>,  \
      (const void*)gram_staged_kernel<9, DT>,  (const void*)gram_staged_kernel<10, DT>, \
      (const void*)gram_staged_kernel<11, DT>, (const void*)gram_staged_kernel<12, DT>, \
      (const void*)gram_staged_kernel<13, DT>, (const void*)gram_staged_kernel<14, DT>, \
      (const void*)gram_staged_kernel<15, DT>, (const void*)gram_staged_kernel<16, DT>}

}  // namespace bkmoo
