// Internal definitions shared by the translation units of the bkmoo CUDA
// library: workspace layout, kernel argument blocks, 16-byte vector access
// and the chunk -> bucket lookup.  Not part of the C ABI (include/bkmoo.h).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "bkmoo.h"

namespace bkmoo {

constexpr int kMaxK = 16;
// Largest K the fused persistent kernel is built for: above it the per-thread
// streaming state (K(K+1)/2 accumulators, K vectors in flight) no longer fits
// the register file, and the three-pass path runs instead.
constexpr int kFusedMaxK = 8;
constexpr int kThreads = 256;              // CTA size of the streaming kernels
constexpr int kWarps = kThreads / 32;
constexpr int kVecPerThread = 16;          // 16-byte vectors per thread per Gram chunk
constexpr uint32_t kMagic = 0x4f4d4b42u;   // "BKMO"
constexpr int kSolveWarpsPerBlock = 4;
constexpr int kFusedMaxCtas = 2048;        // upper bound of the fused grid
// Fused kernel: 11 streaming warps and one solver warp per CTA (12 warps:
// registers are allocated to warps in groups of four, so 9 warps would cost
// as many registers as 12); each group of CTAs keeps the CTA partials of its
// last kFusedRing buckets in a ring.
constexpr int kFusedStreamWarps = 11;
constexpr int kFusedThreads = 32 * (kFusedStreamWarps + 1);
constexpr int kFusedRing = 4;
// cp.async stages per streaming lane of the fused kernel: about 14 K-vector
// sets in flight per lane (~80 KB per SM with 11 streaming warps).
__host__ __device__ constexpr int fused_stages(int K) {
  return K <= 1 ? 12 : K == 2 ? 8 : K == 3 ? 6 : K == 4 ? 5 : K <= 6 ? 4 : 3;
}
__host__ __device__ constexpr int fused_smem_bytes(int K) {
  return fused_stages(K) * K * 16 * 32 * kFusedStreamWarps;
}
// A bucket with more than kGroupMinChunks chunks has its chunk partials
// pre-reduced in groups of kGroupChunks (group_reduce_kernel, solve.cu)
// before the per-bucket reduction reads them: one warp would otherwise read
// every partial of a huge bucket (the one-bucket "global" variant) alone.
constexpr int64_t kGroupChunks = 512;
constexpr int64_t kGroupMinChunks = 1024;

__host__ __device__ constexpr int tri(int K) { return K * (K + 1) / 2; }
__host__ __device__ constexpr int elems_per_vec(int dtype) { return dtype == BKMOO_F32 ? 4 : 8; }
__host__ __device__ constexpr int64_t chunk_elems(int dtype) {
  return (int64_t)kThreads * kVecPerThread * elems_per_vec(dtype);
}

// First 256 bytes of every workspace.
struct WsHeader {
  uint32_t magic;
  int32_t K;
  int32_t in_dtype;
  int32_t status;        // device-side error word: BKMOO_OK or the first error
  int64_t n_buckets;
  int64_t n_elems;
  int64_t n_chunks;
  int64_t chunk_elems;
  uint64_t plan_hash;
  int64_t reserved[25];
};
static_assert(sizeof(WsHeader) == 256, "header is one 256-byte block");

// Byte offsets of the workspace regions (identical on host and device).
struct WsLayout {
  size_t offsets;        // int64 [B + 1]   bucket boundaries (elements)
  size_t chunk_prefix;   // int64 [B + 1]   first Gram chunk of each bucket
  size_t partials;       // double [n_chunks][P] per-chunk Gram partials
  size_t beta;           // float [B][K]    coefficients of the last resolve
  size_t total;          // end of the regions above
  // fused path only (bkmoo_resolve with BKMOO_FLAG_FUSED):
  size_t arrive;         // int32 [B]      CTAs of bucket b's group done with its Gram
  size_t ready;          // int32 [B + 1]  1 once beta of bucket b is written;
                         //                [B] counts the buckets published
  size_t ring;           // double [kFusedRing][2 kFusedMaxCtas][P] CTA partials
  size_t total_fused;
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Host-side plan helpers shared by every entry point.
// Offsets start at 0 and increase strictly (no empty bucket).
inline bool offsets_ok(const int64_t* off, int64_t B) {
  if (!off || B < 0 || off[0] != 0) return false;
  for (int64_t b = 0; b < B; ++b)
    if (off[b + 1] <= off[b]) return false;
  return true;
}

// Gram chunks of a plan: each bucket is cut into chunks of ch elements, the
// last one short.
inline int64_t count_chunks(const int64_t* off, int64_t B, int64_t ch) {
  int64_t n = 0;
  for (int64_t b = 0; b < B; ++b) n += (off[b + 1] - off[b] + ch - 1) / ch;
  return n;
}

// FNV-1a over the 64-bit words that define a plan (K, dtype, B, offsets);
// kept in the workspace header and checked by every kernel.
inline uint64_t plan_hash(int32_t K, int32_t dt, const int64_t* off, int64_t B) {
  uint64_t h = 0xcbf29ce484222325ull;
  auto mix = [&h](uint64_t x) {
    h ^= x;
    h *= 0x100000001b3ull;
  };
  mix((uint64_t)K);
  mix((uint64_t)dt);
  mix((uint64_t)B);
  for (int64_t b = 0; b <= B; ++b) mix((uint64_t)off[b]);
  return h;
}

__host__ __device__ inline WsLayout ws_layout(int K, int64_t B, int64_t n_chunks) {
  WsLayout L;
  size_t at = sizeof(WsHeader);
  L.offsets = at;
  at = align256(at + sizeof(int64_t) * (size_t)(B + 1));
  L.chunk_prefix = at;
  at = align256(at + sizeof(int64_t) * (size_t)(B + 1));
  L.partials = at;
  at = align256(at + sizeof(double) * (size_t)n_chunks * (size_t)tri(K));
  L.beta = at;
  at = align256(at + sizeof(float) * (size_t)B * (size_t)K);
  L.total = at;
  L.arrive = at;
  at = align256(at + sizeof(int32_t) * (size_t)B);
  L.ready = at;
  at = align256(at + sizeof(int32_t) * (size_t)(B + 1));
  L.ring = at;
  at = align256(at + sizeof(double) * kFusedRing * 2 * (size_t)kFusedMaxCtas * (size_t)tri(K));
  L.total_fused = at;
  return L;
}

struct GradPtrs {
  const void* p[kMaxK];
};

// Everything a kernel needs to find its data.
struct PlanView {
  WsHeader* hdr;
  const int64_t* offsets;
  const int64_t* chunk_prefix;
  double* partials;
  float* beta;
  int64_t n_buckets;
  int64_t n_chunks;
  int64_t chunk_elems;
  uint64_t plan_hash;
  int32_t K;
  int32_t in_dtype;
  // The part of the plan one launch works on: chunks [c_lo, c_hi) of buckets
  // [b_lo, b_hi) (the whole plan except in the windowed host-memory path).
  int64_t c_lo, c_hi;
  int64_t b_lo, b_hi;
  int64_t max_chunks;   // most chunks in one bucket of the plan (host-computed)
};

// Whole-plan window of a view whose n_buckets and n_chunks are set.
__host__ __device__ inline void full_window(PlanView& v) {
  v.c_lo = 0;
  v.c_hi = v.n_chunks;
  v.b_lo = 0;
  v.b_hi = v.n_buckets;
}

// The fused path's view: the plan plus the synchronisation arrays.  CTA c
// belongs to group c % n_groups; bucket b is resolved by group b % n_groups.
struct FusedView {
  PlanView v;
  int32_t* arrive;
  int32_t* ready;
  double* ring;          // [n_groups][kFusedRing][group_ctas][P]
  float* out_weights;
  int32_t* out_status;
  int32_t n_groups;
  int32_t group_ctas;    // rows of a ring slot: CTAs of the largest group
  int32_t lookahead;     // buckets a warp's Gram may run ahead of its combination
};

struct SolveParams {
  int32_t rule;
  int32_t max_iter;
  double tol;
  double cagrad_c;
  uint64_t seed;
  uint64_t step;
  uint32_t flags;
};

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

__device__ __forceinline__ bool header_ok(const PlanView& v) {
  const WsHeader* h = v.hdr;
  return h->magic == kMagic && h->plan_hash == v.plan_hash && h->K == v.K &&
         h->in_dtype == v.in_dtype && h->n_buckets == v.n_buckets &&
         h->n_chunks == v.n_chunks;
}

__device__ __forceinline__ void record_error(WsHeader* h, int code) {
  atomicCAS(&h->status, 0, code);
}

// Bucket b with chunk_prefix[b] <= w < chunk_prefix[b+1]; `hint` is tried
// first (chunks of one CTA increase monotonically).
__device__ __forceinline__ int64_t find_bucket(const int64_t* cp, int64_t B, int64_t w,
                                               int64_t hint) {
  if (hint < B && cp[hint] <= w && w < cp[hint + 1]) return hint;
  if (hint + 1 < B && cp[hint + 1] <= w && w < cp[hint + 2]) return hint + 1;
  int64_t lo = 0, hi = B;
  while (hi - lo > 1) {
    int64_t mid = (lo + hi) >> 1;
    if (cp[mid] <= w) lo = mid;
    else hi = mid;
  }
  return lo;
}

// 16-byte loads.  `nc`: read-only path, no L1 allocation (streams that are
// read once by this kernel).  `cs`: coherent, evict-first (combine, which
// may write in place over one of the inputs).
__device__ __forceinline__ uint4 ld16_nc(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}
__device__ __forceinline__ uint4 ld16_cs(const void* p) {
  uint4 r;
  asm volatile("ld.global.cs.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}
__device__ __forceinline__ void st16_cs(void* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ void st8_cs(void* p, uint2 v) {
  asm volatile("st.global.cs.v2.u32 [%0], {%1,%2};" ::"l"(p), "r"(v.x), "r"(v.y) : "memory");
}

__device__ __forceinline__ uint32_t word(const uint4& r, int i) {
  return i == 0 ? r.x : i == 1 ? r.y : i == 2 ? r.z : r.w;
}

// Element e of a 16-byte vector as fp32 (bf16 widened exactly).
template <int DT>
__device__ __forceinline__ float vec_elem(const uint4& r, int e) {
  if (DT == BKMOO_F32) return __uint_as_float(word(r, e));
  const uint32_t w = word(r, e >> 1);
  return (e & 1) ? __uint_as_float(w & 0xffff0000u) : __uint_as_float(w << 16);
}

template <int DT>
__device__ __forceinline__ float load_scalar(const void* base, int64_t i) {
  if (DT == BKMOO_F32) return static_cast<const float*>(base)[i];
  const uint16_t h = static_cast<const uint16_t*>(base)[i];
  return __uint_as_float((uint32_t)h << 16);
}

// ---------------------------------------------------------------------------
// Kernel tables and launchers
// ---------------------------------------------------------------------------

// Gram-pass kernels, signature (GradPtrs, PlanView); gram_f32.cu / gram_bf16.cu.
const void* gram_partials_fn_f32(int K);
const void* gram_partials_fn_bf16(int K);

// Gram-pass kernels with a per-thread shared-memory prefetch (same signature,
// kThreads threads, gram_prefetch_smem(K) bytes of dynamic shared memory) for
// K >= gram_prefetch_min_k(); nullptr below; gram_prefetch.cu.
const void* gram_prefetch_fn(int K, int dt);
int gram_prefetch_smem(int K);
int gram_prefetch_min_k();

// Combine kernels with a per-thread shared-memory prefetch (same signature,
// combine_prefetch_smem(K) bytes of dynamic shared memory), every K;
// combine_prefetch.cu, combine_prefetch_k9_16.cu.  Measured faster than
// combine_kernel on GB300 (K = 2..8: 2-6.5 %).
#ifndef BKMOO_COMBINE_PREFETCH
#define BKMOO_COMBINE_PREFETCH 1
#endif
const void* combine_prefetch_fn(int K, int dti, int dto);
const void* combine_prefetch_fn_k9_16(int K, int dti, int dto);
int combine_prefetch_smem(int K);

// Combine kernels, signature (GradPtrs, PlanView, void* out); combine_*.cu.
const void* combine_fn_f32(int K, int dtype_out);
const void* combine_fn_bf16(int K, int dtype_out);

// Fused kernels, signature (GradPtrs, FusedView, SolveParams, void* out); fused_*.cu.
const void* fused_fn_f32_k1_4(int K, int dtype_out);
const void* fused_fn_f32_k5_6(int K, int dtype_out);
const void* fused_fn_f32_k7_8(int K, int dtype_out);
const void* fused_fn_bf16_k1_4(int K, int dtype_out);
const void* fused_fn_bf16_k5_6(int K, int dtype_out);
const void* fused_fn_bf16_k7_8(int K, int dtype_out);

// Cluster-per-bucket fused kernels (fused_cluster.cu), K <= kClusterMaxK,
// signature (GradPtrs, PlanView, SolveParams, float* out_weights,
// int32_t* out_status, void* out, int head), clusters of kClusterCtas CTAs
// of kClusterThreads threads (15 streaming warps and one solver warp) with
// fused_cluster_smem(K) bytes of dynamic shared memory.
constexpr int kClusterMaxK = 4;
constexpr int kClusterCtas = 8;
constexpr int kClusterStreamWarps = 15;
constexpr int kClusterStreamThreads = 32 * kClusterStreamWarps;
constexpr int kClusterThreads = kClusterStreamThreads + 32;
const void* fused_cluster_fn(int K, int dti, int dto);
int fused_cluster_smem(int K);

// solve.cu
cudaError_t launch_solve(const PlanView& v, const SolveParams& p, float* out_weights,
                         int32_t* out_status, cudaStream_t s);
cudaError_t launch_gram_finalize(const PlanView& v, double* out_gram, cudaStream_t s);
// The fp64 division / square-root helpers of the fast solvers, element-wise
// (self-test of their accuracy against the correctly rounded operations).
cudaError_t launch_selftest_fp64(int op, const double* a, const double* b, double* out, int64_t n,
                                 cudaStream_t s);
// After a Gram pass over the view's window: the group pre-reduction of its
// large buckets (a no-op when no bucket has more than kGroupMinChunks chunks).
cudaError_t launch_group_reduce(const PlanView& v, cudaStream_t s);

}  // namespace bkmoo
