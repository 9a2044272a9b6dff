// Host side of the C ABI (include/bkmoo.h): argument checks, the bucket plan,
// the workspace image, the launch sequence Gram -> solve -> combine on the
// caller's stream (whole plan, a bucket range, or windows of buckets staged
// from host memory), and the fused persistent launch.  Nothing here
// allocates device memory (the host path creates two copy streams and a few
// events per call).
#include <cuda_runtime.h>

#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <utility>
#include <vector>

#include "common.cuh"

using namespace bkmoo;

namespace {

constexpr int32_t kVersion = 200;  // 0.2.0: bucket-range and host-memory entry points

bool dtype_ok(int32_t dt) { return dt == BKMOO_F32 || dt == BKMOO_BF16; }
int elem_bytes(int32_t dt) { return dt == BKMOO_F32 ? 4 : 2; }
bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p & (a - 1)) == 0; }

struct LaunchCache {
  std::mutex mu;
  std::map<int, int> sms;
  std::map<std::pair<int, const void*>, int> occ;
};
LaunchCache& cache() {
  static LaunchCache c;
  return c;
}

// Resident CTAs of `fn` on the current device times its SM count.  A kernel
// with dynamic shared memory gets its limit raised to that size once (the
// default limit of 48 KiB counts static and dynamic shared memory together).
cudaError_t persistent_grid(const void* fn, int threads, int* grid, int dyn_smem = 0) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  LaunchCache& c = cache();
  std::lock_guard<std::mutex> lk(c.mu);
  auto it = c.sms.find(dev);
  if (it == c.sms.end()) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    it = c.sms.emplace(dev, n).first;
  }
  auto key = std::make_pair(dev, fn);
  auto jt = c.occ.find(key);
  if (jt == c.occ.end()) {
    int n = 0;
    if (dyn_smem > 0) {
      e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn_smem);
      if (e != cudaSuccess) return e;
    }
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, threads, dyn_smem);
    if (e != cudaSuccess) return e;
    jt = c.occ.emplace(key, n < 1 ? 1 : n).first;
  }
  *grid = it->second * jt->second;
  return cudaSuccess;
}

const void* gram_fn(int K, int dt) {
  return dt == BKMOO_F32 ? gram_partials_fn_f32(K) : gram_partials_fn_bf16(K);
}
const void* combine_fn(int K, int dti, int dto) {
  return dti == BKMOO_F32 ? combine_fn_f32(K, dto) : combine_fn_bf16(K, dto);
}
const void* fused_fn(int K, int dti, int dto) {
  if (dti == BKMOO_F32)
    return K <= 4 ? fused_fn_f32_k1_4(K, dto)
                  : (K <= 6 ? fused_fn_f32_k5_6(K, dto) : fused_fn_f32_k7_8(K, dto));
  return K <= 4 ? fused_fn_bf16_k1_4(K, dto)
                : (K <= 6 ? fused_fn_bf16_k5_6(K, dto) : fused_fn_bf16_k7_8(K, dto));
}

// Fused-path sizing.  The bytes that pass through L2 between a bucket's Gram
// read and its re-read are about (lookahead + 1) buckets per group, so the
// group count is the budget over that (at least 1, at most one group per 4
// CTAs and one per bucket).  The budget is a fraction of L2 (3/4: measured
// re-reads of more than about 76 MB of 126 MB fall to HBM speed on this
// part, but a lookahead of one bucket and this budget measured fastest).
// BKMOO_FUSED_L2_BUDGET (bytes) and BKMOO_FUSED_LOOKAHEAD (buckets) override
// the defaults.
struct FusedShape {
  int n_groups;
  int lookahead;
};
FusedShape fused_shape(int grid, int64_t n_buckets, double bucket_bytes, int l2_bytes) {
  double budget = 0.75 * (double)l2_bytes;
  int lookahead = 1;
  if (const char* e = std::getenv("BKMOO_FUSED_L2_BUDGET")) {
    const double x = std::atof(e);
    if (x > 0) budget = x;
  }
  if (const char* e = std::getenv("BKMOO_FUSED_LOOKAHEAD")) {
    const int x = std::atoi(e);
    if (x >= 0 && x <= kFusedRing - 2) lookahead = x;
  }
  double ng = budget / ((lookahead + 1) * (bucket_bytes > 1.0 ? bucket_bytes : 1.0));
  int64_t n = (int64_t)ng;
  const int64_t cap = grid / 4 > 0 ? grid / 4 : 1;
  if (n > cap) n = cap;
  if (n > n_buckets) n = n_buckets;
  if (n < 1) n = 1;
  return FusedShape{(int)n, lookahead};
}

// The fused path: one cooperative (co-resident) launch of kFusedThreads per
// CTA, one CTA per SM.
int launch_fused(const GradPtrs& g, const PlanView& v, const SolveParams& sp, void* ws,
                 float* out_weights, int32_t* out_status, void* out, int dto,
                 double bucket_bytes_max, cudaStream_t s) {
  const WsLayout L = ws_layout(v.K, v.n_buckets, v.n_chunks);
  char* base = static_cast<char*>(ws);
  if (cudaMemsetAsync(&v.hdr->status, 0, sizeof(int32_t), s) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (v.n_buckets == 0) return BKMOO_OK;
  if (cudaMemsetAsync(base + L.arrive, 0, L.ring - L.arrive, s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  const void* fn = fused_fn(v.K, v.in_dtype, dto);
  int grid = 0;
  if (persistent_grid(fn, kFusedThreads, &grid, fused_smem_bytes(v.K)) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  if (grid > kFusedMaxCtas) grid = kFusedMaxCtas;
  if (grid < 1) return BKMOO_ERR_CUDA;
  int dev = 0, l2 = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  const FusedShape sh = fused_shape(grid, v.n_buckets, bucket_bytes_max, l2);
  FusedView f;
  f.v = v;
  f.arrive = reinterpret_cast<int32_t*>(base + L.arrive);
  f.ready = reinterpret_cast<int32_t*>(base + L.ready);
  f.ring = reinterpret_cast<double*>(base + L.ring);
  f.out_weights = out_weights;
  f.out_status = out_status;
  f.n_groups = sh.n_groups;
  f.group_ctas = (grid + sh.n_groups - 1) / sh.n_groups;
  f.lookahead = sh.lookahead;
  GradPtrs ga = g;
  SolveParams spa = sp;
  void* outp = out;
  void* args[] = {&ga, &f, &spa, &outp};
  if (cudaLaunchCooperativeKernel(fn, dim3(grid), dim3(kFusedThreads), args,
                                  fused_smem_bytes(v.K), s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

// The cluster-per-bucket fused path: as many clusters of kClusterCtas CTAs
// as can be resident at once, at most one per bucket (clusters never wait
// for one another).  `head`: items per streaming thread of the next
// bucket's Gram read before a combination, to cover the rule's solve
// (environment variable BKMOO_CLUSTER_HEAD overrides it, for tuning).
int launch_fused_cluster(const GradPtrs& g, const PlanView& v, const SolveParams& sp,
                         float* out_weights, int32_t* out_status, void* out, int dto,
                         int64_t smax, cudaStream_t s) {
  if (cudaMemsetAsync(&v.hdr->status, 0, sizeof(int32_t), s) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (v.n_buckets == 0) return BKMOO_OK;
  const void* fn = fused_cluster_fn(v.K, v.in_dtype, dto);
  if (!fn) return BKMOO_ERR_INVALID;
  const int smem = fused_cluster_smem(v.K);
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, int> clusters;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return BKMOO_ERR_CUDA;
  int ncl = 0;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto key = std::make_pair(dev, fn);
    auto it = clusters.find(key);
    if (it == clusters.end()) {
      if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
          cudaSuccess)
        return BKMOO_ERR_CUDA;
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = kClusterCtas;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(kClusterCtas);
      cfg.blockDim = dim3(kClusterThreads);
      cfg.dynamicSmemBytes = (size_t)smem;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) return BKMOO_ERR_CUDA;
      it = clusters.emplace(key, n).first;
    }
    ncl = it->second;
  }
  if (ncl < 1) return BKMOO_ERR_CUDA;
  if ((int64_t)ncl > v.n_buckets) ncl = (int)v.n_buckets;
  // look-ahead: 512 bytes of gradients per streaming thread (32 / K items),
  // or the whole next bucket when it has at most 24 items per thread
  // (measured best on GB300: K = 2 16 items, K = 3 11, K = 4 8-12 at 2 MiB
  // fp32 buckets, the whole bucket at 1 MiB)
  const int64_t eb = elem_bytes(v.in_dtype), epv = 16 / eb;
  const int64_t items = (smax / epv / kClusterCtas + kClusterStreamThreads - 1) / kClusterStreamThreads;
  int64_t h = items <= 24 ? items : 32 / v.K;
  if (h < 2) h = 2;
  int head = (int)h;
  if (const char* e = std::getenv("BKMOO_CLUSTER_HEAD")) {
    const int h = std::atoi(e);
    if (h >= 0) head = h;
  }
  GradPtrs ga = g;
  PlanView va = v;
  SolveParams spa = sp;
  float* ow = out_weights;
  int32_t* os = out_status;
  void* outp = out;
  void* args[] = {&ga, &va, &spa, &ow, &os, &outp, &head};
  if (cudaLaunchKernel(fn, dim3(ncl * kClusterCtas), dim3(kClusterThreads), args, (size_t)smem,
                       s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

// Path of bkmoo_resolve (see bkmoo_resolve_path in bkmoo.h): 0 three
// launches, 1 cluster-per-bucket fused kernel, 2 grid-synchronised fused
// kernel.
int choose_path(int32_t K, int32_t dt, int32_t rule, const int64_t* off, int64_t B,
                uint32_t flags) {
  if (flags & BKMOO_FLAG_THREE_PASS) return 0;
  if (flags & BKMOO_FLAG_FUSED) {
    if (K <= kClusterMaxK && !(flags & BKMOO_FLAG_TEST_WITHHOLD)) return 1;
    return K <= kFusedMaxK ? 2 : 0;
  }
  // measured on GB300 (1e9 elements per language, MGDA, fused / three
  // launches): the cluster kernel is faster for tiny plans, where one
  // launch instead of three is what counts (33 / 43 us), and for K = 2..4
  // when buckets are large enough to amortise each bucket's hand-offs
  // (>= 2 MiB) and small enough that the buckets in flight stay in L2:
  // fp32 K = 2 2.71 / 2.97 ms at 2 MiB, 2.50 / 2.95 at 4 MiB; K = 3 3.43 /
  // 3.95 at 2 MiB; K = 4 4.59 / 5.07 at 2 MiB, 4.74 / 5.06 at 3 MiB; 1 MiB
  // buckets are slower or tie, and K x bucket above 12 MiB (fp32) or
  // outside 6..12 MiB (bf16) ties or loses.  CAGrad, whose solve takes
  // 5.5-7 us, gains only from 8 MiB of fp32 gradients per bucket (K = 4
  // 2 MiB 4.95 / 5.06, K = 2 4 MiB 2.73 / 2.93; K = 2 2 MiB and bf16 lose).
  if (B < 1) return 0;
  if (K <= 2 && B <= 8 && off[B] <= ((int64_t)1 << 22)) return 1;
  if (K < 2 || K > kClusterMaxK) return 0;
  int64_t smax = 0;
  for (int64_t b = 0; b < B; ++b) smax = off[b + 1] - off[b] > smax ? off[b + 1] - off[b] : smax;
  const double mib = 1024.0 * 1024.0;
  const double bytes = (double)smax * elem_bytes(dt), total = bytes * K;
  if (bytes < 2.0 * mib) return 0;
  if (total > 12.0 * mib || (dt != BKMOO_F32 && total < 6.0 * mib)) return 0;
  if (rule == BKMOO_CAGRAD && (dt != BKMOO_F32 || total < 8.0 * mib)) return 0;
  int64_t big = 0;
  for (int64_t b = 0; b < B; ++b)
    if (2 * (off[b + 1] - off[b]) >= smax) big += off[b + 1] - off[b];
  return big * 10 >= off[B] * 9 ? 1 : 0;
}

// Common checks of bkmoo_gram / bkmoo_resolve; fills the plan view.
int prepare(const void* const* grads, int32_t K, int32_t dt, const int64_t* offsets,
            int64_t B, void* ws, size_t ws_bytes, PlanView* v, GradPtrs* g) {
  if (K < 1 || K > kMaxK || !dtype_ok(dt) || !grads || !ws) return BKMOO_ERR_INVALID;
  if (!offsets_ok(offsets, B)) return BKMOO_ERR_INVALID;
  if (!aligned(ws, 256)) return BKMOO_ERR_INVALID;
  for (int k = 0; k < K; ++k)
    if (!grads[k] || !aligned(grads[k], 16)) return BKMOO_ERR_INVALID;
  const int64_t ch = chunk_elems(dt);
  const int64_t nch = count_chunks(offsets, B, ch);
  const WsLayout L = ws_layout(K, B, nch);
  if (ws_bytes < L.total_fused) return BKMOO_ERR_WORKSPACE;
  char* base = static_cast<char*>(ws);
  v->hdr = reinterpret_cast<WsHeader*>(base);
  v->offsets = reinterpret_cast<const int64_t*>(base + L.offsets);
  v->chunk_prefix = reinterpret_cast<const int64_t*>(base + L.chunk_prefix);
  v->partials = reinterpret_cast<double*>(base + L.partials);
  v->beta = reinterpret_cast<float*>(base + L.beta);
  v->n_buckets = B;
  v->n_chunks = nch;
  v->chunk_elems = ch;
  v->plan_hash = plan_hash(K, dt, offsets, B);
  v->K = K;
  v->in_dtype = dt;
  v->max_chunks = 0;
  for (int64_t b = 0; b < B; ++b) {
    const int64_t n = (offsets[b + 1] - offsets[b] + ch - 1) / ch;
    if (n > v->max_chunks) v->max_chunks = n;
  }
  full_window(*v);
  std::memset(g, 0, sizeof(*g));
  for (int k = 0; k < K; ++k) g->p[k] = grads[k];
  return BKMOO_OK;
}

// Gram pass over the view's window; `reset` clears the workspace status word
// first (once per call of the C ABI, not per window).
int launch_gram_pass(const GradPtrs& g, const PlanView& v, cudaStream_t s, bool reset = true) {
  if (reset && cudaMemsetAsync(&v.hdr->status, 0, sizeof(int32_t), s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  const int64_t nch = v.c_hi - v.c_lo;
  if (nch <= 0) return BKMOO_OK;
  // large K: the variant that prefetches into shared memory (gram_prefetch.cu)
  const bool pf = v.K >= gram_prefetch_min_k();
  const void* fn = pf ? gram_prefetch_fn(v.K, v.in_dtype) : gram_fn(v.K, v.in_dtype);
  const int smem = pf ? gram_prefetch_smem(v.K) : 0;
  int grid = 0;
  if (persistent_grid(fn, kThreads, &grid, smem) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (grid > nch) grid = (int)nch;
  GradPtrs ga = g;
  PlanView va = v;
  void* args[] = {&ga, &va};
  if (cudaLaunchKernel(fn, dim3(grid), dim3(kThreads), args, smem, s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  if (launch_group_reduce(v, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

int launch_combine(const GradPtrs& g, const PlanView& v, void* out, int32_t out_dtype,
                   cudaStream_t s) {
  const int64_t nch = v.c_hi - v.c_lo;
  if (nch <= 0) return BKMOO_OK;
  const bool pf = BKMOO_COMBINE_PREFETCH != 0;
  const void* fn = pf ? combine_prefetch_fn(v.K, v.in_dtype, out_dtype)
                      : combine_fn(v.K, v.in_dtype, out_dtype);
  const int smem = pf ? combine_prefetch_smem(v.K) : 0;
  int grid = 0;
  if (persistent_grid(fn, kThreads, &grid, smem) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (grid > nch) grid = (int)nch;
  PlanView va = v;
  GradPtrs ga = g;
  void* outp = out;
  void* args[] = {&ga, &va, &outp};
  if (cudaLaunchKernel(fn, dim3(grid), dim3(kThreads), args, smem, s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

bool params_ok(const bkmoo_params& p) {
  return p.max_iter >= 0 && p.cagrad_c >= 0.0 && p.cagrad_c < 1.0 && p.tol >= 0.0;
}

SolveParams solve_params(int32_t rule, const bkmoo_params& prm) {
  SolveParams sp;
  sp.rule = rule;
  sp.max_iter = prm.max_iter;
  sp.tol = prm.tol;
  sp.cagrad_c = prm.cagrad_c;
  sp.seed = prm.seed;
  sp.step = prm.step;
  sp.flags = prm.flags;
  return sp;
}

// Checks shared by bkmoo_resolve and bkmoo_resolve_buckets; fills the
// effective parameters, the plan view and the gradient pointers.
int resolve_args(const void* const* grads, int32_t K, int32_t in_dtype, const int64_t* offsets,
                 int64_t n_buckets, int32_t rule, const bkmoo_params* p, const void* out_dir,
                 int32_t out_dtype, void* ws, size_t ws_bytes, bkmoo_params* prm, PlanView* v,
                 GradPtrs* g) {
  if (rule < BKMOO_MGDA || rule > BKMOO_MEAN || !dtype_ok(out_dtype)) return BKMOO_ERR_INVALID;
  if (!out_dir || !aligned(out_dir, 16)) return BKMOO_ERR_INVALID;
  if (p) *prm = *p;
  else bkmoo_default_params(prm);
  if (!params_ok(*prm)) return BKMOO_ERR_INVALID;
  int r = prepare(grads, K, in_dtype, offsets, n_buckets, ws, ws_bytes, v, g);
  if (r != BKMOO_OK) return r;
  // out_dir may be exactly one gradient (same dtype); any other overlap is refused.
  const uintptr_t N = (uintptr_t)offsets[n_buckets];
  const uintptr_t o0 = (uintptr_t)out_dir, o1 = o0 + N * elem_bytes(out_dtype);
  for (int k = 0; k < K; ++k) {
    const uintptr_t g0 = (uintptr_t)grads[k], g1 = g0 + N * elem_bytes(in_dtype);
    if (o0 < g1 && g0 < o1 && !(o0 == g0 && out_dtype == in_dtype)) return BKMOO_ERR_INVALID;
  }
  return BKMOO_OK;
}

// ---------------------------------------------------------------------------
// Host-memory path (bkmoo_resolve_host): windows of whole buckets streamed
// through three device staging slots (measured on GB300: 3-5 % faster end to
// end than two, whose output copies held back the next windows' inputs).
// ---------------------------------------------------------------------------

constexpr int kHostSlots = 3;

// Each slot has K input regions and one output region, each 256-byte
// aligned, with one 16-byte vector of slack so that a window may start at
// any element and still keep vector alignment.
size_t region_bytes(int64_t elems, int32_t dt) {
  return align256((size_t)elems * elem_bytes(dt) + 16);
}

size_t staging_bytes_for(int32_t K, int32_t dti, int32_t dto, int64_t elems) {
  return (size_t)kHostSlots * ((size_t)K * region_bytes(elems, dti) + region_bytes(elems, dto));
}

// Elements of one language a slot holds for a staging buffer of `bytes`: the
// largest cap with staging_bytes_for(cap) <= bytes.
int64_t slot_capacity(int32_t K, int32_t dti, int32_t dto, size_t bytes) {
  const int64_t per_elem = K * elem_bytes(dti) + elem_bytes(dto);
  int64_t lo = 0, hi = (int64_t)(bytes / kHostSlots) / per_elem + 1;  // fits, does not fit
  if (staging_bytes_for(K, dti, dto, 0) > bytes) return 0;
  while (hi - lo > 1) {
    const int64_t mid = lo + (hi - lo) / 2;
    if (staging_bytes_for(K, dti, dto, mid) <= bytes) lo = mid;
    else hi = mid;
  }
  return lo;
}

}  // namespace

extern "C" {

void bkmoo_default_params(bkmoo_params* p) {
  if (!p) return;
  p->max_iter = 256;
  p->tol = 1e-12;
  p->cagrad_c = 0.5;
  p->seed = 0;
  p->step = 0;
  p->flags = BKMOO_FLAG_CLOSED_FORM_K2 | BKMOO_FLAG_POLISH;
  p->events = nullptr;
}

int bkmoo_plan(const int64_t* param_sizes, int32_t n_params, int32_t elem_bytes_,
               int64_t bucket_bytes, int64_t* out_offsets, int64_t out_cap,
               int64_t* n_buckets) {
  if (!n_buckets || n_params < 0 || (n_params > 0 && !param_sizes) || elem_bytes_ <= 0 ||
      bucket_bytes <= 0)
    return BKMOO_ERR_INVALID;
  const int64_t cap = bucket_bytes / elem_bytes_;
  if (cap < 1) return BKMOO_ERR_INVALID;
  for (int32_t i = 0; i < n_params; ++i)
    if (param_sizes[i] < 0) return BKMOO_ERR_INVALID;

  // Walk the tensors last-registered first; `fill` is the open bucket's size
  // and `end` the flat position reached so far.
  std::vector<int64_t> bounds;
  bounds.push_back(0);
  int64_t fill = 0, end = 0;
  for (int32_t i = n_params; i-- > 0;) {
    int64_t left = param_sizes[i];
    if (left == 0) continue;
    if (fill > 0 && fill + left > cap) {  // does not fit: close the open bucket
      bounds.push_back(end);
      fill = 0;
    }
    while (left > cap) {  // oversize tensor: whole cap-sized pieces
      end += cap;
      bounds.push_back(end);
      left -= cap;
    }
    fill += left;
    end += left;
  }
  if (fill > 0) bounds.push_back(end);
  *n_buckets = (int64_t)bounds.size() - 1;
  if (!out_offsets) return BKMOO_OK;
  if (out_cap < (int64_t)bounds.size()) return BKMOO_ERR_BUFFER_TOO_SMALL;
  std::memcpy(out_offsets, bounds.data(), sizeof(int64_t) * bounds.size());
  return BKMOO_OK;
}

int bkmoo_workspace_size(int32_t K, int32_t in_dtype, const int64_t* offsets,
                         int64_t n_buckets, size_t* bytes) {
  if (!bytes || K < 1 || K > kMaxK || !dtype_ok(in_dtype) || !offsets_ok(offsets, n_buckets))
    return BKMOO_ERR_INVALID;
  const int64_t nch = count_chunks(offsets, n_buckets, chunk_elems(in_dtype));
  *bytes = ws_layout(K, n_buckets, nch).total_fused;
  return BKMOO_OK;
}

int bkmoo_workspace_init(int32_t K, int32_t in_dtype, const int64_t* offsets,
                         int64_t n_buckets, void* ws, size_t ws_bytes, void* stream) {
  if (K < 1 || K > kMaxK || !dtype_ok(in_dtype) || !ws || !aligned(ws, 256) ||
      !offsets_ok(offsets, n_buckets))
    return BKMOO_ERR_INVALID;
  const int64_t ch = chunk_elems(in_dtype);
  const int64_t nch = count_chunks(offsets, n_buckets, ch);
  const WsLayout L = ws_layout(K, n_buckets, nch);
  if (ws_bytes < L.total_fused) return BKMOO_ERR_WORKSPACE;
  // Host image of header + bucket table, copied in one transfer.
  std::vector<unsigned char> img(L.partials, 0);
  WsHeader h;
  std::memset(&h, 0, sizeof h);
  h.magic = kMagic;
  h.K = K;
  h.in_dtype = in_dtype;
  h.status = BKMOO_OK;
  h.n_buckets = n_buckets;
  h.n_elems = offsets[n_buckets];
  h.n_chunks = nch;
  h.chunk_elems = ch;
  h.plan_hash = plan_hash(K, in_dtype, offsets, n_buckets);
  std::memcpy(img.data(), &h, sizeof h);
  std::memcpy(img.data() + L.offsets, offsets, sizeof(int64_t) * (size_t)(n_buckets + 1));
  int64_t* cp = reinterpret_cast<int64_t*>(img.data() + L.chunk_prefix);
  cp[0] = 0;
  for (int64_t b = 0; b < n_buckets; ++b) cp[b + 1] = cp[b] + (offsets[b + 1] - offsets[b] + ch - 1) / ch;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(ws, img.data(), img.size(), cudaMemcpyHostToDevice, s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

int bkmoo_gram(const void* const* grads, int32_t K, int32_t in_dtype, const int64_t* offsets,
               int64_t n_buckets, double* out_gram, void* ws, size_t ws_bytes, void* stream) {
  if (!out_gram && n_buckets > 0) return BKMOO_ERR_INVALID;
  PlanView v;
  GradPtrs g;
  int r = prepare(grads, K, in_dtype, offsets, n_buckets, ws, ws_bytes, &v, &g);
  if (r != BKMOO_OK) return r;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  r = launch_gram_pass(g, v, s);
  if (r != BKMOO_OK) return r;
  if (launch_gram_finalize(v, out_gram, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

int bkmoo_resolve(const void* const* grads, int32_t K, int32_t in_dtype, const int64_t* offsets,
                  int64_t n_buckets, int32_t rule, const bkmoo_params* p, void* out_dir,
                  int32_t out_dtype, float* out_weights, int32_t* out_status, void* ws,
                  size_t ws_bytes, void* stream) {
  bkmoo_params prm;
  PlanView v;
  GradPtrs g;
  int r = resolve_args(grads, K, in_dtype, offsets, n_buckets, rule, p, out_dir, out_dtype, ws,
                       ws_bytes, &prm, &v, &g);
  if (r != BKMOO_OK) return r;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaEvent_t* ev = static_cast<cudaEvent_t*>(prm.events);
  const SolveParams sp = solve_params(rule, prm);
  if (ev && cudaEventRecord(ev[0], s) != cudaSuccess) return BKMOO_ERR_CUDA;
  const int path = choose_path(K, in_dtype, rule, offsets, n_buckets, prm.flags);
  int64_t nmax = 0;
  if (path != 0)
    for (int64_t b = 0; b < n_buckets; ++b)
      if (offsets[b + 1] - offsets[b] > nmax) nmax = offsets[b + 1] - offsets[b];
  if (path == 1) {
    r = launch_fused_cluster(g, v, sp, out_weights, out_status, out_dir, out_dtype, nmax, s);
    if (r != BKMOO_OK) return r;
    for (int i = 1; i < 4; ++i)
      if (ev && cudaEventRecord(ev[i], s) != cudaSuccess) return BKMOO_ERR_CUDA;
    return BKMOO_OK;
  }
  if (path == 2) {
    r = launch_fused(g, v, sp, ws, out_weights, out_status, out_dir, out_dtype,
                     (double)nmax * (K * elem_bytes(in_dtype) + elem_bytes(out_dtype)), s);
    if (r != BKMOO_OK) return r;
    for (int i = 1; i < 4; ++i)
      if (ev && cudaEventRecord(ev[i], s) != cudaSuccess) return BKMOO_ERR_CUDA;
    return BKMOO_OK;
  }
  r = launch_gram_pass(g, v, s);
  if (r != BKMOO_OK) return r;
  if (ev && cudaEventRecord(ev[1], s) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (launch_solve(v, sp, out_weights, out_status, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (ev && cudaEventRecord(ev[2], s) != cudaSuccess) return BKMOO_ERR_CUDA;
  r = launch_combine(g, v, out_dir, out_dtype, s);
  if (r != BKMOO_OK) return r;
  if (ev && cudaEventRecord(ev[3], s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

int bkmoo_resolve_buckets(const void* const* grads, int32_t K, int32_t in_dtype,
                          const int64_t* offsets, int64_t n_buckets, int64_t b_lo, int64_t b_hi,
                          int32_t rule, const bkmoo_params* p, void* out_dir, int32_t out_dtype,
                          float* out_weights, int32_t* out_status, void* ws, size_t ws_bytes,
                          void* stream) {
  bkmoo_params prm;
  PlanView v;
  GradPtrs g;
  int r = resolve_args(grads, K, in_dtype, offsets, n_buckets, rule, p, out_dir, out_dtype, ws,
                       ws_bytes, &prm, &v, &g);
  if (r != BKMOO_OK) return r;
  if (b_lo < 0 || b_hi > n_buckets || b_lo > b_hi) return BKMOO_ERR_INVALID;
  if (b_lo == b_hi) return BKMOO_OK;
  v.b_lo = b_lo;
  v.b_hi = b_hi;
  int64_t c = 0;
  for (int64_t b = 0; b < b_lo; ++b) c += (offsets[b + 1] - offsets[b] + v.chunk_elems - 1) / v.chunk_elems;
  v.c_lo = c;
  for (int64_t b = b_lo; b < b_hi; ++b) c += (offsets[b + 1] - offsets[b] + v.chunk_elems - 1) / v.chunk_elems;
  v.c_hi = c;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const SolveParams sp = solve_params(rule, prm);
  r = launch_gram_pass(g, v, s, false);
  if (r != BKMOO_OK) return r;
  if (launch_solve(v, sp, out_weights, out_status, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return launch_combine(g, v, out_dir, out_dtype, s);
}

int bkmoo_host_staging_size(int32_t K, int32_t in_dtype, int32_t out_dtype,
                            const int64_t* offsets, int64_t n_buckets, int64_t window_elems,
                            size_t* bytes) {
  if (!bytes || K < 1 || K > kMaxK || !dtype_ok(in_dtype) || !dtype_ok(out_dtype) ||
      !offsets_ok(offsets, n_buckets) || window_elems < 0)
    return BKMOO_ERR_INVALID;
  int64_t w = window_elems;
  for (int64_t b = 0; b < n_buckets; ++b)
    if (offsets[b + 1] - offsets[b] > w) w = offsets[b + 1] - offsets[b];
  *bytes = staging_bytes_for(K, in_dtype, out_dtype, w);
  return BKMOO_OK;
}

int bkmoo_resolve_host(const void* const* host_grads, int32_t K, int32_t in_dtype,
                       const int64_t* offsets, int64_t n_buckets, int32_t rule,
                       const bkmoo_params* p, void* host_out, int32_t out_dtype,
                       float* out_weights, int32_t* out_status, void* ws, size_t ws_bytes,
                       void* staging, size_t staging_bytes, void* stream) {
  if (rule < BKMOO_MGDA || rule > BKMOO_MEAN || !dtype_ok(out_dtype) || !host_out || !staging ||
      !aligned(staging, 256))
    return BKMOO_ERR_INVALID;
  bkmoo_params prm;
  if (p) prm = *p;
  else bkmoo_default_params(&prm);
  if (!params_ok(prm)) return BKMOO_ERR_INVALID;
  // The kernels address the staging slots, never the host buffers; `prepare`
  // checks the plan and workspace (its pointer checks see the host pointers).
  PlanView v;
  GradPtrs unused;
  int r = prepare(host_grads, K, in_dtype, offsets, n_buckets, ws, ws_bytes, &v, &unused);
  if (r != BKMOO_OK) return r;
  const int ei = elem_bytes(in_dtype), eo = elem_bytes(out_dtype);
  const int64_t N = offsets[n_buckets];
  {  // host_out may be exactly one gradient (same dtype); any other overlap is refused.
    const uintptr_t o0 = (uintptr_t)host_out, o1 = o0 + (uintptr_t)N * eo;
    for (int k = 0; k < K; ++k) {
      const uintptr_t g0 = (uintptr_t)host_grads[k], g1 = g0 + (uintptr_t)N * ei;
      if (o0 < g1 && g0 < o1 && !(o0 == g0 && out_dtype == in_dtype)) return BKMOO_ERR_INVALID;
    }
  }
  const int64_t cap = slot_capacity(K, in_dtype, out_dtype, staging_bytes);
  for (int64_t b = 0; b < n_buckets; ++b)
    if (offsets[b + 1] - offsets[b] > cap) return BKMOO_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(&v.hdr->status, 0, sizeof(int32_t), s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  if (n_buckets == 0) return BKMOO_OK;
  const SolveParams sp = solve_params(rule, prm);

  // Slot layout: K input regions then the output region, each of
  // region_bytes(cap) bytes.
  const size_t rin = region_bytes(cap, in_dtype), rout = region_bytes(cap, out_dtype);
  const size_t slot_bytes = (size_t)K * rin + rout;
  char* const stage = static_cast<char*>(staging);
  const int vec_in = 16 / ei;  // elements per 16-byte input vector

  // Copy streams and events live for this call only; destroying them while
  // work is queued is legal (their resources go once the work completes).
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaEvent_t ev_start = nullptr, in_ready[kHostSlots] = {}, in_free[kHostSlots] = {},
              out_ready[kHostSlots] = {}, out_free[kHostSlots] = {};
  bool ok = cudaStreamCreateWithFlags(&h2d, cudaStreamNonBlocking) == cudaSuccess &&
            cudaStreamCreateWithFlags(&d2h, cudaStreamNonBlocking) == cudaSuccess &&
            cudaEventCreateWithFlags(&ev_start, cudaEventDisableTiming) == cudaSuccess;
  for (int i = 0; ok && i < kHostSlots; ++i)
    ok = cudaEventCreateWithFlags(&in_ready[i], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&in_free[i], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&out_ready[i], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&out_free[i], cudaEventDisableTiming) == cudaSuccess;
  // Both copy streams start after the work already queued on `stream`.
  ok = ok && cudaEventRecord(ev_start, s) == cudaSuccess &&
       cudaStreamWaitEvent(h2d, ev_start, 0) == cudaSuccess &&
       cudaStreamWaitEvent(d2h, ev_start, 0) == cudaSuccess;

  const int64_t ch = v.chunk_elems;
  int64_t b0 = 0, c_next = 0;
  for (int64_t win = 0; ok && b0 < n_buckets; ++win) {
    // the window: whole buckets b0 .. b1-1, at most `cap` elements
    int64_t b1 = b0 + 1;
    while (b1 < n_buckets && offsets[b1 + 1] - offsets[b0] <= cap) ++b1;
    const int slot = (int)(win % kHostSlots);
    const int64_t lo = offsets[b0], hi = offsets[b1], n = hi - lo;
    // element `lo` sits at the same offset within a 16-byte vector as in a
    // 16-byte-aligned buffer, so the kernels' vector/scalar split holds
    const int64_t base = lo / vec_in * vec_in;
    char* sin = stage + (size_t)slot * slot_bytes;
    char* sout = sin + (size_t)K * rin;
    if (win >= kHostSlots) ok = ok && cudaStreamWaitEvent(h2d, in_free[slot], 0) == cudaSuccess;
    for (int k = 0; ok && k < K; ++k)
      ok = cudaMemcpyAsync(sin + (size_t)k * rin + (size_t)(lo - base) * ei,
                           static_cast<const char*>(host_grads[k]) + (size_t)lo * ei,
                           (size_t)n * ei, cudaMemcpyHostToDevice, h2d) == cudaSuccess;
    ok = ok && cudaEventRecord(in_ready[slot], h2d) == cudaSuccess;

    // Kernel pointers are shifted so that global element i of the plan is
    // addressed at (region + (i - base) * e): only [lo, hi) is touched.
    GradPtrs gw;
    std::memset(&gw, 0, sizeof gw);
    for (int k = 0; k < K; ++k)
      gw.p[k] = reinterpret_cast<const void*>((uintptr_t)(sin + (size_t)k * rin) -
                                              (uintptr_t)base * ei);
    void* outw = reinterpret_cast<void*>((uintptr_t)sout - (uintptr_t)base * eo);
    PlanView vw = v;
    vw.b_lo = b0;
    vw.b_hi = b1;
    // chunk range of the window: chunks are numbered bucket by bucket
    vw.c_lo = c_next;
    for (int64_t b = b0; b < b1; ++b) c_next += (offsets[b + 1] - offsets[b] + ch - 1) / ch;
    vw.c_hi = c_next;
    ok = ok && cudaStreamWaitEvent(s, in_ready[slot], 0) == cudaSuccess;
    if (win >= kHostSlots) ok = ok && cudaStreamWaitEvent(s, out_free[slot], 0) == cudaSuccess;
    if (ok) r = launch_gram_pass(gw, vw, s, false);
    ok = ok && r == BKMOO_OK && launch_solve(vw, sp, out_weights, out_status, s) == cudaSuccess;
    if (ok) r = launch_combine(gw, vw, outw, out_dtype, s);
    ok = ok && r == BKMOO_OK && cudaEventRecord(in_free[slot], s) == cudaSuccess &&
         cudaEventRecord(out_ready[slot], s) == cudaSuccess;

    ok = ok && cudaStreamWaitEvent(d2h, out_ready[slot], 0) == cudaSuccess &&
         cudaMemcpyAsync(static_cast<char*>(host_out) + (size_t)lo * eo,
                         sout + (size_t)(lo - base) * eo, (size_t)n * eo,
                         cudaMemcpyDeviceToHost, d2h) == cudaSuccess &&
         cudaEventRecord(out_free[slot], d2h) == cudaSuccess;
    b0 = b1;
  }
  // `stream` completes only after the last copy back.
  ok = ok && cudaEventRecord(ev_start, d2h) == cudaSuccess &&
       cudaStreamWaitEvent(s, ev_start, 0) == cudaSuccess;
  if (h2d) cudaStreamDestroy(h2d);
  if (d2h) cudaStreamDestroy(d2h);
  if (ev_start) cudaEventDestroy(ev_start);
  for (int i = 0; i < kHostSlots; ++i) {
    if (in_ready[i]) cudaEventDestroy(in_ready[i]);
    if (in_free[i]) cudaEventDestroy(in_free[i]);
    if (out_ready[i]) cudaEventDestroy(out_ready[i]);
    if (out_free[i]) cudaEventDestroy(out_free[i]);
  }
  if (!ok) return r != BKMOO_OK ? r : BKMOO_ERR_CUDA;
  return BKMOO_OK;
}

int bkmoo_workspace_status(const void* ws, void* stream, int32_t* status) {
  if (!ws || !status || !aligned(ws, 256)) return BKMOO_ERR_INVALID;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return BKMOO_ERR_CUDA;
  const WsHeader* h = static_cast<const WsHeader*>(ws);
  int32_t st = 0;
  if (cudaMemcpy(&st, &h->status, sizeof st, cudaMemcpyDeviceToHost) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  *status = st;
  return BKMOO_OK;
}

const char* bkmoo_status_string(int32_t status) {
  switch (status) {
    case BKMOO_OK: return "ok";
    case BKMOO_ERR_INVALID: return "invalid argument";
    case BKMOO_ERR_CUDA: return "CUDA error";
    case BKMOO_ERR_NONFINITE: return "non-finite Gram matrix (beta = 1/K)";
    case BKMOO_ERR_WORKSPACE: return "workspace too small or not initialised for this plan";
    case BKMOO_ERR_TIMEOUT: return "bounded device wait timed out";
    case BKMOO_ERR_BUFFER_TOO_SMALL: return "output buffer too small";
    case BKMOO_ERR_NOT_CONVERGED: return "solver stopped at its iteration cap";
    default: return "unknown status";
  }
}

int32_t bkmoo_version(void) { return kVersion; }

int bkmoo_resolve_path(int32_t K, int32_t in_dtype, int32_t rule, const int64_t* offsets,
                       int64_t n_buckets, uint32_t flags, int32_t* path) {
  if (!path || K < 1 || K > kMaxK || !dtype_ok(in_dtype) || rule < BKMOO_MGDA ||
      rule > BKMOO_MEAN || !offsets_ok(offsets, n_buckets))
    return BKMOO_ERR_INVALID;
  *path = choose_path(K, in_dtype, rule, offsets, n_buckets, flags);
  return BKMOO_OK;
}

int bkmoo_selftest_fp64(int32_t op, const double* a, const double* b, double* out, int64_t n,
                        void* stream) {
  if ((op != 0 && op != 1) || n < 0 || (n > 0 && (!a || !out || (op == 0 && !b))))
    return BKMOO_ERR_INVALID;
  return launch_selftest_fp64(op, a, b, out, n, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? BKMOO_OK
             : BKMOO_ERR_CUDA;
}

}  // extern "C"
