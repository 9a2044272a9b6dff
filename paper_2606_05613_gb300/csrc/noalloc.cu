// bkmoo_gram_noalloc: the Gram pass with its scratch in a static device
// array instead of a caller-supplied workspace.
//
// Some callers have device buffers for their inputs and outputs but no way to
// obtain more device memory: a hook inside a training framework that is
// handed the gradient buckets and an output buffer while every byte of device
// memory belongs to the framework's caching allocator, or a C caller in a
// process where another component owns device allocation.  For them this
// entry point keeps the Gram pass's scratch (the bucket table and the
// per-chunk partial sums) in `g_scratch`, a file-scope __device__ array of
// kNoallocScratchBytes that every GPU which loads this library holds until the
// process exits.  It calls no cudaMalloc, cudaFree or other allocating routine.
//
// Host code never touches g_scratch by name: in host code the name is only a
// stand-in, not a device address.  Each call made outside stream capture
// looks the address up in the current context with cudaGetSymbolAddress
// (with that device current) and passes it to the kernels; a call made
// while its stream is being captured reuses the last address seen on that
// device, so the first call on each device should come before any capture.
//
// All calls share the one array and it keeps whatever the last call left
// there.  Every call rewrites the header (including its status word, which
// must start at zero) and the bucket table before the Gram kernels read them,
// and the kernels overwrite every partial they later read, so nothing stale is
// used.  Calls whose work overlaps on the GPU (different streams, or different
// host threads on one device) race on the array and must be serialised by the
// caller.
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

#include "common.cuh"

namespace bkmoo {
namespace {

constexpr size_t kNoallocScratchBytes = (size_t)BKMOO_NOALLOC_SCRATCH_BYTES;
constexpr int64_t kNoallocMaxBuckets = BKMOO_NOALLOC_MAX_BUCKETS;
constexpr int kSlice = 224;      // bucket-table entries per set-up launch
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kNoallocScratchBytes];

// One slice of the bucket table, passed by value as kernel parameters
// (under 4 KB), so the table reaches the device without a copy call.
struct TableSlice {
  WsHeader hdr;      // written by the launch that carries the last slice
  int64_t first;     // index of off[0] in the full table
  int32_t count;     // entries off[0 .. count] are valid
  int32_t last;
  int64_t off[kSlice + 1];
  int64_t cp[kSlice + 1];
};

__global__ void noalloc_table_kernel(const TableSlice t, unsigned char* scratch,
                                     size_t offsets_at, size_t prefix_at) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i <= t.count) {
    reinterpret_cast<int64_t*>(scratch + offsets_at)[t.first + i] = t.off[i];
    reinterpret_cast<int64_t*>(scratch + prefix_at)[t.first + i] = t.cp[i];
  }
  if (t.last && i == 0) *reinterpret_cast<WsHeader*>(scratch) = t.hdr;
}

std::mutex g_addr_mu;
void* g_addr[kMaxDevices] = {};

// Device address of g_scratch in the current context.  Outside stream
// capture it is looked up on every call (cudaGetSymbolAddress allocates
// nothing and is cheap once the module is loaded), so a context rebuilt
// after cudaDeviceReset, or another context made current on the same
// device, gets its own address; the last address seen on each device is
// kept for calls made while `s` is being captured, when the runtime call is
// avoided.  The first call on a device must therefore come before any
// capture.
int scratch_address(cudaStream_t s, unsigned char** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return BKMOO_ERR_CUDA;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  const bool capturing =
      cudaStreamIsCapturing(s, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone;
  if (capturing) (void)cudaGetLastError();   // an implicit-capture error is not sticky
  std::lock_guard<std::mutex> lk(g_addr_mu);
  if (!capturing) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) return BKMOO_ERR_CUDA;
    g_addr[dev] = p;
  }
  if (!g_addr[dev]) return BKMOO_ERR_CUDA;   // first call on this device during capture
  *out = static_cast<unsigned char*>(g_addr[dev]);
  return BKMOO_OK;
}

}  // namespace
}  // namespace bkmoo

using namespace bkmoo;

extern "C" int bkmoo_gram_noalloc(const void* const* grads, int32_t K, int32_t in_dtype,
                                  const int64_t* offsets, int64_t n_buckets, double* out_gram,
                                  void* stream) {
  if (K < 1 || K > kMaxK || (in_dtype != BKMOO_F32 && in_dtype != BKMOO_BF16) || !grads ||
      !offsets_ok(offsets, n_buckets) || (n_buckets > 0 && !out_gram))
    return BKMOO_ERR_INVALID;
  for (int k = 0; k < K; ++k)
    if (!grads[k] || ((uintptr_t)grads[k] & 15u)) return BKMOO_ERR_INVALID;
  const int64_t ch = chunk_elems(in_dtype);
  const int64_t nch = count_chunks(offsets, n_buckets, ch);
  const WsLayout L = ws_layout(K, n_buckets, nch);
  if (n_buckets > kNoallocMaxBuckets || L.total > kNoallocScratchBytes)
    return BKMOO_ERR_WORKSPACE;  // larger than the static scratch
  if (n_buckets == 0) return BKMOO_OK;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned char* scratch = nullptr;
  int r = scratch_address(s, &scratch);
  if (r != BKMOO_OK) return r;

  // Bucket table and header, slice by slice through kernel parameters.
  TableSlice t;
  std::memset(&t, 0, sizeof t);
  t.hdr.magic = kMagic;
  t.hdr.K = K;
  t.hdr.in_dtype = in_dtype;
  t.hdr.status = BKMOO_OK;
  t.hdr.n_buckets = n_buckets;
  t.hdr.n_elems = offsets[n_buckets];
  t.hdr.n_chunks = nch;
  t.hdr.chunk_elems = ch;
  t.hdr.plan_hash = plan_hash(K, in_dtype, offsets, n_buckets);
  int64_t prefix = 0;
  for (int64_t first = 0; first < n_buckets; first += kSlice) {
    const int32_t count = (int32_t)((n_buckets - first) < kSlice ? (n_buckets - first) : kSlice);
    t.first = first;
    t.count = count;
    t.last = (first + count == n_buckets) ? 1 : 0;
    for (int i = 0; i <= count; ++i) {
      const int64_t b = first + i;
      t.off[i] = offsets[b];
      t.cp[i] = prefix;
      if (i < count) prefix += (offsets[b + 1] - offsets[b] + ch - 1) / ch;
    }
    const int threads = 256;
    noalloc_table_kernel<<<(count + threads) / threads, threads, 0, s>>>(t, scratch, L.offsets,
                                                                         L.chunk_prefix);
    if (cudaGetLastError() != cudaSuccess) return BKMOO_ERR_CUDA;
  }

  PlanView v;
  v.hdr = reinterpret_cast<WsHeader*>(scratch);
  v.offsets = reinterpret_cast<const int64_t*>(scratch + L.offsets);
  v.chunk_prefix = reinterpret_cast<const int64_t*>(scratch + L.chunk_prefix);
  v.partials = reinterpret_cast<double*>(scratch + L.partials);
  v.beta = reinterpret_cast<float*>(scratch + L.beta);
  v.n_buckets = n_buckets;
  v.n_chunks = nch;
  v.chunk_elems = ch;
  v.plan_hash = t.hdr.plan_hash;
  v.K = K;
  v.in_dtype = in_dtype;
  v.max_chunks = 0;
  for (int64_t b = 0; b < n_buckets; ++b) {
    const int64_t nb = (offsets[b + 1] - offsets[b] + ch - 1) / ch;
    if (nb > v.max_chunks) v.max_chunks = nb;
  }
  full_window(v);
  GradPtrs g;
  std::memset(&g, 0, sizeof g);
  for (int k = 0; k < K; ++k) g.p[k] = grads[k];

  // the same Gram-pass kernel as bkmoo_gram (the prefetching variant for large K)
  const bool pf = K >= gram_prefetch_min_k();
  const void* fn = pf ? gram_prefetch_fn(K, in_dtype)
                      : (in_dtype == BKMOO_F32 ? gram_partials_fn_f32(K) : gram_partials_fn_bf16(K));
  const int smem = pf ? gram_prefetch_smem(K) : 0;
  int dev = 0, sms = 0, per_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      (smem > 0 &&
       cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kThreads, smem) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  int64_t grid = (int64_t)sms * (per_sm < 1 ? 1 : per_sm);
  if (grid > nch) grid = nch;
  void* args[] = {&g, &v};
  if (cudaLaunchKernel(fn, dim3((unsigned)grid), dim3(kThreads), args, smem, s) != cudaSuccess)
    return BKMOO_ERR_CUDA;
  if (launch_group_reduce(v, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  if (launch_gram_finalize(v, out_gram, s) != cudaSuccess) return BKMOO_ERR_CUDA;
  return BKMOO_OK;
}
