// Cluster-per-bucket fused resolve kernels, K = 1..kClusterMaxK, fp32 / bf16 in and out.
#include "fused_cluster.cuh"

namespace bkmoo {
namespace {
#define BKMOO_FCL_ROW(K, DTI)                                                 \
  {(const void*)fused_cluster_kernel<K, DTI, BKMOO_F32>,                      \
   (const void*)fused_cluster_kernel<K, DTI, BKMOO_BF16>}
#define BKMOO_FCL_TABLE(DTI)                                                  \
  {BKMOO_FCL_ROW(1, DTI), BKMOO_FCL_ROW(2, DTI), BKMOO_FCL_ROW(3, DTI),       \
   BKMOO_FCL_ROW(4, DTI)}
static const void* const kFclF32[4][2] = BKMOO_FCL_TABLE(BKMOO_F32);
static const void* const kFclBf16[4][2] = BKMOO_FCL_TABLE(BKMOO_BF16);
}  // namespace
const void* fused_cluster_fn(int K, int dti, int dto) {
  if (K < 1 || K > kClusterMaxK) return nullptr;
  return dti == BKMOO_F32 ? kFclF32[K - 1][dto] : kFclBf16[K - 1][dto];
}
int fused_cluster_smem(int K) { return cluster_smem_bytes(K); }
}  // namespace bkmoo
