// Combination kernels with a per-thread shared-memory prefetch, K = 1..8
// (K = 9..16: combine_prefetch_k9_16.cu).
#include "combine_prefetch.cuh"

namespace bkmoo {
namespace {
#define BKMOO_CPF_ROW(K, DTI)                                                 \
  {(const void*)combine_prefetch_kernel<K, DTI, BKMOO_F32>,                   \
   (const void*)combine_prefetch_kernel<K, DTI, BKMOO_BF16>}
#define BKMOO_CPF_TABLE(DTI)                                                  \
  {BKMOO_CPF_ROW(1, DTI), BKMOO_CPF_ROW(2, DTI), BKMOO_CPF_ROW(3, DTI),       \
   BKMOO_CPF_ROW(4, DTI), BKMOO_CPF_ROW(5, DTI), BKMOO_CPF_ROW(6, DTI),       \
   BKMOO_CPF_ROW(7, DTI), BKMOO_CPF_ROW(8, DTI)}
static const void* const kCpfF32[8][2] = BKMOO_CPF_TABLE(BKMOO_F32);
static const void* const kCpfBf16[8][2] = BKMOO_CPF_TABLE(BKMOO_BF16);
}  // namespace
const void* combine_prefetch_fn(int K, int dti, int dto) {
  if (K >= 9 && K <= kMaxK) return combine_prefetch_fn_k9_16(K, dti, dto);
  if (K < 1 || K > 8) return nullptr;
  return dti == BKMOO_F32 ? kCpfF32[K - 1][dto] : kCpfBf16[K - 1][dto];
}
int combine_prefetch_smem(int K) { return combine_prefetch_smem_bytes(K); }
}  // namespace bkmoo
