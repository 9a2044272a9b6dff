// Combination kernels with a per-thread shared-memory prefetch, K = 9..16.
#include "combine_prefetch.cuh"

namespace bkmoo {
namespace {
#define BKMOO_CPF_ROW(K, DTI)                                                 \
  {(const void*)combine_prefetch_kernel<K, DTI, BKMOO_F32>,                   \
   (const void*)combine_prefetch_kernel<K, DTI, BKMOO_BF16>}
#define BKMOO_CPF_TABLE(DTI)                                                  \
  {BKMOO_CPF_ROW(9, DTI),  BKMOO_CPF_ROW(10, DTI), BKMOO_CPF_ROW(11, DTI),    \
   BKMOO_CPF_ROW(12, DTI), BKMOO_CPF_ROW(13, DTI), BKMOO_CPF_ROW(14, DTI),    \
   BKMOO_CPF_ROW(15, DTI), BKMOO_CPF_ROW(16, DTI)}
static const void* const kCpfF32[8][2] = BKMOO_CPF_TABLE(BKMOO_F32);
static const void* const kCpfBf16[8][2] = BKMOO_CPF_TABLE(BKMOO_BF16);
}  // namespace
const void* combine_prefetch_fn_k9_16(int K, int dti, int dto) {
  if (K < 9 || K > 16) return nullptr;
  return dti == BKMOO_F32 ? kCpfF32[K - 9][dto] : kCpfBf16[K - 9][dto];
}
}  // namespace bkmoo
