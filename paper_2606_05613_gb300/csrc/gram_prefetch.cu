// Gram-pass kernels with a per-thread shared-memory prefetch (used for K >=
// kPrefetchMinK).
#include "gram_prefetch.cuh"

namespace bkmoo {
namespace {
BKMOO_GRAM_PREFETCH_TABLE(BKMOO_F32);
}
namespace bf {
namespace {
BKMOO_GRAM_PREFETCH_TABLE(BKMOO_BF16);
}
}  // namespace bf
const void* gram_prefetch_fn(int K, int dt) {
  if (K < kPrefetchMinK || K > kMaxK) return nullptr;
  return dt == BKMOO_F32 ? kGramPrefetchTable[K - 1] : bf::kGramPrefetchTable[K - 1];
}
int gram_prefetch_smem(int K) { return prefetch_smem_bytes(K); }
int gram_prefetch_min_k() { return kPrefetchMinK; }
}  // namespace bkmoo
