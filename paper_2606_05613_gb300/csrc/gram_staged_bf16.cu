// Shared-memory-staged Gram-pass kernels for bf16 gradients, K = 1..16.
#include "gram_staged.cuh"

namespace bkmoo {
namespace {
BKMOO_GRAM_STAGED_TABLE(BKMOO_BF16);
}
const void* gram_staged_fn_bf16(int K) { return kGramStagedTable[K - 1]; }
}  // namespace bkmoo
