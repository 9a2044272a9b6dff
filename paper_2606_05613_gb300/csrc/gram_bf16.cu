// Gram-pass kernels for bf16 gradients, K = 1..16.
#include "gram_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_GRAM_TABLE(BKMOO_BF16);
}
const void* gram_partials_fn_bf16(int K) { return kGramTable[K - 1]; }
}  // namespace bkmoo
