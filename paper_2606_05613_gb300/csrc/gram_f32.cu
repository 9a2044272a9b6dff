// Gram-pass kernels for fp32 gradients, K = 1..16.
#include "gram_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_GRAM_TABLE(BKMOO_F32);
}
const void* gram_partials_fn_f32(int K) { return kGramTable[K - 1]; }
}  // namespace bkmoo
