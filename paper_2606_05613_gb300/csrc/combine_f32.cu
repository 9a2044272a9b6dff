// Combination kernels for fp32 gradients, K = 1..16, fp32 or bf16 output.
#include "combine_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_COMBINE_TABLE(BKMOO_F32);
}
const void* combine_fn_f32(int K, int dtype_out) { return kCombineTable[K - 1][dtype_out]; }
}  // namespace bkmoo
