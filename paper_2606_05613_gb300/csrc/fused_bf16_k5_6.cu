// Fused resolve kernels for bf16 gradients, K = 5..6, fp32 or bf16 output.
#include "fused_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_FUSED_TABLE2(BKMOO_BF16, 5);
}
const void* fused_fn_bf16_k5_6(int K, int dtype_out) { return kFusedTable[K - 5][dtype_out]; }
}  // namespace bkmoo
