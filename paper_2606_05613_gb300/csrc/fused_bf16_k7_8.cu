// Fused resolve kernels for bf16 gradients, K = 7..8, fp32 or bf16 output.
#include "fused_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_FUSED_TABLE2(BKMOO_BF16, 7);
}
const void* fused_fn_bf16_k7_8(int K, int dtype_out) { return kFusedTable[K - 7][dtype_out]; }
}  // namespace bkmoo
