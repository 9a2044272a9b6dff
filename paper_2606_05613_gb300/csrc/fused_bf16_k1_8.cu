// Fused resolve kernels for bf16 gradients, K = 1..8, fp32 or bf16 output.
#include "fused_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_FUSED_TABLE8(BKMOO_BF16, 1);
}
const void* fused_fn_bf16_k1_8(int K, int dtype_out) { return kFusedTable[K - 1][dtype_out]; }
}  // namespace bkmoo
