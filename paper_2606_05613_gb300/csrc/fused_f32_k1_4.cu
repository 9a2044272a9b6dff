// Fused resolve kernels for f32 gradients, K = 1..4, fp32 or bf16 output.
#include "fused_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_FUSED_TABLE4(BKMOO_F32, 1);
}
const void* fused_fn_f32_k1_4(int K, int dtype_out) { return kFusedTable[K - 1][dtype_out]; }
}  // namespace bkmoo
