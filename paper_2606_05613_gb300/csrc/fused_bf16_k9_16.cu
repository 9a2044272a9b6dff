// Fused resolve kernels for bf16 gradients, K = 9..16, fp32 or bf16 output.
#include "fused_impl.cuh"

namespace bkmoo {
namespace {
BKMOO_FUSED_TABLE8(BKMOO_BF16, 9);
}
const void* fused_fn_bf16_k9_16(int K, int dtype_out) { return kFusedTable[K - 9][dtype_out]; }
}  // namespace bkmoo
