// Shared-memory-staged Gram-pass kernels for f32 gradients, K = 1..16.
#include "gram_staged.cuh"

namespace bkmoo {
namespace {
BKMOO_GRAM_STAGED_TABLE(BKMOO_F32);
}
const void* gram_staged_fn_f32(int K) { return kGramStagedTable[K - 1]; }
int gram_staged_threads() { return kStagedThreads; }
int gram_staged_smem(int K) {
  static const int kSmem[kMaxK] = {
      staged_smem_bytes(1),  staged_smem_bytes(2),  staged_smem_bytes(3),  staged_smem_bytes(4),
      staged_smem_bytes(5),  staged_smem_bytes(6),  staged_smem_bytes(7),  staged_smem_bytes(8),
      staged_smem_bytes(9),  staged_smem_bytes(10), staged_smem_bytes(11), staged_smem_bytes(12),
      staged_smem_bytes(13), staged_smem_bytes(14), staged_smem_bytes(15), staged_smem_bytes(16)};
  return kSmem[K - 1];
}
}  // namespace bkmoo
