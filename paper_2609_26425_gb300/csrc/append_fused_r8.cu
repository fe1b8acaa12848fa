// append_fused_r8.cu -- the fused append kernel (append_fused.cuh) for PSAC
// rank 8, in a translation unit of its own so the ranks compile in parallel.
#include "append_fused.cuh"

namespace qwm {

cudaError_t append_fused_r8(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  return launch_fused_rank<8>(a, maps, st);
}

}  // namespace qwm
