// append_fused_r16.cu -- the fused append kernel (append_fused.cuh) for PSAC
// rank 16, in a translation unit of its own so the ranks compile in parallel.
#include "append_fused.cuh"

namespace qwm {

cudaError_t append_fused_r16(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  return launch_fused_rank<16>(a, maps, st);
}

}  // namespace qwm
