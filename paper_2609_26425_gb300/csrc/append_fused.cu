// append_fused.cu -- the fused append kernel (append_fused.cuh): tensor maps,
// dispatch on the PSAC rank, and the instances without PSAC.
#include "append_fused.cuh"

namespace qwm {

cudaError_t append_fused_r0(const AppendArgs& a, const CUtensorMap* maps, cudaStream_t st) {
  return launch_fused_rank<0>(a, maps, st);
}

cudaError_t launch_append_fused(const AppendArgs& a, cudaStream_t st) {
  alignas(64) CUtensorMap maps[4];
  const int Npad = (a.L.C + 15) & ~15;
  if (!make_token_map(&maps[0], a.k, a.N, a.L.H, 128) || !make_token_map(&maps[1], a.v, a.N, a.L.H, 128) ||
      !make_table_map(&maps[2], a.kc, a.L.C, a.L.H, Npad) || !make_table_map(&maps[3], a.vc, a.L.C, a.L.H, Npad))
    return cudaErrorInvalidValue;
  switch (a.L.r) {
    case 0: return append_fused_r0(a, maps, st);
    case 8: return append_fused_r8(a, maps, st);
    case 16: return append_fused_r16(a, maps, st);
    case 32: return append_fused_r32(a, maps, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace qwm
