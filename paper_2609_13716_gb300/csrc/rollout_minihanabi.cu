// rollout_minihanabi.cu -- kernel instantiations for the Mini Hanabi rules.
#include "env_minihanabi.cuh"
#include "rollout_impl.cuh"
#include "xplay_tc.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(minihanabi, EnvMiniHanabi)

cudaError_t minihanabi_xplay_tc(const XpTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  return launch_xp_tc<EnvMiniHanabi>(a, grid, smem, s);
}
cudaError_t minihanabi_xplay_tc_smem_limit(size_t smem) { return xp_tc_smem_limit<EnvMiniHanabi>(smem); }
}  // namespace aht
