// rollout_hanabi.cu -- kernel instantiations for the hanabi rules.
#include "env_hanabi.cuh"
#include "rollout_impl.cuh"
#include "xplay_tc.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(hanabi, EnvHanabi)

cudaError_t hanabi_xplay_tc(const XpTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  return launch_xp_tc<EnvHanabi>(a, grid, smem, s);
}
cudaError_t hanabi_xplay_tc_smem_limit(size_t smem) { return xp_tc_smem_limit<EnvHanabi>(smem); }
}  // namespace aht
