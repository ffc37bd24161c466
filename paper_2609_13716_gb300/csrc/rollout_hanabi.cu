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
cudaError_t hanabi_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                             uint32_t* out, cudaStream_t s) {
  return launch_obs_words<EnvHanabi>(state, n, env, seat, words, out, s);
}
}  // namespace aht
