// rollout_overcooked.cu -- kernel instantiations for the overcooked rules.
#include "env_overcooked.cuh"
#include "rollout_impl.cuh"
#include "xplay_tc.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(overcooked, EnvOvercooked)

cudaError_t overcooked_xplay_tc(const XpTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  return launch_xp_tc<EnvOvercooked>(a, grid, smem, s);
}
cudaError_t overcooked_xplay_tc_smem_limit(size_t smem) { return xp_tc_smem_limit<EnvOvercooked>(smem); }

size_t xp_tc_smem_bytes(const WideDims& w) { return xp_tc_layout(w).total; }
size_t xp_tc_state_bytes(const WideDims& w) { return xp_tc_layout(w).a_bytes; }
cudaError_t overcooked_obs_words(const uint32_t* state, int64_t n, const DevEnv& env, int seat, int words,
                             uint32_t* out, cudaStream_t s) {
  return launch_obs_words<EnvOvercooked>(state, n, env, seat, words, out, s);
}
}  // namespace aht
