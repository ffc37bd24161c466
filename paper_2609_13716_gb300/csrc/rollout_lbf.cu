// rollout_lbf.cu -- kernel instantiations for the lbf rules (CUDA-core and tensor-core).
#include "env_lbf.cuh"
#include "rollout_impl.cuh"
#include "rollout_tc.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(lbf, EnvLbf)

cudaError_t lbf_ppo_tc(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  const TrajPtrs& u = a.traj1;
  const bool ippo = u.obs || u.actions || u.tm_actions || u.logp || u.values || u.rewards ||
                    u.dones || u.last_value;
  // collection with a dense first layer (plain, or IPPO on contiguous tiles): one warp
  // group per agent (rollout_tc2.cuh)
  if (!a.tc.sparse && (!ippo || !a.gather)) return lbf_ppo_tc2(a, grid, smem, s);
  return LaunchTc<EnvLbf>::ppo(a, grid, smem, s);
}

cudaError_t lbf_xplay_tc(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  // a dense first layer: one warp group per agent (rollout_tc2.cuh)
  if (!a.tc.sparse) return lbf_xplay_tc2(a, grid, smem, s);
  return LaunchTc<EnvLbf>::xplay(a, grid, smem, s);
}
}  // namespace aht
