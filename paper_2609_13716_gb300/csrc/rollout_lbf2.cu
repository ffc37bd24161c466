// rollout_lbf2.cu -- the LBF PPO collection kernel with one warp group per agent.
#include "env_lbf.cuh"
#include "rollout_tc2.cuh"

namespace aht {
cudaError_t lbf_ppo_tc2(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  const TrajPtrs& u = a.traj1;
  const bool ippo = u.obs || u.actions || u.tm_actions || u.logp || u.values || u.rewards ||
                    u.dones || u.last_value;
  return ippo ? LaunchTc2<EnvLbf>::ippo(a, grid, smem, s) : LaunchTc2<EnvLbf>::ppo(a, grid, smem, s);
}
cudaError_t lbf_xplay_tc2(const PpoTcArgs& a, int grid, size_t smem, cudaStream_t s) {
  return LaunchTc2<EnvLbf>::xplay(a, grid, smem, s);
}
}  // namespace aht
