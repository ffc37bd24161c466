// rollout_lbf.cu -- kernel instantiations for the lbf rules.
#include "env_lbf.cuh"
#include "rollout_impl.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(lbf, EnvLbf)
}  // namespace aht
