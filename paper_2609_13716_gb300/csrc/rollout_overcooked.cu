// rollout_overcooked.cu -- kernel instantiations for the overcooked rules.
#include "env_overcooked.cuh"
#include "rollout_impl.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(overcooked, EnvOvercooked)
}  // namespace aht
