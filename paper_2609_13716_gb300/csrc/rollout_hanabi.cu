// rollout_hanabi.cu -- kernel instantiations for the hanabi rules.
#include "env_hanabi.cuh"
#include "rollout_impl.cuh"

namespace aht {
AHT_DEFINE_ENV_LAUNCHERS(hanabi, EnvHanabi)
}  // namespace aht
