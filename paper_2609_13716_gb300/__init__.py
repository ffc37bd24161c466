"""GB300 (sm_103a) batched ad hoc teamwork rollouts: env stepping, population MLP policies,
GAE and cross-play matrices in hand-written CUDA kernels behind a C ABI (include/aht.h).

Modules:
  build      -- compiles csrc/*.cu into _build/libaht.so (nvcc, sm_103a)
  aht        -- ctypes binding of the C ABI (argument marshalling only)
  workloads  -- seeded synthetic workloads and weights (no method arithmetic)
"""
