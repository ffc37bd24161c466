"""Shared helpers of the GPU parity tests: contexts from workloads, oracle twins, tolerances."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

# Floating-point tolerance of logits, values and logp against the fp64 oracle:
# |gpu - oracle| <= REL * |oracle| + REL * rms(oracle)   (REL = 1e-4)
REL = 1e-4
# GAE is checked teacher-forced (oracle fed the GPU's own r, v, d, V_T), fp32 vs fp64.
GAE_REL = 1e-5
# A sampled action may differ only where the oracle's u lies within this of a CDF edge.
CDF_MARGIN = 1e-5


def require_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    aht.load()


def close(gpu, ref, rel=REL):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    rms = np.sqrt(np.mean(ref ** 2)) if ref.size else 0.0
    err = np.abs(gpu - ref)
    bound = rel * np.abs(ref) + rel * rms
    ok = err <= bound
    return bool(ok.all()), float((err / np.maximum(bound, 1e-30)).max()) if ref.size else 0.0


def torch_pop(wl, pop_np):
    dt = torch.float32 if wl.weight_dtype == W.FP32 else torch.bfloat16
    return [[(torch.from_numpy(Wt).to("cuda", dt), torch.from_numpy(b).to("cuda", dt))
             for Wt, b in p] for p in pop_np]


def make_ctx(wl, n_envs, seed=None, pop_np=None, env=None):
    pop_np = pop_np if pop_np is not None else W.population(wl)
    env = env or wl.env
    ctx = aht.aht_create(env, torch_pop(wl, pop_np), n_envs,
                         wl.env_seed if seed is None else seed,
                         has_value_head=[int(v) for v in wl.value_head[:len(pop_np)]],
                         weight_dtype=aht.AHT_FP32 if wl.weight_dtype == W.FP32 else aht.AHT_BF16)
    return ctx, pop_np


def oracle_of(env, pop_np):
    return O.env_desc(*env.astuple()), O.Policies(pop_np)


def np_(t):
    return t.detach().cpu().numpy()
