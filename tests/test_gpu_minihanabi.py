"""Mini Hanabi (3 colours x 3 ranks) on the GPU against the oracle: forced-action env
rules (states, observations, rewards, dones bit-exact), cross-play to termination on the
streamed tensor-core kernel (bf16 256-wide policies) and on the CUDA-core kernel (fp32
64-wide), and the illegal-action error."""
import ctypes as C
import dataclasses

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, require_gpu
from test_gpu_env import _run_forced
from test_gpu_xplay import check, run_xplay

pytestmark = pytest.mark.gpu

WL = W.WORKLOADS["minihanabi_xplay_16x16x32"]


def _legal_random(rng):
    def fn(t, st):
        n = st.shape[0]
        acts = np.zeros((n, 2), np.uint8)
        legal = np.zeros(10, np.uint8)
        for e in range(n):
            s = O.MiniHanabiState.from_buffer(st[e])
            O.lib().orc_mhanabi_legal(C.byref(s), legal.ctypes.data_as(C.c_void_p))
            acts[e, s.turn % 2] = rng.choice(np.flatnonzero(legal))
            acts[e, 1 - s.turn % 2] = rng.integers(0, 10)   # ignored seat
        return acts
    return fn


def test_minihanabi_forced_random_legal():
    require_gpu()
    rng = np.random.default_rng(21)
    dones = _run_forced(WL.env, WL, 700, 5, _legal_random(rng), 90)
    assert dones >= 700


def test_minihanabi_xplay_tensor_core_to_termination():
    require_gpu()
    ego, tm, P = [0, 3, 9], [16, 31], 45
    ctx, pop_np = make_ctx(WL, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 100)
    ref = check(WL, pop_np, ego, tm, P, 100, out, WL.env_seed)
    assert (ref["steps"] >= 1).all() and (ref["steps"] <= 40).all()


def test_minihanabi_xplay_cuda_cores_fp32():
    require_gpu()
    wl = dataclasses.replace(WL, hidden=(64, 64), weight_dtype=W.FP32)
    ego, tm, P = [1, 2], [17, 20], 70
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 100)
    check(wl, pop_np, ego, tm, P, 100, out, wl.env_seed)


def test_minihanabi_illegal_forced_action_latches_error():
    require_gpu()
    ctx, _ = make_ctx(WL, 4, seed=1)
    acts = torch.full((4, 2), 2, dtype=torch.uint8, device="cuda")   # discard at 3 tokens
    aht.aht_step_forced(ctx, acts)
    with pytest.raises(aht.AhtError) as e:
        aht.aht_sync(ctx)
    assert e.value.status == aht.AHT_EDEVICE
    aht.aht_sync(ctx)
