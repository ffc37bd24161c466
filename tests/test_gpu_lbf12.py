"""LBF 12x12 (the paper's second LBF grid): cross-play and PPO collection on the GPU against
the oracle.  The 576-feature observation is past the fused tensor-core rollout's input
width, so these run the CUDA-core rollout and cross-play kernels; the protocol is the
7x7 one (bit-exact env quantities, sampled actions equal away from a CDF edge)."""
import numpy as np
import pytest

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu
from test_gpu_rollout import check_rollout
from test_gpu_xplay import check, run_xplay

pytestmark = pytest.mark.gpu


def test_lbf12_xplay_small():
    require_gpu()
    wl = W.WORKLOADS["lbf12x12_xplay_8x16x128"]
    ego, tm, P = [0, 5], [8, 20, 23], 70          # ragged pairs
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 128)
    ref = check(wl, pop_np, ego, tm, P, 128, out, wl.env_seed)
    assert (ref["steps"] <= 128).all()


def test_lbf12_ppo_rollout_two_calls():
    require_gpu()
    wl = W.WORKLOADS["lbf12x12_ppo_4096x128"]
    N, T = 600, 30
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    for call in range(2):
        traj = aht.traj_buffers(ctx, T)
        aht.aht_rollout(ctx, 0, wl.pool, T, traj)
        aht.aht_sync(ctx)
        check_rollout(wl, pop_np, traj, st, wl.env_seed, call * T, T, 0, list(wl.pool))
