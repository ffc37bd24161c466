"""Rule-based LBF teammates inside the tensor-core rollout and cross-play kernels, against
the oracle.  A heuristic teammate draws nothing, so its every action must equal the
oracle's rule exactly (never a flagged CDF edge); the ego's actions, observations,
rewards, dones and returns follow the usual rollout / cross-play protocol."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu
from test_gpu_rollout import check_rollout
from test_gpu_xplay import check, run_xplay

pytestmark = pytest.mark.gpu

ALL = [O.heuristic_id(n) for n in O.LBF_HEURISTICS]


def test_ppo_rollout_with_heuristic_and_network_teammates():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    N, T = 2000, 60                      # 16 teammate blocks, the last one ragged
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    pool = ALL + [1, 2, 3]
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 0, pool, T, traj)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, T, 0, pool)
    tm = np_(traj["teammate"])
    assert (tm < 0).any() and (tm > 0).any()


def test_fp32_context_heuristic_pool():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, pop_np = make_ctx(wl, 256)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, 256)
    pool = [O.heuristic_id("seq_nearest_agent"), O.heuristic_id("greedy_closest_avg")]
    traj = aht.traj_buffers(ctx, 50)
    aht.aht_rollout(ctx, 0, pool, 50, traj)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, 50, 0, pool)


def test_xplay_against_every_heuristic():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_xplay_8x16x256"]
    ego, tm, P = [0, 3], ALL + [8], 40
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 128)
    ref = check(wl, pop_np, ego, tm, P, 128, out, wl.env_seed)
    assert (ref["steps"] >= 1).all()
    # the static variant runs the same kernel: the same matrix
    m2 = torch.empty(len(ego), len(tm), device="cuda")
    aht.aht_reset(ctx, wl.env_seed)
    aht.aht_xplay_matrix_static(ctx, ego, tm, P, 128, m2)
    aht.aht_sync(ctx)
    assert torch.equal(m2, out[0])


def test_heuristic_ids_rejected_where_unsupported():
    require_gpu()
    wl = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    ctx, _ = make_ctx(wl, 64)
    m = torch.empty(1, 1, device="cuda")
    with pytest.raises(aht.AhtError):
        aht.aht_xplay_matrix(ctx, [0], [-1], 64, 10, m)
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, _ = make_ctx(wl, 128)
    traj = aht.traj_buffers(ctx, 4)
    with pytest.raises(aht.AhtError):
        aht.aht_rollout(ctx, 0, [-1 - O.LBF_HEURISTICS.__len__()], 4, traj)
