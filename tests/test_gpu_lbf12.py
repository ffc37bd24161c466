"""LBF 12x12 (the paper's second LBF grid): cross-play and PPO collection on the GPU against
the oracle.  The 576-feature observation is past the 256 tensor-memory columns of the
fused rollout's first-layer operand, so the tensor-core kernels take the first layer on
CUDA cores from the observation's changed features (and IPPO and per-episode calls run
the CUDA-core kernels); the protocol is the 7x7 one (bit-exact env quantities, sampled
actions equal away from a CDF edge)."""
import dataclasses

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


def test_lbf12_xplay_against_rule_teammates_and_fp32_and_bf16():
    require_gpu()
    wl = W.WORKLOADS["lbf12x12_xplay_8x16x128"]
    ego, tm, P = [1, 3], [O.heuristic_id("greedy_lowest_level"), O.heuristic_id("entitled"), 9], 40
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 128)
    check(wl, pop_np, ego, tm, P, 128, out, wl.env_seed)
    # the 12x12 PPO population is bf16 (128 hidden): its cross-play too
    wl2 = W.WORKLOADS["lbf12x12_ppo_4096x128"]
    ctx2, pop2 = make_ctx(wl2, 2 * 3 * 33)
    out2 = run_xplay(ctx2, [0, 2], [1, 4, 7], 33, 60)
    check(wl2, pop2, [0, 2], [1, 4, 7], 33, 60, out2, wl2.env_seed)


def test_lbf12_ippo_and_per_episode_calls():
    require_gpu()
    from test_gpu_ippo import check_seat1
    wl = dataclasses.replace(W.WORKLOADS["lbf12x12_ppo_4096x128"],
                             value_head=(1, 1) + (0,) * 7)
    wl = dataclasses.replace(wl, env=dataclasses.replace(wl.env, episode_len=9))
    N, T = 300, 20
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    t0, t1 = aht.traj_buffers(ctx, T), aht.traj_buffers(ctx, T)
    aht.aht_rollout_ippo(ctx, 0, 1, T, t0, t1)
    aht.aht_sync(ctx)
    st1 = st.copy()
    check_rollout(wl, pop_np, t0, st, wl.env_seed, 0, T, 0, [1])
    check_seat1(wl, pop_np, t0, t1, st1, wl.env_seed, 0, T, 0, 1)
    ep = np.zeros(N, np.uint32)
    # episodes that ended in the IPPO call began at their reset step
    dn = np_(t0["dones"])
    for t in range(T):
        ep[dn[t] == 1] = t + 1
    traj = aht.traj_buffers(ctx, T)
    tms = torch.empty(T, N, dtype=torch.int32, device="cuda")
    aht.aht_rollout_resample(ctx, 0, [2, 3, 4], T, traj, tms)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, T, T, 0, [2, 3, 4], ep_step=ep,
                  resample=True, teammates=tms)


def test_lbf9x9_xplay_and_ppo_take_the_sparse_path():
    """A grid between the two paper sizes: 9x9 x 4 channels = 324 features (past 256
    tensor-memory columns), random 1-2 foods and level 2 agents, cross-play and a PPO call."""
    require_gpu()
    base = W.WORKLOADS["lbf12x12_xplay_8x16x128"]
    env = dataclasses.replace(base.env, width=9, height=9, n_food=2, max_agent_level=2, episode_len=40)
    wl = dataclasses.replace(base, env=env, n_policies=6, value_head=(1,) + (0,) * 5)
    ego, tm, P = [0, 1], [2, 5], 50
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    out = run_xplay(ctx, ego, tm, P, 40)
    check(wl, pop_np, ego, tm, P, 40, out, wl.env_seed)
    N, T = 200, 25
    ctx2, _ = make_ctx(wl, N, pop_np=pop_np)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    traj = aht.traj_buffers(ctx2, T)
    aht.aht_rollout(ctx2, 0, [3, 4], T, traj)
    aht.aht_sync(ctx2)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, T, 0, [3, 4])


def test_lbf12_ppo_full_size_4096x128_sampled():
    """The bench's 12x12 PPO configuration (32-env tiles); the oracle replays a sample."""
    require_gpu()
    wl = W.WORKLOADS["lbf12x12_ppo_4096x128"]
    ctx, pop_np = make_ctx(wl, wl.n_envs)
    traj = aht.traj_buffers(ctx, wl.T)
    aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj)
    aht.aht_sync(ctx)
    ids = np.unique(np.concatenate([[0, wl.n_envs - 1], np.random.default_rng(3).integers(0, wl.n_envs, 30)]))
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_envs(d, wl.env_seed, ids)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, wl.T, wl.ego_id, list(wl.pool), env_ids=ids)
