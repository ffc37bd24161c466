"""Per-episode teammate resampling (aht_rollout_resample) against the oracle.

Every env's teammate at every step must equal the oracle's (the draw of the episode's
first step, exact), and the trajectory follows the usual rollout protocol (observations,
rewards, dones exact; sampled actions equal away from CDF edges; logp / values / V_T
within the rollout tolerance; GAE teacher-forced).  Cases: the bf16 tensor-core kernel
with network and rule teammates, fp32-split weights, the CUDA-core kernel, calls that
carry episodes across, a per-call aht_rollout before a per-episode one, the checkpoint, and
the full 16384 x 128 launch on sampled envs."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu
from test_gpu_rollout import check_rollout

pytestmark = pytest.mark.gpu


def run_and_check(wl, ctx, pop_np, st, ep, step0, T, ego, pool, env_ids=None):
    """One per-episode call on the GPU, replayed by the oracle (st and ep advance)."""
    traj = aht.traj_buffers(ctx, T)
    tms = torch.empty(T, ctx.n_envs, dtype=torch.int32, device="cuda")
    aht.aht_rollout_resample(ctx, ego, pool, T, traj, tms)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, step0, T, ego, pool, env_ids=env_ids,
                  ep_step=ep, resample=True, teammates=tms)
    return traj, np_(tms)


def short_lbf(wl, ep_len):
    return dataclasses.replace(wl, env=dataclasses.replace(wl.env, episode_len=ep_len))


def test_bf16_network_and_rule_teammates_two_calls():
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_ppo_16384x128"], 9)
    N, T = 1000, 30
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    ep = np.zeros(N, np.uint32)
    pool = list(range(1, 9)) + [O.heuristic_id("greedy_closest_self"), O.heuristic_id("entitled")]
    for call in range(2):
        _, tms = run_and_check(wl, ctx, pop_np, st, ep, call * T, T, 0, pool)
        # teammates do change within a call (episodes of at most 9 steps), by episode
        assert (tms[1:] != tms[:-1]).any()
        assert set(np.unique(tms)) == set(pool)
    assert aht.aht_step_counter(ctx) == 2 * T


def test_fp32_split_weights():
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_xplay_8x16x256"], 7)
    N, T = 300, 25
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    run_and_check(wl, ctx, pop_np, st, np.zeros(N, np.uint32), 0, T, 0, list(range(8, 24)))


def test_cuda_core_kernel():
    require_gpu()
    base = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    wl = dataclasses.replace(base, env=dataclasses.replace(base.env, episode_len=6))
    N, T = 130, 20
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    run_and_check(wl, ctx, pop_np, st, np.zeros(N, np.uint32), 0, T, 2, [9, 10, 11])


def test_per_call_rollout_then_per_episode_call():
    """A per-call aht_rollout also records where episodes begin, so a per-episode call
    after it draws from the right steps."""
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_ppo_16384x128"], 11)
    N, T = 400, 20
    ctx, pop_np = make_ctx(wl, N)
    d, pols = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    ep = np.zeros(N, np.uint32)
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 0, [3, 4], T, traj)
    aht.aht_sync(ctx)
    acts = np.stack([np_(traj["actions"]), np_(traj["tm_actions"])], -1)
    ref = O.rollout(d, pols, wl.env_seed, st, 0, T, 0, [3, 4], forced=acts, n_threads=8, ep_step=ep)
    assert ref["rc"] == 0 and (ep > 0).any()
    run_and_check(wl, ctx, pop_np, st, ep, T, T, 0, [1, 2, 5])


def test_checkpoint_carries_episode_starts():
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_ppo_16384x128"], 9)
    ctx, _ = make_ctx(wl, 700)
    pool = [1, 2, 3, 4, 5]
    aht.aht_rollout_resample(ctx, 0, pool, 13, aht.traj_buffers(ctx, 13))
    snap = aht.aht_get_state(ctx)
    out = []
    for rep in range(2):
        if rep:
            aht.aht_set_state(ctx, snap)
        t = aht.traj_buffers(ctx, 21)
        tms = torch.empty(21, 700, dtype=torch.int32, device="cuda")
        aht.aht_rollout_resample(ctx, 0, pool, 21, t, tms)
        aht.aht_sync(ctx)
        out.append((t, tms))
    for k in out[0][0]:
        if out[0][0][k] is not None:
            assert torch.equal(out[0][0][k], out[1][0][k]), k
    assert torch.equal(out[0][1], out[1][1])


def test_full_size_16384x128_sampled_envs():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, pop_np = make_ctx(wl, wl.n_envs)
    ids = np.unique(np.concatenate([[0, 1, wl.n_envs - 1],
                                    np.random.default_rng(1).integers(0, wl.n_envs, 45)]))
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_envs(d, wl.env_seed, ids)
    _, tms = run_and_check(wl, ctx, pop_np, st, np.zeros(len(ids), np.uint32), 0, wl.T,
                           wl.ego_id, list(wl.pool), env_ids=ids)
    # every pool member is met, and each env changes teammate at its episode ends only
    assert set(np.unique(tms)) == set(wl.pool)


@pytest.mark.parametrize("N,pool_size", [(1, 3), (131, 256), (300, 1)])
def test_edge_sizes_and_pools(N, pool_size):
    """One env; a ragged batch with a 256-entry pool (more groups than envs, most of them
    empty, indices up to 255); a one-member pool."""
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_ppo_16384x128"], 6)
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    pool = [1 + (k * 7) % 32 for k in range(pool_size)]
    ep = np.zeros(N, np.uint32)
    for call in range(2):
        run_and_check(wl, ctx, pop_np, st, ep, call * 17, 17, 0, pool)


def test_rule_teammates_only():
    require_gpu()
    wl = short_lbf(W.WORKLOADS["lbf7x7_ppo_16384x128"], 10)
    N = 257
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    pool = [O.heuristic_id(n) for n in O.LBF_HEURISTICS]
    _, tms = run_and_check(wl, ctx, pop_np, st, np.zeros(N, np.uint32), 0, 40, 0, pool)
    assert (tms < 0).all()
