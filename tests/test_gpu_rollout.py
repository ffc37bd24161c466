"""PPO rollout collection on the GPU vs the oracle.

Protocol: the oracle replays every env with the GPU's own joint actions.  Observations,
rewards, dones, teammate assignments and auto-resets must be bit-exact; the GPU's
action must equal the oracle's own fp64 sample wherever the oracle's u lies at least
1e-5 from a CDF edge; logp, values and V_T agree within the fp32/fp64 tolerance; GAE is
checked teacher-forced on the GPU's own r, v, d and V_T.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import CDF_MARGIN, GAE_REL, close, make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu


def check_rollout(wl, pop_np, traj, states, seed, step0, T, ego, pool, env_ids=None, ep_step=None,
                  resample=False, teammates=None):
    """Replays the GPU's applied actions in the oracle and compares.  ep_step / resample:
    per-episode teammates (teammates: the GPU's per-step teammate ids, compared exactly)."""
    d, pols = oracle_of(wl.env, pop_np)
    sel = slice(None) if env_ids is None else env_ids
    acts = np.stack([np_(traj["actions"])[:, sel], np_(traj["tm_actions"])[:, sel]], -1)
    ref = O.rollout(d, pols, seed, states, step0, T, ego, pool, forced=acts, n_threads=8,
                    env_ids=env_ids, ep_step=ep_step, resample=resample)
    if teammates is not None:
        assert np.array_equal(np_(teammates)[:, sel], ref["teammates_t"]), "per-step teammates"
    assert ref["rc"] == 0
    assert np.array_equal(np_(traj["teammate"])[sel], ref["teammate"]), "teammate draw"
    if traj.get("obs") is not None:
        assert np.array_equal(np_(traj["obs"])[:, sel], ref["obs"]), "observations"
    assert np.array_equal(np_(traj["rewards"])[:, sel], ref["rewards"]), "rewards"
    assert np.array_equal(np_(traj["dones"])[:, sel], ref["dones"]), "dones"
    agree = (ref["own_actions"] == acts) | (ref["margin"] < CDF_MARGIN)
    assert agree.all(), f"{(~agree).sum()} sampled actions differ away from a CDF edge"
    flagged = (ref["margin"] < CDF_MARGIN).sum()
    ok, worst = close(np_(traj["logp"])[:, sel], ref["logp"])
    assert ok, f"logp {worst:.3g}"
    if wl.value_head[ego]:
        ok, worst = close(np_(traj["values"])[:, sel], ref["values"])
        assert ok, f"values {worst:.3g}"
        ok, worst = close(np_(traj["last_value"])[sel], ref["last_value"])
        assert ok, f"V_T {worst:.3g}"
    # teacher-forced GAE
    r = np_(traj["rewards"])[:, sel]
    v = np_(traj["values"])[:, sel]
    dn = np_(traj["dones"])[:, sel]
    vl = np_(traj["last_value"])[sel]
    a_ref, t_ref = O.gae(r, v, dn, vl, 0.99, 0.95)
    ok, worst = close(np_(traj["advantages"])[:, sel], a_ref, GAE_REL)
    assert ok, f"advantages {worst:.3g}"
    ok, worst = close(np_(traj["targets"])[:, sel], t_ref, GAE_REL)
    assert ok, f"targets {worst:.3g}"
    return flagged


def test_c0_rollout_64x50_fp32():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, pop_np = make_ctx(wl, 64)
    traj = aht.traj_buffers(ctx, 50)
    aht.aht_rollout(ctx, 0, [1], 50, traj)
    aht.aht_sync(ctx)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, 64)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, 50, 0, [1])


def test_ppo_bf16_population_two_calls_and_ragged_groups():
    # The 33-policy bf16 population of the 16384-env workload on 1000 envs: 32 teammate
    # groups of ragged sizes, two consecutive calls (the env state and step counter carry).
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    N, T = 1000, 40
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    for call in range(2):
        traj = aht.traj_buffers(ctx, T)
        aht.aht_rollout(ctx, 0, wl.pool, T, traj)
        aht.aht_sync(ctx)
        check_rollout(wl, pop_np, traj, st, wl.env_seed, call * T, T, 0, list(wl.pool))
    assert aht.aht_step_counter(ctx) == 2 * T


def test_overcooked_ppo_rollout():
    require_gpu()
    wl = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    N, T = 130, 30
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 2, [9, 10, 11], T, traj)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, T, 2, [9, 10, 11])


def test_checkpoint_resume_is_bit_exact():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, _ = make_ctx(wl, 700)
    traj0 = aht.traj_buffers(ctx, 13)
    aht.aht_rollout(ctx, 0, wl.pool, 13, traj0)
    snap = aht.aht_get_state(ctx)
    a = aht.traj_buffers(ctx, 21)
    aht.aht_rollout(ctx, 0, wl.pool, 21, a)
    aht.aht_set_state(ctx, snap)
    assert aht.aht_step_counter(ctx) == 13
    b = aht.traj_buffers(ctx, 21)
    aht.aht_rollout(ctx, 0, wl.pool, 21, b)
    aht.aht_sync(ctx)
    for k in a:
        if a[k] is not None:
            assert torch.equal(a[k], b[k]), k


def test_full_size_16384x128_sampled_envs():
    # The bench launch configuration; the oracle replays a sample of 48 envs.
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, pop_np = make_ctx(wl, wl.n_envs)
    traj = aht.traj_buffers(ctx, wl.T)
    aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj)
    aht.aht_sync(ctx)
    ids = np.unique(np.concatenate([[0, 1, wl.n_envs - 1],
                                    np.random.default_rng(0).integers(0, wl.n_envs, 45)]))
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_envs(d, wl.env_seed, ids)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, wl.T, wl.ego_id, list(wl.pool), env_ids=ids)
    # every env's teammate draw, bit-exact against the oracle's (one step of all envs)
    ref = O.rollout(d, O.Policies(pop_np), wl.env_seed, O.reset_all(d, wl.env_seed, wl.n_envs), 0, 1,
                    wl.ego_id, list(wl.pool), n_threads=8)
    assert ref["rc"] == 0
    assert np.array_equal(np_(traj["teammate"]), ref["teammate"]), "teammate draws"
    # properties over all envs: dones at most every 50 steps, rewards in [0, 1]
    r = np_(traj["rewards"])
    assert (r >= 0).all() and (r <= 1.0 + 1e-6).all()
    assert (np_(traj["dones"]).sum(0) >= 2).all()


@pytest.mark.parametrize("N,pool", [
    (1, list(range(1, 33)) * 8),             # one env, a 256-entry pool: one tile
    (300, list(range(1, 33)) * 8),           # most of 256 groups empty or single-env
    (517, [5, 5, 5, 7]),                     # repeated ids: entries are drawn, not ids
    (2000, [-1, 3, -12, 4, -6]),             # rule teammates among networks
])
def test_per_call_teammate_groups_edge_cases(N, pool):
    """Per-call teammate draws grouped into gathered tensor-core tiles: a single env,
    empty and single-env groups, repeated pool ids and rule teammates."""
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    T = 12
    ctx, pop_np = make_ctx(wl, N)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 0, pool, T, traj)
    aht.aht_sync(ctx)
    check_rollout(wl, pop_np, traj, st, wl.env_seed, 0, T, 0, pool)


def test_traj_copy_to_pinned_host_and_device():
    # aht_traj_copy (the API's trajectory download) delivers every field bit for bit, to
    # pinned host buffers and to another set of device buffers; a field missing on either
    # side is skipped.
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    N, T = 300, 12
    ctx, _ = make_ctx(wl, N)
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 0, wl.pool, T, traj, 0.99, 0.95)
    host = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in traj.items()}
    host["targets"] = None
    dev = aht.traj_buffers(ctx, T)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    aht.aht_sync(ctx)
    aht.aht_traj_copy(traj, host, N, T, ctx.obs_dim, stream)
    aht.aht_traj_copy(traj, dev, N, T, ctx.obs_dim, stream)
    stream.synchronize()
    for k, v in traj.items():
        if host[k] is not None:
            assert torch.equal(host[k], v.cpu()), k
        assert torch.equal(dev[k].cpu(), v.cpu()), k
    with pytest.raises(ValueError):  # the binding checks the shapes (the C call: test_abi)
        aht.aht_traj_copy(traj, host, 0, T, ctx.obs_dim, stream)
