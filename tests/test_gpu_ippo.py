"""IPPO collection (both seats learn: aht_rollout_ippo) against the oracle.

Seat 0's trajectory must be the one aht_rollout writes for the pool {policy1} (the same
draws and states, bit for bit); seat 1's is checked against the oracle's teammate-seat
outputs: observations, actions, rewards and dones exactly, logp / values / V_T within the
rollout tolerance, GAE teacher-forced.  Both kernels: the tensor-core rollout (bf16 and
fp32-split weights) and the CUDA-core one (the wide Overcooked-style kitchen policies)."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import GAE_REL, close, make_ctx, np_, oracle_of, require_gpu
from test_gpu_rollout import check_rollout

pytestmark = pytest.mark.gpu


def check_seat1(wl, pop_np, traj0, traj1, states, seed, step0, T, p0, p1, env_ids=None):
    d, pols = oracle_of(wl.env, pop_np)
    sel = slice(None) if env_ids is None else env_ids
    g = lambda k: np_(traj1[k])[:, sel] if traj1[k].dim() > 1 else np_(traj1[k])[sel]
    acts = np.stack([np_(traj0["actions"])[:, sel], np_(traj0["tm_actions"])[:, sel]], -1)
    ref = O.rollout(d, pols, seed, states, step0, T, p0, [p1], forced=acts, n_threads=8,
                    env_ids=env_ids)
    assert ref["rc"] == 0
    assert np.array_equal(g("obs"), ref["obs_tm"]), "seat-1 observations"
    assert np.array_equal(g("actions"), acts[..., 1])
    assert np.array_equal(g("tm_actions"), acts[..., 0])
    assert np.array_equal(g("rewards"), ref["rewards"])
    assert np.array_equal(g("dones"), ref["dones"])
    ok, worst = close(g("logp"), ref["logp_tm"])
    assert ok, f"seat-1 logp {worst:.3g}"
    ok, worst = close(g("values"), ref["values_tm"])
    assert ok, f"seat-1 values {worst:.3g}"
    ok, worst = close(g("last_value"), ref["last_value_tm"])
    assert ok, f"seat-1 V_T {worst:.3g}"
    a_ref, t_ref = O.gae(g("rewards"), g("values"), g("dones"), g("last_value"), 0.99, 0.95)
    ok, worst = close(g("advantages"), a_ref, GAE_REL)
    assert ok, f"seat-1 advantages {worst:.3g}"
    ok, worst = close(g("targets"), t_ref, GAE_REL)
    assert ok, f"seat-1 targets {worst:.3g}"


def run_case(wl, N, T, p0, p1, calls=1):
    ctx, pop_np = make_ctx(wl, N)
    ref_ctx, _ = make_ctx(wl, N, pop_np=pop_np)
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, N)
    for call in range(calls):
        traj0 = aht.traj_buffers(ctx, T)
        traj1 = aht.traj_buffers(ctx, T)
        aht.aht_rollout_ippo(ctx, p0, p1, T, traj0, traj1)
        plain = aht.traj_buffers(ref_ctx, T)
        aht.aht_rollout(ref_ctx, p0, [p1], T, plain)
        aht.aht_sync(ctx)
        aht.aht_sync(ref_ctx)
        for k in ("obs", "actions", "tm_actions", "logp", "values", "rewards", "dones",
                  "advantages", "targets", "last_value", "teammate"):
            assert torch.equal(traj0[k], plain[k]), f"seat-0 {k} differs from aht_rollout"
        st1 = st.copy()
        check_rollout(wl, pop_np, traj0, st, wl.env_seed, call * T, T, p0, [p1])
        check_seat1(wl, pop_np, traj0, traj1, st1, wl.env_seed, call * T, T, p0, p1)
        assert np.array_equal(st, st1)
    return ctx, traj0, traj1


def test_ippo_bf16_tensor_core_two_calls_ragged():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ippo_16384x128"]
    run_case(wl, 1000, 40, 0, 1, calls=2)          # 8 tiles, the last one ragged


def test_ippo_fp32_split_weights():
    require_gpu()
    wl = dataclasses.replace(W.WORKLOADS["lbf7x7_64x50_fp32"], value_head=(1, 1))
    run_case(wl, 64, 50, 1, 0)                     # seats swapped: policy 1 in seat 0


def test_ippo_cuda_core_kernel():
    require_gpu()
    base = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    wl = dataclasses.replace(base, value_head=(1,) * base.n_policies)
    run_case(wl, 130, 30, 2, 9)


def test_ippo_learners_consume_both_seats():
    """One IPPO iteration: a learner per seat updates on its own trajectory and pushes its
    weights back; the next collection runs, and the pushed policies are the ones used."""
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ippo_16384x128"]
    N, T = 512, 16
    ctx, pop_np = make_ctx(wl, N)
    traj = [aht.traj_buffers(ctx, T), aht.traj_buffers(ctx, T)]
    aht.aht_rollout_ippo(ctx, 0, 1, T, traj[0], traj[1])
    learners = []
    for seat in range(2):
        layers = [(torch.from_numpy(np.asarray(Wt, np.float32)), torch.from_numpy(np.asarray(bb, np.float32)))
                  for Wt, bb in pop_np[seat]]
        L = aht.aht_learner_create(wl.env.obs_dim, wl.env.n_actions, layers, epochs=1,
                                   minibatches=2, seed=seat)
        aht.aht_sync(ctx)
        aht.aht_ppo_update(L, traj[seat])
        aht.aht_learner_push(L, ctx, seat)
        aht.aht_learner_sync(L)
        learners.append(L)
    # the context's seat-1 policy is now the learner's weights, rounded to bf16
    obs = traj[1]["obs"][0].contiguous()
    p = torch.empty(learners[1].n_params, device="cuda")
    aht.aht_learner_get(learners[1], p)
    aht.aht_learner_sync(learners[1])
    flat = W.round_to_bf16(np_(p)).astype(np.float64)
    D, H, A = wl.env.obs_dim, 128, wl.env.n_actions + 1
    sizes = np.cumsum([0, H * D, H, H * H, H, A * H, A])
    parts = [flat[sizes[i]:sizes[i + 1]] for i in range(6)]
    pushed = [(parts[0].reshape(H, D), parts[1]), (parts[2].reshape(H, H), parts[3]),
              (parts[4].reshape(A, H), parts[5])]
    want = O.Policies([pushed]).outputs(0, np_(obs))
    before = O.Policies(pop_np).outputs(1, np_(obs))
    out = torch.empty(N, A, device="cuda")
    aht.aht_policy_forward(ctx, 1, obs, out)
    aht.aht_sync(ctx)
    ok, worst = close(np_(out), want)
    assert ok, f"pushed seat-1 policy {worst:.3g}"
    assert np.abs(want - before).max() > 1e-4        # and it moved
    t2 = [aht.traj_buffers(ctx, T), aht.traj_buffers(ctx, T)]
    aht.aht_rollout_ippo(ctx, 0, 1, T, t2[0], t2[1])
    aht.aht_sync(ctx)
    assert torch.isfinite(t2[1]["logp"]).all() and (t2[1]["logp"] <= 0).all()


def test_ippo_rejects_rule_and_out_of_range_seat1():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ippo_16384x128"]
    ctx, _ = make_ctx(wl, 128)
    t0, t1 = aht.traj_buffers(ctx, 4), aht.traj_buffers(ctx, 4)
    for bad in (-1, 2):
        with pytest.raises(aht.AhtError):
            aht.aht_rollout_ippo(ctx, 0, bad, 4, t0, t1)


def test_ippo_full_size_16384x128_sampled():
    """The bench's IPPO configuration; the oracle replays a sample of the envs."""
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ippo_16384x128"]
    ctx, pop_np = make_ctx(wl, wl.n_envs)
    t0, t1 = aht.traj_buffers(ctx, wl.T), aht.traj_buffers(ctx, wl.T)
    aht.aht_rollout_ippo(ctx, 0, 1, wl.T, t0, t1)
    aht.aht_sync(ctx)
    ids = np.unique(np.concatenate([[0, wl.n_envs - 1], np.random.default_rng(2).integers(0, wl.n_envs, 30)]))
    d, _ = oracle_of(wl.env, pop_np)
    st = O.reset_envs(d, wl.env_seed, ids)
    st1 = st.copy()
    check_rollout(wl, pop_np, t0, st, wl.env_seed, 0, wl.T, 0, [1], env_ids=ids)
    check_seat1(wl, pop_np, t0, t1, st1, wl.env_seed, 0, wl.T, 0, 1, env_ids=ids)
