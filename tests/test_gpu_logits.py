"""Every output of the tensor-core kernels' policy evaluations against the fp64 oracle.

The rollout and cross-play tests see only what the kernels keep (the sampled action, its
logp, the ego's value).  Here the parity hook (aht_debug_logits) records each
evaluation's whole output vector -- every logit, and the value row where the policy has
one -- and each element is compared with the oracle's forward of the same observation
(protocol M3: |g - o| <= 1e-4 |o| + 1e-4 rms(o) over the tensor), for every MLP shape the
tensor-core kernels run:
  - the two-warp-group kernel: PPO collection with bf16 196-128-128-7 ego and
    196-128-128-6 teammates (gathered tiles, contiguous tiles) and fp32 196-64-64-6
    (split weights); IPPO collection (both seats' networks); LBF cross-play with fp32
    196-64-64-6 (split weights, frozen envs evaluated too);
  - LBF 12x12 PPO collection with the sparse first layer (576-128-128);
  - cross-play on the streamed kernel: Overcooked 520-256-256-6, Hanabi 660-512-512-20
    and Mini Hanabi 156-256-256-10.
Every case has at least 1200 evaluated rows per seat and step range."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import close, make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu
S = aht.AHT_DEBUG_STRIDE


def ppo_logits(wl_name, N, T, pool, ego=0, ippo=False):
    """Runs one collection call with the hook set; returns the GPU outputs, the
    trajectory and the oracle's forced replay."""
    wl = W.WORKLOADS[wl_name]
    ctx, pop_np = make_ctx(wl, N)
    buf = torch.full((T, N, 2, S), float("nan"), device="cuda")
    aht.aht_debug_logits(ctx, buf)
    traj = aht.traj_buffers(ctx, T)
    if ippo:
        traj1 = aht.traj_buffers(ctx, T)
        aht.aht_rollout_ippo(ctx, ego, pool[0], T, traj, traj1)
    else:
        aht.aht_rollout(ctx, ego, pool, T, traj)
    aht.aht_sync(ctx)
    aht.aht_debug_logits(ctx, None)
    d, pols = oracle_of(wl.env, pop_np)
    acts = np.stack([np_(traj["actions"]), np_(traj["tm_actions"])], -1)
    ref = O.rollout(d, pols, wl.env_seed, O.reset_all(d, wl.env_seed, N), 0, T, ego, pool,
                    forced=acts, n_threads=8)
    assert ref["rc"] == 0
    return wl, pols, np_(buf), np_(traj["obs"]), ref


def check_ppo(wl, pols, g, obs, ref, ego, n_act):
    T, N = obs.shape[:2]
    n_ego = pols.arr[ego].n_out
    want = np.stack([pols.outputs(ego, obs[t]) for t in range(T)])
    ok, worst = close(g[:, :, 0, :n_ego], want)
    assert ok, f"ego outputs {worst:.3g}"
    assert np.isnan(g[:, :, 0, 8:]).all() and (g[:, :, 0, n_ego:8] == 0).all()
    tm = ref["teammate"]
    nets = tm >= 0
    if nets.any():
        got, exp = [], []
        for pid in np.unique(tm[nets]):
            sel = tm == pid
            n_out = pols.arr[pid].n_out
            for t in range(T):
                got.append(g[t, sel, 1, :n_out])
                exp.append(pols.outputs(int(pid), ref["obs_tm"][t, sel]))
        ok, worst = close(np.concatenate(got), np.concatenate(exp))
        assert ok, f"teammate outputs {worst:.3g}"
    assert np.isnan(g[:, ~nets, 1]).all()  # rule teammates evaluate no network


@pytest.mark.parametrize("pool", [list(range(1, 33)), [5]], ids=["gathered", "contiguous"])
def test_ppo_bf16_outputs(pool):
    require_gpu()
    wl, pols, g, obs, ref = ppo_logits("lbf7x7_ppo_16384x128", 1200, 4, pool)
    check_ppo(wl, pols, g, obs, ref, 0, 6)


def test_ppo_bf16_outputs_with_rule_teammates():
    require_gpu()
    wl, pols, g, obs, ref = ppo_logits("lbf7x7_ppo_16384x128", 1300, 3, [3, -2, 7, -9])
    check_ppo(wl, pols, g, obs, ref, 0, 6)


def test_ppo_fp32_split_outputs():
    require_gpu()
    wl, pols, g, obs, ref = ppo_logits("lbf7x7_64x50_fp32", 1200, 4, [1])
    check_ppo(wl, pols, g, obs, ref, 0, 6)


def test_ippo_outputs():
    require_gpu()
    wl, pols, g, obs, ref = ppo_logits("lbf7x7_ippo_16384x128", 1200, 3, [1], ippo=True)
    check_ppo(wl, pols, g, obs, ref, 0, 6)


def test_lbf12_sparse_first_layer_outputs():
    require_gpu()
    wl, pols, g, obs, ref = ppo_logits("lbf12x12_ppo_4096x128", 1200, 3, [1, 2, 3, 4])
    check_ppo(wl, pols, g, obs, ref, 0, 6)


@pytest.mark.parametrize("name,ego,tm,P,steps", [
    ("lbf7x7_xplay_8x16x256", [0, 7], [8, 15, 23], 200, 24),
    ("overcooked5x4_xplay_8x8x64", [0, 1], [8, 9], 300, 6),
    ("hanabi_xplay_16x16x32", [0, 5], [16, 30], 300, 100),      # to termination
    ("minihanabi_xplay_16x16x32", [1, 2], [17, 20], 300, 100),
])
def test_xplay_outputs(name, ego, tm, P, steps):
    require_gpu()
    wl = W.WORKLOADS[name]
    n = len(ego) * len(tm) * P
    ctx, pop_np = make_ctx(wl, n)
    buf = torch.full((steps, n, 2, S), float("nan"), device="cuda")
    aht.aht_debug_logits(ctx, buf)
    matrix = torch.empty(len(ego), len(tm), device="cuda")
    actions = torch.empty(steps, n, 2, dtype=torch.uint8, device="cuda")
    aht.aht_xplay_matrix(ctx, ego, tm, P, steps, matrix, actions=actions)
    aht.aht_sync(ctx)
    aht.aht_debug_logits(ctx, None)
    d, pols = oracle_of(wl.env, pop_np)
    ref = O.xplay(d, pols, wl.env_seed, 0, ego, tm, P, steps, forced=np_(actions), n_threads=8,
                  logit_stride=S)
    assert ref["rc"] == 0
    g, want = np_(buf), ref["logits"]
    n_out = pols.arr[ego[0]].n_out
    live = np.isfinite(want[..., 0])               # the oracle's evaluations
    assert live.sum() >= 1200
    assert np.isfinite(g[..., 0][live]).all()      # each one was made on the GPU too
    ok, worst = close(g[..., :n_out][live], want[..., :n_out][live])
    assert ok, f"outputs {worst:.3g}"


def test_hook_rejects_a_short_buffer():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, _ = make_ctx(wl, 256)
    buf = torch.zeros(4 * 256 * 2 * S - 1, device="cuda")
    aht.aht_debug_logits(ctx, buf)
    traj = aht.traj_buffers(ctx, 4)
    with pytest.raises(aht.AhtError):
        aht.aht_rollout(ctx, 0, [1, 2], 4, traj)
    assert aht.aht_step_counter(ctx) == 0      # nothing launched, the counter stays
    aht.aht_debug_logits(ctx, None)
    aht.aht_rollout(ctx, 0, [1, 2], 4, traj)
    aht.aht_sync(ctx)
