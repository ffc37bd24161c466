"""GPU parity of the PPO ego update (aht_ppo_grad / aht_ppo_update) against the fp64 oracle.

Inputs: a trajectory collected by the ORACLE's own rollout of the LBF 7x7 PPO workload's
ego against its teammate pool (oracle GAE for advantages and targets), with N(0, 0.15)
noise on the recorded log-probabilities so that some ratios leave the clip band; the
learner starts from the workload's seeded ego weights.  Nothing the oracle reads comes
from the GPU.

Tolerances, from the arithmetic of the GPU path (activations and gradients carried as
two bf16, ~2^-17 relative; tanh within 1e-6; fp32 accumulation; W1, W2 as bf16 on both
sides):
  - gradient: |g - o| <= 1e-4 |o| + 1e-4 rms(o of that tensor) (the form of the logit
    tolerance of the rollout);
  - loss diagnostics: 1e-5 relative + 1e-6; the clip fraction counts a ratio decision,
    which may flip for ratios within the arithmetic's error of the band edge: 2 / B;
  - one optimiser step (the first, m_hat = g, v_hat = g^2): the step lr g / (|g| + eps)
    moves by at most lr eps dg / (|g| - dg + eps)^2 for a gradient error dg (capped at
    2 lr where |g| <= dg), plus the fp32 rounding of the weight.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W
from gpu_util import require_gpu

pytestmark = pytest.mark.gpu

WL = "lbf7x7_ppo_16384x128"
REL = 1e-4


def make_batch(T, N, seed):
    wl = W.WORKLOADS[WL]
    d = O.env_desc(*wl.env.astuple())
    pop = W.population(wl)
    st = O.reset_all(d, seed, N)
    out = O.rollout(d, O.Policies(pop), seed, st, 0, T, wl.ego_id, list(wl.pool), n_threads=8)
    adv, tgt = O.gae(out["rewards"], out["values"].astype(np.float32), out["dones"],
                     out["last_value"].astype(np.float32), wl.gamma, wl.lam)
    rng = np.random.default_rng(seed + 100)
    b = dict(obs=out["obs"], actions=out["actions"][..., 0].copy(),
             logp=(out["logp"] + rng.normal(0, 0.15, (T, N))).astype(np.float32),
             values=out["values"].astype(np.float32), advantages=adv.astype(np.float32),
             targets=tgt.astype(np.float32))
    return b, pop[wl.ego_id], wl


def setup(T=8, N=512, data_seed=3, **cfg):
    """cfg: the learner's configuration (seed = its permutation key)."""
    require_gpu()
    b, ego, wl = make_batch(T, N, data_seed)
    traj = {k: torch.from_numpy(np.ascontiguousarray(v)).cuda() for k, v in b.items()}
    layers = [(torch.from_numpy(np.asarray(Wt, np.float32)), torch.from_numpy(np.asarray(bb, np.float32)))
              for Wt, bb in ego]
    L = aht.aht_learner_create(wl.env.obs_dim, wl.env.n_actions, layers, **cfg)
    net = O.ppo_net(wl.env.obs_dim, 128, 128, wl.env.n_actions)
    p0 = O.flat_params([(np.asarray(Wt, np.float64), np.asarray(bb, np.float64)) for Wt, bb in ego])
    return L, traj, O.PpoBatchNp(**b), net, p0


def hp_of(L, **kw):
    c = dict(L.cfg)
    c.update(kw)
    return O.ppo_hp(**c)


def tensor_slices(net):
    D, H, O_ = net.obs_dim, 128, net.n_act + 1
    sizes = [H * D, H, H * H, H, O_ * H, O_]
    off = np.cumsum([0] + sizes)
    return [slice(off[i], off[i + 1]) for i in range(6)]


def check_grad(g, o, net):
    for sl in tensor_slices(net):
        rms = np.sqrt(np.mean(o[sl] ** 2))
        err = np.abs(g[sl] - o[sl])
        bound = REL * np.abs(o[sl]) + REL * rms
        assert (err <= bound).all(), f"gradient slice {sl}: max err/bound {(err / bound).max():.3f}"


def check_stats(s, o, B):
    np.testing.assert_allclose(s[:5], o[:5], rtol=1e-5, atol=1e-6)
    assert abs(s[5] - o[5]) <= 2.0 / B + 1e-7


@pytest.mark.parametrize("epoch,mb", [(0, 0), (0, 3), (1, 2)])
def test_minibatch_gradient(epoch, mb):
    L, traj, batch, net, p0 = setup(epochs=2, minibatches=4, seed=11)
    S = batch.S
    B = S // 4
    g = torch.empty(L.n_params, device="cuda")
    st = torch.empty(6, device="cuda")
    aht.aht_ppo_grad(L, traj, epoch, mb, g, st)
    aht.aht_learner_sync(L)
    idx = O.perm(11, epoch, S)[mb * B:(mb + 1) * B]
    go, so = O.ppo_grad(net, p0, batch, idx, hp_of(L, epoch0=0), n_threads=8)
    check_grad(g.cpu().numpy().astype(np.float64), go, net)
    check_stats(st.cpu().numpy().astype(np.float64), so, B)


def test_single_tile_and_single_minibatch():
    """The smallest batch (one 64-sample tile, one CTA) and a full-batch minibatch."""
    L, traj, batch, net, p0 = setup(T=1, N=64, data_seed=5, epochs=1, minibatches=1)
    g = torch.empty(L.n_params, device="cuda")
    st = torch.empty(6, device="cuda")
    aht.aht_ppo_grad(L, traj, 0, 0, g, st)
    aht.aht_learner_sync(L)
    idx = O.perm(0, 0, 64)
    go, so = O.ppo_grad(net, p0, batch, idx, hp_of(L, epoch0=0))
    check_grad(g.cpu().numpy().astype(np.float64), go, net)
    check_stats(st.cpu().numpy().astype(np.float64), so, 64)


def test_first_adam_step_matches_oracle():
    L, traj, batch, net, p0 = setup(epochs=1, minibatches=1, seed=2, max_grad_norm=0.5)
    stats = torch.empty(1, 6, device="cuda")
    aht.aht_ppo_update(L, traj, stats)
    aht.aht_learner_sync(L)
    p_gpu = torch.empty(L.n_params, device="cuda")
    t, upd = aht.aht_learner_get(L, p_gpu)
    assert (t, upd) == (1, 1)
    p_gpu = p_gpu.cpu().numpy().astype(np.float64)
    hp = hp_of(L, epoch0=0)
    idx = O.perm(2, 0, batch.S)
    g, so = O.ppo_grad(net, p0, batch, idx, hp, n_threads=8)
    norm = np.linalg.norm(g)
    scale = hp.max_grad_norm / norm if norm >= hp.max_grad_norm else 1.0
    p, m, v = p0.copy(), np.zeros_like(p0), np.zeros_like(p0)
    O.adam_step(p, m, v, 0, g.copy(), hp)
    gc = g * scale
    dg = np.zeros_like(g)
    for sl in tensor_slices(net):
        dg[sl] = (REL * np.abs(g[sl]) + REL * np.sqrt(np.mean(g[sl] ** 2))) * scale
    slack = np.maximum(np.abs(gc) - dg, 0.0) + hp.adam_eps
    bound = np.minimum(2 * hp.lr, hp.lr * hp.adam_eps * dg / slack ** 2) + 2.0 ** -23 * np.abs(p) + 1e-12
    err = np.abs(p_gpu - p)
    assert (err <= bound).all(), f"max err/bound {(err / bound).max():.3f}"
    assert np.abs(p - p0).max() > 0.9 * hp.lr        # the step really moved the weights
    check_stats(stats.cpu().numpy()[0].astype(np.float64), so, batch.S)


def test_update_tracks_oracle_over_epochs_and_minibatches():
    """2 epochs x 4 minibatches: each minibatch's permutation slice, step count and
    loss diagnostics; the weights stay within the per-step bound summed over steps."""
    L, traj, batch, net, p0 = setup(epochs=2, minibatches=4, seed=11)
    stats = torch.empty(8, 6, device="cuda")
    aht.aht_ppo_update(L, traj, stats)
    aht.aht_learner_sync(L)
    p_gpu = torch.empty(L.n_params, device="cuda")
    t, upd = aht.aht_learner_get(L, p_gpu)
    assert (t, upd) == (8, 1)
    p, m, v = p0.copy(), np.zeros_like(p0), np.zeros_like(p0)
    hp = hp_of(L, epoch0=0)
    t_o, so = O.ppo_update(net, p, m, v, 0, batch, hp, n_threads=8)
    assert t_o == 8
    dp = np.abs(p_gpu.cpu().numpy().astype(np.float64) - p)
    assert dp.max() <= 2 * hp.lr * 8
    assert dp.mean() <= 0.01 * hp.lr
    sg = stats.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(sg[:, :5], so[:, :5], rtol=1e-3, atol=1e-5)
    assert np.abs(sg[:, 5] - so[:, 5]).max() <= 4.0 / (batch.S // 4)


def test_deterministic_and_state_round_trip():
    L, traj, batch, net, p0 = setup(epochs=1, minibatches=2, seed=4)
    n = L.n_params
    p_a, m_a, v_a = (torch.empty(n, device="cuda") for _ in range(3))
    start = [torch.empty(n, device="cuda") for _ in range(3)]
    aht.aht_learner_get(L, *start)
    aht.aht_ppo_update(L, traj)
    t1, u1 = aht.aht_learner_get(L, p_a, m_a, v_a)
    # back to the start: the same update gives the same bits
    aht.aht_learner_set(L, start[0], start[1], start[2], t=0, updates=0)
    aht.aht_ppo_update(L, traj)
    p_b, m_b, v_b = (torch.empty(n, device="cuda") for _ in range(3))
    t2, u2 = aht.aht_learner_get(L, p_b, m_b, v_b)
    aht.aht_learner_sync(L)
    assert (t1, u1) == (t2, u2) == (2, 1)
    assert torch.equal(p_a, p_b) and torch.equal(m_a, m_b) and torch.equal(v_a, v_b)
    # the next update uses the next epoch counter: a different permutation
    g1, g2 = torch.empty(n, device="cuda"), torch.empty(n, device="cuda")
    aht.aht_learner_set(L, p_a, m_a, v_a, t=2, updates=0)
    aht.aht_ppo_grad(L, traj, 0, 0, g1)
    aht.aht_learner_set(L, p_a, m_a, v_a, t=2, updates=1)
    aht.aht_ppo_grad(L, traj, 0, 0, g2)
    aht.aht_learner_sync(L)
    assert not torch.equal(g1, g2)


def test_push_writes_the_context_policy():
    """After an update, the pushed ego equals a context created from the same weights."""
    L, traj, batch, net, p0 = setup(epochs=1, minibatches=2, seed=6)
    aht.aht_ppo_update(L, traj)
    wl = W.WORKLOADS[WL]
    pop = [[(torch.from_numpy(np.asarray(Wt, np.float32)), torch.from_numpy(np.asarray(bb, np.float32)))
            for Wt, bb in pol] for pol in W.population(wl)[:3]]
    hv = [1, 0, 0]
    ctx = aht.aht_create(wl.env, [[(Wt.cuda(), bb.cuda()) for Wt, bb in pol] for pol in pop], 256,
                         0, has_value_head=hv, weight_dtype=aht.AHT_FP32)
    aht.aht_learner_push(L, ctx, 0)
    p = torch.empty(L.n_params, device="cuda")
    aht.aht_learner_get(L, p)
    aht.aht_learner_sync(L)
    D, H, O_ = wl.env.obs_dim, 128, wl.env.n_actions + 1
    sizes = [H * D, H, H * H, H, O_ * H, O_]
    parts = torch.split(p, sizes)
    ego_new = [(parts[0].view(H, D), parts[1]), (parts[2].view(H, H), parts[3]), (parts[4].view(O_, H), parts[5])]
    ref = aht.aht_create(wl.env, [ego_new] + [[(Wt.cuda(), bb.cuda()) for Wt, bb in pol] for pol in pop[1:]],
                         256, 0, has_value_head=hv, weight_dtype=aht.AHT_FP32)
    obs = traj["obs"][0, :256].contiguous()
    a = torch.empty(256, wl.env.n_actions + 1, device="cuda")
    b = torch.empty_like(a)
    aht.aht_policy_forward(ctx, 0, obs, a)
    aht.aht_policy_forward(ref, 0, obs, b)
    aht.aht_sync(ctx)
    aht.aht_sync(ref)
    assert torch.equal(a, b)
    assert not torch.equal(parts[0].view(H, D).cpu(), pop[0][0][0])
