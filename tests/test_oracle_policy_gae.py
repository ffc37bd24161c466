"""Pins for the oracle's policy forward, masked categorical sampling, GAE and drivers."""
import ctypes as C

import numpy as np
import pytest
import torch

from paper_2609_13716_gb300 import workloads as W


def rand_policy(rng, dims, scale=0.1):
    return [(rng.standard_normal((dims[i + 1], dims[i])) * scale,
             rng.standard_normal(dims[i + 1]) * scale) for i in range(3)]


def test_mlp_matches_torch_float64(orc):
    rng = np.random.default_rng(0)
    pol = rand_policy(rng, [196, 64, 64, 7])
    P = orc.Policies([pol])
    obs = rng.integers(0, 7, size=(50, 196)).astype(np.uint8)
    got = P.outputs(0, obs)
    x = torch.from_numpy(obs.astype(np.float64))
    for W_, b in pol:
        x = x @ torch.from_numpy(W_).T + torch.from_numpy(b)
        if W_ is not pol[-1][0]:
            x = torch.tanh(x)
    assert np.allclose(got, x.numpy(), rtol=1e-13, atol=1e-13)


def test_zero_weights_give_bias_and_uniform_policy(orc):
    dims = [196, 64, 64, 6]
    rng = np.random.default_rng(1)
    pol = [(np.zeros((dims[i + 1], dims[i])), np.zeros(dims[i + 1])) for i in range(3)]
    b3 = rng.standard_normal(6)
    P = orc.Policies([pol[:2] + [(np.zeros((6, 64)), b3)]])
    assert np.array_equal(P.outputs(0, np.ones((1, 196), np.uint8))[0], b3)
    legal = np.ones(6, np.uint8)
    for u in (0.0, 0.1, 0.49, 0.5, 0.83, 0.999):
        a, lp, _ = orc.sample(np.zeros(6), legal, u)
        assert a == int(np.floor(u * 6)) and abs(lp + np.log(6)) < 1e-15


def test_sample_is_inverse_cdf_of_masked_softmax(orc):
    rng = np.random.default_rng(2)
    for _ in range(300):
        K = int(rng.choice([6, 20]))
        z = rng.standard_normal(K) * 3
        legal = (rng.random(K) < 0.7).astype(np.uint8)
        legal[rng.integers(K)] = 1
        u = rng.random()
        a, lp, mg = orc.sample(z, legal, u)
        p = np.where(legal == 1, np.exp(z - z[legal == 1].max()), 0.0)
        cdf = np.cumsum(p) / p.sum()
        assert a == int(np.searchsorted(cdf, u, side="right"))
        assert legal[a] == 1
        logsm = torch.log_softmax(torch.from_numpy(np.where(legal == 1, z, -np.inf)), 0).numpy()
        assert abs(lp - logsm[a]) < 1e-12
        assert abs(mg - np.abs(u - cdf).min()) < 1e-12


def test_onehot_last_layer_is_deterministic_argmax(orc):
    dims = [196, 64, 64, 6]
    pol = [(np.zeros((dims[i + 1], dims[i])), np.zeros(dims[i + 1])) for i in range(3)]
    b3 = np.zeros(6)
    b3[4] = 60.0   # a margin of e^60
    P = orc.Policies([pol[:2] + [(np.zeros((6, 64)), b3)]])
    z = P.outputs(0, np.zeros((1, 196), np.uint8))[0]
    for u in np.linspace(1e-6, 0.999999, 17):   # u = 0 picks action 0 (S_0 = e^-60 > 0)
        assert orc.sample(z, np.ones(6, np.uint8), u)[0] == 4


def _gae_inputs(rng, T=40, N=7, p_done=0.1):
    r = rng.standard_normal((T, N)).astype(np.float32)
    v = rng.standard_normal((T, N)).astype(np.float32)
    d = (rng.random((T, N)) < p_done).astype(np.uint8)
    vl = rng.standard_normal(N).astype(np.float32)
    return r, v, d, vl


def test_gae_lambda_one_is_discounted_return_minus_value(orc):
    rng = np.random.default_rng(3)
    r, v, d, vl = _gae_inputs(rng, p_done=0.0)
    g = 0.99
    adv, tgt = orc.gae(r, v, d, vl, g, 1.0)
    T = r.shape[0]
    for t in range(T):
        ret = sum(g ** (k - t) * r[k].astype(np.float64) for k in range(t, T)) + g ** (T - t) * vl.astype(np.float64)
        assert np.allclose(adv[t], ret - v[t], atol=1e-11)
        assert np.allclose(tgt[t], ret, atol=1e-11)


def test_gae_lambda_zero_is_td_error(orc):
    rng = np.random.default_rng(4)
    r, v, d, vl = _gae_inputs(rng)
    g = 0.99
    adv, _ = orc.gae(r, v, d, vl, g, 0.0)
    vnext = np.concatenate([v[1:], vl[None]], 0).astype(np.float64)
    delta = r.astype(np.float64) + g * (1 - d) * vnext - v
    assert np.allclose(adv, delta, atol=1e-13)


def test_gae_geometric_closed_form(orc):
    T, N, g, lam, c = 64, 3, 0.99, 0.95, 0.5
    r = np.full((T, N), c, np.float32)
    z = np.zeros((T, N), np.float32)
    adv, _ = orc.gae(r, z, z.astype(np.uint8), np.zeros(N, np.float32), g, lam)
    for t in range(T):
        n = T - t
        q = g * lam
        assert np.allclose(adv[t], c * (1 - q ** n) / (1 - q), atol=1e-12)


def test_gae_done_cuts_recursion(orc):
    rng = np.random.default_rng(5)
    r, v, d, vl = _gae_inputs(rng, p_done=0.0)
    d[10] = 1
    a1, _ = orc.gae(r, v, d, vl, 0.99, 0.95)
    r2 = r.copy()
    r2[11:] += 5.0   # changes after the cut must not reach t <= 10
    v2 = v.copy()
    v2[11:] -= 2.0
    a2, _ = orc.gae(r2, v2, d, vl + 1, 0.99, 0.95)
    assert np.array_equal(a1[:11], a2[:11])
    assert not np.allclose(a1[11:], a2[11:])


def test_rollout_matches_stepwise_replay(orc):
    # The PPO driver = reset + per-step forced stepping with auto-reset at step t+1.
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    d = orc.env_desc(*wl.env.astuple())
    pols = orc.Policies(W.population(wl))
    N, T, seed = 16, 120, 9
    st = orc.reset_all(d, seed, N)
    out = orc.rollout(d, pols, seed, st, 0, T, 0, [1])
    assert out["rc"] == 0
    st2 = orc.reset_all(d, seed, N)
    for t in range(T):
        rc, _, team, dones, obs2 = orc.step_forced(d, seed, t, st2, out["actions"][t])
        assert rc == 0
        assert np.array_equal(team, out["rewards"][t]) and np.array_equal(dones, out["dones"][t])
        if t + 1 < T:
            assert np.array_equal(obs2[:, 0], out["obs"][t + 1])
            assert np.array_equal(obs2[:, 1], out["obs_tm"][t + 1])
    assert np.array_equal(st, st2)
    assert out["dones"].sum() >= N   # 50-step episodes: every env resets at least once
    # free running: applied actions are the oracle's own samples
    assert np.array_equal(out["actions"], out["own_actions"])


def test_rollout_teammate_draw_is_per_env(orc):
    """Sec. 3: the ego meets teammates drawn uniformly from the training pool.  Per call,
    every env draws its own: env e plays pool[floor(x |pool| / 2^32)], x = word 0 of the
    counter (e, step0, stream 3).  Checked at the 16,384 envs of the PPO workload: the
    rule for every env (x from the Philox pinned against Triton), a chi-square over 32
    pool members, neighbouring envs independent (no block structure), and a new draw
    when step0 changes."""
    from scipy import stats
    d = orc.env_desc(orc.LBF, 7, 7, 3, 3, 50)
    od, K = orc.obs_dim(d), orc.n_actions(d)
    rng = np.random.default_rng(2)
    pols = orc.Policies([[(rng.standard_normal((n, m)) * 0.1, rng.standard_normal(n) * 0.1)
                          for m, n in ((od, 4), (4, 4), (4, K))] for _ in range(33)])
    N, seed = 16384, 2
    pool = list(range(1, 33))
    st = orc.reset_all(d, seed, N)
    tm = orc.rollout(d, pols, seed, st, 5, 1, 0, pool, n_threads=8)["teammate"]
    x = np.array([orc.draw(seed, e, 5, 3, 0) for e in range(N)], np.uint64)
    assert np.array_equal(tm, np.asarray(pool)[(x * 32) >> 32])
    c = np.bincount(tm - 1, minlength=32)
    assert stats.chisquare(c).pvalue > 1e-3
    # no 128-env (or any) blocks: consecutive envs agree about 1/32 of the time
    same = (tm[1:] == tm[:-1]).mean()
    assert abs(same - 1 / 32) < 5 * np.sqrt((1 / 32) * (31 / 32) / (N - 1))
    # a later call (another step0) draws anew, independently of the first
    tm2 = orc.rollout(d, pols, seed, st, 6, 1, 0, pool, n_threads=8)["teammate"]
    assert abs((tm2 == tm).mean() - 1 / 32) < 0.01


def test_xplay_matrix_is_pair_mean(orc):
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    d = orc.env_desc(*wl.env.astuple())
    pols = orc.Policies(W.population(wl)[:4])
    out = orc.xplay(d, pols, 4, 0, [0, 1], [2, 3], 8, 100, n_threads=4)
    assert out["rc"] == 0
    R = out["returns"].reshape(2, 2, 8).astype(np.float64)
    assert np.array_equal(out["matrix"], R.mean(-1).astype(np.float32))
    assert (out["steps"] <= 97).all() and (out["steps"] > 0).all()
    # Hanabi returns are integers in [0, 25]
    assert np.array_equal(R, np.round(R)) and R.min() >= 0 and R.max() <= 25
    # only the acting seat samples
    acts = out["actions"]
    for s in range(100):
        live = acts[s, :, 0] != 255
        assert (acts[s, :, 1 - s % 2] == 255).all()
        assert ((acts[s, :, s % 2] != 255) == (out["steps"] > s)).all()


def test_xplay_logits_output_is_what_the_sampler_used(orc):
    """The cross-play logits output (a parity-test record) is the forward the oracle
    sampled from: re-sampling it with the same draw gives the recorded own action, and an
    independent torch fp64 forward of the seat-0 reset observation gives the same values."""
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    d = orc.env_desc(*wl.env.astuple())
    layers = W.population(wl)[:4]
    pols = orc.Policies(layers)
    out = orc.xplay(d, pols, 4, 0, [0, 1], [2, 3], 3, 100, n_threads=4, logit_stride=32)
    assert out["rc"] == 0
    L, own = out["logits"], out["own_actions"]
    n = 0
    for s in range(6):
        for e in range(12):
            seat = s % 2
            if own[s, e, seat] == 255:
                assert np.isnan(L[s, e, seat]).all()
                continue
            assert np.isnan(L[s, e, 1 - seat]).all()      # only the acting seat runs
            z = L[s, e, seat, :20]
            assert np.isnan(L[s, e, seat, 20:]).all()
            u = (int(orc.draw(4, e, s, seat, 0)) >> 8) * 2.0 ** -24
            if s == 0:
                st = orc.reset_envs(d, 4, [e])
                legal = np.zeros(20, np.uint8)
                hs = orc.HanabiState.from_buffer(st)
                orc.lib().orc_hanabi_legal(C.byref(hs), legal.ctypes.data_as(C.c_void_p))
                o = np.zeros(660, np.uint8)
                orc.lib().orc_hanabi_obs(C.byref(hs), 0, o.ctypes.data_as(C.c_void_p))
                pid = [0, 1][e // 6]
                x = torch.from_numpy(o.astype(np.float64))
                for k, (Wt, b) in enumerate(layers[pid]):
                    x = torch.from_numpy(np.asarray(Wt, np.float64)) @ x + torch.from_numpy(np.asarray(b, np.float64))
                    if k < 2:
                        x = torch.tanh(x)
                assert np.allclose(z, x.numpy(), rtol=1e-12, atol=1e-12)
                a, _, _ = orc.sample(z, legal, u)
                assert a == own[s, e, seat]
                n += 1
    assert n == 12
