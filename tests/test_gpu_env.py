"""GPU env rules vs the oracle in forced-action mode: states, observations, rewards, dones
and auto-resets must be bit-exact given identical action sequences."""
import ctypes as C
import dataclasses
import itertools

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu


def _run_forced(env, wl, n_envs, seed, actions_fn, steps):
    ctx, pop_np = make_ctx(wl, n_envs, seed=seed, env=env)
    d, _ = oracle_of(env, pop_np)
    st = O.reset_all(d, seed, n_envs)
    N, od = n_envs, env.obs_dim
    rew = torch.empty(N, 2, device="cuda")
    team = torch.empty(N, device="cuda")
    dones = torch.empty(N, dtype=torch.uint8, device="cuda")
    obs = torch.empty(N, 2, od, dtype=torch.uint8, device="cuda")
    n_done = 0
    for t in range(steps):
        acts = actions_fn(t, st)
        aht.aht_step_forced(ctx, torch.from_numpy(acts).cuda(), rew, team, dones, obs)
        rc, r2, tm, dn, ob = O.step_forced(d, seed, t, st, acts)
        assert rc == 0
        assert np.array_equal(np_(rew), r2), f"per-agent rewards differ at step {t}"
        assert np.array_equal(np_(team), tm), f"team rewards differ at step {t}"
        assert np.array_equal(np_(dones), dn), f"dones differ at step {t}"
        got = np_(obs)
        if not np.array_equal(got, ob):
            bad = np.argwhere((got != ob).any(-1))
            raise AssertionError(f"obs differ at step {t}, (env, seat) {bad[:5].tolist()}")
        n_done += int(dn.sum())
    aht.aht_sync(ctx)
    assert aht.aht_step_counter(ctx) == steps
    return n_done


@pytest.mark.parametrize("w,h,nf,lvl,ep", [(7, 7, 3, 3, 50), (3, 3, 1, 3, 7), (5, 8, 2, 9, 20),
                                           (12, 12, 3, 2, 30)])
def test_lbf_forced_random(w, h, nf, lvl, ep):
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    env = W.EnvSpec(kind=W.LBF, width=w, height=h, n_food=nf, max_agent_level=lvl, episode_len=ep)
    wl2 = dataclasses.replace(wl, env=env)
    rng = np.random.default_rng(w * 100 + h)
    N = 3001   # ragged: not a multiple of any block size
    # bias toward load so that foods get eaten
    acts_all = rng.integers(0, 6, size=(2 * ep + 5, N, 2)).astype(np.uint8)
    acts_all[rng.random(acts_all.shape) < 0.35] = 5
    dones = _run_forced(env, wl2, N, 17, lambda t, st: acts_all[t], 2 * ep + 5)
    assert dones >= N   # every env finished at least one episode and was reset


@pytest.mark.parametrize("nf", [1, 2])
def test_lbf_3x3_enumeration(nf):
    # All 36^3 joint-action sequences of length 3, one per env, each from its own reset.
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    env = W.EnvSpec(kind=W.LBF, width=3, height=3, n_food=nf, max_agent_level=3, episode_len=50)
    wl2 = dataclasses.replace(wl, env=env)
    N = 36 ** 3
    seqs = np.array(list(itertools.product(range(36), repeat=3)), dtype=np.int64)  # [N][3]

    def acts(t, st):
        ja = seqs[:, t]
        return np.stack([ja // 6, ja % 6], -1).astype(np.uint8)

    _run_forced(env, wl2, N, 5, acts, 3)


def test_overcooked_forced_random():
    require_gpu()
    wl = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    env = W.EnvSpec(kind=W.OVERCOOKED, width=5, height=4, episode_len=60, cook_time=4,
                    soup_reward=20)
    wl2 = dataclasses.replace(wl, env=env)
    rng = np.random.default_rng(3)
    N = 1500
    acts_all = rng.integers(0, 6, size=(130, N, 2)).astype(np.uint8)
    acts_all[rng.random(acts_all.shape) < 0.4] = 5
    _run_forced(env, wl2, N, 9, lambda t, st: acts_all[t], 130)


def _legal_random(rng):
    def fn(t, st):
        n = st.shape[0]
        acts = np.zeros((n, 2), np.uint8)
        legal = np.zeros(20, np.uint8)
        for e in range(n):
            s = O.HanabiState.from_buffer(st[e])
            O.lib().orc_hanabi_legal(C.byref(s), legal.ctypes.data_as(C.c_void_p))
            a = rng.choice(np.flatnonzero(legal))
            acts[e, s.turn % 2] = a
            acts[e, 1 - s.turn % 2] = rng.integers(0, 20)   # ignored seat
        return acts
    return fn


def test_hanabi_forced_random_legal():
    require_gpu()
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    rng = np.random.default_rng(11)
    dones = _run_forced(wl.env, wl, 600, 4, _legal_random(rng), 140)
    assert dones >= 600


def test_hanabi_illegal_forced_action_latches_error():
    require_gpu()
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    ctx, _ = make_ctx(wl, 4, seed=1)
    before = aht.aht_get_state(ctx)
    acts = torch.full((4, 2), 5, dtype=torch.uint8, device="cuda")   # discard at 8 tokens
    aht.aht_step_forced(ctx, acts)
    with pytest.raises(aht.AhtError) as e:
        aht.aht_sync(ctx)
    assert e.value.status == aht.AHT_EDEVICE
    after = aht.aht_get_state(ctx)
    hdr = 40
    assert before[hdr:] == after[hdr:]   # env state untouched
    aht.aht_sync(ctx)                    # the status word was cleared
