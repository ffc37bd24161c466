"""The observation rows of the streamed cross-play kernel -- the word-level bit writers of
Overcooked, Hanabi and Mini Hanabi, read through aht_debug_obs_words -- against the fp64
oracle's observations of the same states, bit by bit (feature k = bit k; then the
constant-1 bias input; then zeros), for both seats, along forced play long enough to
reach every section's late-game values: the urgency channel of the kitchen, an empty
Hanabi deck and the final round (play that mostly discards), auto-resets in between."""
import ctypes as C

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu


def _check_rows(env, wl, N, seed, actions_fn, steps, every, state_cls=None):
    ctx, pop_np = make_ctx(wl, N, seed=seed, env=env)
    d, _ = oracle_of(env, pop_np)
    st = O.reset_all(d, seed, N)
    od = env.obs_dim
    words = (od + 32) // 32
    out = torch.zeros(N, words, dtype=torch.int32, device="cuda")
    obs = torch.empty(N, 2, od, dtype=torch.uint8, device="cuda")
    final_rounds = 0
    checked = 0
    for t in range(steps):
        acts = actions_fn(t, st)
        aht.aht_step_forced(ctx, torch.from_numpy(acts).cuda(), None, None, None, obs)
        rc, _, _, _, ob = O.step_forced(d, seed, t, st, acts)
        assert rc == 0
        assert np.array_equal(np_(obs), ob)            # the byte path agrees (as in test_gpu_env)
        in_final = 0 if state_cls is None else sum(state_cls.from_buffer(st[e]).fr >= 0 for e in range(N))
        final_rounds += in_final
        if t % every and not in_final:   # every final-round state is checked
            continue
        for seat in (0, 1):
            aht.aht_debug_obs_words(ctx, seat, out)
            aht.aht_sync(ctx)
            bits = np.unpackbits(np_(out).view(np.uint8), axis=1, bitorder="little")
            want = np.zeros((N, words * 32), np.uint8)
            want[:, :od] = ob[:, seat]
            want[:, od] = 1
            if not np.array_equal(bits, want):
                e, k = np.argwhere(bits != want)[0]
                raise AssertionError(f"step {t} seat {seat}: env {e} feature {k}: "
                                     f"kernel {bits[e, k]} oracle {want[e, k]}")
            checked += 1
    return checked, final_rounds


def _deck_out_actions(rng, state_cls, legal_fn, n_act, discard, hint_lo):
    """Discard when that is legal, else hint, else any legal action: no bombs, so games
    run the deck out and reach the final round."""
    def fn(t, st):
        n = st.shape[0]
        acts = np.zeros((n, 2), np.uint8)
        legal = np.zeros(n_act, np.uint8)
        for e in range(n):
            s = state_cls.from_buffer(st[e])
            legal_fn(C.byref(s), legal.ctypes.data_as(C.c_void_p))
            ok = np.flatnonzero(legal)
            disc = ok[(ok >= discard[0]) & (ok < discard[1])]
            hint = ok[ok >= hint_lo]
            a = rng.choice(disc) if len(disc) else rng.choice(hint) if len(hint) else rng.choice(ok)
            acts[e, s.turn % 2] = a
            acts[e, 1 - s.turn % 2] = rng.integers(0, n_act)   # ignored seat
        return acts
    return fn


def test_hanabi_rows_match_the_oracle():
    require_gpu()
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    rng = np.random.default_rng(31)
    fn = _deck_out_actions(rng, O.HanabiState, O.lib().orc_hanabi_legal, 20, (5, 10), 10)
    checked, final_rounds = _check_rows(wl.env, wl, 160, 7, fn, 120, 3, O.HanabiState)
    assert checked >= 80 and final_rounds > 0


def test_minihanabi_rows_match_the_oracle():
    require_gpu()
    wl = W.WORKLOADS["minihanabi_xplay_16x16x32"]
    rng = np.random.default_rng(32)
    fn = _deck_out_actions(rng, O.MiniHanabiState, O.lib().orc_mhanabi_legal, 10, (2, 4), 4)
    checked, final_rounds = _check_rows(wl.env, wl, 200, 8, fn, 60, 2, O.MiniHanabiState)
    assert checked >= 60 and final_rounds > 0


def test_overcooked_rows_match_the_oracle():
    require_gpu()
    import dataclasses
    wl = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    env = W.EnvSpec(kind=W.OVERCOOKED, width=5, height=4, episode_len=60, cook_time=4, soup_reward=20)
    wl2 = dataclasses.replace(wl, env=env)
    rng = np.random.default_rng(33)
    acts_all = rng.integers(0, 6, size=(130, 600, 2)).astype(np.uint8)
    acts_all[rng.random(acts_all.shape) < 0.4] = 5
    checked, _ = _check_rows(env, wl2, 600, 9, lambda t, st: acts_all[t], 130, 4)
    assert checked >= 60


def test_hook_rejects_lbf_and_bad_seats():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_ppo_16384x128"]
    ctx, _ = make_ctx(wl, 64)
    out = torch.zeros(64, (wl.env.obs_dim + 32) // 32, dtype=torch.int32, device="cuda")
    with pytest.raises(aht.AhtError):
        aht.aht_debug_obs_words(ctx, 0, out)
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    ctx, _ = make_ctx(wl, 8)
    out = torch.zeros(8, (wl.env.obs_dim + 32) // 32, dtype=torch.int32, device="cuda")
    with pytest.raises(aht.AhtError):
        aht.aht_debug_obs_words(ctx, 2, out)
