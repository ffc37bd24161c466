"""Pins for the oracle's 2-player Mini Hanabi (3 colours x 3 ranks; the remaining rules are
the readings stated in aht_oracle.h: ranks (1,1,1,2,2,3) per colour, 2-card hands, 3 info
and 1 life tokens, 10 actions, the full game's rules and observation at this size)."""
import ctypes as C

import numpy as np
import pytest

COPIES = {1: 3, 2: 2, 3: 1}


def reset(orc, seed, env=0):
    s = orc.MiniHanabiState()
    orc.lib().orc_mhanabi_reset(seed, env, 0, C.byref(s))
    return s


def legal(orc, s):
    out = np.zeros(10, np.uint8)
    orc.lib().orc_mhanabi_legal(C.byref(s), out.ctypes.data_as(C.c_void_p))
    return out


def step(orc, s, a):
    team = np.zeros(1, np.float32)
    done = orc.lib().orc_mhanabi_step(C.byref(s), a, team.ctypes.data_as(C.c_void_p))
    return done, float(team[0])


def obs(orc, s, seat):
    out = np.zeros(156, np.uint8)
    orc.lib().orc_mhanabi_obs(C.byref(s), seat, out.ctypes.data_as(C.c_void_p))
    return out


def conserved(s):
    """Every card is in the deck, a hand, the discards or on a firework, exactly once."""
    counts = np.zeros(9, int)
    for k in range(s.ptr, 18):
        counts[s.deck[k]] += 1
    for p in range(2):
        for k in range(s.n_hand[p]):
            counts[s.hand[p][k]] += 1
    for t in range(9):
        counts[t] += s.disc[t]
    for c in range(3):
        for r in range(1, s.fw[c] + 1):
            counts[c * 3 + r - 1] += 1
    want = np.array([COPIES[t % 3 + 1] for t in range(9)])
    return np.array_equal(counts, want)


def test_deal_and_deck(orc):
    for seed in range(20):
        s = reset(orc, seed)
        deck = np.array(s.deck[:])
        assert sorted(np.bincount(deck, minlength=9).tolist()) == [1, 1, 1, 2, 2, 2, 3, 3, 3]
        for t in range(9):
            assert np.count_nonzero(deck == t) == COPIES[t % 3 + 1]
        assert [s.hand[0][0], s.hand[0][1], s.hand[1][0], s.hand[1][1]] == deck[:4].tolist()
        assert (s.ptr, s.info, s.lives, s.score, s.fr, s.turn) == (4, 3, 1, 0, -1, 0)
        assert conserved(s)


def test_legal_mask_by_hand(orc):
    s = reset(orc, 1)
    # seed 1: own hand types (8, 2), partner (1, 0): colour 0 ranks 2 and 1
    s.hand[0][0], s.hand[0][1], s.hand[1][0], s.hand[1][1] = 8, 2, 1, 0
    lg = legal(orc, s)
    # plays yes; discards no (info at its maximum 3); hint colour 0 only; ranks 1 and 2
    assert lg.tolist() == [1, 1, 0, 0, 1, 0, 0, 1, 1, 0]
    s.info = 0
    assert legal(orc, s).tolist() == [1, 1, 1, 1, 0, 0, 0, 0, 0, 0]


def test_play_hint_discard_trace_by_hand(orc):
    s = reset(orc, 1)
    s.hand[0][0], s.hand[0][1], s.hand[1][0], s.hand[1][1] = 0, 4, 1, 8   # R1 G2 | R2 B3
    s.info = 2
    # seat 0 plays slot 0 (red 1): success, reward 1, hand shifts and draws deck[4]
    top = s.deck[4]
    done, r = step(orc, s, 0)
    assert (done, r, s.score, s.fw[0], s.turn) == (0, 1.0, 1, 1, 1)
    assert (s.hand[0][0], s.hand[0][1], s.ptr) == (4, top, 5)
    # seat 1 hints colour 0 (red) to seat 0: no red in (G2, top) unless top is red
    done, r = step(orc, s, 4) if top // 3 == 0 else step(orc, s, 5)
    assert (done, r, s.info) == (0, 0.0, 1)
    # seat 0 discards slot 0 (green 2): info back to 2, discard count
    done, r = step(orc, s, 2)
    assert (done, s.info, s.disc[4]) == (0, 2, 1)
    # the last action as seen by seat 1: partner discarded green 2 from slot 0
    o = obs(orc, s, 1)
    la = o[99:126]
    assert la[1] == 1 and la[2 + 1] == 1 and la[6 + 1] == 1 and la[9 + 1] == 1 and la[12] == 1
    assert la[14 + 4] == 1 and la.sum() == 6


def test_bomb_ends_the_game_and_zeroes_the_return(orc):
    s = reset(orc, 3)
    s.hand[0][0] = 5    # green 3 on an empty green firework: a bomb
    s.score = 0
    done, r = step(orc, s, 0)
    assert done == 1 and s.lives == 0 and r == 0.0
    s = reset(orc, 3)
    s.fw[0], s.score, s.ret = 1, 1, 1.0
    s.hand[0][0] = 2    # red 3 on red 1: a bomb with one point scored
    done, r = step(orc, s, 0)
    assert done == 1 and r == -1.0 and s.ret == 0.0


def test_random_games_keep_the_invariants(orc):
    rng = np.random.default_rng(0)
    lengths = []
    for g in range(300):
        s = reset(orc, g)
        for t in range(100):
            lg = legal(orc, s)
            assert lg.sum() >= 1
            a = int(rng.choice(np.flatnonzero(lg)))
            done, r = step(orc, s, a)
            assert done in (0, 1)
            assert 0 <= s.info <= 3 and 0 <= s.lives <= 1 and 0 <= s.score <= 9
            assert conserved(s)
            o0, o1 = obs(orc, s, 0), obs(orc, s, 1)
            assert o0[:18].sum() == s.n_hand[1] and o1[:18].sum() == s.n_hand[0]
            assert o0[63:66].sum() == s.info and o0[66] == s.lives
            assert o0[67:81].sum() == 18 - s.ptr
            if done:
                break
        assert done == 1
        lengths.append(s.turn)
    assert max(lengths) <= 40


def test_final_round_two_more_turns(orc):
    s = reset(orc, 5)
    s.ptr = 17          # one card left in the deck
    s.info = 0
    done, _ = step(orc, s, 2)    # seat 0 discards and draws the last card
    assert (done, s.ptr, s.fr) == (0, 18, 2)
    done, _ = step(orc, s, 2)    # seat 1: first final turn
    assert (done, s.fr) == (0, 1)
    done, _ = step(orc, s, 2)    # seat 0: the last one
    assert (done, s.fr) == (1, 0)


def test_observation_sections_by_hand(orc):
    s = reset(orc, 7)
    o = obs(orc, s, 0)
    # partner hand one-hot (2 x 9), own knowledge all-ones for 2 slots (2 x 9), same for
    # the partner's, no fireworks, 3 info, 1 life, 14 deck cards, no discards, no last
    # action, no hints, 2 own slots, no final round
    assert o[:18].sum() == 2
    assert o[s.hand[1][0]] == 1 and o[9 + s.hand[1][1]] == 1
    assert o[18:36].all() and o[36:54].all()
    assert not o[54:63].any()
    assert o[63:66].all() and o[66] == 1 and o[67:81].all() and not o[81:99].any()
    assert not o[99:150].any() and o[150:152].all() and o[152] == 0
    assert not o[153:].any()   # the 3 padding features
