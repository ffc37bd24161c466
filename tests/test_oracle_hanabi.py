"""Pins for the oracle's 2-player Hanabi.

Deck: 5 colours x ranks (1,1,1,2,2,3,3,4,4,5); 5-card hands; 8 info and 3 life
tokens; 20 actions (play/discard per slot, colour and rank hints).
"""
import ctypes as C

import numpy as np
import pytest

COPIES = {1: 3, 2: 2, 3: 2, 4: 2, 5: 1}


def reset(orc, seed, env=0):
    s = orc.HanabiState()
    orc.lib().orc_hanabi_reset(seed, env, 0, C.byref(s))
    return s


def legal(orc, s):
    out = np.zeros(20, np.uint8)
    orc.lib().orc_hanabi_legal(C.byref(s), out.ctypes.data_as(C.c_void_p))
    return out


def step(orc, s, a):
    team = np.zeros(1, np.float32)
    done = orc.lib().orc_hanabi_step(C.byref(s), a, team.ctypes.data_as(C.c_void_p))
    return done, float(team[0])


def obs(orc, s, seat):
    out = np.zeros(660, np.uint8)
    orc.lib().orc_hanabi_obs(C.byref(s), seat, out.ctypes.data_as(C.c_void_p))
    return out


def conserved(s):
    counts = np.zeros(25, int)
    for k in range(s.ptr, 50):
        counts[s.deck[k]] += 1
    for p in range(2):
        for k in range(s.n_hand[p]):
            counts[s.hand[p][k]] += 1
    for t in range(25):
        counts[t] += s.disc[t]
    for c in range(5):
        for r in range(1, s.fw[c] + 1):
            counts[c * 5 + r - 1] += 1
    return all(counts[c * 5 + r - 1] == COPIES[r] for c in range(5) for r in range(1, 6))


def test_deal_and_deck_is_a_permutation(orc):
    pos = np.zeros((25, 50))
    for seed in range(400):
        s = reset(orc, seed)
        assert conserved(s)
        assert s.ptr == 10 and s.info == 8 and s.lives == 3 and s.fr == -1
        assert [s.hand[0][k] for k in range(5)] == [s.deck[k] for k in range(5)]
        assert [s.hand[1][k] for k in range(5)] == [s.deck[5 + k] for k in range(5)]
        for k in range(50):
            pos[s.deck[k], k] += 1
    # every card type is spread evenly over deck positions (uniform shuffle)
    for t in range(25):
        share = pos[t] / pos[t].sum()
        assert np.abs(share - 1 / 50).max() < 0.03


def test_legal_mask_hand_cases(orc):
    s = reset(orc, 3)
    m = legal(orc, s)
    assert m[:5].all() and not m[5:10].any()           # 8 info tokens: no discard
    partner = [s.hand[1][k] for k in range(5)]
    for v in range(5):
        assert m[10 + v] == any(c // 5 == v for c in partner)   # hints touching no card
        assert m[15 + v] == any(c % 5 == v for c in partner)    # are illegal
    assert step(orc, s, 5)[0] == -1                     # discarding at 8 tokens rejected
    s.info = 0
    assert not legal(orc, s)[10:].any()
    s.info = 4
    assert legal(orc, s)[5:10].all()


def test_hint_restricts_knowledge(orc):
    s = reset(orc, 11)
    m = legal(orc, s)
    a = int(np.flatnonzero(m[10:15])[0]) + 10
    colour = a - 10
    done, r = step(orc, s, a)
    assert done == 0 and r == 0.0 and s.info == 7 and s.turn == 1
    for k in range(5):
        card = s.hand[1][k]
        colmask = 0x1F << (5 * colour)
        if card // 5 == colour:
            assert s.know[1][k] == colmask and s.hint_col[1][k] == 1 << colour
            assert (s.la_hinted >> k) & 1
        else:
            assert s.know[1][k] == ((1 << 25) - 1) & ~colmask and s.hint_col[1][k] == 0
    o = obs(orc, s, 1)   # seat 1 acts next; its own knowledge sits at [125, 250)
    for k in range(5):
        bits = o[125 + 25 * k: 150 + 25 * k]
        assert int(sum(int(b) << i for i, b in enumerate(bits))) == s.know[1][k]
    la = o[501:554]
    assert la[1] == 1 and la[2 + 2] == 1 and la[6 + colour] == 1   # partner hinted colour


def test_reset_obs_thermometers(orc):
    s = reset(orc, 5)
    o = obs(orc, s, 0)
    for k in range(5):
        assert o[25 * k + s.hand[1][k]] == 1 and o[25 * k: 25 * k + 25].sum() == 1
    assert o[125:250].all() and o[250:375].all()
    assert o[375:400].sum() == 0
    assert o[400:408].all() and o[408:411].all() and o[411:451].all()
    assert o[451:554].sum() == 0 and o[554:654].sum() == 0
    assert o[654:659].all() and o[659] == 0
    assert o.sum() == 5 + 250 + 8 + 3 + 40 + 5


def _cheater(orc, s):
    """Perfect-information policy: play a playable card, else discard a dead or
    duplicated card, else hint (to pass), else discard slot 0."""
    me = s.turn % 2
    m = legal(orc, s)
    hand = [s.hand[me][k] for k in range(s.n_hand[me])]
    for k, c in enumerate(hand):
        if s.fw[c // 5] == c % 5:
            return k
    if m[10:].any():
        return int(np.flatnonzero(m[10:])[0]) + 10
    for k, c in enumerate(hand):
        if c % 5 < s.fw[c // 5]:
            return 5 + k
    return 5


def test_rule_invariants_and_scripted_perfect_game(orc):
    best = 0
    for seed in range(60):
        s = reset(orc, seed)
        rng = np.random.default_rng(seed)
        total = 0.0
        for turn in range(100):
            a = _cheater(orc, s) if seed % 2 == 0 else int(rng.choice(np.flatnonzero(legal(orc, s))))
            assert legal(orc, s)[a]
            done, r = step(orc, s, a)
            total += r
            assert conserved(s)
            assert 0 <= s.score <= 25 and 0 <= s.info <= 8 and 0 <= s.lives <= 3
            assert s.score == sum(s.fw)
            if done:
                break
        assert done == 1 and s.turn <= 97
        assert total == s.ret
        if s.lives == 0:
            assert s.ret == 0.0
        else:
            assert s.ret == s.score
            assert s.score == 25 or (s.fr == 0 and s.ptr == 50)
        if seed % 2 == 0:
            best = max(best, s.score)
            if s.score == 25:
                assert s.ret == 25.0
    assert best == 25


def test_final_round_gives_two_more_turns(orc):
    s = reset(orc, 21)
    # burn the deck by discarding (after spending a token on a hint when at 8)
    while s.ptr < 50:
        m = legal(orc, s)
        a = 5 if m[5] else int(np.flatnonzero(m[10:])[0]) + 10
        done, _ = step(orc, s, a)
        assert done == 0
    assert s.fr == 2
    t_empty = s.turn
    m = legal(orc, s)
    done1, _ = step(orc, s, int(np.flatnonzero(m)[0]))
    m = legal(orc, s)
    done2, _ = step(orc, s, int(np.flatnonzero(m)[0]))
    assert (done1, done2) == (0, 1) and s.turn == t_empty + 2


def test_losing_all_lives_zeroes_return(orc):
    for seed in range(200):
        s = reset(orc, seed)
        # play slot 0 until the game ends; collect one game that scores then bombs out
        rets = []
        while True:
            done, r = step(orc, s, 0)
            rets.append(r)
            if done:
                break
        if s.lives == 0 and max(rets) > 0:
            assert sum(rets) == 0.0 and rets[-1] == -float(sum(1 for x in rets if x == 1.0))
            return
    pytest.fail("no scoring game that lost all lives")
