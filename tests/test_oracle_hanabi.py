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


# Observation offsets of the 660-bit Hanabi encoding (partner hand 125, own knowledge
# 125, partner knowledge 125, fireworks 25, info 8, lives 3, deck 40, discards 50, last
# action 53 = actor 2 | type 4 | colour 5 | rank 5 | slot 5 | card 25 | hinted 5 |
# success 1 | bomb 1, own hints 50, partner hints 50, own slots 5, final round 1).
PH, OK, PK, FW, INFO, LIFE, DECK, DISC, LA, OH, PHH, SLOTS, FR = (
    0, 125, 250, 375, 400, 408, 411, 451, 501, 554, 604, 654, 659)
R, Y, G, Wc, B = range(5)
RANK1 = sum(1 << (c * 5) for c in range(5))       # knowledge bits of every rank-1 card


def card(c, r):
    return c * 5 + r - 1


def scripted_state(orc):
    """Seat 0: R1 G2 B1 Y4 W5; seat 1: G1 R1 Y3 B2 W1; the next draws R3, B4, Y1; the
    rest of the deck in canonical order (the 50 cards are conserved)."""
    s = reset(orc, 0)
    hands = [[card(R, 1), card(G, 2), card(B, 1), card(Y, 4), card(Wc, 5)],
             [card(G, 1), card(R, 1), card(Y, 3), card(B, 2), card(Wc, 1)]]
    head = hands[0] + hands[1] + [card(R, 3), card(B, 4), card(Y, 1)]
    rest = [c * 5 + r - 1 for c in range(5) for r in (1, 1, 1, 2, 2, 3, 3, 4, 4, 5)]
    for x in head:
        rest.remove(x)
    for k, x in enumerate(head + rest):
        s.deck[k] = x
    for p in range(2):
        for k in range(5):
            s.hand[p][k] = hands[p][k]
    assert conserved(s)
    return s


def therm(o, a, n, ones):
    return o[a:a + ones].all() and not o[a + ones:a + n].any()


def last_action(o, *bits):
    want = np.zeros(53, np.uint8)
    want[list(bits)] = 1
    return np.array_equal(o[LA:LA + 53], want)


def test_observation_sections_through_play_hint_discard_and_bomb(orc):
    s = scripted_state(orc)
    full = (1 << 25) - 1
    # turn 0, seat 0 plays R1 from slot 0: a success, then draws R3 into slot 4
    assert step(orc, s, 0) == (0, 1.0)
    o = obs(orc, s, 1)
    partner = [card(G, 2), card(B, 1), card(Y, 4), card(Wc, 5), card(R, 3)]
    assert o[PH:OK].sum() == 5 and all(o[PH + 25 * k + x] for k, x in enumerate(partner))
    assert o[OK:PK].all() and o[PK:FW].all()
    assert o[FW:INFO].sum() == 1 and o[FW + 5 * R + 0] == 1           # red firework at 1
    assert therm(o, INFO, 8, 8) and therm(o, LIFE, 3, 3) and therm(o, DECK, 40, 39)
    assert not o[DISC:LA].any()
    # actor = partner, type play, colour R, rank 1, slot 0, card R1, success
    assert last_action(o, 1, 2 + 0, 6 + R, 11 + 0, 16 + 0, 21 + card(R, 1), 51)
    assert not o[OH:SLOTS].any() and o[SLOTS:FR].all() and o[FR] == 0
    assert o.sum() == 5 + 125 + 125 + 1 + 8 + 3 + 39 + 7 + 5
    # the actor's own view: actor = self
    assert last_action(obs(orc, s, 0), 0, 2 + 0, 6 + R, 11 + 0, 16 + 0, 21 + card(R, 1), 51)

    # turn 1, seat 1 hints rank 1: only seat 0's slot 1 (B1) matches
    assert step(orc, s, 15 + 0) == (0, 0.0)
    o = obs(orc, s, 0)
    for k in range(5):
        bits = sum(int(b) << i for i, b in enumerate(o[OK + 25 * k:OK + 25 * k + 25]))
        assert bits == (RANK1 if k == 1 else full & ~RANK1), k
    assert o[OH:PHH].sum() == 1 and o[OH + 10 * 1 + 5 + 0] == 1        # own slot 1: rank 1
    assert not o[PHH:SLOTS].any()
    assert therm(o, INFO, 8, 7)
    assert last_action(o, 1, 2 + 3, 11 + 0, 46 + 1)                   # hint rank 1, slot 1
    o1 = obs(orc, s, 1)                                                # the hinter's view
    assert np.array_equal(o1[PK:FW], o[OK:PK])
    assert o1[PHH:SLOTS].sum() == 1 and o1[PHH + 10 * 1 + 5] == 1
    assert last_action(o1, 0, 2 + 3, 11 + 0, 46 + 1)

    # turn 2, seat 0 discards W5 from slot 3 and draws B4
    assert step(orc, s, 5 + 3) == (0, 0.0)
    o = obs(orc, s, 1)
    assert o[DISC:LA].sum() == 1 and o[DISC + 10 * Wc + 9] == 1        # the single W5 copy
    assert therm(o, INFO, 8, 8) and therm(o, DECK, 40, 38)
    assert last_action(o, 1, 2 + 1, 6 + Wc, 11 + 4, 16 + 3, 21 + card(Wc, 5))
    # seat 0's hand is now G2 B1 Y4 R3 B4: the hint moved with B1, the new card knows all
    know = [full & ~RANK1, RANK1, full & ~RANK1, full & ~RANK1, full]
    for k in range(5):
        bits = sum(int(b) << i for i, b in enumerate(o[PK + 25 * k:PK + 25 * k + 25]))
        assert bits == know[k], k
    assert o[PHH:SLOTS].sum() == 1 and o[PHH + 10 + 5] == 1

    # turn 3, seat 1 plays B2 from slot 3 on an empty blue firework: a bomb
    assert step(orc, s, 3) == (0, 0.0)
    o = obs(orc, s, 0)
    assert therm(o, LIFE, 3, 2)
    assert o[DISC:LA].sum() == 2 and o[DISC + 10 * Wc + 9] and o[DISC + 10 * B + 3]
    assert last_action(o, 1, 2 + 0, 6 + B, 11 + 1, 16 + 3, 21 + card(B, 2), 52)
    assert o[FW:INFO].sum() == 1 and o[FW + 5 * R] == 1                # score unchanged

    # turn 4, seat 0 hints green: seat 1's hand is G1 R1 Y3 W1 Y1, slot 0 matches
    assert step(orc, s, 10 + G) == (0, 0.0)
    o = obs(orc, s, 1)
    assert o[OH:PHH].sum() == 1 and o[OH + G] == 1                     # own slot 0: green
    bits = sum(int(b) << i for i, b in enumerate(o[OK:OK + 25]))
    assert bits == 0x1F << (5 * G)
    assert last_action(o, 1, 2 + 2, 6 + G, 46 + 0)

    # turn 5, seat 1 discards R1 from slot 1: the first red rank-1 copy
    assert step(orc, s, 5 + 1) == (0, 0.0)
    o = obs(orc, s, 0)
    assert o[DISC:LA].sum() == 3 and o[DISC + 10 * R + 0] == 1 and o[DISC + 10 * R + 1] == 0
    s.disc[card(R, 1)] = 2                                             # a second copy
    o = obs(orc, s, 0)
    assert o[DISC + 10 * R + 0] == 1 and o[DISC + 10 * R + 1] == 1 and o[DISC + 10 * R + 2] == 0
    assert o[DISC + 10 * R + 3] == 0                                   # rank 2 starts at 3


def test_final_round_flag_and_empty_deck_bits(orc):
    s = reset(orc, 21)
    while s.ptr < 50:
        m = legal(orc, s)
        step(orc, s, 5 if m[5] else int(np.flatnonzero(m[10:])[0]) + 10)
    o = obs(orc, s, s.turn % 2)
    assert o[FR] == 1 and not o[DECK:DISC].any()
    assert o[SLOTS:FR].sum() == s.n_hand[s.turn % 2]
