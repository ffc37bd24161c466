"""Pins for the oracle's 5x4 Overcooked-style kitchen.

Layout (x right, y down): row 0 "# O # P #", row 1 "# . . . #", row 2 "D . . . S",
row 3 "# # O # #".  A pot cooks three onions for cook_time steps; a delivered soup pays
soup_reward to the team.
"""
import ctypes as C

import numpy as np

NOOP, N, S, E, W, INTERACT = range(6)
NONE, ONION, DISH, SOUP = range(4)


def desc(orc, ep=400):
    return orc.env_desc(orc.OVERCOOKED, 5, 4, 0, 0, ep, 20, 20)


def step(orc, d, s, a0, a1):
    r = np.zeros(2, np.float32)
    team = np.zeros(1, np.float32)
    done = orc.lib().orc_oc_step(C.byref(d), C.byref(s), a0, a1, r.ctypes.data_as(C.c_void_p),
                                 team.ctypes.data_as(C.c_void_p))
    return float(team[0]), done


def fresh(orc, d):
    s = orc.OcState()
    orc.lib().orc_oc_reset(C.byref(d), C.byref(s))
    return s


def obs(orc, d, s, seat):
    out = np.zeros(520, np.uint8)
    orc.lib().orc_oc_obs(C.byref(d), C.byref(s), seat, out.ctypes.data_as(C.c_void_p))
    return out.reshape(4, 5, 26)


def test_layout(orc):
    L = orc.lib()
    rows = ["#O#P#", "#...#", "D...S", "##O##"]
    code = {"#": 1, ".": 0, "O": 2, "P": 3, "D": 4, "S": 5}
    for y, row in enumerate(rows):
        for x, ch in enumerate(row):
            assert L.orc_oc_cell(x, y) == code[ch]


# Agent 0's scripted soup: three onion trips from the dispenser at (1,0) to the pot at
# (3,0), a dish from (0,2), then the soup to the serving cell (4,2).  Agent 1 steps
# out of the way to (2,2) first and then waits.
ONION_TRIP = [W, W, N, INTERACT, E, E, N, INTERACT]   # from (3,1) back to (3,1)
SCRIPT = ([INTERACT, E, E, N, INTERACT] + ONION_TRIP + ONION_TRIP +
          [W, W, S, W, INTERACT, N, E, E, N])          # to the dish and back, t = 21..29


def test_scripted_soup_and_cook_timer(orc):
    d = desc(orc)
    s = fresh(orc, d)
    log = []
    t = 0
    for a in SCRIPT:
        team, _ = step(orc, d, s, a, W if t == 0 else NOOP)
        log.append((t, s.held[0], s.pot_n, s.pot_timer, team))
        t += 1
    # third onion goes in at step 20: cooking starts with timer = cook_time
    assert log[20][2:4] == (3, 20)
    assert log[4][2] == 1 and log[12][2] == 2
    assert log[25][1] == DISH and (s.ax[0], s.ay[0], s.face[0]) == (3, 1, 0)
    # the pot was cooking at the start of steps 21..40, so it is ready from step 41 on:
    # an interact at step 40 fails and one at step 41 serves the soup into the dish
    while t < 41:
        step(orc, d, s, INTERACT, NOOP)
        assert s.held[0] == DISH, t
        t += 1
    assert s.pot_timer == 0 and s.pot_n == 3
    step(orc, d, s, INTERACT, NOOP)   # t = 41
    assert s.held[0] == SOUP and s.pot_n == 0
    step(orc, d, s, S, NOOP)          # (3,2)
    step(orc, d, s, E, NOOP)          # serving cell is not floor: turn east
    team, _ = step(orc, d, s, INTERACT, NOOP)
    assert team == 20.0 and s.held[0] == NONE and s.ret == 20.0


def test_swap_and_same_target_block(orc):
    d = desc(orc)
    s = fresh(orc, d)
    s.ax[0], s.ay[0], s.ax[1], s.ay[1] = 1, 1, 2, 1
    step(orc, d, s, E, W)   # swap
    assert (s.ax[0], s.ax[1]) == (1, 2) and (s.face[0], s.face[1]) == (2, 3)
    s.ax[0], s.ay[0], s.ax[1], s.ay[1] = 1, 1, 3, 1
    step(orc, d, s, E, W)   # both into (2,1)
    assert (s.ax[0], s.ax[1]) == (1, 3)
    s.ax[0], s.ay[0], s.ax[1], s.ay[1] = 1, 1, 2, 1
    step(orc, d, s, E, E)   # follow into a cell being vacated
    assert (s.ax[0], s.ax[1]) == (2, 3)


def test_counter_place_and_pick(orc):
    d = desc(orc)
    s = fresh(orc, d)
    step(orc, d, s, INTERACT, NOOP)   # onion
    step(orc, d, s, W, NOOP)          # face the counter at (0,1)
    step(orc, d, s, INTERACT, NOOP)
    assert s.held[0] == NONE and s.counter_item[1 * 5 + 0] == ONION
    assert obs(orc, d, s, 1)[1, 0, 15] == 1
    step(orc, d, s, INTERACT, NOOP)
    assert s.held[0] == ONION and s.counter_item[5] == NONE


def test_reset_obs_channels(orc):
    d = desc(orc)
    s = fresh(orc, d)
    o = obs(orc, d, s, 0)
    assert o[1, 1, 0] == 1 and o[1, 1, 2] == 1          # self at (1,1) facing N
    assert o[2, 3, 1] == 1 and o[2, 3, 6] == 1          # other at (3,2) facing N
    assert o[0, 3, 11] == 1 and o[0, 1, 12] == 1 and o[3, 2, 12] == 1
    assert o[2, 0, 13] == 1 and o[2, 4, 14] == 1
    assert o[:, :, 10].sum() == 9 and o[:, :, 25].sum() == 0
    assert o.sum() == 2 * 2 + 9 + 5
    o1 = obs(orc, d, s, 1)
    assert o1[2, 3, 0] == 1 and o1[1, 1, 1] == 1
    s.ep_t = 360
    assert obs(orc, d, s, 0)[:, :, 25].sum() == 20


def test_random_play_invariants(orc):
    d = desc(orc, ep=400)
    L = orc.lib()
    rng = np.random.default_rng(0)
    for env in range(40):
        s = fresh(orc, d)
        acts = rng.integers(0, 6, size=(400, 2))
        # bias toward interact so that items move around
        acts[rng.random((400, 2)) < 0.3] = INTERACT
        for t, (a0, a1) in enumerate(acts):
            team, done = step(orc, d, s, int(a0), int(a1))
            assert team in (0.0, 20.0, 40.0)
            assert 0 <= s.pot_n <= 3 and 0 <= s.pot_timer <= 20
            assert s.pot_timer == 0 or s.pot_n == 3
            for i in range(2):
                assert L.orc_oc_cell(s.ax[i], s.ay[i]) == 0
            assert (s.ax[0], s.ay[0]) != (s.ax[1], s.ay[1])
            assert done == (t == 399)
        assert s.ret % 20 == 0


def test_item_pot_and_holding_channels_along_the_soup_script(orc):
    """Channels 15-24 at hand-worked points of the scripted soup (index (y*5 + x)*26 + c;
    15/16/17 onion/dish/soup on a counter or in a hand at the holder's cell, 18/19/20 pot
    with 1/2/3 onions, 21 cooking, 22 ready, 23 self holding, 24 other holding).  Agent 0
    starts at (1,1), the pot is at (3,0), agent 1 waits at (2,2)."""
    d = desc(orc)
    s = fresh(orc, d)
    POT = (0, 3)                                      # (y, x)

    def ch(seat):
        return obs(orc, d, s, seat)[:, :, 15:25]      # channels 15..24 as [..., 0..9]

    def only(o, *cells):
        """the 10 channels are zero except at the listed (y, x, c) entries"""
        want = np.zeros_like(o)
        for y, x, c in cells:
            want[y, x, c - 15] = 1
        return np.array_equal(o, want)

    t = 0

    def run(a0):
        nonlocal t
        step(orc, d, s, a0, W if t == 0 else NOOP)
        t += 1

    assert only(ch(0)) and only(ch(1))               # empty kitchen
    run(SCRIPT[0])                                    # t0: agent 0 takes an onion at (1,1)
    assert s.held[0] == ONION
    assert only(ch(0), (1, 1, 15), (1, 1, 23))        # onion in own hand, self holding
    assert only(ch(1), (1, 1, 15), (1, 1, 24))        # seen by the other: other holding
    for a in SCRIPT[1:5]:                             # t1..t4: first onion into the pot
        run(a)
    assert s.pot_n == 1
    assert only(ch(0), (*POT, 18)) and only(ch(1), (*POT, 18))
    for a in SCRIPT[5:13]:                            # second onion (t12)
        run(a)
    assert s.pot_n == 2 and only(ch(0), (*POT, 19))
    for a in SCRIPT[13:21]:                           # third onion (t20): cooking starts
        run(a)
    assert (s.pot_n, s.pot_timer) == (3, 20)
    assert only(ch(0), (*POT, 20), (*POT, 21))
    for a in SCRIPT[21:]:                             # to the dish dispenser and back
        run(a)
        if s.held[0] == DISH:
            y, x = s.ay[0], s.ax[0]
            assert only(ch(0), (*POT, 20), (*POT, 21), (y, x, 16), (y, x, 23))
            assert only(ch(1), (*POT, 20), (*POT, 21), (y, x, 16), (y, x, 24))
    assert s.held[0] == DISH and (s.ax[0], s.ay[0]) == (3, 1)
    while t < 41:                                     # still cooking through t40
        assert ch(0)[POT[0], POT[1], 21 - 15] == 1
        run(INTERACT)
    assert s.pot_timer == 0                           # ready after t40
    assert only(ch(0), (*POT, 20), (*POT, 22), (1, 3, 16), (1, 3, 23))
    run(INTERACT)                                     # t41: soup into the dish, pot empties
    assert s.held[0] == SOUP
    assert only(ch(0), (1, 3, 17), (1, 3, 23)) and only(ch(1), (1, 3, 17), (1, 3, 24))
    run(E)                                            # (4,1) is a counter: turn east
    run(INTERACT)                                     # soup placed on the counter at (4,1)
    assert s.held[0] == NONE and s.counter_item[1 * 5 + 4] == SOUP
    assert only(ch(0), (1, 4, 17)) and only(ch(1), (1, 4, 17))
    s.counter_item[0 * 5 + 0] = DISH                  # a dish on the corner counter (0,0)
    assert only(ch(0), (1, 4, 17), (0, 0, 16))
    s.held[1] = ONION                                 # the other agent holds an onion at (2,2)
    assert only(ch(0), (1, 4, 17), (0, 0, 16), (2, 2, 15), (2, 2, 24))
    assert only(ch(1), (1, 4, 17), (0, 0, 16), (2, 2, 15), (2, 2, 23))
