"""Pins of the oracle's rule-based LBF teammates (no GPU).

The paper's LBF heuristic suite (App. F): Greedy picks the next uneaten food online by
closest_self / closest_teammate / closest_avg / lowest_level / highest_level; Sequential
plans a food order before the episode by lexicographic / reverse_lexicographic /
column_major / reverse_column_major / nearest_agent / farthest_agent; Entitled picks a pair
of squares beside a food and waits for the teammate to stand on one before taking the
other and loading.  The movement and
tie rules are the readings stated in aht_oracle.h.  Every expected action below is worked
out by hand from those statements on a 5 x 5 grid (x right, y down; 1 N, 2 S, 3 W, 4 E,
5 load, 0 noop).
"""
import numpy as np
import pytest

import oracle as O

N_, S_, W_, E_, LOAD, NOOP = 1, 2, 3, 4, 5, 0
H = {n: k for k, n in enumerate(O.LBF_HEURISTICS)}


def desc(w=5, h=5, n_food=3):
    return O.env_desc(O.LBF, w, h, n_food, 3, 50)


def state(a0, a1, foods, levels=(1, 1), init1=None, eaten=(0, 0, 0)):
    s = O.LbfState()
    s.ax[0], s.ay[0] = a0
    s.ax[1], s.ay[1] = a1
    s.al[0], s.al[1] = levels
    for k, (x, y, lv) in enumerate(foods):
        s.fx[k], s.fy[k], s.fl[k] = x, y, lv
        s.eaten[k] = eaten[k]
    for k in range(len(foods), 3):
        s.eaten[k] = 1
    s.F = sum(f[2] for f in foods)
    s.ix[0], s.iy[0] = a0
    s.ix[1], s.iy[1] = init1 if init1 is not None else a1
    return s


# agent 1 (the heuristic) at (2, 2), agent 0 at (0, 0); foods: 0 at (4, 2) level 1,
# 1 at (2, 0) level 3, 2 at (0, 4) level 2
BASE = dict(a0=(0, 0), a1=(2, 2), foods=[(4, 2, 1), (2, 0, 3), (0, 4, 2)])


@pytest.mark.parametrize("name,want", [
    # distances from (2,2): 2, 2, 4 -> tie, food 0 (lower index) -> dx = 2: east
    ("greedy_closest_self", E_),
    # from (0,0): 6, 2, 4 -> food 1 (2,0): dy = -2: north
    ("greedy_closest_teammate", N_),
    # sums 8, 4, 8 -> food 1
    ("greedy_closest_avg", N_),
    # levels 1, 3, 2 -> food 0
    ("greedy_lowest_level", E_),
    ("greedy_highest_level", N_),
    # row-major indices 2*5+4 = 14, 0*5+2 = 2, 4*5+0 = 20 -> food 1 first
    ("seq_lexicographic", N_),
    # descending -> food 2 (0,4): dx = -2, dy = 2, tie -> x first: west
    ("seq_reverse_lexicographic", W_),
    # column-major x*5+y: 22, 10, 4 -> food 2
    ("seq_column_major", W_),
    ("seq_reverse_column_major", E_),
])
def test_target_and_first_move_by_hand(name, want):
    s = state(**BASE)
    assert O.lbf_heuristic(desc(), s, 1, H[name]) == want


def test_sequential_plans_use_the_start_position():
    # the agent started at (0, 3): distances 5, 5, 1 -> nearest food 2, farthest food 0
    # (tie with food 1, lower index); it is now at (2, 2)
    s = state(**BASE, init1=(0, 3))
    assert O.lbf_heuristic(desc(), s, 1, H["seq_nearest_agent"]) == W_
    assert O.lbf_heuristic(desc(), s, 1, H["seq_farthest_agent"]) == E_
    # from the current position instead, food 0 / 1 would tie nearest: the plan differs
    s2 = state(**BASE)
    assert O.lbf_heuristic(desc(), s2, 1, H["seq_nearest_agent"]) == E_


def test_load_when_adjacent_and_eaten_foods_skipped():
    s = state(a0=(0, 0), a1=(3, 2), foods=[(4, 2, 1), (2, 0, 3), (0, 4, 2)])
    assert O.lbf_heuristic(desc(), s, 1, H["greedy_closest_self"]) == LOAD
    s = state(a0=(0, 0), a1=(3, 2), foods=[(4, 2, 1), (2, 0, 3), (0, 4, 2)], eaten=(1, 0, 0))
    # food 0 gone: food 1 at (2,0): dx = -1, dy = -2 -> y first: north
    assert O.lbf_heuristic(desc(), s, 1, H["greedy_closest_self"]) == N_
    s = state(a0=(0, 0), a1=(3, 2), foods=[(4, 2, 1), (2, 0, 3), (0, 4, 2)], eaten=(1, 1, 1))
    assert O.lbf_heuristic(desc(), s, 1, H["greedy_closest_self"]) == NOOP


def test_blocked_moves():
    # target (4, 2) straight east, agent 0 on (3, 2): no other axis to try -> noop
    s = state(a0=(3, 2), a1=(2, 2), foods=[(4, 2, 1), (0, 0, 3)])
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["greedy_lowest_level"]) == NOOP
    # target (4, 3): dx = 2, dy = 1 -> east first, but food 1 sits on (3, 2) -> south
    s = state(a0=(0, 0), a1=(2, 2), foods=[(4, 3, 1), (3, 2, 3)])
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["greedy_lowest_level"]) == S_
    # both axes blocked: east (3,2) by agent 0, south (2,3) by food 1 -> noop
    s = state(a0=(3, 2), a1=(2, 2), foods=[(4, 3, 1), (2, 3, 3)])
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["greedy_lowest_level"]) == NOOP
    # at the grid edge: target (0, 4) from (0, 2) along y only
    s = state(a0=(4, 4), a1=(0, 2), foods=[(0, 4, 1)])
    assert O.lbf_heuristic(desc(n_food=1), s, 1, H["greedy_closest_self"]) == S_


def test_seat_zero_plays_the_same_rules():
    s = state(a0=(2, 2), a1=(0, 0), foods=[(4, 2, 1), (2, 0, 3), (0, 4, 2)])
    s.ix[0], s.iy[0] = 2, 2
    assert O.lbf_heuristic(desc(), s, 0, H["greedy_closest_teammate"]) == N_   # teammate at (0,0)
    assert O.lbf_heuristic(desc(), s, 0, H["greedy_closest_self"]) == E_


def test_moves_close_in_on_the_target_random_states():
    """On random states, every unblocked heuristic move shortens the Manhattan distance to
    the food its own criterion ranks first, and 'load' happens exactly when adjacent."""
    rng = np.random.default_rng(0)
    d = desc(7, 7)
    for trial in range(300):
        cells = rng.choice(49, 5, replace=False)
        pos = [(c % 7, c // 7) for c in cells]
        foods = [(x, y, int(rng.integers(1, 5))) for x, y in pos[:3]]
        s = state(pos[3], pos[4], foods, init1=pos[4])
        for name, k in H.items():
            if name == "entitled":
                continue
            a = O.lbf_heuristic(d, s, 1, k)
            assert 0 <= a <= 5
            # the target by brute force over the three foods
            def key(f):
                x, y, lv = foods[f]
                dm = abs(x - pos[4][0]) + abs(y - pos[4][1])
                dt = abs(x - pos[3][0]) + abs(y - pos[3][1])
                return [dm, dt, dm + dt, lv, -lv, y * 7 + x, -(y * 7 + x), x * 7 + y, -(x * 7 + y), dm, -dm][k]
            tgt = min(range(3), key=lambda f: (key(f), f))
            tx, ty, _ = foods[tgt]
            dist = abs(tx - pos[4][0]) + abs(ty - pos[4][1])
            if dist == 1:
                assert a == LOAD, name
                continue
            assert a != LOAD
            if a == NOOP:
                continue
            dx = (a == E_) - (a == W_)
            dy = (a == S_) - (a == N_)
            nx, ny = pos[4][0] + dx, pos[4][1] + dy
            assert abs(tx - nx) + abs(ty - ny) == dist - 1, name


def test_rollout_and_xplay_accept_heuristic_teammates():
    d = desc(7, 7)
    rng = np.random.default_rng(1)
    layers = [(rng.normal(0, 0.1, (16, 196)), rng.normal(0, 0.1, 16)),
              (rng.normal(0, 0.1, (16, 16)), rng.normal(0, 0.1, 16)),
              (rng.normal(0, 0.1, (7, 16)), rng.normal(0, 0.1, 7))]
    pols = O.Policies([layers])
    st = O.reset_all(d, 3, 256)
    pool = [O.heuristic_id("greedy_closest_self"), O.heuristic_id("seq_column_major")]
    out = O.rollout(d, pols, 3, st, 0, 20, 0, pool)
    assert out["rc"] == 0
    assert set(np.unique(out["teammate"])) <= set(pool)
    # the teammate seat's actions are its rule's, and no draw is flagged for it
    assert (out["margin"][..., 1] == 2.0).all()
    xp = O.xplay(d, pols, 4, 0, [0], [O.heuristic_id(n) for n in O.LBF_HEURISTICS], 8, 50)
    assert xp["rc"] == 0 and xp["matrix"].shape == (1, 12)


# Entitled, food 0 at (2, 2) level 2 on a 5 x 5 grid: its pair is W (1, 2) and E (3, 2)
E_FOODS = [(2, 2, 2), (4, 4, 1)]


def test_entitled_waits_until_the_teammate_takes_a_square():
    # agent 0 on neither square: wait, wherever the heuristic (agent 1) stands
    for a1 in [(0, 0), (3, 2), (1, 2), (4, 0)]:
        s = state(a0=(0, 4), a1=a1, foods=E_FOODS)
        assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == NOOP, a1
    # agent 0 on W (1, 2): go to E (3, 2) -- from (4, 0): dx = -1, dy = 2 -> south
    s = state(a0=(1, 2), a1=(4, 0), foods=E_FOODS)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == S_
    # ... and load once standing on it
    s = state(a0=(1, 2), a1=(3, 2), foods=E_FOODS)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == LOAD
    # agent 0 on E: the target is W (1, 2); from (1, 0): dx = 0, dy = 2 -> south
    s = state(a0=(3, 2), a1=(1, 0), foods=E_FOODS)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == S_


def test_entitled_pairs_at_edges_and_next_to_foods():
    # food 0 at (0, 0): W and N off the grid -> pair E (1, 0), S (0, 1)
    foods = [(0, 0, 1), (4, 4, 1)]
    s = state(a0=(0, 1), a1=(3, 0), foods=foods)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == W_   # to (1, 0)
    s = state(a0=(1, 0), a1=(0, 3), foods=foods)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == N_   # to (0, 1)
    # food 1 on (1, 2), W of food 0 at (2, 2): the pair becomes E (3, 2), N (2, 1)
    foods = [(2, 2, 1), (1, 2, 1)]
    s = state(a0=(2, 1), a1=(3, 4), foods=foods)
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == N_   # to (3, 2)
    s = state(a0=(1, 3), a1=(3, 4), foods=foods)                        # (1, 3): no square
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == NOOP
    # food 0 eaten: the pair belongs to food 1 at (4, 4): W (3, 4), N (4, 3)
    s = state(a0=(4, 3), a1=(0, 4), foods=[(2, 2, 1), (4, 4, 1)], eaten=(1, 0, 0))
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == E_
    # all eaten: noop
    s = state(a0=(4, 3), a1=(0, 4), foods=[(2, 2, 1), (4, 4, 1)], eaten=(1, 1, 1))
    assert O.lbf_heuristic(desc(n_food=2), s, 1, H["entitled"]) == NOOP
    # a food in a 1-wide corridor with a single free neighbour has no pair: noop
    d = O.env_desc(O.LBF, 3, 1, 1, 3, 50)
    s = state(a0=(1, 0), a1=(2, 0), foods=[(0, 0, 1)])
    assert O.lbf_heuristic(d, s, 1, H["entitled"]) == NOOP


def test_entitled_pair_load_together():
    """Two Entitled agents off the pair both wait; with the other agent on W, an Entitled
    agent walks to E by the step rule and loads there."""
    d = desc(n_food=2)
    s = state(a0=(0, 4), a1=(4, 4), foods=[(2, 2, 2), (0, 0, 1)])
    assert [O.lbf_heuristic(d, s, seat, H["entitled"]) for seat in (0, 1)] == [NOOP, NOOP]
    s = state(a0=(1, 2), a1=(4, 4), foods=[(2, 2, 2), (0, 0, 1)], levels=(1, 1))
    seen = []
    for t in range(10):
        a = O.lbf_heuristic(d, s, 1, H["entitled"])
        seen.append(a)
        if a == LOAD:
            break
        dx = (a == E_) - (a == W_)
        dy = (a == S_) - (a == N_)
        s.ax[1] += dx
        s.ay[1] += dy
    assert seen[-1] == LOAD and (s.ax[1], s.ay[1]) == (3, 2)
    # (4,4) -N-> (4,3) -W-> (3,3) (tie: x first) -N-> (3,2), then load
    assert seen == [N_, W_, N_, LOAD]
