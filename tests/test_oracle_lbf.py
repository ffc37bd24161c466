"""Pins for the oracle's Level-Based Foraging rules.

Hand-worked cases follow the workload's statement of the game: a load succeeds when
the summed levels of the adjacent loading agents reach the food level, and each loader
is paid food_level * agent_level / normaliser (the readings fix the normaliser as
loader-level sum times the total spawned food level, so a fully eaten grid returns 1).
"""
import ctypes as C
import itertools

import numpy as np
import pytest

NOOP, N, S, W, E, LOAD = range(6)


def desc(orc, w=7, h=7, nf=3, ep=50):
    return orc.env_desc(orc.LBF, w, h, nf, 3, ep)


def state(orc, agents, foods, F=None):
    """agents: [(x, y, level)] * 2; foods: [(x, y, level)] (missing foods are eaten)."""
    s = orc.LbfState()
    for i, (x, y, l) in enumerate(agents):
        s.ax[i], s.ay[i], s.al[i] = x, y, l
    for k in range(3):
        if k < len(foods):
            s.fx[k], s.fy[k], s.fl[k] = foods[k]
            s.eaten[k] = 0
        else:
            s.eaten[k] = 1
    s.F = F if F is not None else sum(f[2] for f in foods)
    return s


def step(orc, d, s, a0, a1):
    r = np.zeros(2, np.float32)
    team = np.zeros(1, np.float32)
    done = orc.lib().orc_lbf_step(C.byref(d), C.byref(s), a0, a1, r.ctypes.data_as(C.c_void_p),
                                  team.ctypes.data_as(C.c_void_p))
    return r, float(team[0]), done


def test_joint_load_pays_by_level(orc):
    d = desc(orc, nf=2)
    # levels (1, 2), food level 3 between them; a second food of level 2 far away: F = 5.
    s = state(orc, [(1, 2, 1), (3, 2, 2)], [(2, 2, 3), (6, 6, 2)])
    r, team, done = step(orc, d, s, LOAD, LOAD)
    assert s.eaten[0] == 1 and s.eaten[1] == 0
    assert r[0] == np.float32(3 * 1) / np.float32(3 * 5)
    assert r[1] == np.float32(3 * 2) / np.float32(3 * 5)
    assert abs(team - 3 / 5) < 1e-7 and not done


def test_single_loader_below_level_fails(orc):
    d = desc(orc, nf=1)
    s = state(orc, [(1, 2, 2), (5, 5, 1)], [(2, 2, 3)])
    r, team, done = step(orc, d, s, LOAD, NOOP)
    assert s.eaten[0] == 0 and team == 0.0 and r.tolist() == [0.0, 0.0]


def test_diagonal_neighbour_does_not_count(orc):
    d = desc(orc, nf=1)
    s = state(orc, [(1, 2, 2), (3, 3, 2)], [(2, 2, 3)])   # agent 1 is diagonal
    r, team, _ = step(orc, d, s, LOAD, LOAD)
    assert s.eaten[0] == 0 and team == 0.0


def test_adjacent_non_loader_does_not_count(orc):
    d = desc(orc, nf=1)
    s = state(orc, [(1, 2, 2), (3, 2, 2)], [(2, 2, 3)])
    r, team, _ = step(orc, d, s, LOAD, NOOP)
    assert s.eaten[0] == 0 and team == 0.0


def test_one_loader_eats_two_adjacent_foods(orc):
    d = desc(orc, nf=2)
    s = state(orc, [(2, 2, 3), (6, 6, 1)], [(1, 2, 2), (3, 2, 3)])   # F = 5
    r, team, done = step(orc, d, s, LOAD, NOOP)
    assert s.eaten[0] == 1 and s.eaten[1] == 1 and done
    # each food pays food_level * 3 / (3 * 5) to the single loader: 2/5 + 3/5
    want = np.float32(np.float32(2 * 3) / np.float32(3 * 5)) + np.float32(np.float32(3 * 3) / np.float32(3 * 5))
    assert r[0] == want and r[1] == 0.0


@pytest.mark.parametrize("a0,blocked_by", [(W, "edge"), (E, "food"), (S, "agent")])
def test_blocked_moves_stay(orc, a0, blocked_by):
    d = desc(orc, nf=1)
    # agent 0 at the west edge (0, 3); food east of it at (1, 3); agent 1 south at (0, 4)
    s = state(orc, [(0, 3, 1), (0, 4, 1)], [(1, 3, 3)])
    step(orc, d, s, a0, NOOP)
    assert (s.ax[0], s.ay[0]) == (0, 3), blocked_by


def test_moving_into_cell_being_vacated_is_blocked(orc):
    d = desc(orc, nf=1)
    s = state(orc, [(2, 2, 1), (3, 2, 1)], [(6, 6, 3)])
    step(orc, d, s, E, E)   # agent 1 moves away but agent 0 targets its current cell
    assert (s.ax[0], s.ay[0]) == (2, 2) and (s.ax[1], s.ay[1]) == (4, 2)


def test_same_target_both_stay(orc):
    d = desc(orc, nf=1)
    s = state(orc, [(1, 2, 1), (3, 2, 1)], [(6, 6, 3)])
    step(orc, d, s, E, W)   # both target (2, 2)
    assert (s.ax[0], s.ay[0], s.ax[1], s.ay[1]) == (1, 2, 3, 2)


def test_compass_directions(orc):
    d = desc(orc, nf=1)
    for a, (dx, dy) in {N: (0, -1), S: (0, 1), W: (-1, 0), E: (1, 0), NOOP: (0, 0), LOAD: (0, 0)}.items():
        s = state(orc, [(3, 3, 1), (0, 0, 1)], [(6, 6, 3)])
        step(orc, d, s, a, NOOP)
        assert (s.ax[0], s.ay[0]) == (3 + dx, 3 + dy)


def test_episode_limit_and_all_eaten_end_episode(orc):
    d = desc(orc, nf=1, ep=3)
    s = state(orc, [(0, 0, 1), (6, 0, 1)], [(6, 6, 3)])
    dones = [step(orc, d, s, NOOP, NOOP)[2] for _ in range(3)]
    assert dones == [0, 0, 1]


def test_obs_is_level_scaled_one_hot(orc):
    d = desc(orc, w=3, h=3, nf=2)
    s = state(orc, [(0, 0, 2), (2, 1, 3)], [(1, 1, 4), (2, 2, 1)])
    s.eaten[1] = 1
    for seat, (me, you) in enumerate([((0, 0), (2, 1)), ((2, 1), (0, 0))]):
        out = np.zeros(36, np.uint8)
        orc.lib().orc_lbf_obs(C.byref(d), C.byref(s), seat, out.ctypes.data_as(C.c_void_p))
        grid = out.reshape(3, 3, 4)   # [y][x][channel]
        want = np.zeros((3, 3, 4), np.uint8)
        want[:, :, 3] = 1
        for (x, y), ch, lvl in [(me, 0, [2, 3][seat]), (you, 1, [3, 2][seat]), ((1, 1), 2, 4)]:
            want[y, x, :] = 0
            want[y, x, ch] = lvl
        assert (grid == want).all(), seat


def test_reset_distribution(orc):
    d = desc(orc)
    st = orc.reset_all(d, 5, 6000)
    S = np.frombuffer(st.tobytes(), dtype=np.int32).reshape(6000, -1)[:, :22]
    ax, ay, al = S[:, 0:2], S[:, 2:4], S[:, 4:6]
    fx, fy, fl, eaten, F = S[:, 6:9], S[:, 9:12], S[:, 12:15], S[:, 15:18], S[:, 18]
    assert ((al >= 1) & (al <= 3)).all()
    assert ((fl >= 1) & (fl <= al.sum(1, keepdims=True))).all()
    assert (F == fl.sum(1)).all() and (eaten == 0).all()
    cells = np.concatenate([fy * 7 + fx, ay * 7 + ax], axis=1)
    assert all(len(set(row)) == 5 for row in cells)   # no two objects share a cell
    lv = np.bincount(al.ravel(), minlength=4)[1:]
    assert np.abs(lv - lv.mean()).max() < 5 * np.sqrt(lv.mean())
    occ = np.bincount(cells.ravel(), minlength=49)
    assert np.abs(occ - occ.mean()).max() < 5 * np.sqrt(occ.mean())


def _enumerate(orc, d, s0, T):
    """Team return of every joint-action sequence of length T from state s0."""
    rets = {}
    for seq in itertools.product(range(36), repeat=T):
        s = orc.LbfState.from_buffer_copy(s0)
        total = 0.0
        for ja in seq:
            if s.done:
                break
            _, team, _ = step(orc, d, s, ja // 6, ja % 6)
            total += team
        rets[seq] = (s.ret, s)
    return rets


def test_brute_force_optimum_hand_derived(orc):
    # 3x3 grid: food level 2 in the centre, level-1 agents in opposite corners.  No
    # single step can eat it; in two steps each agent has exactly two moves to a cell
    # 4-adjacent to the centre (agent 0 E or S, agent 1 W or N), then both load:
    # optimum 1.0 reached by exactly 2 * 2 = 4 of the 36^2 sequences.
    d = desc(orc, w=3, h=3, nf=1)
    s0 = state(orc, [(0, 0, 1), (2, 2, 1)], [(1, 1, 2)])
    r1 = _enumerate(orc, d, s0, 1)
    assert max(v[0] for v in r1.values()) == 0.0
    r2 = _enumerate(orc, d, s0, 2)
    best = [k for k, v in r2.items() if v[0] == 1.0]
    assert len(best) == 4
    assert max(v[0] for v in r2.values()) == 1.0
    for seq in best:
        assert seq[1] == LOAD * 6 + LOAD
        assert seq[0] // 6 in (E, S) and seq[0] % 6 in (W, N)


def test_brute_force_invariants_3x3(orc):
    # All 36^3 joint-action sequences from several random 3x3 starts with 1 and 2 foods:
    # no two objects overlap, 0 <= return <= 1, and return = eaten level sum / F.
    for nf in (1, 2):
        d = desc(orc, w=3, h=3, nf=nf)
        starts = orc.reset_all(d, 99, 3)
        for e in range(3):
            s0 = orc.LbfState.from_buffer_copy(starts[e].tobytes()[:C.sizeof(orc.LbfState)])
            for seq, (ret, s) in _enumerate(orc, d, s0, 3).items():
                assert 0.0 <= ret <= 1.0 + 1e-6
                eaten = sum(s.fl[k] for k in range(nf) if s.eaten[k])
                assert abs(ret - eaten / s.F) < 1e-6
                occ = [(s.ax[0], s.ay[0]), (s.ax[1], s.ay[1])] + \
                      [(s.fx[k], s.fy[k]) for k in range(nf) if not s.eaten[k]]
                assert len(set(occ)) == len(occ)
