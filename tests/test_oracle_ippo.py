"""Pins for the oracle's teammate-seat learner outputs (IPPO, Sec. 3 MARL baseline: both
seats learn with their own PPO).  The seat-1 log-probability, value and bootstrap value
of a rollout are checked against a torch fp64 forward of the teammate's weights on the
recorded seat-1 observations, against the seat-0 outputs of the same rollout with the
seats' policies swapped where the game is symmetric, and against a one-step-longer run."""
import numpy as np
import torch

import oracle as O


def rand_policy(rng, dims, scale=0.3):
    return [(rng.standard_normal((dims[i + 1], dims[i])) * scale,
             rng.standard_normal(dims[i + 1]) * scale) for i in range(3)]


def torch_outputs(pol, obs):
    x = torch.from_numpy(obs.reshape(-1, obs.shape[-1]).astype(np.float64))
    for k, (W_, b) in enumerate(pol):
        x = x @ torch.from_numpy(W_).T + torch.from_numpy(b)
        if k < 2:
            x = torch.tanh(x)
    return x.numpy().reshape(obs.shape[:-1] + (-1,))


def setup(N=40, T=30):
    rng = np.random.default_rng(11)
    d = O.env_desc(O.LBF, 7, 7, 3, 3, 20)
    od, K = 196, 6
    pols = [rand_policy(rng, [od, 16, 16, K + 1]), rand_policy(rng, [od, 16, 16, K + 1]),
            rand_policy(rng, [od, 16, 16, K])]  # the last one has no value row
    return d, pols, K, N, T


def test_teammate_logp_and_value_follow_its_own_network():
    d, pols, K, N, T = setup()
    P = O.Policies(pols)
    st = O.reset_all(d, 5, N)
    out = O.rollout(d, P, 5, st, 0, T, 0, [1])
    assert out["rc"] == 0
    z = torch_outputs(pols[1], out["obs_tm"])                       # [T][N][K+1]
    a1 = out["actions"][..., 1].astype(np.int64)
    lsm = torch.log_softmax(torch.from_numpy(z[..., :K]), -1).numpy()
    want_lp = np.take_along_axis(lsm, a1[..., None], -1)[..., 0]
    assert np.allclose(out["logp_tm"], want_lp, rtol=0, atol=1e-12)
    assert np.allclose(out["values_tm"], z[..., K], rtol=0, atol=1e-12)
    # the ego's outputs come from seat 0's network on seat 0's observations, not these
    z0 = torch_outputs(pols[0], out["obs"])
    assert np.allclose(out["values"], z0[..., K], rtol=0, atol=1e-12)
    assert not np.allclose(out["values"], out["values_tm"])


def test_bootstrap_equals_the_next_steps_value():
    d, pols, K, N, T = setup()
    P = O.Policies(pols)
    st_a = O.reset_all(d, 9, N)
    st_b = st_a.copy()
    short = O.rollout(d, P, 9, st_a, 0, T, 0, [1])
    long = O.rollout(d, P, 9, st_b, 0, T + 1, 0, [1])
    assert np.array_equal(short["actions"], long["actions"][:T])
    assert np.array_equal(short["last_value_tm"], long["values_tm"][T])
    assert np.array_equal(short["last_value"], long["values"][T])


def test_no_value_row_and_rule_teammates_give_zeros():
    d, pols, K, N, T = setup()
    P = O.Policies(pols)
    out = O.rollout(d, P, 3, O.reset_all(d, 3, N), 0, T, 0, [2])
    assert not out["values_tm"].any() and not out["last_value_tm"].any()
    assert out["logp_tm"].max() < 0.0           # a network teammate still has its logp
    out = O.rollout(d, P, 3, O.reset_all(d, 3, N), 0, T, 0, [O.heuristic_id("greedy_closest_self")])
    assert not out["logp_tm"].any() and not out["values_tm"].any() and not out["last_value_tm"].any()


def test_seat_swap_on_a_symmetric_start():
    """LBF with the two agents exchanged (positions and levels): seat 1 of the original
    state sees what seat 0 of the swapped state sees, so the first step's seat-1
    observation and value of rollout (A, B) equal the seat-0 ones of rollout (B, A) on
    the swapped states."""
    d, pols, K, N, T = setup(N=200, T=1)
    P = O.Policies(pols)
    st = O.reset_all(d, 21, N)
    swapped = st.copy()
    for i in range(N):
        a = O.LbfState.from_buffer(swapped[i])
        a.ax[0], a.ax[1] = a.ax[1], a.ax[0]
        a.ay[0], a.ay[1] = a.ay[1], a.ay[0]
        a.al[0], a.al[1] = a.al[1], a.al[0]
    ab = O.rollout(d, P, 21, st, 0, 1, 0, [1])
    ba = O.rollout(d, P, 21, swapped, 0, 1, 1, [0])
    assert np.array_equal(ab["obs_tm"][0], ba["obs"][0])
    assert np.allclose(ab["values_tm"][0], ba["values"][0], rtol=0, atol=0)
    # logp of each seat's own applied action differs only through the action draw
    z = torch_outputs(pols[1], ab["obs_tm"][0])
    lsm = torch.log_softmax(torch.from_numpy(z[:, :K]), -1).numpy()
    a1 = ab["actions"][0, :, 1].astype(np.int64)
    assert np.allclose(ab["logp_tm"][0], lsm[np.arange(N), a1], atol=1e-12)


def test_seat1_rows_are_seat0_rows_with_the_level_channels_swapped():
    """Seat 1's LBF observation differs from seat 0's only in which agent fills the
    observer's and the other agent's level channels (0 and 1); food and empty cells are
    the same for both.  The tensor-core IPPO collection writes seat 1's trajectory rows
    from seat 0's by that swap, so it is checked here on the oracle's own rows, along
    rollouts with auto-resets on the 7x7 and 12x12 grids."""
    rng = np.random.default_rng(5)
    for w, h in [(7, 7), (12, 12)]:
        d = O.env_desc(O.LBF, w, h, 3, 3, 20)
        od = 4 * w * h
        pols = [rand_policy(rng, [od, 16, 16, 7]), rand_policy(rng, [od, 16, 16, 7])]
        st = O.reset_all(d, 3, 64)
        out = O.rollout(d, O.Policies(pols), 3, st, 0, 45, 0, [1])
        assert out["rc"] == 0 and out["dones"].any()
        rows0 = out["obs"].reshape(45, 64, w * h, 4)
        rows1 = out["obs_tm"].reshape(45, 64, w * h, 4)
        assert np.array_equal(rows1, rows0[..., [1, 0, 2, 3]])
        assert (rows0[..., 0] > 0).sum(-1).min() == 1   # each row shows its observer once
