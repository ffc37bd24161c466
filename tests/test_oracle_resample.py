"""Pins for the oracle's per-episode teammate resampling (Sec. 3: the ego meets teammates
drawn from the training set; each episode draws its own).  The reading: the episode of
env e that began at step s plays pool[uniform_int(x, |pool|)], x = word 0 of the Philox
counter (e, s, stream 5); the step each env's episode began is carried in ep_step."""
import numpy as np
import torch

import oracle as O


def rand_policy(rng, dims, scale=0.3):
    return [(rng.standard_normal((dims[i + 1], dims[i])) * scale,
             rng.standard_normal(dims[i + 1]) * scale) for i in range(3)]


def setup(n_pol=5, N=64, ep_len=12):
    rng = np.random.default_rng(4)
    d = O.env_desc(O.LBF, 5, 5, 2, 3, ep_len)
    od, K = O.obs_dim(d), O.n_actions(d)
    pols = [rand_policy(rng, [od, 16, 16, K + 1])] + [rand_policy(rng, [od, 16, 16, K + 1])
                                                      for _ in range(n_pol - 1)]
    return d, pols, K, N


def episode_teammate(seed, env, start, pool):
    x = int(O.draw(seed, env, start, 5, 0))
    return pool[(x * len(pool)) >> 32]


def test_teammate_changes_exactly_at_episode_starts():
    d, pols, K, N = setup()
    P = O.Policies(pols)
    pool = [1, 2, 3, 4]
    ep = np.zeros(N, np.uint32)
    st = O.reset_all(d, 7, N)
    T = 60
    out = O.rollout(d, P, 7, st, 0, T, 0, pool, ep_step=ep, resample=True)
    assert out["rc"] == 0
    tm, dn = out["teammates_t"], out["dones"]
    start = np.zeros(N, np.int64)
    n_episodes = 0
    for t in range(T):
        for e in range(N):
            if t > 0 and dn[t - 1, e]:
                start[e] = t
                n_episodes += 1
            assert tm[t, e] == episode_teammate(7, e, int(start[e]), pool), (t, e)
    assert n_episodes > N                             # episodes of 12 steps or fewer
    start[dn[T - 1] == 1] = T                         # a done at the last step resets at T
    # ep_step ends as the start of each env's current episode
    assert np.array_equal(ep, start.astype(np.uint32))
    # the first episode's teammate also comes out as `teammate`
    assert np.array_equal(out["teammate"], tm[0])


def test_teammate_network_is_the_recorded_one():
    """The teammate's logp of its applied action is that of the policy teammates_t names,
    evaluated (torch fp64) on the recorded seat-1 observation."""
    d, pols, K, N = setup()
    P = O.Policies(pols)
    pool = [1, 2, 3, 4]
    out = O.rollout(d, P, 3, O.reset_all(d, 3, N), 0, 40, 0, pool,
                    ep_step=np.zeros(N, np.uint32), resample=True)
    a1 = out["actions"][..., 1].astype(np.int64)
    for pid in pool:
        sel = out["teammates_t"] == pid
        assert sel.any()
        x = torch.from_numpy(out["obs_tm"][sel].astype(np.float64))
        for k, (W_, b) in enumerate(pols[pid]):
            x = x @ torch.from_numpy(W_).T + torch.from_numpy(b)
            if k < 2:
                x = torch.tanh(x)
        lsm = torch.log_softmax(x[:, :K], -1).numpy()
        want = lsm[np.arange(sel.sum()), a1[sel]]
        assert np.allclose(out["logp_tm"][sel], want, atol=1e-12)
        assert np.allclose(out["values_tm"][sel], x[:, K].numpy(), atol=1e-12)


def test_single_member_pool_matches_per_call_mode():
    d, pols, K, N = setup(N=300)
    P = O.Policies(pols)
    a = O.rollout(d, P, 5, O.reset_all(d, 5, N), 0, 30, 0, [2],
                  ep_step=np.zeros(N, np.uint32), resample=True)
    b = O.rollout(d, P, 5, O.reset_all(d, 5, N), 0, 30, 0, [2])
    for k in ("obs", "obs_tm", "actions", "logp", "values", "rewards", "dones", "logp_tm",
              "teammates_t", "last_value"):
        assert np.array_equal(a[k], b[k]), k


def test_carry_over_between_calls_and_uniform_draws():
    """Two calls of 30 steps equal one call of 60 (ep_step and the states carry), and the
    episode teammates are uniform over the pool (chi-square, 3 dof, p > 0.001)."""
    d, pols, K, N = setup(N=256)
    P = O.Policies(pols)
    pool = [1, 2, 3, 4]
    ep_a, ep_b = np.zeros(N, np.uint32), np.zeros(N, np.uint32)
    st_a, st_b = O.reset_all(d, 11, N), O.reset_all(d, 11, N)
    one = O.rollout(d, P, 11, st_a, 0, 60, 0, pool, ep_step=ep_a, resample=True)
    h1 = O.rollout(d, P, 11, st_b, 0, 30, 0, pool, ep_step=ep_b, resample=True)
    h2 = O.rollout(d, P, 11, st_b, 30, 30, 0, pool, ep_step=ep_b, resample=True)
    assert np.array_equal(one["teammates_t"], np.concatenate([h1["teammates_t"], h2["teammates_t"]]))
    assert np.array_equal(one["actions"], np.concatenate([h1["actions"], h2["actions"]]))
    assert np.array_equal(ep_a, ep_b) and np.array_equal(st_a, st_b)
    # one teammate per episode start
    tm, dn = one["teammates_t"], one["dones"]
    firsts = np.concatenate([tm[:1], tm[1:][dn[:-1] == 1][None]], axis=None)
    counts = np.array([(firsts == p).sum() for p in pool], np.float64)
    exp = counts.sum() / len(pool)
    chi2 = ((counts - exp) ** 2 / exp).sum()
    assert counts.sum() > 1000 and chi2 < 16.27
