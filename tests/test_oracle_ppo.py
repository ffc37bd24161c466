"""Pins of the oracle's PPO ego update (no GPU).

What fixes the values: PPO's clipped surrogate objective with a clipped value loss and an
entropy bonus (Schulman et al. 2017, the algorithm App. C "PPO ego" names), Adam (Kingma &
Ba 2015) and global-norm clipping.  The gradient is pinned by central finite differences
of the oracle's own loss (a dropped term, wrong sign or transposed weight fails it); Adam
and clipping by their closed forms; the permutation by brute force.
"""
import numpy as np
import pytest

import oracle as O


def tiny_problem(seed, D=5, H0=4, H1=3, A=3, S=12, spread=0.3):
    rng = np.random.default_rng(seed)
    net = O.ppo_net(D, H0, H1, A)
    layers = [(rng.normal(0, 0.5, (H0, D)), rng.normal(0, 0.1, H0)),
              (rng.normal(0, 0.5, (H1, H0)), rng.normal(0, 0.1, H1)),
              (rng.normal(0, 0.5, (A + 1, H1)), rng.normal(0, 0.1, A + 1))]
    params = O.flat_params(layers)
    obs = rng.integers(0, 4, (S, D)).astype(np.uint8)
    act = rng.integers(0, A, S).astype(np.uint8)
    logp = np.log(rng.uniform(0.2, 0.5, S)).astype(np.float32)
    val = rng.normal(0, spread, S).astype(np.float32)
    adv = rng.normal(0, 1, S).astype(np.float32)
    tgt = (val + rng.normal(0, spread, S)).astype(np.float32)
    return net, params, O.PpoBatchNp(obs, act, logp, val, adv, tgt)


def loss_at(net, p, batch, idx, hp):
    return O.ppo_grad(net, p, batch, idx, hp)[1][0]


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_gradient_matches_central_differences(seed):
    net, p, batch = tiny_problem(seed)
    idx = np.arange(batch.S)
    hp = O.ppo_hp(round_bf16=0, clip_eps=0.2, ent_coef=0.05, vf_coef=0.7)
    g, _ = O.ppo_grad(net, p, batch, idx, hp)
    h = 1e-6
    fd = np.zeros_like(p)
    for k in range(len(p)):
        e = np.zeros_like(p)
        e[k] = h
        fd[k] = (loss_at(net, p + e, batch, idx, hp) - loss_at(net, p - e, batch, idx, hp)) / (2 * h)
    # the loss has kinks (min, max, clip); none lies within h of these seeded samples
    np.testing.assert_allclose(g, fd, rtol=1e-6, atol=1e-9)
    assert np.abs(g).max() > 1e-3


def test_gradient_terms_separately():
    """Each loss term alone (others' coefficients 0) still matches differences."""
    net, p, batch = tiny_problem(5)
    idx = np.arange(batch.S)
    for kw in (dict(vf_coef=0.0, ent_coef=0.0), dict(vf_coef=1.0, ent_coef=0.0, clip_eps=0.01),
               dict(vf_coef=0.0, ent_coef=1.0)):
        hp = O.ppo_hp(round_bf16=0, **kw)
        g, _ = O.ppo_grad(net, p, batch, idx, hp)
        h = 1e-6
        for k in range(0, len(p), 3):
            e = np.zeros_like(p)
            e[k] = h
            fd = (loss_at(net, p + e, batch, idx, hp) - loss_at(net, p - e, batch, idx, hp)) / (2 * h)
            assert abs(g[k] - fd) <= 1e-6 * abs(fd) + 1e-9, (kw, k, g[k], fd)


def test_bf16_weights_only_enter_through_the_forward():
    """With rounding on, the gradient is the exact-weight gradient at bf16(W1), bf16(W2)."""
    net, p, batch = tiny_problem(7)
    idx = np.arange(batch.S)
    D, H0, H1 = net.obs_dim, net.h0, net.h1
    q = p.copy()
    n1, n2 = H0 * D, H1 * H0
    q[:n1] = [O.bf16_round(w) for w in p[:n1]]
    q[n1 + H0:n1 + H0 + n2] = [O.bf16_round(w) for w in p[n1 + H0:n1 + H0 + n2]]
    g_round, s_round = O.ppo_grad(net, p, batch, idx, O.ppo_hp(round_bf16=1))
    g_exact, s_exact = O.ppo_grad(net, q, batch, idx, O.ppo_hp(round_bf16=0))
    np.testing.assert_array_equal(g_round, g_exact)
    np.testing.assert_array_equal(s_round, s_exact)
    assert not np.array_equal(p, q)


def test_bf16_rounding_nearest_even():
    assert O.bf16_round(1.0 + 2 ** -8) == 1.0                 # tie -> even (1.0)
    assert O.bf16_round(1.0 + 3 * 2 ** -8) == 1.0 + 2 ** -6   # tie -> even (odd mantissa rounds up)
    assert O.bf16_round(1.0 + 3 * 2 ** -9) == 1.0 + 2 ** -7
    assert O.bf16_round(-2.5) == -2.5
    assert O.bf16_round(0.1) == 0.10009765625


def test_ratio_one_and_uniform_policy_closed_forms():
    net, p, batch = tiny_problem(3)
    A = net.n_act
    layers = O.unflat_params(net, p)
    (W3, b3) = layers[2]
    W3[:A] = 0.0
    b3[:A] = 0.0                      # uniform policy: logp = -log A for every action
    p = O.flat_params(layers)
    batch.logp[:] = np.float32(-np.log(A))
    idx = np.arange(batch.S)
    hp = O.ppo_hp(round_bf16=0)
    g, st = O.ppo_grad(net, p, batch, idx, hp)
    # ratio exp(logp - logp_old) = 1 up to the fp32 rounding of logp_old
    assert abs(st[4]) < 1e-7 and st[5] == 0.0
    assert abs(st[1]) < 1e-7          # -mean(normalised advantage) = 0
    assert st[3] == pytest.approx(np.log(A), rel=1e-14)
    # uniform logits are a stationary point of the entropy: no entropy gradient on b3
    hp_e = O.ppo_hp(round_bf16=0, vf_coef=0.0)
    g_e, _ = O.ppo_grad(net, p, batch, idx, hp_e)
    adv = batch.advantages.astype(np.float64)
    a_n = (adv - adv.mean()) / (adv.std() + 1e-8)
    onehot = np.eye(A)[batch.actions]
    # d/d b3_j of -mean(A_n * ratio): ratio = 1, d logp_a / d z_j = [j = a] - 1/A
    want = -(a_n[:, None] * (onehot - 1.0 / A)).mean(axis=0)
    np.testing.assert_allclose(g_e[-(A + 1):-1], want, rtol=1e-6, atol=1e-12)


def test_fully_clipped_samples_have_no_policy_gradient():
    net, p, batch = tiny_problem(4)
    idx = np.arange(batch.S)
    hp = O.ppo_hp(round_bf16=0, vf_coef=0.0, ent_coef=0.0, clip_eps=0.1)
    # push every ratio far past the band in the direction its advantage rewards
    adv = batch.advantages.astype(np.float64)
    a_n = (adv - adv.mean()) / (adv.std() + 1e-8)
    z_logp = np.zeros(batch.S)
    # logp under the policy, from each single-sample diagnostic mean(logp_old - logp)
    for s in range(batch.S):
        _, st = O.ppo_grad(net, p, batch, np.array([s]), hp)
        z_logp[s] = batch.logp[s] - st[4]
    batch.logp[:] = (z_logp - np.where(a_n > 0, 1.0, -1.0)).astype(np.float32)  # ratio e or 1/e
    g, st = O.ppo_grad(net, p, batch, idx, hp)
    assert st[5] == 1.0
    np.testing.assert_array_equal(g, np.zeros_like(g))


def test_adam_first_steps_closed_form():
    rng = np.random.default_rng(9)
    n = 50
    hp = O.ppo_hp(max_grad_norm=0.0, lr=1e-3, adam_eps=1e-5)
    p0 = rng.normal(size=n)
    g1 = rng.normal(0, 1e-3, n)
    g1[:5] = [1e-7, -1e-6, 3e-5, 0.0, -2e-4]
    p, m, v = p0.copy(), np.zeros(n), np.zeros(n)
    t = O.adam_step(p, m, v, 0, g1.copy(), hp)
    assert t == 1
    # bias-corrected moments of one step: m_hat = g, v_hat = g^2
    np.testing.assert_allclose(p, p0 - hp.lr * g1 / (np.abs(g1) + hp.adam_eps), rtol=0, atol=1e-15)
    g2 = rng.normal(0, 1e-3, n)
    t = O.adam_step(p, m, v, t, g2.copy(), hp)
    m2 = 0.9 * 0.1 * g1 + 0.1 * g2
    v2 = 0.999 * 0.001 * g1 ** 2 + 0.001 * g2 ** 2
    step2 = hp.lr * (m2 / (1 - 0.9 ** 2)) / (np.sqrt(v2 / (1 - 0.999 ** 2)) + hp.adam_eps)
    np.testing.assert_allclose(p, p0 - hp.lr * g1 / (np.abs(g1) + hp.adam_eps) - step2, rtol=0, atol=1e-14)


def test_global_norm_clipping():
    rng = np.random.default_rng(10)
    n = 40
    g = rng.normal(0, 1, n)
    norm = np.linalg.norm(g)
    hp = O.ppo_hp(max_grad_norm=0.5, lr=1.0, adam_eps=1e-5)
    p, m, v = np.zeros(n), np.zeros(n), np.zeros(n)
    gg = g.copy()
    O.adam_step(p, m, v, 0, gg, hp)
    np.testing.assert_allclose(np.linalg.norm(gg), 0.5, rtol=1e-14)   # clipped in place
    np.testing.assert_allclose(gg, g * 0.5 / norm, rtol=1e-14)
    # below the threshold nothing changes
    small = g * 0.1 / norm
    s2 = small.copy()
    O.adam_step(np.zeros(n), np.zeros(n), np.zeros(n), 0, s2, hp)
    np.testing.assert_array_equal(s2, small)


@pytest.mark.parametrize("S", [1, 2, 3, 4, 5, 7, 64, 100, 1000, 4096, 5000])
def test_permutation_is_a_bijection(S):
    for seed, epoch in ((0, 0), (7, 3)):
        p = O.perm(seed, epoch, S)
        assert sorted(p.tolist()) == list(range(S))


def test_permutation_depends_on_seed_and_epoch():
    S = 4096
    a, b, c = O.perm(1, 0, S), O.perm(1, 1, S), O.perm(2, 0, S)
    assert not np.array_equal(a, b) and not np.array_equal(a, c)
    assert (a == np.arange(S)).mean() < 0.01     # few fixed points at this size
    np.testing.assert_array_equal(a, O.perm(1, 0, S))


def test_update_is_minibatch_steps_over_the_permutation():
    net, p0, batch = tiny_problem(11, S=16)
    hp = O.ppo_hp(epochs=2, minibatches=4, seed=5, epoch0=3, round_bf16=1)
    p, m, v = p0.copy(), np.zeros_like(p0), np.zeros_like(p0)
    t, stats = O.ppo_update(net, p, m, v, 0, batch, hp)
    assert t == 8 and stats.shape == (8, 6)
    # the same by hand: grad over pi_e(4b .. 4b + 3), then one Adam step
    q, mq, vq, tq = p0.copy(), np.zeros_like(p0), np.zeros_like(p0), 0
    for e in range(2):
        pe = O.perm(5, 3 + e, 16)
        for b in range(4):
            g, st = O.ppo_grad(net, q, batch, pe[4 * b:4 * b + 4], hp)
            np.testing.assert_array_equal(st, stats[e * 4 + b])
            tq = O.adam_step(q, mq, vq, tq, g, hp)
    np.testing.assert_array_equal(p, q)
    np.testing.assert_array_equal(m, mq)
