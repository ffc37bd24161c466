"""Pins for the oracle's recurrent S5 actor-critic (readings in aht_oracle.h): the
recurrence against the explicit sum of powers of the discretised modes, the steady state
of a constant input against the geometric series, the reset, and the dense parts against
torch fp64 layers (small sizes: H = 16, P = 12, F = 32)."""
import numpy as np
import pytest
import torch
from scipy.special import erf

import oracle as O
from paper_2609_13716_gb300 import workloads as W


def small(seed=0, K=20, A=6):
    return W.s5_params(seed, K, A, H=16, P=12, F=32)


def discretised(p):
    lam = p["lam_re"].astype(np.float64) + 1j * p["lam_im"].astype(np.float64)
    dt = np.exp(p["log_dt"].astype(np.float64))
    lbar = np.exp(lam * dt)
    Bbar = ((lbar - 1.0) / lam)[:, None] * (p["B_re"] + 1j * p["B_im"]).astype(np.complex128)
    C = (p["C_re"] + 1j * p["C_im"]).astype(np.complex128)
    return lbar, Bbar, C


def test_recurrence_is_the_sum_of_powers():
    p = small()
    net = O.S5(p)
    lbar, Bbar, C = discretised(p)
    rng = np.random.default_rng(0)
    T = 25
    us = rng.standard_normal((T, net.H))
    state = np.zeros(2 * net.P)
    for t in range(T):
        y = net.ssm_step(us[t], t == 0, state)
        x = sum(lbar ** (t - j) * (Bbar @ us[j]) for j in range(t + 1))
        want = (C @ x).real + p["Dv"] * us[t]
        assert np.allclose(y, want, rtol=1e-12, atol=1e-12), t
        assert np.allclose(state[:net.P] + 1j * state[net.P:], x, rtol=1e-12, atol=1e-12)


def test_constant_input_reaches_the_geometric_steady_state():
    p = small(1)
    net = O.S5(p)
    lbar, Bbar, C = discretised(p)
    assert (np.abs(lbar) < 1).all()
    u = np.random.default_rng(1).standard_normal(net.H)
    state = np.zeros(2 * net.P)
    for t in range(20000):
        y = net.ssm_step(u, t == 0, state)
    x_inf = (Bbar @ u) / (1.0 - lbar)
    slow = np.abs(lbar) ** 20000 > 1e-12     # modes that have not settled
    x = state[:net.P] + 1j * state[net.P:]
    assert np.allclose(x[~slow], x_inf[~slow], rtol=1e-8, atol=1e-10)


def test_reset_starts_a_fresh_sequence():
    net = O.S5(small(2))
    rng = np.random.default_rng(2)
    us = rng.standard_normal((10, net.H))
    a, b = np.zeros(2 * net.P), np.zeros(2 * net.P)
    for t in range(6):
        net.ssm_step(us[t], t == 0, a)
    for t in range(6, 10):
        ya = net.ssm_step(us[t], t == 6, a)      # reset at step 6
        yb = net.ssm_step(us[t], t == 6, b)      # a different history before it
        assert np.array_equal(ya, yb)


def test_dense_parts_match_torch_and_the_step_composes_them():
    p = small(3)
    net = O.S5(p)
    rng = np.random.default_rng(3)
    obs = rng.integers(0, 4, size=net.K).astype(np.uint8)
    t = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    x = t(obs.astype(np.float64))
    e = torch.relu(t(p["We1"]) @ x + t(p["be1"]))
    u_want = torch.relu(t(p["We2"]) @ e + t(p["be2"])).numpy()
    u = net.encode(obs)
    assert np.allclose(u, u_want, rtol=1e-13, atol=1e-13)
    v = rng.standard_normal(net.H)
    legal = np.array([1, 0, 1, 1, 0, 1], np.uint8)
    logits, value = net.heads(v, legal)
    for head, out in (("a", logits), ("c", np.array([value]))):
        h = t(v)
        for i in range(4):
            h = t(p["W" + head][i]) @ h + t(p["b" + head][i])
            if i < 3:
                h = torch.relu(h)
        want = h.numpy()
        if head == "a":
            want = np.where(legal == 1, want, -np.inf)
        assert np.allclose(out, want, rtol=1e-12, atol=1e-12)
    # one full step = heads(u + gelu(y)), gelu(a) = a (1 + erf(a / sqrt 2)) / 2
    state = np.zeros((1, 2 * net.P))
    lg, val = net.step(obs[None], np.array([1], np.uint8), state, legal[None])
    s2 = np.zeros(2 * net.P)
    y = net.ssm_step(u, 1, s2)
    vv = u + y * 0.5 * (1.0 + erf(y / np.sqrt(2.0)))
    lg2, val2 = net.heads(vv, legal)
    assert np.allclose(lg[0], lg2, rtol=1e-12) and abs(val[0] - val2) < 1e-12
    assert np.allclose(state[0], s2, rtol=0, atol=0)
