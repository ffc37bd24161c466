"""The recurrent S5 actor-critic step on the GPU (aht_s5_step) against the fp64 oracle,
at the paper's sizes (H = P = 128, heads of three 1024-unit layers) over an LBF 7x7
observation stream: a sequence of steps with episode resets and legal-action masks.
Tolerance: logits and values |g - o| <= 1e-4 |o| + 1e-4 rms(o) (the dense layers carry
their activations as two bf16, ~2^-17 relative, with fp32 accumulation; the SSM is fp32);
the recurrent state 1e-4 likewise."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import close, np_, require_gpu

pytestmark = pytest.mark.gpu


def lbf_observations(T, N, seed):
    """Real LBF 7x7 observations of seat 0 along forced random play (with auto-resets)."""
    d = O.env_desc(O.LBF, 7, 7, 3, 3, 8)
    st = O.reset_all(d, seed, N)
    rng = np.random.default_rng(seed)
    obs, resets = [], []
    reset = np.ones(N, np.uint8)
    for t in range(T):
        rc, _, _, dones, ob2 = O.step_forced(d, seed, t, st, rng.integers(0, 6, (N, 2)).astype(np.uint8))
        obs.append(ob2[:, 0].copy())
        resets.append(reset.copy())
        reset = dones.astype(np.uint8)
    return np.stack(obs), np.stack(resets)


@pytest.mark.parametrize("N,T", [(300, 6), (1, 3)])
def test_s5_steps_match_the_oracle(N, T):
    require_gpu()
    params = W.s5_params(0, 196, 6)
    pol = aht.aht_s5_create(params, max(N, 64))
    net = O.S5(params)
    obs, resets = lbf_observations(T, N, 5)
    rng = np.random.default_rng(6)
    legal = (rng.random((T, N, 6)) < 0.8).astype(np.uint8)
    legal[..., 0] = 1
    state = torch.zeros(N, 2 * net.P, device="cuda")
    state_ref = np.zeros((N, 2 * net.P))
    logits = torch.empty(N, 6, device="cuda")
    values = torch.empty(N, device="cuda")
    for t in range(T):
        aht.aht_s5_step(pol, torch.from_numpy(obs[t]).cuda(), torch.from_numpy(resets[t]).cuda(), state,
                        logits, values, torch.from_numpy(legal[t]).cuda())
        aht.aht_s5_sync(pol)
        lg_ref, v_ref = net.step(obs[t], resets[t], state_ref, legal[t])
        lg = np_(logits)
        assert np.array_equal(np.isinf(lg), legal[t] == 0), "masked actions"
        finite = legal[t] == 1
        ok, worst = close(lg[finite], lg_ref[finite])
        assert ok, f"logits at step {t}: {worst:.3g}"
        ok, worst = close(np_(values), v_ref)
        assert ok, f"values at step {t}: {worst:.3g}"
        ok, worst = close(np_(state), state_ref)
        assert ok, f"state at step {t}: {worst:.3g}"
    pol.close()


@pytest.mark.parametrize("K,A,H,P,F,N,max_envs,masked", [
    (100, 20, 64, 32, 64, 77, 128, True),     # 20 actions; fewer envs than max_envs
    (37, 32, 32, 96, 288, 5, 5, False),       # 32 actions, no mask; 3 n-tiles of 96 per head
    (10, 1, 32, 32, 32, 300, 300, True),      # one action; 3 row tiles, the last ragged
])
def test_s5_other_shapes(K, A, H, P, F, N, max_envs, masked):
    """Action counts on each register width of the output kernel, the unmasked path,
    narrow heads and ragged env counts, over four steps with resets."""
    require_gpu()
    params = W.s5_params(3, K, A, H=H, P=P, F=F)
    pol = aht.aht_s5_create(params, max_envs)
    net = O.S5(params)
    rng = np.random.default_rng(K)
    state = torch.zeros(N, 2 * P, device="cuda")
    state_ref = np.zeros((N, 2 * P))
    logits = torch.empty(N, A, device="cuda")
    values = torch.empty(N, device="cuda")
    for t in range(4):
        obs = rng.integers(0, 4, (N, K)).astype(np.uint8)
        reset = (rng.random(N) < 0.3).astype(np.uint8) if t else np.ones(N, np.uint8)
        legal = None
        if masked:
            legal = (rng.random((N, A)) < 0.7).astype(np.uint8)
            legal[:, 0] = 1
        aht.aht_s5_step(pol, torch.from_numpy(obs).cuda(), torch.from_numpy(reset).cuda(), state, logits,
                        values, None if legal is None else torch.from_numpy(legal).cuda())
        aht.aht_s5_sync(pol)
        lg_ref, v_ref = net.step(obs, reset, state_ref, legal)
        lg = np_(logits)
        fin = np.isfinite(lg_ref)
        assert np.array_equal(np.isfinite(lg), fin), "masked actions"
        ok, worst = close(lg[fin], lg_ref[fin])
        assert ok, f"logits at step {t}: {worst:.3g}"
        ok, worst = close(np_(values), v_ref)
        assert ok, f"values at step {t}: {worst:.3g}"
        ok, worst = close(np_(state), state_ref)
        assert ok, f"state at step {t}: {worst:.3g}"
    pol.close()


def test_s5_rejects_bad_sizes():
    require_gpu()
    params = W.s5_params(1, 196, 6, H=32, P=32, F=32)
    bad = dict(params)
    bad["lam_re"] = -bad["lam_re"]          # growing modes
    with pytest.raises(aht.AhtError):
        aht.aht_s5_create(bad, 8)
    pol = aht.aht_s5_create(params, 8)
    obs = torch.zeros(9, 196, dtype=torch.uint8, device="cuda")
    with pytest.raises(aht.AhtError):       # more envs than max_envs
        aht.aht_s5_step(pol, obs, torch.zeros(9, dtype=torch.uint8, device="cuda"),
                        torch.zeros(9, 64, device="cuda"), torch.empty(9, 6, device="cuda"),
                        torch.empty(9, device="cuda"))


def test_s5_step_with_another_device_current():
    """A policy created on GPU 0 steps, syncs and is destroyed correctly while another
    device is current: the library makes the policy's device current for each call.
    Needs two GPUs."""
    require_gpu()
    if torch.cuda.device_count() < 2:
        pytest.skip("needs two GPUs")
    N = 64
    params = W.s5_params(0, 196, 6)
    obs, resets = lbf_observations(2, N, 5)
    legal = torch.ones(N, 6, dtype=torch.uint8, device="cuda:0")
    out = []
    for other in (False, True):
        torch.cuda.set_device(0)
        pol = aht.aht_s5_create(params, N)
        state = torch.zeros(N, 2 * O.S5(params).P, device="cuda:0")
        logits = torch.empty(N, 6, device="cuda:0")
        values = torch.empty(N, device="cuda:0")
        if other:
            torch.cuda.set_device(1)
        for t in range(2):
            aht.aht_s5_step(pol, torch.from_numpy(obs[t]).to("cuda:0"), torch.from_numpy(resets[t]).to("cuda:0"),
                            state, logits, values, legal)
        aht.aht_s5_sync(pol)
        pol.close()
        torch.cuda.set_device(0)
        out.append((logits.cpu(), values.cpu()))
    assert torch.equal(out[0][0], out[1][0]) and torch.equal(out[0][1], out[1][1])
