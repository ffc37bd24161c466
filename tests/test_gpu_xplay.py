"""Cross-play matrices on the GPU vs the oracle.

The oracle replays each env with the GPU's recorded actions: per-env returns and
episode lengths are bit-exact, the GPU's actions equal the oracle's own samples away
from CDF edges, and each matrix cell equals the exact mean of its pair's returns.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import CDF_MARGIN, make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu


def run_xplay(ctx, ego, tm, P, S, record=True):
    ne, nt = len(ego), len(tm)
    matrix = torch.empty(ne, nt, device="cuda")
    returns = torch.empty(ne, nt, P, device="cuda")
    steps = torch.empty(ne, nt, P, dtype=torch.int32, device="cuda")
    actions = torch.empty(S, ne * nt * P, 2, dtype=torch.uint8, device="cuda") if record else None
    aht.aht_xplay_matrix(ctx, ego, tm, P, S, matrix, returns, steps, actions)
    aht.aht_sync(ctx)
    return matrix, returns, steps, actions


def check(wl, pop_np, ego, tm, P, S, out, seed, step0=0, env_ids=None):
    matrix, returns, steps, actions = out
    d, pols = oracle_of(wl.env, pop_np)
    acts = np_(actions)
    sel = slice(None) if env_ids is None else env_ids
    ref = O.xplay(d, pols, seed, step0, ego, tm, P, S, forced=acts[:, sel], n_threads=8,
                  env_ids=env_ids)
    assert ref["rc"] == 0
    R = np_(returns).reshape(-1)
    assert np.array_equal(R[sel], ref["returns"]), "returns"
    assert np.array_equal(np_(steps).reshape(-1)[sel], ref["steps"]), "episode lengths"
    live = ref["own_actions"] != 255
    assert np.array_equal(ref["actions"], acts[:, sel]), "applied / recorded actions"
    agree = ~live | (ref["own_actions"] == acts[:, sel]) | (ref["margin"] < CDF_MARGIN)
    assert agree.all(), f"{(~agree).sum()} actions differ away from a CDF edge"
    want = R.reshape(len(ego), len(tm), P).astype(np.float64).mean(-1).astype(np.float32)
    assert np.array_equal(np_(matrix), want), "matrix = exact pair means"
    if env_ids is None:
        assert np.array_equal(np_(matrix), ref["matrix"])
    return ref


def test_lbf_xplay_fp32_small():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_xplay_8x16x256"]
    ctx, pop_np = make_ctx(wl, 2 * 3 * 150)
    ego, tm, P = [0, 7], [8, 15, 23], 150   # ragged: 150 = 128 + 22
    out = run_xplay(ctx, ego, tm, P, 128)
    ref = check(wl, pop_np, ego, tm, P, 128, out, wl.env_seed)
    assert (ref["steps"] <= 128).all()


def test_overcooked_xplay_small():
    require_gpu()
    wl = W.WORKLOADS["overcooked5x4_xplay_8x8x64"]
    ctx, pop_np = make_ctx(wl, 2 * 2 * 70)
    out = run_xplay(ctx, [0, 1], [8, 9], 70, 400)
    ref = check(wl, pop_np, [0, 1], [8, 9], 70, 400, out, wl.env_seed)
    assert (ref["steps"] == 400).all()


def test_hanabi_xplay_small_to_termination():
    require_gpu()
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    ctx, pop_np = make_ctx(wl, 3 * 2 * 40)
    out = run_xplay(ctx, [0, 5, 6], [16, 30], 40, 100)
    ref = check(wl, pop_np, [0, 5, 6], [16, 30], 40, 100, out, wl.env_seed)
    assert (ref["steps"] <= 97).all() and (ref["steps"] >= 1).all()


def test_step_counter_advances_between_calls():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, pop_np = make_ctx(wl, 64)
    a = run_xplay(ctx, [0], [1], 64, 50)
    b = run_xplay(ctx, [0], [1], 64, 50)
    check(wl, pop_np, [0], [1], 64, 50, b, wl.env_seed, step0=50)
    assert not torch.equal(a[1], b[1])   # fresh draws on the second call


@pytest.mark.parametrize("name", ["lbf7x7_xplay_8x16x256", "overcooked5x4_xplay_8x8x64",
                                  "hanabi_xplay_16x16x32", "lbf7x7_xplay_heuristics_8x12x256",
                                  "lbf12x12_xplay_8x16x128", "minihanabi_xplay_16x16x32"])
def test_full_size_xplay_sampled(name):
    """Every cross-play workload the bench times, in its launch configuration; the oracle
    replays a sample of the envs."""
    require_gpu()
    wl = W.WORKLOADS[name]
    n = wl.xplay_envs
    ctx, pop_np = make_ctx(wl, n)
    out = run_xplay(ctx, list(wl.ego_ids), list(wl.tm_ids), wl.envs_per_pair, wl.max_steps)
    ids = np.unique(np.concatenate([[0, n - 1], np.random.default_rng(1).integers(0, n, 30)]))
    check(wl, pop_np, list(wl.ego_ids), list(wl.tm_ids), wl.envs_per_pair, wl.max_steps, out,
          wl.env_seed, env_ids=ids)


@pytest.mark.parametrize("name,P,S", [("overcooked5x4_xplay_8x8x64", 40, 60),
                                      ("lbf7x7_xplay_8x16x256", 70, 40)])
def test_set_policy_reaches_every_kernel_copy(name, P, S):
    # Context A uploads policy 3's weights into slot 0 with aht_set_policy; context B is
    # created with that population.  Same seed and step: the matrices must be identical,
    # so the kernel's own packed copy (streamed tensor-core blocks for Overcooked, split
    # fp32 tensor-core blocks for LBF) was refreshed.
    require_gpu()
    wl = W.WORKLOADS[name]
    pop_np = W.population(wl)
    swapped = [pop_np[3]] + pop_np[1:]
    ego, tm = [0, 1], [wl.tm_ids[0], wl.tm_ids[1]]
    a, _ = make_ctx(wl, len(ego) * len(tm) * P, pop_np=pop_np)
    b, _ = make_ctx(wl, len(ego) * len(tm) * P, pop_np=swapped)
    dt = torch.float32 if wl.weight_dtype == W.FP32 else torch.bfloat16
    host = [(torch.from_numpy(Wt).to(dt), torch.from_numpy(bb).to(dt)) for Wt, bb in pop_np[3]]
    aht.aht_set_policy(a, 0, host, 0, aht.AHT_FP32 if wl.weight_dtype == W.FP32 else aht.AHT_BF16)
    ma = torch.empty(len(ego), len(tm), device="cuda")
    mb = torch.empty_like(ma)
    aht.aht_xplay_matrix(a, ego, tm, P, S, ma)
    aht.aht_xplay_matrix(b, ego, tm, P, S, mb)
    aht.aht_sync(a)
    aht.aht_sync(b)
    assert torch.equal(ma, mb)
