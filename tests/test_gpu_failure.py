"""Failure detection without a GPU fault.

Every wait of the tensor-core kernels on another warp's progress is bounded by
%globaltimer; on expiry the kernel latches a status bit, stops, drains its own work and
returns.  Here a wait is made to expire on purpose (an mbarrier nothing arrives on, a
1 ms limit): the host must read the timeout from aht_sync, and the context must stay
usable for the next call.  First in a one-thread probe, then inside the real kernels
(aht_debug_expire_at): the two-warp-group kernel (collection, IPPO and LBF cross-play),
the sparse-first-layer kernel and the streamed cross-play kernel, each mid-call with MMAs
in flight.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, np_, oracle_of, require_gpu

pytestmark = pytest.mark.gpu


def test_expired_wait_is_reported_and_the_context_stays_usable():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, pop_np = make_ctx(wl, 64)
    aht.aht_debug_expire_wait(ctx, 1_000_000)
    with pytest.raises(aht.AhtError) as e:
        aht.aht_sync(ctx)
    assert e.value.status == aht.AHT_ETIMEOUT
    aht.aht_sync(ctx)                     # the status word was cleared
    # the next rollout runs normally and matches the oracle's replay of its actions
    T = 12
    traj = aht.traj_buffers(ctx, T)
    aht.aht_rollout(ctx, 0, [1], T, traj)
    aht.aht_sync(ctx)
    d, pols = oracle_of(wl.env, pop_np)
    st = O.reset_all(d, wl.env_seed, 64)
    acts = np.stack([np_(traj["actions"]), np_(traj["tm_actions"])], -1)
    ref = O.rollout(d, pols, wl.env_seed, st, 0, T, 0, [1], forced=acts)
    assert ref["rc"] == 0
    assert np.array_equal(np_(traj["obs"]), ref["obs"])
    assert np.array_equal(np_(traj["rewards"]), ref["rewards"])


def test_expire_wait_validates_its_limit():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, _ = make_ctx(wl, 8)
    for bad in (0, -5, 2_000_000_000):
        with pytest.raises(aht.AhtError) as e:
            aht.aht_debug_expire_wait(ctx, bad)
        assert e.value.status == aht.AHT_EINVAL
    aht.aht_sync(ctx)


def expire_then(ctx, call):
    """Runs `call` with the failure hook armed: the kernel's wait expires mid-call and
    aht_sync reports AHT_ETIMEOUT."""
    with pytest.raises(aht.AhtError) as e:
        call()
        aht.aht_sync(ctx)
    assert e.value.status == aht.AHT_ETIMEOUT
    aht.aht_sync(ctx)   # cleared


@pytest.mark.parametrize("wl_name,pool,ippo", [
    ("lbf7x7_ppo_16384x128", [1, 2, 3, 4], False),   # two-group kernel, gathered tiles
    ("lbf7x7_ppo_16384x128", [2], False),            # two-group kernel, contiguous tiles
    ("lbf7x7_ippo_16384x128", [1], True),            # two-group kernel, IPPO
    ("lbf12x12_ppo_4096x128", [1, 2, 3], False),     # sparse first layer, gathered tiles
])
def test_collection_kernel_wait_expires_mid_rollout(wl_name, pool, ippo):
    """The real collection kernels: a wait made to expire at step 5 of 12 takes the abort
    path (MMAs drained, tensor memory freed); the context keeps its pre-call env state,
    and the next call matches the oracle's replay from that state."""
    require_gpu()
    wl = W.WORKLOADS[wl_name]
    N, T = 300, 12
    ctx, pop_np = make_ctx(wl, N)
    traj = aht.traj_buffers(ctx, T)
    traj1 = aht.traj_buffers(ctx, T) if ippo else None

    def run():
        if ippo:
            aht.aht_rollout_ippo(ctx, 0, pool[0], T, traj, traj1)
        else:
            aht.aht_rollout(ctx, 0, pool, T, traj)

    aht.aht_debug_expire_at(ctx, 5, 1_000_000)
    expire_then(ctx, run)
    assert aht.aht_step_counter(ctx) == T
    run()                                   # the hook fired once: a normal call
    aht.aht_sync(ctx)
    d, pols = oracle_of(wl.env, pop_np)
    acts = np.stack([np_(traj["actions"]), np_(traj["tm_actions"])], -1)
    ref = O.rollout(d, pols, wl.env_seed, O.reset_all(d, wl.env_seed, N), T, T, 0, pool,
                    forced=acts, n_threads=8)
    assert ref["rc"] == 0
    assert np.array_equal(np_(traj["obs"]), ref["obs"])
    assert np.array_equal(np_(traj["rewards"]), ref["rewards"])
    assert np.array_equal(np_(traj["dones"]), ref["dones"])
    assert ((ref["own_actions"] == acts) | (ref["margin"] < 1e-5)).all()


@pytest.mark.parametrize("name,ego,tm,P,S,at", [
    ("lbf7x7_xplay_8x16x256", [0, 3], [8, 9], 70, 40, 7),
    ("overcooked5x4_xplay_8x8x64", [0, 1], [8, 9], 40, 30, 4),
    ("hanabi_xplay_16x16x32", [0, 5], [16, 30], 40, 100, 3),
])
def test_cross_play_kernel_wait_expires(name, ego, tm, P, S, at):
    """The real cross-play kernels (LBF one-launch rollout, streamed Overcooked / Hanabi
    steps): the expired wait is reported, the aborted matrix is not passed off as valid,
    and the next matrix matches the oracle (each call resets its envs)."""
    require_gpu()
    from test_gpu_xplay import check, run_xplay
    wl = W.WORKLOADS[name]
    ctx, pop_np = make_ctx(wl, len(ego) * len(tm) * P)
    aht.aht_debug_expire_at(ctx, at, 1_000_000)
    m = torch.zeros(len(ego), len(tm), device="cuda")
    expire_then(ctx, lambda: aht.aht_xplay_matrix(ctx, ego, tm, P, S, m))
    if name.startswith("lbf"):
        assert torch.isnan(m).all()         # every tile gave up: NaN, never stale
    out = run_xplay(ctx, ego, tm, P, S)
    check(wl, pop_np, ego, tm, P, S, out, wl.env_seed, step0=S)


def test_expire_at_validates_its_limit():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    ctx, _ = make_ctx(wl, 8)
    for bad in (0, 2_000_000_000):
        with pytest.raises(aht.AhtError) as e:
            aht.aht_debug_expire_at(ctx, 3, bad)
        assert e.value.status == aht.AHT_EINVAL
    aht.aht_debug_expire_at(ctx, -1, 0)     # clearing needs no limit


@pytest.mark.parametrize("name,n_envs", [
    ("lbf7x7_ppo_16384x128", 500),      # bf16 LBF: tensor-core blocks too
    ("lbf7x7_64x50_fp32", 64),          # fp32 LBF: split-weight blocks
    ("hanabi_xplay_16x16x32", 300),     # streamed cross-play buffers too
])
def test_create_unwinds_every_failed_allocation(name, n_envs):
    """aht_create with its k-th allocation failing, for every k: AHT_ENOMEM, no context,
    and every block it had allocated is freed (the library's live-block count and the
    device's free memory are back where they were); then a normal create succeeds."""
    require_gpu()
    wl = W.WORKLOADS[name]
    import gc
    ctx, _ = make_ctx(wl, n_envs)            # loads the kernels once
    ctx.close()
    gc.collect()                             # contexts of earlier tests go now, not mid-loop
    gc.disable()
    torch.cuda.synchronize()
    base = aht.aht_debug_live_allocs()
    free0 = torch.cuda.mem_get_info()[0]
    k, failed = 1, 0
    while True:
        aht.aht_debug_fail_alloc(k)
        try:
            ctx, _ = make_ctx(wl, n_envs)
        except aht.AhtError as e:
            assert e.status == aht.AHT_ENOMEM, (k, e)
            assert aht.aht_debug_live_allocs() == base, k
            failed += 1
            k += 1
            continue
        finally:
            aht.aht_debug_fail_alloc(0)
        break                                # k exceeds the allocations of one create
    assert failed >= 10                      # every allocation of a create was tried
    assert aht.aht_debug_live_allocs() == base + failed
    ctx.close()
    gc.enable()
    assert aht.aht_debug_live_allocs() == base
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) <= 4 << 20
