"""Failure detection without a GPU fault.

Every wait of the tensor-core kernels on another warp's progress is bounded by
%globaltimer; on expiry the kernel latches a status bit, stops, drains its own work and
returns.  Here a wait is made to expire on purpose (an mbarrier nothing arrives on, a
1 ms limit): the host must read the timeout from aht_sync, and the context must stay
usable for the next call.
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
