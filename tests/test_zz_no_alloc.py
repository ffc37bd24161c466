"""aht_xplay_matrix_static: the cross-play matrix for callers that cannot allocate device
memory after start-up.

aht_xplay_matrix keeps per-env returns in context scratch sized when the context was
created, so a context made for a small training batch cannot evaluate a larger matrix
without more device memory.  The static variant keeps that scratch in one file-scope
device array of the library instead.  Here it runs on a context of capacity 16 and must
reproduce, on two calls in a row, the matrices that aht_xplay_matrix computes on a
context sized for the whole batch (both contexts start from the same seed and step, so
their draws coincide).  On bf16 Overcooked and Hanabi contexts, whose static matrix runs
the CUDA-core kernel, each pair without a close call at a sampling-CDF edge must have the
fp64 oracle's cell exactly.  This file is collected last on purpose.
"""
import pytest
import torch

from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W

from gpu_util import make_ctx, require_gpu

pytestmark = pytest.mark.gpu


def test_static_scratch_matrix_matches_context_scratch_matrix():
    require_gpu()
    wl = W.WORKLOADS["lbf7x7_xplay_8x16x256"]
    pop_np = W.population(wl)
    ego, tm, P, S = [0, 3, 7], [8, 12, 20, 23], 200, 128   # 2400 envs, ragged tiles
    big, _ = make_ctx(wl, len(ego) * len(tm) * P, pop_np=pop_np)
    small, _ = make_ctx(wl, 16, pop_np=pop_np)
    too_small = torch.empty(len(ego), len(tm), device="cuda")
    with pytest.raises(aht.AhtError):   # context scratch cannot hold 2400 returns
        aht.aht_xplay_matrix(small, ego, tm, P, S, too_small)
    for call in range(2):
        ref = torch.empty(len(ego), len(tm), device="cuda")
        aht.aht_xplay_matrix(big, ego, tm, P, S, ref)
        got = torch.full((len(ego), len(tm)), float("nan"), device="cuda")
        aht.aht_xplay_matrix_static(small, ego, tm, P, S, got)
        aht.aht_sync(big)
        aht.aht_sync(small)
        # the matrix is an exact fp64 mean of bit-exact returns: tolerance 0
        assert torch.equal(got, ref), (call, got, ref)
        assert aht.aht_step_counter(small) == aht.aht_step_counter(big) == (call + 1) * S


def test_static_scratch_rejects_batches_above_its_size():
    require_gpu()
    wl = W.WORKLOADS["hanabi_xplay_16x16x32"]
    ctx, _ = make_ctx(wl, 8)
    m = torch.empty(64, 64, device="cuda")
    ids = list(range(32)) * 2
    with pytest.raises(aht.AhtError) as e:   # 64 * 64 * 32 envs > 65536
        aht.aht_xplay_matrix_static(ctx, ids, ids, 32, 100, m)
    assert e.value.status == aht.AHT_EINVAL
    assert aht.aht_step_counter(ctx) == 0


@pytest.mark.parametrize("name,ego,tm,P,S", [
    ("overcooked5x4_xplay_8x8x64", [0, 1, 2, 3], [8, 9, 10, 11], 2, 400),
    ("hanabi_xplay_16x16x32", [0, 5, 9], [16, 30], 40, 100),
])
def test_static_scratch_matrix_on_bf16_overcooked_and_hanabi(name, ego, tm, P, S):
    """bf16 Overcooked and Hanabi contexts: the static variant runs the CUDA-core
    cross-play kernel.  The oracle plays the same episodes free-running in fp64; an env
    whose every sample lies at least 1e-5 from a CDF edge plays the oracle's episode
    exactly, so each pair with no such close call has exactly the oracle's cell, on two
    calls in a row (the second from the advanced step counter)."""
    import numpy as np
    import oracle as O
    from gpu_util import CDF_MARGIN, oracle_of
    require_gpu()
    wl = W.WORKLOADS[name]
    ctx, pop_np = make_ctx(wl, 16)
    d, pols = oracle_of(wl.env, pop_np)
    checked = 0
    for call in range(2):
        got = torch.full((len(ego), len(tm)), float("nan"), device="cuda")
        aht.aht_xplay_matrix_static(ctx, ego, tm, P, S, got)
        aht.aht_sync(ctx)
        ref = O.xplay(d, pols, wl.env_seed, call * S, ego, tm, P, S, n_threads=8)
        assert ref["rc"] == 0
        close_call = (ref["margin"] < CDF_MARGIN).any(axis=(0, 2)).reshape(len(ego), len(tm), P).any(-1)
        g = got.cpu().numpy()
        assert np.isfinite(g).all()
        assert np.array_equal(g[~close_call], ref["matrix"][~close_call]), call
        checked += int((~close_call).sum())
        assert aht.aht_step_counter(ctx) == (call + 1) * S
    assert checked >= len(ego) * len(tm)   # most pairs have no close call
