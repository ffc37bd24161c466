"""aht_xplay_matrix_static: the cross-play matrix for callers that cannot allocate device
memory after start-up.

aht_xplay_matrix keeps per-env returns in context scratch sized when the context was
created, so a context made for a small training batch cannot evaluate a larger matrix
without more device memory.  The static variant keeps that scratch in one file-scope
device array of the library instead.  Here it runs on a context of capacity 16 and must
reproduce, on two calls in a row, the matrices that aht_xplay_matrix computes on a
context sized for the whole batch (both contexts start from the same seed and step, so
their draws coincide).  This file is collected last on purpose.
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
