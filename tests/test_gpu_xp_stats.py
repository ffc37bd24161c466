"""GPU parity of the cross-play matrix consumers (aht_xp_stats) against the fp64 oracle.

Both sides compute in fp64 and round each output to f32 once.  The bounds, the
elementwise outputs (normalised return, regret) and the row maxima of the regret are the
same fp64 operations on the same operands, so they are compared bit for bit (NaN where
the bound is <= 0 included).  The means add the same fp64 terms in another order (the
kernel: lanes then a shuffle tree; the oracle: left to right); the two fp64 sums differ by
a few units in the 53rd bit, so after the f32 rounding they agree to one unit in the last
place (BRDiv, a difference of two means, to 1e-12 of the matrix scale).
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_13716_gb300 import aht
from paper_2609_13716_gb300 import workloads as W
from gpu_util import require_gpu

pytestmark = [pytest.mark.gpu, pytest.mark.filterwarnings("ignore::RuntimeWarning")]


def run_gpu(xp, prior):
    ne, nt = xp.shape
    dev = "cuda"
    x = torch.from_numpy(xp).to(dev)
    up = torch.from_numpy(prior.astype(np.float32)).to(dev)
    o = dict(norm=torch.empty(ne, nt, device=dev), regret=torch.empty(ne, nt, device=dev),
             j_aht=torch.empty(ne, device=dev), j_norm=torch.empty(ne, device=dev),
             max_regret=torch.empty(ne, device=dev),
             worst_tm=torch.empty(ne, dtype=torch.int32, device=dev),
             brdiv=torch.empty(1, device=dev) if ne == nt else None)
    aht.aht_xp_stats(x, up, **o)
    torch.cuda.synchronize()
    res = {k: (v.cpu().numpy() if v is not None else None) for k, v in o.items()}
    res["upper"] = up.cpu().numpy()
    return res


def check(xp, prior):
    g = run_gpu(xp, prior)
    r = O.xp_stats(xp, prior.astype(np.float32).astype(np.float64))
    f = np.float32
    np.testing.assert_array_equal(g["upper"], r["upper"].astype(f))
    for k in ("norm", "regret", "max_regret"):
        np.testing.assert_array_equal(g[k], r[k].astype(f), err_msg=k)
    np.testing.assert_array_equal(g["worst_tm"], r["worst"])
    for k in ("j_aht", "j_norm"):
        want = r[k].astype(f)
        assert (np.isnan(g[k]) == np.isnan(want)).all(), k
        ok = ~np.isnan(want)
        np.testing.assert_array_max_ulp(g[k][ok], want[ok], maxulp=1)
    if r["brdiv"] is not None:
        scale = float(np.abs(xp).max())
        assert abs(float(g["brdiv"][0]) - r["brdiv"]) <= 2.0 ** -24 * abs(r["brdiv"]) + 1e-12 * scale
    return g


@pytest.mark.parametrize("ne,nt,scale,quantum", [
    (1, 1, 1.0, 0.0), (8, 16, 1.0, 0.0), (8, 8, 200.0, 20.0 / 64), (16, 16, 25.0, 1.0 / 32),
    (64, 64, 1.0, 0.0), (33, 17, 3.0, 0.25), (300, 300, 1.0, 0.0), (2048, 3, 5.0, 1.0),
    (5, 2048, 1.0, 0.0), (257, 255, 10.0, 0.5)])
def test_parity_random(ne, nt, scale, quantum):
    require_gpu()
    xp = W.xp_matrix(17 * ne + nt, ne, nt, scale, quantum)
    check(xp, np.full(nt, -np.inf))


def test_parity_priors_ties_and_nonpositive_bounds():
    require_gpu()
    ne, nt = 24, 40
    xp = W.xp_matrix(5, ne, nt, 4.0, 1.0)   # integer scores: many ties for the argmax
    xp[:, 3] = 0.0                          # every return 0: bound 0, NaN normalisation
    xp[:, 7] = -1.0                         # negative bound
    prior = np.full(nt, -np.inf)
    prior[0] = 100.0                        # a prior above every score is kept
    prior[1] = 0.5                          # a prior below is replaced
    prior[2] = np.nan                       # a NaN bound is never exceeded
    g = check(xp, prior)
    assert g["upper"][0] == 100.0 and np.isnan(g["upper"][2])
    assert np.isnan(g["norm"][:, 3]).all() and np.isnan(g["j_norm"]).all()


def test_refinement_over_two_calls_matches_one_call_on_stacked_rows():
    require_gpu()
    a = W.xp_matrix(11, 8, 16)
    b = W.xp_matrix(12, 8, 16, 1.3)
    up = np.full(16, -np.inf)
    g1 = run_gpu(a, up)
    g2 = run_gpu(b, g1["upper"])
    r = O.xp_stats(np.concatenate([a, b]), up)
    np.testing.assert_array_equal(g2["upper"], r["upper"].astype(np.float32))
