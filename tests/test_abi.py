"""The C-ABI library builds for sm_103a, loads, and exports every symbol include/aht.h declares."""
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "aht.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(aht_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_13716_gb300 import build
    path = build.build()
    return path


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ("aht_create", "aht_reset", "aht_rollout", "aht_xplay_matrix", "aht_gae"):
        assert name in syms


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", lib], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\b[TtWw] (aht_\w+)", out))
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, missing


def test_library_loads_and_binding_matches(lib):
    from paper_2609_13716_gb300 import aht
    L = aht.load()
    for s in declared_symbols():
        assert hasattr(L, s), s
    assert set(aht.EXPORTED) <= set(declared_symbols())
    assert L.aht_status_string(1) == b"invalid argument"


def test_host_validation_needs_no_gpu(lib):
    # Argument checks happen before any CUDA call.
    import ctypes as C
    from paper_2609_13716_gb300 import aht
    L = aht.load()
    bad = aht.EnvDesc(0, 2, 7, 3, 3, 50, 0, 0)   # LBF width 2 is invalid
    h = C.c_void_p()
    assert L.aht_create(C.byref(bad), None, 4, 0, None, C.byref(h)) == aht.AHT_EINVAL
    assert b"width" in L.aht_last_error()
    assert L.aht_gae(None, None, None, None, 1, 1, 0.9, 0.9, None, None, None) == aht.AHT_EINVAL
    t = aht.Traj()
    assert L.aht_traj_copy(None, C.byref(t), 1, 1, 1, None) == aht.AHT_EINVAL
    assert L.aht_traj_copy(C.byref(t), C.byref(t), 0, 1, 1, None) == aht.AHT_EINVAL
    L.aht_debug_expire_wait.argtypes = [C.c_void_p, C.c_int64]
    assert L.aht_debug_expire_wait(None, 1000) == aht.AHT_EINVAL
    assert L.aht_debug_obs_words(None, 0, None) == aht.AHT_EINVAL

    out = aht.XpStatsOut()
    fake = C.c_void_p(16)  # never dereferenced: every case below fails a host check
    assert L.aht_xp_stats(None, 2, 2, fake, C.byref(out), None) == aht.AHT_EINVAL
    assert L.aht_xp_stats(fake, 0, 2, fake, C.byref(out), None) == aht.AHT_EINVAL
    assert L.aht_xp_stats(fake, 2, 2049, fake, C.byref(out), None) == aht.AHT_EINVAL
    out.brdiv = 16
    assert L.aht_xp_stats(fake, 2, 3, fake, C.byref(out), None) == aht.AHT_EINVAL
    assert b"square" in L.aht_last_error()
    # PPO learner: host checks before any CUDA call
    cfg = aht.PpoConfig(**aht.PPO_DEFAULTS)
    ptrs = (C.c_void_p * 3)(16, 16, 16)
    out_l = C.c_void_p()
    assert L.aht_learner_create(195, 6, ptrs, ptrs, C.byref(cfg), None, C.byref(out_l)) == aht.AHT_EINVAL
    assert b"obs_dim" in L.aht_last_error()
    assert L.aht_learner_create(196, 8, ptrs, ptrs, C.byref(cfg), None, C.byref(out_l)) == aht.AHT_EINVAL
    bad_cfg = aht.PpoConfig(**dict(aht.PPO_DEFAULTS, minibatches=0))
    assert L.aht_learner_create(196, 6, ptrs, ptrs, C.byref(bad_cfg), None, C.byref(out_l)) == aht.AHT_EINVAL
    assert L.aht_ppo_update(None, None, 64, 1, None) == aht.AHT_EINVAL
    assert L.aht_learner_n_params(None) == -1
