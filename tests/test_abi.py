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


def test_null_handles_and_arguments_are_rejected_before_any_cuda_call(lib):
    # Every entry point that takes a context, learner or S5 handle checks it (and its
    # output pointers) on the host first: AHT_EINVAL and a message, no CUDA call, so
    # none of this needs a GPU.  The destroy calls accept NULL.
    import ctypes as C
    from paper_2609_13716_gb300 import aht
    L = aht.load()
    E = aht.AHT_EINVAL
    fake = C.c_void_p(16)  # never dereferenced: each call fails a host check first
    t = aht.Traj()
    i32 = C.c_int32
    ids = (i32 * 2)(0, 1)
    calls = {
        "aht_sync": lambda: L.aht_sync(None),
        "aht_set_timing": lambda: L.aht_set_timing(None, 1),
        "aht_get_timing": lambda: L.aht_get_timing(None, None, None),
        "aht_get_state": lambda: L.aht_get_state(None, None, None),
        "aht_set_state": lambda: L.aht_set_state(None, None, 0),
        "aht_set_policy": lambda: L.aht_set_policy(None, 0, None, None, 0, 0),
        "aht_step_forced": lambda: L.aht_step_forced(None, None, None),
        "aht_policy_forward": lambda: L.aht_policy_forward(None, 0, None, 1, None),
        "aht_rollout_ippo": lambda: L.aht_rollout_ippo(None, 0, 1, 4, C.byref(t), C.byref(t)),
        "aht_rollout_resample": lambda: L.aht_rollout_resample(None, 0, ids, 2, 4, C.byref(t), None),
        "aht_debug_expire_at": lambda: L.aht_debug_expire_at(None, 1, 1000),
        "aht_debug_logits": lambda: L.aht_debug_logits(None, None, 0),
        "aht_learner_get": lambda: L.aht_learner_get(None, None, None, None, None, None),
        "aht_learner_set": lambda: L.aht_learner_set(None, None, None, None, 0, 0),
        "aht_learner_push": lambda: L.aht_learner_push(None, None, 0),
        "aht_learner_sync": lambda: L.aht_learner_sync(None),
        "aht_ppo_grad": lambda: L.aht_ppo_grad(None, C.byref(t), 1, 1, 0, 0, None, None),
        "aht_s5_step": lambda: L.aht_s5_step(None, fake, fake, fake, 1, fake, fake, fake),
        "aht_s5_sync": lambda: L.aht_s5_sync(None),
    }
    L.aht_xplay_matrix_static.argtypes = [C.c_void_p, C.POINTER(i32), i32, C.POINTER(i32), i32, i32,
                                          i32, C.c_void_p]
    L.aht_xplay_matrix_static.restype = C.c_int
    calls["aht_xplay_matrix_static"] = lambda: L.aht_xplay_matrix_static(None, ids, 1, ids, 1, 4, 4, fake)
    L.aht_debug_tanh.argtypes = [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]
    L.aht_debug_tanh.restype = C.c_int
    calls["aht_debug_tanh"] = lambda: L.aht_debug_tanh(None, None, 4, None)
    out = C.c_void_p(16)
    calls["aht_s5_create (NULL params)"] = lambda: L.aht_s5_create(None, 16, None, C.byref(out))
    calls["aht_s5_create (NULL out)"] = lambda: L.aht_s5_create(None, 16, None, None)
    for name, call in calls.items():
        assert call() == E, name
        assert L.aht_last_error(), name
    assert out.value is None  # aht_s5_create clears *out before it fails
    L.aht_destroy(None)
    L.aht_learner_destroy(None)
    L.aht_s5_destroy(None)


def test_s5_create_checks_its_sizes_and_arrays_on_the_host(lib):
    # aht_s5_create validates the model sizes, max_envs, every parameter array and the
    # sign of Re(lambda) (the S5 recurrence must decay) before it allocates or touches
    # the device.
    import ctypes as C
    import numpy as np
    from paper_2609_13716_gb300 import aht
    L = aht.load()
    keep = []

    def arr(n, v=0.1):
        a = np.full(n, v, np.float32)
        keep.append(a)
        return a.ctypes.data_as(C.POINTER(C.c_float))

    def params(**kw):
        p = aht.S5Params()
        p.obs_dim, p.n_actions, p.H, p.P, p.F = 196, 6, 128, 128, 1024
        for f in ("We1", "be1", "We2", "be2", "lam_im", "log_dt", "B_re", "B_im", "C_re", "C_im", "D"):
            setattr(p, f, arr(4))
        p.lam_re = arr(128, -0.5)
        for l in range(4):
            p.Wa[l], p.ba[l], p.Wc[l], p.bc[l] = arr(4), arr(4), arr(4), arr(4)
        for k, v in kw.items():
            setattr(p, k, v)
        return p

    out = C.c_void_p()
    cases = [
        (params(H=100), 16, b"multiples of 32"),
        (params(P=160), 16, b"P <= 128"),
        (params(n_actions=33), 16, b"n_actions"),
        (params(obs_dim=0), 16, b"obs_dim"),
        (params(), 0, b"max_envs"),
        (params(), (1 << 20) + 1, b"max_envs"),
        (params(D=None), 16, b"NULL parameter array"),
        (params(lam_re=arr(128, 0.0)), 16, b"negative"),
    ]
    p = params()
    p.Wc[3] = None
    cases.append((p, 16, b"NULL head array"))
    for prm, n, msg in cases:
        assert L.aht_s5_create(C.byref(prm), n, None, C.byref(out)) == aht.AHT_EINVAL, msg
        assert msg in L.aht_last_error(), (msg, L.aht_last_error())
        assert out.value is None
