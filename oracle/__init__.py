"""CPU oracle for the batched ad hoc teamwork rollout path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and
``--impl reference`` legs may import this package.  The product package
(``paper_2609_13716_gb300``) never imports it and shares no code with it.

The C++ source (``aht_oracle.cpp``) is compiled on first use into ``oracle/_build``
with plain ``g++ -O2 -ffp-contract=off`` (no intrinsics, no fast-math), so fp32 reward
arithmetic is IEEE single on x86-64 and aarch64 alike.  This module only marshals
arguments; every step of the oracle's arithmetic lives in the C++ file.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_SRC = [os.path.join(_HERE, "aht_oracle.cpp"), os.path.join(_HERE, "ppo_oracle.cpp"),
        os.path.join(_HERE, "s5_oracle.cpp")]
_HDR = os.path.join(_HERE, "aht_oracle.h")
_lock = threading.Lock()
_lib = None

LBF, OVERCOOKED, HANABI, MINI_HANABI = 0, 1, 2, 3
STREAM_ACT0, STREAM_ACT1, STREAM_RESET, STREAM_TEAMMATE = 0, 1, 2, 3
STATE_BYTES = 768
# LBF heuristic teammates: teammate id -1 - k (App. F LBF suite; rules in aht_oracle.h)
LBF_HEURISTICS = ("greedy_closest_self", "greedy_closest_teammate", "greedy_closest_avg",
                  "greedy_lowest_level", "greedy_highest_level", "seq_lexicographic",
                  "seq_reverse_lexicographic", "seq_column_major", "seq_reverse_column_major",
                  "seq_nearest_agent", "seq_farthest_agent", "entitled")


def heuristic_id(name):
    return -1 - LBF_HEURISTICS.index(name)


def build(force: bool = False) -> str:
    """Compile the oracle shared library (g++, seconds).  Returns its path."""
    os.makedirs(_BUILD, exist_ok=True)
    newest = max(os.path.getmtime(p) for p in _SRC + [_HDR])
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= newest:
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-pthread", "-Wall", "-o", tmp] + _SRC
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


class EnvDesc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("width", C.c_int32), ("height", C.c_int32),
                ("n_food", C.c_int32), ("max_agent_level", C.c_int32),
                ("episode_len", C.c_int32), ("cook_time", C.c_int32),
                ("soup_reward", C.c_int32)]


class LbfState(C.Structure):
    _fields_ = [("ax", C.c_int32 * 2), ("ay", C.c_int32 * 2), ("al", C.c_int32 * 2),
                ("fx", C.c_int32 * 3), ("fy", C.c_int32 * 3), ("fl", C.c_int32 * 3),
                ("eaten", C.c_int32 * 3), ("F", C.c_int32), ("ep_t", C.c_int32),
                ("done", C.c_int32), ("ret", C.c_float), ("ix", C.c_int32 * 2),
                ("iy", C.c_int32 * 2)]


class OcState(C.Structure):
    _fields_ = [("ax", C.c_int32 * 2), ("ay", C.c_int32 * 2), ("face", C.c_int32 * 2),
                ("held", C.c_int32 * 2), ("pot_n", C.c_int32), ("pot_timer", C.c_int32),
                ("counter_item", C.c_int32 * 20), ("ep_t", C.c_int32), ("done", C.c_int32),
                ("ret", C.c_float)]


class MiniHanabiState(C.Structure):
    _fields_ = [("deck", C.c_int32 * 18), ("ptr", C.c_int32),
                ("hand", (C.c_int32 * 2) * 2), ("n_hand", C.c_int32 * 2),
                ("know", (C.c_uint32 * 2) * 2), ("hint_col", (C.c_uint32 * 2) * 2),
                ("hint_rank", (C.c_uint32 * 2) * 2), ("fw", C.c_int32 * 3),
                ("info", C.c_int32), ("lives", C.c_int32), ("score", C.c_int32),
                ("disc", C.c_int32 * 9), ("fr", C.c_int32), ("turn", C.c_int32),
                ("la_valid", C.c_int32), ("la_actor", C.c_int32), ("la_type", C.c_int32),
                ("la_colour", C.c_int32), ("la_rank", C.c_int32), ("la_slot", C.c_int32),
                ("la_card", C.c_int32), ("la_hinted", C.c_int32), ("la_success", C.c_int32),
                ("la_bomb", C.c_int32), ("done", C.c_int32), ("ret", C.c_float)]


class HanabiState(C.Structure):
    _fields_ = [("deck", C.c_int32 * 50), ("ptr", C.c_int32),
                ("hand", (C.c_int32 * 5) * 2), ("n_hand", C.c_int32 * 2),
                ("know", (C.c_uint32 * 5) * 2), ("hint_col", (C.c_uint32 * 5) * 2),
                ("hint_rank", (C.c_uint32 * 5) * 2), ("fw", C.c_int32 * 5),
                ("info", C.c_int32), ("lives", C.c_int32), ("score", C.c_int32),
                ("disc", C.c_int32 * 25), ("fr", C.c_int32), ("turn", C.c_int32),
                ("la_valid", C.c_int32), ("la_actor", C.c_int32), ("la_type", C.c_int32),
                ("la_colour", C.c_int32), ("la_rank", C.c_int32), ("la_slot", C.c_int32),
                ("la_card", C.c_int32), ("la_hinted", C.c_int32), ("la_success", C.c_int32),
                ("la_bomb", C.c_int32), ("done", C.c_int32), ("ret", C.c_float)]


class Mlp(C.Structure):
    _fields_ = [("obs_dim", C.c_int32), ("h0", C.c_int32), ("h1", C.c_int32),
                ("n_out", C.c_int32),
                ("W1", C.POINTER(C.c_double)), ("b1", C.POINTER(C.c_double)),
                ("W2", C.POINTER(C.c_double)), ("b2", C.POINTER(C.c_double)),
                ("W3", C.POINTER(C.c_double)), ("b3", C.POINTER(C.c_double))]


_P = C.c_void_p


class PpoNet(C.Structure):
    _fields_ = [("obs_dim", C.c_int32), ("h0", C.c_int32), ("h1", C.c_int32), ("n_act", C.c_int32)]


class PpoHp(C.Structure):
    _fields_ = [("epochs", C.c_int32), ("minibatches", C.c_int32), ("lr", C.c_double),
                ("clip_eps", C.c_double), ("vf_coef", C.c_double), ("ent_coef", C.c_double),
                ("max_grad_norm", C.c_double), ("adam_b1", C.c_double), ("adam_b2", C.c_double),
                ("adam_eps", C.c_double), ("seed", C.c_uint64), ("epoch0", C.c_int64),
                ("round_bf16", C.c_int32)]


class PpoBatch(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("actions", C.c_void_p), ("logp", C.c_void_p),
                ("values", C.c_void_p), ("advantages", C.c_void_p), ("targets", C.c_void_p)]


class RolloutIO(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("n_envs", C.c_int64), ("step0", C.c_int64),
                ("T", C.c_int32), ("ego_id", C.c_int32), ("pool", _P), ("pool_size", C.c_int32),
                ("forced", _P), ("env_ids", _P), ("states", _P), ("n_threads", C.c_int32),
                ("teammate", _P), ("obs", _P), ("obs_tm", _P), ("actions", _P),
                ("own_actions", _P), ("margin", _P), ("logits", _P), ("logp", _P),
                ("values", _P), ("rewards", _P), ("dones", _P), ("last_value", _P),
                ("logp_tm", _P), ("values_tm", _P), ("last_value_tm", _P),
                ("resample", C.c_int32), ("ep_step", _P), ("teammates_t", _P)]


class XplayIO(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("step0", C.c_int64), ("ego_ids", _P),
                ("n_ego", C.c_int32), ("tm_ids", _P), ("n_tm", C.c_int32),
                ("envs_per_pair", C.c_int32), ("max_steps", C.c_int32), ("forced", _P),
                ("env_ids", _P), ("n_sel", C.c_int64), ("n_threads", C.c_int32), ("returns", _P), ("steps", _P), ("actions", _P),
                ("own_actions", _P), ("margin", _P), ("matrix", _P), ("logits", _P),
                ("logit_stride", C.c_int32)]


def lib() -> C.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            L.orc_philox4x32_10.argtypes = [C.c_uint32, C.c_uint32, _P, _P]
            L.orc_draw.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32]
            L.orc_draw.restype = C.c_uint32
            L.orc_uniform_int.argtypes = [C.c_uint32, C.c_uint32]
            L.orc_uniform_int.restype = C.c_uint32
            L.orc_u01.argtypes = [C.c_uint32]
            L.orc_u01.restype = C.c_double
            for f in ("orc_obs_dim", "orc_n_actions", "orc_check_desc"):
                getattr(L, f).argtypes = [C.POINTER(EnvDesc)]
                getattr(L, f).restype = C.c_int32
            L.orc_lbf_reset.argtypes = [C.POINTER(EnvDesc), C.c_uint64, C.c_uint32, C.c_uint32, C.POINTER(LbfState)]
            L.orc_lbf_step.argtypes = [C.POINTER(EnvDesc), C.POINTER(LbfState), C.c_int32, C.c_int32, _P, _P]
            L.orc_lbf_step.restype = C.c_int32
            L.orc_lbf_obs.argtypes = [C.POINTER(EnvDesc), C.POINTER(LbfState), C.c_int32, _P]
            L.orc_lbf_heuristic.argtypes = [C.POINTER(EnvDesc), C.POINTER(LbfState), C.c_int32, C.c_int32]
            L.orc_lbf_heuristic.restype = C.c_int32
            L.orc_oc_cell.argtypes = [C.c_int32, C.c_int32]
            L.orc_oc_cell.restype = C.c_int32
            L.orc_oc_reset.argtypes = [C.POINTER(EnvDesc), C.POINTER(OcState)]
            L.orc_oc_step.argtypes = [C.POINTER(EnvDesc), C.POINTER(OcState), C.c_int32, C.c_int32, _P, _P]
            L.orc_oc_step.restype = C.c_int32
            L.orc_oc_obs.argtypes = [C.POINTER(EnvDesc), C.POINTER(OcState), C.c_int32, _P]
            L.orc_hanabi_reset.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.POINTER(HanabiState)]
            L.orc_hanabi_legal.argtypes = [C.POINTER(HanabiState), _P]
            L.orc_hanabi_step.argtypes = [C.POINTER(HanabiState), C.c_int32, _P]
            L.orc_hanabi_step.restype = C.c_int32
            L.orc_hanabi_obs.argtypes = [C.POINTER(HanabiState), C.c_int32, _P]
            L.orc_mhanabi_reset.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.POINTER(MiniHanabiState)]
            L.orc_mhanabi_legal.argtypes = [C.POINTER(MiniHanabiState), _P]
            L.orc_mhanabi_step.argtypes = [C.POINTER(MiniHanabiState), C.c_int32, _P]
            L.orc_mhanabi_step.restype = C.c_int32
            L.orc_mhanabi_obs.argtypes = [C.POINTER(MiniHanabiState), C.c_int32, _P]
            L.orc_mlp_forward.argtypes = [C.POINTER(Mlp), _P, _P]
            L.orc_sample.argtypes = [_P, _P, C.c_int32, C.c_double, _P, _P, _P]
            L.orc_logp.argtypes = [_P, _P, C.c_int32, C.c_int32]
            L.orc_logp.restype = C.c_double
            L.orc_gae.argtypes = [_P, _P, _P, _P, C.c_int64, C.c_int32, C.c_double, C.c_double, _P, _P]
            L.orc_rollout.argtypes = [C.POINTER(EnvDesc), C.POINTER(Mlp), C.c_int32, C.POINTER(RolloutIO)]
            L.orc_rollout.restype = C.c_int32
            L.orc_reset_all.argtypes = [C.POINTER(EnvDesc), C.c_uint64, C.c_int64, C.c_int64, _P]
            L.orc_reset_all.restype = C.c_int32
            L.orc_reset_envs.argtypes = [C.POINTER(EnvDesc), C.c_uint64, _P, C.c_int64, C.c_int64, _P]
            L.orc_reset_envs.restype = C.c_int32
            L.orc_step_forced.argtypes = [C.POINTER(EnvDesc), C.c_uint64, C.c_int64, C.c_int64, _P, _P, _P, _P, _P, _P]
            L.orc_step_forced.restype = C.c_int32
            L.orc_xplay.argtypes = [C.POINTER(EnvDesc), C.POINTER(Mlp), C.c_int32, C.POINTER(XplayIO)]
            L.orc_xplay.restype = C.c_int32
            L.orc_policy_outputs.argtypes = [C.POINTER(Mlp), _P, C.c_int64, _P]
            L.orc_ppo_n_params.argtypes = [C.POINTER(PpoNet)]
            L.orc_ppo_n_params.restype = C.c_int64
            L.orc_bf16_round.argtypes = [C.c_double]
            L.orc_bf16_round.restype = C.c_double
            L.orc_perm_index.argtypes = [C.c_uint64, C.c_int64, C.c_int64, C.c_int64]
            L.orc_perm_index.restype = C.c_int64
            L.orc_ppo_grad.argtypes = [C.POINTER(PpoNet), _P, C.POINTER(PpoBatch), _P, C.c_int64,
                                       C.POINTER(PpoHp), _P, _P, C.c_int32]
            L.orc_adam_step.argtypes = [C.c_int64, _P, _P, _P, _P, _P, C.POINTER(PpoHp)]
            L.orc_ppo_update.argtypes = [C.POINTER(PpoNet), _P, _P, _P, _P, C.POINTER(PpoBatch),
                                         C.c_int64, C.POINTER(PpoHp), _P, C.c_int32]
            L.orc_xp_stats.argtypes = [_P, C.c_int32, C.c_int32, _P, _P, _P, _P, _P, _P, _P, _P]
            _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


# ---------------------------------------------------------------------------------
# Thin marshalling helpers.
# ---------------------------------------------------------------------------------
def env_desc(kind, width=0, height=0, n_food=0, max_agent_level=0, episode_len=0,
             cook_time=0, soup_reward=0) -> EnvDesc:
    return EnvDesc(kind, width, height, n_food, max_agent_level, episode_len, cook_time,
                   soup_reward)


def obs_dim(d: EnvDesc) -> int:
    return lib().orc_obs_dim(C.byref(d))


def n_actions(d: EnvDesc) -> int:
    return lib().orc_n_actions(C.byref(d))


def philox(key, ctr):
    out = np.zeros(4, np.uint32)
    c = np.asarray(ctr, np.uint32)
    lib().orc_philox4x32_10(int(key[0]), int(key[1]), _ptr(c), _ptr(out))
    return out


def draw(seed, env, step, stream, n):
    return lib().orc_draw(seed, env, step, stream, n)


class Policies:
    """fp64 copies of a population's weights (exact for fp32 and bf16 inputs)."""

    def __init__(self, layers):
        # layers: list per policy of [(W1, b1), (W2, b2), (W3, b3)], any float dtype.
        self._keep = []
        arr = (Mlp * len(layers))()
        for p, pol in enumerate(layers):
            ws = [np.ascontiguousarray(np.asarray(a, dtype=np.float64)) for wb in pol for a in wb]
            self._keep.append(ws)
            W1, b1, W2, b2, W3, b3 = ws
            dp = C.POINTER(C.c_double)
            arr[p] = Mlp(W1.shape[1], W1.shape[0], W2.shape[0], W3.shape[0],
                         W1.ctypes.data_as(dp), b1.ctypes.data_as(dp),
                         W2.ctypes.data_as(dp), b2.ctypes.data_as(dp),
                         W3.ctypes.data_as(dp), b3.ctypes.data_as(dp))
        self.arr = arr
        self.n = len(layers)

    def outputs(self, pid, obs_u8):
        obs_u8 = np.ascontiguousarray(obs_u8, np.uint8)
        n = obs_u8.shape[0]
        out = np.zeros((n, self.arr[pid].n_out), np.float64)
        lib().orc_policy_outputs(C.byref(self.arr[pid]), _ptr(obs_u8), n, _ptr(out))
        return out


def sample(z, legal, u):
    z = np.ascontiguousarray(z, np.float64)
    legal = np.ascontiguousarray(legal, np.uint8)
    a = C.c_int32()
    lp = C.c_double()
    mg = C.c_double()
    lib().orc_sample(_ptr(z), _ptr(legal), len(z), float(u), C.byref(a), C.byref(lp), C.byref(mg))
    return a.value, lp.value, mg.value


def gae(r, v, d, v_last, gamma, lam):
    r = np.ascontiguousarray(r, np.float32)
    v = np.ascontiguousarray(v, np.float32)
    d = np.ascontiguousarray(d, np.uint8)
    v_last = np.ascontiguousarray(v_last, np.float32)
    T, N = r.shape
    adv = np.zeros((T, N), np.float64)
    tgt = np.zeros((T, N), np.float64)
    lib().orc_gae(_ptr(r), _ptr(v), _ptr(d), _ptr(v_last), N, T, gamma, lam, _ptr(adv), _ptr(tgt))
    return adv, tgt


def new_states(n):
    return np.zeros((n, STATE_BYTES), np.uint8)


def reset_all(d, seed, n, step=0):
    st = new_states(n)
    rc = lib().orc_reset_all(C.byref(d), seed, n, step, _ptr(st))
    assert rc == 0, rc
    return st


def reset_envs(d, seed, ids, step=0):
    ids = np.ascontiguousarray(ids, np.int64)
    st = new_states(len(ids))
    rc = lib().orc_reset_envs(C.byref(d), seed, _ptr(ids), len(ids), step, _ptr(st))
    assert rc == 0, rc
    return st


def step_forced(d, seed, step, states, actions):
    n = states.shape[0]
    od = obs_dim(d)
    actions = np.ascontiguousarray(actions, np.uint8)
    rew2 = np.zeros((n, 2), np.float32)
    team = np.zeros(n, np.float32)
    dones = np.zeros(n, np.uint8)
    obs2 = np.zeros((n, 2, od), np.uint8)
    rc = lib().orc_step_forced(C.byref(d), seed, n, step, _ptr(states), _ptr(actions),
                               _ptr(rew2), _ptr(team), _ptr(dones), _ptr(obs2))
    return rc, rew2, team, dones, obs2


def rollout(d, pols: Policies, seed, states, step0, T, ego_id, pool, forced=None, n_threads=1,
            env_ids=None, ep_step=None, resample=False):
    """PPO collection.  Returns a dict of numpy arrays; states are updated in place.
    env_ids: global env index of each state row (default 0..N-1).  ep_step: uint32 [N]
    step at which each env's episode began, updated in place at auto-resets; resample:
    per-episode teammates (needs ep_step)."""
    N = states.shape[0]
    if env_ids is not None:
        env_ids = np.ascontiguousarray(env_ids, np.int64)
        assert env_ids.shape == (N,)
    od = obs_dim(d)
    K = n_actions(d)
    n_out = pols.arr[ego_id].n_out
    pool = np.ascontiguousarray(pool, np.int32)
    out = dict(
        teammate=np.zeros(N, np.int32), obs=np.zeros((T, N, od), np.uint8),
        obs_tm=np.zeros((T, N, od), np.uint8), actions=np.zeros((T, N, 2), np.uint8),
        own_actions=np.zeros((T, N, 2), np.uint8), margin=np.zeros((T, N, 2), np.float64),
        logits=np.zeros((T, N, n_out), np.float64), logp=np.zeros((T, N), np.float64),
        values=np.zeros((T, N), np.float64), rewards=np.zeros((T, N), np.float32),
        dones=np.zeros((T, N), np.uint8), last_value=np.zeros(N, np.float64),
        logp_tm=np.zeros((T, N), np.float64), values_tm=np.zeros((T, N), np.float64),
        last_value_tm=np.zeros(N, np.float64), teammates_t=np.zeros((T, N), np.int32))
    if ep_step is not None:
        assert ep_step.dtype == np.uint32 and ep_step.shape == (N,) and ep_step.flags.c_contiguous
    if forced is not None:
        forced = np.ascontiguousarray(forced, np.uint8)
        assert forced.shape == (T, N, 2)
    io = RolloutIO(seed=seed, n_envs=N, step0=step0, T=T, ego_id=ego_id, pool=_ptr(pool),
                   pool_size=len(pool), forced=_ptr(forced), env_ids=_ptr(env_ids),
                   states=_ptr(states), resample=int(resample), ep_step=_ptr(ep_step),
                   n_threads=n_threads, **{k: _ptr(v) for k, v in out.items()})
    rc = lib().orc_rollout(C.byref(d), pols.arr, pols.n, C.byref(io))
    out["rc"] = rc
    return out


def xplay(d, pols: Policies, seed, step0, ego_ids, tm_ids, P, max_steps, forced=None,
          n_threads=1, record=True, env_ids=None, logit_stride=0):
    """Cross-play.  env_ids: run only these global env indices (rows of the outputs).
    logit_stride > 0: also the acting seats' policy outputs, [max_steps][rows][2][stride]
    (NaN where a seat did not act)."""
    ego_ids = np.ascontiguousarray(ego_ids, np.int32)
    tm_ids = np.ascontiguousarray(tm_ids, np.int32)
    N = len(ego_ids) * len(tm_ids) * P
    if env_ids is not None:
        env_ids = np.ascontiguousarray(env_ids, np.int64)
        N = len(env_ids)
    out = dict(returns=np.zeros(N, np.float32), steps=np.zeros(N, np.int32),
               matrix=np.zeros((len(ego_ids), len(tm_ids)), np.float32))
    if record:
        out.update(actions=np.zeros((max_steps, N, 2), np.uint8),
                   own_actions=np.zeros((max_steps, N, 2), np.uint8),
                   margin=np.zeros((max_steps, N, 2), np.float64))
    if logit_stride:
        out["logits"] = np.full((max_steps, N, 2, logit_stride), np.nan)
    if forced is not None:
        forced = np.ascontiguousarray(forced, np.uint8)
    io = XplayIO(seed=seed, step0=step0, ego_ids=_ptr(ego_ids), n_ego=len(ego_ids),
                 tm_ids=_ptr(tm_ids), n_tm=len(tm_ids), envs_per_pair=P, max_steps=max_steps,
                 forced=_ptr(forced), env_ids=_ptr(env_ids),
                 n_sel=0 if env_ids is None else len(env_ids), n_threads=n_threads,
                 logit_stride=logit_stride, **{k: _ptr(v) for k, v in out.items()})
    rc = lib().orc_xplay(C.byref(d), pols.arr, pols.n, C.byref(io))
    out["rc"] = rc
    return out


def xp_stats(xp, upper=None):
    """Cross-play matrix consumers (App. B upper bounds, Sec. 3 J_AHT, App. A regret and
    BRDiv objective) of an fp32 [n_ego][n_tm] matrix; ``upper`` is the prior bound per
    teammate (default -inf).  Returns fp64 arrays (``brdiv`` None unless square)."""
    xp = np.ascontiguousarray(xp, np.float32)
    ne, nt = xp.shape
    up = np.full(nt, -np.inf) if upper is None else np.array(upper, np.float64)
    out = dict(norm=np.zeros((ne, nt)), regret=np.zeros((ne, nt)), j_aht=np.zeros(ne),
               j_norm=np.zeros(ne), max_regret=np.zeros(ne), worst=np.zeros(ne, np.int32))
    bd = np.zeros(1)
    lib().orc_xp_stats(_ptr(xp), ne, nt, _ptr(up), _ptr(out["norm"]), _ptr(out["regret"]),
                       _ptr(out["j_aht"]), _ptr(out["j_norm"]), _ptr(out["max_regret"]),
                       _ptr(out["worst"]), _ptr(bd) if ne == nt else None)
    out["upper"] = up
    out["brdiv"] = float(bd[0]) if ne == nt else None
    return out


# ---------------------------------------------------------------------------------
# PPO ego update (ppo_oracle.cpp)
# ---------------------------------------------------------------------------------
PPO_DEFAULTS = dict(epochs=4, minibatches=4, lr=2.5e-4, clip_eps=0.2, vf_coef=0.5, ent_coef=0.01,
                    max_grad_norm=0.5, adam_b1=0.9, adam_b2=0.999, adam_eps=1e-5, seed=0,
                    epoch0=0, round_bf16=1)


def ppo_hp(**kw):
    d = dict(PPO_DEFAULTS)
    d.update(kw)
    return PpoHp(**d)


def ppo_net(obs_dim, h0, h1, n_act):
    return PpoNet(obs_dim, h0, h1, n_act)


def ppo_n_params(net):
    return int(lib().orc_ppo_n_params(C.byref(net)))


def flat_params(layers):
    """[(W1, b1), (W2, b2), (W3, b3)] -> one fp64 vector in the oracle's order."""
    return np.concatenate([np.asarray(a, np.float64).ravel() for wb in layers for a in wb])


def unflat_params(net, p):
    D, H0, H1, O = net.obs_dim, net.h0, net.h1, net.n_act + 1
    sizes = [(H0, D), (H0,), (H1, H0), (H1,), (O, H1), (O,)]
    out, i = [], 0
    for sh in sizes:
        n = int(np.prod(sh))
        out.append(np.asarray(p[i:i + n]).reshape(sh))
        i += n
    return [(out[0], out[1]), (out[2], out[3]), (out[4], out[5])]


class PpoBatchNp:
    """Flattened (time-major) trajectory arrays, kept alive for the C structure."""

    def __init__(self, obs, actions, logp, values, advantages, targets):
        D = obs.shape[-1]
        self.obs = np.ascontiguousarray(obs, np.uint8).reshape(-1, D)
        self.actions = np.ascontiguousarray(actions, np.uint8).ravel()
        self.logp = np.ascontiguousarray(logp, np.float32).ravel()
        self.values = np.ascontiguousarray(values, np.float32).ravel()
        self.advantages = np.ascontiguousarray(advantages, np.float32).ravel()
        self.targets = np.ascontiguousarray(targets, np.float32).ravel()
        self.S = self.actions.size
        self.c = PpoBatch(*(_ptr(a) for a in (self.obs, self.actions, self.logp, self.values,
                                               self.advantages, self.targets)))


def perm_index(seed, epoch, S, x):
    return int(lib().orc_perm_index(seed, epoch, S, x))


def perm(seed, epoch, S):
    return np.array([perm_index(seed, epoch, S, x) for x in range(S)], np.int64)


def bf16_round(w):
    return float(lib().orc_bf16_round(float(w)))


def ppo_grad(net, params, batch: PpoBatchNp, idx, hp, n_threads=1):
    params = np.ascontiguousarray(params, np.float64)
    idx = np.ascontiguousarray(idx, np.int64)
    grad = np.zeros(ppo_n_params(net))
    stats = np.zeros(6)
    lib().orc_ppo_grad(C.byref(net), _ptr(params), C.byref(batch.c), _ptr(idx), len(idx),
                       C.byref(hp), _ptr(grad), _ptr(stats), n_threads)
    return grad, stats


def adam_step(params, m, v, t, grad, hp):
    """In place on params, m, v, grad (fp64 arrays); returns the new step count."""
    tt = C.c_int64(t)
    lib().orc_adam_step(len(params), _ptr(params), _ptr(m), _ptr(v), C.byref(tt), _ptr(grad),
                        C.byref(hp))
    return tt.value


def ppo_update(net, params, m, v, t, batch: PpoBatchNp, hp, n_threads=1):
    """In place on params, m, v (fp64); returns (t, stats [E*M][6])."""
    tt = C.c_int64(t)
    stats = np.zeros((hp.epochs * hp.minibatches, 6))
    lib().orc_ppo_update(C.byref(net), _ptr(params), _ptr(m), _ptr(v), C.byref(tt),
                         C.byref(batch.c), batch.S, C.byref(hp), _ptr(stats), n_threads)
    return tt.value, stats


def lbf_heuristic(d, state, seat, k):
    return int(lib().orc_lbf_heuristic(C.byref(d), C.byref(state), seat, k))


# ---- S5 recurrent actor-critic (s5_oracle.cpp) ------------------------------------------
class S5Net(C.Structure):
    _fields_ = [("obs_dim", C.c_int32), ("n_actions", C.c_int32), ("H", C.c_int32),
                ("P", C.c_int32), ("F", C.c_int32),
                ("We1", _P), ("be1", _P), ("We2", _P), ("be2", _P),
                ("lam_re", _P), ("lam_im", _P), ("log_dt", _P),
                ("B_re", _P), ("B_im", _P), ("C_re", _P), ("C_im", _P), ("Dv", _P),
                ("Wa", _P * 4), ("ba", _P * 4), ("Wc", _P * 4), ("bc", _P * 4)]


S5_KEYS = ("We1", "be1", "We2", "be2", "lam_re", "lam_im", "log_dt", "B_re", "B_im",
           "C_re", "C_im", "Dv")


class S5:
    """fp64 copies of an S5 actor-critic's parameters (a dict of arrays: the S5_KEYS and
    lists Wa, ba, Wc, bc of four arrays each) and the oracle's entry points."""

    def __init__(self, params):
        self.p = {k: np.ascontiguousarray(np.asarray(params[k], np.float64)) for k in S5_KEYS}
        for k in ("Wa", "ba", "Wc", "bc"):
            self.p[k] = [np.ascontiguousarray(np.asarray(a, np.float64)) for a in params[k]]
        H, K = self.p["We1"].shape
        self.H, self.K = H, K
        self.P = self.p["lam_re"].shape[0]
        self.F = self.p["Wa"][0].shape[0]
        self.A = self.p["Wa"][3].shape[0]
        net = S5Net(obs_dim=K, n_actions=self.A, H=H, P=self.P, F=self.F)
        for k in S5_KEYS:
            setattr(net, k, _ptr(self.p[k]))
        for k in ("Wa", "ba", "Wc", "bc"):
            arr = (_P * 4)(*[_ptr(a) for a in self.p[k]])
            setattr(net, k, arr)
        self.net = net
        L = lib()
        if not getattr(L, "_s5_typed", False):
            L.orc_s5_encode.argtypes = [C.POINTER(S5Net), _P, _P]
            L.orc_s5_ssm_step.argtypes = [C.POINTER(S5Net), _P, C.c_int32, _P, _P]
            L.orc_s5_heads.argtypes = [C.POINTER(S5Net), _P, _P, _P, _P]
            L.orc_s5_step.argtypes = [C.POINTER(S5Net), _P, _P, _P, C.c_int64, _P, _P, _P, C.c_int32]
            L._s5_typed = True

    def encode(self, obs):
        obs = np.ascontiguousarray(obs, np.uint8)
        u = np.zeros(self.H)
        lib().orc_s5_encode(C.byref(self.net), _ptr(obs), _ptr(u))
        return u

    def ssm_step(self, u, reset, state):
        u = np.ascontiguousarray(u, np.float64)
        y = np.zeros(self.H)
        lib().orc_s5_ssm_step(C.byref(self.net), _ptr(u), int(reset), _ptr(state), _ptr(y))
        return y

    def heads(self, v, legal=None):
        v = np.ascontiguousarray(v, np.float64)
        logits, value = np.zeros(self.A), np.zeros(1)
        legal = None if legal is None else np.ascontiguousarray(legal, np.uint8)
        lib().orc_s5_heads(C.byref(self.net), _ptr(v), _ptr(legal), _ptr(logits), _ptr(value))
        return logits, float(value[0])

    def step(self, obs, reset, state, legal=None, n_threads=8):
        """One step for n envs; state [n][2P] (float64) is updated in place."""
        obs = np.ascontiguousarray(obs, np.uint8)
        reset = np.ascontiguousarray(reset, np.uint8)
        n = obs.shape[0]
        assert state.dtype == np.float64 and state.shape == (n, 2 * self.P) and state.flags.c_contiguous
        legal = None if legal is None else np.ascontiguousarray(legal, np.uint8)
        logits, values = np.zeros((n, self.A)), np.zeros(n)
        lib().orc_s5_step(C.byref(self.net), _ptr(obs), _ptr(reset), _ptr(legal), n, _ptr(state),
                          _ptr(logits), _ptr(values), n_threads)
        return logits, values
