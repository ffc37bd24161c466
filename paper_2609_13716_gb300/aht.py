"""Python binding of libaht.so (include/aht.h): argument marshalling only.

Every step of the rollout path runs in the CUDA kernels behind the C ABI; this module
converts torch tensors to device pointers, checks shapes and dtypes, and raises
``AhtError`` for a non-OK status.  There is no CPU fallback: if the library has not
been built (``paper_2609_13716_gb300.build.build()``), importing the functions raises.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import torch

from . import build as _build

AHT_OK, AHT_EINVAL, AHT_ENOMEM, AHT_ECUDA, AHT_ETIMEOUT, AHT_EDEVICE = range(6)
AHT_LBF, AHT_OVERCOOKED, AHT_HANABI, AHT_MINI_HANABI = range(4)
AHT_FP32, AHT_BF16 = 0, 1

EXPORTED = ["aht_create", "aht_destroy", "aht_reset", "aht_rollout", "aht_xplay_matrix",
            "aht_gae", "aht_step_forced", "aht_policy_forward", "aht_get_state",
            "aht_set_state", "aht_step_counter", "aht_sync", "aht_last_error",
            "aht_status_string", "aht_set_policy", "aht_set_timing", "aht_get_timing",
            "aht_xplay_matrix_static", "aht_debug_tanh", "aht_debug_expire_wait",
            "aht_xp_stats", "aht_learner_create", "aht_learner_destroy", "aht_learner_n_params",
            "aht_ppo_update", "aht_ppo_grad", "aht_learner_get", "aht_learner_set",
            "aht_learner_push", "aht_learner_sync", "aht_rollout_ippo", "aht_rollout_resample",
            "aht_s5_create", "aht_s5_destroy", "aht_s5_step", "aht_s5_sync", "aht_traj_copy"]


class AhtError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"aht status {status}: {msg}")
        self.status = status


class EnvDesc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("width", C.c_int32), ("height", C.c_int32),
                ("n_food", C.c_int32), ("max_agent_level", C.c_int32),
                ("episode_len", C.c_int32), ("cook_time", C.c_int32),
                ("soup_reward", C.c_int32)]


class PopDesc(C.Structure):
    _fields_ = [("n_policies", C.c_int32), ("obs_dim", C.c_int32), ("hidden0", C.c_int32),
                ("hidden1", C.c_int32), ("n_actions", C.c_int32),
                ("has_value_head", C.POINTER(C.c_int32)), ("weight_dtype", C.c_int32),
                ("W", C.POINTER(C.c_void_p)), ("b", C.POINTER(C.c_void_p))]


class Traj(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("actions", C.c_void_p), ("tm_actions", C.c_void_p),
                ("logp", C.c_void_p), ("values", C.c_void_p), ("rewards", C.c_void_p),
                ("dones", C.c_void_p), ("advantages", C.c_void_p), ("targets", C.c_void_p),
                ("last_value", C.c_void_p), ("teammate", C.c_void_p), ("gamma", C.c_float),
                ("lambda_", C.c_float)]


class XplayOut(C.Structure):
    _fields_ = [("matrix", C.c_void_p), ("returns", C.c_void_p), ("steps", C.c_void_p),
                ("actions", C.c_void_p)]


class XpStatsOut(C.Structure):
    _fields_ = [("norm", C.c_void_p), ("regret", C.c_void_p), ("j_aht", C.c_void_p),
                ("j_norm", C.c_void_p), ("max_regret", C.c_void_p), ("worst_tm", C.c_void_p),
                ("brdiv", C.c_void_p)]


class PpoConfig(C.Structure):
    _fields_ = [("epochs", C.c_int32), ("minibatches", C.c_int32), ("lr", C.c_float),
                ("clip_eps", C.c_float), ("vf_coef", C.c_float), ("ent_coef", C.c_float),
                ("max_grad_norm", C.c_float), ("adam_b1", C.c_float), ("adam_b2", C.c_float),
                ("adam_eps", C.c_float), ("seed", C.c_uint64)]


PPO_DEFAULTS = dict(epochs=4, minibatches=4, lr=2.5e-4, clip_eps=0.2, vf_coef=0.5, ent_coef=0.01,
                    max_grad_norm=0.5, adam_b1=0.9, adam_b2=0.999, adam_eps=1e-5, seed=0)


class StepOut(C.Structure):
    _fields_ = [("rewards", C.c_void_p), ("team", C.c_void_p), ("dones", C.c_void_p),
                ("obs", C.c_void_p)]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load() -> C.CDLL:
    """Loads libaht.so (built in-tree).  Raises if it is missing: no fallback exists."""
    global _lib
    with _lock:
        if _lib is None:
            path = library_path()
            if not os.path.exists(path):
                raise ImportError(f"libaht.so not built ({path}); run "
                                  "paper_2609_13716_gb300.build.build() first")
            L = C.CDLL(path)
            vp, i32, i64, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64
            L.aht_create.argtypes = [C.POINTER(EnvDesc), C.POINTER(PopDesc), i64, u64, vp, C.POINTER(vp)]
            L.aht_destroy.argtypes = [vp]
            L.aht_destroy.restype = None
            L.aht_reset.argtypes = [vp, u64]
            L.aht_rollout.argtypes = [vp, i32, C.POINTER(i32), i32, i32, C.POINTER(Traj)]
            L.aht_rollout_ippo.argtypes = [vp, i32, i32, i32, C.POINTER(Traj), C.POINTER(Traj)]
            L.aht_s5_create.argtypes = [C.POINTER(S5Params), i64, vp, C.POINTER(vp)]
            L.aht_s5_create.restype = C.c_int
            L.aht_s5_destroy.argtypes = [vp]
            L.aht_s5_destroy.restype = None
            L.aht_s5_step.argtypes = [vp, vp, vp, vp, i64, vp, vp, vp]
            L.aht_s5_step.restype = C.c_int
            L.aht_s5_sync.argtypes = [vp]
            L.aht_s5_sync.restype = C.c_int
            L.aht_rollout_resample.argtypes = [vp, i32, C.POINTER(i32), i32, i32, C.POINTER(Traj), vp]
            L.aht_xplay_matrix.argtypes = [vp, C.POINTER(i32), i32, C.POINTER(i32), i32, i32, i32, C.POINTER(XplayOut)]
            L.aht_gae.argtypes = [vp, vp, vp, vp, i64, i32, C.c_float, C.c_float, vp, vp, vp]
            L.aht_traj_copy.argtypes = [C.POINTER(Traj), C.POINTER(Traj), i64, i32, i32, vp]
            L.aht_xp_stats.argtypes = [vp, i32, i32, vp, C.POINTER(XpStatsOut), vp]
            L.aht_step_forced.argtypes = [vp, vp, C.POINTER(StepOut)]
            L.aht_learner_create.argtypes = [i32, i32, C.POINTER(vp), C.POINTER(vp), C.POINTER(PpoConfig),
                                             vp, C.POINTER(vp)]
            L.aht_learner_destroy.argtypes = [vp]
            L.aht_learner_destroy.restype = None
            L.aht_learner_n_params.argtypes = [vp]
            L.aht_learner_n_params.restype = i64
            L.aht_ppo_update.argtypes = [vp, C.POINTER(Traj), i64, i32, vp]
            L.aht_ppo_grad.argtypes = [vp, C.POINTER(Traj), i64, i32, i32, i32, vp, vp]
            L.aht_learner_get.argtypes = [vp, vp, vp, vp, C.POINTER(i64), C.POINTER(i64)]
            L.aht_learner_set.argtypes = [vp, vp, vp, vp, i64, i64]
            L.aht_learner_push.argtypes = [vp, vp, i32]
            L.aht_learner_sync.argtypes = [vp]
            L.aht_policy_forward.argtypes = [vp, i32, vp, i64, vp]
            L.aht_get_state.argtypes = [vp, vp, C.POINTER(C.c_size_t)]
            L.aht_set_state.argtypes = [vp, vp, C.c_size_t]
            L.aht_set_policy.argtypes = [vp, i32, C.POINTER(vp), C.POINTER(vp), i32, i32]
            L.aht_set_timing.argtypes = [vp, i32]
            L.aht_get_timing.argtypes = [vp, C.POINTER(C.c_double), C.POINTER(i64)]
            L.aht_debug_fail_alloc.argtypes = [i64]
            L.aht_debug_fail_alloc.restype = C.c_int
            L.aht_debug_live_allocs.argtypes = []
            L.aht_debug_live_allocs.restype = i64
            L.aht_debug_expire_at.argtypes = [vp, i32, i64]
            L.aht_debug_expire_at.restype = C.c_int
            L.aht_debug_logits.argtypes = [vp, vp, i64]
            L.aht_debug_logits.restype = C.c_int
            L.aht_debug_obs_words.argtypes = [vp, i32, vp]
            L.aht_debug_obs_words.restype = C.c_int
            L.aht_step_counter.argtypes = [vp]
            L.aht_step_counter.restype = i64
            L.aht_sync.argtypes = [vp]
            L.aht_last_error.argtypes = []
            L.aht_last_error.restype = C.c_char_p
            L.aht_status_string.argtypes = [C.c_int]
            L.aht_status_string.restype = C.c_char_p
            for f in ("aht_learner_create", "aht_ppo_update", "aht_ppo_grad", "aht_learner_get",
                      "aht_learner_set", "aht_learner_push", "aht_learner_sync"):
                getattr(L, f).restype = C.c_int
            for f in ("aht_create", "aht_reset", "aht_rollout", "aht_rollout_ippo", "aht_rollout_resample",
                      "aht_xplay_matrix",
                      "aht_gae", "aht_xp_stats",
                      "aht_step_forced", "aht_policy_forward", "aht_get_state", "aht_set_state",
                      "aht_sync", "aht_set_policy", "aht_set_timing", "aht_get_timing"):
                getattr(L, f).restype = C.c_int
            _lib = L
    return _lib


def _check(status):
    if status != AHT_OK:
        raise AhtError(status, load().aht_last_error().decode())


def _ptr(t, dtype=None, shape=None, name="tensor"):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


class Context:
    """Owns an aht_ctx handle (aht_destroy on close / garbage collection)."""

    def __init__(self, handle, env, n_envs, obs_dim, n_actions, stream):
        self.handle = handle
        self.env = env
        self.n_envs = n_envs
        self.obs_dim = obs_dim
        self.n_actions = n_actions
        self.stream = stream

    def close(self):
        if self.handle:
            load().aht_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def aht_create(env, population, n_envs, seed, has_value_head=None, weight_dtype=AHT_BF16,
               stream=None) -> Context:
    """env: workloads.EnvSpec; population: per policy [(W1, b1), (W2, b2), (W3, b3)] torch
    tensors (CUDA or CPU, fp32 or bf16 matching weight_dtype), row-major [out][in]."""
    L = load()
    dt = torch.float32 if weight_dtype == AHT_FP32 else torch.bfloat16
    keep, Ws, bs = [], [], []
    for pol in population:
        for W, b in pol:
            W = W.to(dt).contiguous()
            b = b.to(dt).contiguous()
            keep += [W, b]
            Ws.append(W.data_ptr())
            bs.append(b.data_ptr())
    n = len(population)
    hv = (C.c_int32 * n)(*(has_value_head or [0] * n))
    Warr = (C.c_void_p * len(Ws))(*Ws)
    barr = (C.c_void_p * len(bs))(*bs)
    h0 = population[0][0][0].shape[0]
    h1 = population[0][1][0].shape[0]
    pop = PopDesc(n, env.obs_dim, h0, h1, env.n_actions, hv, weight_dtype, Warr, barr)
    desc = EnvDesc(*env.astuple())
    handle = C.c_void_p()
    s = _stream(stream)
    _check(L.aht_create(C.byref(desc), C.byref(pop), n_envs, seed, s, C.byref(handle)))
    del keep
    return Context(handle, env, n_envs, env.obs_dim, env.n_actions, s)


def aht_reset(ctx: Context, seed: int):
    _check(load().aht_reset(ctx.handle, seed))


def traj_buffers(ctx: Context, T: int, device="cuda", obs=True):
    """Allocates (with torch) the caller-owned trajectory tensors of aht_rollout."""
    N = ctx.n_envs
    z = lambda shape, dt: torch.empty(shape, dtype=dt, device=device)
    return dict(obs=z((T, N, ctx.obs_dim), torch.uint8) if obs else None,
                actions=z((T, N), torch.uint8), tm_actions=z((T, N), torch.uint8),
                logp=z((T, N), torch.float32), values=z((T, N), torch.float32),
                rewards=z((T, N), torch.float32), dones=z((T, N), torch.uint8),
                advantages=z((T, N), torch.float32), targets=z((T, N), torch.float32),
                last_value=z((N,), torch.float32), teammate=z((N,), torch.int32))


def _traj(ctx: Context, T, traj: dict, gamma, lam):
    N = ctx.n_envs
    f32, u8 = torch.float32, torch.uint8
    g = traj.get
    return Traj(_ptr(g("obs"), u8, (T, N, ctx.obs_dim), "obs"),
             _ptr(g("actions"), u8, (T, N), "actions"),
             _ptr(g("tm_actions"), u8, (T, N), "tm_actions"),
             _ptr(g("logp"), f32, (T, N), "logp"), _ptr(g("values"), f32, (T, N), "values"),
             _ptr(g("rewards"), f32, (T, N), "rewards"), _ptr(g("dones"), u8, (T, N), "dones"),
             _ptr(g("advantages"), f32, (T, N), "advantages"),
             _ptr(g("targets"), f32, (T, N), "targets"),
             _ptr(g("last_value"), f32, (N,), "last_value"),
             _ptr(g("teammate"), torch.int32, (N,), "teammate"), gamma, lam)


def aht_rollout(ctx: Context, ego_id, pool, T, traj: dict, gamma=0.99, lam=0.95):
    t = _traj(ctx, T, traj, gamma, lam)
    pool = list(pool)
    parr = (C.c_int32 * len(pool))(*pool)
    _check(load().aht_rollout(ctx.handle, ego_id, parr, len(pool), T, C.byref(t)))


def aht_rollout_resample(ctx: Context, ego_id, pool, T, traj: dict, teammates=None,
                         gamma=0.99, lam=0.95):
    """PPO collection with a fresh teammate per episode; teammates: int32 [T][N] or None."""
    t = _traj(ctx, T, traj, gamma, lam)
    pool = list(pool)
    parr = (C.c_int32 * len(pool))(*pool)
    tm = _ptr(teammates, torch.int32, (T, ctx.n_envs), "teammates")
    _check(load().aht_rollout_resample(ctx.handle, ego_id, parr, len(pool), T, C.byref(t), tm))


def aht_rollout_ippo(ctx: Context, policy0, policy1, T, traj0: dict, traj1: dict,
                     gamma=0.99, lam=0.95):
    """IPPO collection: traj0 gets seat 0's (policy0) trajectory, traj1 seat 1's."""
    t0 = _traj(ctx, T, traj0, gamma, lam)
    t1 = _traj(ctx, T, traj1, gamma, lam)
    _check(load().aht_rollout_ippo(ctx.handle, policy0, policy1, T, C.byref(t0), C.byref(t1)))


def aht_xplay_matrix(ctx: Context, ego_ids, tm_ids, envs_per_pair, max_steps, matrix,
                     returns=None, steps=None, actions=None):
    ne, nt, P = len(ego_ids), len(tm_ids), envs_per_pair
    out = XplayOut(_ptr(matrix, torch.float32, (ne, nt), "matrix"),
                   _ptr(returns, torch.float32, (ne, nt, P), "returns"),
                   _ptr(steps, torch.int32, (ne, nt, P), "steps"),
                   _ptr(actions, torch.uint8, (max_steps, ne * nt * P, 2), "actions"))
    ea = (C.c_int32 * ne)(*ego_ids)
    ta = (C.c_int32 * nt)(*tm_ids)
    _check(load().aht_xplay_matrix(ctx.handle, ea, ne, ta, nt, P, max_steps, C.byref(out)))


def aht_xplay_matrix_static(ctx: Context, ego_ids, tm_ids, envs_per_pair, max_steps, matrix):
    """aht_xplay_matrix with its per-env return scratch in the library's static device
    array instead of the context's memory (see include/aht.h)."""
    L = load()
    L.aht_xplay_matrix_static.argtypes = [C.c_void_p, C.POINTER(C.c_int32), C.c_int32,
                                          C.POINTER(C.c_int32), C.c_int32, C.c_int32,
                                          C.c_int32, C.c_void_p]
    L.aht_xplay_matrix_static.restype = C.c_int
    ne, nt = len(ego_ids), len(tm_ids)
    ea = (C.c_int32 * ne)(*ego_ids)
    ta = (C.c_int32 * nt)(*tm_ids)
    _check(L.aht_xplay_matrix_static(ctx.handle, ea, ne, ta, nt, envs_per_pair, max_steps,
                                     _ptr(matrix, torch.float32, (ne, nt), "matrix")))


def aht_debug_tanh(x, y, stream=None):
    """The tensor-core epilogue's tanh applied elementwise (test hook)."""
    L = load()
    L.aht_debug_tanh.argtypes = [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]
    L.aht_debug_tanh.restype = C.c_int
    n = x.numel()
    _check(L.aht_debug_tanh(_ptr(x, torch.float32, None, "x"), _ptr(y, torch.float32, (n,), "y"),
                            n, _stream(stream)))


def aht_gae(rewards, values, dones, v_last, gamma, lam, advantages, targets=None, stream=None):
    T, N = rewards.shape
    f32 = torch.float32
    _check(load().aht_gae(_ptr(rewards, f32, (T, N), "rewards"), _ptr(values, f32, (T, N), "values"),
                          _ptr(dones, torch.uint8, (T, N), "dones"), _ptr(v_last, f32, (N,), "v_last"),
                          N, T, gamma, lam, _ptr(advantages, f32, (T, N), "advantages"),
                          _ptr(targets, f32, (T, N), "targets"), _stream(stream)))


def _ptr_pinned_or_cuda(t, dtype, shape, name):
    """A CUDA tensor, or a pinned host tensor (the trajectory copy's host side)."""
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not (t.is_cuda or t.is_pinned()):
        raise TypeError(f"{name} must be a CUDA tensor or a pinned host tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t.data_ptr()


def aht_traj_copy(src: dict, dst: dict, n_envs: int, T: int, obs_dim: int, stream=None):
    """Copies every trajectory field present in both ``src`` and ``dst`` (dicts as from
    traj_buffers; CUDA or pinned host tensors), enqueued on ``stream``."""
    f32, u8 = torch.float32, torch.uint8
    shapes = dict(obs=((T, n_envs, obs_dim), u8), actions=((T, n_envs), u8), tm_actions=((T, n_envs), u8),
                  logp=((T, n_envs), f32), values=((T, n_envs), f32), rewards=((T, n_envs), f32),
                  dones=((T, n_envs), u8), advantages=((T, n_envs), f32), targets=((T, n_envs), f32),
                  last_value=((n_envs,), f32), teammate=((n_envs,), torch.int32))

    def side(d):
        return Traj(*[_ptr_pinned_or_cuda(d.get(k), dt, sh, k) for k, (sh, dt) in shapes.items()], 0.0, 0.0)

    a, b = side(src), side(dst)
    _check(load().aht_traj_copy(C.byref(a), C.byref(b), n_envs, T, obs_dim, _stream(stream)))


def aht_xp_stats(xp, upper, norm=None, regret=None, j_aht=None, j_norm=None, max_regret=None,
                 worst_tm=None, brdiv=None, stream=None):
    """Cross-play matrix consumers on the device: ``upper`` (f32 [n_tm]) is refined in
    place; the other outputs are optional preallocated CUDA tensors."""
    ne, nt = xp.shape
    f32 = torch.float32
    out = XpStatsOut(_ptr(norm, f32, (ne, nt), "norm"), _ptr(regret, f32, (ne, nt), "regret"),
                     _ptr(j_aht, f32, (ne,), "j_aht"), _ptr(j_norm, f32, (ne,), "j_norm"),
                     _ptr(max_regret, f32, (ne,), "max_regret"),
                     _ptr(worst_tm, torch.int32, (ne,), "worst_tm"), _ptr(brdiv, f32, (1,), "brdiv"))
    _check(load().aht_xp_stats(_ptr(xp, f32, (ne, nt), "xp"), ne, nt, _ptr(upper, f32, (nt,), "upper"),
                               C.byref(out), _stream(stream)))


def aht_step_forced(ctx: Context, actions, rewards=None, team=None, dones=None, obs=None):
    N = ctx.n_envs
    out = StepOut(_ptr(rewards, torch.float32, (N, 2), "rewards"),
                  _ptr(team, torch.float32, (N,), "team"), _ptr(dones, torch.uint8, (N,), "dones"),
                  _ptr(obs, torch.uint8, (N, 2, ctx.obs_dim), "obs"))
    _check(load().aht_step_forced(ctx.handle, _ptr(actions, torch.uint8, (N, 2), "actions"),
                                  C.byref(out)))


def aht_policy_forward(ctx: Context, policy, obs, out):
    n = obs.shape[0]
    _check(load().aht_policy_forward(ctx.handle, policy,
                                     _ptr(obs, torch.uint8, (n, ctx.obs_dim), "obs"), n,
                                     _ptr(out, torch.float32, (n, ctx.n_actions + 1), "out")))


def aht_get_state(ctx: Context) -> bytes:
    L = load()
    n = C.c_size_t(0)
    _check(L.aht_get_state(ctx.handle, None, C.byref(n)))
    buf = C.create_string_buffer(n.value)
    _check(L.aht_get_state(ctx.handle, buf, C.byref(n)))
    return buf.raw[:n.value]


def aht_set_state(ctx: Context, state: bytes):
    buf = C.create_string_buffer(state, len(state))
    _check(load().aht_set_state(ctx.handle, buf, len(state)))


def aht_set_policy(ctx: Context, policy, layers, has_value_head=0, weight_dtype=AHT_BF16):
    """layers: [(W1, b1), (W2, b2), (W3, b3)] tensors (pinned/pageable host or CUDA)."""
    dt = torch.float32 if weight_dtype == AHT_FP32 else torch.bfloat16
    for W, b in layers:
        if W.dtype != dt or b.dtype != dt or not W.is_contiguous() or not b.is_contiguous():
            raise TypeError(f"weights must be contiguous {dt}")
    Ws = (C.c_void_p * 3)(*[W.data_ptr() for W, _ in layers])
    bs = (C.c_void_p * 3)(*[b.data_ptr() for _, b in layers])
    _check(load().aht_set_policy(ctx.handle, policy, Ws, bs, weight_dtype, has_value_head))


def aht_set_timing(ctx: Context, enable: bool):
    _check(load().aht_set_timing(ctx.handle, int(enable)))


def aht_get_timing(ctx: Context):
    """(summed kernel milliseconds, number of timed launches) since the previous call."""
    ms = C.c_double(0)
    n = C.c_int64(0)
    _check(load().aht_get_timing(ctx.handle, C.byref(ms), C.byref(n)))
    return ms.value, n.value


def aht_step_counter(ctx: Context) -> int:
    return load().aht_step_counter(ctx.handle)


def aht_sync(ctx: Context):
    _check(load().aht_sync(ctx.handle))


AHT_DEBUG_STRIDE = 32


def aht_debug_fail_alloc(n: int):
    """Allocation-failure hook: the n-th allocation aht_create makes from now on fails
    (n <= 0: off)."""
    _check(load().aht_debug_fail_alloc(n))


def aht_debug_live_allocs() -> int:
    """Device and pinned blocks that contexts hold now."""
    return int(load().aht_debug_live_allocs())


def aht_debug_expire_at(ctx: Context, step: int, limit_ns: int):
    """Failure-detection hook: the next tensor-core call waits in vain (bounded by
    limit_ns) at its step ``step`` and aborts; ``step < 0`` clears the hook."""
    _check(load().aht_debug_expire_at(ctx.handle, step, limit_ns))


def aht_debug_logits(ctx: Context, buf):
    """Parity hook: while ``buf`` (a contiguous CUDA fp32 tensor) is set, the tensor-core
    kernels of the next calls write every policy output vector into it, at
    [step][row][seat][AHT_DEBUG_STRIDE]; ``None`` turns it off."""
    if buf is None:
        _check(load().aht_debug_logits(ctx.handle, None, 0))
        return
    _check(load().aht_debug_logits(ctx.handle, _ptr(buf, torch.float32, name="buf"), buf.numel()))


def aht_debug_obs_words(ctx: Context, seat: int, out):
    """Parity hook: the streamed cross-play kernel's observation rows of seat ``seat`` of
    every env's current state, into ``out`` (CUDA int32 [n_envs][(obs_dim + 32) // 32],
    the bits of uint32 words); Overcooked, Hanabi and Mini Hanabi contexts."""
    words = (ctx.obs_dim + 32) // 32
    _check(load().aht_debug_obs_words(ctx.handle, seat, _ptr(out, torch.int32, (ctx.n_envs, words), "out")))


def aht_debug_expire_wait(ctx: Context, limit_ns: int):
    """Failure-detection hook: a kernel's bounded wait on a barrier nothing arrives on
    expires after limit_ns; the next aht_sync raises AhtError with AHT_ETIMEOUT."""
    L = load()
    L.aht_debug_expire_wait.argtypes = [C.c_void_p, C.c_int64]
    L.aht_debug_expire_wait.restype = C.c_int
    _check(L.aht_debug_expire_wait(ctx.handle, int(limit_ns)))


# ---------------------------------------------------------------------------------
# PPO learner
# ---------------------------------------------------------------------------------
class Learner:
    """Owns an aht_learner handle (aht_learner_destroy on close / garbage collection)."""

    def __init__(self, handle, obs_dim, n_actions, n_params, cfg):
        self.handle = handle
        self.obs_dim, self.n_actions, self.n_params, self.cfg = obs_dim, n_actions, n_params, cfg

    def close(self):
        if self.handle:
            load().aht_learner_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def aht_learner_create(obs_dim, n_actions, layers, stream=None, **cfg) -> Learner:
    """layers: [(W1, b1), (W2, b2), (W3, b3)] torch tensors (converted to fp32)."""
    L = load()
    c = dict(PPO_DEFAULTS)
    c.update(cfg)
    conf = PpoConfig(**c)
    keep = [(W.float().contiguous(), b.float().contiguous()) for W, b in layers]
    Ws = (C.c_void_p * 3)(*[W.data_ptr() for W, _ in keep])
    bs = (C.c_void_p * 3)(*[b.data_ptr() for _, b in keep])
    h = C.c_void_p()
    _check(L.aht_learner_create(obs_dim, n_actions, Ws, bs, C.byref(conf), _stream(stream), C.byref(h)))
    del keep
    return Learner(h, obs_dim, n_actions, int(L.aht_learner_n_params(h)), c)


def _ppo_traj(learner, traj, T, N):
    f32, u8 = torch.float32, torch.uint8
    g = traj.get
    return Traj(_ptr(g("obs"), u8, (T, N, learner.obs_dim), "obs"), _ptr(g("actions"), u8, (T, N), "actions"),
                None, _ptr(g("logp"), f32, (T, N), "logp"), _ptr(g("values"), f32, (T, N), "values"),
                None, None, _ptr(g("advantages"), f32, (T, N), "advantages"),
                _ptr(g("targets"), f32, (T, N), "targets"), None, None, 0.0, 0.0)


def aht_ppo_update(learner: Learner, traj: dict, stats=None):
    T, N = traj["actions"].shape
    t = _ppo_traj(learner, traj, T, N)
    E, M = learner.cfg["epochs"], learner.cfg["minibatches"]
    _check(load().aht_ppo_update(learner.handle, C.byref(t), N, T,
                                 _ptr(stats, torch.float32, (E * M, 6), "stats")))


def aht_ppo_grad(learner: Learner, traj: dict, epoch, minibatch, grad, stats=None):
    T, N = traj["actions"].shape
    t = _ppo_traj(learner, traj, T, N)
    _check(load().aht_ppo_grad(learner.handle, C.byref(t), N, T, epoch, minibatch,
                               _ptr(grad, torch.float32, (learner.n_params,), "grad"),
                               _ptr(stats, torch.float32, (6,), "stats")))


def aht_learner_get(learner: Learner, params=None, adam_m=None, adam_v=None):
    n = learner.n_params
    t, u = C.c_int64(0), C.c_int64(0)
    _check(load().aht_learner_get(learner.handle, _ptr(params, torch.float32, (n,), "params"),
                                  _ptr(adam_m, torch.float32, (n,), "adam_m"),
                                  _ptr(adam_v, torch.float32, (n,), "adam_v"), C.byref(t), C.byref(u)))
    return t.value, u.value


def aht_learner_set(learner: Learner, params, adam_m=None, adam_v=None, t=0, updates=0):
    n = learner.n_params
    _check(load().aht_learner_set(learner.handle, _ptr(params, torch.float32, (n,), "params"),
                                  _ptr(adam_m, torch.float32, (n,), "adam_m"),
                                  _ptr(adam_v, torch.float32, (n,), "adam_v"), t, updates))


def aht_learner_push(learner: Learner, ctx: Context, policy):
    _check(load().aht_learner_push(learner.handle, ctx.handle, policy))


def aht_learner_sync(learner: Learner):
    _check(load().aht_learner_sync(learner.handle))


# ---- S5 recurrent actor-critic ----------------------------------------------------------
_FP = C.POINTER(C.c_float)


class S5Params(C.Structure):
    _fields_ = [("obs_dim", C.c_int32), ("n_actions", C.c_int32), ("H", C.c_int32),
                ("P", C.c_int32), ("F", C.c_int32),
                ("We1", _FP), ("be1", _FP), ("We2", _FP), ("be2", _FP),
                ("lam_re", _FP), ("lam_im", _FP), ("log_dt", _FP),
                ("B_re", _FP), ("B_im", _FP), ("C_re", _FP), ("C_im", _FP), ("D", _FP),
                ("Wa", _FP * 4), ("ba", _FP * 4), ("Wc", _FP * 4), ("bc", _FP * 4)]


class S5Policy:
    """Owns an aht_s5 handle (aht_s5_destroy on close / garbage collection)."""

    def __init__(self, handle, obs_dim, n_actions, P):
        self.handle, self.obs_dim, self.n_actions, self.P = handle, obs_dim, n_actions, P

    def close(self):
        if self.handle:
            load().aht_s5_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def aht_s5_create(params, max_envs, stream=None) -> S5Policy:
    """params: dict of host float32 numpy arrays (the keys of workloads.s5_params)."""
    import numpy as np
    keep = {}

    def fp(a):
        a = np.ascontiguousarray(a, np.float32)
        keep[id(a)] = a
        return a.ctypes.data_as(_FP)

    H, K = params["We1"].shape
    P = params["lam_re"].shape[0]
    F = params["Wa"][0].shape[0]
    A = params["Wa"][3].shape[0]
    sp = S5Params(obs_dim=K, n_actions=A, H=H, P=P, F=F)
    for k, f in (("We1", "We1"), ("be1", "be1"), ("We2", "We2"), ("be2", "be2"), ("lam_re", "lam_re"),
                 ("lam_im", "lam_im"), ("log_dt", "log_dt"), ("B_re", "B_re"), ("B_im", "B_im"),
                 ("C_re", "C_re"), ("C_im", "C_im"), ("Dv", "D")):
        setattr(sp, f, fp(params[k]))
    for k in ("Wa", "ba", "Wc", "bc"):
        setattr(sp, k, (_FP * 4)(*[fp(a) for a in params[k]]))
    h = C.c_void_p()
    st = None if stream is None else C.c_void_p(stream.cuda_stream)
    _check(load().aht_s5_create(C.byref(sp), int(max_envs), st, C.byref(h)))
    return S5Policy(h, K, A, P)


def aht_s5_step(pol: S5Policy, obs, reset, state, logits, values, legal=None):
    n = obs.shape[0]
    u8, f32 = torch.uint8, torch.float32
    _check(load().aht_s5_step(pol.handle, _ptr(obs, u8, (n, pol.obs_dim), "obs"),
                              _ptr(reset, u8, (n,), "reset"),
                              _ptr(legal, u8, (n, pol.n_actions), "legal"), n,
                              _ptr(state, f32, (n, 2 * pol.P), "state"),
                              _ptr(logits, f32, (n, pol.n_actions), "logits"),
                              _ptr(values, f32, (n,), "values")))


def aht_s5_sync(pol: S5Policy):
    _check(load().aht_s5_sync(pol.handle))
