"""Seeded synthetic workloads: env descriptions, population shapes and weights.

This module holds no step of the method's arithmetic.  It describes the five
workloads (grid-world rollouts shaped like the paper's LBF, Overcooked and Hanabi
settings, Sec. 4 Table "JaxAHT Environments") and draws the synthetic policy weights
that both the CUDA path and the CPU oracle consume.  There are no trained weights in
this build: every policy is random-init, W and b ~ N(0, 0.1), drawn from
``numpy.random.Generator(numpy.random.Philox(seed))`` with seed = 1000 * workload index +
policy id, then rounded to bf16 for the bf16 workloads.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

LBF, OVERCOOKED, HANABI, MINI_HANABI = 0, 1, 2, 3
FP32, BF16 = 0, 1


@dataclass(frozen=True)
class EnvSpec:
    kind: int
    width: int = 0
    height: int = 0
    n_food: int = 0
    max_agent_level: int = 0
    episode_len: int = 0
    cook_time: int = 0
    soup_reward: int = 0

    @property
    def obs_dim(self) -> int:
        if self.kind == LBF:
            return self.width * self.height * 4
        if self.kind == OVERCOOKED:
            return 5 * 4 * 26
        if self.kind == MINI_HANABI:
            return 156
        return 660

    @property
    def n_actions(self) -> int:
        return {HANABI: 20, MINI_HANABI: 10}.get(self.kind, 6)

    def astuple(self):
        return (self.kind, self.width, self.height, self.n_food, self.max_agent_level,
                self.episode_len, self.cook_time, self.soup_reward)


@dataclass(frozen=True)
class Workload:
    name: str
    index: int                 # seed family: weights use 1000 * index + policy id
    env: EnvSpec
    hidden: tuple              # (h0, h1)
    weight_dtype: int          # FP32 or BF16
    n_policies: int
    value_head: tuple          # per-policy: 1 if the last layer has a value row
    mode: str                  # "ppo" or "xplay"
    env_seed: int
    # PPO collection
    n_envs: int = 0
    T: int = 0
    ego_id: int = 0
    pool: tuple = ()
    gamma: float = 0.99
    lam: float = 0.95
    # cross-play
    ego_ids: tuple = ()
    tm_ids: tuple = ()
    envs_per_pair: int = 0
    max_steps: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def xplay_envs(self) -> int:
        return len(self.ego_ids) * len(self.tm_ids) * self.envs_per_pair


LBF7 = dict(kind=LBF, width=7, height=7, n_food=3, max_agent_level=3)


def _lbf(ep):
    return EnvSpec(episode_len=ep, **LBF7)


WORKLOADS = {
    # 64 LBF 7x7 envs, 50-step episodes, one ego + one teammate fp32 196-64-64-6 MLP.
    "lbf7x7_64x50_fp32": Workload(
        name="lbf7x7_64x50_fp32", index=0, env=_lbf(50), hidden=(64, 64), weight_dtype=FP32,
        n_policies=2, value_head=(0, 0), mode="ppo", env_seed=0, n_envs=64, T=50, ego_id=0,
        pool=(1,), ego_ids=(0,), tm_ids=(1,), envs_per_pair=64, max_steps=50),
    # LBF 7x7 cross-play: 8 egos x 16 teammates, 256 envs per pair, 128-step episodes.
    "lbf7x7_xplay_8x16x256": Workload(
        name="lbf7x7_xplay_8x16x256", index=1, env=_lbf(128), hidden=(64, 64),
        weight_dtype=FP32, n_policies=24, value_head=(0,) * 24, mode="xplay", env_seed=1,
        ego_ids=tuple(range(8)), tm_ids=tuple(range(8, 24)), envs_per_pair=256,
        max_steps=128),
    # The same 8 egos (same seeds) against the 12 rule-based LBF teammates (ids -1..-12).
    "lbf7x7_xplay_heuristics_8x12x256": Workload(
        name="lbf7x7_xplay_heuristics_8x12x256", index=1, env=_lbf(128), hidden=(64, 64),
        weight_dtype=FP32, n_policies=8, value_head=(0,) * 8, mode="xplay", env_seed=1,
        ego_ids=tuple(range(8)), tm_ids=tuple(-1 - k for k in range(12)), envs_per_pair=256,
        max_steps=128),
    # LBF 12x12 (the paper's second LBF grid, Sec. 4 Table "JaxAHT Environments"): 8 egos
    # x 16 teammates, 128 envs per pair, 128-step episodes, fp32 576-64-64-6 MLPs.
    "lbf12x12_xplay_8x16x128": Workload(
        name="lbf12x12_xplay_8x16x128", index=6, env=EnvSpec(kind=LBF, width=12, height=12, n_food=3,
                                                           max_agent_level=3, episode_len=128),
        hidden=(64, 64), weight_dtype=FP32, n_policies=24, value_head=(0,) * 24, mode="xplay",
        env_seed=6, ego_ids=tuple(range(8)), tm_ids=tuple(range(8, 24)), envs_per_pair=128,
        max_steps=128),
    # LBF 12x12 PPO collection: 4096 envs x 128 steps, ego 576-128-128-(6+1) vs 8 teammates, bf16.
    "lbf12x12_ppo_4096x128": Workload(
        name="lbf12x12_ppo_4096x128", index=7, env=EnvSpec(kind=LBF, width=12, height=12, n_food=3,
                                                         max_agent_level=3, episode_len=50),
        hidden=(128, 128), weight_dtype=BF16, n_policies=9, value_head=(1,) + (0,) * 8, mode="ppo",
        env_seed=7, n_envs=4096, T=128, ego_id=0, pool=tuple(range(1, 9))),
    # LBF 7x7 PPO collection: 16384 envs x 128 steps, ego actor-critic 196-128-128-(6+1),
    # teammates drawn uniformly from a 32-policy population, bf16 weights.
    "lbf7x7_ppo_16384x128": Workload(
        name="lbf7x7_ppo_16384x128", index=2, env=_lbf(50), hidden=(128, 128),
        weight_dtype=BF16, n_policies=33, value_head=(1,) + (0,) * 32, mode="ppo",
        env_seed=2, n_envs=16384, T=128, ego_id=0, pool=tuple(range(1, 33))),
    # IPPO collection (both seats learn): two bf16 196-128-128-(6+1) policies with value
    # rows, 16384 envs x 128 steps, seat 0 = policy 0, seat 1 = policy 1 in every env.
    "lbf7x7_ippo_16384x128": Workload(
        name="lbf7x7_ippo_16384x128", index=9, env=_lbf(50), hidden=(128, 128),
        weight_dtype=BF16, n_policies=2, value_head=(1, 1), mode="ppo",
        env_seed=9, n_envs=16384, T=128, ego_id=0, pool=(1,)),
    # 5x4 kitchen: 8 x 8 pairs, 64 envs per pair (4096 envs), 400-step episodes,
    # 520-256-256-6 bf16 MLPs.
    "overcooked5x4_xplay_8x8x64": Workload(
        name="overcooked5x4_xplay_8x8x64", index=3,
        env=EnvSpec(kind=OVERCOOKED, width=5, height=4, episode_len=400, cook_time=20,
                    soup_reward=20),
        hidden=(256, 256), weight_dtype=BF16, n_policies=16, value_head=(0,) * 16,
        mode="xplay", env_seed=3, ego_ids=tuple(range(8)), tm_ids=tuple(range(8, 16)),
        envs_per_pair=64, max_steps=400),
    # 2-player Hanabi: 16 x 16 pairs, 32 envs per pair (8192 envs), to termination,
    # 660-512-512-20 bf16 MLPs with illegal-action masking.
    "hanabi_xplay_16x16x32": Workload(
        name="hanabi_xplay_16x16x32", index=4, env=EnvSpec(kind=HANABI, episode_len=0),
        hidden=(512, 512), weight_dtype=BF16, n_policies=32, value_head=(0,) * 32,
        mode="xplay", env_seed=4, ego_ids=tuple(range(16)), tm_ids=tuple(range(16, 32)),
        envs_per_pair=32, max_steps=100),
    # 2-player Mini Hanabi (3 colours x 3 ranks): 16 x 16 pairs, 32 envs per pair, to
    # termination, 156-256-256-10 bf16 MLPs with illegal-action masking.
    "minihanabi_xplay_16x16x32": Workload(
        name="minihanabi_xplay_16x16x32", index=8, env=EnvSpec(kind=MINI_HANABI, episode_len=0),
        hidden=(256, 256), weight_dtype=BF16, n_policies=32, value_head=(0,) * 32,
        mode="xplay", env_seed=8, ego_ids=tuple(range(16)), tm_ids=tuple(range(16, 32)),
        envs_per_pair=32, max_steps=100),
}


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Nearest-even rounding of fp32 values to bf16, returned as exact fp32 values."""
    a = np.ascontiguousarray(a, np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    rounded = ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) << 16
    return rounded.astype(np.uint32).view(np.float32)


def policy_weights(wl: Workload, pid: int, scale: float = 0.1):
    """[(W1, b1), (W2, b2), (W3, b3)] as fp32 arrays, row-major [out][in].

    The last layer has n_actions rows, plus one value row when wl.value_head[pid].
    bf16 workloads return fp32 arrays holding bf16-representable values.
    """
    rng = np.random.Generator(np.random.Philox(1000 * wl.index + pid))
    dims = [wl.env.obs_dim, wl.hidden[0], wl.hidden[1],
            wl.env.n_actions + (1 if wl.value_head[pid] else 0)]
    layers = []
    for i in range(3):
        W = (rng.standard_normal((dims[i + 1], dims[i])) * scale).astype(np.float32)
        b = (rng.standard_normal(dims[i + 1]) * scale).astype(np.float32)
        if wl.weight_dtype == BF16:
            W, b = round_to_bf16(W), round_to_bf16(b)
        layers.append((W, b))
    return layers


def population(wl: Workload, scale: float = 0.1):
    return [policy_weights(wl, p, scale) for p in range(wl.n_policies)]


def random_actions(seed: int, shape, n_actions: int) -> np.ndarray:
    """Uniform forced actions for env-rule parity tests."""
    rng = np.random.Generator(np.random.Philox(seed))
    return rng.integers(0, n_actions, size=shape, dtype=np.uint8)


def xp_matrix(seed: int, n_ego: int, n_tm: int, scale: float = 1.0,
              quantum: float = 0.0) -> np.ndarray:
    """Synthetic cross-play return matrix [n_ego][n_tm] (f32) shaped like the paper's (App.
    B figures): entries uniform in [0, 0.6) * scale, the matched pairs of the leading
    diagonal 0.4 * scale higher.  ``quantum`` > 0 rounds every entry to a multiple of it
    (integer game scores averaged over a fixed number of episodes), which makes ties."""
    rng = np.random.Generator(np.random.Philox(seed))
    m = rng.uniform(0.0, 0.6, (n_ego, n_tm))
    k = min(n_ego, n_tm)
    m[np.arange(k), np.arange(k)] += 0.4
    m *= scale
    if quantum > 0:
        m = np.round(m / quantum) * quantum
    return m.astype(np.float32)


def s5_params(seed: int, obs_dim: int, n_actions: int, H: int = 128, P: int = 128, F: int = 1024):
    """Synthetic parameters of the recurrent S5 actor-critic (random init, no training).

    Dense layers (encoder and both heads) are N(0, 1/fan_in) and rounded to bf16 (the
    GPU runs them as bf16 GEMMs); the SSM's continuous-time modes have decay rates
    exp(U(log 0.05, 0)) (lambda_re = -rate), frequencies U(-pi, pi) and log steps
    U(log 1e-3, log 1e-1); B and C are complex N(0, 1/(2 fan_in)), D is N(0, 1); all fp32.
    Returns a dict of float32 arrays: We1 be1 We2 be2 lam_re lam_im log_dt B_re B_im C_re
    C_im Dv, and lists Wa ba Wc bc of the heads' four layers."""
    rng = np.random.Generator(np.random.Philox(90000 + seed))
    f32 = lambda a: np.asarray(a, np.float32)

    def dense(rows, cols):
        W = round_to_bf16(f32(rng.standard_normal((rows, cols)) / np.sqrt(cols)))
        b = round_to_bf16(f32(rng.standard_normal(rows) * 0.1))
        return W, b

    p = {}
    p["We1"], p["be1"] = dense(H, obs_dim)
    p["We2"], p["be2"] = dense(H, H)
    p["lam_re"] = f32(-np.exp(rng.uniform(np.log(0.05), 0.0, P)))
    p["lam_im"] = f32(rng.uniform(-np.pi, np.pi, P))
    p["log_dt"] = f32(rng.uniform(np.log(1e-3), np.log(1e-1), P))
    p["B_re"] = f32(rng.standard_normal((P, H)) / np.sqrt(2 * H))
    p["B_im"] = f32(rng.standard_normal((P, H)) / np.sqrt(2 * H))
    p["C_re"] = f32(rng.standard_normal((H, P)) / np.sqrt(2 * P))
    p["C_im"] = f32(rng.standard_normal((H, P)) / np.sqrt(2 * P))
    p["Dv"] = f32(rng.standard_normal(H))
    for head, out in (("a", n_actions), ("c", 1)):
        dims = [H, F, F, F, out]
        Ws, bs = [], []
        for i in range(4):
            W, b = dense(dims[i + 1], dims[i])
            Ws.append(W)
            bs.append(b)
        p["W" + head], p["b" + head] = Ws, bs
    return p
