"""Benchmark: PPO rollout collection of 16384 LBF 7x7 envs x 128 steps with GAE, on GB300.

One step = one aht_rollout call over the whole batch: per env-step, the ego (196-128-128-7
actor-critic) and a teammate drawn from a 32-policy population (196-128-128-6) run,
actions are sampled, the env steps, the trajectory (obs, actions, logp, values, rewards,
dones) streams to HBM, then V_T and GAE advantages/targets are formed.  Weights are
synthetic (N(0, 0.1), bf16); there are no trained policies in this build.

Prints ONE JSON line (rank 0).  `--impl reference` times the CPU oracle instead, on a
bounded sample of the same workload.  Multi-GPU (torchrun): every rank runs its own
independent batch (weak scaling, no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "lbf7x7_ppo_16384x128"
METRIC = "env-steps/sec (LBF 7x7 PPO rollout collection + GAE, ego vs 32-policy population)"
UNIT = "env-steps/s"
L2_BYTES = 129 * 2 ** 20


def mlp_flops(dims):
    return 2 * sum(dims[i] * dims[i + 1] for i in range(len(dims) - 1))


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-xplay", action="store_true")
    p.add_argument("--no-ppo", action="store_true")
    # PPO update only, on the trajectory of one rollout (profiling; not a bench line)
    p.add_argument("--ppo-only", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    # profiling of a smaller case of the same kernel (not a bench line)
    p.add_argument("--n-envs", type=int, default=None)
    p.add_argument("--T", type=int, default=None)
    p.add_argument("--no-e2e", action="store_true")
    # cross-play only (profiling of the cross-play kernels; not a bench line)
    p.add_argument("--xplay-only", default=None,
                   help="comma-separated cross-play workloads to time without the rollout")
    return p.parse_args()


def max_over_ranks(value, device):
    """The largest value over all ranks (timings only: the data path has no collective)."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t)


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


# ------------------------------------------------------------------------------------
# CPU oracle timing (the reported baseline; never tuned)
# ------------------------------------------------------------------------------------
def oracle_rate(wl, target_s, seed_offset=0):
    """Times the oracle's free-running PPO collection on a bounded env sample sized for
    about target_s seconds on all host cores.  Returns (env-steps/s, threads, sample)."""
    import numpy as np
    import oracle as O
    from paper_2609_13716_gb300 import workloads as W
    threads = os.cpu_count() or 1
    d = O.env_desc(*wl.env.astuple())
    pols = O.Policies(W.population(wl))
    n = max(threads, 2 * threads)
    st = O.reset_all(d, wl.env_seed, n)
    t0 = time.perf_counter()
    O.rollout(d, pols, wl.env_seed, st, 0, wl.T, wl.ego_id, list(wl.pool), n_threads=threads)
    rate = n * wl.T / (time.perf_counter() - t0)
    n = int(min(wl.n_envs, max(threads, rate * target_s / wl.T)))
    n = max(threads, n // threads * threads)
    ids = np.arange(n, dtype=np.int64) * (wl.n_envs // n)   # spread over the batch
    st = O.reset_envs(d, wl.env_seed, ids)
    t0 = time.perf_counter()
    out = O.rollout(d, pols, wl.env_seed, st, 0, wl.T, wl.ego_id, list(wl.pool),
                    n_threads=threads, env_ids=ids)
    adv = O.gae(out["rewards"], out["values"].astype(np.float32), out["dones"],
                out["last_value"].astype(np.float32), wl.gamma, wl.lam)
    dt = time.perf_counter() - t0
    sample = f"{n} of {wl.n_envs} envs x {wl.T} steps (rollout + GAE), free-running fp64 oracle"
    return n * wl.T / dt, threads, sample, dt


def oracle_rate_1thread(wl, target_s):
    """The oracle's free-running PPO collection (rollout + GAE) on one host thread, on a
    bounded env sample sized for about target_s seconds.  Returns (env-steps/s, sample)."""
    import numpy as np
    import oracle as O
    from paper_2609_13716_gb300 import workloads as W
    d = O.env_desc(*wl.env.astuple())
    pols = O.Policies(W.population(wl))
    n = 4
    for _ in range(2):  # the first pilot also pays one-time costs
        t0 = time.perf_counter()
        O.rollout(d, pols, wl.env_seed, O.reset_all(d, wl.env_seed, n), 0, wl.T, wl.ego_id,
                  list(wl.pool), n_threads=1)
        rate = n * wl.T / (time.perf_counter() - t0)
    n = int(min(wl.n_envs, max(4, rate * target_s / wl.T)))
    ids = np.arange(n, dtype=np.int64) * (wl.n_envs // n)
    st = O.reset_envs(d, wl.env_seed, ids)
    t0 = time.perf_counter()
    out = O.rollout(d, pols, wl.env_seed, st, 0, wl.T, wl.ego_id, list(wl.pool), n_threads=1,
                    env_ids=ids)
    O.gae(out["rewards"], out["values"].astype(np.float32), out["dones"],
          out["last_value"].astype(np.float32), wl.gamma, wl.lam)
    dt = time.perf_counter() - t0
    return n * wl.T / dt, f"{n} of {wl.n_envs} envs x {wl.T} steps (rollout + GAE) on 1 thread"


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return
    from paper_2609_13716_gb300 import workloads as W
    wl = W.WORKLOADS[WORKLOAD]
    import oracle as O
    O.build()
    per_step_s = max(2.0, 60.0 / max(1, args.steps + args.warmup))
    for _ in range(args.warmup):
        oracle_rate(wl, 0.5)
    rates, dts = [], []
    sample = ""
    threads = 1
    for _ in range(args.steps):
        r, threads, sample, dt = oracle_rate(wl, per_step_s)
        rates.append(r)
        dts.append(dt)
    value = statistics.median(rates)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 0,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * wl.n_envs * wl.T / value,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "n_envs": wl.n_envs, "T": wl.T, "pool": len(wl.pool)},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": sample + "; each step is such a sample, ms_per_step is "
                                   "scaled to the full batch"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------
# GPU arm
# ------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for name, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# the sources the fused rollout kernel is compiled from
ROLLOUT_SOURCES = ("rollout_tc2.cuh", "rollout_tc.cuh", "tc_common.cuh", "env_lbf.cuh", "aht_common.cuh",
                   "mlp_simt.cuh", "rollout_impl.cuh", "kernels.h", "rollout_lbf.cu", "rollout_lbf2.cu")


def csrc_hash():
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2609_13716_gb300", "csrc")
    for f in ROLLOUT_SOURCES:
        h.update(open(os.path.join(d, f), "rb").read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel):
    """Per-launch DRAM bytes from the committed ncu summary, if it still matches the source."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    want = csrc_hash()
    for ln in open(path):
        kv = dict(x.split("=", 1) for x in ln.split() if "=" in x)
        if kv.get("kernel") == kernel and kv.get("csrc_sha") == want:
            return float(kv["dram_bytes_per_launch"])
    return None


def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    rank, local, world = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2609_13716_gb300 import aht, workloads as W
    from paper_2609_13716_gb300 import build as B
    B.build()
    peaks = {}
    pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(pk):
        peaks = json.load(open(pk))
    bf16_peak = peaks.get("bf16_tflops", 1900.0)
    bf16_sustained = peaks.get("bf16_tflops_sustained", 1700.0)
    hbm_peak = peaks.get("hbm_gbs", 6800.0)
    peak_src = "measured" if peaks else "fallback"

    if args.xplay_only:
        xp = run_xplay(args, aht, W, torch, bf16_peak, args.xplay_only.split(","))
        if rank == 0:
            print(json.dumps({"xplay": xp}), flush=True)
        return
    wl = W.WORKLOADS[WORKLOAD]
    N, T = args.n_envs or wl.n_envs, args.T or wl.T
    pop_np = W.population(wl)
    pop = [[(torch.from_numpy(Wt).to("cuda", torch.bfloat16), torch.from_numpy(b).to("cuda", torch.bfloat16))
            for Wt, b in p] for p in pop_np]
    ctx = aht.aht_create(wl.env, pop, N, wl.env_seed + 7919 * rank,
                         has_value_head=list(wl.value_head), weight_dtype=aht.AHT_BF16)
    traj = aht.traj_buffers(ctx, T)
    scrub = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")   # > L2
    stream = torch.cuda.current_stream()

    def step():
        aht.aht_rollout(ctx, wl.ego_id, wl.pool, T, traj, wl.gamma, wl.lam)

    if args.ppo_only:
        step()
        pu = run_ppo_update(args, aht, wl, pop_np, traj, torch, bf16_peak, stream)
        if rank == 0:
            print(json.dumps({"ppo_update": pu}), flush=True)
        return

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()

    # ---- timed region: K rollouts, L2 scrubbed between them (outside the events) ----
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    stops = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    dev_index = local
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        dev_index = int(vis.split(",")[local])
    aht.aht_get_timing(ctx)
    aht.aht_set_timing(ctx, True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev_index) as clocks:
        time.sleep(0.3)   # let the sampler start before the timed launches
        for k in range(args.steps):
            scrub.fill_(k & 0xFF)
            starts[k].record(stream)
            step()
            stops[k].record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    aht.aht_set_timing(ctx, False)
    kernel_ms, kernel_launches = aht.aht_get_timing(ctx)
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, stops)]
    ms = sum(step_ms) / len(step_ms)
    ms_max = max_over_ranks(ms, "cuda")
    aht.aht_sync(ctx)

    # ---- end to end: ego weights from pinned host memory in, whole trajectory out ------
    # Through the library's API: aht_set_policy uploads the ego's weights, aht_rollout
    # collects, aht_traj_copy downloads.  Two trajectory buffers, as a user would
    # double-buffer: step k's trajectory is copied to pinned host memory on a copy stream
    # while step k + 1 runs on the library's stream.  Every step's upload and download
    # lies inside the timed region, which ends when the last download has landed.
    ego_host = [(W_.to(torch.bfloat16).cpu().pin_memory(), b.to(torch.bfloat16).cpu().pin_memory())
                for W_, b in [(torch.from_numpy(a), torch.from_numpy(c)) for a, c in pop_np[wl.ego_id]]]
    e2e_ms = []
    h2d = sum(W_.numel() * 2 + b.numel() * 2 for W_, b in ego_host)
    d2h = sum(v.numel() * v.element_size() for v in traj.values() if v is not None)
    if not args.no_e2e:
        trajs = [traj, aht.traj_buffers(ctx, T)]
        hosts = [{k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in t.items() if v is not None}
                 for t in trajs]
        copy_stream = torch.cuda.Stream()
        rolled = [torch.cuda.Event(), torch.cuda.Event()]
        copied = [torch.cuda.Event(), torch.cuda.Event()]

        def e2e_step(k):
            b = k % 2
            stream.wait_event(copied[b])            # buffer b's previous download is done
            aht.aht_set_policy(ctx, wl.ego_id, ego_host, 1, aht.AHT_BF16)
            aht.aht_rollout(ctx, wl.ego_id, wl.pool, T, trajs[b], wl.gamma, wl.lam)
            rolled[b].record(stream)
            copy_stream.wait_event(rolled[b])
            aht.aht_traj_copy(trajs[b], hosts[b], N, T, wl.env.obs_dim, copy_stream)
            copied[b].record(copy_stream)

        for k in range(2):
            e2e_step(k)
        torch.cuda.synchronize()
        e2e_s, e2e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e2e_s.record(stream)
        for k in range(args.steps):
            e2e_step(k)
        stream.wait_stream(copy_stream)
        e2e_e.record(stream)
        torch.cuda.synchronize()
        e2e_ms = [e2e_s.elapsed_time(e2e_e) / args.steps]
    aht.aht_sync(ctx)
    e2e_ms_max = max_over_ranks(sum(e2e_ms) / max(1, len(e2e_ms)), "cuda")

    # ---- roofline of the dominant kernel (the fused rollout) ----------------------------
    env_steps = N * T
    ego_dims = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions + 1]
    tm_dims = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions]
    flops_per_env_step = mlp_flops(ego_dims) + mlp_flops(tm_dims)          # 169,216
    flops_launch = env_steps * flops_per_env_step + N * mlp_flops(ego_dims)  # + V_T forward
    bytes_per_env_step = wl.env.obs_dim + 1 + 1 + 4 + 4 + 4 + 1              # obs, a, a_tm, logp, v, r, d
    kern_ms = kernel_ms / max(1, kernel_launches)
    achieved_tflops = flops_launch / (kern_ms * 1e-3) / 1e12
    achieved_gbs = env_steps * bytes_per_env_step / (kern_ms * 1e-3) / 1e9
    traffic = recorded_traffic("ppo2_tc_kernel")

    line = None
    if rank == 0:
        value = world * env_steps / (ms_max * 1e-3)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_max,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic (random-init N(0,0.1) bf16 weights, seeded envs)",
            "config": {"workload": WORKLOAD, "n_envs": N, "T": T, "pool": len(wl.pool),
                       "episode_len": wl.env.episode_len, "weights": "bf16",
                       "l2": "scrubbed: 256 MB write between timed steps (outside the events); "
                             "each step also writes a 449 MB trajectory",
                       "parallelism": f"{world} independent replicas" if world > 1 else "1 GPU"},
            "roofline": {"bound": "tensor", "achieved": achieved_tflops, "peak": bf16_peak,
                         "unit": "TFLOP/s", "frac": achieved_tflops / bf16_peak,
                         "traffic": traffic, "kernel": "ppo2_tc_kernel<EnvLbf, bf16, gathered tiles>",
                         "kernel_ms": kern_ms, "flops_per_launch": flops_launch,
                         "peak_source": f"{peak_src} bf16 burst",
                         "frac_of_sustained": achieved_tflops / bf16_sustained,
                         "hbm": {"achieved_gbs": achieved_gbs, "peak_gbs": hbm_peak,
                                 "frac": achieved_gbs / hbm_peak,
                                 "bytes_per_launch": env_steps * bytes_per_env_step}},
            "e2e": None if not e2e_ms else
                   {"value": world * env_steps / (float(e2e_ms_max) * 1e-3), "unit": UNIT,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": 3 * args.steps,
            "clocks": clocks.summary(),
        }
    if line is not None and not args.n_envs and not args.T:
        line["c0"] = run_c0(aht, W, torch, stream)
        line["ippo"] = run_ippo(aht, W, torch, stream, bf16_peak)
        line["resample"] = run_resample(aht, wl, pop, torch, stream, bf16_peak)
        line["lbf12x12_ppo"] = run_lbf12_ppo(aht, W, torch, stream, bf16_peak)
        line["s5"] = run_s5(aht, W, torch, stream, bf16_peak)
    if not args.no_ppo:
        pu = run_ppo_update(args, aht, wl, pop_np, traj, torch, bf16_peak, stream)
        if line is not None:
            line["ppo_update"] = pu
    if not args.no_xplay:
        xp = run_xplay(args, aht, W, torch, bf16_peak, bf16_sustained=bf16_sustained)
        if line is not None:
            line["xplay"] = xp
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, cores, sample, _ = oracle_rate(wl, args.cpu_seconds)
        v1, sample1 = oracle_rate_1thread(wl, min(4.0, args.cpu_seconds / 3))
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": sample, "value_1_thread": v1, "sample_1_thread": sample1}
    if line is not None:
        print(json.dumps(line), flush=True)
    ctx.close()
    if world > 1:
        dist.destroy_process_group()


def run_c0(aht, W, torch, stream):
    """The smallest configuration (64 LBF 7x7 envs x 50 steps, fp32 64-wide MLPs): too
    small to fill the GPU, so only its latency and env-steps/s are reported."""
    import numpy as np
    wl = W.WORKLOADS["lbf7x7_64x50_fp32"]
    pop = [[(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda()) for Wt, b in p]
           for p in W.population(wl)]
    ctx = aht.aht_create(wl.env, pop, wl.n_envs, wl.env_seed, weight_dtype=aht.AHT_FP32, stream=stream)
    traj = aht.traj_buffers(ctx, wl.T)
    for _ in range(3):
        aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    K = 10
    ev[0].record(stream)
    for _ in range(K):
        aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj)
    ev[1].record(stream)
    torch.cuda.synchronize()
    aht.aht_sync(ctx)
    ms = ev[0].elapsed_time(ev[1]) / K
    ctx.close()
    return {"workload": wl.name, "ms_per_call": ms, "env_steps_per_s": wl.n_envs * wl.T / (ms * 1e-3),
            "bound": "latency (64 envs fill one tile; no roofline target)"}


def run_ippo(aht, W, torch, stream, bf16_peak):
    """IPPO collection (both seats learn): 16384 LBF 7x7 envs x 128 steps, two bf16
    196-128-128-(6+1) policies, both seats' trajectories and GAE.  ms per call from CUDA
    events (L2 scrubbed between calls, outside the events) and the tensor roofline of the
    fused rollout kernel's algorithmic FLOPs (both forwards per env-step, both V_T)."""
    wl = W.WORKLOADS["lbf7x7_ippo_16384x128"]
    pop = [[(torch.from_numpy(Wt).to("cuda", torch.bfloat16), torch.from_numpy(b).to("cuda", torch.bfloat16))
            for Wt, b in p] for p in W.population(wl)]
    ctx = aht.aht_create(wl.env, pop, wl.n_envs, wl.env_seed, has_value_head=list(wl.value_head),
                         weight_dtype=aht.AHT_BF16, stream=stream)
    t0, t1 = aht.traj_buffers(ctx, wl.T), aht.traj_buffers(ctx, wl.T)
    scrub = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")

    def call():
        aht.aht_rollout_ippo(ctx, 0, 1, wl.T, t0, t1, wl.gamma, wl.lam)

    for _ in range(3):
        call()
    torch.cuda.synchronize()
    K = 5
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    aht.aht_get_timing(ctx)
    aht.aht_set_timing(ctx, True)
    for k in range(K):
        scrub.fill_(k & 0xFF)
        ev[k][0].record(stream)
        call()
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    aht.aht_set_timing(ctx, False)
    kernel_ms, launches = aht.aht_get_timing(ctx)
    aht.aht_sync(ctx)
    ctx.close()
    ms = sum(a.elapsed_time(b) for a, b in ev) / K
    kern_ms = kernel_ms / max(1, launches)
    dims = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions + 1]
    flops = (wl.n_envs * wl.T + wl.n_envs) * 2 * mlp_flops(dims)
    achieved = flops / (kern_ms * 1e-3) / 1e12
    return {"workload": wl.name, "ms_per_call": ms, "env_steps_per_s": wl.n_envs * wl.T / (ms * 1e-3),
            "learner_samples_per_s": 2 * wl.n_envs * wl.T / (ms * 1e-3), "kernel_ms": kern_ms,
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": bf16_peak, "unit": "TFLOP/s",
                         "frac": achieved / bf16_peak, "flops_per_launch": flops}}


def run_resample(aht, wl, pop, torch, stream, bf16_peak):
    """The bench workload with a fresh teammate per episode (aht_rollout_resample): one
    fused-rollout launch per step, each grouping its own rows by the envs' current
    teammates (steps after the first start as programmatic dependents of the step
    before), plus the first draw and GAE: T + 2 launches per call.  ms per call from CUDA
    events (L2 scrubbed between calls, outside the events); then a second pass with the
    library's per-launch timing on (its event records between the launches serialise
    them) for the rollout kernels' summed time.  The roofline is taken on the whole call."""
    ctx = aht.aht_create(wl.env, pop, wl.n_envs, wl.env_seed, has_value_head=list(wl.value_head),
                         weight_dtype=aht.AHT_BF16, stream=stream)
    traj = aht.traj_buffers(ctx, wl.T)
    scrub = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")

    def call():
        aht.aht_rollout_resample(ctx, wl.ego_id, wl.pool, wl.T, traj, None, wl.gamma, wl.lam)

    for _ in range(3):
        call()
    torch.cuda.synchronize()
    K = 5
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    for k in range(K):
        scrub.fill_(k & 0xFF)
        ev[k][0].record(stream)
        call()
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    aht.aht_get_timing(ctx)
    aht.aht_set_timing(ctx, True)
    for k in range(K):
        scrub.fill_(k & 0xFF)
        call()
    torch.cuda.synchronize()
    aht.aht_set_timing(ctx, False)
    kernel_ms, launches = aht.aht_get_timing(ctx)
    aht.aht_sync(ctx)
    ctx.close()
    ms = sum(a.elapsed_time(b) for a, b in ev) / K
    rollout_ms = kernel_ms / K           # the T fused-rollout launches of one call
    ego = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions + 1]
    tm = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions]
    flops = wl.n_envs * wl.T * (mlp_flops(ego) + mlp_flops(tm)) + wl.n_envs * mlp_flops(ego)
    achieved = flops / (ms * 1e-3) / 1e12  # the whole call: its rollout launches overlap
    return {"workload": wl.name + "_per_episode_teammates", "ms_per_call": ms,
            "env_steps_per_s": wl.n_envs * wl.T / (ms * 1e-3), "rollout_kernels_ms": rollout_ms,
            "launches_per_call": wl.T + 2,
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": bf16_peak, "unit": "TFLOP/s",
                         "frac": achieved / bf16_peak, "flops_per_call": flops}}


def run_lbf12_ppo(aht, W, torch, stream, bf16_peak):
    """PPO collection on the 12x12 grid: 4096 envs x 128 steps, ego 576-128-128-(6+1) vs
    8 bf16 teammates, on the tensor-core rollout with the sparse first layer.  ms per
    call from CUDA events (L2 scrubbed between calls, outside the events); the roofline
    counts dense-equivalent MLP FLOPs."""
    wl = W.WORKLOADS["lbf12x12_ppo_4096x128"]
    pop = [[(torch.from_numpy(Wt).to("cuda", torch.bfloat16), torch.from_numpy(b).to("cuda", torch.bfloat16))
            for Wt, b in p] for p in W.population(wl)]
    ctx = aht.aht_create(wl.env, pop, wl.n_envs, wl.env_seed, has_value_head=list(wl.value_head),
                         weight_dtype=aht.AHT_BF16, stream=stream)
    traj = aht.traj_buffers(ctx, wl.T)
    scrub = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")
    for _ in range(3):
        aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj, wl.gamma, wl.lam)
    torch.cuda.synchronize()
    K = 5
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    aht.aht_get_timing(ctx)
    aht.aht_set_timing(ctx, True)
    for k in range(K):
        scrub.fill_(k & 0xFF)
        ev[k][0].record(stream)
        aht.aht_rollout(ctx, wl.ego_id, wl.pool, wl.T, traj, wl.gamma, wl.lam)
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    aht.aht_set_timing(ctx, False)
    kernel_ms, launches = aht.aht_get_timing(ctx)
    aht.aht_sync(ctx)
    ctx.close()
    ms = sum(a.elapsed_time(b) for a, b in ev) / K
    kern_ms = kernel_ms / max(1, launches)
    ego = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions + 1]
    tm = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions]
    flops = wl.n_envs * wl.T * (mlp_flops(ego) + mlp_flops(tm)) + wl.n_envs * mlp_flops(ego)
    achieved = flops / (kern_ms * 1e-3) / 1e12
    return {"workload": wl.name, "ms_per_call": ms, "env_steps_per_s": wl.n_envs * wl.T / (ms * 1e-3),
            "kernel_ms": kern_ms,
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": bf16_peak, "unit": "TFLOP/s",
                         "frac": achieved / bf16_peak, "flops_per_launch": flops,
                         "flops_basis": "dense-equivalent MLP FLOPs; the first layer is formed on CUDA "
                                        "cores from the observation's changed features"}}


def run_s5(aht, W, torch, stream, bf16_peak, n=16384, K=10):
    """The recurrent S5 actor-critic step (App. B sizes: model 128, state 128, heads of three
    1024-unit layers) for n LBF 7x7 observations (196 features, 6 actions): encoder, the
    diagonal recurrence with 1 % of envs resetting, both heads, masked logits.  ms per step
    from CUDA events on the policy's stream (L2 scrubbed between steps, outside the events);
    the roofline counts the model's FLOPs once (the GPU runs the split-activation layers
    twice: hi and lo bf16 halves)."""
    obs_dim, A, H, P, F = 196, 6, 128, 128, 1024
    pol = aht.aht_s5_create(W.s5_params(0, obs_dim, A), n, stream=stream)
    g = torch.Generator(device="cuda").manual_seed(3)
    obs = torch.randint(0, 3, (n, obs_dim), dtype=torch.uint8, device="cuda", generator=g)
    reset = (torch.rand(n, device="cuda", generator=g) < 0.01).to(torch.uint8)
    legal = torch.ones(n, A, dtype=torch.uint8, device="cuda")
    state = torch.zeros(n, 2 * P, device="cuda")
    logits = torch.empty(n, A, device="cuda")
    values = torch.empty(n, device="cuda")
    scrub = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    for _ in range(3):
        aht.aht_s5_step(pol, obs, reset, state, logits, values, legal)
    aht.aht_s5_sync(pol)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    with torch.cuda.stream(stream):
        for k in range(K):
            scrub.fill_(k & 0xFF)
            ev[k][0].record(stream)
            aht.aht_s5_step(pol, obs, reset, state, logits, values, legal)
            ev[k][1].record(stream)
    torch.cuda.synchronize()
    pol.close()
    ms = sum(a.elapsed_time(b) for a, b in ev) / K
    dense = mlp_flops([obs_dim, H, H]) + mlp_flops([H, F, F, F, A]) + mlp_flops([H, F, F, F, 1])
    ssm = 2 * (2 * P * H) + 8 * P + 2 * (H * 2 * P)
    flops = n * (dense + ssm)
    achieved = flops / (ms * 1e-3) / 1e12
    return {"workload": f"s5_actor_critic_lbf7x7_{n}", "ms_per_step": ms,
            "env_steps_per_s": n / (ms * 1e-3), "tcgen05_gemm_launches": 7, "own_kernel_launches": 9,
            "library_gemm_launches": 0,
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": bf16_peak, "unit": "TFLOP/s",
                         "frac": achieved / bf16_peak, "flops_per_step": flops,
                         "flops_basis": "model FLOPs of the encoder, SSM and heads, counted once; "
                                        "the split layers execute twice as many"}}


PPO_FLOPS_PER_SAMPLE = 204032   # forward 84,736 + backward 119,296 (dW1, dW2, dh1, dW3, dh2)


def run_ppo_update(args, aht, wl, pop_np, traj, torch, bf16_peak, stream):
    """The PPO ego update (4 epochs x 4 minibatches, Adam) over the trajectory the last
    timed rollout wrote: ms per update, sample-epochs/s and the fraction of the tensor
    roofline of its algorithmic FLOPs; beside it the fp64 oracle's gradient rate on a
    bounded sample of the same trajectory."""
    import numpy as np
    T, N = traj["actions"].shape
    layers = [(torch.from_numpy(np.asarray(Wt, np.float32)), torch.from_numpy(np.asarray(b, np.float32)))
              for Wt, b in pop_np[wl.ego_id]]
    L = aht.aht_learner_create(wl.env.obs_dim, wl.env.n_actions, layers, stream=stream)
    start = [torch.empty(L.n_params, device="cuda") for _ in range(3)]
    aht.aht_learner_get(L, *start)
    for _ in range(2):
        aht.aht_ppo_update(L, traj)
    torch.cuda.synchronize()
    K = max(3, min(args.steps, 10))
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record(stream)
    for _ in range(K):
        aht.aht_ppo_update(L, traj)
    ev[1].record(stream)
    torch.cuda.synchronize()
    aht.aht_learner_sync(L)
    ms = ev[0].elapsed_time(ev[1]) / K
    E, M = L.cfg["epochs"], L.cfg["minibatches"]
    samples = T * N * E
    tflops = samples * PPO_FLOPS_PER_SAMPLE / (ms * 1e-3) / 1e12
    res = {"workload": f"ppo_update_lbf7x7_{N}x{T}_{E}ep_{M}mb", "ms_per_update": ms,
           "sample_epochs_per_s": samples / (ms * 1e-3),
           "gpu_launches_per_update": 2 + 3 * E * M,
           "roofline": {"bound": "tensor", "achieved": tflops, "peak": bf16_peak, "unit": "TFLOP/s",
                        "frac": tflops / bf16_peak, "flops_per_update": samples * PPO_FLOPS_PER_SAMPLE}}
    L.close()
    if not args.no_cpu_baseline:
        import oracle as O
        b = {k: traj[k][:, :1024].contiguous().cpu().numpy() for k in
             ("obs", "actions", "logp", "values", "advantages", "targets")}
        batch = O.PpoBatchNp(**b)
        net = O.ppo_net(wl.env.obs_dim, wl.hidden[0], wl.hidden[1], wl.env.n_actions)
        p0 = O.flat_params([(np.asarray(Wt, np.float64), np.asarray(bb, np.float64)) for Wt, bb in pop_np[wl.ego_id]])
        threads = os.cpu_count() or 1
        n = min(batch.S, 32768)
        idx = np.arange(n, dtype=np.int64)
        t0 = time.perf_counter()
        O.ppo_grad(net, p0, batch, idx, O.ppo_hp(), n_threads=threads)
        dt = time.perf_counter() - t0
        res["cpu_baseline"] = {"value": n / dt, "unit": "sample-epochs/s", "cores": threads, "kind": "oracle",
                               "sample": f"gradient of one {n}-sample minibatch of the same trajectory, fp64"}
    return res


XPLAY_WORKLOADS = ("lbf7x7_xplay_8x16x256", "lbf7x7_xplay_heuristics_8x12x256",
                   "lbf12x12_xplay_8x16x128", "overcooked5x4_xplay_8x8x64", "hanabi_xplay_16x16x32",
                   "minihanabi_xplay_16x16x32")


def run_xplay(args, aht, W, torch, bf16_peak, names=XPLAY_WORKLOADS, bf16_sustained=1717.4):
    """Cross-play matrices: cells/s and active env-steps/s of each cross-play workload, and
    the fraction of the tensor roofline (MLP FLOPs of the env-steps that actually ran, one
    forward per acting agent, at the bf16 peak)."""
    res = {}
    for name in names:
        wl = W.WORKLOADS[name]
        dt = torch.bfloat16 if wl.weight_dtype == W.BF16 else torch.float32
        pop = [[(torch.from_numpy(Wt).to("cuda", dt), torch.from_numpy(b).to("cuda", dt)) for Wt, b in p]
               for p in W.population(wl)]
        n = wl.xplay_envs
        ctx = aht.aht_create(wl.env, pop, n, wl.env_seed,
                             weight_dtype=aht.AHT_BF16 if wl.weight_dtype == W.BF16 else aht.AHT_FP32)
        ne, nt = len(wl.ego_ids), len(wl.tm_ids)
        matrix = torch.empty(ne, nt, device="cuda")
        steps = torch.empty(ne, nt, wl.envs_per_pair, dtype=torch.int32, device="cuda")
        call = lambda: aht.aht_xplay_matrix(ctx, list(wl.ego_ids), list(wl.tm_ids),
                                            wl.envs_per_pair, wl.max_steps, matrix, None, steps)
        for _ in range(3):
            call()
        torch.cuda.synchronize()
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        K = max(3, args.steps)
        s.record()
        for _ in range(K):
            call()
        e.record()
        torch.cuda.synchronize()
        ms = s.elapsed_time(e) / K
        active = int(steps.sum())
        # the matrix's consumers (bounds, normalised returns, regret, J_AHT, BRDiv)
        upper = torch.full((nt,), float("-inf"), device="cuda")
        so = dict(norm=torch.empty(ne, nt, device="cuda"), regret=torch.empty(ne, nt, device="cuda"),
                  j_aht=torch.empty(ne, device="cuda"), j_norm=torch.empty(ne, device="cuda"),
                  max_regret=torch.empty(ne, device="cuda"),
                  worst_tm=torch.empty(ne, dtype=torch.int32, device="cuda"),
                  brdiv=torch.empty(1, device="cuda") if ne == nt else None)
        for _ in range(3):
            aht.aht_xp_stats(matrix, upper, **so)
        torch.cuda.synchronize()
        # one small kernel per call: replay a CUDA graph of 50 calls, so that the host's
        # per-call binding overhead does not leave the device idle between them
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for _ in range(50):
                aht.aht_xp_stats(matrix, upper, **so)
        graph.replay()
        torch.cuda.synchronize()
        s.record()
        graph.replay()
        e.record()
        torch.cuda.synchronize()
        stats_us = s.elapsed_time(e) / 50 * 1e3
        aht.aht_sync(ctx)
        ctx.close()
        dims = [wl.env.obs_dim, *wl.hidden, wl.env.n_actions]
        acting = 1 if wl.env.kind in (W.HANABI, W.MINI_HANABI) else 2   # one actor per turn
        if min(wl.tm_ids) < 0:                              # rule-based teammates: no network
            acting = 1
        flops = active * acting * mlp_flops(dims)
        tflops = flops / (ms * 1e-3) / 1e12
        res[name] = {"cells_per_s": ne * nt / (ms * 1e-3), "ms_per_matrix": ms,
                     "active_env_steps": active, "active_env_steps_per_s": active / (ms * 1e-3),
                     "weights": "bf16" if wl.weight_dtype == W.BF16 else "f32",
                     "roofline": {"bound": "tensor", "achieved": tflops, "peak": bf16_peak,
                                  "unit": "TFLOP/s", "frac": tflops / bf16_peak,
                                  "frac_of_sustained": tflops / bf16_sustained,
                                  "flops_per_matrix": flops},
                     "xp_stats_us": stats_us}
        if wl.env.kind == W.LBF and wl.env.obs_dim > 255:
            # wider than the tensor-memory operand: the first layer adds only the
            # observation's changed features to a per-policy constant (CUDA cores), so
            # these are dense-equivalent FLOPs
            res[name]["roofline"]["flops_basis"] = (
                "dense-equivalent MLP FLOPs; the first layer is formed on CUDA cores from the "
                "observation's changed features, the second on the tensor cores")
    return res


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
