#!/usr/bin/env python
"""Throughput of the batched AUV rollout step on GB300 (env-steps/s).

One bench step = one PPO collection pass of the 65,536-env workload: a
T = 128-step rollout (observation, policy network, Gaussian action,
thruster allocation, 4 physics substeps, reward, done, auto-reset) writing
the full SoA trajectory (obs, act, logp, rew, done), followed by the value
network over the stored observations.  Prints one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun (N > 1) each rank steps its own shard of envs (env ids offset
by rank, weak scaling, no data-path collective); rank 0 prints.
`--impl reference` times the CPU oracle (test infrastructure) on a bounded
sample of the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2512_13359_gb300 import workloads as W  # noqa: E402

L2_BYTES = 129 * 1024 * 1024


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="ppo_65536")
    ap.add_argument("--n-envs", type=int, default=None)
    ap.add_argument("--rollout-steps", type=int, default=None)
    ap.add_argument("--mlp", default=None, choices=[None, "fp32", "bf16", "tf32"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the fp32 workloads' rollouts of the default line")
    ap.add_argument("--no-replay", action="store_true",
                    help="skip the physics-only measurement of the default line")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--replay", action="store_true",
                    help="physics only: action replay (env_step_actions), FP32 roofline")
    ap.add_argument("--ppo", action="store_true",
                    help="time the PPO update (ppo_update) on one rollout's trajectory")
    ap.add_argument("--ppo-precision", default="bf16", choices=["fp32", "tf32", "bf16"])
    ap.add_argument("--minibatch", type=int, default=65536)
    ap.add_argument("--epochs", type=int, default=4)
    ap.add_argument("--n-minibatches", type=int, default=None,
                    help="minibatches per epoch (default: all rows / minibatch)")
    ap.add_argument("--adjoint", action="store_true",
                    help="time the control-step adjoint (env_adjoint) over an action window")
    ap.add_argument("--window", type=int, default=32, help="adjoint / SHAC window length")
    ap.add_argument("--shac", action="store_true",
                    help="time SHAC's closed-loop window (env_shac_window)")
    ap.add_argument("--rbuf", action="store_true",
                    help="time replay-buffer insert (a rollout's trajectory) and sampling")
    ap.add_argument("--invalloc", action="store_true",
                    help="time the inverse thruster allocation over the envs")
    ap.add_argument("--gae", action="store_true",
                    help="advantage estimation (env_gae) over one rollout, HBM roofline")
    ap.add_argument("--probes", action="store_true",
                    help="roofline probes: FFMA chain, tanh.approx.f32 and ex2.approx.f32 chains, "
                         "cuBLAS tf32/bf16 GEMM, tcgen05 MMA cost per instruction by N")
    ap.add_argument("--sweep", action="store_true",
                    help="batch-size sweep 1,024 .. 1,048,576 envs x 256 steps (one line per size)")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sm_max_mhz": 2070.0}, "fallback"


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# algorithmic work per env-step
# ---------------------------------------------------------------------------
def mlp_flops(in_dim, hidden, out):
    return 2 * (in_dim * hidden + hidden * hidden + hidden * out)


def traj_bytes_per_env_step(w, keys):
    b = dict(obs=4 * W.obs_dim(w), act=4 * W.act_dim(w), logp=4, value=4, rew=4, done=1)
    return sum(b[k] for k in keys)


def dyn_flops_per_env_step(w):
    return PAPER_DYN_FLOPS_PER_ENV_STEP if W.is_paper(w) else DYN_FLOPS_PER_ENV_STEP


# ---------------------------------------------------------------------------
# reference arm / CPU baseline: the oracle on a bounded sample
# ---------------------------------------------------------------------------
def oracle_api(w):
    """(model, batch class, reset, rollout) of the oracle for w's model."""
    from oracle import oracle as O
    if W.is_paper(w):
        return O.paper_model(w), O.PaperBatch, O.paper_reset, O.paper_rollout
    return O.model(w), O.Batch, O.reset, O.rollout


def oracle_sample_rate(w, T, target_s, max_envs=4096):
    """Time the CPU oracle on a sample of envs over T steps; env-steps/s on
    one host core.  The sample grows until it takes about target_s."""
    m, Batch, reset, rollout = oracle_api(w)
    pw = W.policy_weights(w)
    vw = W.value_weights(w) if w["has_value"] else None
    n = 2
    while True:
        b = Batch(np.arange(n))
        reset(m, b)
        t0 = time.perf_counter()
        rollout(m, b, pw, vw, 0, T)
        dt = time.perf_counter() - t0
        if dt >= target_s or n >= max_envs:
            return n * T / dt, n, dt
        n = min(max_envs, max(n * 2, int(n * target_s / max(dt, 1e-3)) + 1))


def _oracle_worker(w, jobs, results):
    """Worker process of OraclePool: runs the oracle rollout of env ids
    [lo, lo + n) for each job (lo, n, T) and reports its seconds."""
    m, Batch, reset, rollout = oracle_api(w)
    pw = W.policy_weights(w)
    vw = W.value_weights(w) if w["has_value"] else None
    while True:
        job = jobs.get()
        if job is None:
            return
        lo, n, T = job
        b = Batch(np.arange(lo, lo + n))
        reset(m, b)
        t0 = time.perf_counter()
        rollout(m, b, pw, vw, 0, T)
        results.put(time.perf_counter() - t0)


class OraclePool:
    """The unchanged oracle on every host core: one spawned process per core
    (spawn, so that no process inherits a CUDA context), each on its own
    range of env ids.  run(n, T) rolls n envs per process over T steps and
    returns the wall seconds of the whole batch."""

    def __init__(self, w, cores=None):
        import multiprocessing as mp
        from oracle import oracle as O
        O.build()
        self.cores = cores or len(os.sched_getaffinity(0))
        ctx = mp.get_context("spawn")
        self.jobs, self.results = ctx.Queue(), ctx.Queue()
        self.procs = [ctx.Process(target=_oracle_worker, args=(w, self.jobs, self.results),
                                  daemon=True) for _ in range(self.cores)]
        for p in self.procs:
            p.start()
        self.run(1, 1)      # every worker has loaded the oracle

    def run(self, n, T):
        t0 = time.perf_counter()
        for k in range(self.cores):
            self.jobs.put((k * n, n, T))
        for _ in range(self.cores):
            self.results.get()
        return time.perf_counter() - t0

    def close(self):
        for _ in self.procs:
            self.jobs.put(None)
        for p in self.procs:
            p.join(timeout=10)


def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from oracle import oracle as O
    O.build()
    T = w["steps"]
    # size one bench step so that K + W steps take about a minute in total;
    # each step rolls n envs on every host core (disjoint env-id ranges)
    rate, _, _ = oracle_sample_rate(w, T, 2.0)
    per_step_s = max(1.0, 60.0 / max(1, args.steps + args.warmup))
    n = max(1, int(rate * per_step_s / T))
    pool = OraclePool(w)
    try:
        times = [pool.run(n, T) for _ in range(args.warmup + args.steps)][args.warmup:]
    finally:
        pool.close()
    sec = sum(times) / len(times)
    value = pool.cores * n * T / sec
    sample = (f"{n} envs x {T} steps of {w['name']} per process per step, {pool.cores} "
              f"processes on disjoint env ids (0..{pool.cores * n - 1})")
    line = {
        "impl": "reference", "metric": "env-steps/s (physics+policy+reward)", "value": value,
        "unit": "env-steps/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w["name"], "n_envs": w["n_envs"], "rollout_steps": T,
                   "substeps": w["substeps"], "mlp": w["mlp"], "sample_envs": n},
        "cpu_baseline": {"value": value, "unit": "env-steps/s", "cores": pool.cores,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "env-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def measure_replay(w, steps, warmup, clocks_on=True, device=0):
    """Dynamics step alone (allocation, substeps, reward, done, reset) over
    a fixed action sequence through env_step_actions: the FP32-bound part of
    the rollout.  Returns (ms per launch, env-steps, achieved TFLOP/s, FP32
    peak TFLOP/s, peak source, clock record)."""
    import torch
    from paper_2512_13359_gb300 import auvenv
    n, T = int(w["n_envs"]), int(w["steps"])
    env = auvenv.Env(w)
    env.reset()
    act = torch.from_numpy(W.replay_actions(1, T, n, act=W.act_dim(w))).cuda()
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        env.step_actions(act, rew, done)
    torch.cuda.synchronize()
    clocks = ClockSampler(device) if clocks_on else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ms = []
    for _ in range(steps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        env.step_actions(act, rew, done)
        e1.record(stream)
        ms.append((e0, e1))
    torch.cuda.synchronize()
    clock_info = clocks.stop() if clocks else None
    step_ms = sum(a.elapsed_time(b) for a, b in ms) / len(ms)
    if env.status().code != 0:
        raise RuntimeError("device status after replay")
    env.close()
    peaks, _ = load_peaks()
    sm_mhz = (clock_info or {}).get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
    n_sm = torch.cuda.get_device_properties(device).multi_processor_count
    fp32_peak = 2 * 128 * n_sm * sm_mhz * 1e6 / 1e12
    achieved = n * T * dyn_flops_per_env_step(w) / (step_ms * 1e-3) / 1e12
    src = f"FP32 pipe 2*128*{n_sm} SMs*{sm_mhz:.0f} MHz (derived)"
    return step_ms, n * T, achieved, fp32_peak, src, clock_info


# The three fp32 workloads: 64 envs x 200 steps with the
# 18-64-64-8 network on CUDA cores (hidden 64 is far below a tensor-core
# tile), and 4,096 / 16,384 envs x 1,000 steps with the 18-256-256-8 network
# on the tensor cores in tf32 (kind::tf32); trajectories of rewards and dones.
CONFIG_LINES = (("tiny_64", "fp32"), ("fp32_4096", "tf32"), ("dr_16384", "tf32"))


def dyn_flops(w):
    """Physics flops per env-step for the workload's substep count (the
    counts behind DYN_FLOPS_PER_ENV_STEP)."""
    if W.is_paper(w):
        return PAPER_DYN_FLOPS_PER_ENV_STEP
    return 141 + 144 + 378 * int(w["substeps"]) + 93 + 72


def measure_config(name, mlp, reps, device=0):
    """Time whole rollouts of one fp32 workload (T = its step count, rewards
    and dones written), L2 flushed before each; returns a result dict."""
    import torch
    from paper_2512_13359_gb300 import auvenv
    w = W.workload(name, mlp=mlp)
    n, T = int(w["n_envs"]), int(w["steps"])
    env = auvenv.Env(w)
    env.set_weights(W.policy_weights(w))
    env.reset()
    traj = env.alloc_traj(T, keys=("rew", "done"))
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    env.rollout(T, traj)
    torch.cuda.synchronize()
    ms = []
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        env.rollout(T, traj)
        e1.record(stream)
        ms.append((e0, e1))
    torch.cuda.synchronize()
    if env.status().code != 0:
        raise RuntimeError(f"device status after the {name} rollouts")
    env.close()
    t_ms = sum(a.elapsed_time(b) for a, b in ms) / len(ms)
    rate = n * T / (t_ms * 1e-3)
    peaks, src = load_peaks()
    pol = mlp_flops(W.obs_dim(w), w["hidden"], w["policy_out"])
    if mlp == "tf32":
        peak = peaks["bf16_tflops"] * 1.1 / 2.25
        # a CTA pair per 128-env tile while the tiles fill at most half the SMs
        n_sm = torch.cuda.get_device_properties(device).multi_processor_count
        kern = "k_rollout_tf32_pair" if 2 * ((n + 127) // 128) <= n_sm else "k_rollout_tf32"
        roof = {"bound": "tensor", "kernel": kern, "achieved": rate * pol / 1e12,
                "peak": peak, "unit": "TFLOP/s", "frac": rate * pol / 1e12 / peak,
                "peak_source": f"bf16 burst, {src}, x tf32/bf16 nominal 1.1/2.25"}
    else:
        n_sm = torch.cuda.get_device_properties(device).multi_processor_count
        peak = 2 * 128 * n_sm * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        ach = rate * (pol + dyn_flops(w)) / 1e12
        roof = {"bound": "alu", "kernel": "k_rollout_fp32", "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak,
                "peak_source": f"FP32 pipe 2*128*{n_sm} SMs*max clock (derived)"}
    return {"workload": name, "mlp": mlp, "n_envs": n, "steps": T, "substeps": w["substeps"],
            "value": rate, "unit": "env-steps/s", "ms_per_rollout": t_ms, "reps": reps,
            "flops_per_env_step": pol + dyn_flops(w), "roofline": roof,
            "trajectory": ["rew", "done"], "l2": "flushed before each rollout"}


def run_replay(args):
    """--replay: the physics-only line of its own."""
    from paper_2512_13359_gb300 import build
    build.build()
    over = {}
    if args.n_envs:
        over["n_envs"] = args.n_envs
    if args.rollout_steps:
        over["steps"] = args.rollout_steps
    w = W.workload(args.workload, **over)
    n, T = int(w["n_envs"]), int(w["steps"])
    step_ms, units, achieved, fp32_peak, src, clock_info = measure_replay(
        w, args.steps, args.warmup, not args.no_clocks)
    line = {
        "metric": "env-steps/s (physics only, action replay)", "value": units / (step_ms * 1e-3),
        "unit": "env-steps/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic",
        "config": {"workload": w["name"], "n_envs_per_gpu": n, "rollout_steps": T,
                   "substeps": w["substeps"], "l2": "flushed between timed steps"},
        "roofline": {"bound": "alu", "kernel": "k_replay", "achieved": achieved, "peak": fp32_peak,
                     "unit": "TFLOP/s", "frac": achieved / fp32_peak, "traffic": None,
                     "flops_per_env_step": dyn_flops_per_env_step(w), "peak_source": src},
        "gpu_launches": args.steps, "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


def run_probes(args):
    """The roofline denominators measured with the library's probes: the FP32
    pipe (FFMA chains at full occupancy) against 2 x 128 x SMs x clock, the
    multi-function unit (tanh.approx.f32 and ex2.approx.f32 chains), the
    tensor pipe for tf32 and bf16 operands (one 8192^3 cuBLAS GEMM each), and
    the tensor pipe's cost per tcgen05 MMA instruction (M = 128, K = 16,
    bf16) for each N the engine issues, one CTA per SM, in SM cycles."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    torch.cuda.init()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    blocks, threads = sms * 8, 256
    sink = torch.zeros(blocks * threads, device="cuda")

    def timed(fn, reps):
        fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            work = fn()
            e1.record()
            torch.cuda.synchronize()
            ts.append((e0.elapsed_time(e1) * 1e-3, work))
        ts.sort()
        t, work = ts[len(ts) // 2]
        return work / t

    clocks = ClockSampler(0) if not args.no_clocks else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ffma = timed(lambda: auvenv.probe_ffma(blocks, threads, 20000, sink), max(args.steps, 5))
    tanh = timed(lambda: auvenv.probe_tanh(blocks, threads, 4000, sink), max(args.steps, 5))
    ex2 = timed(lambda: auvenv.probe_ex2(blocks, threads, 4000, sink), max(args.steps, 5))
    mma, mma_tf32 = {}, {}
    mma_iters = 1024
    cyc = torch.zeros(sms, dtype=torch.int64, device="cuda")
    for tf32, out, k in ((False, mma, 16), (True, mma_tf32, 8)):
        for nn in (16, 32, 64, 128, 256):
            for a_tmem in (False, True):
                for _ in range(2):
                    auvenv.probe_mma(nn, a_tmem, mma_iters, cyc, tf32=tf32)
                torch.cuda.synchronize()
                c = cyc.cpu()
                if int((c == 0).sum()):
                    raise RuntimeError("mma probe: a bounded wait gave up")
                per = float(c.double().median()) / mma_iters
                out[f"n{nn}_{'ts' if a_tmem else 'ss'}"] = {
                    "cycles_per_mma": per, "mac_per_clk_per_sm": 128 * nn * k / per}
    n = 8192
    g = torch.Generator(device="cuda").manual_seed(0)
    a32 = torch.randn(n, n, device="cuda", generator=g)
    b32 = torch.randn(n, n, device="cuda", generator=g)
    c32 = torch.empty(n, n, device="cuda")
    tf32 = timed(lambda: auvenv.probe_gemm("tf32", a32, b32, c32), max(args.steps, 5))
    a16, b16 = a32.to(torch.bfloat16), b32.to(torch.bfloat16)
    bf16 = timed(lambda: auvenv.probe_gemm("bf16", a16, b16, c32), max(args.steps, 5))
    torch.cuda.synchronize()
    clock_info = clocks.stop() if clocks else None
    peaks, src = load_peaks()
    mhz = (clock_info or {}).get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
    derived = 2 * 128 * sms * mhz * 1e6
    line = {
        "metric": "roofline probes", "n_gpus": 1, "steps": max(args.steps, 5), "data": "synthetic",
        "probes": {
            "fp32_ffma_tflops": ffma / 1e12, "fp32_derived_tflops": derived / 1e12,
            "fp32_ffma_frac_of_derived": ffma / derived,
            "mufu_tanh_gops": tanh / 1e9,
            "mufu_tanh_per_clk_per_sm": tanh / (sms * mhz * 1e6),
            "mufu_ex2_gops": ex2 / 1e9,
            "mufu_ex2_per_clk_per_sm": ex2 / (sms * mhz * 1e6),
            "tcgen05_mma_m128_k16_bf16": mma,
            "tcgen05_mma_m128_k8_tf32": mma_tf32,
            "tf32_gemm_tflops": tf32 / 1e12, "bf16_gemm_tflops": bf16 / 1e12,
            "bf16_peak_measured_tflops": peaks.get("bf16_tflops"),
            "tf32_over_bf16": tf32 / bf16, "nominal_tf32_over_bf16": 1.1 / 2.25,
            "gemm_n": n, "sms": sms, "sm_mhz_used": mhz, "peaks_source": src},
        "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


def run_gae(args):
    """Advantage estimation (env_gae) over the workload's trajectory shape,
    fed by one real rollout: the HBM-bound learner input pass, HBM roofline
    (17 B per env-step + the bootstrap values)."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    over = {}
    if args.n_envs:
        over["n_envs"] = args.n_envs
    if args.rollout_steps:
        over["steps"] = args.rollout_steps
    w = W.workload(args.workload, **over)
    n, T = int(w["n_envs"]), int(w["steps"])
    env = auvenv.Env(w)
    env.set_weights(W.policy_weights(w), W.value_weights(w) if w["has_value"] else None)
    env.reset()
    traj = env.alloc_traj(T, keys=("obs", "rew", "done", "value"))
    env.rollout(T, traj)
    last = torch.randn(n, device="cuda")
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    for _ in range(args.warmup):
        env.gae(traj["rew"], traj["done"], traj["value"], last, 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    clocks = ClockSampler(0) if not args.no_clocks else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ms = []
    for _ in range(args.steps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        env.gae(traj["rew"], traj["done"], traj["value"], last, 0.99, 0.95, adv, ret)
        e1.record()
        ms.append((e0, e1))
    torch.cuda.synchronize()
    clock_info = clocks.stop() if clocks else None
    step_ms = sum(a.elapsed_time(b) for a, b in ms) / len(ms)
    peaks, src = load_peaks()
    bytes_ = n * T * 17 + n * 4
    achieved = bytes_ / (step_ms * 1e-3) / 1e9
    line = {
        "metric": "env-steps/s (advantage estimation)", "value": n * T / (step_ms * 1e-3),
        "unit": "env-steps/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic (one rollout's rewards, dones, values)",
        "config": {"workload": w["name"], "n_envs_per_gpu": n, "rollout_steps": T,
                   "gamma": 0.99, "lambda": 0.95, "l2": "flushed between timed steps"},
        "roofline": {"bound": "hbm", "kernel": "k_gae_chunked" if 8 < T <= 512 else "k_gae",
                     "achieved": achieved,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                     "traffic": None, "peak_source": f"HBM copy, {src}"},
        "gpu_launches": args.steps, "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


# DRAM bytes (read + write) of one rollout launch of the 65,536-env x
# 128-step workload, from one ncu capture (dram__bytes_read.sum +
# dram__bytes_write.sum, 1 pass, the first timed rollout of `bench.py
# --steps 2 --warmup 1 --no-e2e --no-cpu-baseline --no-replay --no-clocks`;
# profiles/k_engine_ppo_65536_T128_dram.md), valid while the engine's sources
# hash to ENGINE_SRC_HASH.
ROLLOUT_TRAFFIC_65536x128 = 10_622_976 + 900_608_256
ENGINE_SRC_HASH = "6e8400dd6451a3f1"
ENGINE_SRCS = ("k_bf16.cu", "auv_device.cuh", "tc_ptx.cuh", "auv_bf16.h")


def rollout_traffic(w, n, T):
    import hashlib
    if w["name"] != "ppo_65536" or n != 65536 or T != 128:
        return None
    h = hashlib.sha256()
    for f in ENGINE_SRCS:
        with open(os.path.join(ROOT, "paper_2512_13359_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return ROLLOUT_TRAFFIC_65536x128 if h.hexdigest()[:16] == ENGINE_SRC_HASH else None


def ppo_flops_per_sample(d, h, a):
    """Algorithmic flops of one PPO sample: forward of both MLPs
    (2 x multiply-adds), their weight gradients (same count) and the input
    gradients of layers 2 and 3 (layer 1's input gradient is not needed)."""
    fwd = mlp_flops(d, h, 2 * a) + mlp_flops(d, h, 1)
    return 3 * fwd - 2 * (2 * d * h)


def run_ppo(args):
    """The PPO update (ppo_update: epochs x minibatches of gather, forward,
    loss head, backward, Adam) over the trajectory of one rollout of the
    workload plus env_gae.  Tensor roofline: algorithmic flops of the two
    MLPs' forward and backward per sample."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    over = {}
    if args.n_envs:
        over["n_envs"] = args.n_envs
    if args.rollout_steps:
        over["steps"] = args.rollout_steps
    w = W.workload(args.workload, **over)
    n, T = int(w["n_envs"]), int(w["steps"])
    D, A, H = W.obs_dim(w), W.act_dim(w), int(w["hidden"])
    env = auvenv.Env(w)
    env.set_weights(W.policy_weights(w), W.value_weights(w))
    env.reset()
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    obs = torch.empty((1, D, n), device="cuda")
    env.observe(obs[0])
    last = torch.empty((1, n), device="cuda")
    env.value(obs, last)
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    env.gae(traj["rew"], traj["done"], traj["value"], last[0], 0.99, 0.95, adv, ret)
    batch = dict(obs=traj["obs"], act=traj["act"], logp=traj["logp"], adv=adv, ret=ret)
    B = args.minibatch
    n_mb = args.n_minibatches or (n * T) // B
    L = auvenv.Learner(D, A, H, B, precision=args.ppo_precision, seed=1,
                       logstd_min=w["logstd_min"], logstd_max=w["logstd_max"])
    L.set_weights(W.policy_weights(w), W.value_weights(w))
    stats = torch.empty(8, device="cuda")
    for _ in range(args.warmup):
        L.update(batch, args.epochs, n_mb, stats=stats)
    torch.cuda.synchronize()
    clocks = ClockSampler(0) if not args.no_clocks else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ms = []
    for _ in range(args.steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        L.update(batch, args.epochs, n_mb, stats=stats)
        e1.record()
        ms.append((e0, e1))
    torch.cuda.synchronize()
    clock_info = clocks.stop() if clocks else None
    step_ms = sum(a.elapsed_time(b) for a, b in ms) / len(ms)
    samples = args.epochs * n_mb * B
    fps = ppo_flops_per_sample(D, H, A)
    achieved = samples * fps / (step_ms * 1e-3) / 1e12
    peaks, src = load_peaks()
    if args.ppo_precision == "fp32":
        mhz = peaks.get("sm_max_mhz", 2070.0)
        peak, bound, psrc = 152 * 128 * 2 * mhz * 1e6 / 1e12, "alu", f"FP32 FMA, 152 SMs x 128 lanes at {mhz:.0f} MHz"
    else:
        ratio = 1.0 if args.ppo_precision == "bf16" else 1.1 / 2.25
        peak = peaks["bf16_tflops_sustained"] * ratio
        bound, psrc = "tensor", (f"bf16 sustained, {src}" + ("" if ratio == 1.0 else
                                 " x tf32/bf16 nominal 1.1/2.25"))
    st = stats.cpu().numpy().tolist()
    launches_per_step = 1 + 10 + 1 + 1 + 14 + 2     # gather, fwd, head, stats, bwd, norm+Adam
    line = {
        "metric": "PPO update samples/s", "value": samples / (step_ms * 1e-3),
        "unit": "samples/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32" if args.ppo_precision == "fp32" else args.ppo_precision,
        "data": "synthetic (one rollout of the workload, env_gae advantages)",
        "config": {"workload": w["name"], "n_envs": n, "rollout_steps": T, "rows": n * T,
                   "minibatch": B, "minibatches_per_epoch": n_mb, "epochs": args.epochs,
                   "precision": args.ppo_precision,
                   "l2": "working set per step larger than L2 when B >= 32768"},
        "roofline": {"bound": bound, "kernel": "whole update (the library's GEMMs and learner kernels)",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None, "peak_source": psrc,
                     "flops_per_sample": fps},
        "update_stats": dict(zip(auvenv.PPO_STAT_NAMES, st)),
        "gpu_launches": args.steps * args.epochs * n_mb * launches_per_step,
        "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


# FP32 operations one env-step of env_adjoint executes (forward pass, the
# backward pass's recompute of the step, and the VJPs), by substep count,
# FFMA counted twice: smsp__sass_thread_inst_executed_op_{fadd,fmul,ffma}_pred_on
# of k_adjoint from one ncu capture of `bench.py --adjoint --n-envs 8192`,
# divided by its 262,144 env-steps (674 FADD + 1273 FMUL + 2021 FFMA).
ADJOINT_FLOPS_PER_ENV_STEP = {4: 5988.2}
# The paper model's k_paper_adjoint, counted the same way (4 substeps,
# history of K = 4): `bench.py --adjoint --workload paper_4096 --n-envs 8192`.
PAPER_ADJOINT_FLOPS_PER_ENV_STEP = {4: 4452.3}   # 409 FADD + 979 FMUL + 1532 FFMA


def run_adjoint(args):
    """The reverse-mode adjoint of the Fossen control step over an action
    window (env_adjoint) from the workload's state: forward re-simulation,
    then the backward sweep.  One step = one window over all envs."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    over = {}
    if args.n_envs:
        over["n_envs"] = args.n_envs
    w = W.workload(args.workload, **over)
    n, T = int(w["n_envs"]), int(args.window)
    A = W.act_dim(w)
    S = 61 if W.is_paper(w) else 13
    env = auvenv.Env(w)
    env.reset()
    warm = torch.from_numpy(W.replay_actions(1, 8, n, scale=0.8, act=A)).cuda()
    rew0 = torch.empty((8, n), device="cuda")
    done0 = torch.empty((8, n), dtype=torch.uint8, device="cuda")
    env.step_actions(warm, rew0, done0)
    act = torch.from_numpy(W.replay_actions(2, T, n, scale=0.9, act=A)).cuda()
    coef = torch.tensor([0.99 ** t / (n * T) for t in range(T)], dtype=torch.float32,
                        device="cuda")
    lam_T = torch.randn((S, n), device="cuda") / (n * T)
    g = torch.empty((T, A, n), device="cuda")
    lam_0 = torch.empty((S, n), device="cuda")
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    for _ in range(args.warmup):
        env.adjoint(act, coef, g, lam_T=lam_T, lam_0=lam_0)
    torch.cuda.synchronize()
    clocks = ClockSampler(0) if not args.no_clocks else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ms = []
    for _ in range(args.steps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        env.adjoint(act, coef, g, lam_T=lam_T, lam_0=lam_0)
        e1.record()
        ms.append((e0, e1))
    torch.cuda.synchronize()
    clock_info = clocks.stop() if clocks else None
    assert env.status().code == 0
    step_ms = sum(a.elapsed_time(b) for a, b in ms) / len(ms)
    rate = n * T / (step_ms * 1e-3)
    peaks, src = load_peaks()
    mhz = peaks.get("sm_max_mhz", 2070.0)
    peak = 152 * 128 * 2 * mhz * 1e6 / 1e12
    table = PAPER_ADJOINT_FLOPS_PER_ENV_STEP if W.is_paper(w) else ADJOINT_FLOPS_PER_ENV_STEP
    fps = table.get(int(w["substeps"]))
    achieved = None if fps is None else rate * fps / 1e12
    line = {
        "metric": "adjoint env-steps/s", "value": rate, "unit": "env-steps/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (workload state after 8 replayed steps, random actions)",
        "config": {"workload": w["name"], "n_envs": n, "window": T,
                   "substeps": int(w["substeps"]), "l2": "flushed between timed steps"},
        "roofline": {"bound": "alu",
                     "kernel": "k_paper_adjoint" if W.is_paper(w) else "k_adjoint",
                     "achieved": achieved, "peak": peak,
                     "unit": "TFLOP/s", "frac": None if achieved is None else achieved / peak,
                     "traffic": None,
                     "peak_source": f"FP32 FMA, 152 SMs x 128 lanes at {mhz:.0f} MHz",
                     "flops_per_env_step": fps},
        "gpu_launches": args.steps, "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)


def _timed(args, fn, flush=None):
    import torch
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    ms = []
    for _ in range(args.steps):
        if flush is not None:
            flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        ms.append((e0, e1))
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in ms) / len(ms)


def run_rbuf(args):
    """Replay buffer (rbuf_insert of one 65,536 x 128 rollout trajectory,
    then rbuf_sample of 65,536-transition minibatches).  HBM roofline:
    (2 D + A + 1) * 4 + 1 bytes read and written per transition."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    over = {"n_envs": args.n_envs} if args.n_envs else {}
    w = W.workload(args.workload, **over)
    n, T = int(w["n_envs"]), int(w["steps"])
    D, A = W.obs_dim(w), W.act_dim(w)
    env = auvenv.Env(w)
    env.set_weights(W.policy_weights(w), W.value_weights(w) if w["has_value"] else None)
    env.reset()
    traj = env.alloc_traj(T, keys=("obs", "act", "rew", "done"))
    env.rollout(T, traj)
    last = torch.empty((D, n), device="cuda")
    env.observe(last)
    rb = auvenv.ReplayBuffer(D, A, 1 << 24)
    rec = (2 * D + A + 1) * 4 + 1
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    ins_ms = _timed(args, lambda: rb.insert(traj["obs"], traj["act"], traj["rew"], traj["done"],
                                            last), flush)
    B = 65536
    out = rb.sample(B, 1, 0)
    draws = iter(range(1, 10 ** 9))
    smp_ms = _timed(args, lambda: rb.sample(B, 1, next(draws), out=out), flush)
    peaks, src = load_peaks()
    ins_gbs = 2 * rec * n * T / (ins_ms * 1e-3) / 1e9
    smp_gbs = 2 * rec * B / (smp_ms * 1e-3) / 1e9
    line = {
        "metric": "replay-buffer sampled transitions/s", "value": B / (smp_ms * 1e-3),
        "unit": "transitions/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": smp_ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic (one rollout of the workload)",
        "config": {"workload": w["name"], "capacity": 1 << 24, "minibatch": B,
                   "inserted_per_call": n * T, "l2": "flushed between timed steps"},
        "insert": {"transitions_per_s": n * T / (ins_ms * 1e-3), "ms": ins_ms,
                   "achieved_gbs": ins_gbs, "frac": ins_gbs / peaks["hbm_gbs"]},
        "roofline": {"bound": "hbm", "kernel": "k_rb_sample", "achieved": smp_gbs,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": smp_gbs / peaks["hbm_gbs"],
                     "traffic": None, "peak_source": f"HBM copy, {src}",
                     "bytes_per_transition": 2 * rec},
        "gpu_launches": args.steps, "clocks": None,
    }
    print(json.dumps(line), flush=True)


def run_invalloc(args):
    """Inverse thruster allocation (env_inverse_allocate) of one wrench per
    env; HBM roofline 56 B per row (6 floats in, 8 out)."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    n = args.n_envs or (1 << 24)
    w = W.workload("ppo_65536", n_envs=1024)
    env = auvenv.Env(w)
    wrench = torch.randn((6, n), device="cuda") * 30.0
    cmd = torch.empty((8, n), device="cuda")
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    ms = _timed(args, lambda: env.inverse_allocate(wrench, cmd), flush)
    peaks, src = load_peaks()
    gbs = 56 * n / (ms * 1e-3) / 1e9
    line = {
        "metric": "inverse allocations/s", "value": n / (ms * 1e-3), "unit": "rows/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (N(0, 30^2) wrenches)",
        "config": {"workload": "inverse allocation of the ppo_65536 vehicle", "rows": n,
                   "l2": "flushed between timed steps"},
        "roofline": {"bound": "hbm", "kernel": "k_inverse_alloc", "achieved": gbs,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": gbs / peaks["hbm_gbs"],
                     "traffic": None, "peak_source": f"HBM copy, {src}"},
        "gpu_launches": args.steps, "clocks": None,
    }
    print(json.dumps(line), flush=True)


def run_shac(args):
    """SHAC's actor gradient over one window in closed loop (env_shac_window):
    forward with the policy network, then back-propagation through the
    dynamics, the network and the observation, with the terminal critic.
    FP32 roofline: the policy network's forward, weight gradients and input
    gradients (3 x 148,480 flop per env-step) plus the physics forward and
    adjoint (5,988 flop per env-step, k_adjoint's count)."""
    import torch
    from paper_2512_13359_gb300 import auvenv, build
    build.build()
    over = {"n_envs": args.n_envs} if args.n_envs else {}
    w = W.workload(args.workload, mlp="fp32", **over)
    n, T, H = int(w["n_envs"]), int(args.window), int(w["hidden"])
    env = auvenv.Env(w)
    env.reset()
    pw = torch.from_numpy(W.policy_weights(w, 0.05)).cuda()
    vw = torch.from_numpy(W.value_weights(w, 0.1)).cuda()
    coef = torch.tensor([0.99 ** t / (n * T) for t in range(T)], dtype=torch.float32,
                        device="cuda")
    grad = torch.empty_like(pw)
    prec = "tf32" if args.ppo_precision in ("tf32", "bf16") else "fp32"
    ms = _timed(args, lambda: env.shac_window(pw, vw, coef, 0.99 ** T / n, grad, precision=prec))
    assert env.status().code == 0
    rate = n * T / (ms * 1e-3)
    fps = 3 * mlp_flops(W.obs_dim(w), H, 16) + ADJOINT_FLOPS_PER_ENV_STEP.get(int(w["substeps"]), 0)
    peaks, src = load_peaks()
    mhz = peaks.get("sm_max_mhz", 2070.0)
    if prec == "tf32":
        peak = peaks["bf16_tflops_sustained"] * 1.1 / 2.25
        bound, psrc = "tensor", f"bf16 sustained, {src}, x tf32/bf16 nominal 1.1/2.25"
    else:
        peak = 152 * 128 * 2 * mhz * 1e6 / 1e12
        bound, psrc = "alu", f"FP32 FMA, 152 SMs x 128 lanes at {mhz:.0f} MHz"
    achieved = rate * fps / 1e12
    line = {
        "metric": "SHAC window env-steps/s", "value": rate, "unit": "env-steps/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "tf32" if prec == "tf32" else "f32",
        "data": "synthetic (workload resets, seeded random policy and critic)",
        "config": {"workload": w["name"], "n_envs": n, "window": T, "hidden": H, "precision": prec,
                   "l2": "working set per window (activations of every step) larger than L2"},
        "roofline": {"bound": bound, "kernel": "whole window (the library's GEMMs and adjoint kernels)",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None, "peak_source": psrc,
                     "flops_per_env_step": fps},
        "gpu_launches": args.steps * (17 * T + 16), "clocks": None,
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.shac:
        run_shac(args)
        return
    if args.rbuf:
        run_rbuf(args)
        return
    if args.invalloc:
        run_invalloc(args)
        return
    if args.adjoint:
        run_adjoint(args)
        return
    if args.ppo:
        run_ppo(args)
        return
    if args.replay:
        run_replay(args)
        return
    if args.gae:
        run_gae(args)
        return
    if args.probes:
        run_probes(args)
        return
    if args.sweep:
        base_steps = args.steps
        for n in W.SWEEP_SIZES:
            a = argparse.Namespace(**vars(args))
            a.workload, a.n_envs, a.rollout_steps, a.sweep = "sweep", n, None, False
            a.no_e2e, a.no_cpu_baseline, a.no_replay, a.no_configs = True, True, True, True
            a.steps = max(3, min(base_steps, int(2e8 // (n * 256)) + 3))
            run(a)
        return
    run(args)


def run(args):
    over = {}
    if args.n_envs:
        over["n_envs"] = args.n_envs
    if args.rollout_steps:
        over["steps"] = args.rollout_steps
    if args.mlp:
        over["mlp"] = args.mlp
    w = W.workload(args.workload, **over)
    if args.impl == "reference":
        run_reference(args, w)
        return

    import torch
    from paper_2512_13359_gb300 import shard
    rank, world, local = shard.world()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2512_13359_gb300 import auvenv, build
    if rank == 0 or world == 1:
        build.build()
    shard.barrier(dist)

    T = int(w["steps"])
    w["env_id_base"], n = shard.env_range(rank, int(w["n_envs"]))
    env = auvenv.Env(w)
    pw = W.policy_weights(w)
    vw = W.value_weights(w) if w["has_value"] else None
    env.set_weights(pw, vw)
    env.reset()
    keys = ["obs", "act", "logp", "rew", "done"]
    traj = env.alloc_traj(T, keys=keys)
    value = torch.empty((T, n), dtype=torch.float32, device="cuda") if w["has_value"] else None
    stream = torch.cuda.current_stream()
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")

    def one_step(ev=None):
        if ev:
            ev[0].record(stream)
        env.rollout(T, traj)
        if ev:
            ev[1].record(stream)
        if value is not None:
            env.value(traj["obs"], value)
        if ev:
            ev[2].record(stream)

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()
    st = env.status()
    if st.code != 0:
        raise RuntimeError(f"device status {st.code} after warm-up")

    clocks = ClockSampler(local) if not args.no_clocks else None
    shard.barrier(dist)
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)
    events = []
    for _ in range(args.steps):
        flush.zero_()                       # evict L2 between timed steps
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        one_step(ev)
        events.append(ev)
    torch.cuda.synchronize()
    shard.barrier(dist)
    clock_info = clocks.stop() if clocks else None
    roll_ms = [e[0].elapsed_time(e[1]) for e in events]
    val_ms = [e[1].elapsed_time(e[2]) for e in events]
    step_ms = shard.max_over_ranks(sum(r + v for r, v in zip(roll_ms, val_ms)) / args.steps,
                                   dist, "cuda")
    env_steps = n * T * world
    value_rate = env_steps / (step_ms * 1e-3)
    st = env.status()
    if st.code != 0:
        raise RuntimeError(f"device status {st.code} after timed steps")

    # ---- end to end through the C ABI with host buffers ----
    e2e = None
    if not args.no_e2e:
        # one env_rollout call per pass with page-locked host arrays (the
        # library stages them through device buffers); traj.value makes the
        # same call run the value pass
        h_keys = keys + (["value"] if value is not None else [])
        h_traj = env.alloc_traj(T, keys=h_keys, pinned_host=True)
        h_pw = torch.from_numpy(pw).pin_memory()
        h_vw = torch.from_numpy(vw).pin_memory() if vw is not None else None
        h2d = h_pw.numel() * 4 + (h_vw.numel() * 4 if h_vw is not None else 0)
        d2h = n * T * traj_bytes_per_env_step(w, h_keys)
        for _ in range(2):
            env.set_weights(h_pw, h_vw)
            env.rollout(T, h_traj)
            torch.cuda.synchronize()
        shard.barrier(dist)
        t0 = time.perf_counter()
        for _ in range(max(1, min(args.steps, 5))):
            env.set_weights(h_pw, h_vw)          # step inputs: policy + value weights, H2D
            env.rollout(T, h_traj)               # trajectory (and values) to host memory
            torch.cuda.synchronize()
        e2e_s = shard.max_over_ranks((time.perf_counter() - t0) / max(1, min(args.steps, 5)),
                                     dist, "cuda")
        e2e = {"value": env_steps / e2e_s, "unit": "env-steps/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return

    # ---- roofline of the dominant kernel ----
    peaks, peak_src = load_peaks()
    roll_avg = sum(roll_ms) / len(roll_ms)
    val_avg = sum(val_ms) / len(val_ms) if value is not None else 0.0
    pol_fl = mlp_flops(W.obs_dim(w), w["hidden"], w["policy_out"])
    val_fl = mlp_flops(W.obs_dim(w), w["hidden"], 1) if w["has_value"] else 0
    sm_mhz = (clock_info or {}).get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
    n_sm = torch.cuda.get_device_properties(local).multi_processor_count
    fp32_peak = 2 * 128 * n_sm * sm_mhz * 1e6 / 1e12   # TFLOP/s of the FP32 pipe
    if w["mlp"] == "bf16":
        if roll_avg >= val_avg:
            kern, dur = "rollout_bf16", roll_avg
            flops = n * T * pol_fl          # tensor-core work of the fused rollout
        else:
            kern, dur = "value_bf16", val_avg
            flops = n * T * val_fl
        achieved = flops / (dur * 1e-3) / 1e12
        # each launch (a few ms) is timed on its own: the burst peak applies
        peak = peaks["bf16_tflops"]
        roof = {"bound": "tensor", "kernel": kern, "achieved": achieved, "peak": peak,
                "unit": "TFLOP/s", "frac": achieved / peak,
                "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"],
                "traffic": rollout_traffic(w, n, T) if kern == "rollout_bf16" else None,
                "peak_source": f"bf16 burst, {peak_src}"}
    elif w["mlp"] == "tf32":
        peak = peaks["bf16_tflops"] * 1.1 / 2.25
        achieved = n * T * pol_fl / (roll_avg * 1e-3) / 1e12
        roof = {"bound": "tensor", "kernel": "rollout_tf32", "achieved": achieved, "peak": peak,
                "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                "peak_source": f"bf16 burst, {peak_src}, x tf32/bf16 nominal 1.1/2.25"}
    else:
        kern, dur = "rollout_fp32", roll_avg
        flops = n * T * (pol_fl + val_fl + dyn_flops_per_env_step(w))
        if value is not None and val_avg > roll_avg:
            kern, dur, flops = "value_fp32", val_avg, n * T * val_fl
        elif value is not None:
            flops = n * T * (pol_fl + dyn_flops_per_env_step(w))
        achieved = flops / (dur * 1e-3) / 1e12
        roof = {"bound": "alu", "kernel": kern, "achieved": achieved, "peak": fp32_peak,
                "unit": "TFLOP/s", "frac": achieved / fp32_peak, "traffic": None,
                "peak_source": f"FP32 pipe 2*128*{n_sm} SMs*{sm_mhz:.0f} MHz"}

    cpu = None
    if not args.no_cpu_baseline:
        from oracle import oracle as O
        O.build()
        rate, n_s, dt = oracle_sample_rate(w, T, args.cpu_seconds)
        # then the same sample on every host core at once (disjoint env ids)
        pool = OraclePool(w)
        try:
            wall = pool.run(n_s, T)
        finally:
            pool.close()
        cpu = {"value": pool.cores * n_s * T / wall, "unit": "env-steps/s", "cores": pool.cores,
               "kind": "oracle", "one_core": rate,
               "sample": (f"{n_s} envs x {T} steps of {w['name']} per process, {pool.cores} "
                          f"processes ({wall:.1f} s wall); one thread alone {rate:.0f} "
                          f"env-steps/s ({dt:.1f} s)")}

    # the physics alone (action replay) on the same workload: the FP32
    # roofline of the dynamics step, measured after the timed region
    physics = None
    if not args.no_replay:
        r_ms, r_units, r_ach, r_peak, r_src, r_clk = measure_replay(
            dict(w, env_id_base=0), max(5, min(args.steps, 30)), 3, not args.no_clocks, local)
        physics = {"metric": "env-steps/s (physics only, action replay)",
                   "value": r_units / (r_ms * 1e-3), "unit": "env-steps/s", "ms": r_ms,
                   "kernel": "k_replay" if not W.is_paper(w) else "k_paper_replay",
                   "bound": "alu", "achieved": r_ach, "peak": r_peak, "unit_roofline": "TFLOP/s",
                   "frac": r_ach / r_peak, "flops_per_env_step": dyn_flops_per_env_step(w),
                   "peak_source": r_src, "sm_mhz": (r_clk or {}).get("sm_mhz")}

    # the fp32 workloads (one whole rollout each, timed after the timed region)
    configs = None
    if not args.no_configs and world == 1:
        configs = [measure_config(nm, mlp, 3, local) for nm, mlp in CONFIG_LINES]

    launches_per_step = 1 + (1 if value is not None else 0)
    line = {
        "metric": "env-steps/s (physics+policy+reward)", "value": value_rate,
        "unit": "env-steps/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": {"bf16": "bf16", "tf32": "tf32"}.get(w["mlp"], "f32"),
        "data": "synthetic",
        "config": {"workload": w["name"], "n_envs_per_gpu": n, "rollout_steps": T,
                   "substeps": w["substeps"], "mlp": w["mlp"], "hidden": w["hidden"],
                   "trajectory": keys + (["value"] if value is not None else []),
                   "l2": "flushed between timed steps (2 x L2 buffer written)",
                   "rollout_ms": roll_avg, "value_ms": val_avg},
        "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "physics_only": physics,
        "fp32_workloads": configs,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clock_info,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


# Algorithmic FP32 flops of the non-network part of one env-step with 4
# substeps, counted by running the oracle's formulation with an
# operation-counting scalar: observation 141 + allocation 144 + 4 x 378
# (substep) + reward 93 + action sampling and log-probability 72 (adds,
# multiplies and divides; square roots and transcendentals not counted).
DYN_FLOPS_PER_ENV_STEP = 1962
# The paper model, counted the same way: observation 95 + wrench 6 + 4 x 245
# (substep; the inertia-box constants, 78 flops that the oracle recomputes
# in every substep, are per model, not per step) + reward 185 (including its
# own observation of the post-step state) + sampling six actions 54.
PAPER_DYN_FLOPS_PER_ENV_STEP = 1320

if __name__ == "__main__":
    main()
