#!/usr/bin/env python
"""Benchmark of the rollout / payoff-evaluation path on GB300.

Default workload (one "step"): the PSRO payoff-table sweep on Leduc hold'em,
the largest of the five workloads: a 64 x 64 population of bf16 MLP policies
17-256-256-3 (fp32 accumulation on the tensor cores), 16,384 Monte-Carlo hands
per pair (4,096 pairs, ~67 M hands, ~300 M decisions): deal, observation,
policy forward of the acting seat, masked softmax + Philox draw, transition,
payoff reduction (malib_eval_payoff). Inputs (population, pair table) are
resident in HBM; L2 is flushed (256 MiB write) before every timed step; each
step uses a new seed. --workload selects another of the workloads.

Prints ONE JSON line (rank 0). --impl reference times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "env-steps/sec incl. policy inference and payoff entries/sec on 1 GB300; % of roofline"
UNIT = "env-steps/s"
FP32_LANES_PER_SM = 128
# DRAM bytes (read + write) per launch of each workload's dominant kernel, from
# ncu (dram__bytes_read.sum + dram__bytes_write.sum). The fp32 rollout kernels were captured
# on the benchmark's own workload with the two dram counters alone (one pass);
# about 62 MB of trajectory lines are still dirty in L2 when such a kernel ends,
# so their writes fall that much short of the bytes stored. The spread N=8 bf16
# figure is a one-episode capture x 2 (65,536 environments: one episode's output
# is 15x the L2, so the traffic grows in proportion);
# the evaluation kernels' traffic is the staging of the population, which does
# not grow with the hands per pair; the learner's gradient kernel was captured
# on the learner step's own workload.
NCU_TRAFFIC_PER_LAUNCH = {
    "leduc_eval_f32_t8_kernel": 1441536 + 512,
    "kuhn_eval_kernel": 26880,
    "spread_rollout_f32_kernel<3,18,64,0>": 1373184 + 2559883520,
    "leduc_eval_tc_kernel": 19416064 + 490240,
    "spread_rollout_f32_kernel<3,14,64,1>": 1683968 + 2068428800,
    "spread_rollout_f32_kernel<2,11,64,2>": 1547520 + 1034004736,
    "spread_rollout_tc_kernel": (18220032 + 1910865664) * 2,
    "learn_grad_kernel": 510880512 + 3277568,
    "spread_rollout_f32_kernel<2,8,64,3>": 1031936 + 706821376,
    "spread_rollout_f32_kernel<4,16,64,4>": 3663872 + 2780089856,
    "spread_rollout_f32_kernel<2,14,64,6>": 2387712 + 1377357056,
}


def mlp_flop(dims):
    i, h1, h2, o = dims
    return 2 * (i * h1 + h1 * h2 + h2 * o)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["leduc", "kuhn", "spread3", "adversary3", "speaker_listener",
                                           "leduc_bf16", "spread8", "meta", "learner", "learner_ppo", "push", "tag",
                                           "reference"],
                    default="leduc_bf16")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--hands", type=int, default=None,
                    help="hands per pair (a smaller case for profiler captures)")
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Max of a per-rank number over all ranks (the timing aggregation)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, world: int, device=None) -> float:
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        return json.load(open(p))
    except Exception:
        return {}


def workload(name: str, rank: int, hands=None):
    import workloads
    over = {} if hands is None else {"n_episodes": hands}
    if name == "leduc":
        w = workloads.config(2, **over)
    elif name == "leduc_bf16":
        w = workloads.config(5, **over)
    elif name == "kuhn":
        w = workloads.config(1, **over)
    elif name == "spread8":
        w = workloads.config(4, **({"n_episodes": 2} if hands is None else over))
    elif name == "adversary3":
        w = workloads.adversary(n_envs=4096, pop=16, n_episodes=100 if hands is None else hands)
    elif name == "speaker_listener":
        w = workloads.speaker_listener(n_envs=4096, pop=16, n_episodes=100 if hands is None else hands)
    elif name == "push":
        w = workloads.push(n_envs=4096, pop=16, n_episodes=100 if hands is None else hands)
    elif name == "tag":
        w = workloads.tag(n_envs=4096, pop=16, n_episodes=100 if hands is None else hands)
    elif name == "reference":
        w = workloads.reference(n_envs=4096, pop=16, n_episodes=100 if hands is None else hands)
    else:
        w = workloads.config(3, **({"n_episodes": 100} if hands is None else over))
    return w


def config_of(w, name):
    if name == "leduc":
        return {"workload": f"leduc_holdem_8x8_mlp17-128-128-3_f32_{w.n_episodes}hands",
                "pairs": w.n_pairs, "hands_per_pair": w.n_episodes,
                "policy": "MLP 17-128-128-3 fp32", "population_per_seat": w.rows,
                "l2": "flushed (256 MiB write) before every timed step"}
    if name == "leduc_bf16":
        return {"workload": f"leduc_holdem_64x64_mlp17-256-256-3_bf16_{w.n_episodes}hands",
                "pairs": w.n_pairs, "hands_per_pair": w.n_episodes,
                "policy": "MLP 17-256-256-3 bf16 (fp32 accumulate)", "population_per_seat": w.rows,
                "l2": "flushed (256 MiB write) before every timed step"}
    if name == "spread8":
        return {"workload": f"spread_n8_65536env_mlp34-256-256-5_bf16_{w.n_episodes}episodes",
                "envs": w.n_envs, "combinations": w.n_pairs, "episodes_per_env": w.n_episodes,
                "episode_len": 25, "l2": "trajectory output exceeds L2; flushed as well"}
    if name == "adversary3":
        return {"workload": f"simple_adversary_4096env_mlp14-64-64-5_f32_{w.n_episodes}episodes",
                "envs": w.n_envs, "combinations": w.n_pairs, "episodes_per_env": w.n_episodes,
                "episode_len": 25, "l2": "trajectory output exceeds L2; flushed as well"}
    if name == "speaker_listener":
        return {"workload": f"simple_speaker_listener_4096env_mlp11-64-64-5_f32_{w.n_episodes}episodes",
                "envs": w.n_envs, "combinations": w.n_pairs, "episodes_per_env": w.n_episodes,
                "episode_len": 25, "l2": "trajectory output exceeds L2; flushed as well"}
    if name in ("push", "tag", "reference"):
        return {"workload": f"simple_{name}_4096env_mlp{w.obs_dim}-64-64-{w.n_actions}_f32_{w.n_episodes}episodes",
                "envs": w.n_envs, "combinations": w.n_pairs, "episodes_per_env": w.n_episodes,
                "episode_len": 25, "contact_forces": name != "reference",
                "l2": "trajectory output exceeds L2; flushed as well"}
    if name == "kuhn":
        return {"workload": "kuhn_4x4_tabular_10000hands", "pairs": w.n_pairs,
                "hands_per_pair": w.n_episodes,
                "l2": "flushed (256 MiB write) before every timed step"}
    return {"workload": "spread_n3_4096env_mlp18-64-64-5_f32_100episodes", "envs": w.n_envs,
            "combinations": w.n_pairs, "episodes_per_env": w.n_episodes, "episode_len": 25,
            "l2": "trajectory output (2.5 GB per step) exceeds L2; flushed as well"}


# ----------------------------------------------------------------- CPU oracle
def oracle_leduc_sample(w, target_s: float, threads: int):
    """Times the oracle on the first n hands of every pair, n sized so that the
    run takes about target_s seconds. Returns (decisions/s, sample text)."""
    import numpy as np
    import oracle
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims

    def run(n):
        dec = np.zeros(w.n_pairs, np.int64)
        t0 = time.perf_counter()
        oracle.leduc_eval(params, dims, w.pair_ids, w.n_episodes, w.seed, n_sim=n,
                          decisions=dec, n_threads=threads, bf16=w.policies[0].dtype == 1)
        return time.perf_counter() - t0, int(dec.sum())

    n = 8
    dt, dec = run(n)
    while dt < 0.5 and n < w.n_episodes:
        n = min(w.n_episodes, n * 4)
        dt, dec = run(n)
    n2 = max(1, min(w.n_episodes, int(n * target_s / max(dt, 1e-6))))
    if n2 != n:
        dt, dec = run(n2)
        n = n2
    return dec / dt, f"first {n} hands of each of the {w.n_pairs} pairs ({dec} decisions, {dt:.1f} s)"


def oracle_rollout_sample(w, name, target_s: float, threads: int):
    """Times the oracle's rollout (one episode) on the first n environments, n
    sized so that the run takes about target_s seconds. Returns (env-steps/s,
    sample text)."""
    import oracle
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    bf16 = w.policies[0].dtype == 1

    def run(n, eps=1):
        t0 = time.perf_counter()
        if name == "adversary3":
            oracle.adversary_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, eps, w.seed,
                                     env_lo=0, env_hi=n, n_threads=threads)
        elif name == "speaker_listener":
            oracle.sl_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, eps, w.seed,
                              env_lo=0, env_hi=n, n_threads=threads)
        elif name in ("push", "tag", "reference"):
            roll = {"push": oracle.push_rollout, "tag": oracle.tag_rollout, "reference": oracle.ref_rollout}[name]
            roll(params, dims, w.episode_len, w.n_envs, w.pair_ids, eps, w.seed, env_lo=0, env_hi=n,
                 n_threads=threads)
        else:
            oracle.spread_rollout(params, dims, w.n_agents, w.n_landmarks, w.episode_len, w.n_envs,
                                  w.pair_ids, eps, w.seed, bf16=bf16, env_lo=0, env_hi=n,
                                  n_threads=threads)
        return time.perf_counter() - t0

    n = threads
    dt = run(n)
    while dt < 0.5 and n < w.n_envs:
        n = min(w.n_envs, n * 4)
        dt = run(n)
    eps = 1
    n2 = max(1, min(w.n_envs, int(n * target_s / max(dt, 1e-6))))
    if n2 == w.n_envs and n == w.n_envs:
        # every environment fits: add episodes, the oracle's output kept under 512 MB
        per_ep = w.n_envs * w.episode_len * w.n_agents * (w.obs_dim + 8) * 4
        eps = max(1, min(w.n_episodes, int(target_s / max(dt, 1e-6)), (512 << 20) // per_ep))
    if n2 != n or eps != 1:
        dt = run(n2, eps)
        n = n2
    steps = n * w.episode_len * eps
    return steps / dt, (f"first {n} of the {w.n_envs} environments, {eps} episode(s) of "
                        f"{w.episode_len} steps ({steps} env-steps, {dt:.1f} s)")


def oracle_kuhn_sample(w, target_s: float, threads: int):
    """Times the oracle's Kuhn evaluation on the first n hands of every pair."""
    import numpy as np
    import oracle
    tables = np.stack([p.params for p in w.policies])

    def run(n):
        t0 = time.perf_counter()
        oracle.kuhn_eval(tables, w.pair_ids, n, w.seed, n_threads=threads)
        return time.perf_counter() - t0

    n = 1000
    dt = run(n)
    while dt < 0.5 and n < (1 << 26):
        n *= 4
        dt = run(n)
    n2 = max(1, int(n * target_s / max(dt, 1e-6)))
    if n2 != n:
        dt = run(n2)
        n = n2
    # decisions per hand, exactly: 2, plus a third when seat 0 passes (infoset
    # card * 2) and seat 1 then bets (infoset card * 2), over the 6 deals
    deals = [(a, b) for a in range(3) for b in range(3) if a != b]
    dec = 0.0
    for i, j in w.pair_ids:
        p0, p1 = tables[i].astype(np.float64), tables[j].astype(np.float64)
        dec += n * (2.0 + sum((1.0 - p0[2 * a]) * p1[2 * b] for a, b in deals) / 6.0)
    return dec / dt, (f"first {n} hands of each of the {w.n_pairs} pairs ({dt:.1f} s; decisions "
                      f"counted by their exact expectation per pair)")


def cpu_count():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_step_fn(w, name, threads, per_step):
    """One bounded step of the oracle on workload `w`, sized once so that it
    takes about per_step seconds: returns (step(seed) -> units done, sample
    text). Units are the workload's metric unit (decisions or env-steps)."""
    import numpy as np
    import oracle
    params = [p.params for p in w.policies]
    dims = w.policies[0].dims
    if name in ("leduc", "leduc_bf16"):
        bf16 = w.policies[0].dtype == 1
        _, sample = oracle_leduc_sample(w, per_step, threads)
        n = int(sample.split()[1])

        def step(seed):
            dec = np.zeros(w.n_pairs, np.int64)
            oracle.leduc_eval(params, dims, w.pair_ids, w.n_episodes, seed, n_sim=n,
                              decisions=dec, n_threads=threads, bf16=bf16)
            return int(dec.sum())
        return step, f"per step: first {n} hands of each of the {w.n_pairs} pairs"
    if name == "kuhn":
        rate, sample = oracle_kuhn_sample(w, per_step, threads)
        n = int(sample.split()[1])
        tables = np.stack([p.params for p in w.policies])
        deals = [(a, b) for a in range(3) for b in range(3) if a != b]
        dec = 0.0
        for i, j in w.pair_ids:
            p0, p1 = tables[i].astype(np.float64), tables[j].astype(np.float64)
            dec += n * (2.0 + sum((1.0 - p0[2 * a]) * p1[2 * b] for a, b in deals) / 6.0)

        def step(seed):
            oracle.kuhn_eval(tables, w.pair_ids, n, seed, n_threads=threads)
            return dec
        return step, (f"per step: first {n} hands of each of the {w.n_pairs} pairs (decisions "
                      "counted by their exact expectation per pair)")
    # rollouts: the first n environments, one episode
    _, sample = oracle_rollout_sample(w, name, per_step, threads)
    n = int(sample.split()[1])
    bf16 = w.policies[0].dtype == 1

    def step(seed):
        if name == "adversary3":
            oracle.adversary_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, 1, seed,
                                     env_lo=0, env_hi=n, n_threads=threads)
        elif name == "speaker_listener":
            oracle.sl_rollout(params, dims, w.episode_len, w.n_envs, w.pair_ids, 1, seed,
                              env_lo=0, env_hi=n, n_threads=threads)
        elif name in ("push", "tag", "reference"):
            roll = {"push": oracle.push_rollout, "tag": oracle.tag_rollout, "reference": oracle.ref_rollout}[name]
            roll(params, dims, w.episode_len, w.n_envs, w.pair_ids, 1, seed, env_lo=0, env_hi=n,
                 n_threads=threads)
        else:
            oracle.spread_rollout(params, dims, w.n_agents, w.n_landmarks, w.episode_len, w.n_envs,
                                  w.pair_ids, 1, seed, bf16=bf16, env_lo=0, env_hi=n,
                                  n_threads=threads)
        return n * w.episode_len
    return step, (f"per step: first {n} of the {w.n_envs} environments, one episode of "
                  f"{w.episode_len} steps")


def run_reference(args):
    """The reference arm: the CPU oracle, as it stands, on the host cores, on a
    bounded sample of the same workload as the GPU arm (rank 0 only)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    name = "leduc_bf16" if args.workload == "meta" else args.workload
    w = workload(name, 0, args.hands)
    threads = cpu_count()
    per_step = max(0.2, min(5.0, 150.0 / max(1, args.steps + args.warmup)))
    step, sample = oracle_step_fn(w, name, threads, per_step)
    for k in range(args.warmup):
        step(w.seed + 10_000 + k)
    tot_units, tot_t = 0.0, 0.0
    for k in range(args.steps):
        t0 = time.perf_counter()
        tot_units += step(w.seed + k)
        tot_t += time.perf_counter() - t0
    value = tot_units / tot_t
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * tot_t / max(1, args.steps), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(w, name),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------- GPU arm
def run_ours(args):
    import numpy as np
    import torch

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import Context, alloc_traj, make_spec, policy_desc

    w = workload(args.workload, rank, args.hands)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    ctx = Context(local, stream)
    spec = make_spec(w.env_kind, w.n_agents, w.obs_dim, w.n_actions, w.n_landmarks,
                     w.episode_len, w.n_envs)
    d_params = [torch.from_numpy(p.params).to(dev) for p in w.policies]
    ctx.pop_load(spec, [policy_desc(p.kind, p.dtype, p.seat, p.dims, d)
                        for p, d in zip(w.policies, d_params)])
    d_pairs = torch.from_numpy(w.pair_ids).to(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    seed0 = w.seed + 1_000_003 * rank
    rollout = args.workload in ("spread3", "spread8", "adversary3", "speaker_listener", "push", "tag", "reference")
    if rollout:
        traj = alloc_traj(spec, w.n_episodes)
        steps_per_call = w.n_envs * w.episode_len * w.n_episodes
        flop_per_unit = w.n_agents * mlp_flop(w.policies[0].dims)
    else:
        d_out = torch.empty((w.n_pairs, 4), dtype=torch.float64, device=dev)
        flop_per_unit = mlp_flop(w.policies[0].dims) if w.env_kind == 2 else 0
    tensor = args.workload in ("leduc_bf16", "spread8")

    def step(seed):
        if rollout:
            ctx.rollout(spec, d_pairs, w.n_episodes, seed, traj)
            return steps_per_call
        ctx.eval_payoff(d_pairs, w.n_episodes, seed, d_out)
        return None

    for k in range(args.warmup):
        step(seed0 + 10_000 + k)
    torch.cuda.synchronize(dev)
    ctx.sync()

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    decisions = 0
    ctx.main_kernel_ms(reset=True)
    ctx.set_timing(True)
    launches0 = ctx.launch_count()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clocks:
        for k in range(args.steps):
            flush.zero_()
            ev[k][0].record(stream)
            n = step(seed0 + k)
            ev[k][1].record(stream)
            decisions += n if n is not None else ctx.eval_decisions()
        torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    launches = ctx.launch_count() - launches0
    ctx.set_timing(False)
    ctx.sync()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = sum(step_ms)
    kern_ms, kern_n = ctx.main_kernel_ms(reset=True)
    clk = clocks.summary()

    total_ms_max = max_over_ranks(total_ms, world, dev)
    dec_all = sum_over_ranks(float(decisions), world, dev)
    value = dec_all / (total_ms_max / 1e3)
    entries = sum_over_ranks(float(w.n_pairs * args.steps), world, dev) / (total_ms_max / 1e3)

    peaks = load_peaks()
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    peak_tflops = n_sm * FP32_LANES_PER_SM * 2 * sm_max * 1e6 / 1e12
    achieved = (decisions * flop_per_unit / args.steps) / (kern_ms / kern_n / 1e3) / 1e12 \
        if kern_n else 0.0
    kname = {"leduc": "leduc_eval_f32_t8_kernel", "kuhn": "kuhn_eval_kernel",
             "spread3": "spread_rollout_f32_kernel<3,18,64,0>",
             "adversary3": "spread_rollout_f32_kernel<3,14,64,1>",
             "speaker_listener": "spread_rollout_f32_kernel<2,11,64,2>",
             "push": "spread_rollout_f32_kernel<2,8,64,3>",
             "tag": "spread_rollout_f32_kernel<4,16,64,4>",
             "reference": "spread_rollout_f32_kernel<2,14,64,6>",
             "leduc_bf16": "leduc_eval_tc_kernel",
             "spread8": "spread_rollout_tc_kernel"}[args.workload]
    basis = (f"fp32 FMA: {n_sm} SMs (queried) x {FP32_LANES_PER_SM} lanes x 2 flop"
             f" x {sm_max:.0f} MHz (max SM clock of MEASURED_PEAKS.json)")
    if tensor:
        # the kernel is timed alone, launch by launch, with CUDA events: the
        # burst figure of the measured cuBLAS bf16 GEMM is its peak
        if "bf16_tflops" in peaks:
            peak_tflops = float(peaks["bf16_tflops"])
            basis = "measured cuBLAS bf16 dense GEMM, burst (MEASURED_PEAKS.json bf16_tflops), of measured"
        else:
            peak_tflops = 1900.0
            basis = "fallback bf16 dense burst 1.9 PFLOP/s (no MEASURED_PEAKS.json), of fallback"
    roofline = {"bound": "tensor" if tensor else "alu", "achieved": achieved,
                "peak": peak_tflops, "unit": "TFLOP/s",
                "frac": achieved / peak_tflops if peak_tflops else None,
                "traffic": NCU_TRAFFIC_PER_LAUNCH.get(kname),
                "kernel": kname, "kernel_ms_per_launch": kern_ms / max(1, kern_n),
                "peak_basis": basis,
                "algorithmic": f"{flop_per_unit} flop per env-step (MLP forward, padding excluded)"}
    if clk.get("sm_mhz") and not tensor:
        roofline["frac_at_measured_clock"] = achieved / (peak_tflops * clk["sm_mhz"] / sm_max)
    if args.workload == "kuhn":
        # Kuhn's work is generator arithmetic: one Philox call per deal and one
        # per decision; the ceiling is the measured rate of a Philox-only kernel
        calls = (w.n_pairs * w.n_episodes * args.steps + decisions) / args.steps
        rate = calls / (kern_ms / max(1, kern_n) / 1e3) if kern_n else 0.0
        ceil = philox_ceiling(ctx, stream, n_sm)
        roofline = {"bound": "alu", "achieved": rate / 1e9, "peak": ceil / 1e9,
                    "unit": "Gcall/s (Philox4x32-10)", "frac": rate / ceil,
                    "traffic": None, "kernel": kname,
                    "kernel_ms_per_launch": kern_ms / max(1, kern_n),
                    "peak_basis": f"measured: malib_philox_digest, {n_sm * 8 * 256} threads x "
                                  "4,096 calls per launch, best of 5 (CUDA events)",
                    "algorithmic": "1 Philox4x32-10 call per deal + 1 per decision"}

    e2e = run_e2e(args, ctx, w, spec, dev, rollout) if rank == 0 else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload != "meta":
        if args.workload in ("leduc", "leduc_bf16"):
            rate, sample = oracle_leduc_sample(w, 12.0, cpu_count())
        elif args.workload == "kuhn":
            rate, sample = oracle_kuhn_sample(w, 12.0, cpu_count())
        else:
            rate, sample = oracle_rollout_sample(w, args.workload, 12.0, cpu_count())
        cpu = {"value": rate, "unit": UNIT, "cores": cpu_count(), "kind": "oracle",
               "sample": sample}
    ctx.close()
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16" if tensor else "f32",
                "data": "synthetic", "config": config_of(w, args.workload),
                "payoff_entries_per_s": entries if not rollout else None,
                "env_steps_per_step": decisions / args.steps,
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
                "gpu_launches": launches}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def philox_ceiling(ctx, stream, n_sm):
    """Philox4x32-10 calls per second of the library's arithmetic-only digest
    kernel: best of 5 launches after 3 warm-ups, timed with CUDA events on the
    context's stream."""
    import torch
    n, calls = n_sm * 8 * 256, 4096
    out = torch.empty(n, dtype=torch.int32, device=stream.device)
    best = None
    for k in range(8):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        ctx.philox_digest(0x5EED + k, calls, out)
        b.record(stream)
        b.synchronize()
        if k >= 3:
            ms = a.elapsed_time(b)
            best = ms if best is None else min(best, ms)
    return n * calls / (best / 1e3)


def run_e2e(args, ctx, w, spec, dev, rollout):
    """The same metric through the public API with host buffers: population
    upload from pinned host memory and the pair (or combination) table in; the
    payoff table (evaluation) or the trajectory's rewards (rollout) back."""
    import numpy as np
    import torch
    from paper_2106_07551_gb300 import policy_desc
    if rollout:
        return run_e2e_rollout(args, ctx, w, spec, dev)
    h_params = [torch.from_numpy(p.params).pin_memory() for p in w.policies]
    h_pairs = torch.from_numpy(w.pair_ids).pin_memory()
    h_out = torch.empty((w.n_pairs, 4), dtype=torch.float64).pin_memory()
    descs = [policy_desc(p.kind, p.dtype, p.seat, p.dims, h) for p, h in zip(w.policies, h_params)]
    h2d = sum(h.numel() * 4 for h in h_params) + h_pairs.numel() * 4
    d2h = h_out.numel() * 8
    n = max(1, args.e2e_steps)
    tot, dec = 0.0, 0
    for k in range(n + 1):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        ctx.pop_reset()
        ctx.pop_load(spec, descs)
        ctx.eval_payoff(h_pairs, w.n_episodes, w.seed + 777 + k, h_out)   # returns after D2H
        t1 = time.perf_counter()
        d = ctx.eval_decisions()
        if k > 0:            # first call warms the host path
            tot += t1 - t0
            dec += d
    return {"value": dec / tot, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": n}


def run_e2e_rollout(args, ctx, w, spec, dev):
    """Rollout end to end: population and combination table from pinned host
    memory, the rollout into device trajectory buffers (where a learner on the
    GPU reads them), and every agent-step's reward copied back to pinned host
    memory as the step's result."""
    import torch
    from paper_2106_07551_gb300 import alloc_traj, policy_desc
    h_params = [torch.from_numpy(p.params).pin_memory() for p in w.policies]
    h_pairs = torch.from_numpy(w.pair_ids).pin_memory()
    descs = [policy_desc(p.kind, p.dtype, p.seat, p.dims, h) for p, h in zip(w.policies, h_params)]
    traj = alloc_traj(spec, w.n_episodes)
    h_rew = torch.empty(traj["reward"].shape, dtype=torch.float32).pin_memory()
    h2d = sum(h.numel() * 4 for h in h_params) + h_pairs.numel() * 4
    d2h = h_rew.numel() * 4
    steps_per_call = w.n_envs * w.episode_len * w.n_episodes
    n = max(1, args.e2e_steps)
    tot = 0.0
    for k in range(n + 1):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        ctx.pop_reset()
        ctx.pop_load(spec, descs)
        ctx.rollout(spec, h_pairs, w.n_episodes, w.seed + 777 + k, traj)
        h_rew.copy_(traj["reward"], non_blocking=True)
        ctx.sync()
        torch.cuda.synchronize(dev)
        t1 = time.perf_counter()
        if k > 0:            # first call warms the host path
            tot += t1 - t0
    return {"value": steps_per_call * n / tot, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": n}


# ----------------------------------------------------------------- meta-solver
META_GAMES, META_M, META_N, META_PLAYS = 152, 100, 100, 10_000


def run_meta(args):
    """Fictitious play (the Sec. 4.2 meta-solver) on a batch of payoff tables of
    the paper's largest PSRO population (100 x 100), one game per SM: a step
    is META_PLAYS plays of every game. Also times the LP equilibrium and the
    aggregation on the same tables (reported beside the main value)."""
    import numpy as np
    import torch

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2106_07551_gb300 import Context

    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    ctx = Context(local, stream)
    rng = np.random.default_rng(2106075516 + rank)
    G, m, n, T = META_GAMES, META_M, META_N, META_PLAYS
    tables = rng.normal(size=(G, m, n))
    P = torch.from_numpy(tables).to(dev)
    x = torch.empty((G, m), dtype=torch.float64, device=dev)
    y = torch.empty((G, n), dtype=torch.float64, device=dev)
    b = torch.empty((G, 2), dtype=torch.float64, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        ctx.meta_fictitious_play(P, T, x, y, b)
    torch.cuda.synchronize(dev)
    ctx.sync()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    launches0 = ctx.launch_count()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clocks:
        for k in range(args.steps):
            flush.zero_()
            ev[k][0].record(stream)
            ctx.meta_fictitious_play(P, T, x, y, b)
            ev[k][1].record(stream)
        torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    launches = ctx.launch_count() - launches0
    ctx.sync()
    total_ms = sum(a.elapsed_time(c) for a, c in ev)
    total_ms_max = max_over_ranks(total_ms, world, dev)
    plays_all = sum_over_ranks(float(G * T * args.steps), world, dev)
    value = plays_all / (total_ms_max / 1e3)
    ns_per_play = total_ms / args.steps * 1e6 / T     # per CTA (all games run concurrently)

    # LP and aggregation on the same tables
    v = torch.empty((G,), dtype=torch.float64, device=dev)
    ay = torch.empty((G, m), dtype=torch.float64, device=dev)
    xa = torch.empty((G, n), dtype=torch.float64, device=dev)
    ctx.meta_lp_nash(P, x, y, v)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    ctx.meta_lp_nash(P, x, y, v)
    e1.record(stream)
    ctx.meta_aggregate(P, x, y, ay, xa, v)
    torch.cuda.synchronize(dev)
    ctx.sync()
    lp_ms = e0.elapsed_time(e1)

    # exploitability of uniform mixtures over the whole Leduc 64 x 64 bf16 population
    import workloads
    from paper_2106_07551_gb300 import make_spec, policy_desc
    w5 = workloads.config(5, n_episodes=16)
    spec5 = make_spec(w5.env_kind, w5.n_agents, w5.obs_dim, w5.n_actions)
    ctx.pop_load(spec5, [policy_desc(p.kind, p.dtype, p.seat, p.dims, p.params) for p in w5.policies])
    ids0 = [i for i, p in enumerate(w5.policies) if p.seat == 0]
    ids1 = [i for i, p in enumerate(w5.policies) if p.seat == 1]
    ux, uy = np.full(len(ids0), 1.0 / len(ids0)), np.full(len(ids1), 1.0 / len(ids1))
    expl = ctx.exploitability(ids0, ux, ids1, uy)
    reps = 20
    t0 = time.perf_counter()
    for _ in range(reps):
        expl = ctx.exploitability(ids0, ux, ids1, uy)
    expl_ms = (time.perf_counter() - t0) / reps * 1e3

    e2e = None
    cpu = None
    expl_cpu_s = None
    if rank == 0:
        # e2e: tables from pinned host memory, mixtures and bounds back
        h_tab = torch.from_numpy(tables).pin_memory()
        h_x = torch.empty((G, m), dtype=torch.float64).pin_memory()
        h_y = torch.empty((G, n), dtype=torch.float64).pin_memory()
        h_b = torch.empty((G, 2), dtype=torch.float64).pin_memory()
        reps = max(1, args.e2e_steps // 5)
        t0 = 0.0
        for k in range(reps + 1):
            torch.cuda.synchronize(dev)
            s0 = time.perf_counter()
            P.copy_(h_tab, non_blocking=True)
            ctx.meta_fictitious_play(P, T, x, y, b)
            h_x.copy_(x, non_blocking=True)
            h_y.copy_(y, non_blocking=True)
            h_b.copy_(b, non_blocking=True)
            torch.cuda.synchronize(dev)
            if k > 0:
                t0 += time.perf_counter() - s0
        e2e = {"value": G * T * reps / t0, "unit": "plays/s",
               "h2d_bytes_per_step": int(h_tab.numel() * 8),
               "d2h_bytes_per_step": int((h_x.numel() + h_y.numel() + h_b.numel()) * 8),
               "steps": reps}
        if world == 1 and not args.no_cpu_baseline:
            from oracle import meta_solver as ms
            n_games, t_cpu = 0, 0.0
            while t_cpu < 10.0 and n_games < G:
                s0 = time.perf_counter()
                ms.fictitious_play(tables[n_games], T)
                t_cpu += time.perf_counter() - s0
                n_games += 1
            cpu = {"value": n_games * T / t_cpu, "unit": "plays/s", "cores": 1, "kind": "oracle",
                   "sample": f"{n_games} of the {G} games, {T} plays each ({t_cpu:.1f} s, numpy)"}
            from oracle import exploit as ex
            P5 = [p.params for p in w5.policies]
            t_ex = time.perf_counter()
            ex.leduc_exploitability([P5[i] for i in ids0], ux, [P5[i] for i in ids1], uy,
                                    w5.policies[0].dims, True)
            expl_cpu_s = time.perf_counter() - t_ex
    clk = clocks.summary()
    ctx.close()
    if rank == 0:
        line = {"metric": "fictitious-play plays/sec over a batch of payoff tables",
                "value": value, "unit": "plays/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic",
                "config": {"workload": f"fictitious_play_{G}games_{m}x{n}_{T}plays",
                           "games": G, "rows": m, "cols": n, "plays": T,
                           "l2": "flushed (256 MiB write) before every timed step"},
                "roofline": {"bound": "latency", "achieved": ns_per_play, "peak": None,
                             "unit": "ns per play per game", "frac": None, "traffic": None,
                             "kernel": "fictitious_play_kernel",
                             "note": "each play depends on the previous play's argmax: one CTA "
                                     "barrier and two warp reductions per play bound it"},
                "lp_nash_ms": lp_ms,
                "exploitability": {"workload": "leduc 64x64 bf16 population, uniform mixtures",
                                   "value": expl[2], "ms_per_call": expl_ms,
                                   "oracle_s": expl_cpu_s},
                "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
                "gpu_launches": launches}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


LEARN_EPISODES = 10


def learn_flop(dims):
    """Algorithmic flops of one sample's policy-gradient step: the forward (as
    mlp_flop) and the backward (dL/dh2 and dL/dh1 through W3 and W2, the
    weight gradients of W3, W2, W1; bias sums excluded)."""
    i, h1, h2, a = dims
    return mlp_flop(dims) + 2 * (a * h2 + h2 * h1) + 2 * (a * h2 + h2 * h1 + h1 * i)


def run_learner(args):
    """The learner-side update (Sec. 3.3 independent learning, App. C.2): one
    training iteration of every policy of the spread population (N = 3, 4,096
    envs, population 16, MLP 18-64-64-5 fp32) on LEARN_EPISODES episodes of
    its rollout: malib_learn_pg_batch over the whole population (each policy its
    own independent learner) and one malib_adam_step over all parameters. A step
    covers every sample once (each belongs to one policy)."""
    import numpy as np
    import torch

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    import workloads
    from paper_2106_07551_gb300 import Context, alloc_traj, make_spec, policy_desc

    w = workloads.config(3, n_episodes=LEARN_EPISODES)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    ctx = Context(local, stream)
    ppo = args.workload == "learner_ppo"
    from paper_2106_07551_gb300 import MALIB_DUMP_LOGITS
    spec = make_spec(w.env_kind, w.n_agents, w.obs_dim, w.n_actions, w.n_landmarks, w.episode_len, w.n_envs,
                     MALIB_DUMP_LOGITS if ppo else 0)
    ctx.pop_load(spec, [policy_desc(p.kind, p.dtype, p.seat, p.dims, p.params) for p in w.policies])
    d_pairs = torch.from_numpy(w.pair_ids).to(dev)
    traj = alloc_traj(spec, w.n_episodes, logits=ppo)
    ctx.rollout(spec, d_pairs, w.n_episodes, w.seed + rank, traj)
    dims = w.policies[0].dims
    n_pol = len(w.policies)
    P = int(dims[1] * dims[0] + dims[1] + dims[2] * dims[1] + dims[2] + dims[3] * dims[2] + dims[3])
    grads = torch.zeros((n_pol, P), dtype=torch.float32, device=dev)
    params = torch.from_numpy(np.stack([p.params for p in w.policies]).astype(np.float32)).to(dev)
    m = torch.zeros_like(params)
    v = torch.zeros_like(params)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    samples = w.n_envs * w.episode_len * w.n_episodes * w.n_agents
    state = {"t": 0}

    ids = np.arange(n_pol, dtype=np.int32)

    def step():
        state["t"] += 1
        if ppo:
            ctx.learn_ppo_batch(spec, d_pairs, w.n_episodes, traj, ids, 0.95, 0.001, 0.2, grads)
        else:
            ctx.learn_pg_batch(spec, d_pairs, w.n_episodes, traj, ids, 0.95, 0.001, grads)
        ctx.adam_step(params, grads, m, v, state["t"], 1e-4)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    ctx.sync()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    launches0 = ctx.launch_count()
    ctx.set_timing(True)                 # learn_grad_kernel's own CUDA-event time
    ctx.main_kernel_ms(reset=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clocks:
        for k in range(args.steps):
            flush.zero_()
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    launches = ctx.launch_count() - launches0
    ctx.sync()
    grad_ms, grad_n = ctx.main_kernel_ms(reset=True)
    ctx.set_timing(False)
    total_ms = sum(a.elapsed_time(c) for a, c in ev)
    total_ms_max = max_over_ranks(total_ms, world, dev)
    value = sum_over_ranks(float(samples * args.steps), world, dev) / (total_ms_max / 1e3)
    peaks = load_peaks()
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
    peak = n_sm * FP32_LANES_PER_SM * 2 * sm_max * 1e6 / 1e12
    grad_avg_ms = grad_ms / max(grad_n, 1)
    achieved = samples * learn_flop(dims) / (grad_avg_ms / 1e3) / 1e12
    e2e = None
    cpu = None
    if rank == 0:
        # e2e: the trajectory from pinned host memory, every policy's gradient back
        h_obs = traj["obs"].cpu().pin_memory()
        h_act = traj["action"].cpu().pin_memory()
        h_rew = traj["reward"].cpu().pin_memory()
        h_lg = traj["logits"].cpu().pin_memory() if ppo else None
        h_g = torch.empty_like(grads, device="cpu").pin_memory()
        reps = max(1, args.e2e_steps // 5)
        t_e2e = 0.0
        for k in range(reps + 1):
            torch.cuda.synchronize(dev)
            s0 = time.perf_counter()
            traj["obs"].copy_(h_obs, non_blocking=True)
            traj["action"].copy_(h_act, non_blocking=True)
            traj["reward"].copy_(h_rew, non_blocking=True)
            if ppo:
                traj["logits"].copy_(h_lg, non_blocking=True)
            step()
            h_g.copy_(grads, non_blocking=True)
            torch.cuda.synchronize(dev)
            if k > 0:
                t_e2e += time.perf_counter() - s0
        e2e = {"value": samples * reps / t_e2e, "unit": "samples/s",
               "h2d_bytes_per_step": int(h_obs.numel() * 4 + h_act.numel() + h_rew.numel() * 4 +
                                         (h_lg.numel() * 4 if ppo else 0)),
               "d2h_bytes_per_step": int(h_g.numel() * 4), "steps": reps}
        if world == 1 and not args.no_cpu_baseline:
            from oracle import learner as ol
            tr = {"obs": h_obs.numpy(), "action": h_act.numpy(), "reward": h_rew.numpy()}
            if ppo:
                tr["logits"] = h_lg.numpy()
            n_done, t_cpu, n_s = 0, 0.0, 0
            while t_cpu < 10.0 and n_done < n_pol:
                s0 = time.perf_counter()
                o, a_, r_ = ol.gather(tr, w.pair_ids, w.n_envs, w.n_agents, w.obs_dim, n_done, 0.95)
                if ppo:
                    bl = ol.gather_logits(tr, w.pair_ids, w.n_envs, w.n_agents, n_done)
                    ol.ppo_grad(w.policies[n_done].params, dims, o, a_, r_, bl, 0.001, 0.2)
                else:
                    ol.pg_grad(w.policies[n_done].params, dims, o, a_, r_, 0.001)
                t_cpu += time.perf_counter() - s0
                n_s += o.shape[0]
                n_done += 1
            cpu = {"value": n_s / t_cpu, "unit": "samples/s", "cores": cpu_count(), "kind": "oracle",
                   "sample": f"{n_done} of the {n_pol} policies' gradients ({n_s} samples, {t_cpu:.1f} s, "
                             "numpy fp64)"}
    clk = clocks.summary()
    ctx.close()
    if rank == 0:
        line = {"metric": ("learner samples/sec (PPO clipped-surrogate step and Adam of every policy)" if ppo
                           else "learner samples/sec (policy-gradient step and Adam of every policy)"),
                "value": value, "unit": "samples/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": "synthetic",
                "config": {"workload": f"learner{'_ppo' if ppo else ''}_spread_n3_4096env_mlp18-64-64-5_f32_"
                                       f"{w.n_episodes}episodes_pop{n_pol}", "samples_per_step": samples,
                           "policies": n_pol,
                           "l2": "flushed (256 MiB write) before every timed step"},
                "roofline": {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                             "frac": achieved / peak,
                             "traffic": None if ppo else NCU_TRAFFIC_PER_LAUNCH.get("learn_grad_kernel"),
                             "kernel": "learn_grad_kernel",
                             "peak_basis": f"fp32 FMA: {n_sm} SMs (queried) x {FP32_LANES_PER_SM} lanes x 2 "
                                           f"flop x {sm_max:.0f} MHz",
                             "algorithmic": f"{learn_flop(dims)} flop per sample (forward and backward, "
                                            f"bias sums excluded) x {samples} samples per launch",
                             "kernel_ms": grad_avg_ms, "step_share": grad_avg_ms / (total_ms / args.steps)},
                "cpu_baseline": cpu, "e2e": e2e, "clocks": clk, "gpu_launches": launches}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "meta":
        return run_meta(args)
    if args.workload in ("learner", "learner_ppo"):
        return run_learner(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
