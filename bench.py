#!/usr/bin/env python
"""Benchmark of the batched PPO power-controller path on GB300.

One step = one PPO iteration of the 7B workload (4,096 envs x 512 steps over
a 60,000-sample trace, 5 actions, fp32 16-128-128 policy/value MLPs):
rollout (env + policy + sampler, then the value network), GAE, and the PPO
update (4 epochs x 256 minibatches of 8,192).  Metric: env-steps/s
(E * T per step).  The fleet accounting (1,000,000 compositions of 16
traces x 380,000 samples, windows 1/60/600) is timed in the same run and
reported under "fleet" as window-samples/s.

Timing: W untimed warm-up steps, then K steps each bracketed by CUDA events
on the launch stream; an L2 flush (256 MB write) runs between timed steps,
outside the events.  Multi-GPU (torchrun): independent replicas (one per
rank, seed = rank), barrier + max over ranks; value = all ranks' env-steps
divided by the slowest rank's time.

--impl reference times the CPU oracle on a bounded sample of the same
workload (the paper ships no GPU implementation to compare against).
--ncu-case NAME runs one small case of a hot kernel, sized for ncu captures.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "PPO controller env-steps/s and fleet window-samples/s on 1 GB300; % HBM roofline"
FP32_LANES_PER_SM = 128
N_SM = 152
SM_MAX_MHZ = 2070.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--fleet-n", type=int, default=1_000_000)
    ap.add_argument("--fleet-steps", type=int, default=3)
    ap.add_argument("--no-eval", dest="eval", action="store_false",
                    help="skip the evaluation replay (baseline rules, ledger) and the rule-rollout timing")
    ap.add_argument("--stagger-stride", type=int, default=1,
                    help="candidate offset grid of the greedy staggered schedule (0: skip)")
    ap.add_argument("--cpu-envs", type=int, default=48, help="envs in the oracle CPU sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--r72b-steps", type=int, default=2, help="timed 72B rollouts (0: skip)")
    ap.add_argument("--r72b-envs", type=int, default=65536)
    ap.add_argument("--r72b-horizon", type=int, default=1024)
    ap.add_argument("--r72b-ppo-minibatches", type=int, default=16,
                    help="72B PPO minibatch steps of 65,536 samples timed (0: skip)")
    ap.add_argument("--ncu-case", choices=["ppo7b", "ppo72", "ppostress", "gae", "gae-chunked", "mlp72", "fleet"],
                    default=None,
                    help="run one small named case of a hot kernel (for ncu captures) and exit")
    ap.add_argument("--gae-large", type=int, nargs=2, default=[2048, 262144], metavar=("T", "E"),
                    help="GAE roofline size (Stress: 2048 x 262144); T=0 skips it")
    ap.add_argument("--stress", type=int, nargs=2, default=[262144, 2048], metavar=("E", "T"),
                    help="Stress iteration size (envs, horizon); E=0 skips the leg")
    ap.add_argument("--stress-fleet-n", type=int, default=1_000_000,
                    help="fleet compositions recomputed inside each Stress iteration")
    ap.add_argument("--no-cpu-table", dest="cpu_table", action="store_false",
                    help="skip the per-configuration oracle table (1 core and all host cores)")
    ap.add_argument("--no-roofs", dest="roofs", action="store_false",
                    help="skip the FP32 / INT32 / L2 roof microbenchmarks")
    return ap.parse_args()


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# --------------------------------------------------------------------------- helpers
def ppo_flops_per_sample(D, H, A):
    fwd = (D * H + H * H + H * A) + (D * H + H * H + H)
    bwd = (2 * H * A + 2 * H * H + D * H) + (2 * H + 2 * H * H + D * H)
    return 2 * (fwd + bwd)


def load_traffic(kernel: str):
    """dram bytes per launch from the committed ncu summary, if present."""
    path = os.path.join(ROOT, "profiles", f"{kernel}.md")
    if not os.path.exists(path):
        return None
    for line in open(path):
        if line.strip().startswith("traffic_bytes_per_launch:"):
            v = line.split(":", 1)[1].strip()
            return None if v in ("", "null") else float(v)
    return None


def load_traffic_per_unit(kernel: str, key: str):
    """dram bytes per unit of work (e.g. per env-step) from the committed ncu
    summary, for kernels whose traffic grows with the size of the launch."""
    path = os.path.join(ROOT, "profiles", f"{kernel}.md")
    if not os.path.exists(path):
        return None
    for line in open(path):
        if line.strip().startswith(key + ":"):
            v = line.split(":", 1)[1].strip()
            return None if v in ("", "null") else float(v)
    return None


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """The slowest rank's time (replicas report the whole job's throughput
    against it); NCCL reduces on the device, gloo on the host."""
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(units_per_rank: float, world: int, max_ms: float) -> float:
    """Whole-job throughput of weak-scaled replicas: every rank's units over
    the slowest rank's time."""
    return units_per_rank * world / (max_ms / 1e3)


# --------------------------------------------------------------------------- measured roofs
def measure_roofs(local: int):
    """FP32 FMA (scalar and packed two-lane), INT32 add and L2-read roofs of
    this GPU, each the best of 3 timed throughput loops (pe_roof_probe),
    with the SM clock sampled while they run."""
    from paper_2608_11226_gb300 import pe
    buf = torch.zeros(8 * 1024 * 1024, dtype=torch.float32, device="cuda")  # 32 MB: L2-resident
    clocks = ClockSampler(local)
    clocks.start()
    out = {}
    for name, kind, reps, unit, scale in (("fp32_ffma", pe.PE_ROOF_FFMA, 200000, "TFLOP/s", 1e12),
                                          ("fp32_ffma2", pe.PE_ROOF_FFMA2, 100000, "TFLOP/s", 1e12),
                                          ("int32_add", pe.PE_ROOF_IADD, 100000, "Tops/s", 1e12),
                                          ("l2_read", pe.PE_ROOF_L2, 20, "GB/s", 1e9)):
        best = 0.0
        for _ in range(3):
            ms, units = pe.roof_probe(kind, buf, reps)
            best = max(best, units / (ms / 1e3) / scale)
        out[name] = {"value": best, "unit": unit}
    clk = clocks.stop()
    out["fp32_fma_peak_tflops"] = max(out["fp32_ffma"]["value"], out["fp32_ffma2"]["value"])
    out["clocks"] = clk
    out["how"] = ("pe_roof_probe: 8 CTAs x 256 threads per SM, 8 independent chains per thread "
                  "(FFMA / packed FFMA2 / IADD), or 16-byte L2-only loads over a 32 MB buffer; "
                  "best of 3 launches timed with CUDA events")
    del buf
    return out


# --------------------------------------------------------------------------- our path
class Trainer:
    """State of one 7B PPO training replica on the device."""

    def __init__(self, seed: int):
        from paper_2608_11226_gb300 import pe
        from paper_2608_11226_gb300 import workloads as W
        self.pe, self.W = pe, W
        self.wl = W.make_7b(seed=seed)
        wl = self.wl
        self.E, self.T = wl.env.n_envs, wl.horizon
        self.env = pe.Env(wl.env, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
        self.buf = pe.alloc_rollout(wl.env, wl.net, self.T)
        self.params = torch.from_numpy(W.init_params(wl.net, seed=seed)).cuda()
        self.m = torch.zeros_like(self.params)
        self.v = torch.zeros_like(self.params)
        self.adv = torch.empty(self.T, self.E, device="cuda")
        self.ret = torch.empty_like(self.adv)
        self.stats = torch.zeros(8, device="cuda")
        N = self.E * self.T
        self.ws = torch.empty(pe.ppo_workspace_bytes(wl.net, wl.ppo, N), dtype=torch.uint8, device="cuda")
        self.adam_t = 0
        self.it = 0
        self.seed = seed
        self.steps_per_update = wl.ppo.epochs * ((N + wl.ppo.minibatch - 1) // wl.ppo.minibatch)

    def step(self):
        pe, wl = self.pe, self.wl
        pe.rollout(self.env, wl.net, self.params, self.T, self.it, self.buf)
        pe.gae(self.buf["reward"], self.buf["value"], self.buf["done"], self.buf["last_value"],
               wl.ppo.gamma, wl.ppo.lam, self.adv, self.ret)
        pe.ppo_update(wl.net, wl.ppo, self.params, self.m, self.v, self.adam_t, self.buf["obs"],
                      self.buf["act"], self.buf["logp"], self.adv, self.ret, self.stats, self.ws,
                      seed=1000 + self.seed, iteration=self.it)
        self.adam_t += self.steps_per_update
        self.it += 1


def run_ours(args, world, rank, local):
    from paper_2608_11226_gb300 import build, pe
    from paper_2608_11226_gb300 import workloads as W
    build.build()
    pe.lib()
    roofs = measure_roofs(local) if args.roofs else None
    tr = Trainer(seed=rank)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")  # 256 MB > L2
    for _ in range(args.warmup):
        tr.step()
    torch.cuda.synchronize()
    # ---- timed region (device time, CUDA events on the launch stream)
    for k in range(pe.PE_PROF_KINDS):
        pe.profile_read(k)
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    pe.profile_enable(True)
    stream = torch.cuda.current_stream()
    evs = []
    for _ in range(args.steps):
        flush.fill_(1.0)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        tr.step()
        b.record(stream)
        evs.append((a, b))
    torch.cuda.synchronize()
    pe.profile_enable(False)
    barrier(world)
    clk = clocks.stop()
    total_ms = sum(a.elapsed_time(b) for a, b in evs)
    prof = {pe.profile_kind_name(k): pe.profile_read(k) for k in range(pe.PE_PROF_KINDS)}
    total_ms = max_over_ranks(total_ms, world)
    ms_step = total_ms / args.steps
    env_steps = tr.E * tr.T
    value = job_value(env_steps * args.steps, world, total_ms)
    launches = sum(n for _, n in prof.values())
    # ---- dominant kernel roofline (fp32 FFMA bound)
    gms, gn = prof["ppo_grad"]
    net = tr.wl.net
    # one launch is either the persistent update (all epochs x minibatches) or one minibatch
    samples_per_launch = (tr.E * tr.T * tr.wl.ppo.epochs) if gn == args.steps else tr.wl.ppo.minibatch
    kname = "ppo_persistent_kernel" if gn == args.steps else "ppo_grad_kernel"
    fl_launch = ppo_flops_per_sample(net.obs_dim, net.hidden, net.n_actions) * samples_per_launch
    derived_tflops = N_SM * FP32_LANES_PER_SM * 2 * SM_MAX_MHZ * 1e6 / 1e12
    if roofs:
        peak_tflops = roofs["fp32_fma_peak_tflops"]
        src = ("measured: pe_roof_probe FP32 FMA throughput loop (best of scalar FFMA and packed "
               f"FFMA2) in this run; derived figure {derived_tflops:.1f} TFLOP/s at 2070 MHz")
    else:
        peak_tflops = derived_tflops
        src = "derived: 152 SMs x 128 FP32 lanes x 2 FLOP x 2070 MHz"
    ach = fl_launch / (gms / gn / 1e3) / 1e12 if gn else None
    roof = {"kernel": kname, "bound": "alu", "achieved": ach, "peak": peak_tflops,
            "unit": "TFLOP/s", "frac": (ach / peak_tflops) if ach else None,
            "traffic": load_traffic(kname),
            "peak_source": src, "frac_of_derived": (ach / derived_tflops) if ach else None,
            "avg_launch_ms": gms / gn if gn else None, "launches": gn,
            "flop_per_launch": fl_launch}
    kernels = {k: {"ms_per_step": ms / args.steps, "launches_per_step": n / args.steps,
                   "share": ms / sum(x for x, _ in prof.values()) if n else 0.0}
               for k, (ms, n) in prof.items() if n}
    # GAE roofline (HBM): 17 algorithmic bytes per env-step
    gae_ms, gae_n = prof["gae"]
    gae_gbs = 17.0 * env_steps / (gae_ms / gae_n / 1e3) / 1e9 if gae_n else None
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) if os.path.exists(
        os.path.join(ROOT, "MEASURED_PEAKS.json")) else {"hbm_gbs": 6800.0}
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    # inputs just written by the rollout sit in L2 at this size: no DRAM traffic figure
    gae_roof = {"kernel": gae_kernel_name(tr.E), "bound": "hbm", "achieved": gae_gbs, "peak": hbm,
                "unit": "GB/s", "frac": gae_gbs / hbm if gae_gbs else None,
                "traffic": None}

    # ---- end to end through host buffers: model state uploaded from pinned
    # host memory every step, parameters + statistics + counters read back
    host_in = [x.cpu().pin_memory() for x in (tr.params, tr.m, tr.v)]
    host_out = {k: torch.empty(x.shape, dtype=x.dtype).pin_memory() for k, x in
                (("params", tr.params), ("m", tr.m), ("v", tr.v), ("stats", tr.stats),
                 ("viol", tr.buf["viol"]), ("tokens", tr.buf["tokens"]),
                 ("excess", tr.buf["excess"]), ("energy_q", tr.buf["energy_q"]))}
    h2d = sum(x.numel() * x.element_size() for x in host_in)
    d2h = sum(x.numel() * x.element_size() for x in host_out.values())
    e2e_steps = max(3, args.steps // 2)
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        tr.params.copy_(host_in[0], non_blocking=True)
        tr.m.copy_(host_in[1], non_blocking=True)
        tr.v.copy_(host_in[2], non_blocking=True)
        tr.step()
        for k, dst in host_out.items():
            src = {"params": tr.params, "m": tr.m, "v": tr.v, "stats": tr.stats}.get(k)
            dst.copy_(tr.buf[k] if src is None else src, non_blocking=True)
        torch.cuda.current_stream().synchronize()
        _ = float(host_out["stats"][5])
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    e2e = {"value": env_steps * world * e2e_steps / e2e_s, "unit": "env-steps/s",
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    ppo_stats_last = [float(x) for x in tr.stats.cpu()]
    # ---- fleet accounting
    fleet = run_fleet(args, world, tr, roofs) if args.fleet_n > 0 else None
    evaluation = run_evaluation(args, world, tr, peaks) if args.eval else None
    r72b = run_72b(args, world, peaks, local) if args.r72b_steps > 0 else None
    gae_large = run_gae_large(args, world, peaks) if args.gae_large[0] > 0 else None
    tiny = run_tiny(args, world)
    torch.cuda.empty_cache()
    stress = run_stress(args, world, peaks, local) if args.stress[0] > 0 else None

    out = {"metric": METRIC, "value": value, "unit": "env-steps/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
           "data": "synthetic",
           "config": {"workload": "7b: 4096 envs x 512 steps on a 60,000-sample 7B-GRPO-shaped "
                                  "trace, 5 actions, MLP 16-128-128 fp32, GAE, PPO 4 epochs x "
                                  "minibatch 8192", "n_envs": tr.E, "horizon": tr.T,
                      "parallelism": f"replicas x{world}" if world > 1 else "1 GPU",
                      "l2": "flushed between timed steps (256 MB write)"},
           "roofline": roof, "gae_roofline": gae_roof, "kernels": kernels,
           "gpu_launches": launches, "clocks": clk, "e2e": e2e, "fleet": fleet, "rollout_72b": r72b,
           "gae_roofline_stress_size": gae_large, "evaluation": evaluation,
           "stress_iteration": stress, "tiny_iteration": tiny, "measured_roofs": roofs,
           "ppo_stats_last": ppo_stats_last}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(args.cpu_envs)
    if rank == 0 and world == 1 and args.cpu_table:
        out["per_config"] = per_config_table(out)
    if rank == 0:
        print(json.dumps(out), flush=True)


KWH_PER_Q_SAMPLE = 0.5 / 64.0 / 3.6e6   # one sample of 1/64 W held 0.5 s, in kWh
PRICE_PER_KWH = 0.08                     # Sec. 4.4 / 9.1
CO2_KG_PER_KWH = 0.25                    # New York grid intensity, Sec. 4.4


def run_evaluation(args, world, tr, peaks):
    """Sec. 4.4 evaluation replay of the 7B trace: consecutive 500-step
    episodes covering the trace (119 envs), run under the random policy, the
    threshold heuristic (90% / 70% of the cap), the hysteresis rule (512 /
    510 / 525 W at a 561 W budget, scaled to this budget) and the bench's
    trained network acting deterministically; per arm the violation rates and
    the energy ledger (kWh, $ at 0.08/kWh, kg CO2 at 0.25 kg/kWh, Wh per
    1,000 tokens).  Then the rule rollout's throughput on the 72B env
    (65,536 envs x 1,024 steps)."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    base = W.make_7b(seed=tr.seed)
    L = base.trace.shape[-1]
    offs = W.replay_offsets(L, base.env.episode_len)
    E, T = len(offs), base.env.episode_len
    wl = W.make_7b(n_envs=E, seed=tr.seed)
    spec, net = wl.env, wl.net
    B = spec.budget_q
    arms = {"random": W.random_rule(), "threshold_90_70": W.threshold_rule(B),
            "hysteresis_512_510_525": W.hysteresis_rule(B), "learned_deterministic": None}
    out = {}
    for name, rule in arms.items():
        env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
        pe.set_offsets(env, torch.from_numpy(offs).cuda())
        if rule is None:
            buf = pe.alloc_rollout(spec, net, T)
            pe.rollout(env, net, tr.params, T, 0, buf, deterministic=True)
        else:
            buf = pe.alloc_rule_rollout(spec, T)
            pe.rollout_rule(env, rule, T, 0, buf)
        torch.cuda.synchronize()
        viol = buf["viol"].sum(0).cpu().numpy()
        tok = float(buf["tokens"].double().sum())
        kwh = float(buf["energy_q"].sum()) * KWH_PER_Q_SAMPLE
        out[name] = {"violation_rate_0.5s": float(viol[0]) / (E * T), "violation_rate_30s": float(viol[1]) / (E * T),
                     "tokens": tok, "energy_kwh": kwh, "cost_usd": kwh * PRICE_PER_KWH,
                     "co2_kg": kwh * CO2_KG_PER_KWH, "wh_per_1k_tokens": 1e3 * kwh * 1e3 / tok if tok else None}
        env.close()
    # throughput of the rule rollout at the 72B size
    w72 = W.make_72b(seed=0)
    env = pe.Env(w72.env, torch.from_numpy(w72.trace), torch.from_numpy(w72.phase))
    T72 = 1024
    buf = pe.alloc_rule_rollout(w72.env, T72)
    rule = W.hysteresis_rule(w72.env.budget_q)
    pe.rollout_rule(env, rule, T72, 0, buf)
    torch.cuda.synchronize()
    barrier(world)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    for it in range(2):
        pe.rollout_rule(env, rule, T72, it + 1, buf)
    b.record()
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b), world) / 2
    n = w72.env.n_envs * T72
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    gbs = 6.0 * n / (ms / 1e3) / 1e9  # act 1 + reward 4 + done 1 bytes written per env-step
    env.close()
    return {"arms": out, "config": {"workload": f"7b evaluation replay: {E} consecutive {T}-step episodes "
                                                "covering the 60,000-sample trace", "n_envs": E, "horizon": T},
            "rule_rollout_72b": {"metric": "rule-policy env-steps/s (hysteresis, 72B env)",
                                 "value": n * world / (ms / 1e3), "unit": "env-steps/s", "ms_per_rollout": ms,
                                 "roofline": {"kernel": "rule_rollout_kernel", "bound": "hbm", "achieved": gbs,
                                              "peak": hbm, "unit": "GB/s", "frac": gbs / hbm,
                                              "note": "6 B of buffer writes per env-step; latency-bound"}}}


def run_fleet(args, world, tr=None, roofs=None):
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    fw = W.make_fleet(n_compositions=args.fleet_n)
    G, L = fw.traces.shape
    traces = torch.from_numpy(fw.traces).cuda()
    job = torch.from_numpy(fw.job_of_gpu).cuda()
    off = torch.from_numpy(fw.offsets).cuda()
    N = fw.offsets.shape[0]
    windows = [1, 60, 600]
    counts = torch.empty((N, 3), dtype=torch.int32, device="cuda")
    peaks = torch.empty_like(counts)
    ws = torch.empty(pe.fleet_workspace_bytes(fw.n_jobs, L, fw.horizon), dtype=torch.uint8, device="cuda")
    pe.fleet_windows(traces, job, fw.n_jobs, off, fw.horizon, windows, fw.budget_q, counts, peaks, ws)
    torch.cuda.synchronize()
    for k in range(pe.PE_PROF_KINDS):
        pe.profile_read(k)
    barrier(world)
    pe.profile_enable(True)
    stream = torch.cuda.current_stream()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.fleet_steps):
        pe.fleet_windows(traces, job, fw.n_jobs, off, fw.horizon, windows, fw.budget_q, counts,
                         peaks, ws)
    b.record(stream)
    torch.cuda.synchronize()
    pe.profile_enable(False)
    ms = max_over_ranks(a.elapsed_time(b), world)
    wms, wn = pe.profile_read(pe.PE_PROF_FLEET_WINDOWS)
    pe.profile_read(pe.PE_PROF_FLEET_PREP)
    H = fw.horizon
    ws_per_call = sum(N * (H - w + 1) for w in windows)
    composed = N * H
    c = counts.cpu().numpy()
    p = peaks.cpu().numpy()
    stagger = run_stagger(args, world, fw, traces, job, p, tr) if args.stagger_stride > 0 else None
    return {"metric": "fleet window-samples/s", "value": ws_per_call * world * args.fleet_steps / (ms / 1e3),
            "unit": "window-samples/s", "ms_per_call": ms / args.fleet_steps,
            "config": {"workload": "fleet: 16 traces x 380,000 samples (2x72B@4, 2x14B@2, 4x7B@1), "
                                   f"{N} offset compositions, windows 1/60/600, budget 0.5 x nameplate",
                       "n": N, "horizon": H},
            "kernel_ms_per_launch": wms / wn if wn else None,
            "composed_samples_per_s": composed / (wms / wn / 1e3) if wn else None,
            "logical_l2_gbs": 4.0 * fw.n_jobs * composed / (wms / wn / 1e3) / 1e9 if wn else None,
            "roofline": ({"kernel": "fleet_windows_v4_kernel", "bound": "l2",
                          "achieved": 4.0 * fw.n_jobs * composed / (wms / wn / 1e3) / 1e9,
                          "peak": roofs["l2_read"]["value"], "unit": "GB/s",
                          "frac": 4.0 * fw.n_jobs * composed / (wms / wn / 1e3) / 1e9 / roofs["l2_read"]["value"],
                          "note": "logical bytes: 4 B per job per composed sample, against the measured "
                                  "L2-read roof (32 MB resident buffer)"}
                         if (wn and roofs) else None),
            "violation_fraction_mean": [float(c[:, i].mean() / (H - w + 1)) for i, w in enumerate(windows)],
            "peak_fraction_of_nameplate_max": [float(p[:, i].max() / (64.0 * w) / W.FLEET_NAMEPLATE_W)
                                               for i, w in enumerate(windows)],
            "traffic": load_traffic("fleet_windows_kernel"),
            "strategies": stagger}


def controlled_7b_traces(fw, tr):
    """Sec. 8 "job control": each single-GPU 7B job of the fleet replayed
    through the 7B env under the bench's trained controller, deterministic,
    in consecutive 500-step episodes (Sec. 4.4 replay); its actuated power
    (1/64 W, exact as watts) replaces the raw trace.  The controller's budget
    for a job keeps the 7B study's ratio of budget to full-timeline mean
    power (314.6 / 314.9 W, Sec. 6.1)."""
    import dataclasses
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    base = W.make_7b(seed=tr.seed)
    L = fw.traces.shape[1]
    T = base.env.episode_len
    offs = W.replay_offsets(L, T)
    out = fw.traces.copy()
    jobs7 = [j for j, (kind, gpus) in enumerate(W.FLEET_JOBS) if kind == "7B" and gpus == 1]
    for j in jobs7:
        g = int(np.nonzero(fw.job_of_gpu == j)[0][0])
        x = fw.traces[g]
        spec = dataclasses.replace(base.env, n_envs=len(offs), trace_len=L,
                                   budget_q=W.budget_q(float(x.astype(np.float64).mean()) * 314.6 / 314.9))
        env = pe.Env(spec, torch.from_numpy(np.ascontiguousarray(x.reshape(1, L))),
                     torch.zeros(L, dtype=torch.uint8))
        pe.set_offsets(env, torch.from_numpy(offs).cuda())
        buf = pe.alloc_rollout(spec, base.net, T)
        pe.rollout(env, base.net, tr.params, T, 0, buf, deterministic=True)
        q = buf["q"].cpu().numpy()
        series = x.copy()
        for k, o in enumerate(offs):
            series[o:o + T] = q[:, k].astype(np.float32) / np.float32(64.0)
        out[g] = series
        env.close()
    return out


def run_stagger(args, world, fw, traces, job, peaks_random, tr=None):
    """Sec. 8 fleet operating strategies on the same traces: naive aligned
    starts (composition 0), random starts (the other compositions) and the
    greedy phase-staggered schedule (pe_fleet_stagger over every
    stride-th offset, 30 s window), as 30 s peaks in kW and fractions of the
    6.4 kW nameplate; the greedy's time is reported as candidate
    window-samples/s."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    G, L = fw.traces.shape
    H, J, st, w = fw.horizon, fw.n_jobs, args.stagger_stride, 60
    off = torch.empty(J, dtype=torch.int32, device="cuda")
    pk = torch.empty(J, dtype=torch.int32, device="cuda")
    ws = torch.empty(pe.fleet_stagger_workspace_bytes(J, L, H, st), dtype=torch.uint8, device="cuda")
    pe.fleet_stagger(traces, job, J, H, w, st, off, pk, ws)
    torch.cuda.synchronize()
    barrier(world)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    pe.fleet_stagger(traces, job, J, H, w, st, off, pk, ws)
    b.record()
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b), world)
    ncand = (L + st - 1) // st
    cand_ws = J * ncand * (H - w + 1)
    kw = lambda v: float(v) / (64.0 * w) / 1e3  # noqa: E731  (peak window sum -> mean kW over the window)
    name = W.FLEET_NAMEPLATE_W / 1e3
    rnd = peaks_random[1:, 1] if peaks_random.shape[0] > 1 else peaks_random[:, 1]
    stag = kw(pk[-1].item())
    ctl = None
    if tr is not None:  # staggering combined with job-level control of the 7B jobs
        ctl_traces = torch.from_numpy(controlled_7b_traces(fw, tr)).cuda()
        pk2 = torch.empty_like(pk)
        off2 = torch.empty_like(off)
        pe.fleet_stagger(ctl_traces, job, J, H, w, st, off2, pk2, ws)
        ctl = kw(pk2[-1].item())
    return {"metric": "staggered-schedule candidate window-samples/s",
            "value": cand_ws * world / (ms / 1e3), "unit": "window-samples/s", "ms_per_call": ms,
            "config": {"stride": st, "window": w, "candidates_per_job": ncand, "jobs": J},
            "offsets": [int(x) for x in off.cpu()],
            "peak_30s_kw": {"naive_aligned": kw(peaks_random[0, 1]), "random_median": kw(np.median(rnd)),
                            "random_max": kw(rnd.max()), "phase_staggered": stag,
                            "staggered_with_job_control": ctl},
            "provisioning_fraction": {"naive_aligned": kw(peaks_random[0, 1]) / name,
                                      "random_median": kw(np.median(rnd)) / name,
                                      "phase_staggered": stag / name,
                                      "staggered_with_job_control": ctl / name if ctl else None}}


def run_72b_iteration(args, world, peaks, local, wl, env, params, buf, rws):
    """One whole 72B PPO iteration, timed with CUDA events and clock records:
    the rollout (65,536 envs x 1,024 steps), GAE and the full update (4 epochs
    x 1,024 minibatch steps of 65,536 samples), as the Stress leg times its
    iteration."""
    from paper_2608_11226_gb300 import pe
    net, ppo = wl.net, wl.ppo
    T, E = args.r72b_horizon, wl.env.n_envs
    N = T * E
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty_like(adv)
    m = torch.zeros_like(params)
    v = torch.zeros_like(params)
    stats = torch.zeros(8, device="cuda")
    pws = pe.alloc_workspace(pe.ppo_workspace_bytes(net, ppo, N))
    # warm-up of the update at this size: two minibatch steps
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    nw = 2 * ppo.minibatch
    wppo = type(ppo)(epochs=1, minibatch=ppo.minibatch, ent_coef=ppo.ent_coef)
    pe.ppo_update(net, wppo, params.clone(), m.clone(), v.clone(), 0, buf["obs"].view(-1, net.obs_dim)[:nw],
                  buf["act"].view(-1)[:nw], buf["logp"].view(-1)[:nw], adv.view(-1)[:nw], ret.view(-1)[:nw],
                  stats, pws, seed=7, iteration=0)
    torch.cuda.synchronize()
    barrier(world)
    clocks = ClockSampler(local)
    clocks.start()
    stream = torch.cuda.current_stream()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    ev[0].record(stream)
    pe.rollout(env, net, params, T, 50, buf, lam=1.0, workspace=rws)
    ev[1].record(stream)
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    ev[2].record(stream)
    pe.ppo_update(net, ppo, params, m, v, 0, buf["obs"], buf["act"], buf["logp"], adv, ret, stats, pws,
                  seed=7, iteration=1)
    ev[3].record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    pe.device_check()
    ph = [ev[i].elapsed_time(ev[i + 1]) for i in range(3)]
    total = max_over_ranks(sum(ph), world)
    steps = ppo.epochs * ((N + ppo.minibatch - 1) // ppo.minibatch)
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    ppo_flop = ppo_flops_per_sample(D, H, A) * N * ppo.epochs
    peak = float(peaks.get("bf16_tflops_sustained", 1725.0))
    ppo_tf = ppo_flop / (ph[2] / 1e3) / 1e12
    del pws, adv, ret
    torch.cuda.empty_cache()
    return {"metric": "72B PPO iteration env-steps/s", "value": N * world / (total / 1e3), "unit": "env-steps/s",
            "ms_per_iteration": total,
            "phases_ms": {"rollout": ph[0], "gae": ph[1], "ppo_update": ph[2]},
            "ppo_ms_per_minibatch_step": ph[2] / steps, "ppo_minibatch_steps": steps,
            "config": {"workload": f"72b: {E} envs x {T} steps, MLP 32-256-256 bf16 (tcgen05), GAE, "
                                   f"PPO {ppo.epochs} epochs x minibatch {ppo.minibatch} ({steps} minibatch steps)",
                       "timed": "one iteration after the rollout and update legs; inputs larger than L2"},
            "roofline": {"kernel": "bf16 PPO update (all its kernels)", "bound": "tensor", "achieved": ppo_tf,
                         "peak": peak, "unit": "TFLOP/s", "frac": ppo_tf / peak, "flop": ppo_flop,
                         "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained"},
            "clocks": clk}


def run_72b(args, world, peaks, local=0):
    """The 72B workload's rollout (65,536 envs x 1,024 steps, bf16 32-256-256
    policy/value MLPs on the tcgen05 tensor cores, 4 channels, Eq. 6 reward),
    timed the same way; reports env-steps/s and the tensor-core MLP kernel's
    achieved bf16 TFLOP/s against the measured sustained bf16 peak."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    wl = W.make_72b(n_envs=args.r72b_envs, seed=0)
    spec, net = wl.env, wl.net
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    T, E = args.r72b_horizon, spec.n_envs
    buf = pe.alloc_rollout(spec, net, T)
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    ws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net))
    pe.rollout(env, net, params, T, 0, buf, lam=1.0, workspace=ws)
    pe.device_check()
    for k in range(pe.PE_PROF_KINDS):
        pe.profile_read(k)
    barrier(world)
    # whole rollouts timed with the per-launch event profiler off (its event
    # pairs around ~2,050 launches would add to the rollout's time) ...
    stream = torch.cuda.current_stream()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for it in range(args.r72b_steps):
        pe.rollout(env, net, params, T, it + 1, buf, lam=1.0, workspace=ws)
    b.record(stream)
    torch.cuda.synchronize()
    pe.device_check()
    ms = max_over_ranks(a.elapsed_time(b), world) / args.r72b_steps
    # ... and one more rollout with it on, for the per-kernel device times
    pe.profile_enable(True)
    pe.rollout(env, net, params, T, args.r72b_steps + 1, buf, lam=1.0, workspace=ws)
    torch.cuda.synchronize()
    pe.profile_enable(False)
    pe.device_check()
    prof = {pe.profile_kind_name(k): pe.profile_read(k) for k in range(pe.PE_PROF_KINDS)}
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    pol_flop_all = 2.0 * T * E * (D * H + H * H + H * A)  # every policy launch of one rollout
    val_flop = 2.0 * (T + 1) * E * (D * H + H * H + H)   # the value launches of one rollout
    # GAE over the 72B rollout buffer (T*E = 67M env-steps, 1.14 GB of algorithmic traffic)
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty_like(adv)
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    pe.profile_read(pe.PE_PROF_GAE)
    pe.profile_enable(True)
    for _ in range(3):
        pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    pe.profile_enable(False)
    gms, gn = pe.profile_read(pe.PE_PROF_GAE)
    gae_gbs = 17.0 * T * E / (gms / gn / 1e3) / 1e9 if gn else None
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    ppo72 = run_72b_ppo(args, world, peaks, wl, buf, adv, ret) if args.r72b_ppo_minibatches > 0 else None
    # the Eq. 7 outer loop: lambda fed back from each rollout's 30 s violation rate (target 8%)
    lam_dev = torch.tensor([1.0], device="cuda")
    rate_dev = torch.zeros(1, device="cuda")
    dual = []
    for it in range(3):
        lam_h = float(lam_dev.item())
        pe.rollout(env, net, params, T, 10 + it, buf, lam=lam_h, workspace=ws)
        pe.dual_ascent(buf["viol"], T, lam_dev, rate_dev, target=0.08)
        dual.append({"lambda_in": lam_h, "violation_rate_30s": float(rate_dev.item()),
                     "lambda_out": float(lam_dev.item())})
    del adv, ret
    pms, pn = prof["mlp_policy_tc"]
    vms, vn = prof["mlp_value_tc"]
    peak = float(peaks.get("bf16_tflops_sustained", 1728.9))
    # the policy runs as two chains of E/2-row launches on two streams: the
    # sum of the launches' event times counts time shared with the other
    # chain's env steps, so this figure is a lower bound
    pol = pol_flop_all / (pms / 1e3) / 1e12 if pn else None
    val = val_flop / (vms / 1e3) / 1e12 if vn else None
    it72 = run_72b_iteration(args, world, peaks, local, wl, env, params, buf, ws)
    env.close()
    return {"metric": "72B rollout env-steps/s", "value": E * T * world / (ms / 1e3),
            "unit": "env-steps/s", "ms_per_rollout": ms,
            "config": {"workload": f"72b: {E} envs x {T} steps, 4-channel 22,000-sample trace, "
                                   "16 levels, MLP 32-256-256 bf16 (tcgen05), value on all T*E obs",
                       "n_envs": E, "horizon": T},
            "kernels": {k: {"ms_per_rollout": v[0], "launches_per_rollout": v[1]} for k, v in prof.items() if v[1]},
            "roofline_policy_mlp": {"kernel": f"mlp_bf16_pair_kernel (policy, {pn // max(T, 1)} launches per "
                                              f"step over {E} rows)", "bound": "tensor",
                                    "achieved": pol, "peak": peak, "unit": "TFLOP/s",
                                    "frac": pol / peak if pol else None,
                                    "avg_launch_ms": pms / pn if pn else None,
                                    "traffic": load_traffic("mlp_bf16_pair_kernel")},
            "roofline_value_mlp": {"kernel": "mlp_bf16_pair_kernel (value, T*E rows)", "bound": "tensor",
                                   "achieved": val, "peak": peak, "unit": "TFLOP/s",
                                   "frac": val / peak if val else None},
            "roofline_gae": {"kernel": f"{gae_kernel_name(E)} ({T} x {E})", "bound": "hbm", "achieved": gae_gbs,
                             "peak": hbm, "unit": "GB/s", "frac": gae_gbs / hbm if gae_gbs else None,
                             "avg_launch_ms": gms / gn if gn else None,
                             "traffic": gae_traffic(T * E, E)},
            "ppo_update": ppo72, "dual_ascent_eq7": dual,
            "iteration": it72,
            "cadence": run_72b_cadence(args, world),
            "mixed_families": run_72b_mixed(args, world)}


def run_72b_cadence(args, world):
    """The 72B env at the Sec. 4.5 batch cadence (a step is one generation
    batch of 24-42 samples): 65,536 envs x 64 batch steps on the tcgen05
    policy; reports batch-steps/s and the trace samples consumed per second."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    wl = W.make_72b_cadence(n_envs=args.r72b_envs)
    spec, net = wl.env, wl.net
    T = 64
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    ws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net))
    pe.rollout(env, net, params, T, 0, buf, lam=1.0, workspace=ws)
    torch.cuda.synchronize()
    barrier(world)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    pe.rollout(env, net, params, T, 1, buf, lam=1.0, workspace=ws)
    b.record()
    torch.cuda.synchronize()
    pe.device_check()
    ms = max_over_ranks(a.elapsed_time(b), world)
    samples = int(buf["samples"].sum())
    env.close()
    return {"metric": "72B batch-cadence rollout steps/s", "value": spec.n_envs * T * world / (ms / 1e3),
            "unit": "batch-steps/s", "samples_per_s": samples * world / (ms / 1e3), "ms_per_rollout": ms,
            "mean_samples_per_step": samples / (spec.n_envs * T),
            "config": {"workload": f"72b cadence: {spec.n_envs} envs x {T} batch steps of 24-42 samples, "
                                   "40-batch episodes, MLP 32-256-256 bf16"}}


def run_72b_mixed(args, world):
    """Domain randomisation (Sec. 4.2 G2): the 72B env drawing every episode
    from a 72B-, 14B- or 7B-shaped trace family (own channel count and
    budget), 65,536 envs x 1,024 steps on the tcgen05 policy."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    wl = W.make_72b_mixed(n_envs=args.r72b_envs)
    spec, net = wl.env, wl.net
    T = args.r72b_horizon
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    ws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net))
    pe.rollout(env, net, params, T, 0, buf, lam=1.0, workspace=ws)
    torch.cuda.synchronize()
    barrier(world)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    pe.rollout(env, net, params, T, 1, buf, lam=1.0, workspace=ws)
    b.record()
    torch.cuda.synchronize()
    pe.device_check()
    ms = max_over_ranks(a.elapsed_time(b), world)
    v = buf["viol"].sum(0).cpu().numpy()
    n = spec.n_envs * T
    env.close()
    return {"metric": "72B mixed-family rollout env-steps/s", "value": n * world / (ms / 1e3),
            "unit": "env-steps/s", "ms_per_rollout": ms,
            "violation_rate_30s": float(v[1]) / n,
            "config": {"workload": f"72b mixed families: {spec.n_envs} envs x {T} steps, episodes drawn from "
                                   "72B-/14B-/7B-shaped traces (4/2/1 GPUs, own budgets), MLP 32-256-256 bf16"}}


def run_72b_ppo(args, world, peaks, wl, buf, adv, ret):
    """bf16 PPO update of the 72B networks on the first K x 65,536 samples of
    the 72B rollout (one epoch, K minibatch steps): tensor-core forward over
    the permuted rows, tensor-core backward products, own loss/reduction/Adam.
    Reports samples/s and the whole step's bf16 FLOP rate against the
    measured sustained bf16 peak."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    net = wl.net
    mb = 65536
    n = min(args.r72b_ppo_minibatches * mb, buf["act"].numel())
    ppo = W.PPOSpec(epochs=1, minibatch=mb, ent_coef=0.01)
    D = net.obs_dim
    obs = buf["obs"].view(-1, D)[:n]
    act = buf["act"].view(-1)[:n]
    lpo = buf["logp"].view(-1)[:n]
    a_ = adv.view(-1)[:n]
    r_ = ret.view(-1)[:n]
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    m = torch.zeros_like(params)
    v = torch.zeros_like(params)
    stats = torch.zeros(8, device="cuda")
    ws = pe.alloc_workspace(pe.ppo_workspace_bytes(net, ppo, n))
    pe.ppo_update(net, ppo, params, m, v, 0, obs, act, lpo, a_, r_, stats, ws, seed=7, iteration=0)
    torch.cuda.synchronize()
    for k in range(pe.PE_PROF_KINDS):
        pe.profile_read(k)
    barrier(world)
    # timed with the per-launch event profiler off, then one more update with
    # it on for the per-kernel device times
    stream = torch.cuda.current_stream()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    pe.ppo_update(net, ppo, params, m, v, 1, obs, act, lpo, a_, r_, stats, ws, seed=7, iteration=1)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1), world)
    st = [float(x) for x in stats.cpu()]
    pe.profile_enable(True)
    pe.ppo_update(net, ppo, params, m, v, 2, obs, act, lpo, a_, r_, stats, ws, seed=7, iteration=2)
    torch.cuda.synchronize()
    pe.profile_enable(False)
    prof = {pe.profile_kind_name(k): pe.profile_read(k) for k in range(pe.PE_PROF_KINDS)}
    steps = (n + mb - 1) // mb
    fl = ppo_flops_per_sample(net.obs_dim, net.hidden, net.n_actions) * n
    peak = float(peaks.get("bf16_tflops_sustained", 1728.9))
    ach = fl / (ms / 1e3) / 1e12
    del ws
    return {"metric": "72B PPO update samples/s", "value": n * world / (ms / 1e3), "unit": "samples/s",
            "ms_per_minibatch_step": ms / steps, "minibatch": mb, "steps": steps,
            "kernels": {k: {"ms_per_step": v_[0] / steps, "launches_per_step": v_[1] / steps}
                        for k, v_ in prof.items() if v_[1]},
            "roofline": {"kernel": "bf16 PPO minibatch step (all kernels)", "bound": "tensor",
                         "achieved": ach, "peak": peak, "unit": "TFLOP/s", "frac": ach / peak,
                         "flop_per_sample": ppo_flops_per_sample(net.obs_dim, net.hidden, net.n_actions)},
            "stats": st}


def run_tiny(args, world):
    """One PPO iteration of the Tiny workload (64 envs x 128 steps, fp32
    8-64-64, PPO 4 epochs over one minibatch of the whole rollout), 10 timed
    iterations after 3 warm-up ones."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    wl = W.make_tiny()
    spec, net = wl.env, wl.net
    T, E = wl.horizon, spec.n_envs
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    m = torch.zeros_like(params)
    v = torch.zeros_like(params)
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty_like(adv)
    stats = torch.zeros(8, device="cuda")
    ppo = W.PPOSpec(epochs=4, minibatch=T * E)
    ws = pe.alloc_workspace(pe.ppo_workspace_bytes(net, ppo, T * E))

    def it(k):
        pe.rollout(env, net, params, T, k, buf)
        pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
        pe.ppo_update(net, ppo, params, m, v, 4 * k, buf["obs"], buf["act"], buf["logp"], adv, ret, stats,
                      ws, seed=7, iteration=k)
    for k in range(3):
        it(k)
    torch.cuda.synchronize()
    barrier(world)
    stream = torch.cuda.current_stream()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for k in range(3, 13):
        it(k)
    b.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b), world) / 10
    env.close()
    return {"metric": "Tiny PPO iteration env-steps/s", "value": T * E * world / (ms / 1e3),
            "unit": "env-steps/s", "ms_per_iteration": ms,
            "config": {"workload": "tiny: 64 envs x 128 steps, 4,000-sample trace, 3 actions, MLP 8-64-64 "
                                   "fp32, GAE, PPO 4 epochs x one 8,192-sample minibatch"}}


def run_stress(args, world, peaks, local):
    """One full iteration of the Stress configuration, timed once after a
    short warm-up of each kernel: the rollout of 262,144 envs x 2,048 steps
    over a 4 x 380,000-sample trace (bf16 64-512-512 policy on the tcgen05
    tensor cores with streamed weights, then the value network on every
    observation), GAE, the full PPO update (4 epochs x minibatch 65,536 =
    32,768 minibatch steps), and the fleet windows recomputed at
    --stress-fleet-n compositions.  Reports env-steps/s of the iteration,
    the phase times and the bf16 FLOP rate of the update against the
    measured sustained peak."""
    from paper_2608_11226_gb300 import pe
    from paper_2608_11226_gb300 import workloads as W
    E, T = args.stress
    wl = W.make_stress(n_envs=E, horizon=T)
    spec, net, ppo = wl.env, wl.net, wl.ppo
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    buf["q"] = None
    N = T * E
    params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
    m = torch.zeros_like(params)
    v = torch.zeros_like(params)
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty_like(adv)
    stats = torch.zeros(8, device="cuda")
    rws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net))
    pws = pe.alloc_workspace(pe.ppo_workspace_bytes(net, ppo, N))
    fw = W.make_fleet(n_compositions=args.stress_fleet_n)
    ftr = torch.from_numpy(fw.traces).cuda()
    fjob = torch.from_numpy(fw.job_of_gpu).cuda()
    foff = torch.from_numpy(fw.offsets).cuda()
    fcnt = torch.empty((foff.shape[0], 3), dtype=torch.int32, device="cuda")
    fpk = torch.empty_like(fcnt)
    fws = pe.alloc_workspace(pe.fleet_workspace_bytes(fw.n_jobs, ftr.shape[1], fw.horizon))
    # warm-up: a 4-step rollout, GAE, 2 minibatch steps of the update, one fleet call
    pe.rollout(env, net, params, 4, 0, buf, lam=1.0, workspace=rws)
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    wppo = W.PPOSpec(epochs=1, minibatch=ppo.minibatch, ent_coef=ppo.ent_coef)
    nw = 2 * ppo.minibatch
    pe.ppo_update(net, wppo, params.clone(), m.clone(), v.clone(), 0, buf["obs"].view(-1, net.obs_dim)[:nw],
                  buf["act"].view(-1)[:nw], buf["logp"].view(-1)[:nw], adv.view(-1)[:nw], ret.view(-1)[:nw],
                  stats, pws, seed=7, iteration=0)
    pe.fleet_windows(ftr, fjob, fw.n_jobs, foff, fw.horizon, [1, 60, 600], fw.budget_q, fcnt, fpk, fws)
    torch.cuda.synchronize()
    pe.device_check()
    barrier(world)
    clocks = ClockSampler(local)
    clocks.start()
    stream = torch.cuda.current_stream()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    ev[0].record(stream)
    pe.rollout(env, net, params, T, 1, buf, lam=1.0, workspace=rws)
    ev[1].record(stream)
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
    ev[2].record(stream)
    pe.ppo_update(net, ppo, params, m, v, 0, buf["obs"], buf["act"], buf["logp"], adv, ret, stats, pws,
                  seed=7, iteration=1)
    ev[3].record(stream)
    pe.fleet_windows(ftr, fjob, fw.n_jobs, foff, fw.horizon, [1, 60, 600], fw.budget_q, fcnt, fpk, fws)
    ev[4].record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    pe.device_check()
    ph = [ev[i].elapsed_time(ev[i + 1]) for i in range(4)]
    total = max_over_ranks(sum(ph), world)
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    steps = ppo.epochs * ((N + ppo.minibatch - 1) // ppo.minibatch)
    ppo_flop = ppo_flops_per_sample(D, H, A) * N * ppo.epochs
    roll_flop = 2.0 * N * (D * H + H * H + H * A) + 2.0 * (N + E) * (D * H + H * H + H)
    peak = float(peaks.get("bf16_tflops_sustained", 1725.0))
    ppo_tf = ppo_flop / (ph[2] / 1e3) / 1e12
    roll_tf = roll_flop / (ph[0] / 1e3) / 1e12
    st = [float(x) for x in stats.cpu()]
    out = {"metric": "Stress PPO iteration env-steps/s", "value": N * world / (total / 1e3), "unit": "env-steps/s",
           "ms_per_iteration": total,
           "phases_ms": {"rollout": ph[0], "gae": ph[1], "ppo_update": ph[2], "fleet_windows": ph[3]},
           "config": {"workload": f"stress: {E} envs x {T} steps over a 4 x 380,000-sample 72B-shaped trace, "
                                  "16 levels, MLP 64-512-512 bf16 (tcgen05, streamed weights), GAE, PPO 4 epochs x "
                                  f"minibatch 65,536 ({steps} minibatch steps), fleet windows at "
                                  f"{foff.shape[0]} compositions", "n_envs": E, "horizon": T,
                      "timed": "one iteration after a short warm-up of each kernel; inputs larger than L2"},
           "roofline": {"kernel": "bf16 PPO update (all its kernels)", "bound": "tensor", "achieved": ppo_tf,
                        "peak": peak, "unit": "TFLOP/s", "frac": ppo_tf / peak,
                        "flop": ppo_flop, "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained"},
           "roofline_rollout_mlp": {"kernel": "rollout (policy + value MLP on tcgen05, env step)", "bound": "tensor",
                                    "achieved": roll_tf, "peak": peak, "unit": "TFLOP/s", "frac": roll_tf / peak},
           "gae_gbs": 17.0 * N / (ph[1] / 1e3) / 1e9,
           "fleet_window_samples_per_s": sum(foff.shape[0] * (fw.horizon - w + 1) for w in (1, 60, 600)) / (ph[3] / 1e3),
           "ppo_stats": st, "clocks": clk}
    env.close()
    del buf, adv, ret, pws, rws
    torch.cuda.empty_cache()
    return out


def per_config_table(out):
    """Per configuration: the GPU figure of this run, its roofline fraction,
    and the CPU oracle on 1 core and on all host cores (process-sharded,
    bounded samples; "extrapolated" where the sample is smaller than the
    configuration)."""
    from oracle import cpu_rate
    cpu = cpu_rate.rates()
    r72 = out.get("rollout_72b") or {}
    gpu = {
        "tiny": ((out.get("tiny_iteration") or {}).get("value"), None, "PPO iteration env-steps/s"),
        "7b": (out["value"], (out.get("roofline") or {}).get("frac"), "PPO iteration env-steps/s"),
        "72b": ((r72.get("iteration") or {}).get("value"),
                ((r72.get("iteration") or {}).get("roofline") or {}).get("frac"),
                "PPO iteration env-steps/s (update tensor fraction)"),
        "stress": ((out.get("stress_iteration") or {}).get("value"),
                   ((out.get("stress_iteration") or {}).get("roofline") or {}).get("frac"),
                   "PPO iteration env-steps/s (update tensor fraction)"),
        "fleet": ((out.get("fleet") or {}).get("value"),
                  ((out.get("fleet") or {}).get("roofline") or {}).get("frac"),
                  "window-samples/s (logical L2 fraction)"),
    }
    return {k: {"gpu": gpu[k][0], "gpu_metric": gpu[k][2], "roofline_frac": gpu[k][1], **cpu[k]} for k in cpu}


def gae_kernel_name(E: int) -> str:
    """The GAE kernel the library picks for a batch of E envs (its dispatch
    by width): streamed per env column for wide batches, chunked below."""
    if E >= 196608 and E % 4 == 0:
        return "gae_stream_kernel<4, 8>"
    if E >= 49152:
        return "gae_stream_kernel<1, 16>"
    if E >= 32768:
        return "gae_stream_kernel<1, 32>"
    return "gae_kernel_v (chunked)"


def gae_traffic(env_steps: int, E: int):
    """DRAM bytes of one GAE launch larger than L2, scaled from the committed
    capture's bytes per env-step of the same kernel."""
    key = "traffic_bytes_per_env_step_v4" if E >= 196608 and E % 4 == 0 else "traffic_bytes_per_env_step_v1"
    b = load_traffic_per_unit("gae_stream_kernel", key) if E >= 32768 else None
    return None if b is None else b * env_steps


def run_gae_large(args, world, peaks):
    """GAE alone at the Stress size (2,048 x 262,144 env-steps, 9.1 GB of
    algorithmic traffic), on seeded device-resident inputs."""
    from paper_2608_11226_gb300 import pe
    T, E = args.gae_large
    g = torch.Generator(device="cuda").manual_seed(0)
    r = torch.randn(T, E, device="cuda", generator=g)
    v = torch.randn(T, E, device="cuda", generator=g)
    d = (torch.rand(T, E, device="cuda", generator=g) < 0.002).to(torch.uint8)
    lv = torch.randn(E, device="cuda", generator=g)
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty_like(adv)
    pe.gae(r, v, d, lv, 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    pe.profile_read(pe.PE_PROF_GAE)
    barrier(world)
    pe.profile_enable(True)
    for _ in range(5):
        pe.gae(r, v, d, lv, 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    pe.profile_enable(False)
    gms, gn = pe.profile_read(pe.PE_PROF_GAE)
    ms = max_over_ranks(gms / gn, world)
    gbs = 17.0 * T * E / (ms / 1e3) / 1e9
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    del r, v, d, adv, ret
    torch.cuda.empty_cache()
    return {"kernel": f"{gae_kernel_name(E)} ({T} x {E})", "bound": "hbm", "achieved": gbs, "peak": hbm,
            "unit": "GB/s", "frac": gbs / hbm, "avg_launch_ms": ms,
            "env_steps_per_s": T * E * world / (ms / 1e3), "traffic": gae_traffic(T * E, E)}


# --------------------------------------------------------------------------- CPU oracle
def oracle_iteration(n_envs: int, seed: int = 0, iteration: int = 0):
    """One PPO iteration of the 7B workload on a sample of n_envs envs, by the
    CPU oracle (rollout, value, GAE, PPO update with the minibatch scaled by
    n_envs / 4096 so that the update takes the same 256 minibatch steps)."""
    import oracle as O
    from paper_2608_11226_gb300 import workloads as W
    wl = W.make_7b(seed=seed)
    net = wl.net
    params = W.init_params(net, seed=seed)
    env = O.OracleEnv(wl.env, wl.trace, wl.phase, np.arange(n_envs))
    T = wl.horizon
    t0 = time.perf_counter()
    o = env.rollout(params, net.hidden, False, T, iteration)
    _, v = O.mlp_forward(net, params, o["obs"].reshape(-1, net.obs_dim))
    _, lv = O.mlp_forward(net, params, o["obs_last"])
    adv, ret = O.gae(o["reward"].astype(np.float32), v.reshape(T, n_envs).astype(np.float32),
                     o["done"], lv.astype(np.float32), wl.ppo.gamma, wl.ppo.lam)
    mb = max(1, wl.ppo.minibatch * n_envs // wl.env.n_envs)
    ppo = W.PPOSpec(epochs=wl.ppo.epochs, minibatch=mb)
    P = params.size
    O.ppo_update(net, ppo, params, np.zeros(P), np.zeros(P), 0, o["obs"].reshape(-1, net.obs_dim),
                 o["act_own"].ravel(), o["logp"].astype(np.float32).ravel(),
                 adv.astype(np.float32).ravel(), ret.astype(np.float32).ravel(), 7, iteration)
    return time.perf_counter() - t0, n_envs * T


def cpu_baseline(n_envs: int):
    import oracle as O
    O.build()
    dt, steps = oracle_iteration(n_envs)
    return {"value": steps / dt, "unit": "env-steps/s", "cores": 1, "kind": "oracle",
            "sample": f"one PPO iteration of the 7b workload on {n_envs} of 4096 envs "
                      f"(512 steps each, minibatch scaled to keep 256 minibatch steps); {dt:.1f} s"}


def run_reference(args, world, rank):
    if rank != 0:
        return
    import oracle as O
    O.build()
    n = max(1, args.cpu_envs // 3)
    for _ in range(args.warmup):
        oracle_iteration(n)
    tot = 0.0
    steps = 0
    for k in range(args.steps):
        dt, s = oracle_iteration(n, iteration=k)
        tot += dt
        steps += s
    value = steps / tot
    out = {"metric": METRIC, "value": value, "unit": "env-steps/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot / args.steps * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": "7b: 4096 envs x 512 steps on a 60,000-sample 7B-GRPO-shaped "
                                  "trace, 5 actions, MLP 16-128-128 fp32, GAE, PPO 4 epochs x "
                                  "minibatch 8192", "sample_envs": n},
           "cpu_baseline": {"value": value, "unit": "env-steps/s", "cores": 1, "kind": "oracle",
                            "sample": f"{n} of 4096 envs per step, minibatch scaled to keep 256 "
                                      "minibatch steps"},
           "e2e": {"value": value, "unit": "env-steps/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def run_ncu_case(name: str):
    """Small cases of the hot kernels, sized for ncu captures (a few GB on the
    device at most, inputs larger than L2 where DRAM figures matter); each
    runs its kernel a few times and exits."""
    from paper_2608_11226_gb300 import build, pe
    from paper_2608_11226_gb300 import workloads as W
    build.build()
    pe.lib()
    if name in ("ppo7b", "ppo72", "ppostress"):
        # rollout (32, 16 or 4 steps), GAE, then 3 PPO updates of one epoch (16 minibatch steps each)
        wl = (W.make_7b() if name == "ppo7b" else W.make_72b(n_envs=65536) if name == "ppo72"
              else W.make_stress(n_envs=262144, horizon=4))
        spec, net = wl.env, wl.net
        T = {"ppo7b": 32, "ppo72": 16, "ppostress": 4}[name]
        mb = 8192 if name == "ppo7b" else 65536
        env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
        buf = pe.alloc_rollout(spec, net, T)
        params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
        pe.rollout(env, net, params, T, 0, buf, lam=1.0)
        adv = torch.empty(T, spec.n_envs, device="cuda")
        ret = torch.empty_like(adv)
        pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], 0.99, 0.95, adv, ret)
        ppo = W.PPOSpec(epochs=1, minibatch=mb, ent_coef=wl.ppo.ent_coef)
        m = torch.zeros_like(params)
        v = torch.zeros_like(params)
        st = torch.zeros(8, device="cuda")
        ws = pe.alloc_workspace(pe.ppo_workspace_bytes(net, ppo, buf["act"].numel()))
        steps = (buf["act"].numel() + mb - 1) // mb
        for it in range(3):
            pe.ppo_update(net, ppo, params, m, v, it * steps, buf["obs"], buf["act"], buf["logp"], adv, ret,
                          st, ws, seed=7, iteration=it)
        env.close()
    elif name == "gae-chunked":
        # the chunked kernel of narrower batches: 2,048 x 16,384 (570 MB of
        # algorithmic traffic, more than L2)
        T, E = 2048, 16384
        g = torch.Generator(device="cuda").manual_seed(0)
        r = torch.randn(T, E, device="cuda", generator=g)
        v = torch.randn(T, E, device="cuda", generator=g)
        d = (torch.rand(T, E, device="cuda", generator=g) < 0.002).to(torch.uint8)
        lv = torch.randn(E, device="cuda", generator=g)
        adv = torch.empty(T, E, device="cuda")
        ret = torch.empty_like(adv)
        for _ in range(3):
            pe.gae(r, v, d, lv, 0.99, 0.95, adv, ret)
    elif name == "gae":
        # the two streamed launch shapes: 1,024 x 65,536 (one env per thread,
        # the 72B rollout's shape, 1.1 GB of algorithmic traffic) and
        # 512 x 262,144 (four envs per thread, the Stress width, 2.3 GB)
        for T, E in ((1024, 65536), (512, 262144)):
            g = torch.Generator(device="cuda").manual_seed(0)
            r = torch.randn(T, E, device="cuda", generator=g)
            v = torch.randn(T, E, device="cuda", generator=g)
            d = (torch.rand(T, E, device="cuda", generator=g) < 0.002).to(torch.uint8)
            lv = torch.randn(E, device="cuda", generator=g)
            adv = torch.empty(T, E, device="cuda")
            ret = torch.empty_like(adv)
            for _ in range(3):
                pe.gae(r, v, d, lv, 0.99, 0.95, adv, ret)
            del r, v, d, lv, adv, ret
    elif name == "mlp72":
        # two 72B rollouts of 8 steps over 65,536 envs: 8 policy + 2 value launches each
        wl = W.make_72b(n_envs=65536)
        spec, net = wl.env, wl.net
        T = 8
        env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
        buf = pe.alloc_rollout(spec, net, T)
        params = torch.from_numpy(W.init_params(net, seed=0)).cuda()
        ws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net))
        for it in range(2):
            pe.rollout(env, net, params, T, it, buf, lam=1.0, workspace=ws)
        pe.device_check()
        env.close()
    elif name == "fleet":
        wl = W.make_fleet(n_compositions=20000)
        tr = torch.from_numpy(wl.traces).cuda()
        jg = torch.from_numpy(wl.job_of_gpu).cuda()
        off = torch.from_numpy(wl.offsets).cuda()
        cnt = torch.empty(off.shape[0], len(wl.windows), dtype=torch.int32, device="cuda")
        pk = torch.empty_like(cnt)
        ws = pe.alloc_workspace(pe.fleet_workspace_bytes(wl.n_jobs, tr.shape[1], wl.horizon))
        for _ in range(2):
            pe.fleet_windows(tr, jg, wl.n_jobs, off, wl.horizon, wl.windows, wl.budget_q, cnt, pk, ws)
    torch.cuda.synchronize()
    print(json.dumps({"ncu_case": name, "ok": True}), flush=True)


def main():
    args = parse()
    if args.ncu_case:
        run_ncu_case(args.ncu_case)
        return
    if args.impl == "reference":
        world = int(os.environ.get("WORLD_SIZE", "1"))
        rank = int(os.environ.get("RANK", "0"))
        run_reference(args, world, rank)
        return
    world, rank, local = dist_setup()
    run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
