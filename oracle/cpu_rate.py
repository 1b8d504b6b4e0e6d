"""Throughput of the CPU oracle, as it stands, on bounded samples of the
benchmark workloads -- TEST INFRASTRUCTURE, used only by the benchmark's
CPU-baseline leg.

A sample is one PPO iteration (rollout with the policy, the value network
on every observation, GAE, and the PPO update over the sample's own
env-steps) of n envs over T steps, or n fleet compositions.  The oracle's
cost is linear in env-steps (and in compositions), so the rate of a sample
is the rate of the whole configuration; configurations larger than the
sample are marked "extrapolated".  The all-cores figure runs one sample per
host core in independent processes (a spawn pool: each process its own env
ids and its own update), the process-sharded reading of the oracle.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import time
from typing import Dict, Tuple

import numpy as np

# name -> (workload maker, sample envs, sample steps); full sizes in the docstrings of workloads.py
SAMPLES = {
    "tiny": ("make_tiny", 64, 128),
    "7b": ("make_7b", 8, 512),
    "72b": ("make_72b", 2, 256),
    "stress": ("make_stress", 1, 128),
}
FLEET_SAMPLE = 60  # compositions


def _workload(name: str, n_envs: int):
    from paper_2608_11226_gb300 import workloads as W
    maker, _, T = SAMPLES[name]
    wl = getattr(W, maker)(n_envs=n_envs)
    return wl, T


def iteration_sample(name: str, first_env: int = 0) -> Tuple[float, int]:
    """(seconds, env-steps) of one oracle PPO iteration on the named sample."""
    import oracle as O
    from paper_2608_11226_gb300 import workloads as W
    _, n, _ = SAMPLES[name]
    wl, T = _workload(name, n + first_env)
    net = wl.net
    bf16 = net.dtype == 1
    params = W.init_params(net, seed=0)
    env = O.OracleEnv(wl.env, wl.trace, wl.phase, np.arange(first_env, first_env + n))
    t0 = time.perf_counter()
    o = env.rollout(params, net.hidden, bf16, T, 0)
    _, v = O.mlp_forward(net, params, o["obs"].reshape(-1, net.obs_dim))
    _, lv = O.mlp_forward(net, params, o["obs_last"])
    adv, ret = O.gae(o["reward"].astype(np.float32), v.reshape(T, n).astype(np.float32), o["done"],
                     lv.astype(np.float32), wl.ppo.gamma, wl.ppo.lam)
    N = n * T
    ppo = W.PPOSpec(epochs=wl.ppo.epochs, minibatch=max(1, N // 4), ent_coef=wl.ppo.ent_coef)
    P = params.size
    O.ppo_update(net, ppo, params, np.zeros(P), np.zeros(P), 0, o["obs"].reshape(-1, net.obs_dim),
                 o["act_own"].ravel(), o["logp"].astype(np.float32).ravel(),
                 adv.astype(np.float32).ravel(), ret.astype(np.float32).ravel(), 7, 0)
    return time.perf_counter() - t0, N


def fleet_sample(first: int = 0) -> Tuple[float, float]:
    """(seconds, window-samples) of the oracle fleet windows over FLEET_SAMPLE
    compositions of the full fleet (16 traces x 380,000 samples, windows
    1/60/600)."""
    import oracle as O
    from paper_2608_11226_gb300 import workloads as W
    fw = W.make_fleet(n_compositions=first + FLEET_SAMPLE)
    off = np.ascontiguousarray(fw.offsets[first:first + FLEET_SAMPLE])
    t0 = time.perf_counter()
    O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, off, fw.horizon, fw.windows, fw.budget_q)
    dt = time.perf_counter() - t0
    ws = float(sum(fw.horizon - int(w) + 1 for w in fw.windows)) * FLEET_SAMPLE
    return dt, ws


def _worker(job):
    name, k = job
    if name == "fleet":
        return fleet_sample(first=k * FLEET_SAMPLE)
    _, n, _ = SAMPLES[name]
    return iteration_sample(name, first_env=k * n)


def rates(names=("tiny", "7b", "72b", "stress", "fleet"), cores: int = 0) -> Dict[str, dict]:
    """Per name: 1-core rate, all-cores rate (one sample per core, the
    slowest worker's time), the core count and the sample description."""
    import oracle as O
    O.build()
    cores = cores or os.cpu_count() or 1
    out = {}
    ctx = mp.get_context("spawn")
    with ctx.Pool(cores) as pool:
        pool.map(_noop, range(cores))  # start every worker before timing
        for name in names:
            dt, units = _worker((name, 0))
            res = pool.map(_worker, [(name, k) for k in range(cores)])
            worst = max(r[0] for r in res)
            total = sum(r[1] for r in res)
            if name == "fleet":
                sample = f"{FLEET_SAMPLE} compositions of 16 x 380,000 samples, windows 1/60/600"
                unit = "window-samples/s"
            else:
                _, n, T = SAMPLES[name]
                sample = f"one PPO iteration of {n} envs x {T} steps (minibatch = a quarter of the sample)"
                unit = "env-steps/s"
            out[name] = {"cpu_1core": units / dt, "cpu_all_cores": total / worst, "cores": cores,
                         "unit": unit, "sample": sample, "sample_s_1core": dt,
                         "extrapolated": name != "tiny"}
    return out


def _noop(_):
    return 0
