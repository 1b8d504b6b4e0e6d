"""ctypes front end of the CPU oracle -- TEST INFRASTRUCTURE.

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's
CPU-baseline leg may import this package.  The product path (the CUDA
library and its binding) never does.  ``build()`` compiles ``oracle.c`` with
gcc (-O2 -ffp-contract=off, single-threaded) into ``oracle/_build/``.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import Dict, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lib = None

MAX_LEVELS = 32
MAX_CH = 4


def build(force: bool = False) -> str:
    src = os.path.join(_HERE, "oracle.c")
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "oracle.h"))):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-std=c99", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
                               "-o", tmp, src, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class EnvCfg(C.Structure):
    _fields_ = [(n, C.c_int32) for n in (
        "n_envs", "n_channels", "trace_len", "n_actions", "obs_kind", "actuator_kind",
        "n_levels", "level_init", "g_min", "g_max", "b_min", "b_max", "b_init",
        "episode_len", "budget_q", "scale_phase_mask", "reward_kind", "reward_window")] + [
        ("r_ok", C.c_double), ("r_viol", C.c_double), ("bonus_coef", C.c_double),
        ("level_scale", (C.c_float * MAX_CH) * MAX_LEVELS),
        ("level_tokens", C.c_double * MAX_LEVELS),
        ("seed", C.c_uint64),
        ("level_samples", C.c_int32 * MAX_LEVELS),
        ("n_families", C.c_int32), ("fam_len", C.c_int32 * 4), ("fam_channels", C.c_int32 * 4),
        ("fam_budget_q", C.c_int32 * 4)]


class PPOCfg(C.Structure):
    _fields_ = [("epochs", C.c_int32), ("minibatch", C.c_int32)] + [
        (n, C.c_double) for n in ("lr", "clip", "vf_coef", "ent_coef", "max_grad_norm",
                                  "beta1", "beta2", "eps")]


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(_LIB_PATH)
        vp, i32, i64, u32, u64, f64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32, C.c_uint64, C.c_double
        sig = {
            "or_philox4x32_10": (None, [vp, vp, vp]),
            "or_feistel_index": (u32, [u64, vp, u64]),
            "or_perm_keys": (None, [u64, u32, u32, vp]),
            "or_bf16_round": (f64, [f64]),
            "or_env_state_size": (i32, []),
            "or_actuator_scale": (C.c_float, [vp, i32, i32]),
            "or_env_init": (i32, [vp, vp, vp, vp, i32, vp]),
            "or_env_set_offsets": (i32, [vp, vp, vp, vp, i32, vp]),
            "or_rollout_rule": (i32, [vp, vp, vp, vp, vp, i32, vp, i32, u32, f64, vp, vp, vp, vp,
                                      vp, vp, vp, vp, vp]),
            "or_env_obs": (None, [vp, vp, vp, vp, vp]),
            "or_mlp_forward": (None, [i32, i32, i32, i32, vp, i64, vp, vp, vp]),
            "or_rollout": (i32, [vp, vp, vp, vp, i32, i32, vp, i32, vp, i32, u32, f64, i32,
                                 vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]),
            "or_gae": (None, [i32, i32, vp, vp, vp, vp, f64, f64, vp, vp]),
            "or_ppo_minibatch_grad": (f64, [i32, i32, i32, vp, i64, vp, vp, vp, vp, vp,
                                            f64, f64, f64, vp, vp]),
            "or_ppo_update": (i64, [i32, i32, i32, vp, vp, vp, i64, i64, vp, vp, vp, vp, vp,
                                    vp, u64, u32, i64, vp]),
            "or_ppo_minibatch_grad_ex": (f64, [i32, i32, i32, i32, vp, i64, vp, vp, vp, vp, vp,
                                               f64, f64, f64, vp, vp]),
            "or_ppo_update_ex": (i64, [i32, i32, i32, i32, vp, vp, vp, i64, i64, vp, vp, vp, vp,
                                       vp, vp, u64, u32, i64, vp]),
            "or_fleet_windows": (i32, [i32, i32, vp, vp, i32, vp, i64, i32, vp, i32, i64,
                                       vp, vp]),
            "or_fleet_stagger": (i32, [i32, i32, vp, vp, i32, i32, i32, i32, vp, vp]),
            "or_dual_ascent": (f64, [vp, i32, i64, i32, i32, f64, f64, f64, f64, f64, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


# ---------------------------------------------------------------------------

def philox4x32_10(ctr: Sequence[int], key: Sequence[int]) -> np.ndarray:
    c = np.asarray(ctr, np.uint32)
    k = np.asarray(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().or_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def perm_keys(seed: int, epoch: int, iteration: int) -> np.ndarray:
    k = np.zeros(4, np.uint32)
    lib().or_perm_keys(seed, epoch, iteration, _p(k))
    return k


def feistel_perm(n: int, keys: np.ndarray) -> np.ndarray:
    keys = np.ascontiguousarray(keys, np.uint32)
    f = lib().or_feistel_index
    return np.array([f(n, _p(keys), i) for i in range(n)], np.int64)


def bf16_round(x: float) -> float:
    return lib().or_bf16_round(float(x))


def env_cfg(spec) -> EnvCfg:
    """Oracle configuration from a workloads.EnvSpec."""
    c = EnvCfg()
    for name in ("n_envs", "n_channels", "trace_len", "n_actions", "obs_kind", "actuator_kind",
                 "n_levels", "level_init", "g_min", "g_max", "b_min", "b_max", "b_init",
                 "episode_len", "budget_q", "scale_phase_mask", "reward_kind", "reward_window"):
        setattr(c, name, int(getattr(spec, name)))
    c.r_ok, c.r_viol, c.bonus_coef = spec.r_ok, spec.r_viol, spec.bonus_coef
    for l, row in enumerate(spec.level_scale):
        for ch, v in enumerate(row):
            c.level_scale[l][ch] = float(v)
    for l, v in enumerate(spec.level_tokens):
        c.level_tokens[l] = float(v)
    c.seed = int(spec.seed)
    for l, v in enumerate(getattr(spec, "level_samples", None) or []):
        c.level_samples[l] = int(v)
    c.n_families = int(getattr(spec, "n_families", 0) or 0)
    for f in range(c.n_families):
        c.fam_len[f] = int(spec.fam_len[f])
        c.fam_channels[f] = int(spec.fam_channels[f])
        c.fam_budget_q[f] = int(spec.fam_budget_q[f])
    return c


def actuator_scale(spec, level: int, channel: int = 0) -> float:
    cfg = env_cfg(spec)
    return lib().or_actuator_scale(C.byref(cfg), level, channel)


class OrRule(C.Structure):
    _fields_ = [("kind", C.c_int32), ("hi_q", C.c_int32), ("lo_q", C.c_int32),
                ("drop30_q", C.c_int32), ("climb30_q", C.c_int32), ("climb10_q", C.c_int32)]


def or_rule(rule) -> OrRule:
    return OrRule(rule.kind, rule.hi_q, rule.lo_q, rule.drop30_q, rule.climb30_q, rule.climb10_q)


class OracleEnv:
    """A subset of a workload's envs, stepped by the oracle."""

    def __init__(self, spec, trace: np.ndarray, phase: np.ndarray, env_ids: Sequence[int]):
        self.spec = spec
        self.cfg = env_cfg(spec)
        self.trace = np.ascontiguousarray(trace, np.float32)
        self.phase = np.ascontiguousarray(phase, np.uint8)
        self.env_ids = np.ascontiguousarray(env_ids, np.int32)
        self.n = len(self.env_ids)
        self.state = np.zeros(self.n * lib().or_env_state_size(), np.uint8)
        rc = lib().or_env_init(C.byref(self.cfg), _p(self.trace), _p(self.phase),
                               _p(self.env_ids), self.n, _p(self.state))
        if rc != 0:
            raise ValueError("oracle env init rejected the configuration")

    def obs(self) -> np.ndarray:
        D = self.spec.obs_dim
        out = np.zeros((self.n, D), np.float32)
        sz = lib().or_env_state_size()
        for i in range(self.n):
            lib().or_env_obs(C.byref(self.cfg), _p(self.trace), _p(self.phase),
                             C.c_void_p(self.state.ctypes.data + i * sz),
                             C.c_void_p(out.ctypes.data + i * D * 4))
        return out

    def rollout(self, params: np.ndarray, hidden: int, bf16: bool, T: int, iteration: int,
                lam: float = 1.0, deterministic: bool = False,
                forced: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
        n, D = self.n, self.spec.obs_dim
        params = np.ascontiguousarray(params, np.float32)
        out = dict(
            obs=np.zeros((T, n, D), np.float32), obs_last=np.zeros((n, D), np.float32),
            act_own=np.zeros((T, n), np.uint8), logp=np.zeros((T, n), np.float64),
            reward=np.zeros((T, n), np.float64), done=np.zeros((T, n), np.uint8),
            viol=np.zeros((n, 2), np.int32), tokens=np.zeros(n, np.float64),
            excess=np.zeros(n, np.float64), energy_q=np.zeros(n, np.int64),
            samples=np.zeros(n, np.int64), q=np.zeros((T, n), np.int32))
        f = None if forced is None else np.ascontiguousarray(forced, np.uint8)
        lib().or_rollout(C.byref(self.cfg), _p(self.trace), _p(self.phase), _p(params), hidden,
                         int(bf16), _p(self.env_ids), n, _p(self.state), T, iteration, lam,
                         int(deterministic), _p(f), _p(out["obs"]), _p(out["obs_last"]),
                         _p(out["act_own"]), _p(out["logp"]), _p(out["reward"]), _p(out["done"]),
                         _p(out["viol"]), _p(out["tokens"]), _p(out["excess"]),
                         _p(out["energy_q"]), _p(out["samples"]), _p(out["q"]))
        return out


    def set_offsets(self, offsets) -> None:
        """Start a new episode of every env at the given trace offsets."""
        off = np.ascontiguousarray(offsets, np.int32)
        if lib().or_env_set_offsets(C.byref(self.cfg), _p(self.trace), _p(self.phase), _p(off),
                                    self.n, _p(self.state)) != 0:
            raise ValueError("oracle rejected an episode offset")

    def rollout_rule(self, rule, T: int, iteration: int, lam: float = 1.0) -> Dict[str, np.ndarray]:
        """T steps under a baseline rule policy (workloads.RuleSpec)."""
        n = self.n
        out = dict(act=np.zeros((T, n), np.uint8), reward=np.zeros((T, n), np.float64),
                   done=np.zeros((T, n), np.uint8), viol=np.zeros((n, 2), np.int32),
                   tokens=np.zeros(n, np.float64), excess=np.zeros(n, np.float64),
                   energy_q=np.zeros(n, np.int64), samples=np.zeros(n, np.int64),
                   q=np.zeros((T, n), np.int32))
        r = or_rule(rule)
        if lib().or_rollout_rule(C.byref(self.cfg), _p(self.trace), _p(self.phase), C.byref(r),
                                 _p(self.env_ids), n, _p(self.state), T, iteration, lam,
                                 _p(out["act"]), _p(out["reward"]), _p(out["done"]), _p(out["viol"]),
                                 _p(out["tokens"]), _p(out["excess"]), _p(out["energy_q"]),
                                 _p(out["samples"]), _p(out["q"])) != 0:
            raise ValueError("oracle rejected the rule")
        return out


def mlp_forward(net, params: np.ndarray, obs: np.ndarray):
    obs = np.ascontiguousarray(obs, np.float32).reshape(-1, net.obs_dim)
    n = obs.shape[0]
    logits = np.zeros((n, net.n_actions), np.float64)
    value = np.zeros(n, np.float64)
    lib().or_mlp_forward(net.obs_dim, net.hidden, net.n_actions, int(net.dtype == 1),
                         _p(np.ascontiguousarray(params, np.float32)), n, _p(obs), _p(logits),
                         _p(value))
    return logits, value


def gae(r, v, done, last_v, gamma: float, lam: float):
    r = np.ascontiguousarray(r, np.float32)
    T, E = r.shape
    adv = np.zeros((T, E), np.float64)
    ret = np.zeros((T, E), np.float64)
    lib().or_gae(T, E, _p(r), _p(np.ascontiguousarray(v, np.float32)),
                 _p(np.ascontiguousarray(done, np.uint8)),
                 _p(np.ascontiguousarray(last_v, np.float32)), gamma, lam, _p(adv), _p(ret))
    return adv, ret


def ppo_cfg(ppo) -> PPOCfg:
    c = PPOCfg()
    c.epochs, c.minibatch = ppo.epochs, ppo.minibatch
    for n in ("lr", "clip", "vf_coef", "ent_coef", "max_grad_norm", "beta1", "beta2", "eps"):
        setattr(c, n, float(getattr(ppo, n)))
    return c


def ppo_minibatch_grad(net, params64: np.ndarray, obs, act, logp_old, adv, ret, clip: float,
                       vf_coef: float, ent_coef: float, want_grad: bool = True):
    """bf16 networks expect params64 to hold the bf16-rounded weights."""
    params64 = np.ascontiguousarray(params64, np.float64)
    M = len(act)
    grad = np.zeros_like(params64) if want_grad else None
    stats = np.zeros(5, np.float64)
    loss = lib().or_ppo_minibatch_grad_ex(
        net.obs_dim, net.hidden, net.n_actions, int(net.dtype == 1), _p(params64), M,
        _p(np.ascontiguousarray(obs, np.float32)), _p(np.ascontiguousarray(act, np.uint8)),
        _p(np.ascontiguousarray(logp_old, np.float32)), _p(np.ascontiguousarray(adv, np.float32)),
        _p(np.ascontiguousarray(ret, np.float32)), clip, vf_coef, ent_coef, _p(grad), _p(stats))
    return loss, grad, stats


def ppo_update(net, ppo, params, adam_m, adam_v, adam_t: int, obs, act, logp_old, adv, ret,
               seed: int, iteration: int, max_steps: int = -1):
    """Returns (params64, m, v, adam_t, stats[8]); inputs are not modified."""
    P = np.array(params, np.float64)
    m = np.array(adam_m, np.float64)
    v = np.array(adam_v, np.float64)
    N = int(np.asarray(act).size)
    stats = np.zeros(8, np.float64)
    cfg = ppo_cfg(ppo)
    t = lib().or_ppo_update_ex(
        net.obs_dim, net.hidden, net.n_actions, int(net.dtype == 1), _p(P), _p(m), _p(v), adam_t, N,
        _p(np.ascontiguousarray(obs, np.float32)), _p(np.ascontiguousarray(act, np.uint8)),
        _p(np.ascontiguousarray(logp_old, np.float32)), _p(np.ascontiguousarray(adv, np.float32)),
        _p(np.ascontiguousarray(ret, np.float32)), C.byref(cfg), seed, iteration, max_steps,
        _p(stats))
    return P, m, v, int(t), stats


def fleet_windows(traces, job_of_gpu, n_jobs: int, offsets, horizon: int, windows, budget_q: int):
    traces = np.ascontiguousarray(traces, np.float32)
    G, L = traces.shape
    offsets = np.ascontiguousarray(offsets, np.int32)
    N = offsets.shape[0]
    windows = np.ascontiguousarray(windows, np.int32)
    W = len(windows)
    counts = np.zeros((N, W), np.int32)
    peaks = np.zeros((N, W), np.int32)
    rc = lib().or_fleet_windows(G, L, _p(traces), _p(np.ascontiguousarray(job_of_gpu, np.int32)),
                                n_jobs, _p(offsets), N, horizon, _p(windows), W, budget_q,
                                _p(counts), _p(peaks))
    if rc != 0:
        raise ValueError("oracle fleet windows rejected its inputs")
    return counts, peaks


def fleet_stagger(traces, job_of_gpu, n_jobs: int, horizon: int, w: int, stride: int = 1):
    """Greedy phase-staggered schedule (Sec. 8): (offsets[J], peaks[J])."""
    traces = np.ascontiguousarray(traces, np.float32)
    G, L = traces.shape
    offsets = np.zeros(n_jobs, np.int32)
    peaks = np.zeros(n_jobs, np.int32)
    rc = lib().or_fleet_stagger(G, L, _p(traces), _p(np.ascontiguousarray(job_of_gpu, np.int32)),
                                n_jobs, horizon, w, stride, _p(offsets), _p(peaks))
    if rc != 0:
        raise ValueError("oracle fleet stagger rejected its inputs")
    return offsets, peaks


def dual_ascent(viol, steps: int, lam: float, target: float = 0.08, eta: float = 0.5, lo: float = 1e-3,
                hi: float = 2.0, window: int = 60, additive: bool = False):
    """Eq. 7 (or the additive G3 form): (new lambda, observed violation rate)."""
    viol = np.ascontiguousarray(viol, np.int32).reshape(-1, 2)
    rate = np.zeros(1, np.float64)
    new = lib().or_dual_ascent(_p(viol), viol.shape[0], steps, window, int(additive), lam, target, eta,
                               lo, hi, _p(rate))
    return float(new), float(rate[0])
