"""Python binding of the pe C ABI (include/pe.h): argument marshalling only.

Every step of the path runs in the CUDA kernels of libpe.so.  PyTorch is used
for device memory and streams: tensors are passed to the library as raw
device pointers together with the current CUDA stream.  There is no CPU
fallback: if libpe.so is missing or fails to load, every entry point raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, Optional, Sequence

import torch

from . import workloads as W

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libpe.so")
_lib = None

PE_OK, PE_EINVAL, PE_ENOMEM, PE_ECUDA, PE_EOVERFLOW, PE_ETIMEOUT, PE_ESTATE = range(7)
PE_F32, PE_BF16 = 0, 1
PE_ROLLOUT_DETERMINISTIC = 1
MAX_LEVELS, MAX_CH = 32, 4
(PE_PROF_ROLLOUT, PE_PROF_VALUE, PE_PROF_GAE, PE_PROF_PPO_GRAD, PE_PROF_PPO_REDUCE,
 PE_PROF_PPO_ADAM, PE_PROF_PPO_OTHER, PE_PROF_FLEET_PREP, PE_PROF_FLEET_WINDOWS,
 PE_PROF_MLP_POLICY, PE_PROF_MLP_VALUE) = range(11)
PE_PROF_KINDS = 11


class PEError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"pe status {status}: {msg}")
        self.status = status


class EnvConfig(C.Structure):
    _fields_ = [(n, C.c_int32) for n in (
        "n_envs", "n_channels", "trace_len", "n_actions", "obs_kind", "actuator_kind",
        "n_levels", "level_init", "g_min", "g_max", "b_min", "b_max", "b_init",
        "episode_len", "budget_q", "scale_phase_mask", "reward_kind", "reward_window")] + [
        ("r_ok", C.c_float), ("r_viol", C.c_float), ("bonus_coef", C.c_float),
        ("level_scale", (C.c_float * MAX_CH) * MAX_LEVELS),
        ("level_tokens", C.c_float * MAX_LEVELS),
        ("seed", C.c_uint64),
        ("level_samples", C.c_int32 * MAX_LEVELS),
        ("n_families", C.c_int32), ("fam_len", C.c_int32 * 4), ("fam_channels", C.c_int32 * 4),
        ("fam_budget_q", C.c_int32 * 4)]


class Net(C.Structure):
    _fields_ = [("obs_dim", C.c_int32), ("hidden", C.c_int32), ("n_actions", C.c_int32),
                ("dtype", C.c_int32)]


ROLLOUT_FIELDS = ("obs", "obs_last", "act", "logp", "value", "last_value", "reward", "done", "viol",
                  "tokens", "excess", "energy_q", "samples", "q")


class RolloutBuf(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ROLLOUT_FIELDS]


class Rule(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("kind", "hi_q", "lo_q", "drop30_q", "climb30_q", "climb10_q")]


class PPOConfig(C.Structure):
    _fields_ = [("epochs", C.c_int32), ("minibatch", C.c_int32)] + [
        (n, C.c_float) for n in ("lr", "clip", "vf_coef", "ent_coef", "max_grad_norm",
                                 "beta1", "beta2", "eps")] + [
        ("seed", C.c_uint64), ("iteration", C.c_uint32)]


EXPORTS = (
    "pe_env_create", "pe_env_destroy", "pe_env_state_bytes", "pe_env_save", "pe_env_load",
    "pe_param_count", "pe_rollout_workspace_bytes", "pe_rollout", "pe_value_workspace_bytes",
    "pe_value", "pe_device_check", "pe_gae", "pe_ppo_workspace_bytes",
    "pe_ppo_update", "pe_fleet_workspace_bytes", "pe_fleet_windows", "pe_fleet_windows_noalloc",
    "pe_fleet_stagger_workspace_bytes", "pe_fleet_stagger", "pe_env_set_offsets", "pe_rollout_rule", "pe_rollout_replay", "pe_wait_selftest",
    "pe_dual_ascent", "pe_roof_probe",
    "pe_profile_enable",
    "pe_profile_read", "pe_profile_kind_name", "pe_last_error")


def lib():
    """Load libpe.so (raises if it is missing)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_11226_gb300.build.build()")
        L = C.CDLL(LIB_PATH)
        vp, i32, i64, u32 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32
        sig = {
            "pe_env_create": (i32, [vp, vp, vp, C.POINTER(vp)]),
            "pe_env_destroy": (i32, [vp]),
            "pe_env_state_bytes": (i64, [vp]),
            "pe_env_save": (i32, [vp, vp]),
            "pe_env_load": (i32, [vp, vp]),
            "pe_param_count": (i64, [vp]),
            "pe_rollout_workspace_bytes": (i64, [vp, vp]),
            "pe_rollout": (i32, [vp, vp, vp, i32, u32, C.c_float, i32, vp, vp, i64, vp]),
            "pe_value_workspace_bytes": (i64, [vp]),
            "pe_value": (i32, [vp, vp, vp, i64, vp, vp, i64, vp]),
            "pe_device_check": (i32, [vp]),
            "pe_gae": (i32, [vp, vp, vp, vp, i32, i32, C.c_float, C.c_float, vp, vp, vp]),
            "pe_ppo_workspace_bytes": (i64, [vp, vp, i64]),
            "pe_ppo_update": (i32, [vp, vp, vp, vp, i64, vp, vp, vp, vp, vp, i64, vp, vp, vp,
                                    i64, vp]),
            "pe_fleet_workspace_bytes": (i64, [i32, i32, i32]),
            "pe_fleet_stagger_workspace_bytes": (i64, [i32, i32, i32, i32]),
            "pe_env_set_offsets": (i32, [vp, vp, vp]),
            "pe_dual_ascent": (i32, [vp, i32, i64, i32, i32, C.c_float, C.c_float, C.c_float, C.c_float,
                                     vp, vp, vp]),
            "pe_rollout_rule": (i32, [vp, vp, i32, u32, C.c_float, i32, vp, vp]),
            "pe_rollout_replay": (i32, [vp, vp, i32, u32, C.c_float, i32, vp, vp]),
            "pe_wait_selftest": (i32, [i32, C.c_int64, vp, vp]),
            "pe_fleet_stagger": (i32, [vp, i32, i32, vp, i32, i32, i32, i32, vp, vp, vp, i64, vp]),
            "pe_fleet_windows": (i32, [vp, i32, i32, vp, i32, vp, i64, i32, vp, i32, i64, vp,
                                       vp, vp, i64, vp]),
            "pe_fleet_windows_noalloc": (i32, [vp, i32, i32, vp, i32, vp, i64, i32, vp, i32, i64,
                                               vp, vp, vp]),
            "pe_roof_probe": (i32, [i32, vp, i64, i64, C.POINTER(C.c_double), C.POINTER(C.c_double), vp]),
            "pe_profile_enable": (i32, [i32]),
            "pe_profile_read": (i32, [i32, C.POINTER(C.c_double), C.POINTER(C.c_int64)]),
            "pe_profile_kind_name": (C.c_char_p, [i32]),
            "pe_last_error": (C.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _check(status: int):
    if status != PE_OK:
        raise PEError(status, lib().pe_last_error().decode())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def env_config(spec: W.EnvSpec) -> EnvConfig:
    c = EnvConfig()
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
    for l, v in enumerate(spec.level_samples or []):
        c.level_samples[l] = int(v)
    c.n_families = int(spec.n_families or 0)
    for f in range(c.n_families):
        c.fam_len[f] = int(spec.fam_len[f])
        c.fam_channels[f] = int(spec.fam_channels[f])
        c.fam_budget_q[f] = int(spec.fam_budget_q[f])
    return c


def net_desc(net: W.NetSpec) -> Net:
    return Net(net.obs_dim, net.hidden, net.n_actions, net.dtype)


def param_count(net: W.NetSpec) -> int:
    return int(lib().pe_param_count(C.byref(net_desc(net))))


class Env:
    """E environments over one trace (pe_env_create); the trace may be a
    host or device tensor."""

    def __init__(self, spec: W.EnvSpec, trace: torch.Tensor, phase: torch.Tensor):
        self.spec = spec
        self.cfg = env_config(spec)
        trace = trace.contiguous().to(torch.float32)
        phase = phase.contiguous().to(torch.uint8)
        h = C.c_void_p()
        _check(lib().pe_env_create(C.byref(self.cfg), _ptr(trace), _ptr(phase), C.byref(h)))
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            lib().pe_env_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def state_bytes(self) -> int:
        return int(lib().pe_env_state_bytes(self._h))

    def save(self) -> bytes:
        buf = (C.c_uint8 * self.state_bytes())()
        _check(lib().pe_env_save(self._h, buf))
        return bytes(buf)

    def load(self, image: bytes):
        buf = (C.c_uint8 * len(image)).from_buffer_copy(image)
        _check(lib().pe_env_load(self._h, buf))


def alloc_rollout(spec: W.EnvSpec, net: W.NetSpec, T: int, device="cuda") -> Dict[str, torch.Tensor]:
    E, D = spec.n_envs, net.obs_dim
    odt = torch.float32 if net.dtype == PE_F32 else torch.bfloat16
    kw = dict(device=device)
    return dict(
        obs=torch.empty((T, E, D), dtype=odt, **kw), obs_last=torch.empty((E, D), dtype=odt, **kw),
        act=torch.empty((T, E), dtype=torch.uint8, **kw), logp=torch.empty((T, E), **kw),
        value=torch.empty((T, E), **kw), last_value=torch.empty(E, **kw),
        reward=torch.empty((T, E), **kw), done=torch.empty((T, E), dtype=torch.uint8, **kw),
        viol=torch.empty((E, 2), dtype=torch.int32, **kw), tokens=torch.empty(E, **kw),
        excess=torch.empty(E, **kw), energy_q=torch.empty(E, dtype=torch.int64, **kw),
        samples=torch.empty(E, dtype=torch.int64, **kw), q=torch.empty((T, E), dtype=torch.int32, **kw))


def _rollout_buf(b: Dict[str, Optional[torch.Tensor]]) -> RolloutBuf:
    return RolloutBuf(*[(b[k].data_ptr() if b.get(k) is not None else None) for k in ROLLOUT_FIELDS])


def rollout_workspace_bytes(env: Env, net: W.NetSpec) -> int:
    return int(lib().pe_rollout_workspace_bytes(env._h, C.byref(net_desc(net))))


def alloc_workspace(nbytes: int, device="cuda") -> Optional[torch.Tensor]:
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def rollout(env: Env, net: W.NetSpec, params: torch.Tensor, T: int, iteration: int,
            buf: Dict[str, torch.Tensor], lam: float = 1.0, deterministic: bool = False,
            workspace: Optional[torch.Tensor] = None, stream=None):
    rb = _rollout_buf(buf)
    if workspace is None and net.dtype != PE_F32:
        workspace = alloc_workspace(rollout_workspace_bytes(env, net))
    nbytes = 0 if workspace is None else workspace.numel()
    _check(lib().pe_rollout(env._h, C.byref(net_desc(net)), _ptr(params), T, iteration, lam,
                            PE_ROLLOUT_DETERMINISTIC if deterministic else 0, C.byref(rb),
                            _ptr(workspace), nbytes, _stream(stream)))


def set_offsets(env: Env, offsets: torch.Tensor, stream=None):
    """Start a new episode of every env at offsets[e] (int32 device tensor)."""
    _check(lib().pe_env_set_offsets(env._h, _ptr(offsets), _stream(stream)))


def alloc_rule_rollout(spec: W.EnvSpec, T: int, obs: bool = False, obs_bf16: bool = False,
                       device="cuda") -> Dict[str, torch.Tensor]:
    """Buffers of a rule-policy rollout (observations only if asked for)."""
    E, D = spec.n_envs, spec.obs_dim
    kw = dict(device=device)
    odt = torch.bfloat16 if obs_bf16 else torch.float32
    return dict(
        obs=torch.empty((T, E, D), dtype=odt, **kw) if obs else None,
        obs_last=torch.empty((E, D), dtype=odt, **kw) if obs else None,
        act=torch.empty((T, E), dtype=torch.uint8, **kw), logp=None, value=None, last_value=None,
        reward=torch.empty((T, E), **kw), done=torch.empty((T, E), dtype=torch.uint8, **kw),
        viol=torch.empty((E, 2), dtype=torch.int32, **kw), tokens=torch.empty(E, **kw),
        excess=torch.empty(E, **kw), energy_q=torch.empty(E, dtype=torch.int64, **kw),
        samples=torch.empty(E, dtype=torch.int64, **kw), q=torch.empty((T, E), dtype=torch.int32, **kw))


def rollout_rule(env: Env, rule: W.RuleSpec, T: int, iteration: int, buf: Dict[str, torch.Tensor],
                 lam: float = 1.0, stream=None):
    """T steps of every env under a baseline rule policy (no network)."""
    rb = _rollout_buf(buf)
    obs_bf16 = buf["obs"] is not None and buf["obs"].dtype == torch.bfloat16
    r = Rule(rule.kind, rule.hi_q, rule.lo_q, rule.drop30_q, rule.climb30_q, rule.climb10_q)
    _check(lib().pe_rollout_rule(env._h, C.byref(r), T, iteration, lam, int(obs_bf16), C.byref(rb),
                                 _stream(stream)))


def rollout_replay(env: Env, actions: torch.Tensor, T: int, iteration: int, buf: Dict[str, torch.Tensor],
                   lam: float = 1.0, stream=None):
    """Teacher-forced rollout: env e takes actions[t][e] (uint8, device, [T][E]) at step t."""
    if actions.dtype != torch.uint8 or actions.numel() != T * env.spec.n_envs or not actions.is_contiguous():
        raise ValueError("actions must be a contiguous uint8 tensor of T x n_envs")
    rb = _rollout_buf(buf)
    obs_bf16 = buf["obs"] is not None and buf["obs"].dtype == torch.bfloat16
    _check(lib().pe_rollout_replay(env._h, _ptr(actions), T, iteration, lam, int(obs_bf16), C.byref(rb),
                                   _stream(stream)))


def wait_selftest(mode: int, limit_cycles: int, workspace: torch.Tensor, stream=None):
    """Run one of the library's bounded waits with a short budget (see pe.h);
    raises PEError with PE_ETIMEOUT when the wait gives up."""
    _check(lib().pe_wait_selftest(mode, int(limit_cycles), _ptr(workspace), _stream(stream)))


def dual_ascent(viol: torch.Tensor, steps: int, lam: torch.Tensor, rate: Optional[torch.Tensor] = None,
                target: float = 0.08, eta: float = 0.5, lo: float = 1e-3, hi: float = 2.0, window: int = 60,
                additive: bool = False, stream=None):
    """Eq. 7 update of the device scalar lam (float32) from a rollout's viol counts."""
    _check(lib().pe_dual_ascent(_ptr(viol), viol.shape[0], steps, window, int(additive), target, eta, lo, hi,
                                _ptr(lam), _ptr(rate), _stream(stream)))


def value_workspace_bytes(net: W.NetSpec) -> int:
    return int(lib().pe_value_workspace_bytes(C.byref(net_desc(net))))


def value(net: W.NetSpec, params: torch.Tensor, obs: torch.Tensor, out: torch.Tensor,
          workspace: Optional[torch.Tensor] = None, stream=None):
    n = obs.numel() // net.obs_dim
    if workspace is None and net.dtype != PE_F32:
        workspace = alloc_workspace(value_workspace_bytes(net))
    nbytes = 0 if workspace is None else workspace.numel()
    _check(lib().pe_value(C.byref(net_desc(net)), _ptr(params), _ptr(obs), n, _ptr(out),
                          _ptr(workspace), nbytes, _stream(stream)))


def device_check(stream=None):
    """Synchronise and raise PEError(PE_ETIMEOUT) if a bounded device wait gave up."""
    _check(lib().pe_device_check(_stream(stream)))


def gae(reward, value_, done, last_value, gamma: float, lam: float, adv, ret, stream=None):
    T, E = reward.shape
    _check(lib().pe_gae(_ptr(reward), _ptr(value_), _ptr(done), _ptr(last_value), T, E, gamma,
                        lam, _ptr(adv), _ptr(ret), _stream(stream)))


def ppo_config(ppo: W.PPOSpec, seed: int, iteration: int) -> PPOConfig:
    c = PPOConfig()
    c.epochs, c.minibatch = ppo.epochs, ppo.minibatch
    for n in ("lr", "clip", "vf_coef", "ent_coef", "max_grad_norm", "beta1", "beta2", "eps"):
        setattr(c, n, float(getattr(ppo, n)))
    c.seed, c.iteration = seed, iteration
    return c


def ppo_workspace_bytes(net: W.NetSpec, ppo: W.PPOSpec, n: int) -> int:
    c = ppo_config(ppo, 0, 0)
    return int(lib().pe_ppo_workspace_bytes(C.byref(net_desc(net)), C.byref(c), n))


def ppo_update(net: W.NetSpec, ppo: W.PPOSpec, params, adam_m, adam_v, adam_t: int, obs, act,
               logp_old, adv, ret, stats, workspace, seed: int, iteration: int, stream=None):
    c = ppo_config(ppo, seed, iteration)
    n = act.numel()
    _check(lib().pe_ppo_update(C.byref(net_desc(net)), _ptr(params), _ptr(adam_m), _ptr(adam_v),
                               adam_t, _ptr(obs), _ptr(act), _ptr(logp_old), _ptr(adv), _ptr(ret),
                               n, C.byref(c), _ptr(stats), _ptr(workspace), workspace.numel(),
                               _stream(stream)))


def fleet_workspace_bytes(J: int, L: int, H: int) -> int:
    return int(lib().pe_fleet_workspace_bytes(J, L, H))


def fleet_windows(traces, job_of_gpu, J: int, offsets, H: int, windows: Sequence[int],
                  budget_q: int, counts, peaks, workspace, stream=None):
    G, L = traces.shape
    N = offsets.shape[0]
    w = (C.c_int32 * len(windows))(*[int(x) for x in windows])
    _check(lib().pe_fleet_windows(_ptr(traces), G, L, _ptr(job_of_gpu), J, _ptr(offsets), N, H,
                                  w, len(windows), budget_q, _ptr(counts), _ptr(peaks),
                                  _ptr(workspace), workspace.numel(), _stream(stream)))


def fleet_stagger_workspace_bytes(J: int, L: int, H: int, stride: int) -> int:
    return int(lib().pe_fleet_stagger_workspace_bytes(J, L, H, stride))


def fleet_stagger(traces, job_of_gpu, J: int, H: int, w: int, stride: int, offsets, peaks, workspace,
                  stream=None):
    """Greedy phase-staggered start offsets (offsets[J]) and stage peaks (peaks[J])."""
    G, L = traces.shape
    _check(lib().pe_fleet_stagger(_ptr(traces), G, L, _ptr(job_of_gpu), J, H, w, stride, _ptr(offsets),
                                  _ptr(peaks), _ptr(workspace), workspace.numel(), _stream(stream)))


PE_ROOF_FFMA, PE_ROOF_FFMA2, PE_ROOF_IADD, PE_ROOF_L2 = 0, 1, 2, 3


def roof_probe(kind: int, buf, reps: int, stream=None):
    """(device ms, units) of one timed throughput loop (pe_roof_probe)."""
    ms, units = C.c_double(0.0), C.c_double(0.0)
    _check(lib().pe_roof_probe(kind, _ptr(buf), buf.numel() * buf.element_size(), reps, C.byref(ms),
                               C.byref(units), _stream(stream)))
    return ms.value, units.value


FLEET_NOALLOC_SCRATCH_BYTES = 4 * 1024 * 1024


def fleet_windows_noalloc(traces, job_of_gpu, J: int, offsets, H: int, windows: Sequence[int],
                          budget_q: int, counts, peaks, stream=None):
    """pe_fleet_windows without a workspace, for callers that cannot allocate
    device memory; its scratch is a fixed 4 MiB array inside the library."""
    G, L = traces.shape
    N = offsets.shape[0]
    w = (C.c_int32 * len(windows))(*[int(x) for x in windows])
    _check(lib().pe_fleet_windows_noalloc(_ptr(traces), G, L, _ptr(job_of_gpu), J, _ptr(offsets), N,
                                          H, w, len(windows), budget_q, _ptr(counts), _ptr(peaks),
                                          _stream(stream)))


def profile_enable(on: bool):
    _check(lib().pe_profile_enable(int(bool(on))))


def profile_read(kind: int):
    """(summed device ms, launches) of one kernel kind since the last read."""
    ms = C.c_double()
    n = C.c_int64()
    _check(lib().pe_profile_read(kind, C.byref(ms), C.byref(n)))
    return ms.value, n.value


def profile_kind_name(kind: int) -> str:
    return lib().pe_profile_kind_name(kind).decode()
