"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Tolerances (spec bar): integer counts bit-exact; fp32 env, network and
GAE outputs within 1e-5 relative, measured against max(|ref|, rms(ref)) so
that near-zero entries do not fail a pure relative test; sampled actions
agree on >= 99.9% of steps under teacher forcing (the oracle steps with the
GPU's actions, so one flipped sample cannot cascade).
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_11226_gb300 import pe
from paper_2608_11226_gb300 import workloads as W

pytestmark = pytest.mark.gpu
TOL = 1e-5


def rel_err(gpu, ref):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    floor = np.sqrt(np.mean(ref ** 2)) + 1e-30
    return float(np.max(np.abs(gpu - ref) / np.maximum(np.abs(ref), floor)))


def bf16_ok(gpu, ref, tol=2e-2, tail=1e-3):
    """bf16-network outputs: normwise relative error <= tol, and at most a
    `tail` fraction of elements beyond tol in the rms-floored relative error.
    Rare 1-ulp bf16 rounding flips of hidden activations (fp32 accumulation on
    the GPU, fp64 in the oracle) cascade into a few larger deviations."""
    gpu = np.asarray(gpu, np.float64).ravel()
    ref = np.asarray(ref, np.float64).ravel()
    d = np.abs(gpu - ref)
    norm = d.max() / max(np.abs(ref).max(), 1e-30)
    floor = np.sqrt(np.mean(ref ** 2)) + 1e-30
    frac = float(np.mean(d / np.maximum(np.abs(ref), floor) > tol))
    return norm <= tol and frac <= tail


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_11226_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    pe.lib()


def cpu(t):
    return t.detach().cpu().numpy()


# ------------------------------------------------------------------------ GAE
@pytest.mark.parametrize("T,E", [(1, 1), (37, 100), (512, 4096), (600, 33), (2048, 70)])
def test_gae_parity(T, E):
    g = torch.Generator().manual_seed(T * 1000 + E)
    r = torch.randn(T, E, generator=g)
    v = torch.randn(T, E, generator=g)
    d = (torch.rand(T, E, generator=g) < 0.02).to(torch.uint8)
    lv = torch.randn(E, generator=g)
    dev = [x.cuda() for x in (r, v, d, lv)]
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty(T, E, device="cuda")
    pe.gae(*dev, 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    ra, rr = O.gae(r.numpy(), v.numpy(), d.numpy(), lv.numpy(), 0.99, 0.95)
    assert rel_err(cpu(adv), ra) <= TOL
    assert rel_err(cpu(ret), rr) <= TOL


@pytest.mark.parametrize("T,E", [(64, 16384), (2048, 131072), (1024, 65536), (37, 32771), (300, 131074),
                                 (5, 262144)])
def test_gae_parity_vector_paths(T, E):
    """The wide-batch kernels: the 2-env-per-thread chunked kernel
    (16,384 <= E < 32,768) and the per-column streaming kernel (E >= 32,768;
    2 envs per thread from 131,072 when aligned, else 1), with ragged CTA
    spans (32,771 and 131,074 envs), horizons shorter than, equal to and not a
    multiple of its 16- or 12-step load ring.  Envs are independent, so the
    oracle checks sampled columns including both ends of a CTA span."""
    g = torch.Generator(device="cuda").manual_seed(E)
    r = torch.randn(T, E, device="cuda", generator=g)
    v = torch.randn(T, E, device="cuda", generator=g)
    d = (torch.rand(T, E, device="cuda", generator=g) < 0.02).to(torch.uint8)
    lv = torch.randn(E, device="cuda", generator=g)
    adv = torch.empty(T, E, device="cuda")
    ret = torch.empty(T, E, device="cuda")
    pe.gae(r, v, d, lv, 0.99, 0.95, adv, ret)
    torch.cuda.synchronize()
    rng = np.random.default_rng(T)
    cols = np.unique(np.concatenate([[0, 1, 127, 128, 255, 256, E - 2, E - 1], rng.choice(E, 59, replace=False)]))
    ci = torch.from_numpy(cols).cuda()
    ra, rr = O.gae(cpu(r[:, ci]), cpu(v[:, ci]), cpu(d[:, ci]), cpu(lv[ci]), 0.99, 0.95)
    assert rel_err(cpu(adv[:, ci]), ra) <= TOL
    assert rel_err(cpu(ret[:, ci]), rr) <= TOL


def test_bounded_waits_give_up_and_leave_the_context_usable():
    """Failure detection without a GPU fault: the grid barrier of the
    persistent update with one CTA that never arrives, and an mbarrier that
    nothing completes, both give up after their budget (about 0.1 s here)
    and report PE_ETIMEOUT; the barrier with every CTA arriving passes; the
    context stays usable for a real call afterwards."""
    ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
    pe.wait_selftest(1, 200_000_000, ws)
    for mode in (0, 2):
        with pytest.raises(pe.PEError) as e:
            pe.wait_selftest(mode, 200_000_000, ws)
        assert e.value.status == pe.PE_ETIMEOUT
    pe.device_check()
    r = torch.ones(4, 8, device="cuda")
    adv = torch.empty_like(r)
    ret = torch.empty_like(r)
    pe.gae(r, torch.zeros_like(r), torch.zeros(4, 8, dtype=torch.uint8, device="cuda"),
           torch.zeros(8, device="cuda"), 0.5, 1.0, adv, ret)
    torch.cuda.synchronize()
    assert torch.allclose(adv[0], torch.full((8,), 1.875, device="cuda"))


def test_gae_empty_is_noop():
    z = torch.empty(0, 5, device="cuda")
    pe.gae(z, z, z.to(torch.uint8), torch.empty(5, device="cuda"), 0.99, 0.95, z, z)


# ---------------------------------------------------------------------- fleet
def _fleet_gpu(fw, windows, ws_short=0):
    """ws_short > 0 passes a workspace that many bytes short of
    pe_fleet_workspace_bytes: for J <= 8 that drops the shifted prefix copies
    and the call takes its 4-byte-load path."""
    traces = torch.from_numpy(fw.traces).cuda()
    job = torch.from_numpy(fw.job_of_gpu).cuda()
    off = torch.from_numpy(fw.offsets).cuda()
    N = fw.offsets.shape[0]
    counts = torch.empty((N, len(windows)), dtype=torch.int32, device="cuda")
    peaks = torch.empty_like(counts)
    ws = torch.empty(pe.fleet_workspace_bytes(fw.n_jobs, fw.traces.shape[1], fw.horizon) - ws_short,
                     dtype=torch.uint8, device="cuda")
    pe.fleet_windows(traces, job, fw.n_jobs, off, fw.horizon, windows, fw.budget_q, counts, peaks, ws)
    torch.cuda.synchronize()
    return cpu(counts), cpu(peaks)


def test_fleet_parity_small_bit_exact():
    fw = W.make_fleet(n_compositions=77, length=3001, windows=(1, 60, 600))
    c, p = _fleet_gpu(fw, [1, 60, 600])
    oc, op = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, fw.horizon,
                             fw.windows, fw.budget_q)
    assert np.array_equal(c, oc) and np.array_equal(p, op)


@pytest.mark.parametrize("H", [1, 31, 127, 128, 129, 599, 600, 2500])
@pytest.mark.parametrize("path", ["copies", "one_copy"])
def test_fleet_parity_horizons(H, path):
    fw = W.make_fleet(n_compositions=9, length=2500, windows=(1, 60, 600))
    fw.horizon = H
    windows = [1, 7, 60, 600]
    c, p = _fleet_gpu(fw, windows, ws_short=1 if path == "one_copy" else 0)
    oc, op = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, H, windows, fw.budget_q)
    assert np.array_equal(c, oc) and np.array_equal(p, op)


@pytest.mark.parametrize("windows", [[1, 2, 3, 5], [127, 128, 129, 992], [4, 124, 132, 991]])
def test_fleet_parity_window_alignments(windows):
    """Windows on and off the 4-sample and 128-sample block boundaries of the
    16-byte path, including the largest window; offsets at both trace ends."""
    fw = W.make_fleet(n_compositions=11, length=3000, windows=(1, 60, 600))
    fw.offsets[0, :] = 0
    fw.offsets[1, :] = fw.traces.shape[1] - 1
    fw.offsets[2, :] = np.arange(fw.n_jobs) % 4
    for short in (0, 1):
        c, p = _fleet_gpu(fw, windows, ws_short=short)
        oc, op = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, fw.horizon, windows,
                                 fw.budget_q)
        assert np.array_equal(c, oc) and np.array_equal(p, op)


def test_fleet_parity_more_than_eight_jobs():
    """Twelve jobs over the sixteen traces: the path for fleets of more than
    eight jobs (one prefix copy, stream bases in shared memory)."""
    fw = W.make_fleet(n_compositions=13, length=1800, windows=(1, 60, 600))
    fw.job_of_gpu = (np.arange(fw.traces.shape[0]) % 12).astype(np.int32)
    fw.n_jobs = 12
    fw.offsets = np.random.default_rng(4).integers(0, 1800, (13, 12)).astype(np.int32)
    fw.budget_q = fw.budget_q // 2
    c, p = _fleet_gpu(fw, [1, 60, 600])
    oc, op = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, fw.horizon, [1, 60, 600],
                             fw.budget_q)
    assert np.array_equal(c, oc) and np.array_equal(p, op)
    assert c.sum() > 0


def test_fleet_parity_full_size_sampled():
    """380,000-sample traces and 1,000,000 compositions (the full fleet
    workload); the oracle recomputes a seeded sample of compositions."""
    fw = W.make_fleet()
    c, p = _fleet_gpu(fw, [1, 60, 600])
    rng = np.random.default_rng(11)
    pick = np.concatenate([[0, 1, fw.offsets.shape[0] - 1],
                           rng.choice(fw.offsets.shape[0], 5, replace=False)])
    oc, op = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets[pick], fw.horizon,
                             fw.windows, fw.budget_q)
    assert np.array_equal(c[pick], oc) and np.array_equal(p[pick], op)
    # invariant at every composition: the composed peak never exceeds the
    # sum of per-job peaks (computed by the oracle per job)
    q = np.rint(fw.traces * np.float32(64)).astype(np.int64)
    for wi, w in enumerate((1, 60, 600)):
        per = 0
        for j in range(fw.n_jobs):
            x = q[fw.job_of_gpu == j].sum(0)
            x = np.concatenate([x, x[:w - 1]])  # the trace tiles circularly
            per += np.convolve(x, np.ones(w, np.int64), "valid").max()
        assert p[:, wi].max() <= per


# ------------------------------------------------------------ fleet stagger
def _stagger_gpu(traces, job, J, H, w, stride):
    tr = torch.from_numpy(np.ascontiguousarray(traces, np.float32)).cuda()
    jg = torch.from_numpy(np.ascontiguousarray(job, np.int32)).cuda()
    off = torch.full((J,), -1, dtype=torch.int32, device="cuda")
    pk = torch.full((J,), -1, dtype=torch.int32, device="cuda")
    ws = torch.empty(pe.fleet_stagger_workspace_bytes(J, tr.shape[1], H, max(stride, 1)), dtype=torch.uint8,
                     device="cuda")
    pe.fleet_stagger(tr, jg, J, H, w, stride, off, pk, ws)
    torch.cuda.synchronize()
    return cpu(off), cpu(pk)


@pytest.mark.parametrize("L,H,w,stride", [(500, 500, 60, 1), (997, 800, 20, 7), (300, 1000, 1, 4)])
def test_fleet_stagger_bit_exact(L, H, w, stride):
    """Greedy staggered offsets and stage peaks equal the oracle's exactly
    (ragged candidate grids, horizons shorter and longer than the period)."""
    fw = W.make_fleet(n_compositions=1, length=L, seed=3)
    g_off, g_pk = _stagger_gpu(fw.traces, fw.job_of_gpu, fw.n_jobs, H, w, stride)
    o_off, o_pk = O.fleet_stagger(fw.traces, fw.job_of_gpu, fw.n_jobs, H, w, stride)
    assert np.array_equal(g_off, o_off) and np.array_equal(g_pk, o_pk), (g_off, o_off, g_pk, o_pk)


def test_fleet_stagger_twelve_jobs_bit_exact():
    """Twelve jobs over the sixteen traces (more than the eight streams of one
    composed load): every stage composes the partial-fleet row with one
    candidate job, so the stage count, not the stream count, grows."""
    fw = W.make_fleet(n_compositions=1, length=900, seed=5)
    job = (np.arange(fw.traces.shape[0]) % 12).astype(np.int32)
    g_off, g_pk = _stagger_gpu(fw.traces, job, 12, 700, 60, 3)
    o_off, o_pk = O.fleet_stagger(fw.traces, job, 12, 700, 60, 3)
    assert np.array_equal(g_off, o_off) and np.array_equal(g_pk, o_pk), (g_off, o_off, g_pk, o_pk)


def test_fleet_stagger_full_size_sampled():
    """The 16-GPU, 380,000-sample fleet with every offset a candidate: each
    stage's peak is re-evaluated by the oracle at the chosen offsets, and a
    seeded sample of other candidates (plus offset 0) is never better, nor
    equal at a lower offset."""
    fw = W.make_fleet(n_compositions=1)
    L = fw.traces.shape[1]
    g_off, g_pk = _stagger_gpu(fw.traces, fw.job_of_gpu, fw.n_jobs, L, 60, 1)
    rng = np.random.default_rng(5)
    for j in range(fw.n_jobs):
        sel = fw.job_of_gpu <= j
        tr, jb = fw.traces[sel], fw.job_of_gpu[sel]
        cands = [int(g_off[j])] + [0] + [int(c) for c in rng.integers(0, L, 12)]
        rows = np.tile(g_off[: j + 1], (len(cands), 1)).astype(np.int32)
        rows[:, j] = cands
        _, pk = O.fleet_windows(tr, jb, j + 1, rows, L, [60], 0)
        assert pk[0, 0] == g_pk[j], (j, pk[0, 0], g_pk[j])
        for c, p in zip(cands[1:], pk[1:, 0]):
            assert p > g_pk[j] or (p == g_pk[j] and c >= g_off[j]), (j, c, p, g_off[j], g_pk[j])


def test_fleet_stagger_rejects_bad_arguments():
    fw = W.make_fleet(n_compositions=1, length=200)
    assert pe.fleet_stagger_workspace_bytes(fw.n_jobs, 200, 200, 0) == -1
    with pytest.raises(pe.PEError) as e:
        _stagger_gpu(fw.traces, fw.job_of_gpu, fw.n_jobs, 200, 60, 0)
    assert e.value.status == pe.PE_EINVAL
    with pytest.raises(pe.PEError) as e:
        _stagger_gpu(fw.traces, fw.job_of_gpu, fw.n_jobs, 200, 993, 1)
    assert e.value.status == pe.PE_EINVAL
    bad = fw.job_of_gpu.copy()
    bad[3] = fw.n_jobs
    with pytest.raises(pe.PEError) as e:
        _stagger_gpu(fw.traces, bad, fw.n_jobs, 200, 60, 1)
    assert e.value.status == pe.PE_EINVAL


def test_fleet_rejects_bad_offsets_and_traces():
    fw = W.make_fleet(n_compositions=4, length=700)
    fw.offsets[2, 3] = 700
    with pytest.raises(pe.PEError) as e:
        _fleet_gpu(fw, [1, 60])
    assert e.value.status == pe.PE_EINVAL
    fw = W.make_fleet(n_compositions=4, length=700)
    fw.traces[3, 5] = np.nan
    with pytest.raises(pe.PEError) as e:
        _fleet_gpu(fw, [1, 60])
    assert e.value.status == pe.PE_EOVERFLOW


# -------------------------------------------------------------------- rollout
def _rollout_case(wl, T, iters, sample_envs=None, det=False, lam=1.0):
    spec, net = wl.env, wl.net
    bf16 = net.dtype == pe.PE_BF16
    params = W.init_params(net, seed=1, bias_scale=0.05)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    p_dev = torch.from_numpy(params).cuda()
    ids = np.arange(spec.n_envs) if sample_envs is None else np.asarray(sample_envs)
    ids_d = torch.from_numpy(ids).cuda()
    ora = O.OracleEnv(spec, wl.trace, wl.phase, ids)
    ws = pe.alloc_workspace(pe.rollout_workspace_bytes(env, net)) if bf16 else None
    agree = total = 0
    for it in range(iters):
        pe.rollout(env, net, p_dev, T, it, buf, lam=lam, deterministic=det, workspace=ws)
        pe.device_check()
        g = {}
        for k, v in buf.items():
            sel = v[:, ids_d] if v.dim() >= 2 and k in ("obs", "act", "logp", "value", "reward", "done", "q") else v[ids_d]
            g[k] = cpu(sel.float() if sel.dtype == torch.bfloat16 else sel)
        forced = g["act"]
        o = ora.rollout(params, net.hidden, bf16, T, it, lam=lam, deterministic=det, forced=forced)
        want_obs, want_last = o["obs"], o["obs_last"]
        if bf16:   # the buffer holds observations rounded to bf16 (RNE), as the oracle feeds its network
            want_obs = torch.from_numpy(want_obs).to(torch.bfloat16).float().numpy()
            want_last = torch.from_numpy(want_last).to(torch.bfloat16).float().numpy()
        assert np.array_equal(g["obs"], want_obs), "observations differ"
        assert np.array_equal(g["obs_last"], want_last)
        assert np.array_equal(g["done"], o["done"])
        assert np.array_equal(g["viol"], o["viol"])
        assert np.array_equal(g["energy_q"], o["energy_q"])
        assert np.array_equal(g["samples"], o["samples"])
        assert np.array_equal(g["q"], o["q"])
        assert rel_err(g["reward"], o["reward"]) <= TOL
        assert rel_err(g["tokens"], o["tokens"]) <= TOL
        assert rel_err(g["excess"], o["excess"]) <= TOL
        close = (lambda a, b: bf16_ok(a, b)) if bf16 else (lambda a, b: rel_err(a, b) <= TOL)
        assert close(g["logp"], o["logp"])
        agree += int((o["act_own"] == forced).sum())
        total += forced.size
        _, ov = O.mlp_forward(net, params, o["obs"].reshape(-1, net.obs_dim))
        assert close(g["value"].ravel(), ov)
        _, olv = O.mlp_forward(net, params, o["obs_last"])
        assert close(g["last_value"], olv)
    assert agree / total >= 0.999, agree / total
    env.close()
    return agree / total


def test_rollout_parity_tiny_full():
    _rollout_case(W.make_tiny(), 128, iters=5)   # 640 steps: crosses an episode boundary


def test_rollout_parity_tiny_cadence():
    """The fused fp32 rollout with a cadence table (2, 3 or 5 samples per
    step by level) across an episode boundary."""
    wl = W.make_tiny(n_envs=40)
    wl.env.level_samples = [2, 3, 5]
    _rollout_case(wl, 300, iters=2)


def test_rollout_parity_72b_cadence():
    """The 72B env at the Sec. 4.5 batch cadence (24-42 samples per step,
    40-batch episodes) on the tcgen05 path, crossing episode boundaries."""
    _rollout_case(W.make_72b_cadence(n_envs=128), 30, iters=3, lam=0.7)


def test_rollout_parity_72b_mixed_families():
    """Domain randomisation (Sec. 4.2 G2): the 72B env drawing each episode
    from a 4-GPU 72B-, a 2-GPU 14B- or a 1-GPU 7B-shaped trace family with
    its own budget, on the tcgen05 path across episode boundaries."""
    _rollout_case(W.make_72b_mixed(n_envs=128), 400, iters=3, lam=0.7)


def test_rule_rollout_parity_mixed_families_with_offsets():
    """Rule rollouts on the mixed env, before and after explicit episode
    starts (which keep each env's family)."""
    wl = W.make_72b_mixed(n_envs=64)
    spec = wl.env
    rule = W.threshold_rule(spec.budget_q)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    oenv = O.OracleEnv(spec, wl.trace, wl.phase, range(64))
    for it, T in ((0, 300), (1, 200)):
        buf = pe.alloc_rule_rollout(spec, T)
        pe.rollout_rule(env, rule, T, it, buf, lam=0.5)
        torch.cuda.synchronize()
        ref = oenv.rollout_rule(rule, T, it, lam=0.5)
        for k in ("act", "done", "viol", "energy_q"):
            assert np.array_equal(cpu(buf[k]), ref[k]), k
        if it == 0:
            offs = np.full(64, 100, np.int32)
            pe.set_offsets(env, torch.from_numpy(offs).cuda())
            oenv.set_offsets(offs)
    assert np.array_equal(cpu(buf["energy_q"]), ref["energy_q"])
    env.close()


def test_rule_rollout_parity_72b_cadence():
    wl = W.make_72b_cadence(n_envs=64)
    spec = wl.env
    rule = W.hysteresis_rule(spec.budget_q)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    oenv = O.OracleEnv(spec, wl.trace, wl.phase, range(64))
    for it, T in ((0, 25), (1, 35)):
        buf = pe.alloc_rule_rollout(spec, T)
        pe.rollout_rule(env, rule, T, it, buf, lam=0.5)
        torch.cuda.synchronize()
        ref = oenv.rollout_rule(rule, T, it, lam=0.5)
        for k in ("act", "done", "viol", "energy_q", "samples", "q"):
            assert np.array_equal(cpu(buf[k]), ref[k]), k
        assert rel_err(cpu(buf["reward"]), ref["reward"]) <= TOL
    env.close()


def test_rollout_parity_tiny_ragged_tile():
    _rollout_case(W.make_tiny(n_envs=45), 3, iters=2)


def test_rollout_parity_tiny_deterministic():
    _rollout_case(W.make_tiny(n_envs=40), 64, iters=1, det=True)


def test_rollout_parity_7b_sampled():
    wl = W.make_7b()
    rng = np.random.default_rng(3)
    ids = np.unique(np.concatenate([[0, 31, 32, 4095], rng.choice(4096, 28, replace=False)]))
    _rollout_case(wl, 512, iters=2, sample_envs=ids)


def test_rollout_parity_72b_small():
    """bf16 tensor-core policy/value (D=32, H=256, A=16), 4 channels, Eq. 6
    reward; 512 envs x 600 steps crosses an episode boundary."""
    _rollout_case(W.make_72b(n_envs=512), 600, iters=1, lam=0.7)


def test_rollout_parity_72b_two_chains_ragged():
    """700 envs run as two stream chains split on a tile boundary (384 +
    316 envs, the second ending in a ragged tile); every env is replayed,
    including both sides of the split."""
    _rollout_case(W.make_72b(n_envs=700), 40, iters=2, lam=0.7)


def test_rollout_parity_72b_full_size_sampled():
    """The full 72B workload (65,536 envs x 1,024 steps); the oracle replays
    a seeded sample of envs including both ends and a tile boundary."""
    wl = W.make_72b()
    rng = np.random.default_rng(5)
    ids = np.unique(np.concatenate([[0, 127, 128, 32767, 32768, 65535], rng.choice(65536, 12, replace=False)]))
    _rollout_case(wl, 1024, iters=1, sample_envs=ids)


def test_rollout_parity_stress_small():
    """Stress network (D=64, H=512: weights streamed through a two-slot ring)
    on 512 envs x 520 steps of the 380,000-sample 4-channel trace."""
    _rollout_case(W.make_stress(n_envs=512, horizon=520), 520, iters=1, lam=0.4)


def test_rollout_parity_stress_full_size_sampled():
    """The full Stress workload (262,144 envs x 2,048 steps, 64-512-512 bf16);
    the oracle replays a seeded sample of envs."""
    wl = W.make_stress()
    rng = np.random.default_rng(9)
    ids = np.unique(np.concatenate([[0, 262143], rng.choice(262144, 6, replace=False)]))
    _rollout_case(wl, 2048, iters=1, sample_envs=ids)


def test_value_bf16_stress_ragged():
    net = W.NetSpec(64, 512, 16, pe.PE_BF16)
    params = W.init_params(net, seed=6, bias_scale=0.1)
    for n in (1, 255, 3000):
        obs = torch.randn(n, 64, generator=torch.Generator().manual_seed(n)).to(torch.bfloat16)
        out = torch.empty(n, device="cuda")
        pe.value(net, torch.from_numpy(params).cuda(), obs.cuda(), out)
        pe.device_check()
        _, ov = O.mlp_forward(net, params, obs.float().numpy())
        assert bf16_ok(cpu(out), ov)


def test_value_bf16_parity_ragged():
    net = W.NetSpec(32, 256, 16, pe.PE_BF16)
    params = W.init_params(net, seed=4, bias_scale=0.1)
    for n in (1, 127, 129, 5000):
        obs = torch.randn(n, 32, generator=torch.Generator().manual_seed(n)).to(torch.bfloat16)
        out = torch.empty(n, device="cuda")
        pe.value(net, torch.from_numpy(params).cuda(), obs.cuda(), out)
        pe.device_check()
        _, ov = O.mlp_forward(net, params, obs.float().numpy())
        assert bf16_ok(cpu(out), ov)


def test_env_checkpoint_roundtrip():
    wl = W.make_tiny(n_envs=50)
    params = torch.from_numpy(W.init_params(wl.net, seed=2)).cuda()
    a = pe.Env(wl.env, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    b = pe.Env(wl.env, torch.from_numpy(wl.trace).cuda(), torch.from_numpy(wl.phase).cuda())
    ba, bb = pe.alloc_rollout(wl.env, wl.net, 300), pe.alloc_rollout(wl.env, wl.net, 300)
    pe.rollout(a, wl.net, params, 300, 0, ba)
    pe.rollout(b, wl.net, params, 300, 0, bb)
    img = a.save()
    pe.rollout(a, wl.net, params, 300, 1, ba)
    b.load(img)
    pe.rollout(b, wl.net, params, 300, 1, bb)
    torch.cuda.synchronize()
    for k in ba:
        assert torch.equal(ba[k], bb[k]), k


def test_training_resume_is_bit_exact():
    """Checkpoint/resume of training: two Tiny iterations (rollout, GAE, PPO
    update) run straight equal one iteration, a save of the env state,
    parameters and Adam moments, a restore into fresh objects, and the second
    iteration -- every buffer and statistic bit for bit (the draws are
    counter-based on (seed, iteration, env, step), the reductions fixed-order)."""
    wl = W.make_tiny(n_envs=64)
    spec, net, T = wl.env, wl.net, 128
    ppo = W.PPOSpec(epochs=2, minibatch=2048)
    N = spec.n_envs * T

    def iteration(env, p, m, v, adam_t, it):
        buf = pe.alloc_rollout(spec, net, T)
        pe.rollout(env, net, p, T, it, buf)
        adv = torch.empty(T, spec.n_envs, device="cuda")
        ret = torch.empty_like(adv)
        pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], ppo.gamma, ppo.lam, adv, ret)
        stats = torch.zeros(8, device="cuda")
        ws = torch.empty(pe.ppo_workspace_bytes(net, ppo, N), dtype=torch.uint8, device="cuda")
        pe.ppo_update(net, ppo, p, m, v, adam_t, buf["obs"], buf["act"], buf["logp"], adv, ret, stats, ws,
                      seed=11, iteration=it)
        torch.cuda.synchronize()
        return buf, stats, adam_t + ppo.epochs * ((N + ppo.minibatch - 1) // ppo.minibatch)

    def fresh():
        env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
        p = torch.from_numpy(W.init_params(net, seed=5, bias_scale=0.05)).cuda()
        return env, p, torch.zeros_like(p), torch.zeros_like(p)

    env_a, pa, ma, va = fresh()
    _, _, ta = iteration(env_a, pa, ma, va, 0, 0)
    buf_a, st_a, _ = iteration(env_a, pa, ma, va, ta, 1)

    env_b, pb, mb, vb = fresh()
    _, _, tb = iteration(env_b, pb, mb, vb, 0, 0)
    ckpt = (env_b.save(), pb.cpu(), mb.cpu(), vb.cpu(), tb)
    env_b.close()
    env_c, pc, mc, vc = fresh()
    env_c.load(ckpt[0])
    pc.copy_(ckpt[1]); mc.copy_(ckpt[2]); vc.copy_(ckpt[3])
    buf_c, st_c, _ = iteration(env_c, pc, mc, vc, ckpt[4], 1)

    for k in buf_a:
        if buf_a[k] is not None:
            assert torch.equal(buf_a[k], buf_c[k]), k
    assert torch.equal(pa, pc) and torch.equal(ma, mc) and torch.equal(va, vc)
    assert torch.equal(st_a, st_c)
    env_a.close()
    env_c.close()


def test_env_rejects_bad_trace():
    wl = W.make_tiny(n_envs=4)
    tr = wl.trace.copy()
    tr[0, 100] = np.inf
    with pytest.raises(pe.PEError) as e:
        pe.Env(wl.env, torch.from_numpy(tr), torch.from_numpy(wl.phase))
    assert e.value.status == pe.PE_EOVERFLOW


# ------------------------------------------------------------------------ PPO
def _ppo_inputs(wl, T, seed=0):
    spec, net = wl.env, wl.net
    params = W.init_params(net, seed=seed, bias_scale=0.05)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rollout(spec, net, T)
    p_dev = torch.from_numpy(params).cuda()
    pe.rollout(env, net, p_dev, T, 0, buf)
    adv = torch.empty(T, spec.n_envs, device="cuda")
    ret = torch.empty_like(adv)
    pe.gae(buf["reward"], buf["value"], buf["done"], buf["last_value"], wl.ppo.gamma, wl.ppo.lam, adv, ret)
    torch.cuda.synchronize()
    env.close()
    return params, buf, adv, ret


def _run_ppo(wl, ppo, params, buf, adv, ret, iteration=0):
    net = wl.net
    N = buf["act"].numel()
    p = torch.from_numpy(params).cuda()
    m = torch.zeros_like(p)
    v = torch.zeros_like(p)
    stats = torch.zeros(8, device="cuda")
    ws = torch.empty(pe.ppo_workspace_bytes(net, ppo, N), dtype=torch.uint8, device="cuda")
    pe.ppo_update(net, ppo, p, m, v, 0, buf["obs"], buf["act"], buf["logp"], adv, ret, stats, ws,
                  seed=7, iteration=iteration)
    torch.cuda.synchronize()
    return cpu(p), cpu(m), cpu(v), cpu(stats)


def _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=0, max_steps=-1):
    P = params.size
    return O.ppo_update(wl.net, ppo, params, np.zeros(P), np.zeros(P), 0,
                        cpu(buf["obs"].float()).reshape(-1, wl.net.obs_dim), cpu(buf["act"]).ravel(),
                        cpu(buf["logp"]).ravel(), cpu(adv).ravel(), cpu(ret).ravel(), 7, iteration,
                        max_steps)


def assert_stats(gs, st, min_cnt, tol=TOL):
    """All eight update statistics.  [1] value loss, [2] entropy, [5] total
    loss, [6] last gradient norm: relative.  [0] the clipped surrogate is a
    mean of terms whose normalised advantages sum to zero, so its error is
    measured against max(|pg|, 1).  [3] approximate KL, a mean of about
    (log rho)^2 / 2: relative, plus an absolute floor for the log-ratio noise
    e of the two forward passes (fp32 against fp64 accumulation), which adds
    about mean(|log rho| e) + mean(e^2): 1e-9 for fp32 networks, and
    1e-3 sqrt(2 KL) + 1e-6 for bf16 networks, where a bf16 rounding flip of a
    hidden activation moves a logit by up to about 1e-3.  [4] clip fraction:
    the GPU decides |rho - 1| > clip in fp32, the oracle in fp64, so a sample
    within rounding of the boundary may count on one side only; at most one
    such sample per minibatch step.  [7] step count: exact."""
    assert gs[7] == st[7]
    for k in (1, 2, 5, 6):
        assert abs(gs[k] - st[k]) <= tol * max(abs(st[k]), 1e-3), (k, gs[k], st[k])
    assert abs(gs[0] - st[0]) <= tol * max(abs(st[0]), 1.0), (0, gs[0], st[0])
    floor = 1e-9 if tol <= TOL else 1e-3 * np.sqrt(2.0 * abs(st[3])) + 1e-6
    assert abs(gs[3] - st[3]) <= tol * abs(st[3]) + floor, (3, gs[3], st[3])
    assert abs(gs[4] - st[4]) <= 1.0 / min_cnt + 1e-7, (4, gs[4], st[4])


def assert_update_fp32(gp, gm, gv, P, m, v):
    """fp32 update after several steps: parameters and Adam's first moment
    within the benchmark spec's 1e-5 (rms-floored relative); the second moment is
    quadratic in the gradient, so twice that."""
    assert rel_err(gm, m) <= TOL, rel_err(gm, m)
    assert rel_err(gv, v) <= 2 * TOL, rel_err(gv, v)
    assert rel_err(gp, P) <= TOL, rel_err(gp, P)


def test_ppo_single_step_parity():
    """One minibatch step: Adam's first moment after one step is
    (1 - beta1) * the clipped gradient, so it exposes the gradient itself."""
    wl = W.make_tiny()
    params, buf, adv, ret = _ppo_inputs(wl, 128)
    ppo = W.PPOSpec(epochs=1, minibatch=8192)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret)
    assert t == 1
    assert_update_fp32(gp, gm, gv, P, m, v)
    assert_stats(gs, st, 8192)
    # first step: the policy is the rollout's, rho = 1 on both sides
    assert abs(gs[3]) < 1e-9 and gs[4] == 0.0 and st[4] == 0.0


@pytest.mark.parametrize("clip", [0.2, 0.01])
def test_ppo_ragged_minibatches(clip):
    """3 steps over minibatches of 3000, 3000 and 2192 samples; the small clip
    range makes the later steps clip a share of their samples."""
    wl = W.make_tiny()
    params, buf, adv, ret = _ppo_inputs(wl, 128, seed=1)
    ppo = W.PPOSpec(epochs=1, minibatch=3000, clip=clip)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=5)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=5)
    assert t == 3 and gs[7] == 3
    assert_update_fp32(gp, gm, gv, P, m, v)
    assert_stats(gs, st, 2192)
    assert st[3] > 0.0


@pytest.mark.parametrize("clip", [0.2, 0.01])
def test_ppo_full_update_tiny(clip):
    """4 epochs x 4 minibatches (ragged last one: 8192 = 3*2500 + 692)."""
    wl = W.make_tiny()
    params, buf, adv, ret = _ppo_inputs(wl, 128, seed=3)
    ppo = W.PPOSpec(epochs=4, minibatch=2500, clip=clip)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=2)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=2)
    assert t == 16 and gs[7] == 16
    assert_update_fp32(gp, gm, gv, P, m, v)
    assert_stats(gs, st, 692)
    if clip < 0.1:
        assert st[4] > 0.05   # the clip fraction is exercised


@pytest.mark.parametrize("clip,lr,ent", [(0.2, 3e-4, 0.0), (0.01, 3e-4, 0.0), (0.2, 3e-3, 0.01)])
def test_ppo_7b_multi_epoch_persistent(clip, lr, ent):
    """The 7B networks (16-128-128x5, the persistent update kernel that the
    benchmark runs for 1,024 steps per launch) over 2 epochs x 3 minibatches
    (3000, 3000, 2192) of 8,192 samples: from the second step on, every CTA
    reads the weight images that the previous step's Adam phase rewrote.
    Parameters, both moments and all statistics against the oracle."""
    wl = W.make_7b(n_envs=128)
    params, buf, adv, ret = _ppo_inputs(wl, 64, seed=4)
    ppo = W.PPOSpec(epochs=2, minibatch=3000, clip=clip, lr=lr, ent_coef=ent)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    assert t == 6 and gs[7] == 6
    assert_update_fp32(gp, gm, gv, P, m, v)
    assert_stats(gs, st, 2192)
    assert st[3] > 0.0
    if clip < 0.1 or lr > 1e-3:
        assert st[4] > 0.05


def test_ppo_7b_first_steps():
    wl = W.make_7b(n_envs=512)
    params, buf, adv, ret = _ppo_inputs(wl, 64)
    ppo = W.PPOSpec(epochs=1, minibatch=32768)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret)
    assert rel_err(gm, m) <= TOL and rel_err(gp, P) <= TOL
    assert_stats(gs, st, 32768)


@pytest.mark.parametrize("n", [60, 1000, 4999, 8192])
def test_ppo_7b_single_step_partitions(n):
    """One step over n samples of the 7B networks.  The update gives each CTA
    ceil(n / NC) consecutive samples (NC = 76 per network on 152 SMs, fewer
    for small n), in slices of up to 64 whose tiles stop at the valid rows
    rounded up to 8: n = 60 (8-sample shares, the last one short), 1000
    (14-sample shares, the last CTAs empty), 4999 (a 2-sample second slice)
    and 8192 (the bench's 64 + 44)."""
    wl = W.make_7b(n_envs=512)
    params, buf, adv, ret = _ppo_inputs(wl, 64, seed=4)
    D = wl.net.obs_dim
    sub = {"obs": buf["obs"].reshape(-1, D)[:n].contiguous(), "act": buf["act"].reshape(-1)[:n].contiguous(),
           "logp": buf["logp"].reshape(-1)[:n].contiguous()}
    a_, r_ = adv.reshape(-1)[:n].contiguous(), ret.reshape(-1)[:n].contiguous()
    ppo = W.PPOSpec(epochs=1, minibatch=n)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, sub, a_, r_)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, sub, a_, r_)
    assert t == 1 and gs[7] == 1
    assert rel_err(gm, m) <= TOL and rel_err(gp, P) <= TOL
    assert_stats(gs, st, n)


# ------------------------------------------------------------------ bf16 PPO
BF16_TOL = 2e-2


@pytest.mark.parametrize("preset,E,T", [("72b", 64, 64), ("stress", 32, 64)])
def test_ppo_bf16_single_step(preset, E, T):
    """One minibatch over all N = T*E samples of a bf16 network: tensor-core
    forward over the permuted rows, tensor-core backward, own loss, reduction
    and Adam.  Adam's first moment after one step is 0.1 x the clipped
    gradient."""
    wl = W.make_72b(n_envs=E) if preset == "72b" else W.make_stress(n_envs=E, horizon=T)
    params, buf, adv, ret = _ppo_inputs(wl, T, seed=2)
    ppo = W.PPOSpec(epochs=1, minibatch=T * E, ent_coef=0.01)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    assert t == 1 and gs[7] == 1
    assert bf16_ok(gm, m), (np.abs(gm - m).max() / np.abs(m).max())
    assert_stats(gs, st, T * E, tol=BF16_TOL)


@pytest.mark.parametrize("preset,E,T", [("72b", 320, 128), ("stress", 160, 122)])
def test_ppo_bf16_several_tiles_per_cta(preset, E, T):
    """One minibatch large enough that the persistent kernels take more than
    one tile (pair) per CTA: 72B 40,960 samples = 320 tiles over 152 CTAs
    (the first 16 run two tile pairs, the second half empty); Stress 19,520
    samples = 153 tiles per network, whose forward and backward-data
    launches spread the 306 tiles of both networks over the 152 CTAs (two
    or three each, most CTAs crossing from a policy tile to a value tile).
    Adam's first moment after one step is 0.1 x the clipped gradient."""
    wl = W.make_72b(n_envs=E) if preset == "72b" else W.make_stress(n_envs=E, horizon=T)
    params, buf, adv, ret = _ppo_inputs(wl, T, seed=4)
    ppo = W.PPOSpec(epochs=1, minibatch=T * E, ent_coef=0.01)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=1)
    assert t == 1 and gs[7] == 1
    assert bf16_ok(gm, m), (np.abs(gm - m).max() / np.abs(m).max())
    assert_stats(gs, st, T * E, tol=BF16_TOL)


@pytest.mark.parametrize("preset,E,mb,clip", [("72b", 64, 1500, 0.2), ("72b", 64, 1500, 0.01),
                                              ("stress", 32, 900, 0.01)])
def test_ppo_bf16_ragged_epochs(preset, E, mb, clip):
    """2 epochs x 3 ragged minibatches of T * E = 64 * E samples (72B: 1500,
    1500, 1096; Stress: 900, 900, 248).  The oracle emulates the GPU's bf16
    rounding points, so what remains is fp32 against fp64 accumulation and
    rare 1-ulp rounding flips: the moments, the parameters and their moves
    from the start must agree within the benchmark spec's 2e-2 (rms-floored
    relative; the moves measured 1.4e-2 on the 72B networks, the rest about
    2e-4 there and 1.3e-3 on the wider Stress networks), and the first
    moment also within 5e-3, which a dropped term or a wrongly scaled
    gradient exceeds."""
    T = 64
    wl = W.make_72b(n_envs=E) if preset == "72b" else W.make_stress(n_envs=E, horizon=T)
    params, buf, adv, ret = _ppo_inputs(wl, T, seed=4)
    ppo = W.PPOSpec(epochs=2, minibatch=mb, ent_coef=0.01, clip=clip)
    gp, gm, gv, gs = _run_ppo(wl, ppo, params, buf, adv, ret, iteration=3)
    P, m, v, t, st = _oracle_ppo(wl, ppo, params, buf, adv, ret, iteration=3)
    assert t == 6 and gs[7] == 6
    assert rel_err(gm, m) <= 5e-3, rel_err(gm, m)
    assert rel_err(gv, v) <= BF16_TOL and rel_err(gp, P) <= BF16_TOL
    assert rel_err(gp - params, P - params) <= BF16_TOL, rel_err(gp - params, P - params)
    assert_stats(gs, st, T * E - 2 * mb, tol=BF16_TOL)
    assert st[3] > 0.0
    if clip < 0.1:
        assert st[4] > 0.05


# ------------------------------------------------------- baseline rule policies
def _rule_for(kind, preset, B):
    if kind == 1:
        return W.random_rule()
    if preset == "tiny":  # thresholds between the tiny levels
        return W.threshold_rule(B, 1.1, 0.98) if kind == 2 else W.hysteresis_rule(B, 1.1, 0.98, 1.05)
    return W.threshold_rule(B) if kind == 2 else W.hysteresis_rule(B)


@pytest.mark.parametrize("preset", ["tiny", "7b", "72b"])
@pytest.mark.parametrize("kind", [1, 2, 3])
def test_rule_rollout_parity(preset, kind):
    """Rule-policy rollouts from explicit episode starts, two calls in a row
    (state carried across calls, episode boundaries crossed): actions, done
    flags, violation counts and energy bit-exact; rewards, tokens and excess
    within 1e-5; the final observation bit-exact."""
    E = 64
    wl = {"tiny": W.make_tiny, "7b": W.make_7b, "72b": W.make_72b}[preset](n_envs=E)
    spec = wl.env
    rule = _rule_for(kind, preset, spec.budget_q)
    offs = W.replay_offsets(wl.trace.shape[-1], spec.episode_len)
    offs = np.resize(offs, E).astype(np.int32)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    pe.set_offsets(env, torch.from_numpy(offs).cuda())
    oenv = O.OracleEnv(spec, wl.trace, wl.phase, range(E))
    oenv.set_offsets(offs)
    bf16 = preset == "72b"
    for it, T in ((0, 300), (1, 450)):
        buf = pe.alloc_rule_rollout(spec, T, obs=True, obs_bf16=bf16)
        pe.rollout_rule(env, rule, T, it, buf, lam=0.5)
        torch.cuda.synchronize()
        ref = oenv.rollout_rule(rule, T, it, lam=0.5)
        assert np.array_equal(cpu(buf["act"]), ref["act"])
        assert np.array_equal(cpu(buf["done"]), ref["done"])
        assert np.array_equal(cpu(buf["viol"]), ref["viol"])
        assert np.array_equal(cpu(buf["energy_q"]), ref["energy_q"])
        assert rel_err(cpu(buf["reward"]), ref["reward"]) <= TOL
        assert rel_err(cpu(buf["tokens"]), ref["tokens"]) <= TOL
        assert rel_err(cpu(buf["excess"]), ref["excess"]) <= TOL
        o_last = oenv.obs()
        g_last = cpu(buf["obs_last"].float())
        if bf16:
            o_last = torch.from_numpy(o_last).to(torch.bfloat16).float().numpy()
        assert np.array_equal(g_last, o_last)
    env.close()


@pytest.mark.parametrize("preset", ["tiny", "7b", "72b"])
def test_replay_rollout_parity(preset):
    """Teacher-forced rollouts (pe_rollout_replay) of seeded random actions,
    two calls in a row crossing episode ends, against the oracle stepping
    with the same forced actions: observations (bf16 after RNE for the 72B
    env), done flags, violation counts, energy and per-step power bit-exact;
    rewards, tokens and excess within 1e-5."""
    E = 64
    wl = {"tiny": W.make_tiny, "7b": W.make_7b, "72b": W.make_72b}[preset](n_envs=E)
    spec, net = wl.env, wl.net
    bf16 = preset == "72b"
    params = W.init_params(net, seed=2, bias_scale=0.05)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    oenv = O.OracleEnv(spec, wl.trace, wl.phase, range(E))
    rng = np.random.default_rng(9)
    for it, T in ((0, 300), (1, 450)):
        acts = rng.integers(0, spec.n_actions, (T, E)).astype(np.uint8)
        buf = pe.alloc_rule_rollout(spec, T, obs=True, obs_bf16=bf16)
        pe.rollout_replay(env, torch.from_numpy(acts).cuda(), T, it, buf, lam=0.5)
        torch.cuda.synchronize()
        ref = oenv.rollout(params, net.hidden, bf16, T, it, lam=0.5, forced=acts)
        want_obs, want_last = ref["obs"], ref["obs_last"]
        if bf16:
            want_obs = torch.from_numpy(want_obs).to(torch.bfloat16).float().numpy()
            want_last = torch.from_numpy(want_last).to(torch.bfloat16).float().numpy()
        assert np.array_equal(cpu(buf["act"]), acts)
        assert np.array_equal(cpu(buf["obs"].float()), want_obs)
        assert np.array_equal(cpu(buf["obs_last"].float()), want_last)
        assert np.array_equal(cpu(buf["done"]), ref["done"])
        assert ref["done"].any() or it == 0
        assert np.array_equal(cpu(buf["viol"]), ref["viol"])
        assert np.array_equal(cpu(buf["energy_q"]), ref["energy_q"])
        assert np.array_equal(cpu(buf["samples"]), ref["samples"])
        assert np.array_equal(cpu(buf["q"]), ref["q"])
        assert rel_err(cpu(buf["reward"]), ref["reward"]) <= TOL
        assert rel_err(cpu(buf["tokens"]), ref["tokens"]) <= TOL
        assert rel_err(cpu(buf["excess"]), ref["excess"]) <= TOL
    env.close()


def test_replay_reproduces_policy_rollout():
    """Replaying the actions a 7B policy rollout took, from the same saved env
    state, reproduces that rollout's observations, rewards, done flags,
    counters and final state bit for bit (the same env step on both paths)."""
    wl = W.make_7b(n_envs=256)
    spec, net = wl.env, wl.net
    T = 600
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    snap = env.save()
    p_dev = torch.from_numpy(W.init_params(net, seed=3, bias_scale=0.05)).cuda()
    buf = pe.alloc_rollout(spec, net, T)
    pe.rollout(env, net, p_dev, T, 4, buf, lam=0.7)
    after = env.save()
    env.load(snap)
    rb = pe.alloc_rule_rollout(spec, T, obs=True)
    pe.rollout_replay(env, buf["act"].contiguous(), T, 4, rb, lam=0.7)
    torch.cuda.synchronize()
    for k in ("obs", "obs_last", "act", "reward", "done", "viol", "tokens", "excess", "energy_q", "samples", "q"):
        assert torch.equal(buf[k], rb[k]), k
    assert env.save() == after
    env.close()


def test_replay_rejects_bad_actions():
    wl = W.make_tiny(n_envs=8)
    spec = wl.env
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    acts = torch.zeros((5, 8), dtype=torch.uint8, device="cuda")
    acts[3, 2] = spec.n_actions
    buf = pe.alloc_rule_rollout(spec, 5)
    with pytest.raises(pe.PEError) as e:
        pe.rollout_replay(env, acts, 5, 0, buf)
    assert e.value.status == pe.PE_EINVAL and "outside" in str(e.value)
    env.close()


def test_rule_rollout_full_size_sampled():
    """The 72B env at full size (65,536 envs x 1,024 steps) under the
    hysteresis rule from the random initial offsets; the oracle replays a
    seeded sample of envs."""
    wl = W.make_72b()
    spec = wl.env
    E, T = spec.n_envs, 1024
    rule = W.hysteresis_rule(spec.budget_q)
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    buf = pe.alloc_rule_rollout(spec, T)
    pe.rollout_rule(env, rule, T, 2, buf, lam=1.0)
    torch.cuda.synchronize()
    ids = np.random.default_rng(9).choice(E, 24, replace=False)
    oenv = O.OracleEnv(spec, wl.trace, wl.phase, ids)
    ref = oenv.rollout_rule(rule, T, 2, lam=1.0)
    ids_t = torch.from_numpy(ids).cuda()
    assert np.array_equal(cpu(buf["act"][:, ids_t]), ref["act"])
    assert np.array_equal(cpu(buf["viol"][ids_t]), ref["viol"])
    assert np.array_equal(cpu(buf["energy_q"][ids_t]), ref["energy_q"])
    assert rel_err(cpu(buf["reward"][:, ids_t]), ref["reward"]) <= TOL
    env.close()


def test_set_offsets_rejects_out_of_range():
    wl = W.make_tiny(n_envs=4)
    env = pe.Env(wl.env, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    bad = torch.tensor([60, 100, wl.trace.shape[-1] - wl.env.episode_len + 1, 70], dtype=torch.int32).cuda()
    with pytest.raises(pe.PEError) as e:
        pe.set_offsets(env, bad)
    assert e.value.status == pe.PE_EINVAL
    with pytest.raises(pe.PEError) as e:
        pe.rollout_rule(env, W.RuleSpec(7), 10, 0, pe.alloc_rule_rollout(wl.env, 10))
    assert e.value.status == pe.PE_EINVAL
    env.close()


# ------------------------------------------------------------- dual ascent
def test_dual_ascent_parity_in_a_lagrange_loop():
    """Three 72B rollouts with the Eq. 6 reward, lambda fed back through
    Eq. 7 on the device after each: the observed rates and multipliers
    match the oracle's update applied to the same counts (fp32 lambda)."""
    wl = W.make_72b(n_envs=256)
    spec = wl.env
    env = pe.Env(spec, torch.from_numpy(wl.trace), torch.from_numpy(wl.phase))
    T = 200
    buf = pe.alloc_rule_rollout(spec, T)
    lam = torch.tensor([1.0], device="cuda")
    rate = torch.zeros(1, device="cuda")
    lam_host = 1.0
    for it, (add, tgt) in enumerate(((False, 0.08), (False, 0.02), (True, 0.3))):
        pe.rollout_rule(env, W.random_rule(), T, it, buf, lam=lam_host)
        pe.dual_ascent(buf["viol"], T, lam, rate, target=tgt, additive=add, hi=2.0 if not add else 20.0)
        torch.cuda.synchronize()
        o_lam, o_rate = O.dual_ascent(cpu(buf["viol"]), T, lam_host, target=tgt, additive=add,
                                      hi=2.0 if not add else 20.0)
        assert abs(float(rate.item()) - o_rate) <= 1e-7 * max(o_rate, 1e-3)
        assert abs(float(lam.item()) - o_lam) <= 2e-7 * abs(o_lam)
        lam_host = float(lam.item())
    with pytest.raises(pe.PEError):
        pe.dual_ascent(buf["viol"], T, lam, rate, window=30)
    env.close()
