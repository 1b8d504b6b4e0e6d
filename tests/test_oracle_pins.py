"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: published
known-answer vectors, brute force on tiny inputs, closed forms, finite
differences, library routines for special cases, and invariants.
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_11226_gb300 import workloads as W
from tests.envref import BruteEnv

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------- Philox
def test_philox_known_answers():
    rows = 0
    for line in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")):
        if line.startswith("#") or not line.strip():
            continue
        v = [int(x, 16) for x in line.split()]
        out = O.philox4x32_10(v[0:4], v[4:6])
        assert list(out) == v[6:10]
        rows += 1
    assert rows == 3


# -------------------------------------------------------------------- Feistel
@pytest.mark.parametrize("n", [1, 2, 3, 5, 64, 1000, 8192, 10007])
def test_feistel_is_a_permutation(n):
    keys = O.perm_keys(7, 1, 3)
    p = O.feistel_perm(n, keys)
    assert sorted(p.tolist()) == list(range(n))
    if n >= 64:  # not the identity and differs across epochs
        assert not np.array_equal(p, np.arange(n))
        assert not np.array_equal(p, O.feistel_perm(n, O.perm_keys(7, 2, 3)))


# ----------------------------------------------------------------------- bf16
def test_bf16_round_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(2000) * 10.0 ** rng.integers(-6, 6, 2000),
                        [1.0, -1.0, 1.00390625, 1.01171875, 3.0e-3]])
    ref = torch.tensor(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([O.bf16_round(float(np.float32(v))) for v in x])
    assert np.array_equal(got, ref)


# ------------------------------------------------------------------- actuator
def test_group_size_actuator_formula():
    """Sec. 4.1: P = trace * (0.8 + 0.2 G / G_max), here G_max = 8."""
    spec = W.make_7b(n_envs=4).env
    for G, want in zip(range(3, 9), [0.875, 0.9, 0.925, 0.95, 0.975, 1.0]):
        assert O.actuator_scale(spec, G) == np.float32(want)


# -------------------------------------------------------- env vs brute force
def _brute_compare(wl, n_envs, T, iters=1, seed_actions=0):
    spec = wl.env
    ids = list(range(n_envs))
    env = O.OracleEnv(spec, wl.trace, wl.phase, ids)
    brutes = [BruteEnv(spec, wl.trace.astype(np.float32), wl.phase, e, O.philox4x32_10) for e in ids]
    rng = np.random.default_rng(seed_actions)
    params = W.init_params(wl.net)
    for it in range(iters):
        forced = rng.integers(0, spec.n_actions, size=(T, n_envs)).astype(np.uint8)
        out = env.rollout(params, wl.net.hidden, wl.net.dtype == 1, T, it, lam=0.7, forced=forced)
        for i, b in enumerate(brutes):
            v1 = v60 = 0
            en = smp = 0
            tok = exc = 0.0
            for t in range(T):
                o = b.obs()
                assert np.array_equal(out["obs"][t, i], o), (it, t, i)
                st = b.step(int(forced[t, i]), 0.7, t, it)
                assert out["done"][t, i] == st["done"] and out["q"][t, i] == st["q"]
                assert abs(out["reward"][t, i] - st["r"]) <= 1e-12 * max(1.0, abs(st["r"]))
                v1 += st["v1"]; v60 += st["v60"]; en += st["q"]; smp += st["samples"]
                tok += st["tokens"]; exc += st["excess"]
            assert np.array_equal(out["obs_last"][i], b.obs())
            assert list(out["viol"][i]) == [v1, v60]
            assert out["energy_q"][i] == en
            assert out["samples"][i] == smp
            assert abs(out["tokens"][i] - tok) <= 1e-9 * max(1.0, tok)
            assert abs(out["excess"][i] - exc) <= 1e-9 * max(1.0, exc)


def test_env_72b_cadence_matches_bruteforce():
    """Batch-boundary cadence (Sec. 4.5): a step consumes 24-42 samples by
    level, the Eq. 6 reward sums the batch with its peak 30 s excess, and
    episodes of 40 batches; two iterations cross an episode boundary."""
    wl = W.make_72b_cadence(n_envs=2)
    _brute_compare(wl, 2, 45, iters=2)


def test_env_mixed_families_matches_bruteforce():
    """Domain randomisation (Sec. 4.2 G2): each episode draws its trace
    family (4-GPU 72B-, 2-GPU 14B- or 1-GPU 7B-shaped, each with its own
    budget) from word 1 of the episode draw and its offset from word 0; the
    oracle's per-family view matches the brute-force env across episode
    boundaries, and more than one family is visited."""
    wl = W.make_72b_mixed(n_envs=4)
    _brute_compare(wl, 4, 520, iters=2)
    seen = set()
    for e in range(4):
        b = BruteEnv(wl.env, wl.trace, wl.phase, e, O.philox4x32_10)
        seen.add(b.fam)
        for t in range(3):
            b.reset(t, 0, 1)
            seen.add(b.fam)
    assert len(seen) == 3


def test_env_tiny_matches_bruteforce():
    _brute_compare(W.make_tiny(n_envs=3), 3, 620, iters=2)


def test_env_7b_matches_bruteforce():
    _brute_compare(W.make_7b(n_envs=3), 3, 520)


def test_env_72b_matches_bruteforce():
    wl = W.make_72b(n_envs=2)
    _brute_compare(wl, 2, 510)


def test_env_occ64_matches_bruteforce():
    wl = W._occ_workload("occ64", 2, 3000, W.OBS_OCC64, 32, 64, 0, W.PPOSpec(1, 64))
    _brute_compare(wl, 2, 505)


def _const_spec(level_w_q: int, budget: int):
    """Constant trace whose actuated sample is exactly level_w_q / 64 W."""
    trace = np.full((1, 2000), level_w_q / 64.0, np.float32)
    phase = np.zeros(2000, np.uint8)
    spec = W.EnvSpec(
        n_envs=1, n_channels=1, trace_len=2000, n_actions=2, obs_kind=W.OBS_TINY8,
        actuator_kind=W.ACT_SET_LEVEL, n_levels=2, level_init=0, g_min=0, g_max=1, b_min=1,
        b_max=1, b_init=1, episode_len=500, budget_q=budget, scale_phase_mask=0b11,
        level_scale=[[1.0], [1.0]], level_tokens=[10.0, 10.0], reward_kind=W.REWARD_FIXED,
        reward_window=60, r_ok=1.0, r_viol=-8.0, bonus_coef=0.0, seed=3)
    return spec, trace, phase


@pytest.mark.parametrize("delta,expect", [(1, 1), (0, 0), (-1, 0)])
def test_violation_counts_hand_computed(delta, expect):
    """Eq. 2 on a constant trace at B + delta/64 W: every sample violates iff delta > 0."""
    B = 300 * 64
    spec, trace, phase = _const_spec(B + delta, B)
    env = O.OracleEnv(spec, trace, phase, [0])
    T = 700
    out = env.rollout(np.zeros(W.param_count(8, 4, 2), np.float32), 4, False, T, 0,
                      forced=np.zeros((T, 1), np.uint8))
    assert list(out["viol"][0]) == [expect * T, expect * T]
    assert out["energy_q"][0] == T * (B + delta)
    assert np.all(out["reward"] == (-8.0 if expect else 1.0))
    assert out["done"][:, 0].sum() == 1 and out["done"][499, 0] == 1
    # Eq. 3: X = max(0, P30 - B) * dt = (1/64 W) * 0.5 s per violating sample
    assert out["excess"][0] == pytest.approx(expect * T * 0.5 / 64.0, rel=1e-12)


def test_episode_offsets_in_range():
    wl = W.make_7b(n_envs=256)
    env = O.OracleEnv(wl.env, wl.trace, wl.phase, list(range(256)))
    st = env.state.view(np.int32).reshape(256, -1)
    pos = st[:, 0]
    assert pos.min() >= 60 and pos.max() <= wl.env.trace_len - 500
    assert len(np.unique(pos)) > 200


# ------------------------------------------------------------------------ MLP
def _torch_mlp(net, params, obs, bf16=False):
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    p = torch.tensor(params.astype(np.float64))
    sizes = [H * D, H, H * H, H, A * H, A, H * D, H, H * H, H, H, 1]
    parts = list(torch.split(p, sizes))
    x = torch.tensor(obs.astype(np.float64))

    def rb(t):
        return t.float().to(torch.bfloat16).double() if bf16 else t

    def net_fwd(W1, b1, W2, b2, W3, b3, out):
        h = rb(torch.tanh(rb(x) @ rb(W1.view(H, D)).T + b1))
        h = rb(torch.tanh(h @ rb(W2.view(H, H)).T + b2))
        return h @ rb(W3.view(out, H)).T + b3

    return net_fwd(*parts[:6], A).numpy(), net_fwd(*parts[6:], 1).numpy()[:, 0]


@pytest.mark.parametrize("bf16", [False, True])
def test_mlp_matches_torch(bf16):
    net = W.NetSpec(16, 32, 5, int(bf16))
    params = W.init_params(net, seed=3, bias_scale=0.1)
    obs = np.random.default_rng(1).standard_normal((50, 16)).astype(np.float32)
    lg, v = O.mlp_forward(net, params, obs)
    tl, tv = _torch_mlp(net, params, obs, bf16)
    tol = 1e-12 if not bf16 else 1e-2
    assert np.allclose(lg, tl, rtol=tol, atol=tol) and np.allclose(v, tv, rtol=tol, atol=tol)


def test_mlp_hand_computed_2_2_2():
    net = W.NetSpec(2, 2, 2, 0)
    # policy W1=[[1,0],[0,1]] b1=0; W2=[[1,1],[0,-1]] b2=[0,0.5]; W3=[[1,0],[0,2]] b3=[0.1,0]
    pol = [1, 0, 0, 1, 0, 0, 1, 1, 0, -1, 0, 0.5, 1, 0, 0, 2, 0.1, 0]
    val = [2, 0, 0, 0, 0, 0, 1, 0, 0, 0, 0, 0, 3, 0, -1]
    params = np.array(pol + val, np.float32)
    x = np.array([[0.5, -0.25]], np.float32)
    lg, v = O.mlp_forward(net, params, x)
    h1 = np.tanh([0.5, -0.25])
    h2 = np.tanh([h1[0] + h1[1], -h1[1] + 0.5])
    assert lg[0] == pytest.approx([h2[0] + float(np.float32(0.1)), 2 * h2[1]], rel=1e-12)
    g = np.tanh(np.tanh(1.0))
    assert v[0] == pytest.approx(3 * g - 1.0, rel=1e-12)


def test_mlp_zero_weights_uniform():
    net = W.NetSpec(8, 16, 3, 0)
    params = np.zeros(W.param_count(8, 16, 3), np.float32)
    params[-1] = 0.75  # value output bias
    lg, v = O.mlp_forward(net, params, np.ones((4, 8), np.float32))
    assert np.all(lg == 0.0) and np.all(v == 0.75)


# -------------------------------------------------------------------- sampler
def _bias_only_params(net, b3):
    p = np.zeros(W.param_count(net.obs_dim, net.hidden, net.n_actions), np.float32)
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    off = H * D + H + H * H + H + A * H
    p[off:off + A] = b3
    return p


def test_sampler_inverse_cdf_and_frequencies():
    wl = W.make_7b(n_envs=64)
    b3 = np.array([0.3, -1.0, 1.2, 0.0, -0.4], np.float32)
    params = _bias_only_params(wl.net, b3)
    ids = list(range(64))
    env = O.OracleEnv(wl.env, wl.trace, wl.phase, ids)
    T = 512
    out = env.rollout(params, wl.net.hidden, False, T, 5)
    z = b3.astype(np.float64)
    pr = np.exp(z - z.max()) / np.exp(z - z.max()).sum()
    cdf = np.cumsum(pr)
    key = [wl.env.seed & 0xFFFFFFFF, wl.env.seed >> 32]
    for t in range(0, T, 37):
        for i in ids:
            u = (int(O.philox4x32_10([i, t, 5, 0], key)[0]) >> 8) / 2.0 ** 24
            assert out["act_own"][t, i] == int(np.searchsorted(cdf, u, side="right"))
    counts = np.bincount(out["act_own"].ravel(), minlength=5)
    n = counts.sum()
    sigma = np.sqrt(n * pr * (1 - pr))
    assert np.all(np.abs(counts - n * pr) < 5 * sigma)
    lp = np.log(pr)
    assert np.allclose(out["logp"], lp[out["act_own"]], rtol=1e-12, atol=1e-12)
    det = O.OracleEnv(wl.env, wl.trace, wl.phase, ids).rollout(params, wl.net.hidden, False, 8, 5,
                                                                deterministic=True)
    assert np.all(det["act_own"] == 2)


# ------------------------------------------------------------------------ GAE
def test_gae_closed_form_constant():
    T, E, g, l, r, v = 50, 3, 0.99, 0.95, 0.75, 2.0  # r, v exact in fp32
    adv, ret = O.gae(np.full((T, E), r), np.full((T, E), v), np.zeros((T, E)), np.full(E, v), g, l)
    t = np.arange(T)
    want = (r + (g - 1) * v) * (1 - (g * l) ** (T - t)) / (1 - g * l)
    assert np.allclose(adv[:, 0], want, rtol=1e-12)
    assert np.allclose(ret, adv + v)


def test_gae_special_cases():
    rng = np.random.default_rng(0)
    T, E = 40, 4
    r = rng.standard_normal((T, E)).astype(np.float32)
    v = rng.standard_normal((T, E)).astype(np.float32)
    lv = rng.standard_normal(E).astype(np.float32)
    d = (rng.random((T, E)) < 0.1).astype(np.uint8)
    r64, v64, lv64 = r.astype(np.float64), v.astype(np.float64), lv.astype(np.float64)
    vn = np.vstack([v64[1:], lv64[None]])
    # lambda = 0: A = delta
    adv, _ = O.gae(r, v, d, lv, 0.99, 0.0)
    assert np.allclose(adv, r64 + 0.99 * (1 - d) * vn - v64, rtol=1e-12, atol=1e-12)
    # gamma = lambda = 1, no dones: A_t = sum_{k>=t} r_k + V_T - V_t
    adv, _ = O.gae(r, v, np.zeros_like(d), lv, 1.0, 1.0)
    want = np.cumsum(r64[::-1], 0)[::-1] + lv64[None] - v64
    assert np.allclose(adv, want, rtol=1e-10, atol=1e-10)
    # every step terminal: A_t = r_t - V_t
    adv, _ = O.gae(r, v, np.ones_like(d), lv, 0.99, 0.95)
    assert np.allclose(adv, r64 - v64, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------------------ PPO
def _ppo_batch(net, M, seed=0):
    rng = np.random.default_rng(seed)
    obs = rng.standard_normal((M, net.obs_dim)).astype(np.float32)
    act = rng.integers(0, net.n_actions, M).astype(np.uint8)
    lpo = (np.log(1.0 / net.n_actions) + 0.3 * rng.standard_normal(M)).astype(np.float32)
    adv = rng.standard_normal(M).astype(np.float32)
    ret = rng.standard_normal(M).astype(np.float32)
    return obs, act, lpo, adv, ret


def _torch_ppo_loss(net, params, obs, act, lpo, adv, ret, clip, vf, ent):
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    p = torch.tensor(params, dtype=torch.float64, requires_grad=True)
    sizes = [H * D, H, H * H, H, A * H, A, H * D, H, H * H, H, H, 1]
    W1, b1, W2, b2, W3, b3, V1, c1, V2, c2, V3, c3 = torch.split(p, sizes)
    x = torch.tensor(obs, dtype=torch.float64)
    z = torch.tanh(torch.tanh(x @ W1.view(H, D).T + b1) @ W2.view(H, H).T + b2) @ W3.view(A, H).T + b3
    V = (torch.tanh(torch.tanh(x @ V1.view(H, D).T + c1) @ V2.view(H, H).T + c2) @ V3.view(1, H).T + c3)[:, 0]
    logp_all = torch.log_softmax(z, -1)
    lp = logp_all[torch.arange(len(act)), torch.tensor(act, dtype=torch.long)]
    a = torch.tensor(adv, dtype=torch.float64)
    a = (a - a.mean()) / (a.std() + 1e-8)
    rho = torch.exp(lp - torch.tensor(lpo, dtype=torch.float64))
    pg = -torch.min(rho * a, torch.clamp(rho, 1 - clip, 1 + clip) * a).mean()
    vl = ((torch.tensor(ret, dtype=torch.float64) - V) ** 2).mean()
    H_ = -(logp_all.exp() * logp_all).sum(-1).mean()
    loss = pg + vf * vl - ent * H_
    loss.backward()
    return loss.item(), p.grad.numpy()


def test_ppo_gradient_matches_autograd_and_finite_differences():
    net = W.NetSpec(6, 8, 4, 0)
    params = W.init_params(net, seed=5, bias_scale=0.1).astype(np.float64)
    batch = _ppo_batch(net, 32)
    loss, grad, _ = O.ppo_minibatch_grad(net, params, *batch, 0.2, 0.5, 0.01)
    tl, tg = _torch_ppo_loss(net, params, *batch, 0.2, 0.5, 0.01)
    assert loss == pytest.approx(tl, rel=1e-12)
    assert np.allclose(grad, tg, rtol=1e-9, atol=1e-12)
    rng = np.random.default_rng(1)
    h = 1e-6
    for k in rng.choice(len(params), 40, replace=False):
        pp, pm = params.copy(), params.copy()
        pp[k] += h
        pm[k] -= h
        lp_, _, _ = O.ppo_minibatch_grad(net, pp, *batch, 0.2, 0.5, 0.01, want_grad=False)
        lm_, _, _ = O.ppo_minibatch_grad(net, pm, *batch, 0.2, 0.5, 0.01, want_grad=False)
        fd = (lp_ - lm_) / (2 * h)
        assert abs(fd - grad[k]) <= 1e-6 * max(1.0, abs(grad[k])), k


def _rb(t):
    return t.float().to(torch.bfloat16).double()


class _RoundFwd(torch.autograd.Function):
    """bf16 rounding in the forward pass, identity in the backward pass."""

    @staticmethod
    def forward(ctx, t):
        return _rb(t)

    @staticmethod
    def backward(ctx, g):
        return g


class _RoundBwd(torch.autograd.Function):
    """Identity in the forward pass, bf16 rounding of the incoming gradient."""

    @staticmethod
    def forward(ctx, t):
        return t.clone()

    @staticmethod
    def backward(ctx, g):
        return _rb(g)


class _TanhRound(torch.autograd.Function):
    """y = bf16(tanh(a)); the derivative uses the stored (rounded) y."""

    @staticmethod
    def forward(ctx, a):
        y = _rb(torch.tanh(a))
        ctx.save_for_backward(y)
        return y

    @staticmethod
    def backward(ctx, g):
        (y,) = ctx.saved_tensors
        return g * (1.0 - y * y)


def _torch_ppo_loss_bf16(net, params, obs, act, lpo, adv, ret, clip, vf, ent):
    """Autograd of the bf16 network: weights and inputs rounded on the way in,
    tanh outputs stored rounded, and the gradients at the three product inputs
    (head output, both pre-activations) rounded on the way back; the head bias
    sees the unrounded head gradient."""
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    p = torch.tensor(params, dtype=torch.float64, requires_grad=True)
    sizes = [H * D, H, H * H, H, A * H, A, H * D, H, H * H, H, H, 1]
    W1, b1, W2, b2, W3, b3, V1, c1, V2, c2, V3, c3 = torch.split(p, sizes)
    x = _rb(torch.tensor(obs, dtype=torch.float64))

    def fwd(Wa, ba, Wb, bb, Wc, bc, out):
        h1 = _TanhRound.apply(_RoundBwd.apply(x @ _RoundFwd.apply(Wa.view(H, D)).T + ba))
        h2 = _TanhRound.apply(_RoundBwd.apply(h1 @ _RoundFwd.apply(Wb.view(H, H)).T + bb))
        return _RoundBwd.apply(h2 @ _RoundFwd.apply(Wc.view(out, H)).T) + bc

    z = fwd(W1, b1, W2, b2, W3, b3, A)
    V = fwd(V1, c1, V2, c2, V3, c3, 1)[:, 0]
    logp_all = torch.log_softmax(z, -1)
    lp = logp_all[torch.arange(len(act)), torch.tensor(act, dtype=torch.long)]
    a = torch.tensor(adv, dtype=torch.float64)
    a = (a - a.mean()) / (a.std() + 1e-8)
    rho = torch.exp(lp - torch.tensor(lpo, dtype=torch.float64))
    pg = -torch.min(rho * a, torch.clamp(rho, 1 - clip, 1 + clip) * a).mean()
    vl = ((torch.tensor(ret, dtype=torch.float64) - V) ** 2).mean()
    H_ = -(logp_all.exp() * logp_all).sum(-1).mean()
    loss = pg + vf * vl - ent * H_
    loss.backward()
    return loss.item(), p.grad.numpy()


def test_ppo_bf16_gradient_matches_autograd_with_rounding():
    """bf16 networks: the oracle's hand-written backward equals autograd of
    the network with bf16 rounding at the same points, and differs from the
    unrounded-backward gradient by no more than bf16 rounding."""
    net = W.NetSpec(6, 16, 4, 1)
    params = W.init_params(net, seed=6, bias_scale=0.1).astype(np.float64)
    batch = _ppo_batch(net, 48, seed=2)
    # the minibatch gradient takes the weights already rounded (the update
    # rounds its fp32 masters once per minibatch); biases stay unrounded
    D, H, A = 6, 16, 4
    sizes = [H * D, H, H * H, H, A * H, A, H * D, H, H * H, H, H, 1]
    parts = np.split(params, np.cumsum(sizes)[:-1])
    params = np.concatenate([_rb(torch.tensor(q)).numpy() if i % 2 == 0 else q for i, q in enumerate(parts)])
    loss, grad, _ = O.ppo_minibatch_grad(net, params, *batch, 0.2, 0.5, 0.01)
    tl, tg = _torch_ppo_loss_bf16(net, params, *batch, 0.2, 0.5, 0.01)
    assert loss == pytest.approx(tl, rel=1e-12)
    assert np.allclose(grad, tg, rtol=1e-9, atol=1e-12)
    # the forward of the bf16 network differs from the fp64 one (rounding is applied)
    l64, g64, _ = O.ppo_minibatch_grad(W.NetSpec(6, 16, 4, 0), params, *batch, 0.2, 0.5, 0.01)
    assert 1e-6 < abs(loss - l64) / abs(l64) < 5e-2
    d = np.abs(grad - g64).max() / np.abs(g64).max()
    assert 1e-5 < d < 5e-2


def test_ppo_first_minibatch_ratio_one_policy_loss_zero():
    """With logp_old = logp under the current params, rho = 1 and the
    clipped surrogate is -mean(normalised advantage) = 0."""
    net = W.NetSpec(6, 8, 4, 0)
    params = W.init_params(net, seed=2, bias_scale=0.1)
    obs, act, _, adv, ret = _ppo_batch(net, 64)
    lg, _ = O.mlp_forward(net, params, obs)
    lse = lg.max(1) + np.log(np.exp(lg - lg.max(1, keepdims=True)).sum(1))
    lpo = (lg[np.arange(64), act] - lse).astype(np.float32)
    _, _, st = O.ppo_minibatch_grad(net, params.astype(np.float64), obs, act, lpo, adv, ret,
                                    0.2, 0.5, 0.0)
    assert abs(st[0]) < 1e-6 and st[4] == 0.0 and abs(st[3]) < 1e-12


def test_ppo_clip_cases_two_samples():
    """Two samples, normalised advantages +-1/sqrt(2)*sqrt(2)... rho set via logp_old."""
    net = W.NetSpec(2, 2, 2, 0)
    params = np.zeros(W.param_count(2, 2, 2), np.float64)  # uniform policy, logp = log 0.5
    obs = np.zeros((2, 2), np.float32)
    act = np.array([0, 1], np.uint8)
    adv = np.array([1.0, -1.0], np.float32)   # normalised: +-1/sqrt(2) * ... (mean 0, std sqrt 2)
    ret = np.zeros(2, np.float32)
    an = np.array([1.0, -1.0]) / (np.sqrt(2.0) + 1e-8)
    for rho in (0.5, 0.9, 1.0, 1.1, 1.5):
        lpo = np.full(2, math.log(0.5) - math.log(rho), np.float32)
        r = math.exp(math.log(0.5) - float(np.float32(math.log(0.5) - math.log(rho))))
        _, _, st = O.ppo_minibatch_grad(net, params, obs, act, lpo, adv, ret, 0.2, 0.5, 0.0)
        rc = min(max(r, 0.8), 1.2)
        want = -np.mean(np.minimum(r * an, rc * an))
        assert st[0] == pytest.approx(want, rel=1e-9, abs=1e-12)
        assert st[4] == (1.0 if abs(r - 1) > 0.2 else 0.0)


def test_ppo_adam_first_step_is_signed_lr():
    net = W.NetSpec(6, 8, 4, 0)
    params = W.init_params(net, seed=4, bias_scale=0.1)
    N = 256
    obs, act, lpo, adv, ret = _ppo_batch(net, N, seed=3)
    ppo = W.PPOSpec(epochs=1, minibatch=N, max_grad_norm=1e9)
    P, m, v, t, st = O.ppo_update(net, ppo, params, np.zeros(params.size), np.zeros(params.size), 0,
                                  obs, act, lpo, adv, ret, seed=1, iteration=0, max_steps=1)
    _, g, _ = O.ppo_minibatch_grad(net, params.astype(np.float64), obs, act, lpo, adv, ret,
                                   0.2, 0.5, 0.0)
    step = P - params.astype(np.float64)
    big = np.abs(g) > 1e-5
    assert t == 1 and st[7] == 1
    assert np.allclose(step[big], -3e-4 * np.sign(g[big]), rtol=1e-3)
    # a full-batch minibatch sees every sample once, so the permutation does not matter
    assert np.allclose(m, 0.1 * g, rtol=1e-12, atol=1e-300)


def test_ppo_grad_norm_clip():
    net = W.NetSpec(6, 8, 4, 0)
    params = W.init_params(net, seed=4, bias_scale=0.1)
    obs, act, lpo, adv, ret = _ppo_batch(net, 64, seed=9)
    ppo = W.PPOSpec(epochs=1, minibatch=64, max_grad_norm=1e-3)
    _, m, _, _, st = O.ppo_update(net, ppo, params, np.zeros(params.size), np.zeros(params.size),
                                  0, obs, act, lpo, adv, ret, seed=1, iteration=0, max_steps=1)
    # m = (1 - beta1) * clipped gradient; the clipped gradient has norm max_norm * n / (n + 1e-6)
    n = st[6]
    assert np.linalg.norm(m / 0.1) == pytest.approx(1e-3 * n / (n + 1e-6), rel=1e-9)


class _RoundF32(torch.autograd.Function):
    """fp32 rounding in the forward pass, identity in the backward pass."""

    @staticmethod
    def forward(ctx, t):
        return t.float().double()

    @staticmethod
    def backward(ctx, g):
        return g


def _torch_loss_of(net, p, obs, act, lpo, adv, ret, clip, vf, ent, bf16):
    """The SB3 PPO loss of one minibatch as a function of the fp64 parameter
    tensor p, written independently of the oracle.  bf16 networks see their
    fp32-cast masters with the weights rounded to bf16 (straight-through, so
    the gradient of the rounded weights reaches the masters) and the same
    rounding points as _torch_ppo_loss_bf16."""
    D, H, A = net.obs_dim, net.hidden, net.n_actions
    sizes = [H * D, H, H * H, H, A * H, A, H * D, H, H * H, H, H, 1]
    W1, b1, W2, b2, W3, b3, V1, c1, V2, c2, V3, c3 = torch.split(p, sizes)
    x = torch.tensor(obs, dtype=torch.float64)
    if bf16:
        x = _rb(x)
        wr = lambda w: _RoundFwd.apply(_RoundF32.apply(w))
        br = _RoundF32.apply

        def fwd(Wa, ba, Wb, bb, Wc, bc, out):
            h1 = _TanhRound.apply(_RoundBwd.apply(x @ wr(Wa.view(H, D)).T + br(ba)))
            h2 = _TanhRound.apply(_RoundBwd.apply(h1 @ wr(Wb.view(H, H)).T + br(bb)))
            return _RoundBwd.apply(h2 @ wr(Wc.view(out, H)).T) + br(bc)
    else:
        def fwd(Wa, ba, Wb, bb, Wc, bc, out):
            return torch.tanh(torch.tanh(x @ Wa.view(H, D).T + ba) @ Wb.view(H, H).T + bb) @ Wc.view(out, H).T + bc
    z = fwd(W1, b1, W2, b2, W3, b3, A)
    V = fwd(V1, c1, V2, c2, V3, c3, 1)[:, 0]
    logp_all = torch.log_softmax(z, -1)
    lp = logp_all[torch.arange(len(act)), torch.tensor(act, dtype=torch.long)]
    a = torch.tensor(adv, dtype=torch.float64)
    a = (a - a.mean()) / (a.std() + 1e-8)
    logr = lp - torch.tensor(lpo, dtype=torch.float64)
    rho = torch.exp(logr)
    pg = -torch.min(rho * a, torch.clamp(rho, 1 - clip, 1 + clip) * a).mean()
    vl = ((torch.tensor(ret, dtype=torch.float64) - V) ** 2).mean()
    H_ = -(logp_all.exp() * logp_all).sum(-1).mean()
    with torch.no_grad():
        kl = ((rho - 1) - logr).mean().item()
        cf = ((rho - 1).abs() > clip).double().mean().item()
    return pg + vf * vl - ent * H_, (pg.item(), vl.item(), H_.item(), kl, cf)


def _torch_ppo_update(net, ppo, params, m0, v0, t0, batch, seed, iteration):
    """The whole update loop in torch: per epoch the oracle's Feistel order
    (any permutation is valid; the loop must gather every per-sample array
    through the same index), ragged last minibatch, autograd gradient,
    torch.nn.utils.clip_grad_norm_, torch.optim.Adam resumed from (m0, v0,
    t0).  Returns params, moments, per-step statistics means and step count."""
    obs, act, lpo, adv, ret = batch
    N = len(act)
    p = torch.tensor(np.asarray(params, np.float64), requires_grad=True)
    opt = torch.optim.Adam([p], lr=ppo.lr, betas=(ppo.beta1, ppo.beta2), eps=ppo.eps)
    if t0:
        opt.state[p] = {"step": torch.tensor(float(t0), dtype=torch.float64),
                        "exp_avg": torch.tensor(m0, dtype=torch.float64),
                        "exp_avg_sq": torch.tensor(v0, dtype=torch.float64)}
    acc = np.zeros(5)
    steps = 0
    for ep in range(ppo.epochs):
        perm = O.feistel_perm(N, O.perm_keys(seed, ep, iteration))
        for start in range(0, N, ppo.minibatch):
            idx = perm[start:start + ppo.minibatch]
            opt.zero_grad()
            loss, st = _torch_loss_of(net, p, obs[idx], act[idx], lpo[idx], adv[idx], ret[idx], ppo.clip,
                                      ppo.vf_coef, ppo.ent_coef, net.dtype == 1)
            loss.backward()
            torch.nn.utils.clip_grad_norm_([p], ppo.max_grad_norm)
            opt.step()
            acc += st
            steps += 1
    s = opt.state[p]
    return p.detach().numpy(), s["exp_avg"].numpy(), s["exp_avg_sq"].numpy(), acc / steps, steps


@pytest.mark.parametrize("bf16", [0, 1])
def test_ppo_update_loop_matches_torch_autograd_clip_and_adam(bf16):
    """or_ppo_update_ex over 2 epochs x 3 minibatches (40, 40 and a ragged
    20), resumed from nonzero Adam moments at step 3, against an independent
    torch loop (autograd, clip_grad_norm_, optim.Adam): parameters, both
    moments, the step count and the statistics.  A frozen bias correction,
    moments dropped between minibatches, a gather that takes one array through
    a different index, or a ragged tail normalised over the full minibatch
    size each fail this."""
    net = W.NetSpec(6, 16 if bf16 else 8, 4, bf16)
    params = W.init_params(net, seed=8, bias_scale=0.1).astype(np.float64)
    N = 100
    obs, act, lpo, adv, ret = _ppo_batch(net, N, seed=5)
    adv = (adv + 0.7).astype(np.float32)   # a nonzero mean, so normalisation matters
    ppo = W.PPOSpec(epochs=2, minibatch=40, lr=3e-3, ent_coef=0.01, max_grad_norm=0.5)
    rng = np.random.default_rng(3)
    m0 = 1e-3 * rng.standard_normal(params.size)
    v0 = 1e-5 * rng.random(params.size)
    P, m, v, t, st = O.ppo_update(net, ppo, params, m0, v0, 3, obs, act, lpo, adv, ret, seed=11, iteration=4)
    tp, tm, tv, tst, steps = _torch_ppo_update(net, ppo, params, m0, v0, 3, (obs, act, lpo, adv, ret), 11, 4)
    assert t == 3 + 6 and steps == 6 and st[7] == 6
    assert np.allclose(P, tp, rtol=1e-9, atol=1e-12)
    assert np.allclose(m, tm, rtol=1e-9, atol=1e-14)
    assert np.allclose(v, tv, rtol=1e-9, atol=1e-16)
    # statistics: pg, value loss, entropy, approx KL, clip fraction (means over the steps)
    for k, want in zip((0, 1, 2, 3, 4), tst):
        assert st[k] == pytest.approx(want, rel=1e-9, abs=1e-12), k
    # the steps moved the policy: the later minibatches see rho != 1
    assert st[3] > 0.0
    # and the parameters moved by about lr per step
    assert 0.5 * 3e-3 < np.abs(P - params).max() <= 6 * 3e-3 * (1 + 1e-6)


# ---------------------------------------------------------------------- fleet
def _brute_fleet(traces, job, J, offsets, H, windows, Bq):
    q = np.rint(traces.astype(np.float32) * np.float32(64)).astype(np.int64)
    G, L = q.shape
    N = offsets.shape[0]
    counts = np.zeros((N, len(windows)), np.int64)
    peaks = np.zeros((N, len(windows)), np.int64)
    t = np.arange(H)
    for n in range(N):
        P = sum(q[g, (t + offsets[n, job[g]]) % L] for g in range(G))
        for wi, w in enumerate(windows):
            S = np.array([P[tt - w + 1:tt + 1].sum() for tt in range(w - 1, H)])
            counts[n, wi] = int((S > Bq * w).sum())
            peaks[n, wi] = int(S.max()) if len(S) else 0
    return counts, peaks


def test_fleet_matches_bruteforce():
    rng = np.random.default_rng(0)
    G, L, J = 6, 700, 3
    traces = (300 + 60 * rng.standard_normal((G, L))).astype(np.float32)
    job = np.array([0, 0, 1, 2, 2, 2], np.int32)
    off = rng.integers(0, L, (9, J)).astype(np.int32)
    off[0] = 0
    windows = np.array([1, 7, 60, 600], np.int32)
    Bq = 6 * 300 * 64
    for H in (L, 650, 599, 1):
        c, p = O.fleet_windows(traces, job, J, off, H, windows, Bq)
        bc, bp = _brute_fleet(traces, job, J, off, H, windows, Bq)
        assert np.array_equal(c, bc) and np.array_equal(p, bp)


def test_fleet_invariants():
    fw = W.make_fleet(n_compositions=6, length=3000, windows=(1, 60, 600))
    c, p = O.fleet_windows(fw.traces, fw.job_of_gpu, fw.n_jobs, fw.offsets, fw.horizon,
                           fw.windows, fw.budget_q)
    q = np.rint(fw.traces * np.float32(64)).astype(np.int64)
    # (iii) the aligned composition is the direct sum of the traces
    direct = q.sum(0)
    assert p[0, 0] == direct.max()
    assert c[0, 0] == int((direct > fw.budget_q).sum())
    # (ii) the composed peak never exceeds the sum of per-job peaks (each
    # job's trace tiles circularly, so its windows wrap)
    for wi, w in enumerate(fw.windows):
        per_job = 0
        for j in range(fw.n_jobs):
            pj = q[fw.job_of_gpu == j].sum(0)
            pj = np.concatenate([pj, pj[:w - 1]])
            per_job += np.convolve(pj, np.ones(w, np.int64), "valid").max()
        assert np.all(p[:, wi] <= per_job)
    # (iv) one job and one trace reduce to the single-trace window analysis
    c1, p1 = O.fleet_windows(fw.traces[:1], [0], 1, np.zeros((1, 1), np.int32), fw.horizon,
                             [60], fw.budget_q // 16)
    S = np.convolve(q[0], np.ones(60, np.int64), mode="valid")
    assert c1[0, 0] == int((S > 60 * (fw.budget_q // 16)).sum()) and p1[0, 0] == S.max()


def test_fleet_constant_hand_counted():
    traces = np.full((2, 100), 10.0, np.float32)  # q = 640 each, sum 1280
    off = np.array([[0, 0], [5, 17]], np.int32)
    for Bq, want in ((1279, [100, 41]), (1280, [0, 0])):
        c, p = O.fleet_windows(traces, [0, 1], 2, off, 100, [1, 60], Bq)
        assert c.tolist() == [want, want] and p.tolist() == [[1280, 76800]] * 2


# ------------------------------------------------------------ fleet stagger
def _np_window_peak(series, w):
    c = np.concatenate([[0], np.cumsum(series, dtype=np.int64)])
    S = c[w:] - c[:-w]          # S[t - w + 1] = sum of series[t-w+1 .. t]
    return int(S.max())


def test_fleet_stagger_square_waves_closed_form():
    """Two identical square waves (h samples at a, h at b): the greedy puts
    the second one in anti-phase, offset h, where the 1-sample peak drops
    from 2a to a + b; the first job ties everywhere and takes offset 0.
    With a full-period window every offset ties, so both offsets are 0."""
    h, a, b, L = 5, 300.0, 100.0, 40
    x = np.array(([a] * h + [b] * h) * (L // (2 * h)), np.float32)
    traces = np.stack([x, x])
    off, pk = O.fleet_stagger(traces, [0, 1], 2, L, 1, 1)
    assert off.tolist() == [0, h]
    assert pk.tolist() == [int(64 * a), int(64 * (a + b))]
    off, pk = O.fleet_stagger(traces, [0, 1], 2, L, 2 * h, 1)
    assert off.tolist() == [0, 0]
    assert pk[1] == 2 * h * int(64 * (a + b))  # each job gives h(a + b) per full-period window


def test_fleet_stagger_matches_brute_force():
    """Every stage's choice against an independent numpy search over the
    candidate grid (np.roll for the circular shift, cumulative sums for the
    windows), on a random 5-GPU, 3-job fleet."""
    rng = np.random.default_rng(11)
    G, L, H, w, stride = 5, 47, 47, 6, 3
    traces = rng.uniform(50, 400, size=(G, L)).astype(np.float32)
    job = np.array([0, 0, 1, 2, 2], np.int32)
    off, pk = O.fleet_stagger(traces, job, 3, H, w, stride)
    q = np.rint(traces.astype(np.float32) * np.float32(64)).astype(np.int64)
    qj = np.stack([q[job == j].sum(0) for j in range(3)])
    placed = np.zeros(H, np.int64)
    for j in range(3):
        cands = list(range(0, L, stride))
        peaks = [_np_window_peak(placed + np.roll(qj[j], -o)[:H], w) for o in cands]
        best = int(np.argmin(peaks))          # argmin returns the first (lowest offset) minimum
        assert off[j] == cands[best] and pk[j] == peaks[best], (j, off[j], cands[best])
        placed += np.roll(qj[j], -off[j])[:H]


def test_fleet_stagger_invariants():
    """Stage peaks never fall (each job adds nonnegative power), and the
    second job's choice is no worse than starting it with the first job."""
    wl = W.make_fleet(n_compositions=1, length=600)
    off, pk = O.fleet_stagger(wl.traces, wl.job_of_gpu, wl.n_jobs, 600, 60, 7)
    assert np.all(np.diff(pk) >= 0)
    sel = np.isin(wl.job_of_gpu, [0, 1])
    _, aligned = O.fleet_windows(wl.traces[sel], wl.job_of_gpu[sel], 2,
                                 np.array([[off[0], off[0]]], np.int32), 600, [60], 0)
    assert pk[1] <= aligned[0, 0]
    assert np.all(off % 7 == 0) and np.all(off < 600)


# ------------------------------------------------------- baseline rule policies
def _brute_rule(b, rule, e, t, it):
    """The Sec. 4.4 / 4.5 baseline rules, decided on the brute-force env's
    history (window sums recomputed sample by sample)."""
    s = b.s
    incdec = s.actuator_kind == 1
    hold = 0 if incdec else b.level
    lower = 1 if incdec else max(b.level - 1, 0)
    up = 2 if incdec else min(b.level + 1, s.n_levels - 1)
    if rule.kind == W.RULE_RANDOM:
        u = int(O.philox4x32_10([e, t, it, 0], [s.seed & 0xFFFFFFFF, s.seed >> 32])[0])
        return (u * s.n_actions) >> 32
    if rule.kind == W.RULE_THRESHOLD:
        q = b.Q(0)
        return lower if q > rule.hi_q else (up if q < rule.lo_q else hold)
    s30, s10 = b.S(60), b.S(20)
    if s30 > 60 * rule.drop30_q:
        return lower
    return up if (s30 < 60 * rule.climb30_q and s10 < 20 * rule.climb10_q) else hold


@pytest.mark.parametrize("preset", ["tiny", "7b", "72b"])
@pytest.mark.parametrize("kind", [1, 2, 3])
def test_rule_rollout_matches_bruteforce(preset, kind):
    """Baseline-policy rollouts from explicit episode starts (the evaluation
    replay), across an episode boundary, against the brute-force env driven
    by the same rules."""
    wl = {"tiny": W.make_tiny, "7b": W.make_7b, "72b": W.make_72b}[preset](n_envs=2)
    spec = wl.env
    B = spec.budget_q
    rule = {1: W.random_rule(), 2: W.threshold_rule(B), 3: W.hysteresis_rule(B)}[kind]
    # the tiny trace sits above 0.9 B at every level: thresholds between its
    # levels make both rules move in both directions
    if preset == "tiny" and kind == 2:
        rule = W.threshold_rule(B, 1.1, 0.98)
    if preset == "tiny" and kind == 3:
        rule = W.hysteresis_rule(B, 1.1, 0.98, 1.05)
    if preset == "7b" and kind == 3:  # the 7B 30 s mean stays above 512/561 of B
        rule = W.hysteresis_rule(B, 1.08, 1.0, 1.05)
    offs = W.replay_offsets(wl.trace.shape[-1], spec.episode_len, 2)
    env = O.OracleEnv(spec, wl.trace, wl.phase, [0, 1])
    env.set_offsets(offs)
    T = spec.episode_len + 30
    out = env.rollout_rule(rule, T, 3, lam=0.5)
    for i in range(2):
        b = BruteEnv(spec, wl.trace.astype(np.float32), wl.phase, i, O.philox4x32_10)
        b.reset_at(int(offs[i]))
        v = [0, 0]
        en = 0
        for t in range(T):
            a = _brute_rule(b, rule, i, t, 3)
            assert out["act"][t, i] == a, (t, i)
            st = b.step(a, 0.5, t, 3)
            assert out["done"][t, i] == st["done"]
            assert abs(out["reward"][t, i] - st["r"]) <= 1e-12 * max(1.0, abs(st["r"]))
            v[0] += st["v1"]
            v[1] += st["v60"]
            en += st["q"]
        assert list(out["viol"][i]) == v and out["energy_q"][i] == en
    acts = np.bincount(out["act"].ravel(), minlength=spec.n_actions)
    assert (acts > 0).sum() >= (2 if kind != 1 else spec.n_actions // 2)


def test_threshold_rule_constant_trace_hand_counted():
    """A flat 7B trace at 1.2 B watts (above 0.9 B at every group size): the
    threshold rule lowers G every step, from 4 to the floor 3 after one
    step, so the energy is one sample at s(4) and the rest at s(3); a flat
    trace at 0.5 B raises G every step up to G_max = 8."""
    wl = W.make_7b(n_envs=1)
    spec = wl.env
    L = wl.trace.shape[-1]
    for frac, act, levels in ((1.2, 1, [4, 3]), (0.5, 2, [4, 5, 6, 7, 8])):
        x = np.float32(frac * spec.budget_q / 64.0)
        trace = np.full_like(wl.trace, x)
        phase = np.zeros_like(wl.phase)
        env = O.OracleEnv(spec, trace, phase, [0])
        env.set_offsets([100])
        T = 12
        out = env.rollout_rule(W.threshold_rule(spec.budget_q), T, 0)
        assert np.all(out["act"][:, 0] == act)
        # G in effect at each step: the first action already moves G once
        g = levels[1:] + [levels[-1]] * (T - len(levels) + 1)
        q = [int(np.rint(np.float32(x * O.actuator_scale(spec, G)) * np.float32(64))) for G in g[:T]]
        assert out["energy_q"][0] == sum(q)
    del L


# ------------------------------------------------------------- dual ascent
def test_dual_ascent_eq7_closed_form():
    """Eq. 7: on target the multiplier stays; at twice the target it grows by
    e^eta; at zero violations it shrinks by e^-eta; the clip bounds hold;
    the additive form moves by eta times the relative gap."""
    E, T = 10, 100
    viol = np.zeros((E, 2), np.int32)
    viol[:, 1] = 8                     # 80 of 1000 env-steps: the 8% target exactly
    lam, v = O.dual_ascent(viol, T, 1.0)
    assert v == pytest.approx(0.08) and lam == pytest.approx(1.0, rel=1e-15)
    viol[:, 1] = 16
    lam, v = O.dual_ascent(viol, T, 1.0)
    assert lam == pytest.approx(math.exp(0.5), rel=1e-15)
    viol[:, 1] = 0
    lam, _ = O.dual_ascent(viol, T, 1.0)
    assert lam == pytest.approx(math.exp(-0.5), rel=1e-15)
    viol[:, 1] = 100                   # every step violates
    assert O.dual_ascent(viol, T, 1.9)[0] == 2.0
    assert O.dual_ascent(np.zeros((E, 2)), T, 1e-3)[0] == 1e-3
    viol[:, 0] = 4                     # the instantaneous count: half the target
    lam, v = O.dual_ascent(viol, T, 3.0, window=1, additive=True, hi=20.0)
    assert v == pytest.approx(0.04) and lam == pytest.approx(3.0 - 0.25, rel=1e-15)
