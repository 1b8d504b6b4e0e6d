// Environment of the batched power-control MDP: device-side definitions
// shared by the rollout kernels (fp32 FFMA networks and bf16 tensor-core
// networks).
//
// One environment step consumes one half-second sample of a power trace
// (Sec. 4.1 trace replay).  Actuated power is held in 1/64 W integers, so the
// trailing window sums of Eq. 1 (10 s = 20 samples, 30 s = 60 samples) and
// the violation indicators of Eq. 2 are exact.
#pragma once

#include "common.cuh"

namespace pe {

constexpr int kWShort = 20;  // 10 s
constexpr int kWLong = 60;   // 30 s
constexpr int kRing = 64;    // per-env ring of the last 64 samples (>= kWLong)

// everything a rollout kernel needs to know about the envs (passed by value)
struct EnvDev {
  int32_t E, C, L, A, obs_kind, act_kind, n_levels, level_init;
  int32_t g_min, g_max, b_min, b_max, b_init, ep_len, budget_q, phase_mask;
  int32_t reward_kind, reward_window;
  float r_ok, r_viol, bonus_coef, inv_rate_max;
  float scale[PE_MAX_LEVELS][PE_MAX_CHANNELS];  // actuator table (INCDEC formula pre-evaluated)
  float tokens[PE_MAX_LEVELS];
  int32_t ns[PE_MAX_LEVELS];  // samples per step at each level (1 without a cadence table)
  int32_t cadence;            // a cadence table is set
  int32_t span;               // samples one episode may span: ep_len * max ns
  uint64_t seed;
  // trace families (domain randomisation, Sec. 4.2 G2; one family without
  // it): family f has a [C][fL[f]] trace (channels >= fC[f] are zero), a
  // [fL[f]] phase array and the budget fB[f] in 1/64 W
  int32_t F;
  const float* ftrace[PE_MAX_FAMILIES];
  const uint8_t* fphase[PE_MAX_FAMILIES];
  int32_t fL[PE_MAX_FAMILIES], fC[PE_MAX_FAMILIES], fB[PE_MAX_FAMILIES];
  // persistent env state, SoA
  int32_t* st;     // [7][E]: pos, k, level, prev, b, til, family
  uint8_t* ring;   // [E][64]: level used for the sample at position p (slot p & 63)
  int32_t* sums;   // [E][8]: s_short[4], s_long[4] (per channel)
};

enum { kStPos = 0, kStK, kStLevel, kStPrev, kStB, kStTil, kStFam, kStN };

// one trace family's view (selected with constant indices: the EnvDev
// arrays stay in kernel parameter space)
struct Fam {
  const float* trace;
  const uint8_t* phase;
  int32_t L, C, B;
};

__device__ __forceinline__ Fam fam_of(const EnvDev& env, int f) {
  if (f == 1) return Fam{env.ftrace[1], env.fphase[1], env.fL[1], env.fC[1], env.fB[1]};
  if (f == 2) return Fam{env.ftrace[2], env.fphase[2], env.fL[2], env.fC[2], env.fB[2]};
  if (f == 3) return Fam{env.ftrace[3], env.fphase[3], env.fL[3], env.fC[3], env.fB[3]};
  return Fam{env.ftrace[0], env.fphase[0], env.fL[0], env.fC[0], env.fB[0]};
}

// Per-tile env state staged in shared memory for the whole horizon.
template <int TE, int C>
struct EnvTile {
  int32_t pos[TE], k[TE], level[TE], prev[TE], b[TE], til[TE], fam[TE];
  int32_t s_short[TE][4], s_long[TE][4];
  int32_t q[TE][C][kRing];  // actuated per-channel samples of positions p-64..p-1, slot p & 63
  uint8_t ring[TE][kRing];  // level of each of those samples
};

__device__ __forceinline__ float actuator_scale(const EnvDev& env, int level, int c, int ph) {
  return ((env.phase_mask >> ph) & 1) ? env.scale[level][c] : 1.0f;
}

__device__ __forceinline__ int32_t sample_q(const EnvDev& env, const Fam& fm, int c, int pos, int level) {
  const float x = __ldg(fm.trace + (int64_t)c * fm.L + pos);
  return quant64(x, actuator_scale(env, level, c, __ldg(fm.phase + pos)));
}

// ---------------------------------------------------------------------------
// Two views of one env's state with the same interface:
//   TileAcc -- a slot of an EnvTile in shared memory, with the actuated
//              per-channel samples of the last 64 positions cached;
//   RegAcc  -- scalars in registers, level ring in global memory, samples
//              recomputed from the trace and the ring when needed.
// The features, the step and the reset below are written once over either.
// ---------------------------------------------------------------------------
template <int TE, int C>
struct TileAcc {
  EnvTile<TE, C>& s;
  int e;
  __device__ int32_t& pos() { return s.pos[e]; }
  __device__ int32_t& k() { return s.k[e]; }
  __device__ int32_t& level() { return s.level[e]; }
  __device__ int32_t& prev() { return s.prev[e]; }
  __device__ int32_t& b() { return s.b[e]; }
  __device__ int32_t& til() { return s.til[e]; }
  __device__ int32_t& fam() { return s.fam[e]; }
  __device__ int32_t& ss(int c) { return s.s_short[e][c]; }
  __device__ int32_t& sl(int c) { return s.s_long[e][c]; }
  __device__ uint8_t level_at(int p) const { return s.ring[e][p & (kRing - 1)]; }
  __device__ void set_level_at(int p, int l) { s.ring[e][p & (kRing - 1)] = (uint8_t)l; }
  // actuated sample of channel c at a recent position p (p in [pos-64, pos));
  // fm is the env's family view (unused: the tile caches the samples)
  __device__ int32_t q_at(const EnvDev&, const Fam&, int c, int p) const { return s.q[e][c][p & (kRing - 1)]; }
  __device__ void push(int c, int p, int32_t q) { s.q[e][c][p & (kRing - 1)] = q; }
};

template <int C>
struct RegAcc {
  int32_t pos_, k_, level_, prev_, b_, til_, fam_;
  int32_t ss_[C], sl_[C];
  uint8_t* ring;  // global [64]
  __device__ int32_t& fam() { return fam_; }
  __device__ int32_t& pos() { return pos_; }
  __device__ int32_t& k() { return k_; }
  __device__ int32_t& level() { return level_; }
  __device__ int32_t& prev() { return prev_; }
  __device__ int32_t& b() { return b_; }
  __device__ int32_t& til() { return til_; }
  __device__ int32_t& ss(int c) { return ss_[c]; }
  __device__ int32_t& sl(int c) { return sl_[c]; }
  __device__ uint8_t level_at(int p) const { return ring[p & (kRing - 1)]; }
  __device__ void set_level_at(int p, int l) { ring[p & (kRing - 1)] = (uint8_t)l; }
  // recomputed from the trace of the env's family (view fm) and the level ring
  __device__ int32_t q_at(const EnvDev& env, const Fam& fm, int c, int p) const {
    return sample_q(env, fm, c, p, level_at(p));
  }
  __device__ void push(int, int, int32_t) {}
};

// 60-sample history before the current position at the recorded levels
template <int C, class Acc>
__device__ void rebuild_history(const EnvDev& env, Acc& a) {
  const int p = a.pos();
  const Fam fm = fam_of(env, a.fam());
  for (int c = 0; c < C; ++c) {
    int32_t ss = 0, sl = 0;
    for (int i = 1; i <= kWLong; ++i) {
      const int pp = p - i;
      const int32_t q = sample_q(env, fm, c, pp, a.level_at(pp));
      a.push(c, pp, q);
      sl += q;
      if (i <= kWShort) ss += q;
    }
    a.ss(c) = ss;
    a.sl(c) = sl;
  }
}

// new episode at trace offset o (Sec. 4.5: warm start at the default level)
template <int C, class Acc>
__device__ void env_reset_at(const EnvDev& env, Acc& a, int o) {
  a.pos() = o;
  a.k() = 0;
  a.level() = env.level_init;
  a.prev() = env.level_init;
  a.b() = env.b_init;
  a.til() = 0;
  for (int i = 0; i < kRing; ++i) a.set_level_at(i, env.level_init);
  rebuild_history<C>(env, a);
}

// new episode at a random offset (Sec. 4.1); with several trace families,
// word 1 of the draw picks the episode's family (Sec. 4.2 G2) and word 0
// the offset inside that family's trace
template <int C, class Acc>
__device__ void env_reset(const EnvDev& env, Acc& a, uint32_t eg, uint32_t t, uint32_t it,
                          uint32_t purpose) {
  const u32x4 w = philox10(u32x4{eg, t, it, purpose}, (uint32_t)env.seed, (uint32_t)(env.seed >> 32));
  a.fam() = env.F > 1 ? (int)__umulhi(w.y, (uint32_t)env.F) : 0;
  const uint32_t span = (uint32_t)(fam_of(env, a.fam()).L - env.span - kWLong + 1);
  env_reset_at<C>(env, a, kWLong + (int)__umulhi(w.x, span));
}

template <int C, class Acc>
__device__ __forceinline__ int32_t Qc(const EnvDev& env, Acc& a, const Fam& fm, int c, int i) {
  return a.q_at(env, fm, c, a.pos() - 1 - i);
}

template <int C, class Acc>
__device__ __forceinline__ int32_t Qcl(const EnvDev& env, Acc& a, const Fam& fm, int i) {
  int32_t v = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) v += Qc<C>(env, a, fm, c, i);
  return v;
}

// Observation feature f (fp32 quotient of exact integers; all power
// quantities are normalised by the budget B).
//   TINY8 (Sec. 4.1): 5 latest samples, headroom, phase, level
//   7B16: 8 latest samples, 30 s mean, 30 s slack, phase, G, b, 10 s mean, 5 s slope, 0
//   OCC32/OCC64: Eq. 5 eight-vector, then per-channel recent samples and means
//   fm: the env's family view, fam_of(env, a.fam()), taken once per step by
//   callers that write a whole observation
template <int C, int OBS, class Acc>
__device__ __forceinline__ float feature(const EnvDev& env, Acc& a, const Fam& fm, int f) {
  const int64_t B = fm.B;
  if (OBS == PE_OBS_TINY8) {
    if (f < 5) return ratio_i(Qcl<C>(env, a, fm, 4 - f), B);
    if (f == 5) return ratio_i(B - Qcl<C>(env, a, fm, 0), B);
    if (f == 6) return (float)__ldg(fm.phase + a.pos() - 1);
    return ratio_i(a.level(), env.n_levels - 1);
  }
  int64_t S20 = 0, S60 = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    S20 += a.ss(c);
    S60 += a.sl(c);
  }
  if (OBS == PE_OBS_7B16) {
    if (f < 8) return ratio_i(Qcl<C>(env, a, fm, 7 - f), B);
    switch (f) {
      case 8: return ratio_i(S60, kWLong * B);
      case 9: return ratio_i(kWLong * B - S60, kWLong * B);
      case 10: return (float)__ldg(fm.phase + a.pos() - 1);
      case 11: return ratio_i(a.level() - env.g_min, env.g_max - env.g_min);
      case 12: return ratio_i(a.b() - env.b_min, env.b_max - env.b_min);
      case 13: return ratio_i(S20, kWShort * B);
      case 14: return ratio_i((int64_t)Qcl<C>(env, a, fm, 0) - Qcl<C>(env, a, fm, 10), B);
      default: return 0.0f;
    }
  }
  // OCC32 / OCC64 (Eq. 5 core)
  switch (f) {
    case 0: return ratio_i(Qcl<C>(env, a, fm, 0), B);
    case 1: return ratio_i(S20, kWShort * B);
    case 2: return ratio_i(S60, kWLong * B);
    case 3: return ratio_i(kWLong * B - S60, kWLong * B);
    case 4: return ratio_i((int64_t)Qcl<C>(env, a, fm, 0) - Qcl<C>(env, a, fm, 10), B);
    case 5: return ratio_i(a.level() + 1, env.n_levels);
    case 6: return ratio_i(a.prev() + 1, env.n_levels);
    case 7: return fminf(env.cadence ? ratio_i(env.ns[a.level()], 40) : ratio_i(a.til(), 40), 1.0f);
    default: break;
  }
  if (OBS == PE_OBS_OCC32) {
    if (f < 24) {
      const int c = (f - 8) >> 2, i = (f - 8) & 3;
      return c < fm.C ? ratio_i((int64_t)fm.C * Qc<C>(env, a, fm, c, 3 - i), B) : 0.0f;
    }
    if (f < 28) {
      const int c = f - 24;
      return c < fm.C ? ratio_i((int64_t)fm.C * a.sl(c), kWLong * B) : 0.0f;
    }
    return 0.0f;
  }
  // OCC64
  if (f < 56) {
    const int c = (f - 8) / 12, i = (f - 8) % 12;
    return c < fm.C ? ratio_i((int64_t)fm.C * Qc<C>(env, a, fm, c, 11 - i), B) : 0.0f;
  }
  if (f < 60) {
    const int c = f - 56;
    return c < fm.C ? ratio_i((int64_t)fm.C * a.ss(c), kWShort * B) : 0.0f;
  }
  const int c = f - 60;
  return c < fm.C ? ratio_i((int64_t)fm.C * a.sl(c), kWLong * B) : 0.0f;
}

// All D features of an Eq. 5 observation (OCC32 / OCC64) for an env whose
// samples are recomputed from the trace (RegAcc): the actuated samples the
// features read -- positions pos-1 .. pos-NB and pos-11, every channel -- are
// fetched once, with all their loads independent, instead of per feature.
// The arithmetic is feature()'s, so the results are the same bits.
template <int C, int OBS, int D>
__device__ __forceinline__ void features_eq5(const EnvDev& env, RegAcc<C>& a, const Fam& fm, float (&o)[D]) {
  static_assert(OBS == PE_OBS_OCC32 || OBS == PE_OBS_OCC64, "Eq. 5 observations");
  constexpr int NB = OBS == PE_OBS_OCC32 ? 4 : 12;  // recent samples per channel
  constexpr int NP = NB > 10 ? NB : NB + 1;          // back positions read, pos-11 included
  const int p0 = a.pos() - 1;
  uint8_t lv[NP], ph[NP];
  float x[C][NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const int pp = p0 - (i < NB ? i : 10);
    lv[i] = a.level_at(pp);
    ph[i] = __ldg(fm.phase + pp);
#pragma unroll
    for (int c = 0; c < C; ++c) x[c][i] = __ldg(fm.trace + (int64_t)c * fm.L + pp);
  }
  int32_t q[C][NP];
#pragma unroll
  for (int i = 0; i < NP; ++i)
#pragma unroll
    for (int c = 0; c < C; ++c) q[c][i] = quant64(x[c][i], actuator_scale(env, lv[i], c, ph[i]));
  const int i10 = NB > 10 ? 10 : NB;
  int32_t Q0 = 0, Q10 = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    Q0 += q[c][0];
    Q10 += q[c][i10];
  }
  const int64_t B = fm.B;
  int64_t S20 = 0, S60 = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    S20 += a.ss(c);
    S60 += a.sl(c);
  }
  o[0] = ratio_i(Q0, B);
  o[1] = ratio_i(S20, kWShort * B);
  o[2] = ratio_i(S60, kWLong * B);
  o[3] = ratio_i(kWLong * B - S60, kWLong * B);
  o[4] = ratio_i((int64_t)Q0 - Q10, B);
  o[5] = ratio_i(a.level() + 1, env.n_levels);
  o[6] = ratio_i(a.prev() + 1, env.n_levels);
  o[7] = fminf(env.cadence ? ratio_i(env.ns[a.level()], 40) : ratio_i(a.til(), 40), 1.0f);
  if (OBS == PE_OBS_OCC32) {
#pragma unroll
    for (int f = 8; f < 24; ++f) {
      const int c = (f - 8) >> 2, i = (f - 8) & 3;
      o[f] = c < fm.C ? ratio_i((int64_t)fm.C * q[c][3 - i], B) : 0.0f;
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) o[24 + c] = c < fm.C ? ratio_i((int64_t)fm.C * a.sl(c), kWLong * B) : 0.0f;
#pragma unroll
    for (int f = 28; f < D; ++f) o[f] = 0.0f;
  } else {
#pragma unroll
    for (int f = 8; f < 56; ++f) {
      const int c = (f - 8) / 12, i = (f - 8) % 12;
      o[f] = c < fm.C ? ratio_i((int64_t)fm.C * q[c][11 - i], B) : 0.0f;
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      o[56 + c] = c < fm.C ? ratio_i((int64_t)fm.C * a.ss(c), kWShort * B) : 0.0f;
      o[60 + c] = c < fm.C ? ratio_i((int64_t)fm.C * a.sl(c), kWLong * B) : 0.0f;
    }
  }
}

template <int C, int OBS, class Acc>
__device__ __forceinline__ float feature(const EnvDev& env, Acc& a, int f) {
  return feature<C, OBS>(env, a, fam_of(env, a.fam()), f);
}

struct StepOut {
  float reward, tokens, excess;
  int32_t q, v1, v60, done, samples;
};

// Apply action act and consume one sample (Sec. 4.1 actuator and action set
// with the Sec. 4.2 floor g_min; Eqs. 1-3; G1 or Eq. 6 reward).
template <int C, class Acc>
__device__ __forceinline__ StepOut env_step(const EnvDev& env, Acc& a, int act, float lambda) {
  int nl = a.level();
  if (env.act_kind == PE_ACT_INCDEC) {
    if (act == 1 && nl > env.g_min) --nl;
    if (act == 2 && nl < env.g_max) ++nl;
    if (act == 3 && a.b() > env.b_min) a.b() -= 1;
    if (act == 4 && a.b() < env.b_max) a.b() += 1;
  } else {
    nl = act;
  }
  a.til() = (nl != a.level()) ? 0 : a.til() + 1;
  a.prev() = a.level();
  a.level() = nl;
  // consume the step's samples (one, or a generation batch with a cadence
  // table): windows, violations and excess per sample; tokens and excess
  // summed; the Eq. 6 peak term is the batch's largest 30 s excess
  const Fam fm = fam_of(env, a.fam());
  const int64_t B60 = (int64_t)kWLong * fm.B;
  float rate = env.tokens[nl];
  if (env.act_kind == PE_ACT_INCDEC) rate = __fdiv_rn(rate * (float)a.b(), (float)env.b_init);
  StepOut o;
  o.q = 0;
  o.v1 = 0;
  o.v60 = 0;
  o.tokens = 0.0f;
  o.excess = 0.0f;
  float peak_w = 0.0f, fixed = 0.0f;
  const int n = env.ns[nl];
  for (int i = 0; i < n; ++i) {
    const int p = a.pos();
    const int ph = __ldg(fm.phase + p);
    int32_t Q = 0;
    int64_t S60 = 0;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const int32_t qin = quant64(__ldg(fm.trace + (int64_t)c * fm.L + p), actuator_scale(env, nl, c, ph));
      const int32_t q20 = a.q_at(env, fm, c, p - kWShort);
      const int32_t q60 = a.q_at(env, fm, c, p - kWLong);
      a.ss(c) += qin - q20;
      a.sl(c) += qin - q60;
      a.push(c, p, qin);
      Q += qin;
      S60 += a.sl(c);
    }
    a.set_level_at(p, nl);  // after the window updates: slot p & 63 held position p - 64
    const int v1 = Q > fm.B, v60 = S60 > B60;
    const float exc_w = v60 ? __fdiv_rn(__ll2float_rn(S60 - B60), 3840.0f) : 0.0f;  // watts over B
    o.q += Q;
    o.v1 += v1;
    o.v60 += v60;
    o.excess += exc_w * 0.5f;                                                         // Eq. 3, W*s
    o.tokens += ph == 0 ? rate : 0.0f;
    peak_w = fmaxf(peak_w, exc_w);
    if (env.reward_kind != PE_REWARD_LAGRANGE) {
      const int viol = env.reward_window == 1 ? v1 : v60;
      fixed += (viol ? env.r_viol : env.r_ok) + env.bonus_coef * rate * env.inv_rate_max;
    }
    a.pos() = p + 1;
  }
  o.samples = n;
  o.reward = env.reward_kind == PE_REWARD_LAGRANGE
                 ? o.tokens / 1000.0f - lambda * o.excess - 2.0f * lambda * peak_w  // Eq. 6
                 : fixed;
  a.k() += 1;
  o.done = a.k() == env.ep_len;
  return o;
}

template <int TE, int C>
__device__ void load_tile(const EnvDev& env, EnvTile<TE, C>& s, int e0, int ne) {
  for (int e = threadIdx.x; e < ne; e += blockDim.x) {
    const int g = e0 + e;
    s.pos[e] = env.st[kStPos * env.E + g];
    s.k[e] = env.st[kStK * env.E + g];
    s.level[e] = env.st[kStLevel * env.E + g];
    s.prev[e] = env.st[kStPrev * env.E + g];
    s.b[e] = env.st[kStB * env.E + g];
    s.til[e] = env.st[kStTil * env.E + g];
    s.fam[e] = env.st[kStFam * env.E + g];
    for (int i = 0; i < kRing; ++i) s.ring[e][i] = env.ring[(int64_t)g * kRing + i];
    TileAcc<TE, C> a{s, e};
    rebuild_history<C>(env, a);
  }
}

template <int TE, int C>
__device__ void store_tile(const EnvDev& env, const EnvTile<TE, C>& s, int e0, int ne) {
  for (int e = threadIdx.x; e < ne; e += blockDim.x) {
    const int g = e0 + e;
    env.st[kStPos * env.E + g] = s.pos[e];
    env.st[kStK * env.E + g] = s.k[e];
    env.st[kStLevel * env.E + g] = s.level[e];
    env.st[kStPrev * env.E + g] = s.prev[e];
    env.st[kStB * env.E + g] = s.b[e];
    env.st[kStTil * env.E + g] = s.til[e];
    env.st[kStFam * env.E + g] = s.fam[e];
    for (int i = 0; i < kRing; ++i) env.ring[(int64_t)g * kRing + i] = s.ring[e][i];
    for (int c = 0; c < 4; ++c) {
      env.sums[(int64_t)g * 8 + c] = c < C ? s.s_short[e][c] : 0;
      env.sums[(int64_t)g * 8 + 4 + c] = c < C ? s.s_long[e][c] : 0;
    }
  }
}

// register view of env g (level ring stays in global memory)
template <int C>
__device__ __forceinline__ RegAcc<C> load_reg(const EnvDev& env, int g) {
  RegAcc<C> a;
  a.pos_ = env.st[kStPos * env.E + g];
  a.k_ = env.st[kStK * env.E + g];
  a.level_ = env.st[kStLevel * env.E + g];
  a.prev_ = env.st[kStPrev * env.E + g];
  a.b_ = env.st[kStB * env.E + g];
  a.til_ = env.st[kStTil * env.E + g];
  a.fam_ = env.st[kStFam * env.E + g];
  a.ring = env.ring + (int64_t)g * kRing;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    a.ss_[c] = env.sums[(int64_t)g * 8 + c];
    a.sl_[c] = env.sums[(int64_t)g * 8 + 4 + c];
  }
  return a;
}

template <int C>
__device__ __forceinline__ void store_reg(const EnvDev& env, int g, const RegAcc<C>& a) {
  env.st[kStPos * env.E + g] = a.pos_;
  env.st[kStK * env.E + g] = a.k_;
  env.st[kStLevel * env.E + g] = a.level_;
  env.st[kStPrev * env.E + g] = a.prev_;
  env.st[kStB * env.E + g] = a.b_;
  env.st[kStTil * env.E + g] = a.til_;
  env.st[kStFam * env.E + g] = a.fam_;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    env.sums[(int64_t)g * 8 + c] = c < C ? a.ss_[c] : 0;
    env.sums[(int64_t)g * 8 + 4 + c] = c < C ? a.sl_[c] : 0;
  }
}

// categorical sample by inverse CDF (or argmax), returns action and its log-prob
template <int A>
__device__ __forceinline__ int sample_action(const float* z, uint32_t r, bool det, float* logp) {
  float m = z[0];
  int amax = 0;
#pragma unroll
  for (int j = 1; j < A; ++j)
    if (z[j] > m) {
      m = z[j];
      amax = j;
    }
  float S = 0.0f;
#pragma unroll
  for (int j = 0; j < A; ++j) S += expf(z[j] - m);
  int a = A - 1;
  if (det) {
    a = amax;
  } else {
    const float u = (float)(r >> 8) * (1.0f / 16777216.0f);
    const float target = u * S;
    float c = 0.0f;
#pragma unroll
    for (int j = 0; j < A; ++j) {
      c += expf(z[j] - m);
      if (target < c) {
        a = j;
        break;
      }
    }
  }
  *logp = z[a] - m - logf(S);
  return a;
}

}  // namespace pe
