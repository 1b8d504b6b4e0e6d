// Baseline rule policies of the evaluation (Sec. 4.4 random policy and
// threshold heuristic, Sec. 4.5 hysteresis rule) and explicit episode starts
// for the full-trace replay.
//
// A rule rollout needs no network, so one thread runs one env through the
// whole horizon in registers (its level ring in global memory): decide from
// the state before the step, step (actuator, Eqs. 1-3, reward), record the
// action, reward and done flag, and the per-call counters.
#include <cuda_bf16.h>

#include "env.cuh"

namespace pe {

// host-side twin declared in api.cu
struct RuleArgs {
  int32_t kind, hi_q, lo_q, drop30_q, climb30_q, climb10_q;
  int32_t T, obs_bf16;
  uint32_t it;
  float lambda;
  const uint8_t* forced;  // [T][E] actions of a replay (kind kRuleReplay)
};

// a replay (teacher-forced rollout): env e takes action forced[t][e] at step t
constexpr int32_t kRuleReplay = 4;

// lower / raise move one level: G for the inc/dec actuator (actions 1 and 2;
// the env keeps G in [g_min, g_max]), the level index otherwise (clamped)
template <int C>
__device__ __forceinline__ int rule_action(const EnvDev& env, RegAcc<C>& a, const RuleArgs& r, uint32_t e,
                                           uint32_t t) {
  if (r.kind == kRuleReplay) return r.forced[(int64_t)t * env.E + e];
  const bool incdec = env.act_kind == PE_ACT_INCDEC;
  const int lvl = a.level();
  const int hold = incdec ? 0 : lvl;
  const int lower = incdec ? 1 : (lvl > 0 ? lvl - 1 : 0);
  const int raise = incdec ? 2 : (lvl < env.n_levels - 1 ? lvl + 1 : env.n_levels - 1);
  if (r.kind == PE_RULE_RANDOM) return (int)__umulhi(draw32(env.seed, e, t, r.it, kDrawAction), (uint32_t)env.A);
  if (r.kind == PE_RULE_THRESHOLD) {
    const int32_t q = Qcl<C>(env, a, fam_of(env, a.fam()), 0);  // latest actuated cluster sample
    return q > r.hi_q ? lower : (q < r.lo_q ? raise : hold);
  }
  int64_t s10 = 0, s30 = 0;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    s10 += a.ss(c);
    s30 += a.sl(c);
  }
  if (s30 > (int64_t)kWLong * r.drop30_q) return lower;
  return (s30 < (int64_t)kWLong * r.climb30_q && s10 < (int64_t)kWShort * r.climb10_q) ? raise : hold;
}

template <int C, int OBS, int D>
__device__ __forceinline__ void write_obs(const EnvDev& env, RegAcc<C>& a, void* dst, int bf16) {
  const Fam fm = fam_of(env, a.fam());
  if constexpr (OBS == PE_OBS_OCC32 || OBS == PE_OBS_OCC64) {
    float v[D];
    features_eq5<C, OBS, D>(env, a, fm, v);
    if (bf16) {
      __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(dst);
#pragma unroll
      for (int f = 0; f < D; ++f) o[f] = __float2bfloat16_rn(v[f]);
    } else {
      float* o = reinterpret_cast<float*>(dst);
#pragma unroll
      for (int f = 0; f < D; ++f) o[f] = v[f];
    }
    return;
  }
  if (bf16) {
    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(dst);
#pragma unroll 1
    for (int f = 0; f < D; ++f) o[f] = __float2bfloat16_rn(feature<C, OBS>(env, a, fm, f));
  } else {
    float* o = reinterpret_cast<float*>(dst);
#pragma unroll 1
    for (int f = 0; f < D; ++f) o[f] = feature<C, OBS>(env, a, fm, f);
  }
}

template <int C, int OBS, int D>
__global__ void __launch_bounds__(128) rule_rollout_kernel(EnvDev env, RuleArgs r, pe_rollout_buf buf) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= env.E) return;
  RegAcc<C> acc = load_reg<C>(env, e);
  const size_t ob = r.obs_bf16 ? 2 : 4;
  int32_t v1 = 0, v60 = 0;
  float tok = 0.0f, exc = 0.0f;
  int64_t en = 0, smp = 0;
  for (int t = 0; t < r.T; ++t) {
    const int64_t row = (int64_t)t * env.E + e;
    if (buf.obs) write_obs<C, OBS, D>(env, acc, reinterpret_cast<char*>(buf.obs) + row * D * ob, r.obs_bf16);
    const int act = rule_action<C>(env, acc, r, (uint32_t)e, (uint32_t)t);
    const StepOut so = env_step<C>(env, acc, act, r.lambda);
    buf.act[row] = (uint8_t)act;
    buf.reward[row] = so.reward;
    buf.done[row] = (uint8_t)so.done;
    if (buf.q) buf.q[row] = so.q;
    v1 += so.v1;
    v60 += so.v60;
    tok += so.tokens;
    exc += so.excess;
    en += so.q;
    smp += so.samples;
    if (so.done) env_reset<C>(env, acc, (uint32_t)e, (uint32_t)t, r.it, kDrawReset);
  }
  if (buf.obs_last) write_obs<C, OBS, D>(env, acc, reinterpret_cast<char*>(buf.obs_last) + (int64_t)e * D * ob, r.obs_bf16);
  buf.viol[2 * e] = v1;
  buf.viol[2 * e + 1] = v60;
  buf.tokens[e] = tok;
  buf.excess[e] = exc;
  buf.energy_q[e] = en;
  if (buf.samples) buf.samples[e] = smp;
  store_reg<C>(env, e, acc);
}

// every env starts a new episode at offsets[e]; offsets outside
// [60, L - episode_len] set *flag and leave that env unchanged
template <int C>
__global__ void env_offsets_kernel(EnvDev env, const int32_t* __restrict__ offsets, int32_t* __restrict__ flag) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= env.E) return;
  const int o = offsets[e];
  const int fam = env.st[kStFam * env.E + e];
  if (o < kWLong || o > fam_of(env, fam).L - env.span) {
    atomicOr(flag, 1);
    return;
  }
  RegAcc<C> a;
  a.ring = env.ring + (int64_t)e * kRing;
  a.fam() = fam;  // the env keeps its episode's trace family
  env_reset_at<C>(env, a, o);
  store_reg<C>(env, e, a);
}

// a replay's actions must lie in [0, A)
__global__ void replay_check_kernel(const uint8_t* __restrict__ act, int64_t n, int A, int32_t* __restrict__ flag) {
  int bad = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    bad |= act[i] >= A;
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(flag, 1);
}

pe_status replay_check(const uint8_t* act, int64_t n, int A, int32_t* flag, cudaStream_t st) {
  PE_TRY_CUDA(cudaMemsetAsync(flag, 0, sizeof(int32_t), st));
  replay_check_kernel<<<(int)std::min<int64_t>(ceil_div(n, 256), 4096), 256, 0, st>>>(act, n, A, flag);
  PE_CHECK_LAUNCH("replay_check_kernel");
  int32_t host = 0;
  PE_TRY_CUDA(cudaMemcpyAsync(&host, flag, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  if (host) return fail(PE_EINVAL, "replay action outside [0, A)");
  return PE_OK;
}

pe_status rule_rollout(const EnvDev& env, const RuleArgs& r, const pe_rollout_buf& buf, cudaStream_t st) {
  const int grid = ceil_div(env.E, 128);
  ProfScope ps(PE_PROF_ROLLOUT, st);
  if (env.C == 1 && env.obs_kind == PE_OBS_TINY8)
    rule_rollout_kernel<1, PE_OBS_TINY8, 8><<<grid, 128, 0, st>>>(env, r, buf);
  else if (env.C == 1 && env.obs_kind == PE_OBS_7B16)
    rule_rollout_kernel<1, PE_OBS_7B16, 16><<<grid, 128, 0, st>>>(env, r, buf);
  else if (env.C == 4 && env.obs_kind == PE_OBS_OCC32)
    rule_rollout_kernel<4, PE_OBS_OCC32, 32><<<grid, 128, 0, st>>>(env, r, buf);
  else if (env.C == 4 && env.obs_kind == PE_OBS_OCC64)
    rule_rollout_kernel<4, PE_OBS_OCC64, 64><<<grid, 128, 0, st>>>(env, r, buf);
  else
    return fail(PE_EINVAL, "rule rollout: unsupported env (C=%d, obs kind %d)", env.C, env.obs_kind);
  PE_CHECK_LAUNCH("rule_rollout_kernel");
  return PE_OK;
}

pe_status env_set_offsets(const EnvDev& env, const int32_t* offsets, int32_t* flag, cudaStream_t st) {
  const int grid = ceil_div(env.E, 128);
  PE_TRY_CUDA(cudaMemsetAsync(flag, 0, sizeof(int32_t), st));
  switch (env.C) {
    case 1: env_offsets_kernel<1><<<grid, 128, 0, st>>>(env, offsets, flag); break;
    case 2: env_offsets_kernel<2><<<grid, 128, 0, st>>>(env, offsets, flag); break;
    case 3: env_offsets_kernel<3><<<grid, 128, 0, st>>>(env, offsets, flag); break;
    default: env_offsets_kernel<4><<<grid, 128, 0, st>>>(env, offsets, flag); break;
  }
  PE_CHECK_LAUNCH("env_offsets_kernel");
  int32_t h = 0;
  PE_TRY_CUDA(cudaMemcpyAsync(&h, flag, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  if (h) return fail(PE_EINVAL, "episode offset outside [60, L - episode_len x max(level_samples)]");
  return PE_OK;
}

// Dual ascent on the Eq. 6 multiplier (Eq. 7; the additive G3 form with the
// same relative gap): one block sums the rollout's violation counts exactly
// (int64), then one thread updates lambda in place.  The scalar update runs
// in fp64 (a handful of operations).
__global__ void __launch_bounds__(1024) dual_ascent_kernel(const int32_t* __restrict__ viol, int E, int64_t steps,
                                                           int col, int additive, float target, float eta, float lo,
                                                           float hi, float* __restrict__ lambda,
                                                           float* __restrict__ rate) {
  __shared__ long long red[32];
  long long n = 0;
  for (int e = threadIdx.x; e < E; e += blockDim.x) n += viol[2 * e + col];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long t = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    const double v = (double)t / ((double)E * (double)steps);
    const double gap = (v - (double)target) / (double)target;
    double l = additive ? (double)*lambda + (double)eta * gap : (double)*lambda * exp((double)eta * gap);
    l = l < (double)lo ? (double)lo : (l > (double)hi ? (double)hi : l);
    *lambda = (float)l;
    if (rate) *rate = (float)v;
  }
}

pe_status dual_ascent(const int32_t* viol, int E, int64_t steps, int window, int additive, float target,
                      float eta, float lo, float hi, float* lambda, float* rate, cudaStream_t st) {
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    dual_ascent_kernel<<<1, 1024, 0, st>>>(viol, E, steps, window == 1 ? 0 : 1, additive, target, eta, lo, hi,
                                           lambda, rate);
  }
  PE_CHECK_LAUNCH("dual_ascent_kernel");
  return PE_OK;
}

}  // namespace pe
