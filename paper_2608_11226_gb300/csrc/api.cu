// C ABI of the pe library: argument validation, object lifetime and kernel
// dispatch.  Every argument error is detected here, before any launch.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include "env.cuh"
#include "mlp_f32.cuh"

namespace pe {

static thread_local char g_err[512] = "";

pe_status fail(pe_status code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

pe_status cuda_fail(cudaError_t err, const char* what) {
  snprintf(g_err, sizeof(g_err), "CUDA error %d (%s) in %s", (int)err, cudaGetErrorString(err), what);
  return PE_ECUDA;
}

void clear_error() { g_err[0] = 0; }

// ---------------------------------------------------------------------------
// launch profiling
// ---------------------------------------------------------------------------
struct ProfRec {
  int kind;
  cudaEvent_t a, b;
};
static std::mutex g_prof_mu;
static bool g_prof_on = false;
static std::vector<cudaEvent_t> g_prof_pool;
static std::vector<ProfRec> g_prof_recs;
static thread_local cudaEvent_t g_prof_open = nullptr;

static cudaEvent_t prof_event() {
  if (!g_prof_pool.empty()) {
    cudaEvent_t e = g_prof_pool.back();
    g_prof_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

void prof_mark(int kind, cudaStream_t st, bool begin) {
  if (!g_prof_on) return;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (begin) {
    g_prof_open = prof_event();
    if (g_prof_open) cudaEventRecord(g_prof_open, st);
  } else if (g_prof_open) {
    cudaEvent_t b = prof_event();
    if (b) {
      cudaEventRecord(b, st);
      g_prof_recs.push_back(ProfRec{kind, g_prof_open, b});
    } else {
      g_prof_pool.push_back(g_prof_open);
    }
    g_prof_open = nullptr;
  }
}

// defined in the kernel translation units
pe_status rollout_f32(const EnvDev& env, const pe_net& net, const float* params, int T, uint32_t it,
                      float lambda, int det, const pe_rollout_buf& buf, cudaStream_t st);
pe_status value_f32(const pe_net& net, const float* params, const float* obs, int64_t n,
                    float* value, cudaStream_t st);
pe_status gae_launch(const float* r, const float* v, const uint8_t* d, const float* last_v, int T,
                     int E, float gamma, float lam, float* adv, float* ret, cudaStream_t st);
int64_t ppo_ws_bytes_f32(const pe_net& net, const pe_ppo_config& cfg, int64_t N);
pe_status ppo_update_f32(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                         const float* obs, const uint8_t* act, const float* logp_old,
                         const float* adv, const float* ret, int64_t N, const pe_ppo_config& cfg,
                         float* stats, void* ws, cudaStream_t st);
int64_t ppo_ws_bytes_bf16(const pe_net& net, const pe_ppo_config& cfg, int64_t N);
pe_status ppo_update_bf16(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                          const void* obs, const uint8_t* act, const float* logp_old, const float* adv,
                          const float* ret, int64_t N, const pe_ppo_config& cfg, float* stats, void* ws,
                          cudaStream_t st);
int64_t fleet_ws_bytes(int J, int L, int H);
int64_t fleet_ws_min_bytes(int J, int L, int H);
struct RuleArgs {
  int32_t kind, hi_q, lo_q, drop30_q, climb30_q, climb10_q;
  int32_t T, obs_bf16;
  uint32_t it;
  float lambda;
  const uint8_t* forced;
};
constexpr int32_t kRuleReplay = 4;
pe_status rule_rollout(const EnvDev& env, const RuleArgs& r, const pe_rollout_buf& buf, cudaStream_t st);
pe_status replay_check(const uint8_t* act, int64_t n, int A, int32_t* flag, cudaStream_t st);
pe_status wait_selftest(int mode, int64_t limit_cycles, void* ws, cudaStream_t st);
pe_status env_set_offsets(const EnvDev& env, const int32_t* offsets, int32_t* flag, cudaStream_t st);
pe_status dual_ascent(const int32_t* viol, int E, int64_t steps, int window, int additive, float target,
                      float eta, float lo, float hi, float* lambda, float* rate, cudaStream_t st);
int64_t fleet_stagger_ws_bytes(int J, int L, int H, int stride);
pe_status fleet_stagger_launch(const float* traces, int G, int L, const int32_t* job_of_gpu, int J, int H,
                               int w, int stride, int32_t* offsets_out, int32_t* peaks_out, void* workspace,
                               cudaStream_t st);
int64_t rollout_bf16_ws_bytes(const pe_net& net, int64_t E);
pe_status rollout_bf16(const EnvDev& env, const pe_net& net, const float* params, int T, uint32_t it,
                       float lambda, int det, const pe_rollout_buf& buf, void* ws, cudaStream_t st);
pe_status value_bf16(const pe_net& net, const float* params, const void* obs, int64_t n, float* value,
                     void* ws, cudaStream_t st);
int64_t value_bf16_ws_bytes(const pe_net& net);
pe_status device_check(cudaStream_t st);
pe_status fleet_launch(const float* traces, int G, int L, const int32_t* job_of_gpu, int J,
                       const int32_t* offsets, int64_t N, int H, const int32_t* windows, int W,
                       int64_t budget_q, int32_t* counts, int32_t* peaks, void* workspace,
                       int64_t workspace_bytes, cudaStream_t st);

static int obs_width(int kind) {
  switch (kind) {
    case PE_OBS_TINY8: return 8;
    case PE_OBS_7B16: return 16;
    case PE_OBS_OCC32: return 32;
    case PE_OBS_OCC64: return 64;
    default: return -1;
  }
}

// first episode of every env (Sec. 4.1 random offset, warm-started history and
// window sums), through the same reset as later episodes
template <int C>
__global__ void env_init_kernel(EnvDev env) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= env.E) return;
  RegAcc<C> a;
  a.ring = env.ring + (int64_t)e * kRing;
  env_reset<C>(env, a, (uint32_t)e, 0u, 0u, kDrawInit);
  store_reg<C>(env, e, a);
}

static void launch_env_init(const EnvDev& d) {
  const int grid = ceil_div(d.E, 256);
  switch (d.C) {
    case 1: env_init_kernel<1><<<grid, 256>>>(d); break;
    case 2: env_init_kernel<2><<<grid, 256>>>(d); break;
    case 3: env_init_kernel<3><<<grid, 256>>>(d); break;
    default: env_init_kernel<4><<<grid, 256>>>(d); break;
  }
}

}  // namespace pe

using namespace pe;

struct pe_env {
  pe_env_config cfg;
  EnvDev dev;
  int device;
  int32_t* flag;  // device word for set-up checks (episode offsets)
};

extern "C" {

const char* pe_last_error(void) { return g_err; }

static const char* kProfNames[PE_PROF_KINDS] = {
    "rollout", "value", "gae", "ppo_grad", "ppo_reduce", "ppo_adam", "ppo_other",
    "fleet_prepare", "fleet_windows", "mlp_policy_tc", "mlp_value_tc"};

const char* pe_profile_kind_name(int32_t kind) {
  return (kind >= 0 && kind < PE_PROF_KINDS) ? kProfNames[kind] : "";
}

pe_status pe_profile_enable(int32_t on) {
  clear_error();
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_on = on != 0;
  return PE_OK;
}

pe_status pe_profile_read(int32_t kind, double* total_ms, int64_t* launches) {
  clear_error();
  if (kind < 0 || kind >= PE_PROF_KINDS || !total_ms || !launches) return fail(PE_EINVAL, "bad profile query");
  std::lock_guard<std::mutex> lk(g_prof_mu);
  double ms = 0.0;
  int64_t n = 0;
  std::vector<ProfRec> keep;
  for (const ProfRec& r : g_prof_recs) {
    if (r.kind != kind) {
      keep.push_back(r);
      continue;
    }
    PE_TRY_CUDA(cudaEventSynchronize(r.b));
    float t = 0.0f;
    PE_TRY_CUDA(cudaEventElapsedTime(&t, r.a, r.b));
    ms += t;
    ++n;
    g_prof_pool.push_back(r.a);
    g_prof_pool.push_back(r.b);
  }
  g_prof_recs.swap(keep);
  *total_ms = ms;
  *launches = n;
  return PE_OK;
}

int64_t pe_param_count(const pe_net* net) {
  if (!net) return -1;
  return mlp_layout(net->obs_dim, net->hidden, net->n_actions).total;
}

static pe_status check_env_config(const pe_env_config* c) {
  if (c->n_envs < 1) return fail(PE_EINVAL, "n_envs must be >= 1");
  if (c->n_channels < 1 || c->n_channels > PE_MAX_CHANNELS) return fail(PE_EINVAL, "n_channels must be in [1, 4]");
  if (c->episode_len < 1) return fail(PE_EINVAL, "episode_len must be >= 1");
  int32_t nmax = 1;
  for (int l = 0; l < PE_MAX_LEVELS; ++l) {
    if (c->level_samples[l] < 0 || c->level_samples[l] > 1024)
      return fail(PE_EINVAL, "level_samples[%d] outside [0, 1024]", l);
    if (c->level_samples[l] > nmax) nmax = c->level_samples[l];
  }
  if (c->n_families < 0 || c->n_families > PE_MAX_FAMILIES) return fail(PE_EINVAL, "n_families must be in [0, 4]");
  const int nf = c->n_families > 1 ? c->n_families : 1;
  for (int f = 0; f < nf; ++f) {
    const int64_t L = c->n_families > 1 ? c->fam_len[f] : c->trace_len;
    const int32_t ch = c->n_families > 1 ? c->fam_channels[f] : c->n_channels;
    const int64_t B = c->n_families > 1 ? c->fam_budget_q[f] : c->budget_q;
    if (L < (int64_t)c->episode_len * nmax + kWLong)
      return fail(PE_EINVAL, "trace length (%lld) must be >= episode_len x max(level_samples) + 60", (long long)L);
    if (ch < 1 || ch > c->n_channels) return fail(PE_EINVAL, "family channel count outside [1, n_channels]");
    if (B < 1 || B * kWLong * PE_MAX_CHANNELS >= INT32_MAX) return fail(PE_EINVAL, "budget_q out of range");
  }
  if (obs_width(c->obs_kind) < 0) return fail(PE_EINVAL, "unknown obs_kind %d", c->obs_kind);
  if (c->n_levels < 1 || c->n_levels > PE_MAX_LEVELS) return fail(PE_EINVAL, "n_levels must be in [1, 32]");
  if (c->level_init < 0 || c->level_init >= c->n_levels) return fail(PE_EINVAL, "level_init out of range");
  if (c->actuator_kind == PE_ACT_INCDEC) {
    if (c->n_actions != 5) return fail(PE_EINVAL, "the inc/dec actuator has 5 actions");
    if (c->g_min < 0 || c->g_max >= c->n_levels || c->g_max <= 0 || c->g_min > c->g_max ||
        c->level_init < c->g_min || c->level_init > c->g_max)
      return fail(PE_EINVAL, "group-size range [g_min, g_max] invalid");
    if (c->b_min < 1 || c->b_min > c->b_max || c->b_init < c->b_min || c->b_init > c->b_max ||
        (c->obs_kind == PE_OBS_7B16 && c->b_max == c->b_min))
      return fail(PE_EINVAL, "batch range [b_min, b_max] invalid");
  } else if (c->actuator_kind == PE_ACT_SET_LEVEL) {
    if (c->n_actions < 1 || c->n_actions > c->n_levels) return fail(PE_EINVAL, "n_actions must be in [1, n_levels]");
    if (c->obs_kind == PE_OBS_TINY8 && c->n_levels < 2) return fail(PE_EINVAL, "TINY8 needs >= 2 levels");
  } else {
    return fail(PE_EINVAL, "unknown actuator_kind %d", c->actuator_kind);
  }
  if (c->obs_kind == PE_OBS_7B16 && c->actuator_kind != PE_ACT_INCDEC)
    return fail(PE_EINVAL, "7B16 observations need the inc/dec actuator");
  (void)0;  // budgets checked per trace family above
  if (c->reward_kind != PE_REWARD_FIXED && c->reward_kind != PE_REWARD_LAGRANGE)
    return fail(PE_EINVAL, "unknown reward_kind");
  if (c->reward_window != 1 && c->reward_window != kWLong) return fail(PE_EINVAL, "reward_window must be 1 or 60");
  return PE_OK;
}

pe_status pe_env_create(const pe_env_config* cfg, const float* trace, const uint8_t* phase,
                        pe_env** out) {
  clear_error();
  if (!cfg || !trace || !phase || !out) return fail(PE_EINVAL, "null argument");
  *out = nullptr;
  pe_status s = check_env_config(cfg);
  if (s != PE_OK) return s;
  const int C = cfg->n_channels, L = cfg->trace_len, E = cfg->n_envs;
  // trace families (one: the single [C][L] trace)
  const int F = cfg->n_families > 1 ? cfg->n_families : 1;
  int32_t fL[PE_MAX_FAMILIES], fC[PE_MAX_FAMILIES], fB[PE_MAX_FAMILIES];
  int64_t ftoff[PE_MAX_FAMILIES], fpoff[PE_MAX_FAMILIES], tot_t = 0, tot_p = 0;
  for (int f = 0; f < F; ++f) {
    fL[f] = cfg->n_families > 1 ? cfg->fam_len[f] : L;
    fC[f] = cfg->n_families > 1 ? cfg->fam_channels[f] : C;
    fB[f] = cfg->n_families > 1 ? cfg->fam_budget_q[f] : cfg->budget_q;
    ftoff[f] = tot_t;
    fpoff[f] = tot_p;
    tot_t += (int64_t)C * fL[f];
    tot_p += fL[f];
  }
  // host copies for validation (trace and phase may live in host or device memory)
  std::vector<float> h((size_t)tot_t);
  std::vector<uint8_t> ph((size_t)tot_p);
  PE_TRY_CUDA(cudaMemcpy(h.data(), trace, sizeof(float) * h.size(), cudaMemcpyDefault));
  PE_TRY_CUDA(cudaMemcpy(ph.data(), phase, ph.size(), cudaMemcpyDefault));
  for (int64_t i = 0; i < tot_p; ++i)
    if (ph[i] > 7) return fail(PE_EINVAL, "phase label %d at %lld outside [0, 7]", (int)ph[i], (long long)i);
  pe_env* env = new pe_env();
  env->cfg = *cfg;
  EnvDev& d = env->dev;
  memset(&d, 0, sizeof(d));
  d.E = E; d.C = C; d.L = fL[0]; d.A = cfg->n_actions; d.obs_kind = cfg->obs_kind;
  d.act_kind = cfg->actuator_kind; d.n_levels = cfg->n_levels; d.level_init = cfg->level_init;
  d.g_min = cfg->g_min; d.g_max = cfg->g_max; d.b_min = cfg->b_min; d.b_max = cfg->b_max;
  d.b_init = cfg->b_init; d.ep_len = cfg->episode_len; d.budget_q = fB[0];
  d.F = F;
  for (int f = 0; f < F; ++f) {
    d.fL[f] = fL[f];
    d.fC[f] = fC[f];
    d.fB[f] = fB[f];
  }
  d.phase_mask = cfg->scale_phase_mask; d.reward_kind = cfg->reward_kind;
  d.reward_window = cfg->reward_window; d.r_ok = cfg->r_ok; d.r_viol = cfg->r_viol;
  d.bonus_coef = cfg->bonus_coef; d.seed = cfg->seed;
  // actuator table: Sec. 4.1 formula for the group-size actuator, else the given table
  for (int l = 0; l < PE_MAX_LEVELS; ++l)
    for (int c = 0; c < PE_MAX_CHANNELS; ++c) {
      if (cfg->actuator_kind == PE_ACT_INCDEC)
        d.scale[l][c] = (float)(0.8 + 0.2 * (double)l / (double)cfg->g_max);
      else
        d.scale[l][c] = cfg->level_scale[l][c];
    }
  for (int l = 0; l < PE_MAX_LEVELS; ++l) d.tokens[l] = cfg->level_tokens[l];
  int32_t nmax = 1;
  d.cadence = 0;
  for (int l = 0; l < PE_MAX_LEVELS; ++l) {
    d.ns[l] = cfg->level_samples[l] > 0 ? cfg->level_samples[l] : 1;
    if (cfg->level_samples[l] > 0) d.cadence = 1;
    if (d.ns[l] > nmax) nmax = d.ns[l];
  }
  d.span = cfg->episode_len * nmax;
  double rmax = 0.0;
  if (cfg->actuator_kind == PE_ACT_INCDEC) {
    for (int l = cfg->g_min; l <= cfg->g_max; ++l)
      rmax = fmax(rmax, (double)cfg->level_tokens[l] * cfg->b_max / cfg->b_init);
  } else {
    for (int l = 0; l < cfg->n_levels; ++l) rmax = fmax(rmax, (double)cfg->level_tokens[l]);
  }
  d.inv_rate_max = rmax > 0 ? (float)(1.0 / rmax) : 0.0f;
  // fixed-point range: every actuated sample and every 60-sample cluster sum must fit in int32
  double qmax = 0.0;
  for (int c = 0; c < C; ++c) {
    float smax = 1.0f;
    for (int l = 0; l < cfg->n_levels; ++l) smax = fmaxf(smax, d.scale[l][c]);
    if (!(smax >= 0.0f) || !std::isfinite(smax)) { delete env; return fail(PE_EINVAL, "actuator scale not finite"); }
    for (int f = 0; f < F; ++f) {
      if (c >= fC[f]) continue;  // channels a family does not have are never read
      for (int i = 0; i < fL[f]; ++i) {
        const float x = h[(size_t)(ftoff[f] + (int64_t)c * fL[f] + i)];
        if (!std::isfinite(x) || x < 0.0f) { delete env; return fail(PE_EOVERFLOW, "trace sample (%d, %d) of family %d is not a finite non-negative power", c, i, f); }
        qmax = fmax(qmax, (double)x * smax * 64.0);
      }
    }
  }
  if (qmax * C * kWLong >= 2147483000.0) { delete env; return fail(PE_EOVERFLOW, "trace too large for the 1/64 W fixed point"); }
  cudaError_t e1 = cudaGetDevice(&env->device);
  float* dtrace = nullptr;
  uint8_t* dphase = nullptr;
  int32_t* st = nullptr;
  uint8_t* ring = nullptr;
  int32_t* sums = nullptr;
  int32_t* flag = nullptr;
  if (e1 == cudaSuccess) e1 = cudaMalloc(&dtrace, sizeof(float) * h.size());
  if (e1 == cudaSuccess) e1 = cudaMalloc(&dphase, ph.size());
  if (e1 == cudaSuccess) e1 = cudaMalloc(&st, sizeof(int32_t) * kStN * (size_t)E);
  if (e1 == cudaSuccess) e1 = cudaMalloc(&ring, (size_t)kRing * E);
  if (e1 == cudaSuccess) e1 = cudaMalloc(&sums, sizeof(int32_t) * 8 * (size_t)E);
  if (e1 == cudaSuccess) e1 = cudaMalloc(&flag, sizeof(int32_t));
  if (e1 != cudaSuccess) {
    cudaFree(dtrace); cudaFree(dphase); cudaFree(st); cudaFree(ring); cudaFree(sums); cudaFree(flag);
    delete env;
    return e1 == cudaErrorMemoryAllocation ? fail(PE_ENOMEM, "device allocation failed")
                                           : cuda_fail(e1, "pe_env_create");
  }
  for (int f = 0; f < F; ++f) {
    d.ftrace[f] = dtrace + ftoff[f];
    d.fphase[f] = dphase + fpoff[f];
  }
  d.st = st; d.ring = ring; d.sums = sums;
  env->flag = flag;
  PE_TRY_CUDA(cudaMemcpy(dtrace, h.data(), sizeof(float) * h.size(), cudaMemcpyHostToDevice));
  PE_TRY_CUDA(cudaMemcpy(dphase, ph.data(), ph.size(), cudaMemcpyHostToDevice));
  launch_env_init(d);  // one-time set-up, not profiled
  PE_CHECK_LAUNCH("env_init_kernel");
  PE_TRY_CUDA(cudaDeviceSynchronize());
  *out = env;
  return PE_OK;
}

pe_status pe_env_destroy(pe_env* env) {
  clear_error();
  if (!env) return PE_OK;
  cudaFree((void*)env->dev.ftrace[0]);
  cudaFree((void*)env->dev.fphase[0]);
  cudaFree(env->dev.st);
  cudaFree(env->dev.ring);
  cudaFree(env->dev.sums);
  cudaFree(env->flag);
  delete env;
  return PE_OK;
}

int64_t pe_env_state_bytes(const pe_env* env) {
  if (!env) return -1;
  return (int64_t)env->dev.E * (kStN * 4 + kRing + 8 * 4);
}

pe_status pe_env_save(const pe_env* env, void* host_dst) {
  clear_error();
  if (!env || !host_dst) return fail(PE_EINVAL, "null argument");
  const size_t E = (size_t)env->dev.E;
  char* p = reinterpret_cast<char*>(host_dst);
  PE_TRY_CUDA(cudaDeviceSynchronize());
  PE_TRY_CUDA(cudaMemcpy(p, env->dev.st, E * kStN * 4, cudaMemcpyDeviceToHost));
  PE_TRY_CUDA(cudaMemcpy(p + E * kStN * 4, env->dev.ring, E * kRing, cudaMemcpyDeviceToHost));
  PE_TRY_CUDA(cudaMemcpy(p + E * (kStN * 4 + kRing), env->dev.sums, E * 32, cudaMemcpyDeviceToHost));
  return PE_OK;
}

pe_status pe_env_load(pe_env* env, const void* host_src) {
  clear_error();
  if (!env || !host_src) return fail(PE_EINVAL, "null argument");
  const size_t E = (size_t)env->dev.E;
  const char* p = reinterpret_cast<const char*>(host_src);
  const int32_t* st = reinterpret_cast<const int32_t*>(p);
  const uint8_t* ring = reinterpret_cast<const uint8_t*>(p + E * kStN * 4);
  const pe_env_config& c = env->cfg;
  for (size_t e = 0; e < E; ++e) {
    const int32_t pos = st[kStPos * E + e], k = st[kStK * E + e];
    if (pos < kWLong || pos + (c.episode_len - k) > c.trace_len || k < 0 || k >= c.episode_len)
      return fail(PE_EINVAL, "state image: env %zu has an invalid position", e);
    for (int f = kStLevel; f <= kStPrev; ++f)
      if (st[f * E + e] < 0 || st[f * E + e] >= c.n_levels) return fail(PE_EINVAL, "state image: bad level");
    for (int i = 0; i < kRing; ++i)
      if (ring[e * kRing + i] >= c.n_levels) return fail(PE_EINVAL, "state image: bad level ring");
  }
  PE_TRY_CUDA(cudaDeviceSynchronize());
  PE_TRY_CUDA(cudaMemcpy(env->dev.st, p, E * kStN * 4, cudaMemcpyHostToDevice));
  PE_TRY_CUDA(cudaMemcpy(env->dev.ring, p + E * kStN * 4, E * kRing, cudaMemcpyHostToDevice));
  PE_TRY_CUDA(cudaMemcpy(env->dev.sums, p + E * (kStN * 4 + kRing), E * 32, cudaMemcpyHostToDevice));
  return PE_OK;
}

static pe_status check_net(const pe_net* net) {
  if (!net) return fail(PE_EINVAL, "null network");
  if (net->obs_dim < 1 || net->hidden < 4 || net->n_actions < 1 || (net->dtype != PE_F32 && net->dtype != PE_BF16))
    return fail(PE_EINVAL, "invalid network description");
  return PE_OK;
}

pe_status pe_env_set_offsets(pe_env* env, const int32_t* offsets, void* stream) {
  clear_error();
  if (!env || !offsets) return fail(PE_EINVAL, "null argument");
  return env_set_offsets(env->dev, offsets, env->flag, reinterpret_cast<cudaStream_t>(stream));
}

pe_status pe_rollout_rule(pe_env* env, const pe_rule* rule, int32_t horizon, uint32_t iteration, float lambda,
                          int32_t obs_bf16, const pe_rollout_buf* buf, void* stream) {
  clear_error();
  if (!env || !rule || !buf) return fail(PE_EINVAL, "null argument");
  if (rule->kind < PE_RULE_RANDOM || rule->kind > PE_RULE_HYSTERESIS) return fail(PE_EINVAL, "unknown rule kind %d", rule->kind);
  if (horizon < 1) return fail(PE_EINVAL, "horizon must be >= 1");
  if ((int64_t)horizon * env->dev.E > (int64_t)INT32_MAX) return fail(PE_EINVAL, "horizon * n_envs too large");
  if (!buf->act || !buf->reward || !buf->done || !buf->viol || !buf->tokens || !buf->excess || !buf->energy_q)
    return fail(PE_EINVAL, "null rollout buffer field");
  RuleArgs r{rule->kind, rule->hi_q, rule->lo_q, rule->drop30_q, rule->climb30_q, rule->climb10_q,
             horizon, obs_bf16 ? 1 : 0, iteration, lambda, nullptr};
  return rule_rollout(env->dev, r, *buf, reinterpret_cast<cudaStream_t>(stream));
}

pe_status pe_wait_selftest(int32_t mode, int64_t limit_cycles, void* workspace, void* stream) {
  clear_error();
  if (mode < 0 || mode > 2) return fail(PE_EINVAL, "mode must be 0, 1 or 2");
  if (limit_cycles < 1000 || limit_cycles > 8000000000LL) return fail(PE_EINVAL, "limit_cycles outside [1e3, 8e9]");
  if (!workspace) return fail(PE_EINVAL, "null workspace");
  return wait_selftest(mode, limit_cycles, workspace, reinterpret_cast<cudaStream_t>(stream));
}

pe_status pe_rollout_replay(pe_env* env, const uint8_t* actions, int32_t horizon, uint32_t iteration, float lambda,
                            int32_t obs_bf16, const pe_rollout_buf* buf, void* stream) {
  clear_error();
  if (!env || !actions || !buf) return fail(PE_EINVAL, "null argument");
  if (horizon < 1) return fail(PE_EINVAL, "horizon must be >= 1");
  if ((int64_t)horizon * env->dev.E > (int64_t)INT32_MAX) return fail(PE_EINVAL, "horizon * n_envs too large");
  if (!buf->act || !buf->reward || !buf->done || !buf->viol || !buf->tokens || !buf->excess || !buf->energy_q)
    return fail(PE_EINVAL, "null rollout buffer field");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  pe_status s = replay_check(actions, (int64_t)horizon * env->dev.E, env->dev.A, env->flag, st);
  if (s != PE_OK) return s;
  RuleArgs r{kRuleReplay, 0, 0, 0, 0, 0, horizon, obs_bf16 ? 1 : 0, iteration, lambda, actions};
  return rule_rollout(env->dev, r, *buf, st);
}

pe_status pe_dual_ascent(const int32_t* viol, int32_t n_envs, int64_t steps, int32_t window, int32_t additive,
                         float target, float eta, float lambda_min, float lambda_max, float* lambda, float* rate,
                         void* stream) {
  clear_error();
  if (!viol || !lambda) return fail(PE_EINVAL, "null argument");
  if (n_envs < 1 || steps < 1) return fail(PE_EINVAL, "n_envs >= 1 and steps >= 1 required");
  if (window != 1 && window != 60) return fail(PE_EINVAL, "window must be 1 or 60");
  if (!(target > 0.0f && target < 1.0f)) return fail(PE_EINVAL, "target must be in (0, 1)");
  if (!(lambda_min >= 0.0f && lambda_max >= lambda_min) || !std::isfinite(eta) || !std::isfinite(lambda_max))
    return fail(PE_EINVAL, "need 0 <= lambda_min <= lambda_max and a finite eta");
  return dual_ascent(viol, n_envs, steps, window, additive ? 1 : 0, target, eta, lambda_min, lambda_max, lambda,
                     rate, reinterpret_cast<cudaStream_t>(stream));
}

int64_t pe_rollout_workspace_bytes(const pe_env* env, const pe_net* net) {
  if (!env || !net) return -1;
  if (net->dtype == PE_F32) return 0;
  return rollout_bf16_ws_bytes(*net, env->dev.E);
}

static bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

pe_status pe_rollout(pe_env* env, const pe_net* net, const float* params, int32_t horizon,
                     uint32_t iteration, float lambda, int32_t flags, const pe_rollout_buf* buf,
                     void* workspace, int64_t workspace_bytes, void* stream) {
  clear_error();
  if (!env || !params || !buf) return fail(PE_EINVAL, "null argument");
  pe_status s = check_net(net);
  if (s != PE_OK) return s;
  if (horizon < 1) return fail(PE_EINVAL, "horizon must be >= 1");
  if (net->obs_dim != obs_width(env->cfg.obs_kind) || net->n_actions != env->cfg.n_actions)
    return fail(PE_EINVAL, "network does not match the env (obs_dim %d vs %d, actions %d vs %d)",
                net->obs_dim, obs_width(env->cfg.obs_kind), net->n_actions, env->cfg.n_actions);
  if (!buf->obs || !buf->obs_last || !buf->act || !buf->logp || !buf->value || !buf->last_value ||
      !buf->reward || !buf->done || !buf->viol || !buf->tokens || !buf->excess || !buf->energy_q)
    return fail(PE_EINVAL, "null rollout buffer field");
  if ((int64_t)horizon * env->dev.E > (int64_t)INT32_MAX) return fail(PE_EINVAL, "horizon * n_envs too large");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int det = (flags & PE_ROLLOUT_DETERMINISTIC) ? 1 : 0;
  if (net->dtype == PE_F32) {
    s = rollout_f32(env->dev, *net, params, horizon, iteration, lambda, det, *buf, st);
    if (s != PE_OK) return s;
    s = value_f32(*net, params, reinterpret_cast<const float*>(buf->obs), (int64_t)horizon * env->dev.E,
                  buf->value, st);
    if (s != PE_OK) return s;
    return value_f32(*net, params, reinterpret_cast<const float*>(buf->obs_last), env->dev.E,
                     buf->last_value, st);
  }
  const int64_t need = rollout_bf16_ws_bytes(*net, env->dev.E);
  if (need < 0) return fail(PE_EINVAL, "unsupported bf16 network (D=%d H=%d)", net->obs_dim, net->hidden);
  if (!workspace || workspace_bytes < need)
    return fail(PE_EINVAL, "workspace too small (%lld < %lld bytes)", (long long)workspace_bytes, (long long)need);
  if (misaligned(workspace, 256) || misaligned(buf->obs, 16) || misaligned(buf->obs_last, 16))
    return fail(PE_EINVAL, "bf16 rollout: workspace must be 256-byte and obs buffers 16-byte aligned");
  return rollout_bf16(env->dev, *net, params, horizon, iteration, lambda, det, *buf, workspace, st);
}

int64_t pe_value_workspace_bytes(const pe_net* net) {
  if (!net) return -1;
  if (net->dtype == PE_F32) return 0;
  return value_bf16_ws_bytes(*net);
}

pe_status pe_value(const pe_net* net, const float* params, const void* obs, int64_t n,
                   float* value, void* workspace, int64_t workspace_bytes, void* stream) {
  clear_error();
  pe_status s = check_net(net);
  if (s != PE_OK) return s;
  if (!params || (n > 0 && (!obs || !value))) return fail(PE_EINVAL, "null argument");
  if (n < 0) return fail(PE_EINVAL, "n must be >= 0");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (net->dtype == PE_F32) return value_f32(*net, params, reinterpret_cast<const float*>(obs), n, value, st);
  const int64_t need = value_bf16_ws_bytes(*net);
  if (need < 0) return fail(PE_EINVAL, "unsupported bf16 value network (D=%d H=%d)", net->obs_dim, net->hidden);
  if (!workspace || workspace_bytes < need)
    return fail(PE_EINVAL, "workspace too small (%lld < %lld bytes)", (long long)workspace_bytes, (long long)need);
  if (misaligned(workspace, 256) || misaligned(obs, 16))
    return fail(PE_EINVAL, "bf16 value: workspace must be 256-byte and obs 16-byte aligned");
  return value_bf16(*net, params, obs, n, value, workspace, st);
}

pe_status pe_device_check(void* stream) {
  clear_error();
  return device_check(reinterpret_cast<cudaStream_t>(stream));
}

pe_status pe_gae(const float* reward, const float* value, const uint8_t* done,
                 const float* last_value, int32_t T, int32_t E, float gamma, float lam,
                 float* adv, float* ret, void* stream) {
  clear_error();
  if (T < 0 || E < 0) return fail(PE_EINVAL, "T and E must be >= 0");
  if (T == 0 || E == 0) return PE_OK;
  if (!reward || !value || !done || !last_value || !adv || !ret) return fail(PE_EINVAL, "null argument");
  if ((int64_t)T * E > (int64_t)1 << 40) return fail(PE_EINVAL, "T * E too large");
  if (!std::isfinite(gamma) || !std::isfinite(lam)) return fail(PE_EINVAL, "gamma and lambda must be finite");
  return gae_launch(reward, value, done, last_value, T, E, gamma, lam, adv, ret,
                    reinterpret_cast<cudaStream_t>(stream));
}

static pe_status check_ppo(const pe_net* net, const pe_ppo_config* cfg, int64_t n) {
  pe_status s = check_net(net);
  if (s != PE_OK) return s;
  if (!cfg) return fail(PE_EINVAL, "null PPO config");
  if (cfg->epochs < 1 || cfg->epochs > 16) return fail(PE_EINVAL, "epochs must be in [1, 16]");
  if (cfg->minibatch < 1) return fail(PE_EINVAL, "minibatch must be >= 1");
  if (n < 1 || n > (int64_t)INT32_MAX) return fail(PE_EINVAL, "n_samples must be in [1, 2^31)");
  return PE_OK;
}

static int64_t ppo_ws_bytes(const pe_net& net, const pe_ppo_config& cfg, int64_t n) {
  return net.dtype == PE_BF16 ? ppo_ws_bytes_bf16(net, cfg, n) : ppo_ws_bytes_f32(net, cfg, n);
}

int64_t pe_ppo_workspace_bytes(const pe_net* net, const pe_ppo_config* cfg, int64_t n_samples) {
  if (check_ppo(net, cfg, n_samples) != PE_OK) return -1;
  return ppo_ws_bytes(*net, *cfg, n_samples);
}

pe_status pe_ppo_update(const pe_net* net, float* params, float* adam_m, float* adam_v,
                        int64_t adam_t, const void* obs, const uint8_t* act,
                        const float* logp_old, const float* adv, const float* ret,
                        int64_t n_samples, const pe_ppo_config* cfg, float* stats,
                        void* workspace, int64_t workspace_bytes, void* stream) {
  clear_error();
  pe_status s = check_ppo(net, cfg, n_samples);
  if (s != PE_OK) return s;
  if (!params || !adam_m || !adam_v || !obs || !act || !logp_old || !adv || !ret || !stats || !workspace)
    return fail(PE_EINVAL, "null argument");
  if (adam_t < 0) return fail(PE_EINVAL, "adam_t must be >= 0");
  const int64_t need = ppo_ws_bytes(*net, *cfg, n_samples);
  if (need < 0) return fail(PE_EINVAL, "unsupported PPO network");
  if (workspace_bytes < need) return fail(PE_EINVAL, "workspace too small (%lld < %lld bytes)", (long long)workspace_bytes, (long long)need);
  if (misaligned(workspace, 256) || misaligned(obs, 16))
    return fail(PE_EINVAL, "workspace must be 256-byte and obs 16-byte aligned");
  if (net->dtype == PE_BF16)
    return ppo_update_bf16(*net, params, adam_m, adam_v, adam_t, obs, act, logp_old, adv, ret, n_samples, *cfg,
                           stats, workspace, reinterpret_cast<cudaStream_t>(stream));
  return ppo_update_f32(*net, params, adam_m, adam_v, adam_t, reinterpret_cast<const float*>(obs),
                        act, logp_old, adv, ret, n_samples, *cfg, stats, workspace,
                        reinterpret_cast<cudaStream_t>(stream));
}

int64_t pe_fleet_workspace_bytes(int32_t J, int32_t L, int32_t H) {
  if (J < 1 || L < 1 || H < 0) return -1;
  return fleet_ws_bytes(J, L, H);
}

pe_status pe_fleet_windows(const float* traces, int32_t G, int32_t L, const int32_t* job_of_gpu,
                           int32_t J, const int32_t* offsets, int64_t N, int32_t H,
                           const int32_t* windows, int32_t W, int64_t budget_q,
                           int32_t* counts, int32_t* peaks, void* workspace,
                           int64_t workspace_bytes, void* stream) {
  clear_error();
  if (G < 1 || G > 64) return fail(PE_EINVAL, "G must be in [1, 64]");
  if (J < 1 || J > 32 || J > G) return fail(PE_EINVAL, "J must be in [1, min(32, G)]");
  if (L < 1 || H < 0 || N < 0) return fail(PE_EINVAL, "L >= 1, H >= 0 and N >= 0 required");
  if ((int64_t)L + H > (int64_t)INT32_MAX) return fail(PE_EINVAL, "L + H too large");
  if (W < 1 || W > 4 || !windows) return fail(PE_EINVAL, "W must be in [1, 4] with a host window array");
  for (int k = 0; k < W; ++k)
    if (windows[k] < 1 || windows[k] > 992) return fail(PE_EINVAL, "window %d outside [1, 992]", windows[k]);
  if (budget_q < 0) return fail(PE_EINVAL, "budget_q must be >= 0");
  if (!traces || !job_of_gpu || !workspace || (N > 0 && (!offsets || !counts || !peaks)))
    return fail(PE_EINVAL, "null argument");
  if (workspace_bytes < fleet_ws_min_bytes(J, L, H)) return fail(PE_EINVAL, "workspace too small");
  return fleet_launch(traces, G, L, job_of_gpu, J, offsets, N, H, windows, W, budget_q, counts,
                      peaks, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int64_t pe_fleet_stagger_workspace_bytes(int32_t J, int32_t L, int32_t H, int32_t stride) {
  if (J < 1 || J > 32 || L < 1 || H < 1 || stride < 1) return -1;
  return fleet_stagger_ws_bytes(J, L, H, stride);
}

pe_status pe_fleet_stagger(const float* traces, int32_t G, int32_t L, const int32_t* job_of_gpu,
                           int32_t J, int32_t H, int32_t w, int32_t stride, int32_t* offsets,
                           int32_t* peaks, void* workspace, int64_t workspace_bytes, void* stream) {
  clear_error();
  if (G < 1 || G > 64) return fail(PE_EINVAL, "G must be in [1, 64]");
  if (J < 1 || J > 32 || J > G) return fail(PE_EINVAL, "J must be in [1, min(32, G)]");
  if (L < 1 || H < 1) return fail(PE_EINVAL, "L >= 1 and H >= 1 required");
  if ((int64_t)L + H > (int64_t)INT32_MAX) return fail(PE_EINVAL, "L + H too large");
  if (w < 1 || w > 992) return fail(PE_EINVAL, "window %d outside [1, 992]", w);
  if (stride < 1) return fail(PE_EINVAL, "stride must be >= 1");
  if (!traces || !job_of_gpu || !offsets || !peaks || !workspace) return fail(PE_EINVAL, "null argument");
  if (workspace_bytes < fleet_stagger_ws_bytes(J, L, H, stride)) return fail(PE_EINVAL, "workspace too small");
  return fleet_stagger_launch(traces, G, L, job_of_gpu, J, H, w, stride, offsets, peaks, workspace,
                              reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
