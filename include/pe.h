/*
 * pe.h -- C ABI of the GB300 library for batched, trace-driven training of
 * the PPO power meta-controller of "Cutting AI Datacenter Energy with
 * Reinforcement Learning: Measured Power Control of LLM Training from One
 * GPU to the Fleet" (arxiv 2608.11226).
 *
 * The library runs every step of the path on one GPU (sm_103a):
 *   pe_env_create   -- load a power trace, validate it, place E envs      (Sec. 4.1)
 *   pe_rollout      -- E envs x T steps: observe, policy, sample, actuate,
 *                      windows, reward; then the value network            (Sec. 4.1, 4.2, Eqs. 1-6)
 *   pe_gae          -- reverse-time generalised advantage estimation       (Sec. 4.2)
 *   pe_ppo_update   -- epochs x minibatches of clipped-loss PPO with Adam  (Sec. 4.2, 4.5)
 *   pe_fleet_windows-- composed fleet traces, window violation counts and
 *                      peaks over 0.5 s / 30 s / 5 min windows             (Sec. 7, 8, Eqs. 1-2)
 *
 * Conventions
 *  - Every buffer argument is a DEVICE pointer owned by the caller, unless
 *    the argument says "host".  The library owns only the opaque pe_env.
 *  - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL = the legacy default stream).  Argument errors are detected before
 *    any launch and returned synchronously; nothing is launched then.
 *  - No call except pe_env_create/pe_env_destroy allocates device memory;
 *    scratch space is a caller-provided workspace whose size the matching
 *    *_workspace_bytes function returns.
 *  - On a non-zero status, pe_last_error() returns a thread-local message.
 *  - No C++ exception crosses this interface.
 *
 * Units: one environment step consumes one half-second power sample
 * (Delta t = 0.5 s, Sec. 4.4).  Power inside the library is an int32 in
 * 1/64 W: q = rint(P * 64) of the fp32 actuated power P, so that window sums
 * and violation counts are exact integers.
 */
#ifndef PE_H
#define PE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t pe_status;
#define PE_OK 0
#define PE_EINVAL 1     /* bad argument (null pointer, size, unsupported shape) */
#define PE_ENOMEM 2     /* device allocation failed (pe_env_create only) */
#define PE_ECUDA 3      /* a CUDA runtime call or launch failed */
#define PE_EOVERFLOW 4  /* trace outside the fixed-point range */
#define PE_ETIMEOUT 5   /* a bounded device-side wait gave up */
#define PE_ESTATE 6     /* object in the wrong state */

#define PE_MAX_LEVELS 32
#define PE_MAX_FAMILIES 4
#define PE_MAX_CHANNELS 4

/* actuator kinds */
#define PE_ACT_SET_LEVEL 0 /* action a selects actuator level a (Table 4 concurrency levels) */
#define PE_ACT_INCDEC 1    /* Sec. 4.1: hold, G-1, G+1, batch-1, batch+1 */
/* observation kinds (width D) */
#define PE_OBS_TINY8 0  /* D=8: Sec. 4.1 state */
#define PE_OBS_7B16 1   /* D=16: last 8 samples, 30 s mean, budget slack, phase, G, b, 10 s mean, 5 s slope */
#define PE_OBS_OCC32 2  /* D=32: Eq. 5 eight-vector + per-channel last 4 samples + per-channel 30 s means */
#define PE_OBS_OCC64 3  /* D=64: Eq. 5 eight-vector + per-channel last 12 + per-channel 10 s and 30 s means */
/* reward kinds */
#define PE_REWARD_FIXED 0    /* Sec. 4.2 G1: +r_ok / r_viol per step plus a throughput bonus */
#define PE_REWARD_LAGRANGE 1 /* Eq. 6 per step: T/1000 - lambda X - 2 lambda max(0, P30 - B) */
/* network element types */
#define PE_F32 0
#define PE_BF16 1
/* pe_rollout flags */
#define PE_ROLLOUT_DETERMINISTIC 1 /* argmax action, lowest index on ties (Sec. 4.4 evaluation) */

/* Environment configuration (Sec. 4.1 MDP; Sec. 4.5 windows and budget).
 * Actuated power of channel c at level l is the fp32 product
 *   P = x_c(p) * s(l, c)  when bit phase(p) of scale_phase_mask is set, else x_c(p),
 * where s(l, c) = level_scale[l][c] for PE_ACT_SET_LEVEL and, for the
 * group-size actuator PE_ACT_INCDEC, s(G) = (float)(0.8 + (0.2 * G) / g_max)
 * evaluated in double (Sec. 4.1).  Tokens per generation-phase sample are
 * level_tokens[l] (times b / b_init for PE_ACT_INCDEC); 0 in other phases. */
typedef struct pe_env_config {
  int32_t n_envs;           /* E >= 1 */
  int32_t n_channels;       /* C in [1, 4]: per-GPU channels summed into cluster power */
  int32_t trace_len;        /* L >= episode_len + 60 */
  int32_t n_actions;        /* A: 5 for INCDEC, n_levels for SET_LEVEL */
  int32_t obs_kind;         /* PE_OBS_* */
  int32_t actuator_kind;    /* PE_ACT_* */
  int32_t n_levels;         /* levels in the tables (INCDEC: g_max + 1) */
  int32_t level_init;       /* level (or G) at every episode start */
  int32_t g_min, g_max;     /* INCDEC group-size range; g_min = 3 is the Sec. 4.2 (G4) floor */
  int32_t b_min, b_max, b_init; /* INCDEC batch-size range and start */
  int32_t episode_len;      /* steps per episode (500, Sec. 4.1) */
  int32_t budget_q;         /* budget B in 1/64 W */
  int32_t scale_phase_mask; /* bit k: samples of phase k are actuated */
  int32_t reward_kind;      /* PE_REWARD_* */
  int32_t reward_window;    /* FIXED reward: violation over 1 sample or 60 samples (30 s) */
  float r_ok, r_viol, bonus_coef; /* FIXED reward: +1, -8, throughput bonus coefficient */
  float level_scale[PE_MAX_LEVELS][PE_MAX_CHANNELS];
  float level_tokens[PE_MAX_LEVELS];
  uint64_t seed;            /* Philox4x32-10 key */
  /* Batch-boundary cadence (Sec. 4.5, Sec. 6.5): samples one step consumes
   * at each level, in [1, 1024]; all zero: one sample per step.  With a
   * table, a step is one generation batch: the windows, violations (Eq. 2)
   * and excess (Eq. 3) advance sample by sample, tokens and excess are
   * summed over the batch, and the Eq. 6 reward takes the batch's largest
   * 30 s excess as its peak term; the Eq. 5 feature d_{k-1}/20 becomes the
   * batch just completed, level_samples[level] x 0.5 s / 20 s.  Episodes
   * are episode_len batches, drawn so that episode_len x max(level_samples)
   * samples fit in the trace. */
  int32_t level_samples[PE_MAX_LEVELS];
  /* Domain randomisation (Sec. 4.2, design G2): n_families in [2, 4] trace
   * families, 0 or 1 for the single trace.  Every episode start draws its
   * family f = floor(w1 * n_families / 2^32) from word 1 of the episode's
   * Philox draw (word 0 keeps choosing the offset, now inside family f).
   * Family f has fam_len[f] samples, fam_channels[f] <= n_channels GPUs and
   * the budget fam_budget_q[f] (1/64 W), which normalises its state and
   * decides its violations (the cap-relative state of G2).  With families,
   * pe_env_create's trace is family-major [f][n_channels][fam_len[f]]
   * (channels at or above fam_channels[f] are ignored) and its phase array
   * [f][fam_len[f]]; trace_len and budget_q are then unused. */
  int32_t n_families;
  int32_t fam_len[PE_MAX_FAMILIES], fam_channels[PE_MAX_FAMILIES], fam_budget_q[PE_MAX_FAMILIES];
} pe_env_config;

/* Policy/value network: two separate tanh MLPs obs_dim -> hidden -> hidden
 * -> {n_actions logits, 1 value} (Sec. 4.2 MLP actor-critic).  Parameters are
 * one flat fp32 vector, row-major W[out][in]:
 *   policy: W1[H][D] b1[H] W2[H][H] b2[H] W3[A][H] b3[A]
 *   value : V1[H][D] c1[H] V2[H][H] c2[H] V3[1][H] c3[1]
 * Supported (D, H, A, dtype): (8,64,3,F32), (16,128,5,F32), (32,256,16,BF16),
 * (64,512,16,BF16).  A BF16 network
 * keeps fp32 master parameters; the library rounds weights, observations and
 * hidden activations to bf16 and accumulates in fp32. */
typedef struct pe_net {
  int32_t obs_dim, hidden, n_actions, dtype;
} pe_net;

/* Rollout buffer, time-major [T][E] (row t holds env 0..E-1).  All device
 * pointers, caller-owned; every one is written by pe_rollout. */
typedef struct pe_rollout_buf {
  void* obs;          /* [T][E][D] fp32 (or bf16 for a BF16 network): observation before step t */
  void* obs_last;     /* [E][D] observation after the last step */
  uint8_t* act;       /* [T][E] action taken */
  float* logp;        /* [T][E] log-probability of the action under the policy */
  float* value;       /* [T][E] value of obs[t] */
  float* last_value;  /* [E]    value of obs_last */
  float* reward;      /* [T][E] */
  uint8_t* done;      /* [T][E] 1 if the episode ended with step t */
  int32_t* viol;      /* [E][2] violating steps of this call: instantaneous (Eq. 2, w=0.5 s), 30 s (Eq. 2) */
  float* tokens;      /* [E]    generated tokens of this call */
  float* excess;      /* [E]    integrated excess of this call, W*s (Eq. 3) */
  int64_t* energy_q;  /* [E]    sum of actuated cluster power over the call, 1/64 W per sample */
  int64_t* samples;   /* [E]    trace samples consumed this call (optional, NULL skips); with a
                       *        cadence table the violation counts are per sample, so rates
                       *        divide by this count */
  int32_t* q;         /* [T][E] actuated cluster power of step t, 1/64 W (summed over the
                       *        batch's samples with a cadence table); optional, NULL skips */
} pe_rollout_buf;

/* PPO configuration (Sec. 4.2 / 4.5; SB3 defaults where the paper is silent) */
typedef struct pe_ppo_config {
  int32_t epochs;        /* passes over the rollout */
  int32_t minibatch;     /* samples per minibatch; the last one of an epoch may be smaller */
  float lr, clip, vf_coef, ent_coef, max_grad_norm, beta1, beta2, eps;
  uint64_t seed;         /* Philox key of the minibatch permutation */
  uint32_t iteration;    /* PPO iteration (part of the permutation counter) */
} pe_ppo_config;

typedef struct pe_env pe_env;

/* Create E environments over one trace (Sec. 4.1 trace replay).
 *  trace: [C][L] fp32 watts, host or device memory (copied).
 *  phase: [L] uint8 phase label per sample (0 generation, 1 update; Sec. 4.4).
 * Every env starts an episode at offset 60 + floor(u * (L - episode_len - 59) / 2^32),
 * u = Philox4x32-10(key = seed, ctr = (env, 0, 0, 2)).out[0]; its 60-sample
 * history is warm-started at level_init.
 * Errors: PE_EINVAL (sizes, kinds, tables), PE_EOVERFLOW (a sample that is
 * not finite, negative, or whose actuated 60-sample window sum could exceed
 * int32), PE_ENOMEM, PE_ECUDA.  Synchronous. */
pe_status pe_env_create(const pe_env_config* cfg, const float* trace, const uint8_t* phase,
                        pe_env** out);
pe_status pe_env_destroy(pe_env* env);

/* Checkpoint: the env state is a flat byte image (host memory). */
int64_t pe_env_state_bytes(const pe_env* env);
pe_status pe_env_save(const pe_env* env, void* host_dst);
pe_status pe_env_load(pe_env* env, const void* host_src);

int64_t pe_param_count(const pe_net* net);

/* One rollout of `horizon` steps for all envs (Sec. 4.1 MDP, Sec. 4.2
 * controller), continuing each env where the previous call left it.
 * Step t of env e: observation -> policy logits -> action (inverse CDF of
 * softmax at u = (philox >> 8) 2^-24, ctr = (e, t, iteration, 0)) -> actuator
 * -> consume one sample -> windows (Eq. 1: 10 s = 20 samples, 30 s = 60)
 * -> violation (Eq. 2), excess (Eq. 3), tokens, reward -> episode end after
 * episode_len steps, new offset from ctr = (e, t, iteration, 1).
 * Then the value network on every observation and on obs_last.
 *  lambda: Lagrange multiplier of Eq. 6 (PE_REWARD_LAGRANGE only).
 *  workspace: >= pe_rollout_workspace_bytes(env, net) bytes of device memory
 *  (0 for fp32 networks: NULL is accepted).  BF16 networks (D=32, H=256 or
 *  D=64, H=512; A=16, 4 channels) run on the tcgen05 tensor cores; their
 *  workspace must be 256-byte and buf->obs / obs_last 16-byte aligned.
 * Errors: PE_EINVAL (unsupported network, null buffer, horizon < 1, small
 * workspace), PE_ECUDA; a bounded tensor-core wait that gives up on the
 * device is reported by pe_device_check. */
int64_t pe_rollout_workspace_bytes(const pe_env* env, const pe_net* net);
pe_status pe_rollout(pe_env* env, const pe_net* net, const float* params, int32_t horizon,
                     uint32_t iteration, float lambda, int32_t flags, const pe_rollout_buf* buf,
                     void* workspace, int64_t workspace_bytes, void* stream);

/* Episodes that start at given trace offsets (the evaluation replay of
 * Sec. 4.4 walks a trace in consecutive 500-step episodes): every env starts
 * a new episode at offsets[e], with its 60-sample history warm-started at
 * the default level as at any episode start.
 *  offsets: [E] int32 device memory, each in [60, L - episode_len].
 * The call waits for the device-side range check.
 * Errors: PE_EINVAL (null argument, an offset out of range; the envs with
 * valid offsets are reset), PE_ECUDA. */
pe_status pe_env_set_offsets(pe_env* env, const int32_t* offsets, void* stream);

/* Baseline rule policies of the evaluation, in place of the network
 * (Sec. 4.4: random policy and the threshold heuristic that lowers the group
 * size above 90% of the cap and raises it below 70%; Sec. 4.5: the
 * hysteresis rule that drops a level when the 30 s mean exceeds 512 W and
 * climbs when the 30 s mean is below 510 W and the 10 s mean below 525 W, at
 * a 561 W budget).  "Lower" and "raise" move G for the inc/dec actuator
 * (actions 1 and 2) and the level index otherwise (clamped to the table).
 * Thresholds are integers in 1/64 W, so decisions are exact:
 *  RANDOM:     a = floor(u * A / 2^32), u = Philox(key = seed, ctr = (e, t, iteration, 0)).out[0];
 *  THRESHOLD:  lower if the latest cluster sample q > hi_q, raise if q < lo_q, else hold;
 *  HYSTERESIS: lower if S30 > 60 drop30_q; raise if S30 < 60 climb30_q and
 *              S10 < 20 climb10_q (Eq. 1 window sums), else hold. */
#define PE_RULE_RANDOM 1
#define PE_RULE_THRESHOLD 2
#define PE_RULE_HYSTERESIS 3
typedef struct pe_rule {
  int32_t kind;
  int32_t hi_q, lo_q;                      /* THRESHOLD, 1/64 W */
  int32_t drop30_q, climb30_q, climb10_q;  /* HYSTERESIS, window means in 1/64 W */
} pe_rule;

/* horizon steps of every env under a rule policy, with the same step,
 * episode-end and counter semantics as pe_rollout.  buf: act, reward, done,
 * viol, tokens, excess and energy_q are required; obs and obs_last are
 * optional (NULL skips them; fp32, or bf16 when obs_bf16 != 0); logp, value
 * and last_value are not touched.
 * Errors: PE_EINVAL (unknown rule, null field, horizon < 1, unsupported env), PE_ECUDA. */
pe_status pe_rollout_rule(pe_env* env, const pe_rule* rule, int32_t horizon, uint32_t iteration,
                          float lambda, int32_t obs_bf16, const pe_rollout_buf* buf, void* stream);

/* Teacher-forced rollout (replay of a given action sequence): env e takes
 * action actions[t][e] at step t and steps exactly as in pe_rollout (actuator,
 * Eqs. 1-3, reward, episode ends and resets drawn from `iteration`), with no
 * network: replaying the actions a pe_rollout call took, from the same env
 * state, reproduces its observations, rewards, done flags and counters.  It
 * serves recorded controllers, constant schedules and parity checks in which
 * one flipped sample must not change the rest of a trajectory.
 *  actions: [horizon][E] uint8 device memory, each in [0, A); checked on the
 *  device first (the call waits for the check; nothing runs on a bad value).
 *  buf: as pe_rollout_rule (act receives a copy of the actions; obs/obs_last
 *  optional, fp32 or bf16 by obs_bf16; logp, value, last_value untouched).
 * Errors: PE_EINVAL (null argument or field, horizon < 1, an action outside
 * [0, A), unsupported env), PE_ECUDA. */
pe_status pe_rollout_replay(pe_env* env, const uint8_t* actions, int32_t horizon, uint32_t iteration,
                            float lambda, int32_t obs_bf16, const pe_rollout_buf* buf, void* stream);

/* Self-test of the library's bounded waits (failure detection without a GPU
 * fault): every spin-wait in the kernels gives up after a clock64 budget,
 * records an error word and returns, so the context stays usable.  This call
 * runs the same waits with budget limit_cycles (in SM clock cycles):
 *  mode 0: the persistent update's grid barrier, 2 CTAs, one of which never
 *          arrives -> the wait runs out -> PE_ETIMEOUT;
 *  mode 1: the same barrier with both CTAs arriving -> PE_OK;
 *  mode 2: an mbarrier wait (as in the tensor-core kernels) that nothing
 *          completes -> PE_ETIMEOUT.
 *  workspace: >= 16 bytes of device memory.  The call waits for the result.
 * Errors: PE_EINVAL (mode outside [0, 2], limit_cycles outside [1e3, 8e9],
 * null workspace), PE_ETIMEOUT (a wait gave up, as modes 0 and 2 intend),
 * PE_ECUDA. */
pe_status pe_wait_selftest(int32_t mode, int64_t limit_cycles, void* workspace, void* stream);

/* Dual ascent on the Lagrange multiplier of the Eq. 6 reward (Eq. 7,
 * Sec. 4.5; the G3 design of Sec. 4.2), from a rollout's violation counts:
 *   v = sum_e viol[e][w] / (n_envs * steps)   (w: 1 = instantaneous, 60 = 30 s window)
 *   multiplicative (additive = 0, Eq. 7): lambda <- clip(lambda exp(eta (v - target) / target), lo, hi)
 *   additive (additive = 1, G3):          lambda <- clip(lambda + eta (v - target) / target, lo, hi)
 *  viol: [n_envs][2] int32 device (pe_rollout_buf.viol); steps: the rollout's horizon;
 *  lambda: device float, read and updated in place; rate: device float out (v), or NULL.
 * The paper's Eq. 7 settings are eta = 0.5, [lo, hi] = [1e-3, 2]; its G3 run used a target of 8%.
 * pe_rollout takes lambda by value, so a caller that feeds the update back reads 4 bytes per
 * iteration.
 * Errors: PE_EINVAL (null pointer, sizes, window not 1 or 60, target outside (0, 1), bounds), PE_ECUDA. */
pe_status pe_dual_ascent(const int32_t* viol, int32_t n_envs, int64_t steps, int32_t window, int32_t additive,
                         float target, float eta, float lambda_min, float lambda_max, float* lambda, float* rate,
                         void* stream);

/* Value network on n observations (fp32, or bf16 for a BF16 network).
 * workspace: >= pe_value_workspace_bytes(net) bytes (0 for fp32); for a BF16
 * network the workspace must be 256-byte and obs 16-byte aligned. */
int64_t pe_value_workspace_bytes(const pe_net* net);
pe_status pe_value(const pe_net* net, const float* params, const void* obs, int64_t n,
                   float* value, void* workspace, int64_t workspace_bytes, void* stream);

/* Generalised advantage estimation (gamma, lambda per Sec. 4.2), time-major:
 *   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,  V_T = last_value,
 *   A_t = delta_t + gamma lambda (1 - d_t) A_{t+1},  ret_t = A_t + V_t.
 * reward, value, adv, ret: [T][E] fp32; done: [T][E] uint8; last_value: [E].
 * Errors: PE_EINVAL. */
pe_status pe_gae(const float* reward, const float* value, const uint8_t* done,
                 const float* last_value, int32_t T, int32_t E, float gamma, float lam,
                 float* adv, float* ret, void* stream);

/* PPO update over n_samples = T*E rollout samples (Sec. 4.2; SB3 loss):
 * for each epoch a Feistel permutation of [0, n) keyed by
 * Philox(key = seed, ctr = (epoch, 0, iteration, 3)); each minibatch
 * normalises its advantages, forms the clipped surrogate, value loss and
 * entropy bonus, clips the global gradient norm and takes one Adam step.
 *  params, adam_m, adam_v: [P] fp32, updated in place.
 *  adam_t: Adam steps taken before this call (host value).
 *  obs [n][D] (dtype of the net), act, logp_old, adv, ret: rollout/GAE buffers.
 *  stats: [8] fp32 out: mean pg loss, value loss, entropy, approx KL,
 *         clip fraction, total loss; last pre-clip gradient norm; step count.
 *  workspace: >= pe_ppo_workspace_bytes(...) bytes of device memory, 256-byte
 *  aligned; obs 16-byte aligned (rows are read as 16-byte vectors).
 * BF16 networks: the forward pass rounds the weights (not the biases) of the
 * fp32 masters to bf16 once per minibatch; the head gradient and the hidden
 * pre-activation gradients enter the backward products as bf16 with fp32
 * accumulation; Adam updates the fp32 masters.  stats[7] = -1 if a bounded
 * wait of the tensor-core forward timed out.
 * Errors: PE_EINVAL (unsupported network, sizes, small workspace), PE_ECUDA. */
int64_t pe_ppo_workspace_bytes(const pe_net* net, const pe_ppo_config* cfg, int64_t n_samples);
pe_status pe_ppo_update(const pe_net* net, float* params, float* adam_m, float* adam_v,
                        int64_t adam_t, const void* obs, const uint8_t* act,
                        const float* logp_old, const float* adv, const float* ret,
                        int64_t n_samples, const pe_ppo_config* cfg, float* stats,
                        void* workspace, int64_t workspace_bytes, void* stream);

/* Fleet window accounting (Sec. 7 window analysis, Sec. 8 fleet
 * composition).  Composition n starts job j at offset o[n][j] (a job's GPUs
 * share it; traces tile circularly with period L):
 *   P_n(t) = sum_g q_g((t + o[n][job(g)]) mod L),  t in [0, H)
 *   S_w(t) = sum_{tau = t-w+1}^{t} P_n(tau)         t in [w-1, H)
 *   counts[n][i] = #{t : S_w(t) > budget_q * w},  peaks[n][i] = max_t S_w(t)  (0 if H < w)
 * with q_g = rint(64 * trace) in 1/64 W.
 *  traces: [G][L] fp32 watts; job_of_gpu: [G] in [0, J); offsets: [N][J] in [0, L)
 *  (all device memory); windows: [W] HOST array, W in [1, 4], each w in [1, 992];
 *  counts, peaks: [N][W] int32 (device).
 *  workspace: pe_fleet_workspace_bytes(J, L, H) bytes.  For J <= 8 that size
 *  holds four copies of the per-job prefix sums, each shifted by one sample,
 *  so that the counts use 16-byte loads; a smaller workspace, down to the one
 *  copy of J * (L + H + 128) words plus 1 KiB, gives the same results through
 *  4-byte loads.
 * The call validates the traces on the device and waits for that check
 * (one small device-to-host read on `stream`) before launching the counts.
 * Errors: PE_EINVAL (sizes, pointers, job map or offsets out of range),
 * PE_EOVERFLOW (a sample that is not finite or negative, or a composed
 * window sum or budget_q * w that could exceed int32), PE_ECUDA. */
int64_t pe_fleet_workspace_bytes(int32_t J, int32_t L, int32_t H);
pe_status pe_fleet_windows(const float* traces, int32_t G, int32_t L, const int32_t* job_of_gpu,
                           int32_t J, const int32_t* offsets, int64_t N, int32_t H,
                           const int32_t* windows, int32_t W, int64_t budget_q,
                           int32_t* counts, int32_t* peaks, void* workspace,
                           int64_t workspace_bytes, void* stream);

/* Phase-staggered fleet schedule (Sec. 8, Table 9 "Phase-staggered"): a
 * greedy scheduler places the jobs one at a time in index order 0..J-1.  Job
 * j takes the start offset o from the grid {0, stride, 2 stride, ...} below L
 * that minimises the peak w-sample window sum of the partial fleet of jobs
 * 0..j (jobs 0..j-1 at their chosen offsets; composition and windows as in
 * pe_fleet_windows, t in [w-1, H)); equal peaks go to the lowest offset.
 *  traces [G][L] fp32 watts, job_of_gpu [G] in [0, J) (device memory);
 *  w in [1, 992] (60 = the 30 s window); stride >= 1 (1 = every offset).
 *  offsets: [J] int32 out, the chosen start offsets; peaks: [J] int32 out,
 *  the partial fleet's peak window sum (1/64 W x samples) once job j is
 *  placed (both device memory).
 *  workspace: >= pe_fleet_stagger_workspace_bytes(J, L, H, stride) bytes.
 * Like pe_fleet_windows, the call waits for the device-side trace check
 * before the J stages; the stages themselves run without host round trips.
 * Errors: PE_EINVAL (sizes, pointers, job map), PE_EOVERFLOW (bad sample or
 * an int32 window sum out of range), PE_ECUDA. */
int64_t pe_fleet_stagger_workspace_bytes(int32_t J, int32_t L, int32_t H, int32_t stride);
pe_status pe_fleet_stagger(const float* traces, int32_t G, int32_t L, const int32_t* job_of_gpu,
                           int32_t J, int32_t H, int32_t w, int32_t stride, int32_t* offsets,
                           int32_t* peaks, void* workspace, int64_t workspace_bytes, void* stream);

/* pe_fleet_windows for callers that cannot allocate device memory -- code
 * inside a host process whose device memory belongs to another allocator
 * (a framework's caching allocator, a service with a fixed memory budget),
 * or a control loop that must not add allocations to its timeline.
 * The paper has no counterpart: this is a deployment convenience.
 * Same arguments and results as pe_fleet_windows without the workspace: the
 * scratch is one file-scope device array of PE_FLEET_NOALLOC_SCRATCH_BYTES
 * (4 MiB); the 16-byte path runs when its four prefix copies fit.  Requests
 * whose single copy (about J * (L + H + 128) * 4 bytes) does not fit return
 * PE_EINVAL with that limit in the message, before any launch.
 * Set-up: the first call on a device, with that device current, looks up
 * the array's device address (cudaGetSymbolAddress).  Under lazy module
 * loading, the CUDA default, that lookup is also when the driver loads the
 * array's module and reserves the 4 MiB on the device, once; the device
 * then holds it until the process exits.  Make that first call at set-up
 * time, before any stream capture.  The address is looked up again only if
 * the device's context changed (after cudaDeviceReset).
 * The calls allocate nothing (no cudaMalloc, no cudaFree, no allocating
 * library routine).  Like pe_fleet_windows, every call waits on `stream`
 * for the device-side validation read before it launches the counts, so it
 * returns only once the preparation kernels have finished.  All calls share
 * the array, which keeps the last call's contents: calls that overlap on the
 * GPU (other streams, other host threads) race. */
#define PE_FLEET_NOALLOC_SCRATCH_BYTES (4 * 1024 * 1024)
pe_status pe_fleet_windows_noalloc(const float* traces, int32_t G, int32_t L,
                                   const int32_t* job_of_gpu, int32_t J, const int32_t* offsets,
                                   int64_t N, int32_t H, const int32_t* windows, int32_t W,
                                   int64_t budget_q, int32_t* counts, int32_t* peaks,
                                   void* stream);

/* Launch profiling (off by default).  When enabled, every kernel launch of
 * the library is bracketed by a pair of CUDA events recorded on the launch's
 * stream; pe_profile_read waits for the recorded events of one kernel kind,
 * returns the summed device time and the launch count, and clears that kind.
 * Kinds: */
#define PE_PROF_ROLLOUT 0
#define PE_PROF_VALUE 1
#define PE_PROF_GAE 2
#define PE_PROF_PPO_GRAD 3
#define PE_PROF_PPO_REDUCE 4
#define PE_PROF_PPO_ADAM 5
#define PE_PROF_PPO_OTHER 6
#define PE_PROF_FLEET_PREP 7
#define PE_PROF_FLEET_WINDOWS 8
#define PE_PROF_MLP_POLICY 9  /* tensor-core policy network launches (bf16 rollout) */
#define PE_PROF_MLP_VALUE 10  /* tensor-core value network launches */
#define PE_PROF_KINDS 11
pe_status pe_profile_enable(int32_t on);
pe_status pe_profile_read(int32_t kind, double* total_ms, int64_t* launches);
const char* pe_profile_kind_name(int32_t kind);

/* Measured roofs for the roofline fractions of the kernels that neither HBM
 * nor the tensor cores bound (measurement support; the paper has no
 * counterpart).  One warm-up and one timed launch of a throughput loop over
 * 8 CTAs of 256 threads per SM, timed with CUDA events on `stream`; the call
 * waits for the result.
 *  kind 0 (PE_ROOF_FFMA):  scalar fp32 FMA, units = FLOPs (2 per FMA), reps = loop trips;
 *  kind 1 (PE_ROOF_FFMA2): packed two-lane fp32 FMA, units = FLOPs;
 *  kind 2 (PE_ROOF_IADD):  int32 adds, units = adds;
 *  kind 3 (PE_ROOF_L2):    16-byte loads cached in L2 only over buf[4096, bytes),
 *                          reps passes, units = bytes (pick a buffer L2 holds).
 *  buf: >= 64 KiB of device memory, 16-byte aligned (its first 4 KiB are
 *  scratch words the loops keep alive and never write in practice).
 *  ms: host out, device time of the timed launch; units: host out.
 * Errors: PE_EINVAL (kind, sizes, alignment), PE_ECUDA. */
#define PE_ROOF_FFMA 0
#define PE_ROOF_FFMA2 1
#define PE_ROOF_IADD 2
#define PE_ROOF_L2 3
pe_status pe_roof_probe(int32_t kind, void* buf, int64_t bytes, int64_t reps, double* ms, double* units,
                        void* stream);

/* Synchronise `stream`, then report device-side errors of earlier launches:
 * PE_ETIMEOUT if a bounded tensor-core wait gave up (the flag is cleared). */
pe_status pe_device_check(void* stream);

/* Message for the last non-OK status on this thread ("" if none). */
const char* pe_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* PE_H */
