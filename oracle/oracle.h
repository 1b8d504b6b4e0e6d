/*
 * CPU oracle for the batched PPO power-controller path -- TEST INFRASTRUCTURE.
 *
 * A plain, slow, single-threaded C99 statement of what the GPU path computes,
 * written from the paper ("Cutting AI Datacenter Energy with Reinforcement
 * Learning", Sec. 4.1-4.5, Eqs. 1-7, Sec. 7-8).  It shares no code, header,
 * table or constant generator with the CUDA library; only the seeded input
 * generators (traces, initial weights, offsets) feed both.  Only the test
 * suite, the smoke check and the benchmark's CPU-baseline leg may load it.
 *
 * Precision: fp64 wherever the paper fixes none (network, sampler, GAE, PPO,
 * rewards).  Three decisions are taken in fp32 exactly as the device does,
 * because they decide integers or define the observation type: the
 * multiplicative actuator (one fp32 multiply, then rint to 1/64 W), the
 * observation features (fp32 quotient of two exact integers, the float32
 * observation space of a Gymnasium Box) and, for bf16 networks, the bf16
 * rounding points of the forward pass.
 *
 * Parity status: every function below is pinned by tests under tests/
 * (Philox known answers, brute-force windows, closed-form GAE, finite
 * differences for the PPO gradient, hand-counted violations).
 */
#ifndef PE_ORACLE_H
#define PE_ORACLE_H
#include <stdint.h>

#define OR_MAX_LEVELS 32
#define OR_MAX_CH 4
#define OR_RING 64
#define OR_MAX_FAM 4

enum { OR_ACT_SET_LEVEL = 0, OR_ACT_INCDEC = 1 };
enum { OR_OBS_TINY8 = 0, OR_OBS_7B16 = 1, OR_OBS_OCC32 = 2, OR_OBS_OCC64 = 3 };
enum { OR_REWARD_FIXED = 0, OR_REWARD_LAGRANGE = 1 };
enum { OR_PURPOSE_ACTION = 0, OR_PURPOSE_RESET = 1, OR_PURPOSE_INIT = 2, OR_PURPOSE_PERM = 3 };

typedef struct {
  int32_t n_envs, n_channels, trace_len, n_actions;
  int32_t obs_kind, actuator_kind, n_levels, level_init;
  int32_t g_min, g_max, b_min, b_max, b_init;
  int32_t episode_len, budget_q, scale_phase_mask;
  int32_t reward_kind, reward_window;
  double r_ok, r_viol, bonus_coef;
  float level_scale[OR_MAX_LEVELS][OR_MAX_CH];
  double level_tokens[OR_MAX_LEVELS];
  uint64_t seed;
  /* batch-boundary cadence (Sec. 4.5): samples one step consumes at each
   * level; all zero: one sample per step */
  int32_t level_samples[OR_MAX_LEVELS];
  /* domain randomisation (Sec. 4.2, design G2): n_families trace families;
   * family f has fam_len[f] samples, fam_channels[f] GPUs (<= n_channels)
   * and budget fam_budget_q[f].  The trace buffer is family-major
   * [f][n_channels][fam_len[f]] and the phase buffer [f][fam_len[f]].
   * 0 or 1 family: the single trace of trace_len / n_channels / budget_q. */
  int32_t n_families;
  int32_t fam_len[OR_MAX_FAM], fam_channels[OR_MAX_FAM], fam_budget_q[OR_MAX_FAM];
} or_env_cfg;

typedef struct {
  int32_t pos;         /* next trace position to consume */
  int32_t k;           /* steps taken in the current episode */
  int32_t level;       /* actuator level (group size G for the inc/dec actuator) */
  int32_t prev_level;  /* level in effect during the previous step */
  int32_t b;           /* batch size (inc/dec actuator) */
  int32_t til;         /* steps since the last level change */
  uint8_t ring[OR_RING];           /* level used for the sample at position p, at p & 63 */
  int32_t s_short[OR_MAX_CH];      /* 10 s window sum (20 samples), per channel */
  int32_t s_long[OR_MAX_CH];       /* 30 s window sum (60 samples), per channel */
  int32_t fam;                     /* trace family of the current episode */
} or_env_state;

enum { OR_RULE_RANDOM = 1, OR_RULE_THRESHOLD = 2, OR_RULE_HYSTERESIS = 3 };

typedef struct {
  int32_t kind;
  int32_t hi_q, lo_q;                      /* threshold rule, 1/64 W */
  int32_t drop30_q, climb30_q, climb10_q;  /* hysteresis rule, 1/64 W (window means) */
} or_rule;

typedef struct {
  int32_t epochs, minibatch;
  double lr, clip, vf_coef, ent_coef, max_grad_norm, beta1, beta2, eps;
} or_ppo_cfg;

#ifdef __cplusplus
extern "C" {
#endif

void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
uint32_t or_feistel_index(uint64_t n, const uint32_t keys[4], uint64_t i);
void or_perm_keys(uint64_t seed, uint32_t epoch, uint32_t iteration, uint32_t keys[4]);
double or_bf16_round(double x);
int32_t or_env_state_size(void);
float or_actuator_scale(const or_env_cfg* cfg, int32_t level, int32_t c);
int32_t or_env_init(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                    const int32_t* env_ids, int32_t n, or_env_state* states);
void or_env_obs(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                const or_env_state* st, float* obs);
void or_mlp_forward(int32_t D, int32_t H, int32_t A, int32_t bf16, const float* params,
                    int64_t n, const float* obs, double* logits, double* value);
int32_t or_rollout(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                   const float* params, int32_t hidden, int32_t bf16,
                   const int32_t* env_ids, int32_t n, or_env_state* states,
                   int32_t T, uint32_t iteration, double lambda, int32_t deterministic,
                   const uint8_t* forced, float* obs, float* obs_last, uint8_t* act_own,
                   double* logp_taken, double* reward, uint8_t* done, int32_t* viol,
                   double* tokens, double* excess, int64_t* energy_q, int64_t* samples,
                   int32_t* qout);
int32_t or_env_set_offsets(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                           const int32_t* offsets, int32_t n, or_env_state* states);
int32_t or_rollout_rule(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                        const or_rule* rule, const int32_t* env_ids, int32_t n,
                        or_env_state* states, int32_t T, uint32_t iteration, double lambda,
                        uint8_t* act, double* reward, uint8_t* done, int32_t* viol,
                        double* tokens, double* excess, int64_t* energy_q, int64_t* samples,
                        int32_t* qout);
double or_dual_ascent(const int32_t* viol, int32_t E, int64_t steps, int32_t window, int32_t additive,
                      double lambda, double target, double eta, double lo, double hi, double* rate);
void or_gae(int32_t T, int32_t E, const float* r, const float* v, const uint8_t* done,
            const float* last_v, double gamma, double lam, double* adv, double* ret);
double or_ppo_minibatch_grad(int32_t D, int32_t H, int32_t A, const double* params, int64_t M,
                             const float* obs, const uint8_t* act, const float* logp_old,
                             const float* adv, const float* ret, double clip, double vf_coef,
                             double ent_coef, double* grad, double* stats);
double or_ppo_minibatch_grad_ex(int32_t D, int32_t H, int32_t A, int32_t bf16, const double* params,
                                int64_t M, const float* obs, const uint8_t* act,
                                const float* logp_old, const float* adv, const float* ret,
                                double clip, double vf_coef, double ent_coef, double* grad,
                                double* stats);
int64_t or_ppo_update_ex(int32_t D, int32_t H, int32_t A, int32_t bf16, double* params,
                         double* adam_m, double* adam_v, int64_t adam_t, int64_t N,
                         const float* obs, const uint8_t* act, const float* logp_old,
                         const float* adv, const float* ret, const or_ppo_cfg* cfg, uint64_t seed,
                         uint32_t iteration, int64_t max_steps, double* stats);
int64_t or_ppo_update(int32_t D, int32_t H, int32_t A, double* params, double* adam_m,
                      double* adam_v, int64_t adam_t, int64_t N, const float* obs,
                      const uint8_t* act, const float* logp_old, const float* adv,
                      const float* ret, const or_ppo_cfg* cfg, uint64_t seed,
                      uint32_t iteration, int64_t max_steps, double* stats);
int32_t or_fleet_windows(int32_t G, int32_t L, const float* traces, const int32_t* job_of_gpu,
                         int32_t J, const int32_t* offsets, int64_t N, int32_t H,
                         const int32_t* windows, int32_t W, int64_t budget_q,
                         int32_t* counts, int32_t* peaks);
int32_t or_fleet_stagger(int32_t G, int32_t L, const float* traces, const int32_t* job_of_gpu,
                         int32_t J, int32_t H, int32_t w, int32_t stride, int32_t* offsets,
                         int32_t* peaks);

#ifdef __cplusplus
}
#endif
#endif
