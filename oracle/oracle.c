/*
 * CPU oracle for the batched PPO power-controller path -- TEST INFRASTRUCTURE
 * (see oracle.h).  Plain single-threaded C99, compiled with
 * -O2 -ffp-contract=off so that no multiply-add is fused behind our back.
 *
 * Readings of the paper that this file fixes (all listed with their reasons
 * in the design notes): one environment step consumes one half-second
 * sample; windows are trailing and inclusive of the newest sample
 * (w = 1, 20, 60, 600 samples for 0.5 s, 10 s, 30 s, 5 min); power is held
 * in 1/64 W integers so that window sums and violation counts are exact.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
 * easy as 1, 2, 3", SC'11): ten rounds of two 32x32->64 multiplies on a
 * 128-bit counter under a 64-bit key that is bumped by the Weyl constants
 * between rounds.
 * ---------------------------------------------------------------------- */
#define OR_PHILOX_M0 0xD2511F53u
#define OR_PHILOX_M1 0xCD9E8D57u
#define OR_PHILOX_W0 0x9E3779B9u
#define OR_PHILOX_W1 0xBB67AE85u

void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += OR_PHILOX_W0;
      k1 += OR_PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)OR_PHILOX_M0 * (uint64_t)c0;
    uint64_t p1 = (uint64_t)OR_PHILOX_M1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

static void draw_4(uint64_t seed, uint32_t a, uint32_t b, uint32_t c, uint32_t d, uint32_t out[4]) {
  uint32_t ctr[4] = {a, b, c, d};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  or_philox4x32_10(ctr, key, out);
}

static uint32_t draw_u32(uint64_t seed, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  uint32_t out[4];
  draw_4(seed, a, b, c, d, out);
  return out[0];
}

/* ------------------------------------------------------------------------
 * Minibatch order: a 4-round balanced Feistel network over the smallest
 * even-bit domain that holds n indices, with cycle walking back into
 * [0, n) (Black & Rogaway, "Ciphers with arbitrary finite domains", 2002).
 * The round function is the "lowbias32" integer hash (C. Wellons, 2018).
 * ---------------------------------------------------------------------- */
static uint32_t lowbias32(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7feb352du;
  x ^= x >> 15;
  x *= 0x846ca68bu;
  x ^= x >> 16;
  return x;
}

static uint64_t feistel_once(uint64_t x, int half, const uint32_t keys[4]) {
  uint64_t mask = (1ull << half) - 1ull;
  uint64_t L = x >> half, R = x & mask;
  for (int r = 0; r < 4; ++r) {
    uint64_t F = (uint64_t)lowbias32((uint32_t)R ^ keys[r]) & mask;
    uint64_t nL = R, nR = L ^ F;
    L = nL;
    R = nR;
  }
  return (L << half) | R;
}

uint32_t or_feistel_index(uint64_t n, const uint32_t keys[4], uint64_t i) {
  int bits = 2;
  while ((1ull << bits) < n) ++bits;
  if (bits & 1) ++bits;
  int half = bits / 2;
  uint64_t y = feistel_once(i, half, keys);
  while (y >= n) y = feistel_once(y, half, keys);
  return (uint32_t)y;
}

void or_perm_keys(uint64_t seed, uint32_t epoch, uint32_t iteration, uint32_t keys[4]) {
  uint32_t ctr[4] = {epoch, 0u, iteration, (uint32_t)OR_PURPOSE_PERM};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  or_philox4x32_10(ctr, key, keys);
}

/* bf16 = 8 significant bits; round-to-nearest-even of a double */
double or_bf16_round(double x) {
  if (x == 0.0 || !isfinite(x)) return x;
  int e;
  double m = frexp(x, &e);
  return ldexp(nearbyint(ldexp(m, 8)), e - 8);
}

/* ------------------------------------------------------------------------
 * Environment (Sec. 4.1 trace replay with a multiplicative actuator; the
 * Sec. 4.5 windows of Eq. 1, violations of Eq. 2, excess of Eq. 3 and the
 * Lagrangian reward of Eq. 6).
 * ---------------------------------------------------------------------- */
#define OR_W_SHORT 20 /* 10 s at 0.5 s per sample */
#define OR_W_LONG 60  /* 30 s */
#define OR_DT 0.5

int32_t or_env_state_size(void) { return (int32_t)sizeof(or_env_state); }

/* Sec. 4.1: power = trace * (0.8 + 0.2 G / G_max) for the group-size
 * actuator; a per-level table for the level actuators (Sec. 4.5, Table 4). */
float or_actuator_scale(const or_env_cfg* cfg, int32_t level, int32_t c) {
  if (cfg->actuator_kind == OR_ACT_INCDEC)
    return (float)(0.8 + 0.2 * (double)level / (double)cfg->g_max);
  return cfg->level_scale[level][c];
}

/* actuated power of channel c at trace position pos under `level`, in 1/64 W */
static int32_t q_of(const or_env_cfg* cfg, const float* trace, const uint8_t* phase, int32_t c,
                    int32_t pos, int32_t level) {
  float x = trace[(int64_t)c * cfg->trace_len + pos];
  float s = ((cfg->scale_phase_mask >> phase[pos]) & 1) ? or_actuator_scale(cfg, level, c) : 1.0f;
  float p = x * s;
  return (int32_t)rintf(p * 64.0f);
}

/* channel c, i samples before the newest consumed one */
static int32_t q_back(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                      const or_env_state* st, int32_t c, int32_t i) {
  int32_t pos = st->pos - 1 - i;
  return q_of(cfg, trace, phase, c, pos, st->ring[pos & (OR_RING - 1)]);
}

static int32_t qc_back(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                       const or_env_state* st, int32_t i) {
  int32_t s = 0;
  for (int32_t c = 0; c < cfg->n_channels; ++c) s += q_back(cfg, trace, phase, st, c, i);
  return s;
}

/* Batch-boundary cadence (Sec. 4.5): with a level table, one step is one
 * generation batch and consumes level_samples[level] samples; without one,
 * a step is one sample. */
static int32_t cadence_on(const or_env_cfg* cfg) {
  for (int32_t l = 0; l < OR_MAX_LEVELS; ++l)
    if (cfg->level_samples[l] > 0) return 1;
  return 0;
}

static int32_t step_samples(const or_env_cfg* cfg, int32_t level) {
  return cfg->level_samples[level] > 0 ? cfg->level_samples[level] : 1;
}

static int32_t max_step_samples(const or_env_cfg* cfg) {
  int32_t m = 1;
  for (int32_t l = 0; l < OR_MAX_LEVELS; ++l)
    if (cfg->level_samples[l] > m) m = cfg->level_samples[l];
  return m;
}

/* samples one episode may span */
static int32_t episode_span(const or_env_cfg* cfg) { return cfg->episode_len * max_step_samples(cfg); }

/* The env as one trace family sees it (domain randomisation, Sec. 4.2 G2):
 * the family's length, channel count and budget, and its slices of the
 * family-major trace and phase buffers.  One family: the env itself. */
static void fam_view(const or_env_cfg* cfg, const float* trace, const uint8_t* phase, int32_t f,
                     or_env_cfg* cf, const float** tr, const uint8_t** ph) {
  *cf = *cfg;
  *tr = trace;
  *ph = phase;
  if (cfg->n_families <= 1) return;
  int64_t to = 0, po = 0;
  for (int32_t g = 0; g < f; ++g) {
    to += (int64_t)cfg->n_channels * cfg->fam_len[g];
    po += cfg->fam_len[g];
  }
  cf->trace_len = cfg->fam_len[f];
  cf->n_channels = cfg->fam_channels[f];
  cf->budget_q = cfg->fam_budget_q[f];
  *tr = trace + to;
  *ph = phase + po;
}

/* Sec. 4.1: episodes start at a randomised offset; the history window is
 * warm-started at the default setting (Sec. 4.5 warm start). */
static void env_reset_at(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                         or_env_state* st, int32_t o) {
  st->pos = o;
  st->k = 0;
  st->level = cfg->level_init;
  st->prev_level = cfg->level_init;
  st->b = cfg->b_init;
  st->til = 0;
  for (int i = 0; i < OR_RING; ++i) st->ring[i] = (uint8_t)cfg->level_init;
  for (int32_t c = 0; c < OR_MAX_CH; ++c) {
    st->s_short[c] = 0;
    st->s_long[c] = 0;
  }
  for (int32_t c = 0; c < cfg->n_channels; ++c) {
    for (int32_t i = 1; i <= OR_W_LONG; ++i) {
      int32_t q = q_of(cfg, trace, phase, c, o - i, cfg->level_init);
      st->s_long[c] += q;
      if (i <= OR_W_SHORT) st->s_short[c] += q;
    }
  }
}

/* word 1 of the episode draw picks the trace family (G2 domain
 * randomisation), word 0 the offset inside that family's trace */
static void env_reset(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                      or_env_state* st, uint32_t e, uint32_t t, uint32_t it, uint32_t purpose) {
  uint32_t w[4];
  draw_4(cfg->seed, e, t, it, purpose, w);
  const int32_t f = cfg->n_families > 1 ? (int32_t)(((uint64_t)w[1] * (uint64_t)cfg->n_families) >> 32) : 0;
  or_env_cfg cf;
  const float* tr;
  const uint8_t* ph;
  fam_view(cfg, trace, phase, f, &cf, &tr, &ph);
  uint32_t span = (uint32_t)(cf.trace_len - episode_span(&cf) - OR_W_LONG + 1);
  env_reset_at(&cf, tr, ph, st, OR_W_LONG + (int32_t)(((uint64_t)w[0] * (uint64_t)span) >> 32));
  st->fam = f;
}

/* Episodes that start at given offsets (the evaluation replay of Sec. 4.4
 * walks the trace in consecutive 500-step episodes); each offset must leave
 * the 60-sample history and one full episode inside the trace. */
int32_t or_env_set_offsets(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                           const int32_t* offsets, int32_t n, or_env_state* states) {
  for (int32_t i = 0; i < n; ++i) {
    or_env_cfg cf;
    const float* tr;
    const uint8_t* ph;
    fam_view(cfg, trace, phase, states[i].fam, &cf, &tr, &ph);
    if (offsets[i] < OR_W_LONG || offsets[i] > cf.trace_len - episode_span(&cf)) return 1;
  }
  for (int32_t i = 0; i < n; ++i) {
    or_env_cfg cf;
    const float* tr;
    const uint8_t* ph;
    fam_view(cfg, trace, phase, states[i].fam, &cf, &tr, &ph);
    env_reset_at(&cf, tr, ph, &states[i], offsets[i]);
  }
  return 0;
}

int32_t or_env_init(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                    const int32_t* env_ids, int32_t n, or_env_state* states) {
  if (cfg->n_families > 1) {
    for (int32_t f = 0; f < cfg->n_families; ++f)
      if (cfg->fam_len[f] < episode_span(cfg) + OR_W_LONG) return 1;
  } else if (cfg->trace_len < episode_span(cfg) + OR_W_LONG) {
    return 1;
  }
  for (int32_t i = 0; i < n; ++i)
    env_reset(cfg, trace, phase, &states[i], (uint32_t)env_ids[i], 0u, 0u, OR_PURPOSE_INIT);
  return 0;
}

static float ratio(int64_t num, int64_t den) { return (float)num / (float)den; }

/* Observation vectors: Sec. 4.1 (TINY8), the 7B state of the workload
 * (last 8 samples, 30 s mean, budget slack), Eq. 5 (OCC32 / OCC64 core),
 * all normalised by the budget B. */
static void env_obs_view(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                         const or_env_state* st, float* f) {
  const int64_t B = cfg->budget_q;
  const int32_t C = cfg->n_channels;
  int64_t S20 = 0, S60 = 0;
  for (int32_t c = 0; c < C; ++c) {
    S20 += st->s_short[c];
    S60 += st->s_long[c];
  }
  int32_t Q0 = qc_back(cfg, trace, phase, st, 0);
  switch (cfg->obs_kind) {
    case OR_OBS_TINY8:
      for (int i = 0; i < 5; ++i) f[i] = ratio(qc_back(cfg, trace, phase, st, 4 - i), B);
      f[5] = ratio(B - Q0, B);
      f[6] = (float)phase[st->pos - 1];
      f[7] = ratio(st->level, cfg->n_levels - 1);
      break;
    case OR_OBS_7B16:
      for (int i = 0; i < 8; ++i) f[i] = ratio(qc_back(cfg, trace, phase, st, 7 - i), B);
      f[8] = ratio(S60, OR_W_LONG * B);
      f[9] = ratio(OR_W_LONG * B - S60, OR_W_LONG * B);
      f[10] = (float)phase[st->pos - 1];
      f[11] = ratio(st->level - cfg->g_min, cfg->g_max - cfg->g_min);
      f[12] = ratio(st->b - cfg->b_min, cfg->b_max - cfg->b_min);
      f[13] = ratio(S20, OR_W_SHORT * B);
      f[14] = ratio((int64_t)Q0 - qc_back(cfg, trace, phase, st, 10), B);
      f[15] = 0.0f;
      break;
    case OR_OBS_OCC32:
    case OR_OBS_OCC64: {
      /* d / 20 s: per-sample steps use the time since the last level change,
       * the batch cadence the duration of the batch just completed */
      float d = cadence_on(cfg) ? ratio(step_samples(cfg, st->level), 40) : ratio(st->til, 40);
      f[0] = ratio(Q0, B);
      f[1] = ratio(S20, OR_W_SHORT * B);
      f[2] = ratio(S60, OR_W_LONG * B);
      f[3] = ratio(OR_W_LONG * B - S60, OR_W_LONG * B);
      f[4] = ratio((int64_t)Q0 - qc_back(cfg, trace, phase, st, 10), B);
      f[5] = ratio(st->level + 1, cfg->n_levels);
      f[6] = ratio(st->prev_level + 1, cfg->n_levels);
      f[7] = d < 1.0f ? d : 1.0f;
      if (cfg->obs_kind == OR_OBS_OCC32) {
        for (int c = 0; c < 4; ++c) {
          for (int i = 0; i < 4; ++i)
            f[8 + 4 * c + i] =
                c < C ? ratio((int64_t)C * q_back(cfg, trace, phase, st, c, 3 - i), B) : 0.0f;
          f[24 + c] = c < C ? ratio((int64_t)C * st->s_long[c], OR_W_LONG * B) : 0.0f;
          f[28 + c] = 0.0f;
        }
      } else {
        for (int c = 0; c < 4; ++c) {
          for (int i = 0; i < 12; ++i)
            f[8 + 12 * c + i] =
                c < C ? ratio((int64_t)C * q_back(cfg, trace, phase, st, c, 11 - i), B) : 0.0f;
          f[56 + c] = c < C ? ratio((int64_t)C * st->s_short[c], OR_W_SHORT * B) : 0.0f;
          f[60 + c] = c < C ? ratio((int64_t)C * st->s_long[c], OR_W_LONG * B) : 0.0f;
        }
      }
      break;
    }
    default:
      break;
  }
}

void or_env_obs(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                const or_env_state* st, float* f) {
  or_env_cfg cf;
  const float* tr;
  const uint8_t* ph;
  fam_view(cfg, trace, phase, st->fam, &cf, &tr, &ph);
  env_obs_view(&cf, tr, ph, st, f);
}

static double token_rate(const or_env_cfg* cfg, int32_t level, int32_t b) {
  if (cfg->actuator_kind == OR_ACT_INCDEC)
    return cfg->level_tokens[level] * (double)b / (double)cfg->b_init;
  return cfg->level_tokens[level];
}

static double token_rate_max(const or_env_cfg* cfg) {
  double m = 0.0;
  int32_t lo = cfg->actuator_kind == OR_ACT_INCDEC ? cfg->g_min : 0;
  int32_t hi = cfg->actuator_kind == OR_ACT_INCDEC ? cfg->g_max : cfg->n_levels - 1;
  int32_t b = cfg->actuator_kind == OR_ACT_INCDEC ? cfg->b_max : cfg->b_init;
  for (int32_t l = lo; l <= hi; ++l) {
    double r = token_rate(cfg, l, b);
    if (r > m) m = r;
  }
  return m;
}

typedef struct {
  double reward, tokens, excess;
  int32_t v1, v60, done, samples;
  int64_t q;
} or_step_out;

/* One environment step: apply the action (Sec. 4.1 action set, G >= 3 floor
 * of Sec. 4.2 via g_min), consume one half-second sample, update the
 * windows (Eq. 1), score violation (Eq. 2), excess (Eq. 3) and reward
 * (G1 design of Sec. 4.2, or Eq. 6). */
static or_step_out env_step(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                            or_env_state* st, int32_t a, double lambda) {
  or_step_out o;
  int32_t new_level = st->level;
  if (cfg->actuator_kind == OR_ACT_INCDEC) {
    switch (a) {
      case 1: if (new_level > cfg->g_min) --new_level; break;
      case 2: if (new_level < cfg->g_max) ++new_level; break;
      case 3: if (st->b > cfg->b_min) --st->b; break;
      case 4: if (st->b < cfg->b_max) ++st->b; break;
      default: break;
    }
  } else {
    new_level = a;
  }
  st->til = (new_level != st->level) ? 0 : st->til + 1;
  st->prev_level = st->level;
  st->level = new_level;

  /* consume the step's samples: windows (Eq. 1), violations (Eq. 2) and
   * excess (Eq. 3) per sample; tokens and excess summed over the step; the
   * Eq. 6 peak term takes the step's largest 30 s excess */
  const int64_t B = cfg->budget_q;
  const int32_t ns = step_samples(cfg, new_level);
  const double rate = token_rate(cfg, new_level, st->b);
  o.q = 0;
  o.v1 = 0;
  o.v60 = 0;
  o.tokens = 0.0;
  o.excess = 0.0;
  double peak_w = 0.0, fixed = 0.0;
  for (int32_t i = 0; i < ns; ++i) {
    const int32_t p = st->pos;
    st->ring[p & (OR_RING - 1)] = (uint8_t)new_level;
    int32_t Q = 0;
    int64_t S60 = 0;
    for (int32_t c = 0; c < cfg->n_channels; ++c) {
      int32_t qin = q_of(cfg, trace, phase, c, p, new_level);
      int32_t p20 = p - OR_W_SHORT, p60 = p - OR_W_LONG;
      int32_t q20 = q_of(cfg, trace, phase, c, p20, st->ring[p20 & (OR_RING - 1)]);
      int32_t q60 = q_of(cfg, trace, phase, c, p60, st->ring[p60 & (OR_RING - 1)]);
      st->s_short[c] += qin - q20;
      st->s_long[c] += qin - q60;
      Q += qin;
      S60 += st->s_long[c];
    }
    const int32_t v1 = Q > B, v60 = S60 > (int64_t)OR_W_LONG * B;
    const double excess_w = v60 ? (double)(S60 - (int64_t)OR_W_LONG * B) / (64.0 * OR_W_LONG) : 0.0;
    const double tok = phase[p] == 0 ? rate : 0.0;
    o.q += Q;
    o.v1 += v1;
    o.v60 += v60;
    o.excess += excess_w * OR_DT;
    o.tokens += tok;
    if (excess_w > peak_w) peak_w = excess_w;
    if (cfg->reward_kind != OR_REWARD_LAGRANGE) {
      int32_t viol = cfg->reward_window == 1 ? v1 : v60;
      fixed += (viol ? cfg->r_viol : cfg->r_ok) + cfg->bonus_coef * rate / token_rate_max(cfg);
    }
    st->pos = p + 1;
  }
  o.samples = ns;
  if (cfg->reward_kind == OR_REWARD_LAGRANGE)
    o.reward = o.tokens / 1000.0 - lambda * o.excess - 2.0 * lambda * peak_w;
  else
    o.reward = fixed;
  st->k += 1;
  o.done = st->k == cfg->episode_len;
  return o;
}

/* ------------------------------------------------------------------------
 * Policy / value networks: SB3's default MLP actor-critic (Sec. 4.2), two
 * separate tanh MLPs D -> H -> H -> {A logits, 1 value}.  Canonical flat
 * layout (row-major W[out][in]):
 *   policy: W1[H][D] b1[H] W2[H][H] b2[H] W3[A][H] b3[A]
 *   value : V1[H][D] c1[H] V2[H][H] c2[H] V3[1][H] c3[1]
 * ---------------------------------------------------------------------- */
typedef struct {
  int64_t w1, b1, w2, b2, w3, b3, v1, c1, v2, c2, v3, c3, total;
} or_layout;

static or_layout layout_of(int32_t D, int32_t H, int32_t A) {
  or_layout L;
  int64_t o = 0;
  L.w1 = o; o += (int64_t)H * D;
  L.b1 = o; o += H;
  L.w2 = o; o += (int64_t)H * H;
  L.b2 = o; o += H;
  L.w3 = o; o += (int64_t)A * H;
  L.b3 = o; o += A;
  L.v1 = o; o += (int64_t)H * D;
  L.c1 = o; o += H;
  L.v2 = o; o += (int64_t)H * H;
  L.c2 = o; o += H;
  L.v3 = o; o += H;
  L.c3 = o; o += 1;
  L.total = o;
  return L;
}

/* fp32 parameters -> fp64, with the weight matrices rounded to bf16 for a
 * bf16 network (biases stay fp32) */
static double* params_to_double(int32_t D, int32_t H, int32_t A, const float* p, int32_t bf16) {
  or_layout L = layout_of(D, H, A);
  double* d = (double*)malloc(sizeof(double) * (size_t)L.total);
  for (int64_t i = 0; i < L.total; ++i) d[i] = (double)p[i];
  if (bf16) {
    int64_t mats[6][2] = {{L.w1, (int64_t)H * D}, {L.w2, (int64_t)H * H}, {L.w3, (int64_t)A * H},
                          {L.v1, (int64_t)H * D}, {L.v2, (int64_t)H * H}, {L.v3, (int64_t)H}};
    for (int m = 0; m < 6; ++m)
      for (int64_t i = 0; i < mats[m][1]; ++i) d[mats[m][0] + i] = or_bf16_round(d[mats[m][0] + i]);
  }
  return d;
}

/* y = tanh(W x + b), optionally rounded to bf16 */
static void dense_tanh(int32_t out, int32_t in, const double* W, const double* b, const double* x,
                       double* y, int32_t bf16) {
  for (int32_t o = 0; o < out; ++o) {
    double acc = 0.0;
    for (int32_t i = 0; i < in; ++i) acc += W[(int64_t)o * in + i] * x[i];
    double h = tanh(acc + b[o]);
    y[o] = bf16 ? or_bf16_round(h) : h;
  }
}

static void dense_lin(int32_t out, int32_t in, const double* W, const double* b, const double* x,
                      double* y) {
  for (int32_t o = 0; o < out; ++o) {
    double acc = 0.0;
    for (int32_t i = 0; i < in; ++i) acc += W[(int64_t)o * in + i] * x[i];
    y[o] = acc + b[o];
  }
}

static void policy_fwd(int32_t D, int32_t H, int32_t A, const double* P, const double* x,
                       double* h1, double* h2, double* z, int32_t bf16) {
  or_layout L = layout_of(D, H, A);
  dense_tanh(H, D, P + L.w1, P + L.b1, x, h1, bf16);
  dense_tanh(H, H, P + L.w2, P + L.b2, h1, h2, bf16);
  dense_lin(A, H, P + L.w3, P + L.b3, h2, z);
}

static double value_fwd(int32_t D, int32_t H, int32_t A, const double* P, const double* x,
                        double* g1, double* g2, int32_t bf16) {
  or_layout L = layout_of(D, H, A);
  double v;
  dense_tanh(H, D, P + L.v1, P + L.c1, x, g1, bf16);
  dense_tanh(H, H, P + L.v2, P + L.c2, g1, g2, bf16);
  dense_lin(1, H, P + L.v3, P + L.c3, g2, &v);
  return v;
}

static void obs_to_double(int32_t D, const float* obs, double* x, int32_t bf16) {
  for (int32_t i = 0; i < D; ++i) x[i] = bf16 ? or_bf16_round((double)obs[i]) : (double)obs[i];
}

void or_mlp_forward(int32_t D, int32_t H, int32_t A, int32_t bf16, const float* params,
                    int64_t n, const float* obs, double* logits, double* value) {
  double* P = params_to_double(D, H, A, params, bf16);
  double* x = (double*)malloc(sizeof(double) * (size_t)D);
  double* h1 = (double*)malloc(sizeof(double) * (size_t)H);
  double* h2 = (double*)malloc(sizeof(double) * (size_t)H);
  for (int64_t i = 0; i < n; ++i) {
    obs_to_double(D, obs + i * D, x, bf16);
    if (logits) policy_fwd(D, H, A, P, x, h1, h2, logits + i * A, bf16);
    if (value) value[i] = value_fwd(D, H, A, P, x, h1, h2, bf16);
  }
  free(x); free(h1); free(h2); free(P);
}

/* ------------------------------------------------------------------------
 * Rollout: for each env, T steps of observe -> policy -> sample -> step.
 * The categorical sample is the inverse CDF of softmax(logits) at
 * u = (philox >> 8) * 2^-24, in index order; the deterministic mode is
 * argmax with the lowest index on ties (Sec. 4.4 evaluation protocol).
 * `forced` (optional, [T][n]) replaces the action taken (teacher forcing);
 * act_own always records the oracle's own choice.
 * ---------------------------------------------------------------------- */
int32_t or_rollout(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                   const float* params, int32_t H, int32_t bf16, const int32_t* env_ids,
                   int32_t n, or_env_state* states, int32_t T, uint32_t iteration,
                   double lambda, int32_t deterministic, const uint8_t* forced, float* obs,
                   float* obs_last, uint8_t* act_own, double* logp_taken, double* reward,
                   uint8_t* done, int32_t* viol, double* tokens, double* excess,
                   int64_t* energy_q, int64_t* samples, int32_t* qout) {
  const int32_t D = cfg->obs_kind == OR_OBS_TINY8   ? 8
                    : cfg->obs_kind == OR_OBS_7B16  ? 16
                    : cfg->obs_kind == OR_OBS_OCC32 ? 32
                                                    : 64;
  const int32_t A = cfg->n_actions;
  double* P = params_to_double(D, H, A, params, bf16);
  double* x = (double*)malloc(sizeof(double) * (size_t)D);
  double* h1 = (double*)malloc(sizeof(double) * (size_t)H);
  double* h2 = (double*)malloc(sizeof(double) * (size_t)H);
  double* z = (double*)malloc(sizeof(double) * (size_t)A);
  float* f = (float*)malloc(sizeof(float) * (size_t)D);
  for (int32_t i = 0; i < n; ++i) {
    or_env_state* st = &states[i];
    const uint32_t e = (uint32_t)env_ids[i];
    int32_t v1 = 0, v60 = 0;
    double tok = 0.0, exc = 0.0;
    int64_t en = 0, smp = 0;
    for (int32_t t = 0; t < T; ++t) {
      const int64_t row = (int64_t)t * n + i;
      or_env_cfg cf;
      const float* tr;
      const uint8_t* ph;
      fam_view(cfg, trace, phase, st->fam, &cf, &tr, &ph);
      env_obs_view(&cf, tr, ph, st, f);
      memcpy(obs + row * D, f, sizeof(float) * (size_t)D);
      obs_to_double(D, f, x, bf16);
      policy_fwd(D, H, A, P, x, h1, h2, z, bf16);
      double m = z[0];
      int32_t amax = 0;
      for (int32_t j = 1; j < A; ++j)
        if (z[j] > m) { m = z[j]; amax = j; }
      double S = 0.0;
      for (int32_t j = 0; j < A; ++j) S += exp(z[j] - m);
      int32_t own;
      if (deterministic) {
        own = amax;
      } else {
        uint32_t r = draw_u32(cfg->seed, e, (uint32_t)t, iteration, OR_PURPOSE_ACTION);
        double u = (double)(r >> 8) * (1.0 / 16777216.0);
        double target = u * S, c = 0.0;
        own = A - 1;
        for (int32_t j = 0; j < A; ++j) {
          c += exp(z[j] - m);
          if (target < c) { own = j; break; }
        }
      }
      int32_t a = forced ? (int32_t)forced[row] : own;
      act_own[row] = (uint8_t)own;
      logp_taken[row] = z[a] - m - log(S);
      or_step_out so = env_step(&cf, tr, ph, st, a, lambda);
      reward[row] = so.reward;
      done[row] = (uint8_t)so.done;
      if (qout) qout[row] = (int32_t)so.q;
      v1 += so.v1;
      v60 += so.v60;
      tok += so.tokens;
      exc += so.excess;
      en += so.q;
      smp += so.samples;
      if (so.done) env_reset(cfg, trace, phase, st, e, (uint32_t)t, iteration, OR_PURPOSE_RESET);
    }
    or_env_obs(cfg, trace, phase, st, f);
    memcpy(obs_last + (int64_t)i * D, f, sizeof(float) * (size_t)D);
    viol[2 * i] = v1;
    viol[2 * i + 1] = v60;
    tokens[i] = tok;
    excess[i] = exc;
    energy_q[i] = en;
    if (samples) samples[i] = smp;
  }
  free(x); free(h1); free(h2); free(z); free(f); free(P);
  return 0;
}

/* ------------------------------------------------------------------------
 * Baseline policies of the evaluation (Sec. 4.4 random policy and threshold
 * heuristic, Sec. 4.5 hysteresis rule), decided from the state before each
 * step.  "Lower" and "raise" move the actuator one level: the group size G
 * for the inc/dec actuator (actions 1 and 2; the env keeps G inside
 * [g_min, g_max]), the level index otherwise (clamped to the table).
 *  random:     a = floor(u32 * A / 2^32), u32 the step's action draw;
 *  threshold:  lower if the latest cluster sample q > hi_q, raise if q < lo_q;
 *  hysteresis: lower if S30 > 60 drop30_q; raise if S30 < 60 climb30_q and
 *              S10 < 20 climb10_q (window sums of Eq. 1 in 1/64 W).
 * ---------------------------------------------------------------------- */
static int32_t rule_action(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                           const or_env_state* st, const or_rule* r, uint32_t e, uint32_t t,
                           uint32_t it) {
  const int32_t incdec = cfg->actuator_kind == OR_ACT_INCDEC;
  const int32_t hold = incdec ? 0 : st->level;
  const int32_t lower = incdec ? 1 : (st->level > 0 ? st->level - 1 : 0);
  const int32_t raise = incdec ? 2 : (st->level < cfg->n_levels - 1 ? st->level + 1 : cfg->n_levels - 1);
  if (r->kind == OR_RULE_RANDOM) {
    const uint32_t u = draw_u32(cfg->seed, e, t, it, OR_PURPOSE_ACTION);
    return (int32_t)(((uint64_t)u * (uint64_t)cfg->n_actions) >> 32);
  }
  if (r->kind == OR_RULE_THRESHOLD) {
    const int32_t q = qc_back(cfg, trace, phase, st, 0);
    if (q > r->hi_q) return lower;
    if (q < r->lo_q) return raise;
    return hold;
  }
  int64_t s10 = 0, s30 = 0;
  for (int32_t c = 0; c < cfg->n_channels; ++c) {
    s10 += st->s_short[c];
    s30 += st->s_long[c];
  }
  if (s30 > (int64_t)OR_W_LONG * r->drop30_q) return lower;
  if (s30 < (int64_t)OR_W_LONG * r->climb30_q && s10 < (int64_t)OR_W_SHORT * r->climb10_q) return raise;
  return hold;
}

int32_t or_rollout_rule(const or_env_cfg* cfg, const float* trace, const uint8_t* phase,
                        const or_rule* rule, const int32_t* env_ids, int32_t n,
                        or_env_state* states, int32_t T, uint32_t iteration, double lambda,
                        uint8_t* act, double* reward, uint8_t* done, int32_t* viol,
                        double* tokens, double* excess, int64_t* energy_q, int64_t* samples,
                        int32_t* qout) {
  if (rule->kind < OR_RULE_RANDOM || rule->kind > OR_RULE_HYSTERESIS) return 1;
  for (int32_t i = 0; i < n; ++i) {
    or_env_state* st = &states[i];
    const uint32_t e = (uint32_t)env_ids[i];
    int32_t v1 = 0, v60 = 0;
    double tok = 0.0, exc = 0.0;
    int64_t en = 0, smp = 0;
    for (int32_t t = 0; t < T; ++t) {
      const int64_t row = (int64_t)t * n + i;
      or_env_cfg cf;
      const float* tr;
      const uint8_t* ph;
      fam_view(cfg, trace, phase, st->fam, &cf, &tr, &ph);
      const int32_t a = rule_action(&cf, tr, ph, st, rule, e, (uint32_t)t, iteration);
      act[row] = (uint8_t)a;
      or_step_out so = env_step(&cf, tr, ph, st, a, lambda);
      reward[row] = so.reward;
      done[row] = (uint8_t)so.done;
      if (qout) qout[row] = (int32_t)so.q;
      v1 += so.v1;
      v60 += so.v60;
      tok += so.tokens;
      exc += so.excess;
      en += so.q;
      smp += so.samples;
      if (so.done) env_reset(cfg, trace, phase, st, e, (uint32_t)t, iteration, OR_PURPOSE_RESET);
    }
    viol[2 * i] = v1;
    viol[2 * i + 1] = v60;
    tokens[i] = tok;
    excess[i] = exc;
    energy_q[i] = en;
    if (samples) samples[i] = smp;
  }
  return 0;
}

/* ------------------------------------------------------------------------
 * Generalised advantage estimation (Schulman et al. 2016; gamma 0.99,
 * lambda 0.95 per Sec. 4.2): delta_t = r_t + g (1-d_t) V_{t+1} - V_t,
 * A_t = delta_t + g l (1-d_t) A_{t+1}, R_t = A_t + V_t; V_T = last value.
 * Buffers are time-major [T][E].
 * ---------------------------------------------------------------------- */
void or_gae(int32_t T, int32_t E, const float* r, const float* v, const uint8_t* done,
            const float* last_v, double gamma, double lam, double* adv, double* ret) {
  for (int32_t e = 0; e < E; ++e) {
    double a_next = 0.0, v_next = (double)last_v[e];
    for (int32_t t = T - 1; t >= 0; --t) {
      int64_t i = (int64_t)t * E + e;
      double nonterm = 1.0 - (double)done[i];
      double delta = (double)r[i] + gamma * v_next * nonterm - (double)v[i];
      double a = delta + gamma * lam * nonterm * a_next;
      adv[i] = a;
      ret[i] = a + (double)v[i];
      a_next = a;
      v_next = (double)v[i];
    }
  }
}

/* ------------------------------------------------------------------------
 * PPO (Schulman et al. 2017) with SB3's loss (Sec. 4.2): per-minibatch
 * advantage normalisation, clipped surrogate, squared-error value loss,
 * entropy bonus.  Returns the minibatch loss; `grad` receives dLoss/dparams.
 * stats: [pg_loss, v_loss, entropy, approx_kl, clip_frac].
 * ---------------------------------------------------------------------- */
/* bf16 networks (bf16 != 0): the forward pass rounds observations, weights
 * and hidden activations to bf16 as in the rollout (P must hold the
 * bf16-rounded weights), and the backward pass feeds every matrix product
 * bf16 operands: the head gradient dz, and the layer gradients
 * da2 = dh2 (1 - h2^2) and da1 = dh1 (1 - h1^2) are rounded to bf16 before
 * they are used; the layer bias gradients sum the rounded values, the head
 * bias gradient the unrounded dz. */
static double rb(double x, int32_t bf16) { return bf16 ? or_bf16_round(x) : x; }

double or_ppo_minibatch_grad_ex(int32_t D, int32_t H, int32_t A, int32_t bf16, const double* P,
                                int64_t M, const float* obs, const uint8_t* act,
                                const float* logp_old, const float* adv, const float* ret,
                                double clip, double vf_coef, double ent_coef, double* grad,
                                double* stats) {
  or_layout L = layout_of(D, H, A);
  double mean = 0.0, var = 0.0, sd = 0.0;
  for (int64_t i = 0; i < M; ++i) mean += (double)adv[i];
  mean /= (double)M;
  if (M > 1) {
    for (int64_t i = 0; i < M; ++i) var += ((double)adv[i] - mean) * ((double)adv[i] - mean);
    var /= (double)(M - 1);
    sd = sqrt(var);
  }
  if (grad) memset(grad, 0, sizeof(double) * (size_t)L.total);
  double* x = (double*)malloc(sizeof(double) * (size_t)D);
  double* h1 = (double*)malloc(sizeof(double) * (size_t)H);
  double* h2 = (double*)malloc(sizeof(double) * (size_t)H);
  double* g1 = (double*)malloc(sizeof(double) * (size_t)H);
  double* g2 = (double*)malloc(sizeof(double) * (size_t)H);
  double* dh = (double*)malloc(sizeof(double) * (size_t)H);
  double* da = (double*)malloc(sizeof(double) * (size_t)H);
  double* z = (double*)malloc(sizeof(double) * (size_t)A);
  double* lp = (double*)malloc(sizeof(double) * (size_t)A);
  double* dz = (double*)malloc(sizeof(double) * (size_t)A);
  double pg = 0.0, vl = 0.0, ent = 0.0, kl = 0.0, cf = 0.0;
  const double invM = 1.0 / (double)M;
  for (int64_t s = 0; s < M; ++s) {
    obs_to_double(D, obs + s * D, x, bf16);
    policy_fwd(D, H, A, P, x, h1, h2, z, bf16);
    double V = value_fwd(D, H, A, P, x, g1, g2, bf16);
    double m = z[0];
    for (int32_t j = 1; j < A; ++j)
      if (z[j] > m) m = z[j];
    double se = 0.0;
    for (int32_t j = 0; j < A; ++j) se += exp(z[j] - m);
    double lse = m + log(se);
    double Hs = 0.0;
    for (int32_t j = 0; j < A; ++j) {
      lp[j] = z[j] - lse;
      Hs -= exp(lp[j]) * lp[j];
    }
    const int32_t a = act[s];
    const double adv_n = M > 1 ? ((double)adv[s] - mean) / (sd + 1e-8) : (double)adv[s];
    const double logr = lp[a] - (double)logp_old[s];
    const double rho = exp(logr);
    const double rc = rho < 1.0 - clip ? 1.0 - clip : (rho > 1.0 + clip ? 1.0 + clip : rho);
    const double s1 = rho * adv_n, s2 = rc * adv_n;
    pg += -(s1 < s2 ? s1 : s2);
    vl += ((double)ret[s] - V) * ((double)ret[s] - V);
    ent += Hs;
    kl += (rho - 1.0) - logr;
    cf += fabs(rho - 1.0) > clip ? 1.0 : 0.0;
    if (!grad) continue;
    /* dL/dlogits */
    const double g_rho = (s1 <= s2) ? -adv_n : 0.0;
    const double dlp = g_rho * rho * invM;
    for (int32_t j = 0; j < A; ++j) {
      double p = exp(lp[j]);
      dz[j] = dlp * ((j == a ? 1.0 : 0.0) - p) + ent_coef * invM * p * (lp[j] + Hs);
    }
    /* policy backward (bf16: dz enters the products rounded; db3 takes it unrounded) */
    for (int32_t j = 0; j < A; ++j) {
      const double dzb = rb(dz[j], bf16);
      for (int32_t k = 0; k < H; ++k) grad[L.w3 + (int64_t)j * H + k] += dzb * h2[k];
      grad[L.b3 + j] += dz[j];
    }
    for (int32_t k = 0; k < H; ++k) {
      double acc = 0.0;
      for (int32_t j = 0; j < A; ++j) acc += P[L.w3 + (int64_t)j * H + k] * rb(dz[j], bf16);
      da[k] = rb(acc * (1.0 - h2[k] * h2[k]), bf16);
    }
    for (int32_t k = 0; k < H; ++k) {
      for (int32_t l = 0; l < H; ++l) grad[L.w2 + (int64_t)k * H + l] += da[k] * h1[l];
      grad[L.b2 + k] += da[k];
    }
    for (int32_t l = 0; l < H; ++l) {
      double acc = 0.0;
      for (int32_t k = 0; k < H; ++k) acc += P[L.w2 + (int64_t)k * H + l] * da[k];
      dh[l] = rb(acc * (1.0 - h1[l] * h1[l]), bf16);
    }
    for (int32_t l = 0; l < H; ++l) {
      for (int32_t d = 0; d < D; ++d) grad[L.w1 + (int64_t)l * D + d] += dh[l] * x[d];
      grad[L.b1 + l] += dh[l];
    }
    /* value backward */
    const double dV = vf_coef * 2.0 * (V - (double)ret[s]) * invM;
    const double dVb = rb(dV, bf16);
    for (int32_t k = 0; k < H; ++k) {
      grad[L.v3 + k] += dVb * g2[k];
      da[k] = rb(P[L.v3 + k] * dVb * (1.0 - g2[k] * g2[k]), bf16);
    }
    grad[L.c3] += dV;
    for (int32_t k = 0; k < H; ++k) {
      for (int32_t l = 0; l < H; ++l) grad[L.v2 + (int64_t)k * H + l] += da[k] * g1[l];
      grad[L.c2 + k] += da[k];
    }
    for (int32_t l = 0; l < H; ++l) {
      double acc = 0.0;
      for (int32_t k = 0; k < H; ++k) acc += P[L.v2 + (int64_t)k * H + l] * da[k];
      dh[l] = rb(acc * (1.0 - g1[l] * g1[l]), bf16);
    }
    for (int32_t l = 0; l < H; ++l) {
      for (int32_t d = 0; d < D; ++d) grad[L.v1 + (int64_t)l * D + d] += dh[l] * x[d];
      grad[L.c1 + l] += dh[l];
    }
  }
  free(x); free(h1); free(h2); free(g1); free(g2); free(dh); free(da); free(z); free(lp); free(dz);
  if (stats) {
    stats[0] = pg * invM;
    stats[1] = vl * invM;
    stats[2] = ent * invM;
    stats[3] = kl * invM;
    stats[4] = cf * invM;
  }
  return pg * invM - ent_coef * ent * invM + vf_coef * vl * invM;
}

double or_ppo_minibatch_grad(int32_t D, int32_t H, int32_t A, const double* P, int64_t M,
                             const float* obs, const uint8_t* act, const float* logp_old,
                             const float* adv, const float* ret, double clip, double vf_coef,
                             double ent_coef, double* grad, double* stats) {
  return or_ppo_minibatch_grad_ex(D, H, A, 0, P, M, obs, act, logp_old, adv, ret, clip, vf_coef,
                                  ent_coef, grad, stats);
}

/* PPO update: `epochs` passes over the N = T*E samples of one rollout, each
 * in a fresh Feistel order split into minibatches of `minibatch` (the last
 * one ragged); every minibatch: gradient, global-norm clip
 * (g *= max_norm / (|g| + 1e-6) when that is < 1), Adam (Kingma & Ba 2015,
 * Algorithm 1).  Returns the Adam step count after the update.
 * stats: [pg, v, entropy, kl, clip_frac, loss, last grad norm, steps]. */
int64_t or_ppo_update_ex(int32_t D, int32_t H, int32_t A, int32_t bf16, double* P, double* adam_m,
                         double* adam_v, int64_t adam_t, int64_t N, const float* obs,
                         const uint8_t* act, const float* logp_old, const float* adv,
                         const float* ret, const or_ppo_cfg* cfg, uint64_t seed,
                         uint32_t iteration, int64_t max_steps, double* stats) {
  or_layout L = layout_of(D, H, A);
  /* the bf16 network computes with its fp32 master parameters rounded to bf16
   * (weights only; biases stay fp32); the Adam step updates the masters */
  double* Pc = bf16 ? (double*)malloc(sizeof(double) * (size_t)L.total) : P;
  const int64_t M = cfg->minibatch;
  const int64_t nmb = (N + M - 1) / M;
  double* g = (double*)malloc(sizeof(double) * (size_t)L.total);
  float* bo = (float*)malloc(sizeof(float) * (size_t)(M * D));
  uint8_t* ba = (uint8_t*)malloc((size_t)M);
  float* bl = (float*)malloc(sizeof(float) * (size_t)M);
  float* bv = (float*)malloc(sizeof(float) * (size_t)M);
  float* br = (float*)malloc(sizeof(float) * (size_t)M);
  double acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int64_t steps = 0;
  for (int32_t ep = 0; ep < cfg->epochs; ++ep) {
    uint32_t keys[4];
    or_perm_keys(seed, (uint32_t)ep, iteration, keys);
    for (int64_t mb = 0; mb < nmb; ++mb) {
      if (max_steps >= 0 && steps >= max_steps) goto done;
      const int64_t start = mb * M;
      const int64_t cnt = (N - start) < M ? (N - start) : M;
      for (int64_t j = 0; j < cnt; ++j) {
        uint32_t idx = or_feistel_index((uint64_t)N, keys, (uint64_t)(start + j));
        memcpy(bo + j * D, obs + (int64_t)idx * D, sizeof(float) * (size_t)D);
        ba[j] = act[idx];
        bl[j] = logp_old[idx];
        bv[j] = adv[idx];
        br[j] = ret[idx];
      }
      double st[5];
      if (bf16) {
        int64_t mats[6][2] = {{L.w1, (int64_t)H * D}, {L.w2, (int64_t)H * H}, {L.w3, (int64_t)A * H},
                              {L.v1, (int64_t)H * D}, {L.v2, (int64_t)H * H}, {L.v3, (int64_t)H}};
        for (int64_t i = 0; i < L.total; ++i) Pc[i] = (double)(float)P[i];
        for (int mm = 0; mm < 6; ++mm)
          for (int64_t i = 0; i < mats[mm][1]; ++i) Pc[mats[mm][0] + i] = or_bf16_round(Pc[mats[mm][0] + i]);
      }
      double loss = or_ppo_minibatch_grad_ex(D, H, A, bf16, Pc, cnt, bo, ba, bl, bv, br, cfg->clip,
                                             cfg->vf_coef, cfg->ent_coef, g, st);
      double nrm = 0.0;
      for (int64_t i = 0; i < L.total; ++i) nrm += g[i] * g[i];
      nrm = sqrt(nrm);
      double coef = cfg->max_grad_norm / (nrm + 1e-6);
      if (coef < 1.0)
        for (int64_t i = 0; i < L.total; ++i) g[i] *= coef;
      adam_t += 1;
      const double bc1 = 1.0 - pow(cfg->beta1, (double)adam_t);
      const double bc2 = 1.0 - pow(cfg->beta2, (double)adam_t);
      for (int64_t i = 0; i < L.total; ++i) {
        adam_m[i] = cfg->beta1 * adam_m[i] + (1.0 - cfg->beta1) * g[i];
        adam_v[i] = cfg->beta2 * adam_v[i] + (1.0 - cfg->beta2) * g[i] * g[i];
        const double mh = adam_m[i] / bc1, vh = adam_v[i] / bc2;
        P[i] -= cfg->lr * mh / (sqrt(vh) + cfg->eps);
      }
      for (int k = 0; k < 5; ++k) acc[k] += st[k];
      acc[5] += loss;
      acc[6] = nrm;
      steps += 1;
    }
  }
done:
  if (stats) {
    for (int k = 0; k < 6; ++k) stats[k] = steps ? acc[k] / (double)steps : 0.0;
    stats[6] = acc[6];
    stats[7] = (double)steps;
  }
  free(g); free(bo); free(ba); free(bl); free(bv); free(br);
  if (bf16) free(Pc);
  return adam_t;
}

int64_t or_ppo_update(int32_t D, int32_t H, int32_t A, double* P, double* adam_m, double* adam_v,
                      int64_t adam_t, int64_t N, const float* obs, const uint8_t* act,
                      const float* logp_old, const float* adv, const float* ret,
                      const or_ppo_cfg* cfg, uint64_t seed, uint32_t iteration,
                      int64_t max_steps, double* stats) {
  return or_ppo_update_ex(D, H, A, 0, P, adam_m, adam_v, adam_t, N, obs, act, logp_old, adv, ret,
                          cfg, seed, iteration, max_steps, stats);
}

/* ------------------------------------------------------------------------
 * Fleet accounting (Sec. 7-8): composition n places job j's trace at start
 * offset o[n][j] (tiled circularly over the common horizon), sums the
 * per-GPU powers P_n(t) = sum_g q_g((t + o[n][job(g)]) mod L), forms the
 * trailing window sums S_w(t) over w samples (Eq. 1 without the 1/w) for
 * t in [w-1, H), and counts S_w(t) > B w (Eq. 2) and the peak S_w.
 * ---------------------------------------------------------------------- */
int32_t or_fleet_windows(int32_t G, int32_t L, const float* traces, const int32_t* job_of_gpu,
                         int32_t J, const int32_t* offsets, int64_t N, int32_t H,
                         const int32_t* windows, int32_t W, int64_t budget_q, int32_t* counts,
                         int32_t* peaks) {
  for (int32_t g = 0; g < G; ++g)
    if (job_of_gpu[g] < 0 || job_of_gpu[g] >= J) return 1;
  int32_t* q = (int32_t*)malloc(sizeof(int32_t) * (size_t)G * (size_t)L);
  for (int64_t i = 0; i < (int64_t)G * L; ++i) q[i] = (int32_t)rintf(traces[i] * 64.0f);
  int64_t* P = (int64_t*)malloc(sizeof(int64_t) * (size_t)(H > 0 ? H : 1));
  for (int64_t n = 0; n < N; ++n) {
    for (int32_t t = 0; t < H; ++t) {
      int64_t s = 0;
      for (int32_t g = 0; g < G; ++g) {
        int64_t o = offsets[n * J + job_of_gpu[g]];
        s += q[(int64_t)g * L + (int32_t)(((int64_t)t + o) % L)];
      }
      P[t] = s;
    }
    for (int32_t wi = 0; wi < W; ++wi) {
      const int32_t w = windows[wi];
      int64_t S = 0, peak = 0;
      int32_t cnt = 0;
      for (int32_t t = 0; t < H; ++t) {
        S += P[t];
        if (t >= w) S -= P[t - w];
        if (t >= w - 1) {
          if (S > budget_q * (int64_t)w) ++cnt;
          if (S > peak) peak = S;
        }
      }
      counts[n * W + wi] = cnt;
      peaks[n * W + wi] = (int32_t)peak;
    }
  }
  free(P);
  free(q);
  return 0;
}

/* ------------------------------------------------------------------------
 * Phase-staggered fleet schedule (Sec. 8): a greedy scheduler places the
 * jobs one at a time, in index order.  Job j takes the start offset o from
 * the candidate grid {0, s, 2s, ...} below L that minimises the peak w-sample
 * window sum of the partial fleet made of jobs 0..j (the earlier jobs at the
 * offsets already chosen), over t in [w-1, H); among equal peaks the lowest
 * offset wins.  offsets[j] gets the choice and peaks[j] the partial fleet's
 * peak once job j is placed.  Returns 1 on a bad job map.
 * ---------------------------------------------------------------------- */
int32_t or_fleet_stagger(int32_t G, int32_t L, const float* traces, const int32_t* job_of_gpu,
                         int32_t J, int32_t H, int32_t w, int32_t stride, int32_t* offsets,
                         int32_t* peaks) {
  for (int32_t g = 0; g < G; ++g)
    if (job_of_gpu[g] < 0 || job_of_gpu[g] >= J) return 1;
  /* per-job power series q_j(t) = sum over the job's GPUs of rint(64 x_g(t)) */
  int64_t* qj = (int64_t*)calloc((size_t)J * (size_t)L, sizeof(int64_t));
  for (int32_t g = 0; g < G; ++g)
    for (int32_t t = 0; t < L; ++t)
      qj[(int64_t)job_of_gpu[g] * L + t] += (int64_t)rintf(traces[(int64_t)g * L + t] * 64.0f);
  int64_t* placed = (int64_t*)calloc((size_t)(H > 0 ? H : 1), sizeof(int64_t));
  int64_t* series = (int64_t*)malloc(sizeof(int64_t) * (size_t)(H > 0 ? H : 1));
  for (int32_t j = 0; j < J; ++j) {
    int64_t best_peak = -1;
    int32_t best_o = 0;
    for (int64_t o = 0; o < L; o += stride) {
      for (int32_t t = 0; t < H; ++t) series[t] = placed[t] + qj[(int64_t)j * L + (int32_t)(((int64_t)t + o) % L)];
      int64_t S = 0, peak = 0;
      for (int32_t t = 0; t < H; ++t) {
        S += series[t];
        if (t >= w) S -= series[t - w];
        if (t >= w - 1 && S > peak) peak = S;
      }
      if (best_peak < 0 || peak < best_peak) {
        best_peak = peak;
        best_o = (int32_t)o;
      }
    }
    offsets[j] = best_o;
    peaks[j] = (int32_t)best_peak;
    for (int32_t t = 0; t < H; ++t) placed[t] += qj[(int64_t)j * L + (int32_t)(((int64_t)t + best_o) % L)];
  }
  free(series);
  free(placed);
  free(qj);
  return 0;
}

/* ------------------------------------------------------------------------
 * Dual ascent on the Lagrange multiplier of Eq. 6 (Eq. 7, Sec. 4.5; the G3
 * design of Sec. 4.2): with the observed violation rate v = (violating
 * steps) / (env-steps) over the last rollout (window = 1: instantaneous,
 * 60: the 30 s window of Eq. 2) and target delta,
 *   multiplicative (Eq. 7): lambda <- clip(lambda exp(eta (v - delta) / delta), lo, hi)
 *   additive (G3):          lambda <- clip(lambda + eta (v - delta) / delta, lo, hi)
 * viol is [E][2] (instantaneous, 30 s) as the rollout writes it.
 * Returns the new lambda; *rate gets v.
 * ---------------------------------------------------------------------- */
double or_dual_ascent(const int32_t* viol, int32_t E, int64_t steps, int32_t window, int32_t additive,
                      double lambda, double target, double eta, double lo, double hi, double* rate) {
  int64_t n = 0;
  for (int32_t e = 0; e < E; ++e) n += viol[2 * e + (window == 1 ? 0 : 1)];
  const double v = (double)n / ((double)E * (double)steps);
  const double gap = (v - target) / target;
  double l = additive ? lambda + eta * gap : lambda * exp(eta * gap);
  if (l < lo) l = lo;
  if (l > hi) l = hi;
  if (rate) *rate = v;
  return l;
}
