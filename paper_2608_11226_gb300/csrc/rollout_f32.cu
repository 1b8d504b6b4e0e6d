// Fused rollout for fp32 policy networks (Tiny: 8-64-64x3, 7B: 16-128-128x5).
//
// One CTA owns a tile of TE envs for the whole horizon (the loop over t is
// sequential, envs are independent).  The policy weights and the tile's env
// state stay in shared memory; per step the CTA computes the observation
// features, the two tanh layers and the logits with FFMA register tiles,
// samples with Philox, steps the envs and writes one row of the time-major
// rollout buffer.  The value network does not steer the rollout, so it runs
// afterwards over all T*E observations as a separate, fully parallel kernel.
#include "env.cuh"
#include "mlp_f32.cuh"

namespace pe {

template <int D, int H, int A, int TE, int C, int OBS>
struct RolloutF32Smem {
  float w1t[D * H], b1[H], w2t[H * H], b2[H], w3[A * H], b3[(A + 3) / 4 * 4];
  float xt[D * TE], h1t[H * TE], h2t[H * TE], logits[TE * A];
  EnvTile<TE, C> env;
};

template <int D, int H, int A, int TE, int C, int OBS>
__global__ void __launch_bounds__(TE / 4 * H / 4)
    rollout_f32_kernel(EnvDev env, const float* __restrict__ params, int T, uint32_t it,
                       float lambda, int det, pe_rollout_buf buf) {
  using Smem = RolloutF32Smem<D, H, A, TE, C, OBS>;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& s = *reinterpret_cast<Smem*>(smem_raw);
  const int e0 = blockIdx.x * TE;
  const int ne = min(TE, env.E - e0);
  const MlpLayout Lp = mlp_layout(D, H, A);
  load_transposed(params + Lp.w1, s.w1t, H, D);
  load_transposed(params + Lp.w2, s.w2t, H, H);
  load_copy(params + Lp.b1, s.b1, H);
  load_copy(params + Lp.b2, s.b2, H);
  load_copy(params + Lp.w3, s.w3, A * H);
  load_copy(params + Lp.b3, s.b3, A);
  load_tile<TE, C>(env, s.env, e0, ne);
  __syncthreads();

  float* obs_out = reinterpret_cast<float*>(buf.obs);
  int32_t v1 = 0, v60 = 0;
  int64_t energy = 0, smp = 0;
  float tok = 0.0f, exc = 0.0f;
  const int tid = threadIdx.x;

  for (int t = 0; t <= T; ++t) {
    // (1) observation features -> xT (and the buffer row)
    float* dst = t < T ? obs_out + ((int64_t)t * env.E + e0) * D
                       : reinterpret_cast<float*>(buf.obs_last) + (int64_t)e0 * D;
    for (int idx = tid; idx < TE * D; idx += blockDim.x) {
      const int e = idx / D, f = idx % D;
      float v = 0.0f;
      if (e < ne) {
        TileAcc<TE, C> acc{s.env, e};
        v = feature<C, OBS>(env, acc, f);
        dst[idx] = v;
      }
      s.xt[f * TE + e] = v;
    }
    if (t == T) break;
    __syncthreads();
    // (2)-(4) policy network
    dense_tanh_t<TE, D, H>(s.xt, s.w1t, s.b1, s.h1t);
    __syncthreads();
    dense_tanh_t<TE, H, H>(s.h1t, s.w2t, s.b2, s.h2t);
    __syncthreads();
    head_t<TE, H, A>(s.h2t, s.w3, s.b3, s.logits);
    __syncthreads();
    // (5) sample, actuate, consume one sample, reward
    if (tid < ne) {
      const int e = tid;
      const uint32_t eg = (uint32_t)(e0 + e);
      const uint32_t r = det ? 0u : draw32(env.seed, eg, (uint32_t)t, it, kDrawAction);
      float lp;
      const int a = sample_action<A>(s.logits + e * A, r, det != 0, &lp);
      TileAcc<TE, C> acc{s.env, e};
      const StepOut so = env_step<C>(env, acc, a, lambda);
      const int64_t row = (int64_t)t * env.E + eg;
      buf.act[row] = (uint8_t)a;
      buf.logp[row] = lp;
      buf.reward[row] = so.reward;
      buf.done[row] = (uint8_t)so.done;
      if (buf.q) buf.q[row] = so.q;
      v1 += so.v1;
      v60 += so.v60;
      energy += so.q;
      smp += so.samples;
      tok += so.tokens;
      exc += so.excess;
      if (so.done) env_reset<C>(env, acc, eg, (uint32_t)t, it, kDrawReset);
    }
    __syncthreads();
  }
  if (tid < ne) {
    const int g = e0 + tid;
    buf.viol[2 * g] = v1;
    buf.viol[2 * g + 1] = v60;
    buf.tokens[g] = tok;
    buf.excess[g] = exc;
    buf.energy_q[g] = energy;
    if (buf.samples) buf.samples[g] = smp;
  }
  store_tile<TE, C>(env, s.env, e0, ne);
}

template <int D, int H, int TE>
struct ValueF32Smem {
  float w1t[D * H], b1[H], w2t[H * H], b2[H], w3[H], b3[4];
  float xt[D * TE], h1t[H * TE], h2t[H * TE], out[TE];
};

// value network over n observation rows (persistent over tiles of TE rows)
template <int D, int H, int TE>
__global__ void __launch_bounds__(TE / 4 * H / 4)
    value_f32_kernel(const float* __restrict__ params, int A, const float* __restrict__ obs,
                     int64_t n, float* __restrict__ value) {
  using Smem = ValueF32Smem<D, H, TE>;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& s = *reinterpret_cast<Smem*>(smem_raw);
  const MlpLayout Lp = mlp_layout(D, H, A);
  load_transposed(params + Lp.v1, s.w1t, H, D);
  load_transposed(params + Lp.v2, s.w2t, H, H);
  load_copy(params + Lp.c1, s.b1, H);
  load_copy(params + Lp.c2, s.b2, H);
  load_copy(params + Lp.v3, s.w3, H);
  load_copy(params + Lp.c3, s.b3, 1);
  const int64_t tiles = (n + TE - 1) / TE;
  for (int64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
    const int64_t r0 = tile * TE;
    const int nr = (int)(n - r0 < (int64_t)TE ? n - r0 : (int64_t)TE);
    __syncthreads();
    for (int idx = threadIdx.x; idx < TE * D; idx += blockDim.x) {
      const int e = idx / D, f = idx % D;
      s.xt[f * TE + e] = e < nr ? __ldg(obs + r0 * D + idx) : 0.0f;
    }
    __syncthreads();
    dense_tanh_t<TE, D, H>(s.xt, s.w1t, s.b1, s.h1t);
    __syncthreads();
    dense_tanh_t<TE, H, H>(s.h1t, s.w2t, s.b2, s.h2t);
    __syncthreads();
    head_t<TE, H, 1>(s.h2t, s.w3, s.b3, s.out);
    __syncthreads();
    for (int e = threadIdx.x; e < nr; e += blockDim.x) value[r0 + e] = s.out[e];
  }
}

// ---------------------------------------------------------------------------
// host launchers
// ---------------------------------------------------------------------------
template <int D, int H, int A, int TE, int C, int OBS>
static pe_status launch_rollout(const EnvDev& env, const float* params, int T, uint32_t it,
                                float lambda, int det, const pe_rollout_buf& buf,
                                cudaStream_t st) {
  using Smem = RolloutF32Smem<D, H, A, TE, C, OBS>;
  auto kern = rollout_f32_kernel<D, H, A, TE, C, OBS>;
  const int bytes = (int)sizeof(Smem);
  PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
  {
    ProfScope ps(PE_PROF_ROLLOUT, st);
    kern<<<ceil_div(env.E, TE), TE / 4 * H / 4, bytes, st>>>(env, params, T, it, lambda, det, buf);
  }
  PE_CHECK_LAUNCH("rollout_f32_kernel");
  return PE_OK;
}

template <int D, int H, int TE>
static pe_status launch_value(const float* params, int A, const float* obs, int64_t n,
                              float* value, cudaStream_t st) {
  if (n <= 0) return PE_OK;
  using Smem = ValueF32Smem<D, H, TE>;
  auto kern = value_f32_kernel<D, H, TE>;
  const int bytes = (int)sizeof(Smem);
  PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
  int dev = 0, sms = 0, per_sm = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  PE_TRY_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, TE / 4 * H / 4, bytes));
  const int64_t tiles = (n + TE - 1) / TE;
  const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
  const int grid = (int)(tiles < cap ? tiles : cap);
  {
    ProfScope ps(PE_PROF_VALUE, st);
    kern<<<grid, TE / 4 * H / 4, bytes, st>>>(params, A, obs, n, value);
  }
  PE_CHECK_LAUNCH("value_f32_kernel");
  return PE_OK;
}

pe_status rollout_f32(const EnvDev& env, const pe_net& net, const float* params, int T,
                      uint32_t it, float lambda, int det, const pe_rollout_buf& buf,
                      cudaStream_t st) {
  constexpr int TE = 32;
  if (net.obs_dim == 8 && net.hidden == 64 && net.n_actions == 3 && env.C == 1 &&
      env.obs_kind == PE_OBS_TINY8)
    return launch_rollout<8, 64, 3, TE, 1, PE_OBS_TINY8>(env, params, T, it, lambda, det, buf, st);
  if (net.obs_dim == 16 && net.hidden == 128 && net.n_actions == 5 && env.C == 1 &&
      env.obs_kind == PE_OBS_7B16)
    return launch_rollout<16, 128, 5, TE, 1, PE_OBS_7B16>(env, params, T, it, lambda, det, buf, st);
  return fail(PE_EINVAL, "unsupported fp32 network/env combination (D=%d H=%d A=%d C=%d obs=%d)",
              net.obs_dim, net.hidden, net.n_actions, env.C, env.obs_kind);
}

pe_status value_f32(const pe_net& net, const float* params, const float* obs, int64_t n,
                    float* value, cudaStream_t st) {
  constexpr int TE = 32;
  if (net.obs_dim == 8 && net.hidden == 64)
    return launch_value<8, 64, TE>(params, net.n_actions, obs, n, value, st);
  if (net.obs_dim == 16 && net.hidden == 128)
    return launch_value<16, 128, TE>(params, net.n_actions, obs, n, value, st);
  return fail(PE_EINVAL, "unsupported fp32 value network (D=%d H=%d)", net.obs_dim, net.hidden);
}

}  // namespace pe
