// PPO update for fp32 policy/value networks (Sec. 4.2; SB3's clipped
// surrogate, squared-error value loss, entropy bonus, global-norm gradient
// clipping and Adam).
//
// The update runs as one cooperative launch (ppo_persistent_kernel) of one
// CTA per SM: NC policy-role CTAs and NC value-role CTAs (their gradients are
// independent).  Every minibatch step is three phases behind bounded grid
// barriers:
//   1. gradient: each CTA takes ceil(cnt / NC) consecutive samples of the
//      minibatch (Feistel order) in slices of 128 (one slice for the 7B
//      minibatch), runs forward and backward with the activations
//      feature-major in shared memory (4x4 register tiles, packed two-lane
//      FMA), writes the hidden-layer weight-gradient tiles straight into its
//      fp32 partial gradient row (later slices add to it) and the rest of the
//      row after the last slice; its weights arrive as one bulk copy of a
//      per-role image laid out like shared memory;
//   2. reduce: a fixed-order fp32 sum of the NC partial rows of each network
//      and per-CTA sums of squares (deterministic);
//   3. Adam: global norm in a fixed order, clip factor, Adam step on each
//      CTA's slice of the parameters, which also rewrites the role images.
// The three-launch loop (ppo_grad_kernel, ppo_reduce_kernel,
// ppo_adam_kernel) computes the same sums and is the fallback when the
// cooperative launch is not available.  The per-minibatch advantage
// mean/std (which depend only on the permutation) are computed for all
// minibatches up front.
#include <algorithm>
#include <cmath>
#include <vector>

#include <cstddef>

#include "mlp_f32.cuh"
#include "tc.cuh"

namespace pe {

constexpr int kPpoS = 128;          // samples per slice (a 7B CTA's whole share of a minibatch)
constexpr int kPpoLD = kPpoS + 4;   // row stride of feature-major activations
constexpr int kPpoNT = 512;         // threads per gradient CTA
constexpr int kPpoRT = 4;           // sample rows per thread tile in the dense layers
constexpr int kPpoMaxEpochs = 16;
constexpr int kPpoMaxNC = 128;      // CTAs per network: above half the SMs of any GB300

struct FeistelSet {
  Feistel f[kPpoMaxEpochs];
};

// Reductions are fp32 with a fixed order (per-thread sequential sums, a
// fixed shuffle tree, then warps in order): deterministic, and off the FP64
// pipe, which on this part runs a few operations per SM per clock.
__device__ __forceinline__ float block_sum_f(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float t = 0.0f;
  for (int i = 0; i < nw; ++i) t += red[i];
  return t;
}

// advantage mean and 1/(std + 1e-8) (unbiased std) of every minibatch
__global__ void ppo_advstats_kernel(const float* __restrict__ adv, int64_t N, int M, int nmb,
                                    FeistelSet perms, float2* __restrict__ out) {
  __shared__ float red[32];
  const int mb = blockIdx.x, ep = blockIdx.y;
  const Feistel& f = perms.f[ep];
  const int64_t start = (int64_t)mb * M;
  const int cnt = (int)(N - start < (int64_t)M ? N - start : (int64_t)M);
  float s = 0.0f;
  for (int j = threadIdx.x; j < cnt; j += blockDim.x) s += __ldg(adv + feistel_index(f, start + j));
  const float mean = block_sum_f(s, red) / (float)cnt;
  float q = 0.0f;
  for (int j = threadIdx.x; j < cnt; j += blockDim.x) {
    const float a = __ldg(adv + feistel_index(f, start + j)) - mean;
    q = fmaf(a, a, q);
  }
  const float ss = block_sum_f(q, red);
  if (threadIdx.x == 0) {
    if (cnt > 1) {
      const float sd = sqrtf(ss / (float)(cnt - 1));
      out[ep * nmb + mb] = make_float2(mean, 1.0f / (sd + 1e-8f));
    } else {
      out[ep * nmb + mb] = make_float2(0.0f, 1.0f);  // a 1-sample minibatch is not normalised
    }
  }
}

// Dense-layer register tiles for the sample slices: a thread owns RT
// sample rows x 4 neurons; a warp covers 2 row groups x 16 neuron groups (the
// fastest of the warp shapes measured on the 7B network: 2x16, 4x8, 8x4 and
// 16x2 lie within 3% of each other).
template <int TE, int N, int RT>
__device__ __forceinline__ bool dense_job(int j, int& eg, int& ng) {
  constexpr int EG = TE / RT, NG = N / 4, BE = EG / 2;  // BE: 2-row-group blocks along the slice
  static_assert(EG % 2 == 0 && NG % 16 == 0, "dense tile layout");
  const int wb = j >> 5, lane = j & 31;
  eg = (wb % BE) * 2 + (lane & 1);
  ng = (wb / BE) * 16 + (lane >> 1);
  return ng < NG;
}

// outT[n][e] = tanh(b[n] + sum_k inT[k][e] WT[k][n]) for samples e < SV (a
// multiple of RT; later rows are left as they are); WT rows are LDW floats apart.
// Neuron pairs accumulate with the packed two-lane FMA (__ffma2_rn: two
// round-to-nearest fused multiply-adds, the same results as fmaf, in one
// instruction), the sample value broadcast to both lanes.
template <int TE, int K, int N, int LD, int RT, int LDW = N>
__device__ __forceinline__ void dense_fwd_w(const float* __restrict__ inT, const float* __restrict__ WT,
                                            const float* __restrict__ bias, float* __restrict__ outT, int SV) {
  constexpr int JOBS = (TE / RT) * (N / 4);
  for (int j = threadIdx.x; j < JOBS; j += blockDim.x) {
    int eg, ng;
    if (!dense_job<TE, N, RT>(j, eg, ng) || eg * RT >= SV) continue;
    float2 acc2[RT][2];
#pragma unroll
    for (int r = 0; r < RT; ++r) acc2[r][0] = acc2[r][1] = make_float2(0.0f, 0.0f);
#pragma unroll 8
    for (int k = 0; k < K; ++k) {
      float xv[RT];
      load_rt<RT>(inT + k * LD + eg * RT, xv);
      const float4 w = *reinterpret_cast<const float4*>(WT + k * LDW + ng * 4);
      const float2 w01 = make_float2(w.x, w.y), w23 = make_float2(w.z, w.w);
#pragma unroll
      for (int r = 0; r < RT; ++r) {
        const float2 xx = make_float2(xv[r], xv[r]);
        acc2[r][0] = __ffma2_rn(xx, w01, acc2[r][0]);
        acc2[r][1] = __ffma2_rn(xx, w23, acc2[r][1]);
      }
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const float bb = bias[ng * 4 + c];
      float o[RT];
#pragma unroll
      for (int r = 0; r < RT; ++r) o[r] = tanhf(((c & 1) ? acc2[r][c >> 1].y : acc2[r][c >> 1].x) + bb);
      store_rt<RT>(outT + (ng * 4 + c) * LD + eg * RT, o);
    }
  }
}

// back through a tanh layer, in place, from the transposed weights:
//   hT[k][e] <- (sum_n inT[n][e] W[n][k]) * (1 - hT[k][e]^2),  W[n][k] = WT[k][n]
// A thread owns RT = 4 samples x 4 outputs k; per 4 n it loads a 4x4 block of
// WT (rows k, columns n..n+3) and of inT and does 64 FMAs as 32 packed
// two-lane FMAs over sample pairs (the weight broadcast to both lanes).  A warp covers 16
// sample groups x 2 output groups, so its WT loads touch two rows (4 rows
// apart, different banks with the padded stride) and are broadcasts.
template <int TE, int K, int N, int LD, int LDW>
__device__ __forceinline__ void dense_bwd_wt(const float* __restrict__ inT, const float* __restrict__ WT,
                                             float* hT, int SV) {
  constexpr int RT = 4, EG = TE / RT, NG = N / 4, JOBS = EG * NG;
  static_assert(K % 4 == 0 && EG % 16 == 0, "backward tile layout");
  for (int j = threadIdx.x; j < JOBS; j += blockDim.x) {
    const int eg = j % EG, kg = j / EG;
    if (eg * RT >= SV) continue;  // samples past the slice's valid rows
    float2 acc2[2][4];  // acc2[rp][c] = (acc[2 rp][c], acc[2 rp + 1][c])
#pragma unroll
    for (int c = 0; c < 4; ++c) acc2[0][c] = acc2[1][c] = make_float2(0.0f, 0.0f);
#pragma unroll 2
    for (int n = 0; n < K; n += 4) {
      float4 w[4], d[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) w[c] = *reinterpret_cast<const float4*>(WT + (kg * 4 + c) * LDW + n);
#pragma unroll
      for (int q = 0; q < 4; ++q) d[q] = *reinterpret_cast<const float4*>(inT + (n + q) * LD + eg * RT);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float wc[4] = {w[c].x, w[c].y, w[c].z, w[c].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 ww = make_float2(wc[q], wc[q]);
          acc2[0][c] = __ffma2_rn(make_float2(d[q].x, d[q].y), ww, acc2[0][c]);
          acc2[1][c] = __ffma2_rn(make_float2(d[q].z, d[q].w), ww, acc2[1][c]);
        }
      }
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      float h[RT], o[RT];
      load_rt<RT>(hT + (kg * 4 + c) * LD + eg * RT, h);
      const float a4[4] = {acc2[0][c].x, acc2[0][c].y, acc2[1][c].x, acc2[1][c].y};
#pragma unroll
      for (int r = 0; r < RT; ++r) o[r] = a4[r] * (1.0f - h[r] * h[r]);
      store_rt<RT>(hT + (kg * 4 + c) * LD + eg * RT, o);
    }
  }
}

// dst[m][n] (+)= sum_s aT[m][s] bT[n][s] (weight gradients).  Each thread owns
// 4x4 tiles whose rows and columns are interleaved (m = mg + i*M/4,
// n = ng + j*N/4); a warp covers WM x WN (mg, ng) pairs, so one float4 load of
// the warp touches WM (or WN) distinct rows in distinct shared-memory bank
// groups: one wavefront each.
template <int M, int N, int NT>
struct WGradAcc {
  static constexpr int MG = M / 4, NG = N / 4;
  static constexpr int WN = NG < 4 ? NG : 4, WM = 32 / WN;
  static constexpr int TM = (MG + WM - 1) / WM, TN = NG / WN;
  static constexpr int NWARP = NT / 32, WT = TM * TN, PER = (WT + NWARP - 1) / NWARP;
  __device__ __forceinline__ bool job(int q, int& mg, int& ng) const {
    const int wt = (int)(threadIdx.x >> 5) + q * NWARP, lane = threadIdx.x & 31;
    mg = (wt / TN) * WM + lane / WN;
    ng = (wt % TN) * WN + lane % WN;
    return wt < WT && mg < MG;
  }
  // dst (+)= sum_s aT[m][s] bT[n][s] over s < SV, one 4x4 tile at a time (16
  // packed accumulators live), even and odd samples in the two lanes of a
  // packed two-lane FMA and added at the end; rows of dst ld floats apart
  template <int S, int LD>
  __device__ __forceinline__ void accumulate(const float* __restrict__ aT, const float* __restrict__ bT, int SV,
                                             float* dst, int ld, bool first) const {
#pragma unroll 1
    for (int q = 0; q < PER; ++q) {
      int mg, ng;
      if (!job(q, mg, ng)) continue;
      float2 v2[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) v2[i][j] = make_float2(0.0f, 0.0f);
#pragma unroll 2
      for (int s = 0; s < SV; s += 4) {
        float4 a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) a[i] = *reinterpret_cast<const float4*>(aT + (mg + i * MG) * LD + s);
#pragma unroll
        for (int j = 0; j < 4; ++j) b[j] = *reinterpret_cast<const float4*>(bT + (ng + j * NG) * LD + s);
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            v2[i][j] = __ffma2_rn(make_float2(a[i].x, a[i].y), make_float2(b[j].x, b[j].y), v2[i][j]);
            v2[i][j] = __ffma2_rn(make_float2(a[i].z, a[i].w), make_float2(b[j].z, b[j].w), v2[i][j]);
          }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          float* d = dst + (mg + i * MG) * ld + ng + j * NG;
          const float v = v2[i][j].x + v2[i][j].y;
          *d = first ? v : *d + v;
        }
    }
  }
};

// Shared memory of one gradient CTA: the role's weights (W1 and W2
// transposed, w2t rows padded to H + 4 floats so that rows 4 apart fall in
// different banks; the backward pass reads W2 from the same copy) and one
// 128-sample slice of feature-major activations.  h2t holds h2, then the
// layer-2 pre-activation gradient; h1t holds h1, then the layer-1 one.
template <int H>
__host__ __device__ constexpr int w2t_ld() { return H + 4; }

template <int D, int H, int A>
struct PpoSmem {
  float w1t[D * H], w2t[H * w2t_ld<H>()], w3[A * H], b1[H], b2[H], b3[8];
  float xt[D * kPpoLD], h1t[H * kPpoLD], h2t[H * kPpoLD];
  float z[kPpoS * A];
  float lpo[kPpoS], advn[kPpoS], ret[kPpoS];
  int32_t act[kPpoS], valid[kPpoS];
  float stat[kPpoS / 32][8];
  uint64_t bar_w;  // mbarrier of the weight-image bulk copy (one phase per minibatch step)
};

struct PpoArgs {
  const float* obs;
  const uint8_t* act;
  const float* logp_old;
  const float* adv;
  const float* ret;
  const float* params;
  const float* img;       // [2][RoleImage::SIZE] policy and value weight images
  Feistel perm;
  int64_t start;
  int cnt;
  const float2* advstat;  // (mean, 1/(std+1e-8)) of this minibatch's advantages
  float clip, vf_coef, ent_coef, inv_cnt;
  float* partial;       // [NC][P]
  float* stat_partial;  // [2*NC][8]
  float* grad_out;      // [P] reduced gradient (persistent kernel)
  int32_t* err;  // set when a bounded wait gives up (reported as stats[7] = -1)
  uint32_t wphase;  // parity of this step's weight-image mbarrier phase
  int NC;       // CTAs per network
  int per_cta;  // minibatch samples per CTA, ceil(cnt / NC): CTA c takes [c * per_cta, (c + 1) * per_cta)
  int64_t P, PS;  // parameters; row stride of the partial-sum matrix
};

// Per-role weight image: the prefix of PpoSmem (w1t, padded w2t, w3, b1,
// b2, b3[8]) as it sits in shared memory, kept up to date by the Adam phase
// so that a gradient CTA loads its weights as one contiguous float4 copy.
// Image 0 is the policy network, image 1 the value network (its head is row
// 0 of w3 and b3[0]).  The padding floats of w2t stay zero.
template <int D, int H, int A>
struct RoleImage {
  static constexpr int64_t LDW = w2t_ld<H>();
  static constexpr int64_t W1T = 0, W2T = W1T + (int64_t)D * H, W3 = W2T + (int64_t)H * LDW,
                           B1 = W3 + (int64_t)A * H, B2 = B1 + H, B3 = B2 + H, SIZE = B3 + 8;
  static_assert(SIZE % 4 == 0, "role image is copied as float4");
};

template <int D, int H, int A>
__device__ __forceinline__ void store_image(float* img, int64_t p, float val) {
  using I = RoleImage<D, H, A>;
  const MlpLayout L = mlp_layout(D, H, A);
  const bool pol = p < L.v1;
  float* m = img + (pol ? 0 : I::SIZE);
  const int64_t w1 = pol ? L.w1 : L.v1, b1 = pol ? L.b1 : L.c1, w2 = pol ? L.w2 : L.v2,
                b2 = pol ? L.b2 : L.c2, w3 = pol ? L.w3 : L.v3, b3 = pol ? L.b3 : L.c3;
  if (p < b1) {
    const int64_t q = p - w1;                       // W1[n][k], n = q / D, k = q % D
    m[I::W1T + (q % D) * H + q / D] = val;
  } else if (p < w2) {
    m[I::B1 + (p - b1)] = val;
  } else if (p < b2) {
    const int64_t q = p - w2;                       // W2[n][k], n = q / H, k = q % H
    m[I::W2T + (q % H) * I::LDW + q / H] = val;
  } else if (p < w3) {
    m[I::B2 + (p - b2)] = val;
  } else if (p < b3) {
    m[I::W3 + (p - w3)] = val;
  } else {
    m[I::B3 + (p - b3)] = val;
  }
}

template <int D, int H, int A>
__global__ void ppo_image_kernel(const float* __restrict__ params, float* __restrict__ img) {
  const int64_t P = mlp_layout(D, H, A).total;
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x)
    store_image<D, H, A>(img, p, params[p]);
}

// One role (policy or value network) of the minibatch gradient over this
// CTA's slices: forward, loss, backward; weight-gradient partials in
// registers, written as this CTA's row of the partial-sum matrix.
template <int D, int H, int A, bool POL>
__device__ __forceinline__ bool ppo_role(PpoSmem<D, H, A>& s, const PpoArgs& g, int c) {
  constexpr int NA = POL ? A : 1;
  constexpr int S = kPpoS, LD = kPpoLD;
  static_assert(D % 4 == 0 && H % 32 == 0 && S * (D / 4) <= kPpoNT && S <= kPpoNT && 4 * H <= kPpoNT,
                "gradient CTA layout");
  const MlpLayout Lp = mlp_layout(D, H, A);
  const int64_t oW1 = POL ? Lp.w1 : Lp.v1, oB1 = POL ? Lp.b1 : Lp.c1;
  const int64_t oW2 = POL ? Lp.w2 : Lp.v2, oB2 = POL ? Lp.b2 : Lp.c2;
  const int64_t oW3 = POL ? Lp.w3 : Lp.v3, oB3 = POL ? Lp.b3 : Lp.c3;
  const int tid = threadIdx.x;
  const float2 as = *g.advstat;
  // gather one slice (permuted sample order) of nv <= S samples:
  // observations as float4 rows (one per thread), per-sample scalars by
  // threads < S; rows past nv are zero and marked invalid
  auto gather = [&](int base, int nv) {
    constexpr int F4 = D / 4;
    if (tid < S * F4) {
      const int si = tid / F4, f = tid % F4;
      float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      if (si < nv) {
        const uint32_t idx = feistel_index(g.perm, g.start + base + si);
        v = __ldg(reinterpret_cast<const float4*>(g.obs + (int64_t)idx * D) + f);
      }
      s.xt[(4 * f + 0) * LD + si] = v.x;
      s.xt[(4 * f + 1) * LD + si] = v.y;
      s.xt[(4 * f + 2) * LD + si] = v.z;
      s.xt[(4 * f + 3) * LD + si] = v.w;
    }
    if (tid < S) {
      const int si = tid;
      const int ok = si < nv;
      s.valid[si] = ok;
      if (ok) {
        const uint32_t idx = feistel_index(g.perm, g.start + base + si);
        s.act[si] = __ldg(g.act + idx);
        s.lpo[si] = __ldg(g.logp_old + idx);
        s.advn[si] = (__ldg(g.adv + idx) - as.x) * as.y;
        s.ret[si] = __ldg(g.ret + idx);
      } else {
        s.act[si] = 0;
        s.lpo[si] = s.advn[si] = s.ret[si] = 0.0f;
      }
    }
  };
  // the role's weight image, one bulk copy into shared memory completed on
  // an mbarrier (its bytes all in flight at once).  Inside the persistent
  // update other CTAs rewrite the image between minibatches with ordinary
  // stores, made visible to this CTA by the grid barrier; the proxy fences
  // order those writes, and this CTA's earlier reads of the weights, before
  // the copy.  Every thread waits, bounded, before the first slice.
  {
    using I = RoleImage<D, H, A>;
    using Sm = PpoSmem<D, H, A>;
    static_assert(offsetof(Sm, b3) == sizeof(float) * (size_t)I::B3, "image matches shared memory");
    static_assert((I::SIZE * sizeof(float)) % 16 == 0, "bulk copy size");
    if (tid == 0) {
      asm volatile("fence.proxy.async.global;" ::: "memory");
      tc::fence_async_smem();
      tc::mbar_expect_tx(&s.bar_w, (uint32_t)(I::SIZE * sizeof(float)));
      tc::bulk_g2s(s.w1t, g.img + (POL ? 0 : I::SIZE), (uint32_t)(I::SIZE * sizeof(float)), &s.bar_w);
    }
  }
  // this CTA's samples [c0, c1) of the minibatch, in slices of S
  const int c0 = c * g.per_cta, c1 = min(c0 + g.per_cta, g.cnt);
  // the first slice's gather overlaps the weight copy, issued above
  if (c0 < c1) gather(c0, min(S, c1 - c0));
  // A wait that gives up (in any thread) stops the whole CTA: thread 0
  // records the error, waits once more (bounded) so that the copy into this
  // CTA's shared memory is no longer in flight, and the role returns false.
  if (!__syncthreads_and(tc::mbar_wait(&s.bar_w, g.wphase))) {
    if (tid == 0) {
      atomicExch(g.err, 1);
      (void)tc::mbar_wait(&s.bar_w, g.wphase);
    }
    __syncthreads();
    return false;
  }
  // weight-gradient tiles live in registers only during their phase; the
  // first slice writes them to this CTA's partial gradient row, later slices
  // (when a CTA's share exceeds S samples) add to it
  float* row = g.partial + (int64_t)c * g.PS;
  int nsl = 0;
  // head backward: thread (k = tid / 4, quarter q = tid % 4) owns row k of the
  // head weight gradient and of the layer-2 bias gradient over samples 4i + q
  const int hk = tid >> 2, hq = tid & 3;
  float g3[NA], gb2 = 0.0f, gb1 = 0.0f, gb3 = 0.0f;
#pragma unroll
  for (int a = 0; a < NA; ++a) g3[a] = 0.0f;
  float st[5] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f};  // pg, entropy, kl, clip, value (threads < S)

  for (int base = c0; base < c1; base += S) {
    // nv valid samples; the tiles cover the first SV rows (nv rounded up to
    // 8: whole 4-row groups, both groups of a warp).  Rows in [nv, SV) are
    // zero-input samples whose loss gradient is zero.
    const int nv = min(S, c1 - base), SV = min(S, (nv + 7) & ~7);
    if (base > c0) {
      __syncthreads();
      gather(base, nv);
    }
    __syncthreads();
    // forward
    dense_fwd_w<S, D, H, LD, kPpoRT>(s.xt, s.w1t, s.b1, s.h1t, SV);
    __syncthreads();
    dense_fwd_w<S, H, H, LD, kPpoRT, w2t_ld<H>()>(s.h1t, s.w2t, s.b2, s.h2t, SV);
    __syncthreads();
    // head: job (sample si = j / 8, K-part q = j % 8) sums k = q, q+8, ...
    // for every action; the 8 parts (adjacent lanes) are shuffle-combined
    static_assert((S * 8) % kPpoNT == 0, "whole head jobs per thread");
    for (int hj = tid; hj < S * 8; hj += kPpoNT) {
      const int q = hj & 7, si = hj >> 3;
      if (si < SV) {  // warp-uniform: a warp covers 4 samples and SV is a multiple of 8
      float acc[NA];
#pragma unroll
      for (int a = 0; a < NA; ++a) acc[a] = 0.0f;
#pragma unroll 4
      for (int k = q; k < H; k += 8) {
        const float h = s.h2t[k * LD + si];
#pragma unroll
        for (int a = 0; a < NA; ++a) acc[a] = fmaf(s.w3[a * H + k], h, acc[a]);
      }
#pragma unroll
      for (int a = 0; a < NA; ++a) {
        acc[a] += __shfl_xor_sync(0xffffffffu, acc[a], 1);
        acc[a] += __shfl_xor_sync(0xffffffffu, acc[a], 2);
        acc[a] += __shfl_xor_sync(0xffffffffu, acc[a], 4);
      }
      if (q == 0)
#pragma unroll
        for (int a = 0; a < NA; ++a) s.z[si * NA + a] = acc[a] + s.b3[a];
      }
    }
    __syncthreads();
    // loss terms and dLoss/dhead per sample (written over the head outputs)
    if (tid < S) {
      float* z = s.z + tid * NA;
      if (!s.valid[tid]) {
#pragma unroll
        for (int j = 0; j < NA; ++j) z[j] = 0.0f;
      } else if (POL) {
        float m = z[0];
#pragma unroll
        for (int j = 1; j < NA; ++j) m = fmaxf(m, z[j]);
        float se = 0.0f;
#pragma unroll
        for (int j = 0; j < NA; ++j) se += expf(z[j] - m);
        const float lse = m + logf(se);
        float lp[NA], p[NA], Hs = 0.0f;
#pragma unroll
        for (int j = 0; j < NA; ++j) {
          lp[j] = z[j] - lse;
          p[j] = expf(lp[j]);
          Hs -= p[j] * lp[j];
        }
        const int a = s.act[tid];
        const float an = s.advn[tid];
        float lpa = 0.0f;
#pragma unroll
        for (int j = 0; j < NA; ++j)
          if (j == a) lpa = lp[j];
        const float logr = lpa - s.lpo[tid];
        const float rho = expf(logr);
        const float rc = fminf(fmaxf(rho, 1.0f - g.clip), 1.0f + g.clip);
        const float s1 = rho * an, s2 = rc * an;
        st[0] += -fminf(s1, s2);
        st[1] += Hs;
        st[2] += kl_term(logr);
        st[3] += fabsf(rho - 1.0f) > g.clip ? 1.0f : 0.0f;
        const float dlp = (s1 <= s2 ? -an : 0.0f) * rho * g.inv_cnt;
#pragma unroll
        for (int j = 0; j < NA; ++j)
          z[j] = dlp * ((j == a ? 1.0f : 0.0f) - p[j]) + g.ent_coef * g.inv_cnt * p[j] * (lp[j] + Hs);
      } else {
        const float V = z[0], R = s.ret[tid];
        st[4] += (R - V) * (R - V);
        z[0] = g.vf_coef * 2.0f * (V - R) * g.inv_cnt;
      }
    }
    __syncthreads();
    // head weight gradient, back through the head into layer 2 (in place over h2)
    if (hk < H) {
      float w3k[NA];
#pragma unroll
      for (int a = 0; a < NA; ++a) w3k[a] = s.w3[a * H + hk];
#pragma unroll 4
      for (int i = 0; i < SV / 4; ++i) {
        const int si = 4 * i + hq;
        const float h = s.h2t[hk * LD + si];
        float d = 0.0f;
#pragma unroll
        for (int a = 0; a < NA; ++a) {
          const float dz = s.z[si * NA + a];
          g3[a] = fmaf(dz, h, g3[a]);
          d = fmaf(w3k[a], dz, d);
        }
        const float d2 = d * (1.0f - h * h);
        s.h2t[hk * LD + si] = d2;
        gb2 += d2;
      }
    }
    if (tid < NA) {
      float acc = 0.0f;
      for (int si = 0; si < S; ++si) acc += s.z[si * NA + tid];
      gb3 += acc;
    }
    __syncthreads();
    // layer-2 weight gradient
    {
      WGradAcc<H, H, kPpoNT> g2;
      g2.template accumulate<S, LD>(s.h2t, s.h1t, SV, row + oW2, H, nsl == 0);
    }
    __syncthreads();
    // back into layer 1 (in place over h1)
    dense_bwd_wt<S, H, H, LD, w2t_ld<H>()>(s.h2t, s.w2t, s.h1t, SV);
    __syncthreads();
    // layer-1 weight and bias gradients (the bias by the warps the tiles leave idle)
    {
      WGradAcc<H, D, kPpoNT> g1;
      g1.template accumulate<S, LD>(s.h1t, s.xt, SV, row + oW1, D, nsl == 0);
    }
    if (tid >= kPpoNT - H) {
      const int n = tid - (kPpoNT - H), lane = tid & 31;
      float acc = 0.0f;
      for (int i = 0; i < S; ++i) {
        const int e = (i + lane) & (S - 1);
        if (e < SV) acc += s.h1t[n * LD + e];
      }
      gb1 += acc;
    }
    ++nsl;
  }
  // the rest of the partial gradient row (the hidden-layer weight gradients
  // are zero if the CTA's share held no sample)
  if (nsl == 0) {
    for (int i = tid; i < H * H; i += blockDim.x) row[oW2 + i] = 0.0f;
    for (int i = tid; i < H * D; i += blockDim.x) row[oW1 + i] = 0.0f;
  }
#pragma unroll
  for (int a = 0; a < NA; ++a) {
    g3[a] += __shfl_xor_sync(0xffffffffu, g3[a], 1);
    g3[a] += __shfl_xor_sync(0xffffffffu, g3[a], 2);
  }
  gb2 += __shfl_xor_sync(0xffffffffu, gb2, 1);
  gb2 += __shfl_xor_sync(0xffffffffu, gb2, 2);
  if (hq == 0 && hk < H) {
#pragma unroll
    for (int a = 0; a < NA; ++a) row[oW3 + (int64_t)a * H + hk] = g3[a];
    row[oB2 + hk] = gb2;
  }
  if (tid >= kPpoNT - H) row[oB1 + tid - (kPpoNT - H)] = gb1;
  if (tid < NA) row[oB3 + tid] = gb3;
  // statistics of the CTA's samples (held by threads < S), fixed shuffle tree
  if (tid < S) {
#pragma unroll
    for (int k = 0; k < 5; ++k)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) st[k] += __shfl_xor_sync(0xffffffffu, st[k], o);
    if ((tid & 31) == 0)
#pragma unroll
      for (int k = 0; k < 5; ++k) s.stat[tid >> 5][k] = st[k];
  }
  __syncthreads();
  if (tid == 0) {
    float* sp = g.stat_partial + (int64_t)((POL ? 0 : g.NC) + c) * 8;
#pragma unroll
    for (int k = 0; k < 5; ++k) {
      float t = 0.0f;
      for (int w = 0; w < S / 32; ++w) t += s.stat[w][k];
      sp[k] = t;
    }
  }
  return true;
}

template <int D, int H, int A>
__global__ void __launch_bounds__(kPpoNT) ppo_grad_kernel(PpoArgs g) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  PpoSmem<D, H, A>& s = *reinterpret_cast<PpoSmem<D, H, A>*>(smem_raw);
  if (threadIdx.x == 0) {
    tc::mbar_init(&s.bar_w, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  if ((int)blockIdx.x < g.NC)
    (void)ppo_role<D, H, A, true>(s, g, blockIdx.x);
  else
    (void)ppo_role<D, H, A, false>(s, g, blockIdx.x - g.NC);
}

// Running minibatch statistics from the per-CTA partials, by one whole warp:
// lane c sums rows c, c + 32, ... in fp32, a fixed xor tree combines the
// lanes, and lane 0 adds the minibatch means to the fp64 running sums
// (pg loss, value loss, entropy, approximate KL, clip fraction, total loss).
// The partials are read through L2: inside the persistent update other CTAs
// wrote them.
__device__ __forceinline__ void fold_stats(const float* stat_partial, int NC, float inv_cnt, float vf_coef,
                                           float ent_coef, double* acc) {
  const int lane = threadIdx.x & 31;
  float v[5] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
  for (int c = lane; c < NC; c += 32) {
    v[0] += __ldcg(stat_partial + c * 8 + 0);
    v[1] += __ldcg(stat_partial + c * 8 + 1);
    v[2] += __ldcg(stat_partial + c * 8 + 2);
    v[3] += __ldcg(stat_partial + c * 8 + 3);
    v[4] += __ldcg(stat_partial + (NC + c) * 8 + 4);
  }
#pragma unroll
  for (int k = 0; k < 5; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
  if (lane == 0) {
    const double ic = inv_cnt;
    acc[0] += (double)v[0] * ic;
    acc[1] += (double)v[4] * ic;
    acc[2] += (double)v[1] * ic;
    acc[3] += (double)v[2] * ic;
    acc[4] += (double)v[3] * ic;
    acc[5] += (double)v[0] * ic + (double)vf_coef * v[4] * ic - (double)ent_coef * v[1] * ic;
  }
}

// ---------------------------------------------------------------------------
// Persistent form of the whole update: one cooperative launch runs every
// minibatch step as three phases separated by grid barriers -- gradient
// partials (as ppo_grad_kernel), a fixed-order reduction of each CTA's slice
// of the parameter vector, and the clipped Adam step on that slice.  The
// cooperative launch guarantees that all CTAs are resident, and every
// barrier wait is bounded: on timeout the kernel records an error and stops.
// ---------------------------------------------------------------------------
struct PpoLoop {
  PpoArgs g;              // per-minibatch fields are filled in by the kernel
  const float2* advstat;  // [epochs][nmb]
  FeistelSet perms;
  int64_t N;
  int minibatch, nmb, epochs;
  float* params;
  float* img;              // role weight images (PpoArgs::img), rewritten by the Adam phase
  float* m;
  float* v;
  float* sq;               // [gridDim.x] per-CTA sums of squares
  double* acc;             // [8] running statistics
  unsigned int* bar;       // monotonic arrival count, zeroed before the launch
  int32_t* err;
  const float* bc;         // [2 * steps]: step_size, 1/sqrt(bc2) per Adam step
  float beta1, beta2, eps, max_norm;
};

// Grid barrier on a monotonic arrival counter (zeroed before the launch):
// the k-th barrier's arrivals are numbered k*G .. k*G + G - 1 (no CTA can
// arrive at barrier k + 1 before all have arrived at k), so each CTA waits
// for the counter to reach (k + 1) * G; the last arrival releases everyone
// with its own atomic, and nothing is reset.  The wait is bounded.  Memory
// order: the block barrier puts the CTA's writes before thread 0's arrival,
// a release at GPU scope; thread 0's polling loads are acquires at GPU
// scope, and the second block barrier puts them before the CTA's reads.
__device__ __forceinline__ bool grid_barrier(unsigned int* bar, int* s_ok, long long limit = 4000000000LL) {
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int old;
    asm volatile("atom.release.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar) : "memory");
    const unsigned int target = (old / gridDim.x + 1u) * gridDim.x;
    bool ok = true;
    const long long t0 = clock64();
    for (;;) {
      unsigned int v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar) : "memory");
      if ((int)(v - target) >= 0) break;
      if (clock64() - t0 > limit) {  // by default about 2 s at the maximum SM clock
        ok = false;
        break;
      }
    }
    *s_ok = ok;
  }
  __syncthreads();
  return *s_ok != 0;
}

// Self-test of the bounded waits (mode 0: the grid barrier with CTA 1 never
// arriving; mode 1: the same barrier with every CTA arriving; mode 2: an
// mbarrier nothing arrives at).  A wait that gives up sets *err.
__global__ void wait_selftest_kernel(unsigned int* bar, int32_t* err, int mode, long long limit) {
  __shared__ int s_ok;
  __shared__ uint64_t mb;
  if (mode == 2) {
    if (threadIdx.x == 0) {
      tc::mbar_init(&mb, 1);
      tc::fence_mbar_init();
    }
    __syncthreads();
    if (!tc::mbar_wait(&mb, 0, limit) && threadIdx.x == 0) atomicExch(err, 1);
    return;
  }
  if (mode == 0 && blockIdx.x == 1) return;  // this CTA never reaches the barrier
  if (!grid_barrier(bar, &s_ok, limit) && threadIdx.x == 0) atomicExch(err, 1);
}

pe_status wait_selftest(int mode, int64_t limit_cycles, void* ws, cudaStream_t st) {
  unsigned int* bar = reinterpret_cast<unsigned int*>(ws);
  int32_t* err = reinterpret_cast<int32_t*>(reinterpret_cast<char*>(ws) + 8);
  PE_TRY_CUDA(cudaMemsetAsync(ws, 0, 16, st));
  long long limit = (long long)limit_cycles;
  if (mode == 2) {
    wait_selftest_kernel<<<1, 32, 0, st>>>(bar, err, mode, limit);
  } else {
    void* args[] = {&bar, &err, &mode, &limit};
    PE_TRY_CUDA(cudaLaunchCooperativeKernel((void*)wait_selftest_kernel, dim3(2), dim3(32), args, 0, st));
  }
  PE_CHECK_LAUNCH("wait_selftest_kernel");
  int32_t host = 0;
  PE_TRY_CUDA(cudaMemcpyAsync(&host, err, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  if (host) return fail(PE_ETIMEOUT, "bounded wait gave up (self-test mode %d)", mode);
  return PE_OK;
}

template <int D, int H, int A>
__global__ void __launch_bounds__(kPpoNT, 1) ppo_persistent_kernel(PpoLoop L) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  PpoSmem<D, H, A>& s = *reinterpret_cast<PpoSmem<D, H, A>*>(smem_raw);
  __shared__ int s_ok;
  __shared__ float s_red[kPpoNT / 32];
  __shared__ float s_norm;
  const int NC = L.g.NC, tid = threadIdx.x;
  const int64_t P = L.g.P;
  const int64_t PS = L.g.PS;
  const int64_t per = ((P + gridDim.x - 1) / gridDim.x + 3) / 4 * 4;
  const int64_t p0 = (int64_t)blockIdx.x * per, p1 = p0 + per < P ? p0 + per : P;
  if (tid == 0) {
    tc::mbar_init(&s.bar_w, 1);
    tc::fence_mbar_init();
  }
  __syncthreads();
  int step = 0;
  for (int ep = 0; ep < L.epochs; ++ep) {
    for (int mb = 0; mb < L.nmb; ++mb, ++step) {
      const int64_t start = (int64_t)mb * L.minibatch;
      const int cnt = (int)(L.N - start < L.minibatch ? L.N - start : L.minibatch);
      PpoArgs g = L.g;
      g.perm = L.perms.f[ep];
      g.start = start;
      g.cnt = cnt;
      g.inv_cnt = 1.0f / (float)cnt;
      g.per_cta = (cnt + NC - 1) / NC;
      g.wphase = (uint32_t)(step & 1);
      g.advstat = L.advstat + (int64_t)ep * L.nmb + mb;
      // phase 1: gradient partials of this CTA's role and samples
      // a role whose weight copy timed out has recorded the error; the CTA
      // stops, and the others give up at their next (bounded) barrier
      const bool role_ok = (int)blockIdx.x < NC ? ppo_role<D, H, A, true>(s, g, blockIdx.x)
                                                : ppo_role<D, H, A, false>(s, g, blockIdx.x - NC);
      if (!role_ok) return;
      if (!grid_barrier(L.bar, &s_ok)) {
        if (tid == 0) atomicExch(L.err, 1);
        return;
      }
      // phase 2: grad[p] = sum_c partial[c][p] in a fixed order (row group
      // rg = c % 8 summed in row order, then the groups in order), and this
      // CTA's sum of squares.  64 float4 columns x 8 row groups per pass; the
      // dead h1 slice buffer holds the group sums.
      float q = 0.0f;
      {
        float* part = s.h1t;
        const int c4 = tid & 63, rg = tid >> 6;
        for (int64_t pb = p0; pb < p1; pb += 256) {
          const int64_t p = pb + 4 * c4;
          float4 acc4 = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
          if (p < p1) {
            for (int h = 0; 8 * h < NC; h += 4) {
              float4 v[4];
#pragma unroll
              for (int u = 0; u < 4; ++u)
                if (rg + 8 * (h + u) < NC)
                  v[u] = __ldcg(reinterpret_cast<const float4*>(g.partial + (int64_t)(rg + 8 * (h + u)) * PS + p));
#pragma unroll
              for (int u = 0; u < 4; ++u)
                if (rg + 8 * (h + u) < NC) {
                  acc4.x += v[u].x;
                  acc4.y += v[u].y;
                  acc4.z += v[u].z;
                  acc4.w += v[u].w;
                }
            }
          }
          *reinterpret_cast<float4*>(part + rg * 256 + 4 * c4) = acc4;
          __syncthreads();
          if (tid < 256 && pb + tid < p1) {
            float gs = 0.0f;
#pragma unroll
            for (int r = 0; r < 8; ++r) gs += part[r * 256 + tid];
            L.g.grad_out[pb + tid] = gs;
            q = fmaf(gs, gs, q);
          }
          __syncthreads();
        }
      }
      const float qb = block_sum_f(q, s_red);
      if (tid == 0) L.sq[blockIdx.x] = qb;
      if (!grid_barrier(L.bar, &s_ok)) {
        if (tid == 0) atomicExch(L.err, 1);
        return;
      }
      // phase 3: global norm (fixed order), clip factor, Adam on this slice.
      // The last CTA, whose parameter slice is the shortest, also folds the
      // minibatch statistics (its warp 1), off the barrier-bound path.
      if (tid < 32) {
        float t = 0.0f;
        for (int b = tid; b < (int)gridDim.x; b += 32) t += __ldcg(L.sq + b);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (tid == 0) s_norm = sqrtf(t);
      } else if (tid < 64 && blockIdx.x == gridDim.x - 1) {
        fold_stats(g.stat_partial, NC, g.inv_cnt, g.vf_coef, g.ent_coef, L.acc);
      }
      __syncthreads();
      const float norm = s_norm;
      const float coef = fminf(1.0f, L.max_norm / (norm + 1e-6f));
      const float step_size = L.bc[2 * step], inv_sqrt_bc2 = L.bc[2 * step + 1];
      for (int64_t p = p0 + tid; p < p1; p += blockDim.x) {
        const float gp = L.g.grad_out[p] * coef;
        const float mp = L.beta1 * L.m[p] + (1.0f - L.beta1) * gp;
        const float vp = L.beta2 * L.v[p] + (1.0f - L.beta2) * gp * gp;
        L.m[p] = mp;
        L.v[p] = vp;
        const float np = L.params[p] - step_size * mp / (sqrtf(vp) * inv_sqrt_bc2 + L.eps);
        L.params[p] = np;
        store_image<D, H, A>(L.img, p, np);
      }
      if (blockIdx.x == 0 && tid == 0) {
        L.acc[6] = norm;
        L.acc[7] += 1.0;
      }
      if (!grid_barrier(L.bar, &s_ok)) {
        if (tid == 0) atomicExch(L.err, 1);
        return;
      }
    }
  }
}

// grad[p] = sum_c partial[c][p] in a fixed order: a block covers 32
// parameters x 8 partial-row groups (row c goes to group c % 8), the groups
// are combined in shared memory in group order.  The last block to finish
// (atomic ticket; no block waits for another) forms the global norm from the
// per-block sums of squares in block order and the minibatch statistics.
constexpr int kRedP = 32, kRedG = 8;

struct ReduceArgs {
  const float* partial;
  const float* stat_partial;  // [2*NC][8]
  int NC;
  int64_t P, PS;
  float* grad;
  float* sq;              // [gridDim.x]
  unsigned int* ticket;   // zeroed before the first launch; the last block re-zeroes it
  float* norm;            // [1] out
  double* acc;            // [8] running statistics
  float vf_coef, ent_coef, inv_cnt;
};

__global__ void __launch_bounds__(kRedP * kRedG) ppo_reduce_kernel(ReduceArgs a) {
  __shared__ float part[kRedG][kRedP];
  __shared__ float red[kRedG];
  __shared__ bool last;
  const int lp = threadIdx.x % kRedP, cg = threadIdx.x / kRedP;
  const int64_t p = (int64_t)blockIdx.x * kRedP + lp;
  float s = 0.0f;
  if (p < a.P)
    for (int c = cg; c < a.NC; c += kRedG) s += __ldg(a.partial + (int64_t)c * a.PS + p);
  part[cg][lp] = s;
  __syncthreads();
  if (cg == 0) {
    float g = 0.0f;
#pragma unroll
    for (int k = 0; k < kRedG; ++k) g += part[k][lp];
    if (p < a.P) a.grad[p] = g;
    float q = p < a.P ? g * g : 0.0f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    if (lp == 0) {
      a.sq[blockIdx.x] = q;
      __threadfence();
      const unsigned int t = atomicAdd(a.ticket, 1u);
      last = (t == gridDim.x - 1);
    }
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  // last block: global norm (fixed order: strided partial sums, then warp tree)
  float q = 0.0f;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += blockDim.x) q += *((volatile float*)a.sq + b);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = q;
  __syncthreads();
  if (threadIdx.x < 32) {
    fold_stats(a.stat_partial, a.NC, a.inv_cnt, a.vf_coef, a.ent_coef, a.acc);
    if (threadIdx.x == 0) {
      float t = 0.0f;
      for (int k = 0; k < kRedG; ++k) t += red[k];
      const float norm = sqrtf(t);
      *a.norm = norm;
      a.acc[6] = norm;
      a.acc[7] += 1.0;
      *a.ticket = 0u;
    }
  }
}

struct AdamArgs {
  float beta1, beta2, step_size, inv_sqrt_bc2, eps, max_norm;
};

template <int D, int H, int A>
__global__ void ppo_adam_kernel(float* __restrict__ params, float* __restrict__ img, float* __restrict__ m,
                                float* __restrict__ v, const float* __restrict__ grad,
                                const float* __restrict__ norm_p, int64_t P, AdamArgs a) {
  const float norm = *norm_p;
  const float coef = fminf(1.0f, a.max_norm / (norm + 1e-6f));
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P;
       p += (int64_t)gridDim.x * blockDim.x) {
    const float gp = grad[p] * coef;
    const float mp = a.beta1 * m[p] + (1.0f - a.beta1) * gp;
    const float vp = a.beta2 * v[p] + (1.0f - a.beta2) * gp * gp;
    m[p] = mp;
    v[p] = vp;
    const float np = params[p] - a.step_size * mp / (sqrtf(vp) * a.inv_sqrt_bc2 + a.eps);
    params[p] = np;
    store_image<D, H, A>(img, p, np);
  }
}

// stats[7] is the Adam step count, or -1 if a bounded grid-barrier wait gave up
__global__ void ppo_finalize_kernel(const double* __restrict__ acc, const int32_t* __restrict__ err,
                                    float* __restrict__ stats) {
  const int k = threadIdx.x;
  if (k < 8) {
    const double n = acc[7] > 0 ? acc[7] : 1.0;
    stats[k] = (float)(k < 6 ? acc[k] / n : acc[k]);
    if (k == 7 && *err) stats[7] = -1.0f;
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
Feistel make_feistel(uint64_t n, uint64_t seed, uint32_t epoch, uint32_t iteration) {
  Feistel f;
  const u32x4 k = philox10(u32x4{epoch, 0u, iteration, kDrawPerm}, (uint32_t)seed, (uint32_t)(seed >> 32));
  f.k[0] = k.x;
  f.k[1] = k.y;
  f.k[2] = k.z;
  f.k[3] = k.w;
  int bits = 2;
  while ((1ull << bits) < n) ++bits;
  if (bits & 1) ++bits;
  f.half = (uint32_t)(bits / 2);
  f.n = n;
  return f;
}

struct PpoPlan {
  int64_t P, N;
  int nmb, NC, nsq, steps;  // NC: the most CTAs per network a launch may use (workspace bound)
  int64_t PS;  // row stride of the partial-sum matrix (P rounded up to 4)
  int64_t off_advstat, off_partial, off_stat, off_grad, off_img, off_sq, off_acc, off_bar, off_bc, total;
};

static int64_t align256(int64_t x) { return (x + 255) / 256 * 256; }

static int64_t img_floats(const pe_net& net) {
  const int64_t D = net.obs_dim, H = net.hidden, A = net.n_actions;
  return D * H + H * (H + 4) + A * H + 2 * H + 8;
}

static PpoPlan ppo_plan(const pe_net& net, const pe_ppo_config& cfg, int64_t N) {
  PpoPlan p;
  p.P = mlp_layout(net.obs_dim, net.hidden, net.n_actions).total;
  p.PS = (p.P + 3) / 4 * 4;
  p.N = N;
  p.nmb = (int)((N + cfg.minibatch - 1) / cfg.minibatch);
  const int ncap = (cfg.minibatch + 7) / 8;  // at least 8 samples per CTA
  p.NC = ncap < kPpoMaxNC ? ncap : kPpoMaxNC;
  p.nsq = (int)((p.P + kRedP - 1) / kRedP);
  p.steps = cfg.epochs * p.nmb;
  int64_t o = 0;
  p.off_advstat = o; o = align256(o + (int64_t)cfg.epochs * p.nmb * 8);
  p.off_partial = o; o = align256(o + (int64_t)p.NC * p.PS * 4);
  p.off_stat = o; o = align256(o + (int64_t)2 * p.NC * 8 * 4);
  p.off_grad = o; o = align256(o + p.P * 4);
  p.off_img = o; o = align256(o + 2 * img_floats(net) * 4);
  p.off_sq = o; o = align256(o + (int64_t)(p.nsq > 2 * p.NC ? p.nsq : 2 * p.NC) * 8);
  p.off_acc = o; o = align256(o + 8 * 8 + 16);
  p.off_bar = o; o = align256(o + 16);
  p.off_bc = o; o = align256(o + (int64_t)p.steps * 8);
  p.total = o;
  return p;
}

// advantage statistics of every (epoch, minibatch), shared with the bf16 update
pe_status launch_advstats(const float* adv, int64_t N, int M, int nmb, int epochs, uint64_t seed,
                          uint32_t iteration, float2* out, cudaStream_t st) {
  if (epochs < 1 || epochs > kPpoMaxEpochs) return fail(PE_EINVAL, "epochs must be in [1, %d]", kPpoMaxEpochs);
  FeistelSet perms{};
  for (int ep = 0; ep < epochs; ++ep) perms.f[ep] = make_feistel((uint64_t)N, seed, ep, iteration);
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    ppo_advstats_kernel<<<dim3(nmb, epochs), 1024, 0, st>>>(adv, N, M, nmb, perms, out);
  }
  PE_CHECK_LAUNCH("ppo_advstats_kernel");
  return PE_OK;
}

int64_t ppo_ws_bytes_f32(const pe_net& net, const pe_ppo_config& cfg, int64_t N) {
  return ppo_plan(net, cfg, N).total;
}

template <int D, int H, int A>
static pe_status ppo_run(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                         const float* obs, const uint8_t* act, const float* logp_old,
                         const float* adv, const float* ret, int64_t N, const pe_ppo_config& cfg,
                         float* stats, char* ws, cudaStream_t st) {
  const PpoPlan pl = ppo_plan(net, cfg, N);
  float2* advstat = reinterpret_cast<float2*>(ws + pl.off_advstat);
  float* partial = reinterpret_cast<float*>(ws + pl.off_partial);
  float* stat_partial = reinterpret_cast<float*>(ws + pl.off_stat);
  float* grad = reinterpret_cast<float*>(ws + pl.off_grad);
  float* img = reinterpret_cast<float*>(ws + pl.off_img);
  float* sq = reinterpret_cast<float*>(ws + pl.off_sq);
  double* acc = reinterpret_cast<double*>(ws + pl.off_acc);
  float* norm = reinterpret_cast<float*>(acc + 8);
  unsigned int* ticket = reinterpret_cast<unsigned int*>(acc + 9);
  PE_TRY_CUDA(cudaMemsetAsync(acc, 0, 8 * sizeof(double) + 16, st));
  FeistelSet perms{};
  for (int ep = 0; ep < cfg.epochs; ++ep) perms.f[ep] = make_feistel((uint64_t)N, cfg.seed, ep, cfg.iteration);
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    ppo_advstats_kernel<<<dim3(pl.nmb, cfg.epochs), 256, 0, st>>>(adv, N, cfg.minibatch, pl.nmb, perms, advstat);
  }
  PE_CHECK_LAUNCH("ppo_advstats_kernel");
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    PE_TRY_CUDA(cudaMemsetAsync(img, 0, 2 * img_floats(net) * sizeof(float), st));  // zero the w2t padding
    ppo_image_kernel<D, H, A><<<ceil_div(pl.P, 256), 256, 0, st>>>(params, img);
  }
  PE_CHECK_LAUNCH("ppo_image_kernel");
  using Smem = PpoSmem<D, H, A>;
  static_assert(sizeof(Smem) + 1024 <= 232448, "gradient CTA shared memory");
  auto kern = ppo_grad_kernel<D, H, A>;
  const int bytes = (int)sizeof(Smem);
  PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
  int dev = 0, sms = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  unsigned int* bar = reinterpret_cast<unsigned int*>(ws + pl.off_bar);
  int32_t* bar_err = reinterpret_cast<int32_t*>(ws + pl.off_bar + 8);
  PE_TRY_CUDA(cudaMemsetAsync(bar, 0, 16, st));
  // cooperative persistent update when every CTA can be resident at once
  auto pk = ppo_persistent_kernel<D, H, A>;
  PE_TRY_CUDA(cudaFuncSetAttribute(pk, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
  int per_sm = 0, coop = 0;
  PE_TRY_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, pk, kPpoNT, bytes));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev));
  // one CTA per SM for each network: as many CTAs as the GPU holds at once
  const int nc = std::min(pl.NC, per_sm * sms / 2);
  if (coop && nc >= 1) {
    std::vector<float> bc(2 * (size_t)pl.steps);
    for (int k = 0; k < pl.steps; ++k) {
      const double tt = (double)(adam_t + k + 1);
      bc[2 * k] = (float)(cfg.lr / (1.0 - std::pow((double)cfg.beta1, tt)));
      bc[2 * k + 1] = (float)(1.0 / std::sqrt(1.0 - std::pow((double)cfg.beta2, tt)));
    }
    float* bc_dev = reinterpret_cast<float*>(ws + pl.off_bc);
    PE_TRY_CUDA(cudaMemcpyAsync(bc_dev, bc.data(), bc.size() * sizeof(float), cudaMemcpyHostToDevice, st));
    PpoLoop L;
    L.g.obs = obs;
    L.g.act = act;
    L.g.logp_old = logp_old;
    L.g.adv = adv;
    L.g.ret = ret;
    L.g.params = params;
    L.g.img = img;
    L.img = img;
    L.g.clip = cfg.clip;
    L.g.vf_coef = cfg.vf_coef;
    L.g.ent_coef = cfg.ent_coef;
    L.g.partial = partial;
    L.g.stat_partial = stat_partial;
    L.g.grad_out = grad;
    L.g.NC = nc;
    L.g.err = bar_err;
    L.g.wphase = 0;
    L.g.P = pl.P;
    L.g.PS = pl.PS;
    L.advstat = advstat;
    L.perms = perms;
    L.N = N;
    L.minibatch = cfg.minibatch;
    L.nmb = pl.nmb;
    L.epochs = cfg.epochs;
    L.params = params;
    L.m = m;
    L.v = v;
    L.sq = sq;
    L.acc = acc;
    L.bar = bar;
    L.err = bar_err;
    L.bc = bc_dev;
    L.beta1 = cfg.beta1;
    L.beta2 = cfg.beta2;
    L.eps = cfg.eps;
    L.max_norm = cfg.max_grad_norm;
    void* kargs[] = {&L};
    {
      ProfScope ps(PE_PROF_PPO_GRAD, st);
      PE_TRY_CUDA(cudaLaunchCooperativeKernel((void*)pk, dim3(2 * nc), dim3(kPpoNT), kargs, (size_t)bytes, st));
    }
    PE_CHECK_LAUNCH("ppo_persistent_kernel");
  } else {
    const int ncf = std::min(pl.NC, 64);
    int64_t t = adam_t;
    for (int ep = 0; ep < cfg.epochs; ++ep) {
      for (int mb = 0; mb < pl.nmb; ++mb) {
        const int64_t start = (int64_t)mb * cfg.minibatch;
        const int cnt = (int)std::min<int64_t>(cfg.minibatch, N - start);
        PpoArgs g;
        g.obs = obs;
        g.act = act;
        g.logp_old = logp_old;
        g.adv = adv;
        g.ret = ret;
        g.params = params;
        g.img = img;
        g.perm = perms.f[ep];
        g.start = start;
        g.cnt = cnt;
        g.clip = cfg.clip;
        g.vf_coef = cfg.vf_coef;
        g.ent_coef = cfg.ent_coef;
        g.inv_cnt = 1.0f / (float)cnt;
        g.partial = partial;
        g.stat_partial = stat_partial;
        g.NC = ncf;
        g.per_cta = (cnt + ncf - 1) / ncf;
        g.err = bar_err;
        g.wphase = 0;  // a fresh mbarrier in every launch
        g.P = pl.P;
        g.PS = pl.PS;
        g.advstat = advstat + (int64_t)ep * pl.nmb + mb;
        {
          ProfScope ps(PE_PROF_PPO_GRAD, st);
          kern<<<2 * ncf, kPpoNT, bytes, st>>>(g);
        }
        PE_CHECK_LAUNCH("ppo_grad_kernel");
        {
          ProfScope ps(PE_PROF_PPO_REDUCE, st);
          ReduceArgs ra;
          ra.partial = partial;
          ra.stat_partial = stat_partial;
          ra.NC = ncf;
          ra.P = pl.P;
          ra.PS = pl.PS;
          ra.grad = grad;
          ra.sq = sq;
          ra.ticket = ticket;
          ra.norm = norm;
          ra.acc = acc;
          ra.vf_coef = cfg.vf_coef;
          ra.ent_coef = cfg.ent_coef;
          ra.inv_cnt = 1.0f / (float)cnt;
          ppo_reduce_kernel<<<pl.nsq, kRedP * kRedG, 0, st>>>(ra);
        }
        PE_CHECK_LAUNCH("ppo_reduce_kernel");
        t += 1;
        const double bc1 = 1.0 - std::pow((double)cfg.beta1, (double)t);
        const double bc2 = 1.0 - std::pow((double)cfg.beta2, (double)t);
        AdamArgs a;
        a.beta1 = cfg.beta1;
        a.beta2 = cfg.beta2;
        a.step_size = (float)(cfg.lr / bc1);
        a.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
        a.eps = cfg.eps;
        a.max_norm = cfg.max_grad_norm;
        {
          ProfScope ps(PE_PROF_PPO_ADAM, st);
          ppo_adam_kernel<D, H, A><<<(int)((pl.P + 255) / 256), 256, 0, st>>>(params, img, m, v, grad, norm, pl.P, a);
        }
        PE_CHECK_LAUNCH("ppo_adam_kernel");
      }
    }
  }
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    ppo_finalize_kernel<<<1, 32, 0, st>>>(acc, bar_err, stats);
  }
  PE_CHECK_LAUNCH("ppo_finalize_kernel");
  return PE_OK;
}

}  // namespace pe

namespace pe {

pe_status ppo_update_f32(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                         const float* obs, const uint8_t* act, const float* logp_old,
                         const float* adv, const float* ret, int64_t N, const pe_ppo_config& cfg,
                         float* stats, void* ws, cudaStream_t st) {
  char* w = reinterpret_cast<char*>(ws);
  if (net.obs_dim == 8 && net.hidden == 64 && net.n_actions == 3)
    return ppo_run<8, 64, 3>(net, params, m, v, adam_t, obs, act, logp_old, adv, ret, N, cfg, stats, w, st);
  if (net.obs_dim == 16 && net.hidden == 128 && net.n_actions == 5)
    return ppo_run<16, 128, 5>(net, params, m, v, adam_t, obs, act, logp_old, adv, ret, N, cfg, stats, w, st);
  return fail(PE_EINVAL, "unsupported fp32 PPO network (D=%d H=%d A=%d)", net.obs_dim, net.hidden,
              net.n_actions);
}

}  // namespace pe
