// PPO update for bf16 networks (72B: 32-256-256x16, Stress: 64-512-512x16;
// Sec. 4.2 loss and optimiser as in the fp32 update).
//
// Per minibatch:
//   forward   -- the tcgen05 tensor-core MLP kernels over the minibatch's
//                Feistel-permuted rows, saving x, h1, h2 (bf16) and the heads;
//   loss      -- one thread per sample: clipped surrogate, value loss,
//                entropy; dLoss/dhead in fp32, rounded to bf16 for the products;
//   backward  -- per network five plain bf16 x bf16 -> fp32 GEMMs through
//                cuBLASLt (dh2 = dz W3, dW2 = da2^T h1, dh1 = da2 W2,
//                dW1 = da1^T x, dW3 = dz^T h2), with the tanh derivative,
//                the bf16 rounding of da2 / da1 and the bias partial sums in
//                an elementwise kernel between them; the weight gradients land
//                directly in the canonical gradient vector;
//   step      -- fixed-order bias reduction, global norm, clip, Adam on the
//                fp32 master parameters.
// Rounding points (which the oracle reproduces): dz, da2 and da1 enter the
// products as bf16; the layer bias gradients sum the rounded values, the head
// bias gradient the fp32 dz.
#include <cublasLt.h>
#include <cuda_bf16.h>

#include <cmath>
#include <map>
#include <mutex>
#include <tuple>
#include <vector>

#include "mlp_f32.cuh"

namespace pe {

// defined in mlp_bf16.cu / ppo_f32.cu
int64_t bf16_image_bytes(const pe_net& net);
pe_status bf16_make_images(const pe_net& net, const float* params, uint8_t* two_images, cudaStream_t st);
pe_status bf16_forward_save(const pe_net& net, const uint8_t* img, const float* params, int value_net,
                            const void* obs, const uint32_t* gather, int64_t n, float* out, int out_stride,
                            __nv_bfloat16* x, __nv_bfloat16* h1, __nv_bfloat16* h2, int32_t* err,
                            cudaStream_t st);
pe_status launch_advstats(const float* adv, int64_t N, int M, int nmb, int epochs, uint64_t seed,
                          uint32_t iteration, float2* out, cudaStream_t st);

constexpr int kHead = 16;        // head rows (logits; the value head padded with zero rows)
constexpr int kRowsPerPart = 32;  // rows summed per bias partial
constexpr int64_t kLtWorkspace = 32ll << 20;

// ---------------------------------------------------------------------------
// cuBLASLt row-major bf16 GEMM: C[M x N] (fp32, ldc) = op(A) op(B) with
// op(A) = A[M x K] (lda) or A stored [K x M] when ta, op(B) = B[K x N] (ldb)
// or B stored [N x K] when tb.  Column-major view: C^T = op(B)^T op(A)^T.
// ---------------------------------------------------------------------------
struct GemmPlan {
  cublasLtMatmulDesc_t op = nullptr;
  cublasLtMatrixLayout_t x = nullptr, y = nullptr, c = nullptr;
  cublasLtMatmulAlgo_t algo;
};

static std::mutex g_lt_mu;
static cublasLtHandle_t g_lt = nullptr;
static std::map<std::tuple<int64_t, int64_t, int64_t, int64_t, int64_t, int64_t, int, int>, GemmPlan> g_plans;

static pe_status lt_check(cublasStatus_t s, const char* what) {
  if (s != CUBLAS_STATUS_SUCCESS) return fail(PE_ECUDA, "cuBLASLt error %d in %s", (int)s, what);
  return PE_OK;
}

#define PE_TRY_LT(expr)                                  \
  do {                                                   \
    pe_status _s = lt_check((expr), #expr);              \
    if (_s != PE_OK) return _s;                          \
  } while (0)

static pe_status gemm_bf16(int64_t M, int64_t N, int64_t K, const __nv_bfloat16* A, int64_t lda, bool ta,
                           const __nv_bfloat16* B, int64_t ldb, bool tb, float* C, int64_t ldc, void* lt_ws,
                           cudaStream_t st) {
  // every operand is 16-byte aligned (workspace offsets and the canonical
  // layout with A = 16); the plans are chosen for exactly that alignment
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B) | reinterpret_cast<uintptr_t>(C)) & 15)
    return fail(PE_EINVAL, "GEMM operand not 16-byte aligned");
  std::lock_guard<std::mutex> lk(g_lt_mu);
  if (!g_lt) PE_TRY_LT(cublasLtCreate(&g_lt));
  int dev = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  const auto key = std::make_tuple(M, N, K, lda, ldb, ldc, (int)ta | ((int)tb << 1), dev);
  auto it = g_plans.find(key);
  if (it == g_plans.end()) {
    GemmPlan p;
    PE_TRY_LT(cublasLtMatmulDescCreate(&p.op, CUBLAS_COMPUTE_32F, CUDA_R_32F));
    const cublasOperation_t ox = tb ? CUBLAS_OP_T : CUBLAS_OP_N, oy = ta ? CUBLAS_OP_T : CUBLAS_OP_N;
    PE_TRY_LT(cublasLtMatmulDescSetAttribute(p.op, CUBLASLT_MATMUL_DESC_TRANSA, &ox, sizeof(ox)));
    PE_TRY_LT(cublasLtMatmulDescSetAttribute(p.op, CUBLASLT_MATMUL_DESC_TRANSB, &oy, sizeof(oy)));
    // X = B in column-major: [N x K] (ld ldb) or, transposed, stored [K x N]
    PE_TRY_LT(cublasLtMatrixLayoutCreate(&p.x, CUDA_R_16BF, tb ? K : N, tb ? N : K, ldb));
    // Y = A in column-major: [K x M] (ld lda) or, transposed, stored [M x K]
    PE_TRY_LT(cublasLtMatrixLayoutCreate(&p.y, CUDA_R_16BF, ta ? M : K, ta ? K : M, lda));
    PE_TRY_LT(cublasLtMatrixLayoutCreate(&p.c, CUDA_R_32F, N, M, ldc));
    cublasLtMatmulPreference_t pref;
    PE_TRY_LT(cublasLtMatmulPreferenceCreate(&pref));
    const uint64_t wsb = (uint64_t)kLtWorkspace;
    PE_TRY_LT(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MAX_WORKSPACE_BYTES, &wsb, sizeof(wsb)));
    const uint32_t align = 16;
    PE_TRY_LT(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_A_BYTES, &align, sizeof(align)));
    PE_TRY_LT(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_B_BYTES, &align, sizeof(align)));
    PE_TRY_LT(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_C_BYTES, &align, sizeof(align)));
    PE_TRY_LT(cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_D_BYTES, &align, sizeof(align)));
    cublasLtMatmulHeuristicResult_t res;
    int found = 0;
    PE_TRY_LT(cublasLtMatmulAlgoGetHeuristic(g_lt, p.op, p.x, p.y, p.c, p.c, pref, 1, &res, &found));
    cublasLtMatmulPreferenceDestroy(pref);
    if (found < 1) return fail(PE_ECUDA, "cuBLASLt found no algorithm for %lldx%lldx%lld", (long long)M, (long long)N, (long long)K);
    p.algo = res.algo;
    it = g_plans.emplace(key, p).first;
  }
  const float one = 1.0f, zero = 0.0f;
  const GemmPlan& p = it->second;
  PE_TRY_LT(cublasLtMatmul(g_lt, p.op, &one, B, p.x, A, p.y, &zero, C, p.c, C, p.c, &p.algo, lt_ws,
                           (size_t)kLtWorkspace, st));
  return PE_OK;
}

// ---------------------------------------------------------------------------
// kernels
// ---------------------------------------------------------------------------
__global__ void perm_index_kernel(Feistel f, int64_t start, int cnt, uint32_t* __restrict__ idx) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j < cnt) idx[j] = feistel_index(f, start + j);
}

// bf16 copies of W2 and of the head (padded to 16 rows) for the backward GEMMs
__global__ void backward_weights_kernel(const float* __restrict__ params, int D, int H, int A,
                                        __nv_bfloat16* __restrict__ wb) {
  const MlpLayout Lp = mlp_layout(D, H, A);
  const int64_t per = (int64_t)H * H + (int64_t)kHead * H;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < 2 * per; i += (int64_t)gridDim.x * blockDim.x) {
    const int net = (int)(i / per);
    const int64_t j = i % per;
    float v;
    if (j < (int64_t)H * H) {
      v = params[(net ? Lp.v2 : Lp.w2) + j];
    } else {
      const int64_t q = j - (int64_t)H * H;
      const int r = (int)(q / H), k = (int)(q % H);
      const int nout = net ? 1 : A;
      v = r < nout ? params[(net ? Lp.v3 : Lp.w3) + (int64_t)r * H + k] : 0.0f;
    }
    wb[i] = __float2bfloat16_rn(v);
  }
}

struct LossArgs {
  const float* zp;  // [cnt][16] policy logits
  const float* zv;  // [cnt] values
  const uint32_t* idx;
  const uint8_t* act;
  const float* logp_old;
  const float* adv;
  const float* ret;
  const float2* advstat;
  int cnt, A;
  float clip, vf_coef, ent_coef, inv_cnt;
  __nv_bfloat16* dzp;  // [cnt][16]
  __nv_bfloat16* dzv;  // [cnt][16], column 0 used
  float* part;         // [nblk][32]: pg, ent, kl, clip, vl, db3[16], dc3
};

constexpr int kLossThreads = 256;
constexpr int kPartW = 32;

__global__ void __launch_bounds__(kLossThreads) ppo_bf16_loss_kernel(LossArgs g) {
  __shared__ float red[kLossThreads / 32][kPartW];
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  float v[kPartW];
#pragma unroll
  for (int k = 0; k < kPartW; ++k) v[k] = 0.0f;
  if (j < g.cnt) {
    const uint32_t i = g.idx[j];
    const float2 as = *g.advstat;
    float z[kHead];
#pragma unroll
    for (int a = 0; a < kHead; ++a) z[a] = a < g.A ? g.zp[(int64_t)j * kHead + a] : -INFINITY;
    float m = z[0];
#pragma unroll
    for (int a = 1; a < kHead; ++a) m = fmaxf(m, z[a]);
    float se = 0.0f;
#pragma unroll
    for (int a = 0; a < kHead; ++a) se += a < g.A ? expf(z[a] - m) : 0.0f;
    const float lse = m + logf(se);
    float lp[kHead], p[kHead], Hs = 0.0f;
#pragma unroll
    for (int a = 0; a < kHead; ++a) {
      lp[a] = a < g.A ? z[a] - lse : 0.0f;
      p[a] = a < g.A ? expf(lp[a]) : 0.0f;
      Hs -= p[a] * lp[a];
    }
    const int act = g.act[i];
    const float an = (g.adv[i] - as.x) * as.y;
    float lpa = 0.0f;
#pragma unroll
    for (int a = 0; a < kHead; ++a)
      if (a == act) lpa = lp[a];
    const float logr = lpa - g.logp_old[i];
    const float rho = expf(logr);
    const float rc = fminf(fmaxf(rho, 1.0f - g.clip), 1.0f + g.clip);
    const float s1 = rho * an, s2 = rc * an;
    v[0] = -fminf(s1, s2);
    v[1] = Hs;
    v[2] = kl_term(logr);
    v[3] = fabsf(rho - 1.0f) > g.clip ? 1.0f : 0.0f;
    const float dlp = (s1 <= s2 ? -an : 0.0f) * rho * g.inv_cnt;
    uint32_t pk[kHead / 2];
#pragma unroll
    for (int a = 0; a < kHead; a += 2) {
      float d0 = 0.0f, d1 = 0.0f;
      if (a < g.A) d0 = dlp * ((a == act ? 1.0f : 0.0f) - p[a]) + g.ent_coef * g.inv_cnt * p[a] * (lp[a] + Hs);
      if (a + 1 < g.A)
        d1 = dlp * ((a + 1 == act ? 1.0f : 0.0f) - p[a + 1]) + g.ent_coef * g.inv_cnt * p[a + 1] * (lp[a + 1] + Hs);
      v[5 + a] = d0;
      v[5 + a + 1] = d1;
      __nv_bfloat162 b2 = __floats2bfloat162_rn(d0, d1);
      pk[a / 2] = *reinterpret_cast<uint32_t*>(&b2);
    }
    uint4* o = reinterpret_cast<uint4*>(g.dzp + (int64_t)j * kHead);
    o[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    o[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
    const float V = g.zv[j], R = g.ret[i];
    v[4] = (R - V) * (R - V);
    const float dV = g.vf_coef * 2.0f * (V - R) * g.inv_cnt;
    v[21] = dV;
    __nv_bfloat162 b2 = __floats2bfloat162_rn(dV, 0.0f);
    uint4* ov = reinterpret_cast<uint4*>(g.dzv + (int64_t)j * kHead);
    ov[0] = make_uint4(*reinterpret_cast<uint32_t*>(&b2), 0u, 0u, 0u);
    ov[1] = make_uint4(0u, 0u, 0u, 0u);
  }
  // fixed-order block partial sums
#pragma unroll
  for (int k = 0; k < kPartW; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int k = 0; k < kPartW; ++k) red[threadIdx.x >> 5][k] = v[k];
  __syncthreads();
  if (threadIdx.x < kPartW) {
    float t = 0.0f;
    for (int w = 0; w < kLossThreads / 32; ++w) t += red[w][threadIdx.x];
    g.part[(int64_t)blockIdx.x * kPartW + threadIdx.x] = t;
  }
}

// da = bf16(dh * (1 - h^2)); column sums of the rounded da per 32-row block
__global__ void bwd_act_kernel(const float* __restrict__ dh, const __nv_bfloat16* __restrict__ h, int cnt,
                               int H, __nv_bfloat16* __restrict__ da, float* __restrict__ part) {
  const int col = blockIdx.y * blockDim.x + threadIdx.x;
  if (col >= H) return;
  const int r0 = blockIdx.x * kRowsPerPart;
  float s = 0.0f;
  for (int r = r0; r < r0 + kRowsPerPart && r < cnt; ++r) {
    const int64_t o = (int64_t)r * H + col;
    const float hv = __bfloat162float(h[o]);
    const __nv_bfloat16 d = __float2bfloat16_rn(dh[o] * (1.0f - hv * hv));
    da[o] = d;
    s += __bfloat162float(d);
  }
  part[(int64_t)blockIdx.x * H + col] = s;
}

struct AssembleArgs {
  float* grad;
  const float* db2p[2];    // [nrb][H] per net
  const float* db1p[2];
  const float* w3g[2];     // [16][H] head weight gradients (padded)
  const float* lossp;      // [nlb][32]
  double* stat5;           // [5] minibatch loss statistics out
  int nrb, nlb, H, A;
  int64_t ob1[2], ob2[2], ob3[2], ow3[2];
};

// bias gradients: one warp per bias element sums its column of partials
// (lane-strided, then a fixed shuffle tree: deterministic); the head weight
// gradients are copied out of their padded 16-row buffers
__global__ void assemble_kernel(AssembleArgs a) {
  const int warp = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  const int nb = 2 * a.H + kHead;  // bias elements per net: b2, b1, b3 (padded)
  if (warp >= 2 * nb && warp < 2 * nb + 5) {
    // minibatch loss statistics (pg, entropy, kl, clip, value) for the Adam kernel
    const int k = warp - 2 * nb;
    double s = 0.0;
    for (int b = lane; b < a.nlb; b += 32) s += (double)a.lossp[(int64_t)b * kPartW + k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) a.stat5[k] = s;
  }
  if (warp < 2 * nb) {
    const int net = warp / nb, j = warp % nb;
    const int nout = net ? 1 : a.A;
    float s = 0.0f;
    if (j < 2 * a.H) {
      const float* src = j < a.H ? a.db2p[net] + j : a.db1p[net] + (j - a.H);
      for (int b = lane; b < a.nrb; b += 32) s += src[(int64_t)b * a.H];
    } else if (j - 2 * a.H < nout) {
      const int col = net ? 21 : 5 + (j - 2 * a.H);
      for (int b = lane; b < a.nlb; b += 32) s += a.lossp[(int64_t)b * kPartW + col];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) {
      if (j < a.H) a.grad[a.ob2[net] + j] = s;
      else if (j < 2 * a.H) a.grad[a.ob1[net] + (j - a.H)] = s;
      else if (j - 2 * a.H < nout) a.grad[a.ob3[net] + (j - 2 * a.H)] = s;
    }
  }
  // head weights: threads of the whole grid stride over 2 x 16 x H entries
  const int64_t tid = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t per = (int64_t)kHead * a.H;
  for (int64_t i = tid; i < 2 * per; i += (int64_t)gridDim.x * blockDim.x) {
    const int net = (int)(i / per);
    const int64_t q = i % per;
    const int r = (int)(q / a.H);
    if (r < (net ? 1 : a.A)) a.grad[a.ow3[net] + q] = a.w3g[net][q];
  }
}

// fp32 sums of squares over 256 fixed blocks (fixed order: deterministic)
__global__ void sumsq_kernel(const float* __restrict__ g, int64_t P, float* __restrict__ sq) {
  __shared__ float red[32];
  float s = 0.0f;
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x)
    s = fmaf(g[p], g[p], s);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    sq[blockIdx.x] = t;
  }
}

struct AdamBf16Args {
  float* params;
  float* m;
  float* v;
  const float* grad;
  const float* sq;
  int nsq;
  int64_t P;
  float beta1, beta2, step_size, inv_sqrt_bc2, eps, max_norm, vf_coef, ent_coef, inv_cnt;
  const double* stat5;
  double* acc;
};

__global__ void adam_bf16_kernel(AdamBf16Args a) {
  __shared__ float s_norm;
  if (threadIdx.x < 32) {
    float t = 0.0f;
    for (int b = threadIdx.x; b < a.nsq; b += 32) t += a.sq[b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0) s_norm = sqrtf(t);
  }
  __syncthreads();
  const float norm = s_norm;
  const float coef = fminf(1.0f, a.max_norm / (norm + 1e-6f));
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < a.P; p += (int64_t)gridDim.x * blockDim.x) {
    const float gp = a.grad[p] * coef;
    const float mp = a.beta1 * a.m[p] + (1.0f - a.beta1) * gp;
    const float vp = a.beta2 * a.v[p] + (1.0f - a.beta2) * gp * gp;
    a.m[p] = mp;
    a.v[p] = vp;
    a.params[p] -= a.step_size * mp / (sqrtf(vp) * a.inv_sqrt_bc2 + a.eps);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    double v5[5];
    for (int k = 0; k < 5; ++k) v5[k] = a.stat5[k];
    const double ic = a.inv_cnt;
    a.acc[0] += v5[0] * ic;
    a.acc[1] += v5[4] * ic;
    a.acc[2] += v5[1] * ic;
    a.acc[3] += v5[2] * ic;
    a.acc[4] += v5[3] * ic;
    a.acc[5] += v5[0] * ic + a.vf_coef * v5[4] * ic - a.ent_coef * v5[1] * ic;
    a.acc[6] = norm;
    a.acc[7] += 1.0;
  }
}

__global__ void finalize_bf16_kernel(const double* __restrict__ acc, const int32_t* __restrict__ err,
                                     float* __restrict__ stats) {
  const int k = threadIdx.x;
  if (k < 8) {
    const double n = acc[7] > 0 ? acc[7] : 1.0;
    stats[k] = (float)(k < 6 ? acc[k] / n : acc[k]);
    if (k == 7 && *err) stats[7] = -1.0f;
  }
}

// ---------------------------------------------------------------------------
// workspace plan
// ---------------------------------------------------------------------------
struct Bf16Plan {
  int64_t P, N;
  int nmb, mb, D, H, A, nrb, nlb, nsq;
  int64_t img;
  int64_t o_adv, o_idx, o_img, o_wb, o_x, o_h[4], o_zp, o_zv, o_dz[2], o_dh, o_da2, o_da1, o_db2[2], o_db1[2],
      o_w3g[2], o_loss, o_grad, o_sq, o_acc, o_stat5, o_lt, total;
};

static int64_t al(int64_t x) { return (x + 1023) / 1024 * 1024; }

static Bf16Plan bf16_plan(const pe_net& net, const pe_ppo_config& cfg, int64_t N) {
  Bf16Plan p;
  p.D = net.obs_dim;
  p.H = net.hidden;
  p.A = net.n_actions;
  p.P = mlp_layout(p.D, p.H, p.A).total;
  p.N = N;
  p.mb = (int)std::min<int64_t>(cfg.minibatch, N);
  p.nmb = (int)((N + cfg.minibatch - 1) / cfg.minibatch);
  p.nrb = (p.mb + kRowsPerPart - 1) / kRowsPerPart;
  p.nlb = (p.mb + kLossThreads - 1) / kLossThreads;
  p.nsq = 256;
  p.img = bf16_image_bytes(net);
  const int64_t mb = p.mb, H = p.H;
  int64_t o = 0;
  p.o_adv = o; o = al(o + (int64_t)cfg.epochs * p.nmb * 8);
  p.o_idx = o; o = al(o + mb * 4);
  p.o_img = o; o = al(o + 2 * p.img);
  p.o_wb = o; o = al(o + 2 * (H * H + kHead * H) * 2);
  p.o_x = o; o = al(o + mb * p.D * 2);
  for (int i = 0; i < 4; ++i) { p.o_h[i] = o; o = al(o + mb * H * 2); }
  p.o_zp = o; o = al(o + mb * kHead * 4);
  p.o_zv = o; o = al(o + mb * 4);
  for (int i = 0; i < 2; ++i) { p.o_dz[i] = o; o = al(o + mb * kHead * 2); }
  p.o_dh = o; o = al(o + mb * H * 4);
  p.o_da2 = o; o = al(o + mb * H * 2);
  p.o_da1 = o; o = al(o + mb * H * 2);
  for (int i = 0; i < 2; ++i) { p.o_db2[i] = o; o = al(o + (int64_t)p.nrb * H * 4); }
  for (int i = 0; i < 2; ++i) { p.o_db1[i] = o; o = al(o + (int64_t)p.nrb * H * 4); }
  for (int i = 0; i < 2; ++i) { p.o_w3g[i] = o; o = al(o + kHead * H * 4); }
  p.o_loss = o; o = al(o + (int64_t)p.nlb * kPartW * 4);
  p.o_grad = o; o = al(o + p.P * 4);
  p.o_sq = o; o = al(o + (int64_t)p.nsq * 8);
  p.o_acc = o; o = al(o + 8 * 8 + 8);
  p.o_stat5 = o; o = al(o + 5 * 8);
  p.o_lt = o; o = al(o + kLtWorkspace);
  p.total = o;
  return p;
}

int64_t ppo_ws_bytes_bf16(const pe_net& net, const pe_ppo_config& cfg, int64_t N) {
  if (bf16_image_bytes(net) < 0) return -1;
  return bf16_plan(net, cfg, N).total;
}

pe_status ppo_update_bf16(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                          const void* obs, const uint8_t* act, const float* logp_old, const float* adv,
                          const float* ret, int64_t N, const pe_ppo_config& cfg, float* stats, void* wsv,
                          cudaStream_t st) {
  if (bf16_image_bytes(net) < 0 || net.n_actions > kHead)
    return fail(PE_EINVAL, "unsupported bf16 PPO network (D=%d H=%d A=%d)", net.obs_dim, net.hidden, net.n_actions);
  const Bf16Plan pl = bf16_plan(net, cfg, N);
  char* ws = reinterpret_cast<char*>(wsv);
  auto at = [&](int64_t off) { return ws + off; };
  float2* advstat = reinterpret_cast<float2*>(at(pl.o_adv));
  uint32_t* idx = reinterpret_cast<uint32_t*>(at(pl.o_idx));
  uint8_t* img = reinterpret_cast<uint8_t*>(at(pl.o_img));
  __nv_bfloat16* wb = reinterpret_cast<__nv_bfloat16*>(at(pl.o_wb));
  __nv_bfloat16* x = reinterpret_cast<__nv_bfloat16*>(at(pl.o_x));
  __nv_bfloat16* h[4];
  for (int i = 0; i < 4; ++i) h[i] = reinterpret_cast<__nv_bfloat16*>(at(pl.o_h[i]));
  float* zp = reinterpret_cast<float*>(at(pl.o_zp));
  float* zv = reinterpret_cast<float*>(at(pl.o_zv));
  __nv_bfloat16* dz[2] = {reinterpret_cast<__nv_bfloat16*>(at(pl.o_dz[0])), reinterpret_cast<__nv_bfloat16*>(at(pl.o_dz[1]))};
  float* dh = reinterpret_cast<float*>(at(pl.o_dh));
  __nv_bfloat16* da2 = reinterpret_cast<__nv_bfloat16*>(at(pl.o_da2));
  __nv_bfloat16* da1 = reinterpret_cast<__nv_bfloat16*>(at(pl.o_da1));
  float* db2[2] = {reinterpret_cast<float*>(at(pl.o_db2[0])), reinterpret_cast<float*>(at(pl.o_db2[1]))};
  float* db1[2] = {reinterpret_cast<float*>(at(pl.o_db1[0])), reinterpret_cast<float*>(at(pl.o_db1[1]))};
  float* w3g[2] = {reinterpret_cast<float*>(at(pl.o_w3g[0])), reinterpret_cast<float*>(at(pl.o_w3g[1]))};
  float* lossp = reinterpret_cast<float*>(at(pl.o_loss));
  float* grad = reinterpret_cast<float*>(at(pl.o_grad));
  float* sq = reinterpret_cast<float*>(at(pl.o_sq));
  double* acc = reinterpret_cast<double*>(at(pl.o_acc));
  int32_t* err = reinterpret_cast<int32_t*>(acc + 8);
  double* stat5 = reinterpret_cast<double*>(at(pl.o_stat5));
  void* lt_ws = at(pl.o_lt);
  const int D = pl.D, H = pl.H, A = pl.A;
  const MlpLayout Lp = mlp_layout(D, H, A);
  PE_TRY_CUDA(cudaMemsetAsync(acc, 0, 8 * 8 + 8, st));
  pe_status s = launch_advstats(adv, N, cfg.minibatch, pl.nmb, cfg.epochs, cfg.seed, cfg.iteration, advstat, st);
  if (s != PE_OK) return s;
  const __nv_bfloat16* wb2[2] = {wb, wb + (int64_t)H * H + kHead * H};
  const __nv_bfloat16* wb3[2] = {wb + (int64_t)H * H, wb + (int64_t)H * H + kHead * H + (int64_t)H * H};
  int64_t t = adam_t;
  for (int ep = 0; ep < cfg.epochs; ++ep) {
    const Feistel f = make_feistel((uint64_t)N, cfg.seed, ep, cfg.iteration);
    for (int mbi = 0; mbi < pl.nmb; ++mbi) {
      const int64_t start = (int64_t)mbi * cfg.minibatch;
      const int cnt = (int)std::min<int64_t>(cfg.minibatch, N - start);
      {
        ProfScope ps(PE_PROF_PPO_OTHER, st);
        perm_index_kernel<<<ceil_div(cnt, 256), 256, 0, st>>>(f, start, cnt, idx);
        backward_weights_kernel<<<256, 256, 0, st>>>(params, D, H, A, wb);
      }
      PE_CHECK_LAUNCH("perm_index/backward_weights");
      s = bf16_make_images(net, params, img, st);
      if (s != PE_OK) return s;
      s = bf16_forward_save(net, img, params, 0, obs, idx, cnt, zp, kHead, x, h[0], h[1], err, st);
      if (s != PE_OK) return s;
      s = bf16_forward_save(net, img + pl.img, params, 1, obs, idx, cnt, zv, 1, nullptr, h[2], h[3], err, st);
      if (s != PE_OK) return s;
      LossArgs la;
      la.zp = zp;
      la.zv = zv;
      la.idx = idx;
      la.act = act;
      la.logp_old = logp_old;
      la.adv = adv;
      la.ret = ret;
      la.advstat = advstat + (int64_t)ep * pl.nmb + mbi;
      la.cnt = cnt;
      la.A = A;
      la.clip = cfg.clip;
      la.vf_coef = cfg.vf_coef;
      la.ent_coef = cfg.ent_coef;
      la.inv_cnt = 1.0f / (float)cnt;
      la.dzp = dz[0];
      la.dzv = dz[1];
      la.part = lossp;
      const int nlb = ceil_div(cnt, kLossThreads), nrb = ceil_div(cnt, kRowsPerPart);
      {
        ProfScope ps(PE_PROF_PPO_OTHER, st);
        ppo_bf16_loss_kernel<<<nlb, kLossThreads, 0, st>>>(la);
      }
      PE_CHECK_LAUNCH("ppo_bf16_loss_kernel");
      for (int net_i = 0; net_i < 2; ++net_i) {
        const __nv_bfloat16* h1 = h[2 * net_i];
        const __nv_bfloat16* h2 = h[2 * net_i + 1];
        float* g = grad;
        ProfScope ps(PE_PROF_PPO_GRAD, st);
        // dh2 = dz W3   [cnt x H], K = 16
        s = gemm_bf16(cnt, H, kHead, dz[net_i], kHead, false, wb3[net_i], H, false, dh, H, lt_ws, st);
        if (s != PE_OK) return s;
        bwd_act_kernel<<<dim3(nrb, ceil_div(H, 256)), 256, 0, st>>>(dh, h2, cnt, H, da2, db2[net_i]);
        // dW2 = da2^T h1   [H x H], K = cnt
        s = gemm_bf16(H, H, cnt, da2, H, true, h1, H, false, g + (net_i ? Lp.v2 : Lp.w2), H, lt_ws, st);
        if (s != PE_OK) return s;
        // dh1 = da2 W2   [cnt x H], K = H
        s = gemm_bf16(cnt, H, H, da2, H, false, wb2[net_i], H, false, dh, H, lt_ws, st);
        if (s != PE_OK) return s;
        bwd_act_kernel<<<dim3(nrb, ceil_div(H, 256)), 256, 0, st>>>(dh, h1, cnt, H, da1, db1[net_i]);
        // dW1 = da1^T x   [H x D], K = cnt
        s = gemm_bf16(H, D, cnt, da1, H, true, x, D, false, g + (net_i ? Lp.v1 : Lp.w1), D, lt_ws, st);
        if (s != PE_OK) return s;
        // dW3 (16 padded rows) = dz^T h2   [16 x H], K = cnt
        s = gemm_bf16(kHead, H, cnt, dz[net_i], kHead, true, h2, H, false, w3g[net_i], H, lt_ws, st);
        if (s != PE_OK) return s;
      }
      PE_CHECK_LAUNCH("bwd_act_kernel");
      AssembleArgs aa;
      aa.grad = grad;
      for (int i = 0; i < 2; ++i) {
        aa.db2p[i] = db2[i];
        aa.db1p[i] = db1[i];
        aa.w3g[i] = w3g[i];
      }
      aa.lossp = lossp;
      aa.stat5 = stat5;
      aa.nrb = nrb;
      aa.nlb = nlb;
      aa.H = H;
      aa.A = A;
      aa.ob1[0] = Lp.b1; aa.ob1[1] = Lp.c1;
      aa.ob2[0] = Lp.b2; aa.ob2[1] = Lp.c2;
      aa.ob3[0] = Lp.b3; aa.ob3[1] = Lp.c3;
      aa.ow3[0] = Lp.w3; aa.ow3[1] = Lp.v3;
      const int asm_warps = 2 * (2 * H + kHead) + 5;
      t += 1;
      AdamBf16Args ad;
      ad.params = params;
      ad.m = m;
      ad.v = v;
      ad.grad = grad;
      ad.sq = sq;
      ad.nsq = pl.nsq;
      ad.P = pl.P;
      ad.beta1 = cfg.beta1;
      ad.beta2 = cfg.beta2;
      ad.step_size = (float)(cfg.lr / (1.0 - std::pow((double)cfg.beta1, (double)t)));
      ad.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(1.0 - std::pow((double)cfg.beta2, (double)t)));
      ad.eps = cfg.eps;
      ad.max_norm = cfg.max_grad_norm;
      ad.vf_coef = cfg.vf_coef;
      ad.ent_coef = cfg.ent_coef;
      ad.inv_cnt = 1.0f / (float)cnt;
      ad.stat5 = stat5;
      ad.acc = acc;
      {
        ProfScope ps(PE_PROF_PPO_ADAM, st);
        assemble_kernel<<<ceil_div(asm_warps * 32, 256), 256, 0, st>>>(aa);
        sumsq_kernel<<<pl.nsq, 256, 0, st>>>(grad, pl.P, sq);
        adam_bf16_kernel<<<ceil_div(pl.P, 256), 256, 0, st>>>(ad);
      }
      PE_CHECK_LAUNCH("ppo bf16 step kernels");
    }
  }
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    finalize_bf16_kernel<<<1, 32, 0, st>>>(acc, err, stats);
  }
  PE_CHECK_LAUNCH("finalize_bf16_kernel");
  return PE_OK;
}

}  // namespace pe
