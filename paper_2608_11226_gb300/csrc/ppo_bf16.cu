// PPO update for bf16 networks (72B: 32-256-256x16, Stress: 64-512-512x16;
// Sec. 4.2 loss and optimiser as in the fp32 update).
//
// Per minibatch:
//   forward   -- the tcgen05 tensor-core MLP kernels over the minibatch's
//                Feistel-permuted rows, saving x, h1, h2 (bf16) as 128-row
//                tile images (the kernels' swizzled shared-memory layout)
//                besides the heads;
//   loss      -- in the forward kernels' head epilogue, one thread per
//                sample: clipped surrogate, value loss, entropy; dLoss/dhead
//                in fp32, rounded to bf16 into dz tile images (zero rows past
//                the minibatch), fixed-order per-warp partials of the
//                head-bias gradients and the statistics;
//   backward  -- on the tensor cores (bwd_bf16.cu): per network the data
//                products and tanh derivatives (da2, da1), then the weight
//                and hidden-bias gradients split over samples with a
//                fixed-order reduction into the canonical gradient vector;
//                for the 72B networks the forward, the loss and the data
//                products of a network run as one kernel (fused_bf16.cu);
//   step      -- the gradient's squared norm (summed with the weight
//                gradients' reduction), clip, Adam on the fp32 master
//                parameters, which also writes the updated weights into the
//                bf16 weight images (built once per call).
// Rounding points (which the oracle reproduces): dz, da2 and da1 enter the
// products as bf16; the layer bias gradients sum the rounded values, the head
// bias gradient the fp32 dz.
#include <cuda_bf16.h>

#include <cmath>

#include "bf16_layout.cuh"
#include "mlp_f32.cuh"

namespace pe {

// defined in mlp_bf16.cu / ppo_f32.cu / bwd_bf16.cu
int64_t bf16_image_bytes(const pe_net& net);
pe_status bf16_make_images(const pe_net& net, const float* params, uint8_t* two_images, cudaStream_t st);
pe_status bf16_forward_loss(const pe_net& net, const uint8_t* img, const float* params, const void* obs,
                            const uint32_t* gather, int64_t n, const PpoHead& lp, const PpoHead& lv,
                            __nv_bfloat16* x, __nv_bfloat16* const h[4], int32_t* err, cudaStream_t st);
pe_status launch_advstats(const float* adv, int64_t N, int M, int nmb, int epochs, uint64_t seed,
                          uint32_t iteration, float2* out, cudaStream_t st);
int64_t bwd_image_bytes(int H);
int64_t wgrad_partial_bytes();
pe_status bf16_backward(const pe_net& net, const float* params, uint8_t* const img[2], const uint8_t* x,
                        const uint8_t* const dz[2], const uint8_t* const h1[2], const uint8_t* const h2[2],
                        uint8_t* const da2[2], uint8_t* const da1[2], int64_t n, float* part, float* grad,
                        const float* lossp, int nlb, double* stat5, float* sq, int32_t* err, bool data_done,
                        cudaStream_t st);
pe_status bf16_bwd_images(const pe_net& net, const float* params, uint8_t* const img[2], cudaStream_t st);
// defined in fused_bf16.cu
bool bf16_fused_supported(const pe_net& net);
pe_status bf16_fused_fwd_bwd(const pe_net& net, const uint8_t* img, const uint8_t* bimg, const float* params,
                             int value_net, const void* obs, const uint32_t* gather, int64_t n, const PpoHead& loss,
                             __nv_bfloat16* x, __nv_bfloat16* h1, __nv_bfloat16* h2, uint8_t* da2, uint8_t* da1,
                             int32_t* err, cudaStream_t st);
int wgrad_reduce_blocks();

constexpr int kHead = 16;   // head rows (logits; the value head padded with zero rows)
constexpr int kTile = 128;  // rows of a tile image

// ---------------------------------------------------------------------------
// kernels
// ---------------------------------------------------------------------------
__global__ void perm_index_kernel(Feistel f, int64_t start, int cnt, uint32_t* __restrict__ idx) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j < cnt) idx[j] = feistel_index(f, start + j);
}

constexpr int kPartW = 32;  // partial row of the fused loss: pg, ent, kl, clip, vl, db3[16], dc3

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
  int A;                // policy actions
  uint8_t* fimg;        // forward weight images of both networks (fstride apart)
  int64_t fstride;
  uint8_t* bimg[2];     // backward weight images (policy, value)
  Feistel nf;           // the next minibatch step's permutation ...
  int64_t nstart;       // ... and its first position
  int ncnt;             // its sample count (0: no next step)
  uint32_t* idx;        // out: its gather indices
};

// Clip and Adam on the fp32 master parameters, writing every updated weight's
// bf16 copy straight into the forward and backward weight images (the next
// minibatch step's operands), so that the images need no rebuild per step;
// the conversion is the image kernels' own (round to nearest even).  The same
// launch writes the next minibatch step's Feistel gather indices (the current
// step's kernels, which read them, have finished).
template <int D, int H>
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
    const float pn = a.params[p] - a.step_size * mp / (sqrtf(vp) * a.inv_sqrt_bc2 + a.eps);
    a.params[p] = pn;
    // the weight's place in the images: network, layer, row, column
    const MlpLayout L = mlp_layout(D, H, a.A);
    int net = -1, mat = 0;
    int64_t q = 0;
    if (p < L.b1) net = 0, mat = 1, q = p - L.w1;
    else if (p >= L.w2 && p < L.b2) net = 0, mat = 2, q = p - L.w2;
    else if (p >= L.w3 && p < L.b3) net = 0, mat = 3, q = p - L.w3;
    else if (p >= L.v1 && p < L.c1) net = 1, mat = 1, q = p - L.v1;
    else if (p >= L.v2 && p < L.c2) net = 1, mat = 2, q = p - L.v2;
    else if (p >= L.v3 && p < L.c3) net = 1, mat = 3, q = p - L.v3;
    if (net >= 0) {
      const int cols = mat == 1 ? D : H;
      const int r = (int)(q / cols), k = (int)(q % cols);
      const __nv_bfloat16 b = __float2bfloat16_rn(pn);
      *reinterpret_cast<__nv_bfloat16*>(a.fimg + net * a.fstride + fwd_img_offset<D, H>(mat, r, k)) = b;
      if (mat >= 2) *reinterpret_cast<__nv_bfloat16*>(a.bimg[net] + bwd_img_offset<H>(mat, r, k)) = b;
    }
  }
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < a.ncnt; j += (int64_t)gridDim.x * blockDim.x)
    a.idx[j] = feistel_index(a.nf, a.nstart + j);
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
  int nmb, mb, rows, D, H, A, nlb, nsq;
  int64_t img, bimg;
  int64_t o_adv, o_idx, o_img, o_bimg, o_x, o_h[4], o_dz[2], o_da2[2], o_da1[2], o_part, o_loss,
      o_grad, o_sq, o_acc, o_stat5, total;
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
  p.rows = (p.mb + kTile - 1) / kTile * kTile;
  p.nmb = (int)((N + cfg.minibatch - 1) / cfg.minibatch);
  p.nlb = p.rows / kTile * 4;  // one partial row per head warp (4 per tile)
  p.nsq = wgrad_reduce_blocks();
  p.img = bf16_image_bytes(net);
  p.bimg = al(bwd_image_bytes(p.H));
  const int64_t rows = p.rows, H = p.H;
  int64_t o = 0;
  p.o_adv = o; o = al(o + (int64_t)cfg.epochs * p.nmb * 8);
  p.o_idx = o; o = al(o + rows * 4);
  p.o_img = o; o = al(o + 2 * p.img);
  p.o_bimg = o; o = al(o + 2 * p.bimg);
  p.o_x = o; o = al(o + rows * p.D * 2);
  for (int i = 0; i < 4; ++i) { p.o_h[i] = o; o = al(o + rows * H * 2); }
  for (int i = 0; i < 2; ++i) { p.o_dz[i] = o; o = al(o + rows * 32); }
  for (int i = 0; i < 2; ++i) { p.o_da2[i] = o; o = al(o + rows * H * 2); }
  for (int i = 0; i < 2; ++i) { p.o_da1[i] = o; o = al(o + rows * H * 2); }
  p.o_part = o; o = al(o + wgrad_partial_bytes());
  p.o_loss = o; o = al(o + (int64_t)p.nlb * kPartW * 4);
  p.o_grad = o; o = al(o + p.P * 4);
  p.o_sq = o; o = al(o + (int64_t)p.nsq * 8);
  p.o_acc = o; o = al(o + 8 * 8 + 8);
  p.o_stat5 = o; o = al(o + 5 * 8);
  p.total = o;
  return p;
}

int64_t ppo_ws_bytes_bf16(const pe_net& net, const pe_ppo_config& cfg, int64_t N) {
  if (bf16_image_bytes(net) < 0 || bwd_image_bytes(net.hidden) < 0) return -1;
  return bf16_plan(net, cfg, N).total;
}

pe_status ppo_update_bf16(const pe_net& net, float* params, float* m, float* v, int64_t adam_t,
                          const void* obs, const uint8_t* act, const float* logp_old, const float* adv,
                          const float* ret, int64_t N, const pe_ppo_config& cfg, float* stats, void* wsv,
                          cudaStream_t st) {
  if (bf16_image_bytes(net) < 0 || bwd_image_bytes(net.hidden) < 0 || net.n_actions > kHead)
    return fail(PE_EINVAL, "unsupported bf16 PPO network (D=%d H=%d A=%d)", net.obs_dim, net.hidden, net.n_actions);
  const Bf16Plan pl = bf16_plan(net, cfg, N);
  char* ws = reinterpret_cast<char*>(wsv);
  auto at = [&](int64_t off) { return ws + off; };
  auto u8 = [&](int64_t off) { return reinterpret_cast<uint8_t*>(ws + off); };
  float2* advstat = reinterpret_cast<float2*>(at(pl.o_adv));
  uint32_t* idx = reinterpret_cast<uint32_t*>(at(pl.o_idx));
  uint8_t* img = u8(pl.o_img);
  uint8_t* const bimg[2] = {u8(pl.o_bimg), u8(pl.o_bimg + pl.bimg)};
  __nv_bfloat16* x = reinterpret_cast<__nv_bfloat16*>(at(pl.o_x));
  __nv_bfloat16* h[4];
  for (int i = 0; i < 4; ++i) h[i] = reinterpret_cast<__nv_bfloat16*>(at(pl.o_h[i]));
  uint8_t* const dz[2] = {u8(pl.o_dz[0]), u8(pl.o_dz[1])};
  uint8_t* const da2[2] = {u8(pl.o_da2[0]), u8(pl.o_da2[1])};
  uint8_t* const da1[2] = {u8(pl.o_da1[0]), u8(pl.o_da1[1])};
  const uint8_t* const dzc[2] = {dz[0], dz[1]};
  const uint8_t* const h1c[2] = {u8(pl.o_h[0]), u8(pl.o_h[2])};
  const uint8_t* const h2c[2] = {u8(pl.o_h[1]), u8(pl.o_h[3])};
  float* part = reinterpret_cast<float*>(at(pl.o_part));
  float* lossp = reinterpret_cast<float*>(at(pl.o_loss));
  float* grad = reinterpret_cast<float*>(at(pl.o_grad));
  float* sq = reinterpret_cast<float*>(at(pl.o_sq));
  double* acc = reinterpret_cast<double*>(at(pl.o_acc));
  int32_t* err = reinterpret_cast<int32_t*>(acc + 8);
  double* stat5 = reinterpret_cast<double*>(at(pl.o_stat5));
  const int A = pl.A;
  PE_TRY_CUDA(cudaMemsetAsync(acc, 0, 8 * 8 + 8, st));
  pe_status s = launch_advstats(adv, N, cfg.minibatch, pl.nmb, cfg.epochs, cfg.seed, cfg.iteration, advstat, st);
  if (s != PE_OK) return s;
  int64_t t = adam_t;
  const bool fused = bf16_fused_supported(net);
  // the bf16 weight images of both networks, built once; each Adam step
  // writes its updated weights into them
  s = bf16_make_images(net, params, img, st);
  if (s == PE_OK) s = bf16_bwd_images(net, params, bimg, st);
  if (s != PE_OK) return s;
  // the first minibatch step's gather indices; each Adam launch writes the next step's
  auto mb_count = [&](int mbi) { return (int)std::min<int64_t>(cfg.minibatch, N - (int64_t)mbi * cfg.minibatch); };
  if (cfg.epochs > 0 && pl.nmb > 0) {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    perm_index_kernel<<<ceil_div(mb_count(0), 256), 256, 0, st>>>(
        make_feistel((uint64_t)N, cfg.seed, 0, cfg.iteration), 0, mb_count(0), idx);
  }
  PE_CHECK_LAUNCH("perm_index_kernel");
  for (int ep = 0; ep < cfg.epochs; ++ep) {
    for (int mbi = 0; mbi < pl.nmb; ++mbi) {
      const int64_t start = (int64_t)mbi * cfg.minibatch;
      const int cnt = mb_count(mbi);
      const int rows = (cnt + kTile - 1) / kTile * kTile;
      // the step after this one (the next minibatch, or the next epoch's first)
      const bool last_mb = mbi + 1 == pl.nmb;
      const int nep = last_mb ? ep + 1 : ep, nmbi = last_mb ? 0 : mbi + 1;
      PpoHead lh;
      lh.act = act;
      lh.logp_old = logp_old;
      lh.adv = adv;
      lh.ret = ret;
      lh.advstat = advstat + (int64_t)ep * pl.nmb + mbi;
      lh.clip = cfg.clip;
      lh.vf_coef = cfg.vf_coef;
      lh.ent_coef = cfg.ent_coef;
      lh.inv_cnt = 1.0f / (float)cnt;
      lh.part = lossp;
      if (fused) {
        // 72B: forward, loss and backward data products of a network in one
        // kernel (its backward images first)
        lh.dz = dz[0];
        s = bf16_fused_fwd_bwd(net, img, bimg[0], params, 0, obs, idx, cnt, lh, x, h[0], h[1], da2[0], da1[0], err,
                               st);
        if (s != PE_OK) return s;
        lh.dz = dz[1];
        s = bf16_fused_fwd_bwd(net, img + pl.img, bimg[1], params, 1, obs, idx, cnt, lh, nullptr, h[2], h[3], da2[1],
                               da1[1], err, st);
      } else {
        // Stress: forward and loss of both networks in one launch
        PpoHead lv = lh;
        lh.dz = dz[0];
        lv.dz = dz[1];
        s = bf16_forward_loss(net, img, params, obs, idx, cnt, lh, lv, x, h, err, st);
      }
      if (s != PE_OK) return s;
      const int nlb = rows / kTile * 4;
      s = bf16_backward(net, params, bimg, reinterpret_cast<const uint8_t*>(x), dzc, h1c, h2c, da2, da1, cnt, part,
                        grad, lossp, nlb, stat5, sq, err, fused, st);
      if (s != PE_OK) return s;
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
      ad.A = A;
      ad.fimg = img;
      ad.fstride = pl.img;
      ad.bimg[0] = bimg[0];
      ad.bimg[1] = bimg[1];
      ad.idx = idx;
      ad.ncnt = nep < cfg.epochs ? mb_count(nmbi) : 0;
      ad.nstart = (int64_t)nmbi * cfg.minibatch;
      ad.nf = make_feistel((uint64_t)N, cfg.seed, (uint32_t)(nep < cfg.epochs ? nep : 0), cfg.iteration);
      {
        ProfScope ps(PE_PROF_PPO_ADAM, st);
        if (pl.D == 32 && pl.H == 256)
          adam_bf16_kernel<32, 256><<<ceil_div(pl.P, 256), 256, 0, st>>>(ad);
        else
          adam_bf16_kernel<64, 512><<<ceil_div(pl.P, 256), 256, 0, st>>>(ad);
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
