// Layouts and helpers shared by the bf16 tensor-core kernels (the forward
// MLPs, the backward data and weight-gradient kernels, and the fused PPO
// forward-backward kernel): the forward-pass extras of the PPO update, the
// head epilogue that computes the PPO loss, the forward and backward weight
// images, and the tanh-derivative step.
#pragma once

#include "common.cuh"
#include "tc.cuh"

namespace pe {

// optional extras of a forward pass used by the PPO update: rows gathered
// through an index array, and the bf16 input and hidden activations saved for
// the backward pass as "tile images": tile t (rows 128 t .. 128 t + 127) is
// stored exactly as the kernel holds it in shared memory (K-major, swizzled:
// x with 64- or 128-byte rows, h1 and h2 with 128-byte rows in H / 64
// blocks), all 128 rows written (rows past n hold the finite activations of
// a zero input), so that the backward kernels bulk-copy them as operands.
struct MlpSave {
  const uint32_t* gather;  // row r of the tile reads obs row gather[r] (NULL: row r)
  __nv_bfloat16* x;        // tiles of 128 x D, or NULL
  __nv_bfloat16* h1;       // tiles of 128 x H, or NULL
  __nv_bfloat16* h2;       // tiles of 128 x H, or NULL
  PpoHead loss;            // loss.dz != NULL: the PPO loss replaces the head output
};

constexpr int kTcRows = 128;     // rows (envs / samples) per tile, the MMA M
constexpr int kTcThreads = 512;  // 16 warps: 4 TMEM lane quadrants x 4 column slices
constexpr int kHeadN = 16;       // head width (logits or value padded to 16)

// Head epilogue of a PPO forward pass for row `row` (0..127) of tile `tile`:
// z[16] are the head accumulators of the row (before the bias).  Called by
// all 32 lanes of a head warp (warp < 4); rows past n contribute zero.  The
// dz row goes to the tile image and, when dz_smem is given, to the same
// place of a shared-memory copy of the tile.
__device__ __forceinline__ void ppo_head_row(const PpoHead& L, int value_net, int A, const float* b3,
                                             const uint32_t* gather, int64_t tile, int row, int64_t n,
                                             const float (&acc)[16], int warp, uint8_t* dz_smem = nullptr) {
  constexpr int kW = 32;
  const int64_t j = tile * kTcRows + row;
  const bool valid = j < n;
  float v[22];
#pragma unroll
  for (int k = 0; k < 22; ++k) v[k] = 0.0f;
  uint32_t pk[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (valid) {
    const uint32_t i = gather[j];
    if (!value_net) {
      const float2 as = *L.advstat;
      float z[kHeadN];
#pragma unroll
      for (int a = 0; a < kHeadN; ++a) z[a] = a < A ? acc[a] + b3[a] : -INFINITY;
      float m = z[0];
#pragma unroll
      for (int a = 1; a < kHeadN; ++a) m = fmaxf(m, z[a]);
      float se = 0.0f;
#pragma unroll
      for (int a = 0; a < kHeadN; ++a) se += a < A ? expf(z[a] - m) : 0.0f;
      const float lse = m + logf(se);
      float lp[kHeadN], pr[kHeadN], Hs = 0.0f;
#pragma unroll
      for (int a = 0; a < kHeadN; ++a) {
        lp[a] = a < A ? z[a] - lse : 0.0f;
        pr[a] = a < A ? expf(lp[a]) : 0.0f;
        Hs -= pr[a] * lp[a];
      }
      const int act = L.act[i];
      const float an = (L.adv[i] - as.x) * as.y;
      float lpa = 0.0f;
#pragma unroll
      for (int a = 0; a < kHeadN; ++a)
        if (a == act) lpa = lp[a];
      const float logr = lpa - L.logp_old[i];
      const float rho = expf(logr);
      const float rc = fminf(fmaxf(rho, 1.0f - L.clip), 1.0f + L.clip);
      const float s1 = rho * an, s2 = rc * an;
      v[0] = -fminf(s1, s2);
      v[1] = Hs;
      v[2] = kl_term(logr);
      v[3] = fabsf(rho - 1.0f) > L.clip ? 1.0f : 0.0f;
      const float dlp = (s1 <= s2 ? -an : 0.0f) * rho * L.inv_cnt;
#pragma unroll
      for (int a = 0; a < kHeadN; a += 2) {
        float d0 = 0.0f, d1 = 0.0f;
        if (a < A) d0 = dlp * ((a == act ? 1.0f : 0.0f) - pr[a]) + L.ent_coef * L.inv_cnt * pr[a] * (lp[a] + Hs);
        if (a + 1 < A)
          d1 = dlp * ((a + 1 == act ? 1.0f : 0.0f) - pr[a + 1]) + L.ent_coef * L.inv_cnt * pr[a + 1] * (lp[a + 1] + Hs);
        v[5 + a] = d0;
        v[5 + a + 1] = d1;
        pk[a / 2] = tc::pack_bf16(d0, d1);
      }
    } else {
      const float V = acc[0] + b3[0], R = L.ret[i];
      v[4] = (R - V) * (R - V);
      const float dV = L.vf_coef * 2.0f * (V - R) * L.inv_cnt;
      v[21] = dV;
      pk[0] = tc::pack_bf16(dV, 0.0f);
    }
  }
  // dz row (zeros past the minibatch): 16-byte chunk c at (c ^ ((row >> 2) & 1)) * 16
  uint8_t* dzr = L.dz + tile * (int64_t)(kTcRows * 32) + row * 32;
  const int sw = (row >> 2) & 1;
  *reinterpret_cast<uint4*>(dzr + (sw << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  *reinterpret_cast<uint4*>(dzr + ((1 ^ sw) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
  if (dz_smem) {
    *reinterpret_cast<uint4*>(dz_smem + row * 32 + (sw << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    *reinterpret_cast<uint4*>(dz_smem + row * 32 + ((1 ^ sw) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
  }
  // this warp's partial row
#pragma unroll
  for (int k = 0; k < 22; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_xor_sync(0xffffffffu, v[k], o);
  if ((threadIdx.x & 31) == 0) {
    float* pr = L.part + (tile * 4 + warp) * kW;
    if (!value_net) {
#pragma unroll
      for (int k = 0; k < 4; ++k) pr[k] = v[k];
#pragma unroll
      for (int k = 5; k < 21; ++k) pr[k] = v[k];
    } else {
      pr[4] = v[4];
      pr[21] = v[21];
    }
  }
}

// byte sizes of the weight image parts of one network (D, H)
template <int D, int H>
struct Img {
  static constexpr int RB1 = D == 32 ? 64 : 128;        // layer-1 row bytes (SW64 for D=32)
  static constexpr int W1 = H * RB1 * (D * 2 / RB1);     // H rows x D bf16
  static constexpr int W2 = H * H * 2;                   // H rows x H bf16 (SW128)
  static constexpr int W3 = kHeadN * H * 2;              // 16 rows x H bf16 (SW128)
  static constexpr int TOTAL = W1 + W2 + W3;
  static constexpr int ACT = kTcRows * H * 2;            // hidden activation tile
  static_assert(D == 32 || D == 64, "obs width");
  static_assert(H % 64 == 0 && H <= 256, "hidden width");
  static_assert(TOTAL + ACT + 3 * 1024 <= 232448, "weights and one activation tile must fit in shared memory");
};

// the streamed forward image of the Stress network (D = 64, H = 512):
// 32 KB stages in consumption order -- W1 as 2 N-halves, W2 as 2 N-halves x
// 8 K-blocks of 64, each 256 rows x 128 bytes (SW128) -- then the head
constexpr int kStageBytes = 32768;
constexpr int kStreamStages = 19;  // per tile (H = 512, D = 64)

template <int D, int H>
struct ImgS {
  static_assert(D == 64 && H == 512, "streamed layout is laid out for D = 64, H = 512");
  static constexpr int HEAD_OFF = 18 * kStageBytes;
  static constexpr int TOTAL = HEAD_OFF + kHeadN * H * 2;  // 592 KB
  __host__ __device__ static int stage_off(int s) { return s * kStageBytes; }
  __host__ __device__ static int stage_bytes(int s) { return s < 18 ? kStageBytes : kHeadN * H * 2; }
};

// byte offset of weight (r, k) of layer mat (1: W1 [H][D], 2: W2 [H][H],
// 3: the head W3 [16][H]) in a network's forward image (Img for H <= 256,
// ImgS for the streamed network)
template <int D, int H>
__host__ __device__ __forceinline__ uint32_t fwd_img_offset(int mat, int r, int k) {
  if constexpr (H > 256) {
    if (mat == 1) return (uint32_t)((r / 256) * kStageBytes) + tc::swz_offset<128>(r % 256, k, 256);
    if (mat == 2)
      return (uint32_t)((2 + (r / 256) * (H / 64) + k / 64) * kStageBytes) + tc::swz_offset<128>(r % 256, k % 64, 256);
    return (uint32_t)ImgS<D, H>::HEAD_OFF + tc::swz_offset<128>(r, k, kHeadN);
  } else {
    using I = Img<D, H>;
    if (mat == 1) return tc::swz_offset<I::RB1>(r, k, H);
    if (mat == 2) return (uint32_t)I::W1 + tc::swz_offset<128>(r, k, H);
    return (uint32_t)(I::W1 + I::W2) + tc::swz_offset<128>(r, k, kHeadN);
  }
}

constexpr int kBwRows = 128;            // samples per tile (MMA M of the data products)
constexpr int kBwStage = 32768;         // one streamed W2^T stage: 256 rows x 64 K, SW128

// backward weight image of one network: W3^T (H rows x 16, K-major SW32),
// then the W2^T stages: stage (h, kb) = rows i in [256 h, 256 h + 256) of
// W2^T, K = o in [64 kb, 64 kb + 64), K-major SW128
template <int H>
struct BwdImg {
  static constexpr int W3T = H * 32;
  static constexpr int NH = H / 256, KB = H / 64, STAGES = NH * KB;
  static constexpr int TOTAL = W3T + STAGES * kBwStage;
  static_assert(W3T % 1024 == 0, "stages start on a swizzle atom");
};

// byte offset in a network's backward image of W2[o][c] (mat = 2; stored as
// W2^T[c][o] in the streamed stages) or of W3[a][o] (mat = 3; stored as
// W3^T[o][a])
template <int H>
__host__ __device__ __forceinline__ uint32_t bwd_img_offset(int mat, int row, int col) {
  using I = BwdImg<H>;
  if (mat == 3) return tc::swz_offset<32>(col, row, H);
  const int o = row, c = col;
  const int stage = (c / 256) * I::KB + o / 64;
  return (uint32_t)(I::W3T + stage * kBwStage) + tc::swz_offset<128>(c % 256, o % 64, 256);
}

// d = bf16(g (1 - h^2)) for 16 columns: g from TMEM, h as 16 packed bf16
__device__ __forceinline__ void tanh_grad16(const float (&g)[16], const uint4 (&h)[2], bool valid,
                                            uint32_t (&pk)[8]) {
  const uint4 a = h[0], b = h[1];
  const uint32_t hw[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float h0 = __uint_as_float(hw[i] << 16), h1 = __uint_as_float(hw[i] & 0xFFFF0000u);
    pk[i] = valid ? tc::pack_bf16(g[2 * i] * (1.0f - h0 * h0), g[2 * i + 1] * (1.0f - h1 * h1)) : 0u;
  }
}

}  // namespace pe
