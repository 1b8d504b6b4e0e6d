// Shared device/host helpers of the pe library (GB300, sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "pe.h"

namespace pe {

// ---------------------------------------------------------------------------
// error reporting (thread-local message behind pe_last_error)
// ---------------------------------------------------------------------------
pe_status fail(pe_status code, const char* fmt, ...);
pe_status cuda_fail(cudaError_t err, const char* what);
void clear_error();

#define PE_TRY_CUDA(expr)                                   \
  do {                                                      \
    cudaError_t _e = (expr);                                \
    if (_e != cudaSuccess) return ::pe::cuda_fail(_e, #expr); \
  } while (0)

#define PE_CHECK_LAUNCH(what)                                  \
  do {                                                         \
    cudaError_t _e = cudaGetLastError();                       \
    if (_e != cudaSuccess) return ::pe::cuda_fail(_e, what);   \
  } while (0)

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11): 10 rounds, key bumped by the Weyl
// increments between rounds.
// ---------------------------------------------------------------------------
struct u32x4 {
  uint32_t x, y, z, w;
};

__host__ __device__ __forceinline__ u32x4 philox10(u32x4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
#ifdef __CUDA_ARCH__
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
#else
    const uint64_t m0 = (uint64_t)0xD2511F53u * c.x, m1 = (uint64_t)0xCD9E8D57u * c.z;
    const uint32_t lo0 = (uint32_t)m0, hi0 = (uint32_t)(m0 >> 32);
    const uint32_t lo1 = (uint32_t)m1, hi1 = (uint32_t)(m1 >> 32);
#endif
    c = u32x4{hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0};
  }
  return c;
}

// counter purposes (4th counter word)
enum : uint32_t { kDrawAction = 0, kDrawReset = 1, kDrawInit = 2, kDrawPerm = 3 };

__host__ __device__ __forceinline__ uint32_t draw32(uint64_t seed, uint32_t a, uint32_t b,
                                                    uint32_t c, uint32_t d) {
  return philox10(u32x4{a, b, c, d}, (uint32_t)seed, (uint32_t)(seed >> 32)).x;
}

// ---------------------------------------------------------------------------
// Minibatch permutation: 4-round balanced Feistel over an even number of
// bits, cycle-walking into [0, n) (Black & Rogaway 2002); round function is
// the lowbias32 integer hash (Wellons 2018) of (R xor round key).
// ---------------------------------------------------------------------------
struct Feistel {
  uint32_t k[4];
  uint32_t half;
  uint64_t n;
};

__host__ __device__ __forceinline__ uint32_t lowbias32(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7feb352du;
  x ^= x >> 15;
  x *= 0x846ca68bu;
  x ^= x >> 16;
  return x;
}

__host__ __device__ __forceinline__ uint64_t feistel_round4(const Feistel& f, uint64_t x) {
  const uint64_t mask = (1ull << f.half) - 1ull;
  uint64_t L = x >> f.half, R = x & mask;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const uint64_t F = (uint64_t)lowbias32((uint32_t)R ^ f.k[r]) & mask;
    const uint64_t t = L ^ F;
    L = R;
    R = t;
  }
  return (L << f.half) | R;
}

// the permuted index; the walk is bounded by the domain size (<= 4n) because
// the Feistel map is a permutation of the domain and i < n lies on a cycle
// that re-enters [0, n)
__host__ __device__ __forceinline__ uint32_t feistel_index(const Feistel& f, uint64_t i) {
  uint64_t y = feistel_round4(f, i);
  const uint64_t limit = 4ull * f.n + 4ull;
  for (uint64_t it = 0; y >= f.n && it < limit; ++it) y = feistel_round4(f, y);
  return (uint32_t)(y < f.n ? y : i % f.n);  // the fallback is unreachable for a permutation
}

Feistel make_feistel(uint64_t n, uint64_t seed, uint32_t epoch, uint32_t iteration);

// ---------------------------------------------------------------------------
// fixed-point power and fp32 feature helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ int32_t quant64(float x, float s) {
  // one fp32 multiply (the actuator), exact scaling by 64, round to nearest even
  return __float2int_rn(__fmul_rn(__fmul_rn(x, s), 64.0f));
}

__device__ __forceinline__ float ratio_i(int64_t num, int64_t den) {
  return __fdiv_rn(__ll2float_rn(num), __ll2float_rn(den));
}

__device__ __forceinline__ float bf16r(float x) {
  // round-to-nearest-even to bf16, returned as fp32
  uint32_t u = __float_as_uint(x);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return __uint_as_float(u & 0xFFFF0000u);
}

// Approximate KL term of one sample, (rho - 1) - log rho with
// rho = exp(x) (Schulman's k3 estimator), without the cancellation of the
// literal fp32 form: for |x| < 1/8 the Taylor series of e^x - 1 - x,
//   x^2/2 (1 + x/3 (1 + x/4 (1 + x/5 (1 + x/6 (1 + x/7))))),
// whose first dropped term is below 2e-8 of the sum; above that the direct
// form, whose cancellation costs less than a few ulps there.
__device__ __forceinline__ float kl_term(float x) {
  if (fabsf(x) < 0.125f) {
    float t = fmaf(x, 1.0f / 7.0f, 1.0f);
    t = fmaf(x * (1.0f / 6.0f), t, 1.0f);
    t = fmaf(x * (1.0f / 5.0f), t, 1.0f);
    t = fmaf(x * (1.0f / 4.0f), t, 1.0f);
    t = fmaf(x * (1.0f / 3.0f), t, 1.0f);
    return 0.5f * x * x * t;
  }
  return expm1f(x) - x;
}

// The PPO loss of a minibatch, taken in the forward pass's head epilogue
// (Sec. 4.2; SB3's clipped surrogate, squared-error value loss and entropy
// bonus).  Row r of the minibatch is sample gather[r]; the thread that reads
// the row's head from TMEM computes the loss terms and dLoss/dhead, writes
// dz -- rounded to bf16 -- into the dz tile image (16 bf16 per row, 32-byte
// rows, 32-byte swizzle; rows past the minibatch are zero), and each head
// warp writes the fixed-order (shuffle tree) sums of its 32 rows as one
// partial row: columns 0-3 pg loss, entropy, approximate KL, clip indicator
// and 5..5+A-1 the policy head-bias gradient (policy network), column 4 the
// value loss and 21 the value head-bias gradient (value network), both from
// the unrounded dz.
struct PpoHead {
  const uint8_t* act;
  const float* logp_old;
  const float* adv;
  const float* ret;
  const float2* advstat;  // (mean, 1 / (std + 1e-8)) of the minibatch's advantages
  float clip, vf_coef, ent_coef, inv_cnt;
  uint8_t* dz;            // dz tile images of this network
  float* part;            // [tiles * 4][32] partial rows
};

inline int ceil_div(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

// launch profiling: brackets a launch with CUDA events when enabled
void prof_mark(int kind, cudaStream_t st, bool begin);
struct ProfScope {
  int kind;
  cudaStream_t st;
  ProfScope(int k, cudaStream_t s) : kind(k), st(s) { prof_mark(kind, st, true); }
  ~ProfScope() { prof_mark(kind, st, false); }
};

}  // namespace pe
