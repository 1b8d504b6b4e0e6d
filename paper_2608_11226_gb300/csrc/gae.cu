// Reverse-time generalised advantage estimation over a time-major [T][E]
// buffer (Sec. 4.2: gamma 0.99, lambda 0.95):
//   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,  A_t = delta_t + gamma lambda (1 - d_t) A_{t+1}.
//
// HBM-bound: 9 bytes in and 8 bytes out per env-step.  A CTA covers 32
// consecutive envs (one coalesced 128-byte row segment per warp load) and
// NW time chunks of CL steps, one chunk per warp.  Each thread first reduces
// its chunk to the affine map A_start = alpha + beta * A_end, the chunk maps
// are chained through shared memory by one warp, and each thread then
// re-runs its chunk from registers with the right carry-in.  Longer horizons
// loop over super-chunks of CL*NW steps from the end.
#include "common.cuh"

namespace pe {

template <int CL, int NW>
__global__ void __launch_bounds__(32 * NW)
    gae_kernel(const float* __restrict__ r, const float* __restrict__ v,
               const uint8_t* __restrict__ d, const float* __restrict__ last_v, int T, int E,
               float gamma, float lam, float* __restrict__ adv, float* __restrict__ ret) {
  __shared__ float sa[NW][32], sb[NW][32], cin[NW + 1][32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int e = blockIdx.x * 32 + lane;
  const bool ok = e < E;
  const float gl = gamma * lam;
  float carry = 0.0f;  // A at the first step after the current super-chunk
  for (int sc_end = T; sc_end > 0; sc_end -= CL * NW) {
    const int sc_start = max(0, sc_end - CL * NW);
    const int t1 = sc_end - w * CL;  // warp 0 holds the latest chunk
    const int t0 = max(sc_start, t1 - CL);
    float rr[CL], vv[CL], nt[CL];
    float vnext = 0.0f;
    if (ok && t1 > t0) vnext = t1 < T ? __ldg(v + (int64_t)t1 * E + e) : __ldg(last_v + e);
#pragma unroll
    for (int i = 0; i < CL; ++i) {
      const int t = t1 - 1 - i;
      rr[i] = vv[i] = nt[i] = 0.0f;
      if (ok && t >= t0) {
        const int64_t o = (int64_t)t * E + e;
        rr[i] = __ldg(r + o);
        vv[i] = __ldg(v + o);
        nt[i] = 1.0f - (float)__ldg(d + o);
      }
    }
    float alpha = 0.0f, beta = 1.0f, vn = vnext;
#pragma unroll
    for (int i = 0; i < CL; ++i) {
      if (t1 - 1 - i >= t0) {
        const float delta = rr[i] + gamma * vn * nt[i] - vv[i];
        const float c = gl * nt[i];
        alpha = delta + c * alpha;
        beta = c * beta;
        vn = vv[i];
      }
    }
    sa[w][lane] = alpha;
    sb[w][lane] = beta;
    __syncthreads();
    if (w == 0) {
      float a = carry;
#pragma unroll 4
      for (int j = 0; j < NW; ++j) {
        cin[j][lane] = a;
        a = sa[j][lane] + sb[j][lane] * a;
      }
      cin[NW][lane] = a;
    }
    __syncthreads();
    float A = cin[w][lane];
    vn = vnext;
#pragma unroll
    for (int i = 0; i < CL; ++i) {
      const int t = t1 - 1 - i;
      if (ok && t >= t0) {
        const float delta = rr[i] + gamma * vn * nt[i] - vv[i];
        A = delta + gl * nt[i] * A;
        const int64_t o = (int64_t)t * E + e;
        adv[o] = A;
        ret[o] = A + vv[i];
        vn = vv[i];
      }
    }
    carry = cin[NW][lane];
    __syncthreads();
  }
}

pe_status gae_launch(const float* r, const float* v, const uint8_t* d, const float* last_v,
                     int T, int E, float gamma, float lam, float* adv, float* ret,
                     cudaStream_t st) {
  constexpr int CL = 16, NW = 16;
  {
    ProfScope ps(PE_PROF_GAE, st);
    gae_kernel<CL, NW><<<ceil_div(E, 32), 32 * NW, 0, st>>>(r, v, d, last_v, T, E, gamma, lam, adv, ret);
  }
  PE_CHECK_LAUNCH("gae_kernel");
  return PE_OK;
}

}  // namespace pe
