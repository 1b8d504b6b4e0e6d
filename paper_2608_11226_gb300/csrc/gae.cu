// Reverse-time generalised advantage estimation over a time-major [T][E]
// buffer (Sec. 4.2: gamma 0.99, lambda 0.95):
//   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,  A_t = delta_t + gamma lambda (1 - d_t) A_{t+1}.
//
// HBM-bound: 9 bytes in and 8 bytes out per env-step.  A thread owns V
// consecutive envs (vector loads/stores; a warp covers 32*V envs of one row)
// and one time chunk of CL steps held in registers; the NW warps of a CTA
// cover NW consecutive chunks.  Each thread first reduces its chunk to the
// affine map A_start = alpha + beta * A_end, warp 0 chains the chunk maps
// through shared memory, and each thread then re-runs its chunk with the
// right carry-in and streams A and R out.  Longer horizons loop over
// super-chunks of CL*NW steps from the end.  That time-parallel form serves
// narrow batches; batches of 32,768 envs or more take the barrier-free
// per-column kernel below.
#include <type_traits>

#include "common.cuh"

namespace pe {

template <int CL, int NW, int V>
__global__ void __launch_bounds__(32 * NW)
    gae_kernel_v(const float* __restrict__ r, const float* __restrict__ v,
                 const uint8_t* __restrict__ d, const float* __restrict__ last_v, int T, int E,
                 float gamma, float lam, float* __restrict__ adv, float* __restrict__ ret) {
  using FV = typename std::conditional<V == 4, float4, typename std::conditional<V == 2, float2, float>::type>::type;
  using BV = typename std::conditional<V == 4, uchar4, typename std::conditional<V == 2, uchar2, unsigned char>::type>::type;
  __shared__ float sa[NW][32 * V], sb[NW][32 * V], cin[NW + 1][32 * V];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int e0 = (blockIdx.x * 32 + lane) * V;   // first env of this thread
  const bool ok = e0 < E;
  const float gl = gamma * lam;
  float carry[V];
#pragma unroll
  for (int u = 0; u < V; ++u) carry[u] = 0.0f;
  for (int sc_end = T; sc_end > 0; sc_end -= CL * NW) {
    const int sc_start = max(0, sc_end - CL * NW);
    const int t1 = sc_end - w * CL;
    const int t0 = max(sc_start, t1 - CL);
    float rr[CL][V], vv[CL][V], nt[CL][V];
    float vnext[V];
#pragma unroll
    for (int u = 0; u < V; ++u) vnext[u] = 0.0f;
    if (ok && t1 > t0) {
      const FV q = t1 < T ? *reinterpret_cast<const FV*>(v + (int64_t)t1 * E + e0) : *reinterpret_cast<const FV*>(last_v + e0);
      const float* qp = reinterpret_cast<const float*>(&q);
#pragma unroll
      for (int u = 0; u < V; ++u) vnext[u] = qp[u];
    }
#pragma unroll
    for (int i = 0; i < CL; ++i) {
      const int t = t1 - 1 - i;
#pragma unroll
      for (int u = 0; u < V; ++u) rr[i][u] = vv[i][u] = nt[i][u] = 0.0f;
      if (ok && t >= t0) {
        const int64_t o = (int64_t)t * E + e0;
        const FV a = __ldcs(reinterpret_cast<const FV*>(r + o));
        const FV b = *reinterpret_cast<const FV*>(v + o);
        const BV c = *reinterpret_cast<const BV*>(d + o);
        const float* ap = reinterpret_cast<const float*>(&a);
        const float* bp = reinterpret_cast<const float*>(&b);
        const unsigned char* cp = reinterpret_cast<const unsigned char*>(&c);
#pragma unroll
        for (int u = 0; u < V; ++u) {
          rr[i][u] = ap[u];
          vv[i][u] = bp[u];
          nt[i][u] = 1.0f - (float)cp[u];
        }
      }
    }
#pragma unroll
    for (int u = 0; u < V; ++u) {
      float alpha = 0.0f, beta = 1.0f, vn = vnext[u];
#pragma unroll
      for (int i = 0; i < CL; ++i) {
        if (t1 - 1 - i >= t0) {
          const float delta = rr[i][u] + gamma * vn * nt[i][u] - vv[i][u];
          const float c = gl * nt[i][u];
          alpha = delta + c * alpha;
          beta = c * beta;
          vn = vv[i][u];
        }
      }
      sa[w][lane * V + u] = alpha;
      sb[w][lane * V + u] = beta;
    }
    __syncthreads();
    if (w == 0) {
#pragma unroll
      for (int u = 0; u < V; ++u) {
        float a = carry[u];
        for (int j = 0; j < NW; ++j) {
          cin[j][lane * V + u] = a;
          a = sa[j][lane * V + u] + sb[j][lane * V + u] * a;
        }
        cin[NW][lane * V + u] = a;
      }
    }
    __syncthreads();
    float A[V], vn[V];
#pragma unroll
    for (int u = 0; u < V; ++u) {
      A[u] = cin[w][lane * V + u];
      vn[u] = vnext[u];
    }
#pragma unroll
    for (int i = 0; i < CL; ++i) {
      const int t = t1 - 1 - i;
      if (ok && t >= t0) {
        float ao[V], ro[V];
#pragma unroll
        for (int u = 0; u < V; ++u) {
          const float delta = rr[i][u] + gamma * vn[u] * nt[i][u] - vv[i][u];
          A[u] = delta + gl * nt[i][u] * A[u];
          ao[u] = A[u];
          ro[u] = A[u] + vv[i][u];
          vn[u] = vv[i][u];
        }
        const int64_t o = (int64_t)t * E + e0;
        __stcs(reinterpret_cast<FV*>(adv + o), *reinterpret_cast<FV*>(ao));
        __stcs(reinterpret_cast<FV*>(ret + o), *reinterpret_cast<FV*>(ro));
      }
    }
#pragma unroll
    for (int u = 0; u < V; ++u) carry[u] = cin[NW][lane * V + u];
    __syncthreads();
  }
}


// Wide batches (E >= 32,768): one thread per V envs walks the whole horizon
// backwards, A_t = delta_t + gamma lambda (1 - d_t) A_{t+1} in the same
// order as the recursion, with no barrier and no shared memory.  The loads of
// the next P steps are kept in flight in a register ring, so each SM holds
// enough outstanding bytes to cover HBM latency; every warp streams
// 32 * V consecutive envs of a row (coalesced).  Measured on GB300: one env
// per thread with 16 loads in flight reaches 74% of the HBM copy peak at
// 65,536 envs (14 warps per SM); at 262,144 envs four envs per thread (8
// steps in flight) keep the launch to one wave and reach 77%, where two
// envs per thread at 94 registers spilled into a second wave (54%).
template <int V, int P>
__global__ void __launch_bounds__(128)
    gae_stream_kernel(const float* __restrict__ r, const float* __restrict__ v, const uint8_t* __restrict__ d,
                      const float* __restrict__ last_v, int T, int E, float gamma, float lam,
                      float* __restrict__ adv, float* __restrict__ ret) {
  using FV = typename std::conditional<V == 4, float4, typename std::conditional<V == 2, float2, float>::type>::type;
  using BV = typename std::conditional<V == 4, uchar4, typename std::conditional<V == 2, uchar2, unsigned char>::type>::type;
  const int e0 = (blockIdx.x * blockDim.x + threadIdx.x) * V;
  if (e0 >= E) return;
  const float gl = gamma * lam;
  FV rb[P], vb[P];
  BV db[P];
  auto load = [&](int k, int t) {
    const int64_t o = (int64_t)t * E + e0;
    rb[k] = __ldcs(reinterpret_cast<const FV*>(r + o));
    vb[k] = __ldcs(reinterpret_cast<const FV*>(v + o));
    db[k] = __ldcs(reinterpret_cast<const BV*>(d + o));
  };
#pragma unroll
  for (int k = 0; k < P; ++k)
    if (T - 1 - k >= 0) load(k, T - 1 - k);
  float A[V], vn[V];
  {
    const FV q = *reinterpret_cast<const FV*>(last_v + e0);
    const float* qp = reinterpret_cast<const float*>(&q);
#pragma unroll
    for (int u = 0; u < V; ++u) {
      A[u] = 0.0f;
      vn[u] = qp[u];
    }
  }
  for (int base = T - 1; base >= 0; base -= P) {
#pragma unroll
    for (int k = 0; k < P; ++k) {
      const int t = base - k;
      if (t >= 0) {
        const float* rp = reinterpret_cast<const float*>(&rb[k]);
        const float* vp = reinterpret_cast<const float*>(&vb[k]);
        const unsigned char* dp = reinterpret_cast<const unsigned char*>(&db[k]);
        float ao[V], ro[V];
#pragma unroll
        for (int u = 0; u < V; ++u) {
          const float nt = 1.0f - (float)dp[u];
          const float delta = rp[u] + gamma * vn[u] * nt - vp[u];
          A[u] = delta + gl * nt * A[u];
          ao[u] = A[u];
          ro[u] = A[u] + vp[u];
          vn[u] = vp[u];
        }
        if (t - P >= 0) load(k, t - P);
        const int64_t o = (int64_t)t * E + e0;
        __stcs(reinterpret_cast<FV*>(adv + o), *reinterpret_cast<FV*>(ao));
        __stcs(reinterpret_cast<FV*>(ret + o), *reinterpret_cast<FV*>(ro));
      }
    }
  }
}

template <int V, int P>
static pe_status gae_stream_run(const float* r, const float* v, const uint8_t* d, const float* last_v, int T,
                                int E, float gamma, float lam, float* adv, float* ret, cudaStream_t st) {
  {
    ProfScope ps(PE_PROF_GAE, st);
    gae_stream_kernel<V, P><<<ceil_div(E / V, 128), 128, 0, st>>>(r, v, d, last_v, T, E, gamma, lam, adv, ret);
  }
  PE_CHECK_LAUNCH("gae_stream_kernel");
  return PE_OK;
}

template <int CL, int NW, int V>
static pe_status gae_run(const float* r, const float* v, const uint8_t* d, const float* last_v, int T,
                         int E, float gamma, float lam, float* adv, float* ret, cudaStream_t st) {
  {
    ProfScope ps(PE_PROF_GAE, st);
    gae_kernel_v<CL, NW, V><<<ceil_div(E / V, 32), 32 * NW, 0, st>>>(r, v, d, last_v, T, E, gamma, lam, adv, ret);
  }
  PE_CHECK_LAUNCH("gae_kernel");
  return PE_OK;
}

pe_status gae_launch(const float* r, const float* v, const uint8_t* d, const float* last_v,
                     int T, int E, float gamma, float lam, float* adv, float* ret,
                     cudaStream_t st) {
  const int64_t n = (int64_t)T * E;
  const bool al4 = (E % 4 == 0) && ((reinterpret_cast<uintptr_t>(r) | reinterpret_cast<uintptr_t>(v) |
                                      reinterpret_cast<uintptr_t>(adv) | reinterpret_cast<uintptr_t>(ret) |
                                      reinterpret_cast<uintptr_t>(last_v)) % 16 == 0) &&
                   reinterpret_cast<uintptr_t>(d) % 4 == 0;
  const bool al2 = (E % 2 == 0) && ((reinterpret_cast<uintptr_t>(r) | reinterpret_cast<uintptr_t>(v) |
                                      reinterpret_cast<uintptr_t>(adv) | reinterpret_cast<uintptr_t>(ret) |
                                      reinterpret_cast<uintptr_t>(last_v)) % 8 == 0) &&
                   reinterpret_cast<uintptr_t>(d) % 2 == 0;
  if (E >= 196608 && al4) return gae_stream_run<4, 8>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
  if (E >= 49152) return gae_stream_run<1, 16>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
  if (E >= 32768) return gae_stream_run<1, 32>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
  if (n >= ((int64_t)1 << 28) && al4) return gae_run<4, 8, 4>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
  if (E >= 16384 && al2) return gae_run<4, 16, 2>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
  return gae_run<8, 32, 1>(r, v, d, last_v, T, E, gamma, lam, adv, ret, st);
}

}  // namespace pe
