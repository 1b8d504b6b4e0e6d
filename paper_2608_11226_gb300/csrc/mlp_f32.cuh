// fp32 building blocks of the policy/value MLPs (FFMA register tiles over
// activations held feature-major in shared memory: xT[feature][row]).
#pragma once

#include "common.cuh"

namespace pe {

// canonical flat parameter layout (row-major W[out][in]):
//   policy W1[H][D] b1[H] W2[H][H] b2[H] W3[A][H] b3[A]
//   value  V1[H][D] c1[H] V2[H][H] c2[H] V3[1][H] c3[1]
struct MlpLayout {
  int64_t w1, b1, w2, b2, w3, b3, v1, c1, v2, c2, v3, c3, total;
};

__host__ __device__ __forceinline__ MlpLayout mlp_layout(int D, int H, int A) {
  MlpLayout L;
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

// dst[k][n] = W[n][k] for W[rows=N][cols=K] in global memory
__device__ __forceinline__ void load_transposed(const float* __restrict__ W, float* dst, int N, int K) {
  for (int i = threadIdx.x; i < N * K; i += blockDim.x) {
    const int k = i / N, n = i % N;
    dst[i] = __ldg(W + (int64_t)n * K + k);
  }
}

__device__ __forceinline__ void load_copy(const float* __restrict__ src, float* dst, int n) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) dst[i] = __ldg(src + i);
}

// RT consecutive floats (RT = 2 or 4) from shared memory
template <int RT>
__device__ __forceinline__ void load_rt(const float* p, float (&v)[RT]) {
  if constexpr (RT == 4) {
    const float4 q = *reinterpret_cast<const float4*>(p);
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  } else {
    const float2 q = *reinterpret_cast<const float2*>(p);
    v[0] = q.x; v[1] = q.y;
  }
}

template <int RT>
__device__ __forceinline__ void store_rt(float* p, const float (&v)[RT]) {
  if constexpr (RT == 4) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  } else {
    *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
  }
}

// outT[n][e] = tanh(b[n] + sum_k inT[k][e] * WT[k][n]) for TE rows; each
// thread owns an RT-row x 4-neuron register tile, accumulated as neuron pairs
// with the packed two-lane FMA (__ffma2_rn: two round-to-nearest fused
// multiply-adds, the same results as fmaf, in one instruction) and the row
// value broadcast to both lanes.  LD is the row stride (in floats) of inT
// and outT.
template <int TE, int K, int N, int LD = TE, int RT = 4>
__device__ __forceinline__ void dense_tanh_t(const float* __restrict__ inT, const float* __restrict__ WT,
                                             const float* __restrict__ bias, float* __restrict__ outT) {
  constexpr int EG = TE / RT, NG = N / 4;
  for (int j = threadIdx.x; j < EG * NG; j += blockDim.x) {
    const int eg = j % EG, ng = j / EG;
    float2 acc2[RT][2];
#pragma unroll
    for (int r = 0; r < RT; ++r) acc2[r][0] = acc2[r][1] = make_float2(0.0f, 0.0f);
#pragma unroll 8
    for (int k = 0; k < K; ++k) {
      float xv[RT];
      load_rt<RT>(inT + k * LD + eg * RT, xv);
      const float4 w = *reinterpret_cast<const float4*>(WT + k * N + ng * 4);
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

// out[e][a] = b[a] + sum_k W[a][k] * hT[k][e]
template <int TE, int K, int NA, int LD = TE>
__device__ __forceinline__ void head_t(const float* __restrict__ hT, const float* __restrict__ W,
                                       const float* __restrict__ bias, float* __restrict__ out) {
  for (int j = threadIdx.x; j < TE * NA; j += blockDim.x) {
    const int e = j % TE, a = j / TE;
    float acc = 0.0f;
#pragma unroll 8
    for (int k = 0; k < K; ++k) acc = fmaf(W[a * K + k], hT[k * LD + e], acc);
    out[e * NA + a] = acc + bias[a];
  }
}

}  // namespace pe
