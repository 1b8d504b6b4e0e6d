// Measured roofs of this GPU for the kernels that are not bound by HBM or the
// tensor cores: the FP32 FMA rate (scalar FFMA and the packed two-lane FFMA
// that the fp32 network kernels use), the L2-to-SM read bandwidth, and the
// INT32 add rate.  Each probe is a plain throughput loop timed with CUDA
// events on the caller's stream; the unit counts are exact (FLOPs, bytes,
// integer operations).  Measurement support only: the paper has no
// counterpart.
#include "common.cuh"

namespace pe {

constexpr int kRoofThreads = 256;
constexpr int kRoofChains = 8;   // independent dependency chains per thread

// FP32 FMA: kRoofChains independent chains of fmaf per thread
__global__ void __launch_bounds__(kRoofThreads) roof_ffma_kernel(int64_t iters, float seed, float* sink) {
  float a[kRoofChains];
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) a[c] = seed + (float)(threadIdx.x + c);
  const float b = 0.999999f, d = 1e-7f;
  for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kRoofChains; ++c) a[c] = fmaf(a[c], b, d);
  }
  float s = 0.0f;
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) s += a[c];
  if (s == 1234.5f) sink[blockIdx.x & 1023] = s;  // never true: keeps the loop alive
}

// packed two-lane FMA (two fp32 FMAs per instruction)
__global__ void __launch_bounds__(kRoofThreads) roof_ffma2_kernel(int64_t iters, float seed, float* sink) {
  float2 a[kRoofChains];
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) a[c] = make_float2(seed + (float)threadIdx.x, seed + (float)c);
  const float2 b = make_float2(0.999999f, 0.999998f), d = make_float2(1e-7f, 2e-7f);
  for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kRoofChains; ++c) a[c] = __ffma2_rn(a[c], b, d);
  }
  float s = 0.0f;
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) s += a[c].x + a[c].y;
  if (s == 1234.5f) sink[blockIdx.x & 1023] = s;
}

// INT32 adds: per iteration a[c] += a[c + 1] around a ring of kRoofChains
// registers (one add each; the ring coupling keeps the compiler from
// replacing the loop by a closed form)
__global__ void __launch_bounds__(kRoofThreads) roof_iadd_kernel(int64_t iters, int seed, int* sink) {
  int a[kRoofChains];
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) a[c] = seed + (int)threadIdx.x * 7 + c;
  for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kRoofChains; ++c) a[c] += a[(c + 1) % kRoofChains];
  }
  int s = 0;
#pragma unroll
  for (int c = 0; c < kRoofChains; ++c) s ^= a[c];
  if (s == 0x12345) sink[blockIdx.x & 1023] = s;
}

// L2 read bandwidth: every thread streams 16-byte loads (cached in L2 only)
// over a buffer that L2 holds, `reps` times
__global__ void __launch_bounds__(kRoofThreads) roof_l2_kernel(const uint4* __restrict__ buf, int64_t n16, int reps,
                                                               unsigned int* sink) {
  uint32_t x = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int r = 0; r < reps; ++r) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += stride) {
      const uint4 v = __ldcg(buf + i);
      x ^= v.x ^ v.y ^ v.z ^ v.w;
    }
  }
  if (x == 0x9e3779b9u) sink[blockIdx.x & 1023] = x;
}

}  // namespace pe

extern "C" pe_status pe_roof_probe(int32_t kind, void* buf, int64_t bytes, int64_t reps, double* ms,
                                   double* units, void* stream) {
  using namespace pe;
  clear_error();
  if (kind < 0 || kind > 3 || !ms || !units || !buf || bytes < 65536 || reps < 1 || reps > (1 << 20))
    return fail(PE_EINVAL, "roof probe: kind in [0, 3], buf of >= 64 KiB, reps in [1, 2^20]");
  if (reinterpret_cast<uintptr_t>(buf) & 15) return fail(PE_EINVAL, "roof probe buffer not 16-byte aligned");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int dev = 0, sms = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  cudaEvent_t e0, e1;
  PE_TRY_CUDA(cudaEventCreate(&e0));
  PE_TRY_CUDA(cudaEventCreate(&e1));
  const int grid = sms * 8;  // 8 CTAs of 256 threads per SM: 64 warps, full occupancy
  const int64_t threads = (int64_t)grid * kRoofThreads;
  double u = 0.0;
  // warm-up launch, then the timed one
  for (int pass = 0; pass < 2; ++pass) {
    if (pass == 1) PE_TRY_CUDA(cudaEventRecord(e0, st));
    switch (kind) {
      case 0:
        roof_ffma_kernel<<<grid, kRoofThreads, 0, st>>>(reps, 1.0f, reinterpret_cast<float*>(buf));
        u = 2.0 * kRoofChains * (double)reps * threads;
        break;
      case 1:
        roof_ffma2_kernel<<<grid, kRoofThreads, 0, st>>>(reps, 1.0f, reinterpret_cast<float*>(buf));
        u = 4.0 * kRoofChains * (double)reps * threads;
        break;
      case 2:
        roof_iadd_kernel<<<grid, kRoofThreads, 0, st>>>(reps, 3, reinterpret_cast<int*>(buf));
        u = (double)kRoofChains * reps * threads;
        break;
      default: {
        // the first 4 KiB of the buffer take the (never written) sink words
        const int64_t n16 = (bytes - 4096) / 16;
        roof_l2_kernel<<<grid, kRoofThreads, 0, st>>>(reinterpret_cast<const uint4*>(
                                                          reinterpret_cast<char*>(buf) + 4096),
                                                      n16, (int)reps, reinterpret_cast<unsigned int*>(buf));
        u = 16.0 * (double)n16 * reps;
      }
    }
    PE_CHECK_LAUNCH("roof probe kernel");
  }
  PE_TRY_CUDA(cudaEventRecord(e1, st));
  PE_TRY_CUDA(cudaEventSynchronize(e1));
  float t = 0.0f;
  PE_TRY_CUDA(cudaEventElapsedTime(&t, e0, e1));
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  *ms = t;
  *units = u;
  return PE_OK;
}
