// Fleet window accounting (Sec. 7 window analysis, Sec. 8 composed fleet).
//
// Prepare: q_g = rint(64 x_g) per GPU, summed per job (a job's GPUs share a
// start offset) into jobq[j][i] = sum_{g in j} q_g(i mod L) for
// i in [0, L + H): with the period unrolled once, composition n reads job j
// at index t + o[n][j] without a modulo.  The buffer (J * (L + H) int32,
// 24 MB for the 8-job, 380,000-sample fleet) stays resident in L2.
//
// Count: one warp per composition walks t in steps of 32.  Lane l forms
// P(t0 + l) from J coalesced loads, a warp-shuffle inclusive scan turns the
// 32 powers into the running prefix sum pre(t) (int32, wrapping: window
// differences pre(t) - pre(t - w) are exact because every true window sum
// is below 2^31, checked on the host), and a 1024-slot shared-memory ring of
// prefixes gives pre(t - w) for every window w <= 992 at once.
#include <algorithm>
#include <climits>

#include "common.cuh"

namespace pe {

constexpr int kFleetRing = 1024;
constexpr int kFleetWarps = 8;
constexpr float kFleetMaxWatts = 65536.0f;

struct FleetWs {
  int32_t* jobq;     // [J][L + H]
  int32_t* maxq;     // [J]
  int32_t* flag;     // [1]: bit 0 bad sample, bit 1 bad job map, bit 2 bad offset
};

__global__ void fleet_prepare_kernel(const float* __restrict__ traces, int G, int L, int H,
                                     const int32_t* __restrict__ job_of_gpu, int J,
                                     FleetWs ws) {
  __shared__ int32_t sjob[64];
  __shared__ int32_t smax[32];
  const int j = blockIdx.y;
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    const int jj = job_of_gpu[g];
    sjob[g] = jj;
    if (jj < 0 || jj >= J) atomicOr(ws.flag, 2);
  }
  __syncthreads();
  const int64_t Lx = (int64_t)L + H;
  int32_t m = 0;
  int bad = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < Lx;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t src = i < L ? i : i % L;
    int32_t s = 0;
    for (int g = 0; g < G; ++g) {
      if (sjob[g] != j) continue;
      const float x = __ldg(traces + (int64_t)g * L + src);
      if (!(x >= 0.0f && x <= kFleetMaxWatts)) {
        bad = 1;
        continue;
      }
      s += __float2int_rn(x * 64.0f);
    }
    ws.jobq[(int64_t)j * Lx + i] = s;
    m = max(m, s);
  }
  if (bad) atomicOr(ws.flag, 1);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) smax[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    int32_t mm = 0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) mm = max(mm, smax[k]);
    atomicMax(ws.maxq + j, mm);
  }
}

__global__ void fleet_check_offsets_kernel(const int32_t* __restrict__ off, int64_t n, int L,
                                           int32_t* flag) {
  int bad = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int32_t o = __ldg(off + i);
    bad |= (o < 0 || o >= L);
  }
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(flag, 4);
}

struct FleetWindows {
  int32_t w[4];
  int32_t bw[4];  // budget_q * w
};

template <int NW>
__global__ void __launch_bounds__(32 * kFleetWarps)
    fleet_windows_kernel(const int32_t* __restrict__ jobq, int J, int64_t Lx,
                         const int32_t* __restrict__ offsets, int64_t N, int H, FleetWindows win,
                         int32_t* __restrict__ counts, int32_t* __restrict__ peaks) {
  __shared__ int32_t ring_all[kFleetWarps][kFleetRing];
  __shared__ int32_t off_all[kFleetWarps][32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * kFleetWarps + wid;
  if (n >= N) return;  // the whole warp leaves together; no block-wide barrier follows
  int32_t* ring = ring_all[wid];
  const int32_t* off = off_all[wid];
  if (lane < J) off_all[wid][lane] = __ldg(offsets + n * J + lane);
  if (lane == 0) ring[kFleetRing - 1] = 0;  // pre(-1) = 0
  __syncwarp();
  int32_t carry = 0;
  int32_t cnt[NW], pk[NW];
#pragma unroll
  for (int k = 0; k < NW; ++k) cnt[k] = pk[k] = 0;
  for (int t0 = 0; t0 < H; t0 += 32) {
    const int t = t0 + lane;
    int32_t P = 0;
    if (t < H)
      for (int j = 0; j < J; ++j) P += __ldg(jobq + (int64_t)j * Lx + off[j] + t);
    int32_t x = P;
#pragma unroll
    for (int dlt = 1; dlt < 32; dlt <<= 1) {
      const int32_t y = __shfl_up_sync(0xffffffffu, x, dlt);
      if (lane >= dlt) x = (int32_t)((uint32_t)x + (uint32_t)y);
    }
    const int32_t pre = (int32_t)((uint32_t)carry + (uint32_t)x);
    carry = __shfl_sync(0xffffffffu, pre, 31);
    ring[t & (kFleetRing - 1)] = pre;
    __syncwarp();
    if (t < H) {
#pragma unroll
      for (int k = 0; k < NW; ++k) {
        const int w = win.w[k];
        if (t >= w - 1) {
          const int32_t S = (int32_t)((uint32_t)pre - (uint32_t)ring[(t - w) & (kFleetRing - 1)]);
          cnt[k] += S > win.bw[k];
          pk[k] = max(pk[k], S);
        }
      }
    }
    __syncwarp();
  }
#pragma unroll
  for (int k = 0; k < NW; ++k) {
    int32_t c = cnt[k], p = pk[k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      c += __shfl_xor_sync(0xffffffffu, c, o);
      p = max(p, __shfl_xor_sync(0xffffffffu, p, o));
    }
    if (lane == 0) {
      counts[n * NW + k] = c;
      peaks[n * NW + k] = p;
    }
  }
}

int64_t fleet_ws_bytes(int J, int L, int H) {
  const int64_t jobq = (int64_t)J * ((int64_t)L + H) * 4;
  return ((jobq + 255) / 256) * 256 + 256 + 256;
}

pe_status fleet_launch(const float* traces, int G, int L, const int32_t* job_of_gpu, int J,
                       const int32_t* offsets, int64_t N, int H, const int32_t* windows, int W,
                       int64_t budget_q, int32_t* counts, int32_t* peaks, void* workspace,
                       cudaStream_t st) {
  char* base = reinterpret_cast<char*>(workspace);
  const int64_t jobq_bytes = ((int64_t)J * ((int64_t)L + H) * 4 + 255) / 256 * 256;
  FleetWs ws;
  ws.jobq = reinterpret_cast<int32_t*>(base);
  ws.maxq = reinterpret_cast<int32_t*>(base + jobq_bytes);
  ws.flag = reinterpret_cast<int32_t*>(base + jobq_bytes + 256);
  PE_TRY_CUDA(cudaMemsetAsync(ws.maxq, 0, 256 + 4, st));
  dim3 grid(ceil_div((int64_t)L + H, 256 * 8), J);
  {
    ProfScope ps(PE_PROF_FLEET_PREP, st);
    fleet_prepare_kernel<<<grid, 256, 0, st>>>(traces, G, L, H, job_of_gpu, J, ws);
  }
  PE_CHECK_LAUNCH("fleet_prepare_kernel");
  if (N > 0) {
    fleet_check_offsets_kernel<<<(int)std::min<int64_t>(ceil_div(N * J, 256), 4096), 256, 0, st>>>(
        offsets, N * J, L, ws.flag);
    PE_CHECK_LAUNCH("fleet_check_offsets_kernel");
  }
  int32_t host[64 + 1];
  PE_TRY_CUDA(cudaMemcpyAsync(host, ws.maxq, sizeof(int32_t) * J, cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaMemcpyAsync(host + 64, ws.flag, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  const int32_t flag = host[64];
  if (flag & 1) return fail(PE_EOVERFLOW, "fleet trace holds a sample that is not finite or outside [0, %g] W", (double)kFleetMaxWatts);
  if (flag & 2) return fail(PE_EINVAL, "job_of_gpu entry outside [0, J)");
  if (flag & 4) return fail(PE_EINVAL, "fleet offset outside [0, L)");
  int64_t sum_max = 0;
  for (int j = 0; j < J; ++j) sum_max += host[j];
  FleetWindows win{};
  for (int k = 0; k < W; ++k) {
    const int64_t w = windows[k];
    if (sum_max * w >= (int64_t)INT_MAX || budget_q * w >= (int64_t)INT_MAX)
      return fail(PE_EOVERFLOW, "window %d: composed window sum may exceed int32", (int)w);
    win.w[k] = (int32_t)w;
    win.bw[k] = (int32_t)(budget_q * w);
  }
  if (N == 0) return PE_OK;
  const int grid_n = (int)((N + kFleetWarps - 1) / kFleetWarps);
  const int64_t Lx = (int64_t)L + H;
  ProfScope ps(PE_PROF_FLEET_WINDOWS, st);
  switch (W) {
    case 1: fleet_windows_kernel<1><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.jobq, J, Lx, offsets, N, H, win, counts, peaks); break;
    case 2: fleet_windows_kernel<2><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.jobq, J, Lx, offsets, N, H, win, counts, peaks); break;
    case 3: fleet_windows_kernel<3><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.jobq, J, Lx, offsets, N, H, win, counts, peaks); break;
    default: fleet_windows_kernel<4><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.jobq, J, Lx, offsets, N, H, win, counts, peaks); break;
  }
  PE_CHECK_LAUNCH("fleet_windows_kernel");
  return PE_OK;
}

}  // namespace pe
