// Fleet window accounting (Sec. 7 window analysis, Sec. 8 composed fleet).
//
// Prepare: q_g = rint(64 x_g) per GPU (1/64 W), summed per job (a job's GPUs
// share a start offset) and turned into a per-job prefix sum over the
// period unrolled once:
//   PREX[j][i] = sum_{k < i} sum_{g in j} q_g(k mod L),  i in [0, L + H],
// kept modulo 2^32 (uint32).  For composition n the running composed prefix
// is then pre(t) = sum_j PREX[j][t + 1 + o[n][j]] (mod 2^32), and every
// window sum is S_w(t) = pre(t) - pre(t - w), exact because the true sum is
// below 2^31 (checked on the host from the per-job maxima).  The prefixes
// (J * (L + H + 1) int32, 24 MB for the 8-job, 380,000-sample fleet) stay
// resident in L2.
//
// Count: one warp per composition walks t in steps of 32; lane l forms
// pre(t0 + l) from J coalesced loads, keeps it in a 1024-slot shared-memory
// ring, and reads pre(t - w) back for every window w <= 992 at once.
#include <algorithm>
#include <climits>

#include "common.cuh"

namespace pe {

constexpr int kFleetRing = 1024;
constexpr int kFleetWarps = 8;
constexpr int kFleetChunk = 8192;   // prefix-scan chunk per block
constexpr float kFleetMaxWatts = 65536.0f;

struct FleetWs {
  uint32_t* prex;    // [J][Lp]
  uint32_t* totals;  // [J][nchunk] chunk sums, then exclusive chunk offsets
  int32_t* maxq;     // [J]
  int32_t* flag;     // [1]: bit 0 bad sample, bit 1 bad job map, bit 2 bad offset
  int64_t Lp;        // row stride of prex
  int nchunk;
};

__device__ __forceinline__ int32_t job_sample(const float* __restrict__ traces, const int8_t* sjob,
                                              int G, int L, int j, int64_t i, int& bad) {
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
  return s;
}

__device__ __forceinline__ void load_jobs(const int32_t* __restrict__ job_of_gpu, int G, int J,
                                          int8_t* sjob, int32_t* flag) {
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    const int jj = job_of_gpu[g];
    sjob[g] = (int8_t)((jj >= 0 && jj < J) ? jj : -1);
    if (jj < 0 || jj >= J) atomicOr(flag, 2);
  }
  __syncthreads();
}

// block sum of uint32 (wrapping) and max of int32 over 256 threads
__device__ __forceinline__ void block_sum_max(uint32_t& s, int32_t& m, uint32_t* ss, int32_t* sm) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
  }
  if ((threadIdx.x & 31) == 0) {
    ss[threadIdx.x >> 5] = s;
    sm[threadIdx.x >> 5] = m;
  }
  __syncthreads();
  s = 0;
  m = 0;
  for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
    s += ss[k];
    m = max(m, sm[k]);
  }
}

// pass 1: per (job, chunk) sum, job maximum, sample validation
__global__ void __launch_bounds__(256) fleet_chunk_sums_kernel(const float* __restrict__ traces, int G, int L, int H,
                                                               const int32_t* __restrict__ job_of_gpu,
                                                               int J, FleetWs ws) {
  __shared__ int8_t sjob[64];
  __shared__ uint32_t ss[8];
  __shared__ int32_t sm[8];
  load_jobs(job_of_gpu, G, J, sjob, ws.flag);
  const int j = blockIdx.y, c = blockIdx.x;
  const int64_t Lx = (int64_t)L + H;
  const int64_t i0 = (int64_t)c * kFleetChunk;
  uint32_t s = 0;
  int32_t m = 0;
  int bad = 0;
  for (int64_t i = i0 + threadIdx.x; i < min(i0 + kFleetChunk, Lx); i += blockDim.x) {
    const int32_t q = job_sample(traces, sjob, G, L, j, i, bad);
    s += (uint32_t)q;
    m = max(m, q);
  }
  if (bad) atomicOr(ws.flag, 1);
  block_sum_max(s, m, ss, sm);
  if (threadIdx.x == 0) {
    ws.totals[(int64_t)j * ws.nchunk + c] = s;
    atomicMax(ws.maxq + j, m);
  }
}

// pass 2: exclusive scan of each job's chunk sums (one warp per job)
__global__ void fleet_chunk_scan_kernel(FleetWs ws) {
  const int j = blockIdx.x, lane = threadIdx.x;
  uint32_t carry = 0;
  for (int c0 = 0; c0 < ws.nchunk; c0 += 32) {
    const int c = c0 + lane;
    const uint32_t v = c < ws.nchunk ? ws.totals[(int64_t)j * ws.nchunk + c] : 0u;
    uint32_t x = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, d);
      if (lane >= d) x += y;
    }
    if (c < ws.nchunk) ws.totals[(int64_t)j * ws.nchunk + c] = carry + x - v;
    carry += __shfl_sync(0xffffffffu, x, 31);
  }
}

// pass 3: prefix within each chunk, offset by the chunk's exclusive sum
__global__ void __launch_bounds__(256) fleet_prefix_kernel(const float* __restrict__ traces, int G, int L, int H,
                                                           const int32_t* __restrict__ job_of_gpu,
                                                           int J, FleetWs ws) {
  __shared__ int8_t sjob[64];
  __shared__ uint32_t wsum[8];
  load_jobs(job_of_gpu, G, J, sjob, ws.flag);
  const int j = blockIdx.y, c = blockIdx.x;
  const int64_t Lx = (int64_t)L + H;
  const int64_t i0 = (int64_t)c * kFleetChunk;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t carry = ws.totals[(int64_t)j * ws.nchunk + c];
  uint32_t* row = ws.prex + (int64_t)j * ws.Lp;
  if (c == 0 && threadIdx.x == 0) row[0] = 0u;
  int bad = 0;
  for (int64_t b = i0; b < min(i0 + kFleetChunk, Lx); b += blockDim.x) {
    const int64_t i = b + threadIdx.x;
    const uint32_t q = i < Lx ? (uint32_t)job_sample(traces, sjob, G, L, j, i, bad) : 0u;
    uint32_t x = q;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, d);
      if (lane >= d) x += y;
    }
    if (lane == 31) wsum[w] = x;
    __syncthreads();
    uint32_t before = 0, total = 0;
    for (int k = 0; k < 8; ++k) {
      if (k < w) before += wsum[k];
      total += wsum[k];
    }
    if (i < Lx) row[i + 1] = carry + before + x;
    carry += total;
    __syncthreads();
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
    fleet_windows_kernel(const uint32_t* __restrict__ prex, int J, int64_t Lp,
                         const int32_t* __restrict__ offsets, int64_t N, int H, FleetWindows win,
                         int32_t* __restrict__ counts, int32_t* __restrict__ peaks) {
  __shared__ uint32_t ring_all[kFleetWarps][kFleetRing];
  __shared__ const uint32_t* base_all[kFleetWarps][32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * kFleetWarps + wid;
  if (n >= N) return;  // the whole warp leaves together; no block-wide barrier follows
  uint32_t* ring = ring_all[wid];
  const uint32_t** base = base_all[wid];
  uint32_t pre_m1 = 0;  // pre(-1) = sum_j PREX[j][o_j]
  if (lane < J) {
    const int32_t o = __ldg(offsets + n * J + lane);
    const uint32_t* b = prex + (int64_t)lane * Lp + o;
    base[lane] = b + 1;
    pre_m1 = __ldg(b);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) pre_m1 += __shfl_xor_sync(0xffffffffu, pre_m1, o);
  if (lane == 0) ring[kFleetRing - 1] = pre_m1;
  __syncwarp();
  const uint32_t* b0 = base[0];
  int32_t cnt[NW], pk[NW];
#pragma unroll
  for (int k = 0; k < NW; ++k) cnt[k] = pk[k] = 0;
  for (int t0 = 0; t0 < H; t0 += 32) {
    const int t = t0 + lane;
    uint32_t pre = 0;
    if (t < H) {
      pre = __ldg(b0 + t);
      for (int j = 1; j < J; ++j) pre += __ldg(base[j] + t);
    }
    ring[t & (kFleetRing - 1)] = pre;
    __syncwarp();
    if (t < H) {
#pragma unroll
      for (int k = 0; k < NW; ++k) {
        const int w = win.w[k];
        if (t >= w - 1) {
          const int32_t S = (int32_t)(pre - ring[(t - w) & (kFleetRing - 1)]);
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

// The same walk for fleets of at most 8 jobs: the J stream pointers live
// in registers (no shared-memory pointer reloads), and each iteration
// issues the loads of two 32-sample blocks before using either.
constexpr int kFleetJMax = 8;

// prefix-array row of each composed stream (stream k reads row r[k]): the
// identity for a fleet, {partial fleet, candidate job} for the stagger
struct StreamRows {
  int32_t r[kFleetJMax];
};
static StreamRows identity_rows() {
  StreamRows m;
  for (int k = 0; k < kFleetJMax; ++k) m.r[k] = k;
  return m;
}

template <int NW>
__global__ void __launch_bounds__(32 * kFleetWarps)
    fleet_windows_j8_kernel(const uint32_t* __restrict__ prex, int J, int64_t Lp, StreamRows rows,
                            const int32_t* __restrict__ offsets, int64_t N, int H, FleetWindows win,
                            int32_t* __restrict__ counts, int32_t* __restrict__ peaks) {
  __shared__ uint32_t ring_all[kFleetWarps][kFleetRing];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * kFleetWarps + wid;
  if (n >= N) return;  // the whole warp leaves together; no block-wide barrier follows
  uint32_t* ring = ring_all[wid];
  // every lane holds all J stream bases (t = 0 at index 1 + o_j); lane j also
  // loads pre(-1)'s term PREX[j][o_j]
  const uint32_t* bp[kFleetJMax];
  uint32_t pre_m1 = 0;
#pragma unroll
  for (int j = 0; j < kFleetJMax; ++j) {
    bp[j] = prex;
    if (j < J) {
      const int32_t o = __ldg(offsets + n * J + j);
      bp[j] = prex + (int64_t)rows.r[j] * Lp + o + 1;
      if (lane == j) pre_m1 = __ldg(bp[j] - 1);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) pre_m1 += __shfl_xor_sync(0xffffffffu, pre_m1, o);
  if (lane == 0) ring[kFleetRing - 1] = pre_m1;
  __syncwarp();
  int32_t cnt[NW], pk[NW];
#pragma unroll
  for (int k = 0; k < NW; ++k) cnt[k] = pk[k] = 0;
  for (int t0 = 0; t0 < H; t0 += 64) {
    const int ta = t0 + lane, tb = t0 + 32 + lane;
    uint32_t pa = 0, pb = 0;
#pragma unroll
    for (int j = 0; j < kFleetJMax; ++j) {
      if (j < J) {
        if (ta < H) pa += __ldg(bp[j] + ta);
        if (tb < H) pb += __ldg(bp[j] + tb);
      }
    }
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int t = half ? tb : ta;
      const uint32_t pre = half ? pb : pa;
      ring[t & (kFleetRing - 1)] = pre;
      __syncwarp();
      if (t < H) {
#pragma unroll
        for (int k = 0; k < NW; ++k) {
          const int w = win.w[k];
          if (t >= w - 1) {
            const int32_t S = (int32_t)(pre - ring[(t - w) & (kFleetRing - 1)]);
            cnt[k] += S > win.bw[k];
            pk[k] = max(pk[k], S);
          }
        }
      }
      __syncwarp();
    }
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

// Fleets of at most 8 jobs with 16-byte loads.  The workspace holds four
// copies of the prefix array, copy c shifted left by c samples
// (X_c[j][x] = PREX[j][x + c], zero past the end), so that for any offset the
// stream of job j starts 16-byte aligned in copy (o_j + 1) & 3.  Each lane
// composes 4 consecutive samples per load; one warp iteration covers 128.
// The 1024-slot ring keeps its size: windows of 128 samples or more read it
// before the block's prefixes are written (their starts all precede the
// block), shorter windows after (their starts lie at most 127 back).
template <bool EDGE, int NW>
__device__ __forceinline__ void fleet_block4(const uint32_t* ring, int T, int H, const uint4& pre,
                                             const FleetWindows& win, bool long_windows,
                                             int32_t (&cnt)[NW], int32_t (&pk)[NW]) {
  const uint32_t pv[4] = {pre.x, pre.y, pre.z, pre.w};
#pragma unroll
  for (int k = 0; k < NW; ++k) {
    const int w = win.w[k];
    if ((w >= 128) != long_windows) continue;
    uint32_t old[4];
    if ((w & 3) == 0) {
      const uint4 o4 = *reinterpret_cast<const uint4*>(ring + ((T - w) & (kFleetRing - 1)));
      old[0] = o4.x; old[1] = o4.y; old[2] = o4.z; old[3] = o4.w;
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) old[i] = ring[(T + i - w) & (kFleetRing - 1)];
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int32_t S = (int32_t)(pv[i] - old[i]);
      const bool in = !EDGE || (T + i < H && T + i >= w - 1);
      cnt[k] += (in && S > win.bw[k]);
      if (in) pk[k] = max(pk[k], S);
    }
  }
}

template <int NW>
__global__ void __launch_bounds__(32 * kFleetWarps)
    fleet_windows_v4_kernel(const uint32_t* __restrict__ prex4, int J, int64_t Lp, int64_t cs, StreamRows rows,
                            const int32_t* __restrict__ offsets, int64_t N, int H, FleetWindows win,
                            int wmax, int32_t* __restrict__ counts, int32_t* __restrict__ peaks) {
  __shared__ __align__(16) uint32_t ring_all[kFleetWarps][kFleetRing];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * kFleetWarps + wid;
  if (n >= N) return;  // the whole warp leaves together; no block-wide barrier follows
  uint32_t* ring = ring_all[wid];
  const uint4* bp[kFleetJMax];
  uint32_t pre_m1 = 0;
#pragma unroll
  for (int j = 0; j < kFleetJMax; ++j) {
    bp[j] = reinterpret_cast<const uint4*>(prex4);
    if (j < J) {
      const int32_t o = __ldg(offsets + n * J + j);
      const int s = o + 1, c = s & 3;
      bp[j] = reinterpret_cast<const uint4*>(prex4 + c * cs + (int64_t)rows.r[j] * Lp + (s - c));
      if (lane == j) pre_m1 = __ldg(prex4 + (int64_t)rows.r[j] * Lp + o);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) pre_m1 += __shfl_xor_sync(0xffffffffu, pre_m1, o);
  if (lane == 0) ring[kFleetRing - 1] = pre_m1;
  __syncwarp();
  int32_t cnt[NW], pk[NW];
#pragma unroll
  for (int k = 0; k < NW; ++k) cnt[k] = pk[k] = 0;
  for (int t0 = 0; t0 < H; t0 += 128) {
    const int T = t0 + 4 * lane;
    uint4 pre = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int j = 0; j < kFleetJMax; ++j) {
      if (j < J) {
        const uint4 v = __ldg(bp[j] + (t0 >> 2) + lane);
        pre.x += v.x; pre.y += v.y; pre.z += v.z; pre.w += v.w;
      }
    }
    const bool edge = t0 < wmax - 1 || t0 + 128 > H;
    if (edge) fleet_block4<true, NW>(ring, T, H, pre, win, true, cnt, pk);
    else fleet_block4<false, NW>(ring, T, H, pre, win, true, cnt, pk);
    __syncwarp();
    *reinterpret_cast<uint4*>(ring + (T & (kFleetRing - 1))) = pre;
    __syncwarp();
    if (edge) fleet_block4<true, NW>(ring, T, H, pre, win, false, cnt, pk);
    else fleet_block4<false, NW>(ring, T, H, pre, win, false, cnt, pk);
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

// copies 1..3 of nrows prefix rows for the 16-byte path (copy 0 is the rows
// themselves, copy c starts cs words after copy c - 1); entries past a row's
// last index are zero in every copy
__global__ void fleet_shift_copies_kernel(uint32_t* __restrict__ rows0, int nrows, int64_t Lp, int64_t cs,
                                          int64_t last) {
  const int64_t total = (int64_t)nrows * Lp;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t x = i % Lp;
    const uint32_t* row = rows0 + (i - x);
    if (x > last) rows0[i] = 0u;
#pragma unroll
    for (int c = 1; c < 4; ++c) rows0[c * cs + i] = x + c <= last ? row[x + c] : 0u;
  }
}

// row stride: PREX[j][0 .. L + H] plus the 127 words a 128-sample block of
// the 16-byte path may read past a stream's end, rounded to 16 bytes
static int64_t fleet_lp(int L, int H) { return (((int64_t)L + H + 1 + 127) + 3) / 4 * 4; }
static int fleet_ncopy(int J, int64_t workspace_bytes, int L, int H);
static int fleet_nchunk(int L, int H) { return (int)((((int64_t)L + H) + kFleetChunk - 1) / kFleetChunk); }

// rows = J job rows plus `extra` working rows, in each of ncopy copies
static int64_t fleet_bytes(int J, int L, int H, int ncopy, int extra = 0) {
  const int64_t prex = ((int64_t)ncopy * (J + extra) * fleet_lp(L, H) * 4 + 255) / 256 * 256;
  const int64_t tot = ((int64_t)J * fleet_nchunk(L, H) * 4 + 255) / 256 * 256;
  return prex + tot + 256 + 256;
}

// the least workspace (one prefix copy, 4-byte loads) and the workspace of
// the 16-byte path (four shifted copies; fleets of at most 8 jobs)
int64_t fleet_ws_min_bytes(int J, int L, int H) { return fleet_bytes(J, L, H, 1); }
int64_t fleet_ws_bytes(int J, int L, int H) { return fleet_bytes(J, L, H, J <= kFleetJMax ? 4 : 1); }
static int fleet_ncopy(int J, int64_t workspace_bytes, int L, int H) {
  return J <= kFleetJMax && workspace_bytes >= fleet_bytes(J, L, H, 4) ? 4 : 1;
}

// Per-job prefix sums (PREX) and validation of the traces, job map and
// offsets; returns the per-job maxima (for the int32 range checks).
static pe_status fleet_prepare(const float* traces, int G, int L, const int32_t* job_of_gpu, int J,
                               const int32_t* offsets, int64_t N, int H, void* workspace, int ncopy,
                               int extra, FleetWs& ws, int64_t& sum_max, cudaStream_t st) {
  char* base = reinterpret_cast<char*>(workspace);
  ws.Lp = fleet_lp(L, H);
  ws.nchunk = fleet_nchunk(L, H);
  const int64_t prex_bytes = ((int64_t)ncopy * (J + extra) * ws.Lp * 4 + 255) / 256 * 256;
  const int64_t tot_bytes = ((int64_t)J * ws.nchunk * 4 + 255) / 256 * 256;
  ws.prex = reinterpret_cast<uint32_t*>(base);
  ws.totals = reinterpret_cast<uint32_t*>(base + prex_bytes);
  ws.maxq = reinterpret_cast<int32_t*>(base + prex_bytes + tot_bytes);
  ws.flag = reinterpret_cast<int32_t*>(base + prex_bytes + tot_bytes + 256);
  PE_TRY_CUDA(cudaMemsetAsync(ws.maxq, 0, 256 + 4, st));
  {
    ProfScope ps(PE_PROF_FLEET_PREP, st);
    const dim3 grid(ws.nchunk, J);
    fleet_chunk_sums_kernel<<<grid, 256, 0, st>>>(traces, G, L, H, job_of_gpu, J, ws);
    fleet_chunk_scan_kernel<<<J, 32, 0, st>>>(ws);
    fleet_prefix_kernel<<<grid, 256, 0, st>>>(traces, G, L, H, job_of_gpu, J, ws);
    if (ncopy == 4)
      fleet_shift_copies_kernel<<<(int)std::min<int64_t>(ceil_div((int64_t)J * ws.Lp, 256), 4096), 256, 0, st>>>(
          ws.prex, J, ws.Lp, (int64_t)(J + extra) * ws.Lp, (int64_t)L + H);
    if (N > 0)
      fleet_check_offsets_kernel<<<(int)std::min<int64_t>(ceil_div(N * J, 256), 4096), 256, 0, st>>>(
          offsets, N * J, L, ws.flag);
  }
  PE_CHECK_LAUNCH("fleet prepare kernels");
  int32_t host[64 + 1];
  PE_TRY_CUDA(cudaMemcpyAsync(host, ws.maxq, sizeof(int32_t) * J, cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaMemcpyAsync(host + 64, ws.flag, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  const int32_t flag = host[64];
  if (flag & 1) return fail(PE_EOVERFLOW, "fleet trace holds a sample that is not finite or outside [0, %g] W", (double)kFleetMaxWatts);
  if (flag & 2) return fail(PE_EINVAL, "job_of_gpu entry outside [0, J)");
  if (flag & 4) return fail(PE_EINVAL, "fleet offset outside [0, L)");
  sum_max = 0;
  for (int j = 0; j < J; ++j) sum_max += host[j];
  return PE_OK;
}

pe_status fleet_launch(const float* traces, int G, int L, const int32_t* job_of_gpu, int J,
                       const int32_t* offsets, int64_t N, int H, const int32_t* windows, int W,
                       int64_t budget_q, int32_t* counts, int32_t* peaks, void* workspace,
                       int64_t workspace_bytes, cudaStream_t st) {
  FleetWs ws;
  int64_t sum_max = 0;
  const int ncopy = fleet_ncopy(J, workspace_bytes, L, H);
  pe_status s = fleet_prepare(traces, G, L, job_of_gpu, J, offsets, N, H, workspace, ncopy, 0, ws, sum_max, st);
  if (s != PE_OK) return s;
  FleetWindows win{};
  int wmax = 0;
  for (int k = 0; k < W; ++k) {
    const int64_t w = windows[k];
    if (sum_max * w >= (int64_t)INT_MAX || budget_q * w >= (int64_t)INT_MAX)
      return fail(PE_EOVERFLOW, "window %d: composed window sum may exceed int32", (int)w);
    win.w[k] = (int32_t)w;
    win.bw[k] = (int32_t)(budget_q * w);
    wmax = std::max(wmax, (int)w);
  }
  if (N == 0) return PE_OK;
  const int grid_n = (int)((N + kFleetWarps - 1) / kFleetWarps);
  const int64_t Lx = ws.Lp;
  ProfScope ps(PE_PROF_FLEET_WINDOWS, st);
  const int64_t cs = (int64_t)J * Lx;
  const StreamRows id = identity_rows();
  if (ncopy == 4) {
    switch (W) {
      case 1: fleet_windows_v4_kernel<1><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, cs, id, offsets, N, H, win, wmax, counts, peaks); break;
      case 2: fleet_windows_v4_kernel<2><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, cs, id, offsets, N, H, win, wmax, counts, peaks); break;
      case 3: fleet_windows_v4_kernel<3><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, cs, id, offsets, N, H, win, wmax, counts, peaks); break;
      default: fleet_windows_v4_kernel<4><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, cs, id, offsets, N, H, win, wmax, counts, peaks); break;
    }
  } else if (J <= kFleetJMax) {
    switch (W) {
      case 1: fleet_windows_j8_kernel<1><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, id, offsets, N, H, win, counts, peaks); break;
      case 2: fleet_windows_j8_kernel<2><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, id, offsets, N, H, win, counts, peaks); break;
      case 3: fleet_windows_j8_kernel<3><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, id, offsets, N, H, win, counts, peaks); break;
      default: fleet_windows_j8_kernel<4><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, id, offsets, N, H, win, counts, peaks); break;
    }
  } else {
    switch (W) {
      case 1: fleet_windows_kernel<1><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, offsets, N, H, win, counts, peaks); break;
      case 2: fleet_windows_kernel<2><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, offsets, N, H, win, counts, peaks); break;
      case 3: fleet_windows_kernel<3><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, offsets, N, H, win, counts, peaks); break;
      default: fleet_windows_kernel<4><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, J, Lx, offsets, N, H, win, counts, peaks); break;
    }
  }
  PE_CHECK_LAUNCH("fleet_windows_kernel");
  return PE_OK;
}

// ---------------------------------------------------------------------------
// Phase-staggered schedule (Sec. 8): jobs placed greedily in index order.
// Stage j composes jobs 0..j with the earlier offsets fixed and job j at
// every candidate c * stride; the windows kernel (first j + 1 jobs of the
// prefix array) gives each candidate's peak, and a one-block argmin keeps
// the lowest candidate among equal peaks.  The chosen offsets never leave
// the device between stages.
// ---------------------------------------------------------------------------
// candidate c's stream offsets: (0 for the partial-fleet row, c * stride)
// from the second stage on, (c * stride) alone for the first job
__global__ void stagger_candidates_kernel(int32_t* __restrict__ cand, int64_t ncand, int per, int stride) {
  const int64_t total = ncand * per;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t c = i / per;
    cand[i] = (int)(i % per) == per - 1 ? (int32_t)(c * stride) : 0;
  }
}

// partial-fleet row R[y] = sum over the placed jobs k < j of PREX[k][o_k + y]
// for y in [0, H] (zero past H): stage j adds job j - 1 at its chosen
// offset (stage 1 starts from zero).  With offset 0, R composes like a job.
__global__ void stagger_compose_kernel(uint32_t* __restrict__ R, const uint32_t* __restrict__ prex, int64_t Lp,
                                       int jprev, const int32_t* __restrict__ chosen, int H) {
  const int32_t o = chosen[jprev];
  const uint32_t* src = prex + (int64_t)jprev * Lp + o;
  for (int64_t y = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; y < Lp; y += (int64_t)gridDim.x * blockDim.x)
    R[y] = y <= H ? (jprev > 0 ? R[y] : 0u) + src[y] : 0u;
}

__global__ void __launch_bounds__(1024) stagger_argmin_kernel(const int32_t* __restrict__ peaks, int64_t ncand,
                                                              int stride, int j, int32_t* __restrict__ chosen,
                                                              int32_t* __restrict__ chosen_peak) {
  __shared__ int32_t sp[32];
  __shared__ int64_t sc[32];
  int32_t bp = INT_MAX;
  int64_t bc = ncand;
  for (int64_t c = threadIdx.x; c < ncand; c += blockDim.x) {
    const int32_t p = peaks[c];
    if (p < bp) {  // ascending scan: the first (lowest) candidate of a tie stays
      bp = p;
      bc = c;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int32_t op = __shfl_xor_sync(0xffffffffu, bp, o);
    const int64_t oc = __shfl_xor_sync(0xffffffffu, bc, o);
    if (op < bp || (op == bp && oc < bc)) {
      bp = op;
      bc = oc;
    }
  }
  if ((threadIdx.x & 31) == 0) {
    sp[threadIdx.x >> 5] = bp;
    sc[threadIdx.x >> 5] = bc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
      if (sp[w] < bp || (sp[w] == bp && sc[w] < bc)) {
        bp = sp[w];
        bc = sc[w];
      }
    chosen[j] = (int32_t)(bc * stride);
    chosen_peak[j] = bp;
  }
}

static int64_t stagger_ncand(int L, int stride) { return ((int64_t)L + stride - 1) / stride; }

// four prefix copies of the J job rows and the partial-fleet row, then two
// candidate offsets and a peak and count per candidate
static int64_t stagger_prefix_bytes(int J, int L, int H) { return fleet_bytes(J, L, H, 4, 1); }

int64_t fleet_stagger_ws_bytes(int J, int L, int H, int stride) {
  const int64_t nc = stagger_ncand(L, stride);
  const int64_t cand = (nc * 2 * 4 + 255) / 256 * 256;
  const int64_t outs = (nc * 4 + 255) / 256 * 256;
  return stagger_prefix_bytes(J, L, H) + cand + 2 * outs;
}

pe_status fleet_stagger_launch(const float* traces, int G, int L, const int32_t* job_of_gpu, int J, int H,
                               int w, int stride, int32_t* offsets_out, int32_t* peaks_out, void* workspace,
                               cudaStream_t st) {
  FleetWs ws;
  int64_t sum_max = 0;
  // job rows 0..J-1 and the partial-fleet row J, in four shifted copies
  pe_status s = fleet_prepare(traces, G, L, job_of_gpu, J, nullptr, 0, H, workspace, 4, 1, ws, sum_max, st);
  if (s != PE_OK) return s;
  if (sum_max * w >= (int64_t)INT_MAX) return fail(PE_EOVERFLOW, "window %d: composed window sum may exceed int32", w);
  const int64_t nc = stagger_ncand(L, stride);
  char* base = reinterpret_cast<char*>(workspace) + stagger_prefix_bytes(J, L, H);
  int32_t* cand = reinterpret_cast<int32_t*>(base);
  int32_t* cnt = reinterpret_cast<int32_t*>(base + (nc * 2 * 4 + 255) / 256 * 256);
  int32_t* pk = cnt + (nc * 4 + 255) / 256 * 64;
  const int64_t cs = (int64_t)(J + 1) * ws.Lp;
  uint32_t* R = ws.prex + (int64_t)J * ws.Lp;
  FleetWindows win{};
  win.w[0] = w;
  win.bw[0] = INT_MAX;  // counts unused
  const int grid_n = (int)((nc + kFleetWarps - 1) / kFleetWarps);
  for (int j = 0; j < J; ++j) {
    // stage j composes two streams: the partial fleet of jobs 0..j-1 (row J,
    // offset 0) and job j at each candidate; the first stage has job 0 alone
    const int per = j == 0 ? 1 : 2;
    StreamRows rows = identity_rows();
    if (j > 0) {
      rows.r[0] = J;
      rows.r[1] = j;
    }
    {
      ProfScope ps(PE_PROF_FLEET_PREP, st);
      if (j > 0) {
        const int gb = (int)std::min<int64_t>(ceil_div(ws.Lp, 256), 4096);
        stagger_compose_kernel<<<gb, 256, 0, st>>>(R, ws.prex, ws.Lp, j - 1, offsets_out, H);
        fleet_shift_copies_kernel<<<gb, 256, 0, st>>>(R, 1, ws.Lp, cs, (int64_t)H);
      }
      stagger_candidates_kernel<<<(int)std::min<int64_t>(ceil_div(nc * per, 256), 4096), 256, 0, st>>>(
          cand, nc, per, stride);
    }
    {
      ProfScope ps(PE_PROF_FLEET_WINDOWS, st);
      fleet_windows_v4_kernel<1><<<grid_n, 32 * kFleetWarps, 0, st>>>(ws.prex, per, ws.Lp, cs, rows, cand, nc, H,
                                                                        win, w, cnt, pk);
    }
    {
      ProfScope ps(PE_PROF_FLEET_PREP, st);
      stagger_argmin_kernel<<<1, 1024, 0, st>>>(pk, nc, stride, j, offsets_out, peaks_out);
    }
    PE_CHECK_LAUNCH("fleet stagger kernels");
  }
  return PE_OK;
}

}  // namespace pe
