// bf16 policy/value MLPs on the 5th-generation tensor cores (tcgen05), and the
// decoupled rollout that uses them (72B workload: D=32, H=256, A=16, C=4;
// Stress: D=64, H=512).
//
// A policy/value network is tanh(W2 tanh(W1 x + b1) + b2) followed by a
// linear head (Sec. 4.2 actor-critic), evaluated on 128-row tiles:
//   - the fp32 master parameters are first converted once per call into a
//     bf16 "weight image": each matrix laid out exactly as the kernels keep
//     it in shared memory (K-major, 128-byte or 64-byte swizzle), W2 in
//     32 KB K-blocks that stream through a two-slot ring;
//   - per layer one thread issues tcgen05.mma (M=128, K=16 per instruction)
//     into TMEM; sixteen warps read the fp32 accumulators back (tcgen05.ld),
//     add the bias, apply tanh, round to bf16 and write the next layer's A
//     operand into shared memory in the swizzled layout;
//   - 72B (mlp_bf16_pair_kernel): two tiles in flight per CTA, so that the
//     epilogue of one overlaps the MMAs of the other; Stress
//     (mlp_bf16_stream_kernel): one tile at a time, its 592 KB of weights
//     streamed, the layer-2 MMAs overlapping the epilogues per 256-column
//     half.
// Precision: bf16 observations, weights and hidden activations, fp32
// accumulation, fp32 bias and tanh -- the quantisation points the oracle
// emulates.
#include <algorithm>
#include <type_traits>

#include "bf16_layout.cuh"
#include "env.cuh"
#include "mlp_f32.cuh"
#include "tc.cuh"

namespace pe {

// set when a bounded tensor-core wait gives up; read and cleared by pe_device_check
__device__ int32_t g_tc_error = 0;

// fp32 canonical parameters -> bf16 swizzled weight image of one network
// (policy: W1 W2 W3 of A rows; value: V1 V2 V3 of 1 row), rows >= nout of the
// head are zero.
template <int D, int H>
__global__ void weight_image_kernel(const float* __restrict__ params, int A, int value_first,
                                    uint8_t* __restrict__ img0, int64_t img_stride) {
  using I = Img<D, H>;
  // blockIdx.y selects the network: value_first + y (0 policy, 1 value)
  const int value_net = value_first + (int)blockIdx.y;
  uint8_t* img = img0 + blockIdx.y * img_stride;
  const MlpLayout Lp = mlp_layout(D, H, A);
  const float* w1 = params + (value_net ? Lp.v1 : Lp.w1);
  const float* w2 = params + (value_net ? Lp.v2 : Lp.w2);
  const float* w3 = params + (value_net ? Lp.v3 : Lp.w3);
  const int nout = value_net ? 1 : A;
  const int total = H * D + H * H + kHeadN * H;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    int mat, r, k;
    float v;
    if (i < H * D) {
      mat = 1, r = i / D, k = i % D, v = w1[i];
    } else if (i < H * D + H * H) {
      const int j = i - H * D;
      mat = 2, r = j / H, k = j % H, v = w2[j];
    } else {
      const int j = i - H * D - H * H;
      mat = 3, r = j / H, k = j % H, v = r < nout ? w3[r * H + k] : 0.0f;
    }
    *reinterpret_cast<__nv_bfloat16*>(img + fwd_img_offset<D, H>(mat, r, k)) = __float2bfloat16_rn(v);
  }
}

// ---------------------------------------------------------------------------
// Streamed variant for networks whose weights do not fit in shared memory
// (Stress: D=64, H=512; 592 KB of bf16 weights).  The 128-row activation
// tile stays resident (128 KB); the weights flow through a two-slot ring of
// 32 KB stages, each the B operand of one (N-half, K-block) of a layer:
//   layer 1: 2 stages (N-halves of W1, K=64), layer 2: 16 stages (2 N-halves x
//   8 K-blocks of W2), head: 1 stage (W3, 16 rows x 8 K-blocks).
// Warp roles: warps 0-15 run the epilogues, warp 16 issues cp.async.bulk for
// stage s into slot s%2 once the MMAs that read the slot's previous stage
// have completed (tcgen05.commit on the slot's "empty" barrier), warp 17
// issues the MMAs.  A layer's 512 accumulator columns fill TMEM, so a tile
// cannot overlap another tile; instead the epilogues hand over per 256-column
// half, and the layer-2 MMAs run beside them:
//   epilogue 1, half A (h1 columns 0-255) -> MMAs of layer-2 N-half 0 over
//   K-blocks 0-3 run during epilogue 1, half B; once half B is written, the
//   rest of N-half 0, then N-half 1;
//   epilogue 2, half A (N-half 0) runs during the N-half 1 MMAs; its first
//   results wait in registers until the N-half 1 MMAs have read h1's first
//   four K-blocks, which h2 overwrites in place;
//   the head accumulates in TMEM columns 256-271, so the next tile's layer-1
//   N-half 0 can start while warps 0-3 copy the head accumulators to shared
//   memory (they compute the loss later, during the next tile's layer-2
//   N-half 0 MMAs) and warps 4-15 write the next tile's X (its rows fetched
//   during the previous epilogue) into the buffer's last K-block, which only
//   epilogue 1, half B overwrites.
// The accumulation order of every accumulator is that of the serial kernel,
// so the results are the same bits.  One launch may also cover two networks
// over the same rows (the policy, then the value network of a PPO forward):
// the tiles of both form one list spread over the persistent CTAs, which
// balances a tile count that is not a multiple of the SM count.
// ---------------------------------------------------------------------------
constexpr int kComputeThreads = 512;
constexpr int kStreamThreads = kComputeThreads + 64;

// the second network of a two-network stream launch (img == NULL: one network)
struct MlpSecond {
  const uint8_t* img;
  MlpSave save;
};

template <int D, int H>
__global__ void weight_image_stream_kernel(const float* __restrict__ params, int A, int value_first,
                                           uint8_t* __restrict__ img0, int64_t img_stride) {
  using I = ImgS<D, H>;
  const int value_net = value_first + (int)blockIdx.y;
  uint8_t* img = img0 + blockIdx.y * img_stride;
  const MlpLayout Lp = mlp_layout(D, H, A);
  const float* w1 = params + (value_net ? Lp.v1 : Lp.w1);
  const float* w2 = params + (value_net ? Lp.v2 : Lp.w2);
  const float* w3 = params + (value_net ? Lp.v3 : Lp.w3);
  const int nout = value_net ? 1 : A;
  const int total = H * D + H * H + kHeadN * H;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    int mat, r, k;
    float v;
    if (i < H * D) {
      mat = 1, r = i / D, k = i % D, v = w1[i];
    } else if (i < H * D + H * H) {
      const int j = i - H * D;
      mat = 2, r = j / H, k = j % H, v = w2[j];
    } else {
      const int j = i - H * D - H * H;
      mat = 3, r = j / H, k = j % H, v = r < nout ? w3[r * H + k] : 0.0f;
    }
    *reinterpret_cast<__nv_bfloat16*>(img + fwd_img_offset<D, H>(mat, r, k)) = __float2bfloat16_rn(v);
  }
}

template <int D, int H>
struct MlpStreamSmem {
  alignas(1024) uint8_t act[kTcRows * H * 2];  // X (last K-block), then h1, then h2 (in place)
  alignas(1024) uint8_t ring[2][kStageBytes];
  float headv[kTcRows][kHeadN];                // the previous tile's head accumulators (warps 0-3)
  float b1[2][H], b2[2][H], b3[2][kHeadN];     // per network of the launch
  uint64_t full[2], empty[2], fin;
  // one completion per tile each: X written (warps 4-15), head read out of
  // TMEM (warps 0-3), layer-1 N-halves done, h1 halves written, layer-2
  // N-half 0 done, N-half 1 past K-block 3, N-half 1 done, h2 written, head done
  uint64_t xin, hd, m1a, m1b, h1a, h1b, m2a, n1lo, m2b, h2in, mh;
  uint32_t tmem_base;
  int32_t err;
};

template <int D, int H>
__global__ void __launch_bounds__(kStreamThreads, 1)
    mlp_bf16_stream_kernel(const uint8_t* __restrict__ img, const float* __restrict__ params, int A,
                           int value_net, const __nv_bfloat16* __restrict__ obs, int64_t n,
                           float* __restrict__ out, int out_stride, int nout, int32_t* __restrict__ err,
                           MlpSave save, MlpSecond second) {
  using I = ImgS<D, H>;
  static_assert(D == 64 && H == 512, "two 256-column halves per layer; X is one 128-byte K-block");
  constexpr int NJ = H / 2 / 4 / 16;                 // 16-column chunks per warp and half
  constexpr int KBH = H / 2 / 64;                    // K-blocks of h per half
  constexpr int kXOff = (H / 64 - 1) * kTcRows * 128;  // X sits in the last K-block of the buffer
  constexpr int XCPR = D / 8;                        // 16-byte observation chunks per row
  constexpr int XCH = (kTcRows * XCPR + 383) / 384;  // per X-writing thread (warps 4-15)
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  MlpStreamSmem<D, H>& s = *reinterpret_cast<MlpStreamSmem<D, H>*>(base);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const MlpLayout Lp = mlp_layout(D, H, A);
  const bool two = second.img != nullptr;
  const int nnet = two ? 2 : 1;
  if (tid == 0) {
    s.err = 0;
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.full[i], 1);
      tc::mbar_init(&s.empty[i], 1);
    }
    tc::mbar_init(&s.fin, 1);
    tc::mbar_init(&s.xin, 12);
    tc::mbar_init(&s.hd, 4);
    tc::mbar_init(&s.m1a, 1);
    tc::mbar_init(&s.m1b, 1);
    tc::mbar_init(&s.h1a, 16);
    tc::mbar_init(&s.h1b, 16);
    tc::mbar_init(&s.m2a, 1);
    tc::mbar_init(&s.n1lo, 1);
    tc::mbar_init(&s.m2b, 1);
    tc::mbar_init(&s.h2in, 16);
    tc::mbar_init(&s.mh, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&s.tmem_base, 512);
  for (int k = 0; k < nnet; ++k) {
    const int vn = two ? k : value_net;
    const int no = two ? (k ? 1 : A) : nout;
    for (int i = tid; i < H; i += blockDim.x) {
      s.b1[k][i] = __ldg(params + (vn ? Lp.c1 : Lp.b1) + i);
      s.b2[k][i] = __ldg(params + (vn ? Lp.c2 : Lp.b2) + i);
    }
    if (tid < kHeadN) s.b3[k][tid] = tid < no ? __ldg(params + (vn ? Lp.c3 : Lp.b3) + tid) : 0.0f;
  }
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = s.tmem_base;
  const int64_t tiles = (n + kTcRows - 1) / kTcRows;  // per network
  const int my_tiles = (int)((tiles * nnet - blockIdx.x + gridDim.x - 1) / gridDim.x);
  // this CTA's k-th tile: its network (ni) and its tile index within that network
  auto tile_of = [&](int k, int& ni) -> int64_t {
    const int64_t g = (int64_t)blockIdx.x + (int64_t)k * gridDim.x;
    ni = g >= tiles ? 1 : 0;
    return g - ni * tiles;
  };
  // a bounded wait that is skipped once the CTA has an error
  auto wt = [&](uint64_t* b, uint32_t par) -> bool {
    if (*reinterpret_cast<volatile int32_t*>(&s.err)) return false;
    if (tc::mbar_wait(b, par)) return true;
    atomicExch(&s.err, 1);
    return false;
  };
  int last_issued = -1;  // producer: global index of its last issued stage
  if (warp == 16) {
    // producer: every stage of every tile of this CTA, in consumption order
    if (lane == 0) {
      int gs = 0;
      bool ok = true;
      for (int t = 0; t < my_tiles && ok; ++t) {
        int ni;
        (void)tile_of(t, ni);
        const uint8_t* timg = ni ? second.img : img;
        for (int st = 0; st < kStreamStages && ok; ++st) {
          const int slot = gs & 1;
          if (gs >= 2 && !wt(&s.empty[slot], ((gs - 2) >> 1) & 1)) {
            ok = false;
            break;
          }
          tc::mbar_expect_tx(&s.full[slot], (uint32_t)I::stage_bytes(st));
          tc::bulk_g2s(s.ring[slot], timg + I::stage_off(st), (uint32_t)I::stage_bytes(st), &s.full[slot]);
          last_issued = gs++;
        }
      }
    }
  } else if (warp == 17) {
    // MMA issuer
    if (lane == 0) {
      const uint32_t xa = tc::smem_u32(s.act);
      constexpr uint32_t kIdN = tc::idesc_bf16(kTcRows, 256);
      constexpr uint32_t kIdH = tc::idesc_bf16(kTcRows, kHeadN);
      int gs = 0;
      auto stage_in = [&]() -> uint32_t {
        const int slot = gs & 1;
        (void)wt(&s.full[slot], (gs >> 1) & 1);
        tc::fence_after();
        return tc::smem_u32(s.ring[slot]);
      };
      auto stage_out = [&]() {
        tc::mma_commit(&s.empty[gs & 1]);
        ++gs;
      };
      // layer 2: K-blocks [k0, k1) of h1 into N-half h (TMEM columns 256 h ..)
      auto layer2 = [&](int h, int k0, int k1) {
#pragma unroll 1
        for (int kb = k0; kb < k1; ++kb) {
          const uint32_t ra = stage_in();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc::mma_bf16(tmem + h * 256, tc::desc_kmajor(xa + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                         tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, (kb | kk) != 0);
          stage_out();
        }
      };
      for (int t = 0; t < my_tiles; ++t) {
        const uint32_t par = t & 1;
        (void)wt(&s.xin, par);
        tc::fence_after();
        // layer 1, N-half h; N-half 1 overwrites the columns of the previous tile's head
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          if (h == 1 && t > 0) {
            (void)wt(&s.hd, par ^ 1);
            tc::fence_after();
          }
          const uint32_t ra = stage_in();
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk)
            tc::mma_bf16(tmem + h * 256, tc::desc_kmajor(xa + kXOff + kk * 32, 1024, tc::kLayoutSW128),
                         tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, kk > 0);
          stage_out();
          tc::mma_commit(h ? &s.m1b : &s.m1a);
        }
        (void)wt(&s.h1a, par);
        tc::fence_after();
        layer2(0, 0, KBH);
        (void)wt(&s.h1b, par);
        tc::fence_after();
        layer2(0, KBH, 2 * KBH);
        tc::mma_commit(&s.m2a);
        layer2(1, 0, KBH);
        tc::mma_commit(&s.n1lo);
        layer2(1, KBH, 2 * KBH);
        tc::mma_commit(&s.m2b);
        // head: TMEM columns 256 .. 271 = H2 W3^T (one 16 KB stage)
        (void)wt(&s.h2in, par);
        tc::fence_after();
        const uint32_t ra = stage_in();
#pragma unroll 1
        for (int kb = 0; kb < H / 64; ++kb)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc::mma_bf16(tmem + 256, tc::desc_kmajor(xa + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                         tc::desc_kmajor(ra + kb * kHeadN * 128 + kk * 32, 1024, tc::kLayoutSW128), kIdH,
                         (kb | kk) != 0);
        stage_out();
        tc::mma_commit(&s.mh);
      }
      // every MMA of this CTA completes before TMEM is released
      tc::mma_commit(&s.fin);
      if (!tc::mbar_wait(&s.fin, 0)) atomicExch(&s.err, 1);
    }
  } else {
    // epilogue warps: four TMEM lane quadrants x four column slices
    const int quad = warp & 3, slice = warp >> 2, row = quad * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const int xt = tid - 128;  // X-writing thread index (warps 4-15)
    uint4 xv[XCH];
    auto fetch_x = [&](int k) {
      int ni = 0;
      const int64_t tl = k < my_tiles ? tile_of(k, ni) : 0;
      const uint32_t* gather = ni ? second.save.gather : save.gather;
#pragma unroll
      for (int q = 0; q < XCH; ++q) {
        const int i = xt + q * 384, r = i / XCPR, c = i % XCPR;
        const int64_t rr = tl * kTcRows + r;
        xv[q] = make_uint4(0, 0, 0, 0);
        if (k < my_tiles && i < kTcRows * XCPR && rr < n) {
          const int64_t src = gather ? (int64_t)__ldg(gather + rr) : rr;
          xv[q] = __ldg(reinterpret_cast<const uint4*>(obs + src * D) + c);
        }
      }
    };
    auto handover = [&](uint64_t* bar) {
      tc::fence_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
    };
    // columns c .. c + 15 of this thread's row: tanh(acc + bias), packed bf16
    auto chunk = [&](int c, const float* bias, uint32_t (&pk)[8]) {
      float v[16];
      tc::tmem_ld16(lane_addr + (uint32_t)c, v);
      tc::tanh16_bf16(v, bias + c, pk);
    };
    // ... into the activation buffer (the next A operand) and the tile image g
    auto put = [&](int c, const uint32_t (&pk)[8], uint8_t* g) {
      const uint32_t o0 = tc::swz_offset<128>(row, c, kTcRows), o1 = tc::swz_offset<128>(row, c + 8, kTcRows);
      const uint4 lo = make_uint4(pk[0], pk[1], pk[2], pk[3]), hi = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      *reinterpret_cast<uint4*>(s.act + o0) = lo;
      *reinterpret_cast<uint4*>(s.act + o1) = hi;
      if (g) {
        *reinterpret_cast<uint4*>(g + o0) = lo;
        *reinterpret_cast<uint4*>(g + o1) = hi;
      }
    };
    // head of this CTA's k-th tile from its 16 accumulators (warps 0-3, one row per thread)
    auto head_out = [&](int k, const float (&v)[16]) {
      int ni;
      const int64_t tl = tile_of(k, ni);
      if (ni) {
        ppo_head_row(second.save.loss, 1, A, s.b3[1], second.save.gather, tl, row, n, v, warp);
      } else if (save.loss.dz) {
        ppo_head_row(save.loss, value_net, A, s.b3[0], save.gather, tl, row, n, v, warp);
      } else if (tl * kTcRows + row < n) {
        float* o = out + (tl * kTcRows + row) * out_stride;
#pragma unroll
        for (int j = 0; j < kHeadN; ++j)
          if (j < nout) o[j] = v[j] + s.b3[0][j];
      }
    };
    if (warp >= 4) fetch_x(0);
    for (int t = 0; t < my_tiles; ++t) {
      const uint32_t par = t & 1;
      int ni;
      const int64_t tile = tile_of(t, ni);
      __nv_bfloat16* const sx = ni ? second.save.x : save.x;
      __nv_bfloat16* const sh1 = ni ? second.save.h1 : save.h1;
      __nv_bfloat16* const sh2 = ni ? second.save.h2 : save.h2;
      uint8_t* const gh1 = sh1 ? reinterpret_cast<uint8_t*>(sh1) + tile * (int64_t)(kTcRows * H * 2) : nullptr;
      uint8_t* const gh2 = sh2 ? reinterpret_cast<uint8_t*>(sh2) + tile * (int64_t)(kTcRows * H * 2) : nullptr;
      const float* const b1 = s.b1[ni];
      const float* const b2 = s.b2[ni];
      if (t > 0) (void)wt(&s.mh, par ^ 1);  // the previous tile's head is done
      tc::fence_after();
      if (warp < 4) {
        // its accumulators out of TMEM (the loss comes later, while the
        // layer-2 MMAs run), so that layer 1 may take the columns
        if (t > 0) {
          float v[16];
          tc::tmem_ld16(lane_addr + 256u, v);
#pragma unroll
          for (int j = 0; j < kHeadN; j += 4)
            *reinterpret_cast<float4*>(&s.headv[row][j]) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
          tc::fence_before();
          __syncwarp();
          if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(&s.hd)) : "memory");
        }
      } else {
        // this tile's X (the previous tile's head MMA has read h2)
#pragma unroll
        for (int q = 0; q < XCH; ++q) {
          const int i = xt + q * 384;
          if (i < kTcRows * XCPR) {
            const int r = i / XCPR, c = i % XCPR;
            const uint32_t off = tc::swz_offset<128>(r, c * 8, kTcRows);
            *reinterpret_cast<uint4*>(s.act + kXOff + off) = xv[q];
            if (sx)
              *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(sx) + tile * (int64_t)(kTcRows * D * 2) + off) =
                  xv[q];
          }
        }
        handover(&s.xin);
      }
      // epilogue 1, half A (h1 K-blocks 0-3), then half B (K-blocks 4-7, the
      // last of which held X: layer-1 N-half 1 is done by then)
      (void)wt(&s.m1a, par);
      tc::fence_after();
#pragma unroll 1
      for (int j = 0; j < NJ; ++j) {
        const int c = slice * (H / 8) + j * 16;
        uint32_t pk[8];
        chunk(c, b1, pk);
        put(c, pk, gh1);
      }
      handover(&s.h1a);
      (void)wt(&s.m1b, par);
      tc::fence_after();
#pragma unroll 1
      for (int j = 0; j < NJ; ++j) {
        const int c = H / 2 + slice * (H / 8) + j * 16;
        uint32_t pk[8];
        chunk(c, b1, pk);
        put(c, pk, gh1);
      }
      handover(&s.h1b);
      // the previous tile's head epilogue, while the rest of layer-2 N-half 0 runs
      if (warp < 4 && t > 0) {
        float v[16];
#pragma unroll
        for (int j = 0; j < kHeadN; j += 4) {
          const float4 q = *reinterpret_cast<const float4*>(&s.headv[row][j]);
          v[j] = q.x, v[j + 1] = q.y, v[j + 2] = q.z, v[j + 3] = q.w;
        }
        head_out(t - 1, v);
      }
      // epilogue 2, half A: h2 overwrites h1's K-blocks 0-3 only after the
      // N-half 1 MMAs have read them; the first two chunks wait in registers
      (void)wt(&s.m2a, par);
      tc::fence_after();
      {
        const int c0 = slice * (H / 8);
        uint32_t p0[8], p1[8];
        chunk(c0, b2, p0);
        chunk(c0 + 16, b2, p1);
        (void)wt(&s.n1lo, par);
        tc::fence_after();
        put(c0, p0, gh2);
        put(c0 + 16, p1, gh2);
#pragma unroll 1
        for (int j = 2; j < NJ; ++j) {
          const int c = c0 + j * 16;
          uint32_t pk[8];
          chunk(c, b2, pk);
          put(c, pk, gh2);
        }
      }
      (void)wt(&s.m2b, par);
      tc::fence_after();
#pragma unroll 1
      for (int j = 0; j < NJ; ++j) {
        const int c = H / 2 + slice * (H / 8) + j * 16;
        uint32_t pk[8];
        chunk(c, b2, pk);
        put(c, pk, gh2);
      }
      handover(&s.h2in);
      // the next tile's observation rows, fetched while its X slot waits for this tile's head MMA
      if (warp >= 4) fetch_x(t + 1);
    }
    // the last tile's head
    if (warp < 4 && my_tiles > 0) {
      (void)wt(&s.mh, (my_tiles - 1) & 1);
      tc::fence_after();
      float v[16];
      tc::tmem_ld16(lane_addr + 256u, v);
      head_out(my_tiles - 1, v);
    }
  }
  tc::fence_before();
  __syncthreads();
  // on an error, the producer waits (bounded) for the copies it may still
  // have in flight (at most one per ring slot) before the CTA leaves
  if (s.err && warp == 16 && lane == 0)
    for (int q = last_issued - 1; q <= last_issued; ++q)
      if (q >= 0) (void)tc::mbar_wait(&s.full[q & 1], (q >> 1) & 1);
  if (tid == 0 && s.err) {
    atomicExch(&g_tc_error, 1);
    if (err) atomicExch(err, 1);
  }
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// Two tiles in flight (72B network, H = 256): with one tile per CTA, the
// chain of layer MMA, then an epilogue that waits for it, then the next MMA
// leaves the tensor core idle during every epilogue and the epilogue warps
// idle during every MMA.  Here a CTA holds two 128-row tiles
// (slots 0 and 1), each with its own activation buffer and its own half of
// TMEM (columns 256 s .. 256 s + 255 for layer 1, layer 2 and the head in
// turn), and runs them half a stage apart: the epilogue of one slot overlaps
// the MMAs of the other.  Shared memory holds two activation tiles (128 KB),
// so W2 (128 KB) is streamed from L2 in 32 KB K-blocks through a two-slot
// ring instead of staying resident; W1, W3 and the biases stay resident.
// Warp roles: warps 0-15 run the epilogues (TMEM -> bias, tanh, bf16 ->
// shared memory), warp 16 streams the W2 stages, warp 17 issues the MMAs.
// The roles hand over through mbarriers (one completion per tile pair):
//   xin[s], h1in[s], h2in[s]: the 16 epilogue warps have written the slot's
//                             X, h1 or h2 (count 16, lane 0 of each warp);
//   mma1[s], mma2[s], head[s]: the slot's layer-1, layer-2, head MMAs are
//                             done (tcgen05.commit).
// The arithmetic of every tile is that of a one-tile kernel (the same MMAs
// in the same order, the same epilogue), so the results are the same bits.
// ---------------------------------------------------------------------------
constexpr int kPairThreads = 576;
constexpr int kPairW2Stage = 32768;  // one K-block of 64 of W2 (256 rows x 128 B)

template <int D, int H>
struct MlpPairSmem {
  alignas(1024) uint8_t act[2][kTcRows * H * 2];  // per slot: X (aliases the start), then h1, then h2
  alignas(1024) uint8_t ring[2][kPairW2Stage];
  alignas(1024) uint8_t w1[Img<D, H>::W1];
  alignas(1024) uint8_t w3[Img<D, H>::W3];
  float b1[H], b2[H], b3[kHeadN];
  uint64_t bar_w, full[2], empty[2], mma1[2], mma2[2], head[2], xin[2], h1in[2], h2in[2];
  uint32_t tmem_base;
  int32_t err;
};

template <int D, int H>
__global__ void __launch_bounds__(kPairThreads, 1)
    mlp_bf16_pair_kernel(const uint8_t* __restrict__ img, const float* __restrict__ params, int A,
                         int value_net, const __nv_bfloat16* __restrict__ obs, int64_t n,
                         float* __restrict__ out, int out_stride, int nout, int32_t* __restrict__ err,
                         MlpSave save) {
  using I = Img<D, H>;
  static_assert(H == 256, "two tiles in flight need 2 x 256 TMEM columns");
  constexpr int KB2 = H / 64;   // W2 stages per tile
  constexpr int CPR = D / 8;    // 16-byte observation chunks per row
  constexpr int XCH = kTcRows * CPR / kTcThreads;
  static_assert(kTcRows * CPR % kTcThreads == 0, "observation chunks per thread");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  MlpPairSmem<D, H>& s = *reinterpret_cast<MlpPairSmem<D, H>*>(base);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const MlpLayout Lp = mlp_layout(D, H, A);
  if (tid == 0) {
    s.err = 0;
    tc::mbar_init(&s.bar_w, 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.full[i], 1);
      tc::mbar_init(&s.empty[i], 1);
      tc::mbar_init(&s.mma1[i], 1);
      tc::mbar_init(&s.mma2[i], 1);
      tc::mbar_init(&s.head[i], 1);
      tc::mbar_init(&s.xin[i], 16);
      tc::mbar_init(&s.h1in[i], 16);
      tc::mbar_init(&s.h2in[i], 16);
    }
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&s.tmem_base, 512);
  for (int i = tid; i < H; i += blockDim.x) {
    s.b1[i] = __ldg(params + (value_net ? Lp.c1 : Lp.b1) + i);
    s.b2[i] = __ldg(params + (value_net ? Lp.c2 : Lp.b2) + i);
  }
  if (tid < kHeadN) s.b3[tid] = tid < nout ? __ldg(params + (value_net ? Lp.c3 : Lp.b3) + tid) : 0.0f;
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = s.tmem_base;
  const int64_t tiles = (n + kTcRows - 1) / kTcRows;
  const int my_tiles = (int)((tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);
  const int npairs = (my_tiles + 1) / 2;
  int last_issued = -1;
  if (warp == 16) {
    // producer: W2's K-blocks for every tile slot, in the issuer's order
    if (lane == 0) {
      int gs = 0;
      for (int p = 0; p < npairs; ++p)
        for (int sl = 0; sl < 2; ++sl)
          for (int kb = 0; kb < KB2; ++kb, ++gs) {
            const int slot = gs & 1;
            if (gs >= 2 && !tc::mbar_wait(&s.empty[slot], ((gs - 2) >> 1) & 1)) atomicExch(&s.err, 1);
            tc::mbar_expect_tx(&s.full[slot], (uint32_t)kPairW2Stage);
            tc::bulk_g2s(s.ring[slot], img + I::W1 + (int64_t)kb * kPairW2Stage, (uint32_t)kPairW2Stage,
                         &s.full[slot]);
            last_issued = gs;
          }
    }
  } else if (warp == 17) {
    // MMA issuer
    if (lane == 0) {
      tc::mbar_expect_tx(&s.bar_w, (uint32_t)(I::W1 + I::W3));
      tc::bulk_g2s(s.w1, img, (uint32_t)I::W1, &s.bar_w);
      tc::bulk_g2s(s.w3, img + I::W1 + I::W2, (uint32_t)I::W3, &s.bar_w);
      if (!tc::mbar_wait(&s.bar_w, 0)) atomicExch(&s.err, 1);
      const uint32_t w1a = tc::smem_u32(s.w1), w3a = tc::smem_u32(s.w3);
      const uint32_t r0a = tc::smem_u32(s.ring[0]), r1a = tc::smem_u32(s.ring[1]);
      constexpr uint32_t kL1 = I::RB1 == 64 ? tc::kLayoutSW64 : tc::kLayoutSW128;
      constexpr uint32_t kIdN = tc::idesc_bf16(kTcRows, H);
      constexpr uint32_t kIdH = tc::idesc_bf16(kTcRows, kHeadN);
      int gs = 0;
      for (int p = 0; p < npairs; ++p) {
        const uint32_t par = p & 1;
        for (int sl = 0; sl < 2; ++sl) {
          if (!tc::mbar_wait(&s.xin[sl], par)) atomicExch(&s.err, 1);
          tc::fence_after();
          const uint32_t xa = tc::smem_u32(s.act[sl]);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk)
            tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(xa + kk * 32, 8 * I::RB1, kL1),
                         tc::desc_kmajor(w1a + kk * 32, 8 * I::RB1, kL1), kIdN, kk > 0);
          tc::mma_commit(&s.mma1[sl]);
        }
        for (int sl = 0; sl < 2; ++sl) {
          if (!tc::mbar_wait(&s.h1in[sl], par)) atomicExch(&s.err, 1);
          tc::fence_after();
          const uint32_t ha = tc::smem_u32(s.act[sl]);
          for (int kb = 0; kb < KB2; ++kb, ++gs) {
            const int slot = gs & 1;
            if (!tc::mbar_wait(&s.full[slot], (gs >> 1) & 1)) atomicExch(&s.err, 1);
            tc::fence_after();
            const uint32_t ra = slot ? r1a : r0a;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(ha + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                           tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, (kb | kk) != 0);
            tc::mma_commit(&s.empty[slot]);
          }
          tc::mma_commit(&s.mma2[sl]);
        }
        for (int sl = 0; sl < 2; ++sl) {
          if (!tc::mbar_wait(&s.h2in[sl], par)) atomicExch(&s.err, 1);
          tc::fence_after();
          const uint32_t ha = tc::smem_u32(s.act[sl]);
#pragma unroll 1
          for (int kb = 0; kb < H / 64; ++kb)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(ha + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                           tc::desc_kmajor(w3a + kb * kHeadN * 128 + kk * 32, 1024, tc::kLayoutSW128), kIdH,
                           (kb | kk) != 0);
          tc::mma_commit(&s.head[sl]);
        }
      }
    }
  } else {
    // epilogue warps
    const int quad = warp & 3, slice = warp >> 2, row = quad * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
    uint4 xv[2][XCH];
    auto fetch_x = [&](int k, uint4 (&dst)[XCH]) {
      const int64_t tl = blockIdx.x + (int64_t)k * gridDim.x;
#pragma unroll
      for (int q = 0; q < XCH; ++q) {
        const int i = tid + q * kTcThreads, r = i / CPR, c = i % CPR;
        const int64_t rr = tl * kTcRows + r;
        dst[q] = make_uint4(0, 0, 0, 0);
        if (k < my_tiles && rr < n) {
          const int64_t src = save.gather ? (int64_t)__ldg(save.gather + rr) : rr;
          dst[q] = __ldg(reinterpret_cast<const uint4*>(obs + src * D) + c);
        }
      }
    };
    // head readout of the tile in slot sl (warps 0-3: one row per thread)
    auto head_out = [&](int sl, int k) {
      if (warp < 4 && k < my_tiles) {
        const int64_t tl = blockIdx.x + (int64_t)k * gridDim.x;
        const int nr = (int)(n - tl * kTcRows < kTcRows ? n - tl * kTcRows : kTcRows);
        float v[16];
        tc::tmem_ld16(lane_base + (uint32_t)(sl * 256), v);
        if (save.loss.dz) {
          ppo_head_row(save.loss, value_net, A, s.b3, save.gather, tl, row, n, v, warp);
        } else if (row < nr) {
          float* o = out + (tl * kTcRows + row) * out_stride;
#pragma unroll
          for (int j = 0; j < kHeadN; ++j)
            if (j < nout) o[j] = v[j] + s.b3[j];
        }
      }
    };
    // hidden layer epilogue of slot sl: tanh(acc + bias) -> bf16 -> act[sl] (+ the tile image)
    auto hidden = [&](int sl, const float* bias, __nv_bfloat16* gsave, int k) {
      const int64_t tl = blockIdx.x + (int64_t)k * gridDim.x;
      uint8_t* g = (gsave && k < my_tiles) ? reinterpret_cast<uint8_t*>(gsave) + tl * (int64_t)(kTcRows * H * 2)
                                           : nullptr;
#pragma unroll
      for (int j = 0; j < H / 64; ++j) {
        const int c = slice * (H / 4) + j * 16;
        float v[16];
        tc::tmem_ld16(lane_base + (uint32_t)(sl * 256 + c), v);
        uint32_t pk[8];
        tc::tanh16_bf16(v, bias + c, pk);
        const uint32_t o0 = tc::swz_offset<128>(row, c, kTcRows), o1 = tc::swz_offset<128>(row, c + 8, kTcRows);
        const uint4 lo = make_uint4(pk[0], pk[1], pk[2], pk[3]), hi = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        *reinterpret_cast<uint4*>(s.act[sl] + o0) = lo;
        *reinterpret_cast<uint4*>(s.act[sl] + o1) = hi;
        if (g) {
          *reinterpret_cast<uint4*>(g + o0) = lo;
          *reinterpret_cast<uint4*>(g + o1) = hi;
        }
      }
    };
    auto handover = [&](uint64_t* bar) {
      tc::fence_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
    };
    fetch_x(0, xv[0]);
    fetch_x(1, xv[1]);
    for (int p = 0; p < npairs; ++p) {
      const uint32_t par = p & 1;
      for (int sl = 0; sl < 2; ++sl) {
        const int k = 2 * p + sl;
        if (p > 0) {
          // the previous tile of this slot: its head is done, read it out;
          // its h2 is no longer needed, so X may overwrite the buffer
          if (!tc::mbar_wait(&s.head[sl], par ^ 1)) atomicExch(&s.err, 1);
          tc::fence_after();
          head_out(sl, k - 2);
        }
        const int64_t tl = blockIdx.x + (int64_t)k * gridDim.x;
#pragma unroll
        for (int q = 0; q < XCH; ++q) {
          const int i = tid + q * kTcThreads, r = i / CPR, c = i % CPR;
          const uint32_t off = tc::swz_offset<I::RB1>(r, c * 8, kTcRows);
          *reinterpret_cast<uint4*>(s.act[sl] + off) = xv[sl][q];
          if (save.x && k < my_tiles)
            *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(save.x) + tl * (int64_t)(kTcRows * D * 2) + off) =
                xv[sl][q];
        }
        handover(&s.xin[sl]);
      }
      fetch_x(2 * p + 2, xv[0]);
      fetch_x(2 * p + 3, xv[1]);
      for (int sl = 0; sl < 2; ++sl) {
        if (!tc::mbar_wait(&s.mma1[sl], par)) atomicExch(&s.err, 1);
        tc::fence_after();
        hidden(sl, s.b1, save.h1, 2 * p + sl);
        handover(&s.h1in[sl]);
      }
      for (int sl = 0; sl < 2; ++sl) {
        if (!tc::mbar_wait(&s.mma2[sl], par)) atomicExch(&s.err, 1);
        tc::fence_after();
        hidden(sl, s.b2, save.h2, 2 * p + sl);
        handover(&s.h2in[sl]);
      }
    }
    if (npairs > 0)
      for (int sl = 0; sl < 2; ++sl) {
        if (!tc::mbar_wait(&s.head[sl], (npairs - 1) & 1)) atomicExch(&s.err, 1);
        tc::fence_after();
        head_out(sl, 2 * (npairs - 1) + sl);
      }
  }
  tc::fence_before();
  __syncthreads();
  if (s.err && warp == 16 && lane == 0 && last_issued >= 0)
    (void)tc::mbar_wait(&s.full[last_issued & 1], (last_issued >> 1) & 1);
  if (tid == 0 && s.err) {
    atomicExch(&g_tc_error, 1);
    if (err) atomicExch(err, 1);
  }
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// decoupled bf16 rollout: per step, an env kernel (one thread per env: act on
// the previous step's logits, then observe) and the tensor-core policy kernel
// ---------------------------------------------------------------------------
struct ActArgs {
  const float* logits;  // [E][16]
  int t;                // step whose action is taken (-1: observe only)
  uint32_t it;
  float lambda;
  int det;
  int T;                // horizon (t + 1 == T: write obs_last)
  int e0, ne;           // the envs [e0, e0 + ne) of this launch
};

template <int C, int OBS, int D, int A>
__global__ void __launch_bounds__(128) env_actobs_kernel(EnvDev env, ActArgs a, pe_rollout_buf buf) {
  const int e = a.e0 + (int)(blockIdx.x * blockDim.x + threadIdx.x);
  if (e >= a.e0 + a.ne) return;
  RegAcc<C> acc = load_reg<C>(env, e);
  if (a.t >= 0) {
    float z[A];
    const float4* lz = reinterpret_cast<const float4*>(a.logits + (int64_t)e * kHeadN);
#pragma unroll
    for (int j = 0; j < A / 4; ++j) {
      const float4 q = lz[j];
      z[4 * j] = q.x;
      z[4 * j + 1] = q.y;
      z[4 * j + 2] = q.z;
      z[4 * j + 3] = q.w;
    }
    const uint32_t r = a.det ? 0u : draw32(env.seed, (uint32_t)e, (uint32_t)a.t, a.it, kDrawAction);
    float lp;
    const int act = sample_action<A>(z, r, a.det != 0, &lp);
    const StepOut so = env_step<C>(env, acc, act, a.lambda);
    // the rollout buffer is not read again during the rollout: streaming
    // stores (evict first) keep L2 for the env state, the rings and the logits
    const int64_t row = (int64_t)a.t * env.E + e;
    __stcs(buf.act + row, (uint8_t)act);
    __stcs(buf.logp + row, lp);
    __stcs(buf.reward + row, so.reward);
    __stcs(buf.done + row, (uint8_t)so.done);
    if (buf.q) __stcs(buf.q + row, so.q);
    if (a.t == 0) {
      buf.viol[2 * e] = so.v1;
      buf.viol[2 * e + 1] = so.v60;
      buf.tokens[e] = so.tokens;
      buf.excess[e] = so.excess;
      buf.energy_q[e] = so.q;
      if (buf.samples) buf.samples[e] = so.samples;
    } else {
      buf.viol[2 * e] += so.v1;
      buf.viol[2 * e + 1] += so.v60;
      buf.tokens[e] += so.tokens;
      buf.excess[e] += so.excess;
      buf.energy_q[e] += so.q;
      if (buf.samples) buf.samples[e] += so.samples;
    }
    if (so.done) env_reset<C>(env, acc, (uint32_t)e, (uint32_t)a.t, a.it, kDrawReset);
  }
  // observation for step t + 1 (or the final one)
  __nv_bfloat16* dst = (a.t + 1 < a.T)
                           ? reinterpret_cast<__nv_bfloat16*>(buf.obs) + ((int64_t)(a.t + 1) * env.E + e) * D
                           : reinterpret_cast<__nv_bfloat16*>(buf.obs_last) + (int64_t)e * D;
  const Fam fm = fam_of(env, acc.fam());
  float o[D];
  features_eq5<C, OBS, D>(env, acc, fm, o);
#pragma unroll
  for (int f0 = 0; f0 < D; f0 += 8) {
    uint32_t p[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) p[i] = tc::pack_bf16(o[f0 + 2 * i], o[f0 + 2 * i + 1]);
    __stcs(reinterpret_cast<uint4*>(dst + f0), make_uint4(p[0], p[1], p[2], p[3]));
  }
  store_reg<C>(env, e, acc);
}

// workspace: weight image (policy), weight image (value), logits [E][16], error word
template <int D, int H, bool STREAM = (H > 256)>
struct NetKind;
template <int D, int H>
struct NetKind<D, H, false> {
  static constexpr bool kStream = false;
  static constexpr int64_t kImgPad = (Img<D, H>::TOTAL + 1023) / 1024 * 1024;
};
template <int D, int H>
struct NetKind<D, H, true> {
  static constexpr bool kStream = true;
  static constexpr int64_t kImgPad = (ImgS<D, H>::TOTAL + 1023) / 1024 * 1024;
};

template <int D, int H>
static int64_t bf16_ws_bytes(int64_t E) {
  return 2 * NetKind<D, H>::kImgPad + (E * kHeadN * 4 + 255) / 256 * 256 + 256;
}

template <int D, int H>
static pe_status launch_mlp(const uint8_t* img, const float* params, int A, int value_net,
                            const void* obs, int64_t n, float* out, int out_stride, int nout,
                            int32_t* err, cudaStream_t st, int prof_kind, MlpSave save = MlpSave{},
                            MlpSecond second = MlpSecond{}) {
  if (n <= 0) return PE_OK;
  int dev = 0, sms = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int64_t tiles = (n + kTcRows - 1) / kTcRows;
  const __nv_bfloat16* o = reinterpret_cast<const __nv_bfloat16*>(obs);
  if constexpr (NetKind<D, H>::kStream) {
    // a two-network launch is the PPO forward: policy first, the loss head on both
    if (second.img && (value_net != 0 || !save.loss.dz || !second.save.loss.dz))
      return fail(PE_EINVAL, "a two-network forward runs the policy, then the value network, with the loss head");
    const int64_t all = second.img ? 2 * tiles : tiles;
    const int grid = (int)(all < sms ? all : sms);
    auto kern = mlp_bf16_stream_kernel<D, H>;
    const int bytes = (int)sizeof(MlpStreamSmem<D, H>) + 1024;
    PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    ProfScope ps(prof_kind, st);
    kern<<<grid, kStreamThreads, bytes, st>>>(img, params, A, value_net, o, n, out, out_stride, nout, err, save,
                                              second);
  } else {
    if (second.img) return fail(PE_EINVAL, "two-network forward launches are for the streamed network");
    auto kern = mlp_bf16_pair_kernel<D, H>;
    const int bytes = (int)sizeof(MlpPairSmem<D, H>) + 1024;
    PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    const int pgrid = (int)std::min<int64_t>((tiles + 1) / 2, sms);
    ProfScope ps(prof_kind, st);
    kern<<<pgrid, kPairThreads, bytes, st>>>(img, params, A, value_net, o, n, out, out_stride, nout, err, save);
  }
  PE_CHECK_LAUNCH("bf16 MLP kernel");
  return PE_OK;
}

template <int D, int H>
static pe_status make_images(const float* params, int A, uint8_t* ws, cudaStream_t st, bool policy) {
  const int64_t img = NetKind<D, H>::kImgPad;
  ProfScope ps(PE_PROF_VALUE, st);
  if constexpr (NetKind<D, H>::kStream) {
    weight_image_stream_kernel<D, H><<<dim3(128, policy ? 2 : 1), 256, 0, st>>>(params, A, policy ? 0 : 1,
                                                                                policy ? ws : ws + img, img);
  } else {
    weight_image_kernel<D, H><<<dim3(64, policy ? 2 : 1), 256, 0, st>>>(params, A, policy ? 0 : 1,
                                                                        policy ? ws : ws + img, img);
  }
  PE_CHECK_LAUNCH("weight_image_kernel");
  return PE_OK;
}

// The envs of a 72B rollout run as two independent chains (the first and
// the second half of the envs, split on a 128-env tile boundary), the first
// on the caller's stream and the second on an auxiliary stream forked from
// it and joined back before the value pass.  Each chain alternates its own
// policy and env-step launches, so an env step (latency-bound, few
// registers, no shared memory) can run beside the other chain's tensor-core
// policy kernel, whose half-size grid leaves SMs free.  Every env's
// arithmetic is the single-chain arithmetic, so the results are the same
// bits.  Measured on GB300 (65,536 envs x 64 steps): 4.89 ms against 5.16 ms
// for one chain.  Forcing the two chains' policy kernels to alternate (an
// event per chain) was slower (5.24 ms), and the streamed Stress network,
// whose policy grid fills every SM, stays on one chain (two: 12.19 against
// 11.94 ms for 262,144 envs x 16 steps).
struct AuxChain {
  cudaStream_t main = nullptr, aux = nullptr;
  cudaEvent_t ev = nullptr;
  pe_status open(cudaStream_t st) {
    main = st;
    PE_TRY_CUDA(cudaEventCreateWithFlags(&ev, cudaEventDisableTiming));
    PE_TRY_CUDA(cudaStreamCreateWithFlags(&aux, cudaStreamNonBlocking));
    PE_TRY_CUDA(cudaEventRecord(ev, main));
    PE_TRY_CUDA(cudaStreamWaitEvent(aux, ev, 0));
    return PE_OK;
  }
  ~AuxChain() {  // join (also on an early error return), then release
    if (aux) {
      if (cudaEventRecord(ev, aux) == cudaSuccess) cudaStreamWaitEvent(main, ev, 0);
      cudaStreamDestroy(aux);
    }
    if (ev) cudaEventDestroy(ev);
  }
};

template <int C, int OBS, int D, int H, int A>
static pe_status rollout_bf16_impl(const EnvDev& env, const float* params, int T, uint32_t it,
                                   float lambda, int det, const pe_rollout_buf& buf, void* wsv,
                                   cudaStream_t st) {
  uint8_t* ws = reinterpret_cast<uint8_t*>(wsv);
  const int64_t img = NetKind<D, H>::kImgPad;
  float* logits = reinterpret_cast<float*>(ws + 2 * img);
  int32_t* err = reinterpret_cast<int32_t*>(ws + 2 * img + (env.E * (int64_t)kHeadN * 4 + 255) / 256 * 256);
  PE_TRY_CUDA(cudaMemsetAsync(err, 0, 4, st));
  pe_status s = make_images<D, H>(params, A, ws, st, true);
  if (s != PE_OK) return s;
  ActArgs a{logits, -1, it, lambda, det, T, 0, env.E};
  {
    ProfScope ps(PE_PROF_ROLLOUT, st);
    env_actobs_kernel<C, OBS, D, A><<<ceil_div(env.E, 128), 128, 0, st>>>(env, a, buf);
  }
  PE_CHECK_LAUNCH("env_actobs_kernel");
  {
    // chains: [0, split) on st, [split, E) on the auxiliary stream (one
    // chain for the streamed network and below two tiles per half)
    const int split = (!NetKind<D, H>::kStream && env.E >= 4 * kTcRows)
                          ? (env.E / 2 + kTcRows - 1) / kTcRows * kTcRows
                          : env.E;
    const int nch = split < env.E ? 2 : 1;
    AuxChain ax;
    if (nch == 2) {
      s = ax.open(st);
      if (s != PE_OK) return s;
    }
    for (int t = 0; t < T; ++t) {
      for (int ch = 0; ch < nch; ++ch) {
        const int e0 = ch ? split : 0, ne = ch ? env.E - split : split;
        const cudaStream_t sc = ch ? ax.aux : st;
        const void* obs_t = reinterpret_cast<const __nv_bfloat16*>(buf.obs) + ((int64_t)t * env.E + e0) * D;
        s = launch_mlp<D, H>(ws, params, A, 0, obs_t, ne, logits + (int64_t)e0 * kHeadN, kHeadN, A, err, sc,
                             PE_PROF_MLP_POLICY);
        if (s != PE_OK) return s;
        a.t = t;
        a.e0 = e0;
        a.ne = ne;
        {
          ProfScope ps(PE_PROF_ROLLOUT, sc);
          env_actobs_kernel<C, OBS, D, A><<<ceil_div(ne, 128), 128, 0, sc>>>(env, a, buf);
        }
        PE_CHECK_LAUNCH("env_actobs_kernel");
      }
    }
  }
  s = launch_mlp<D, H>(ws + img, params, A, 1, buf.obs, (int64_t)T * env.E, buf.value, 1, 1, err, st, PE_PROF_MLP_VALUE);
  if (s != PE_OK) return s;
  return launch_mlp<D, H>(ws + img, params, A, 1, buf.obs_last, env.E, buf.last_value, 1, 1, err, st, PE_PROF_MLP_VALUE);
}

int64_t rollout_bf16_ws_bytes(const pe_net& net, int64_t E) {
  if (net.obs_dim == 32 && net.hidden == 256) return bf16_ws_bytes<32, 256>(E);
  if (net.obs_dim == 64 && net.hidden == 512) return bf16_ws_bytes<64, 512>(E);
  return -1;
}

pe_status rollout_bf16(const EnvDev& env, const pe_net& net, const float* params, int T, uint32_t it,
                       float lambda, int det, const pe_rollout_buf& buf, void* ws, cudaStream_t st) {
  if (net.obs_dim == 32 && net.hidden == 256 && net.n_actions == 16 && env.C == 4 && env.obs_kind == PE_OBS_OCC32)
    return rollout_bf16_impl<4, PE_OBS_OCC32, 32, 256, 16>(env, params, T, it, lambda, det, buf, ws, st);
  if (net.obs_dim == 64 && net.hidden == 512 && net.n_actions == 16 && env.C == 4 && env.obs_kind == PE_OBS_OCC64)
    return rollout_bf16_impl<4, PE_OBS_OCC64, 64, 512, 16>(env, params, T, it, lambda, det, buf, ws, st);
  return fail(PE_EINVAL, "unsupported bf16 network/env combination (D=%d H=%d A=%d C=%d obs=%d)",
              net.obs_dim, net.hidden, net.n_actions, env.C, env.obs_kind);
}

pe_status device_check(cudaStream_t st) {
  PE_TRY_CUDA(cudaStreamSynchronize(st));
  int32_t flag = 0;
  PE_TRY_CUDA(cudaMemcpyFromSymbol(&flag, g_tc_error, sizeof(flag)));
  if (flag) {
    const int32_t zero = 0;
    PE_TRY_CUDA(cudaMemcpyToSymbol(g_tc_error, &zero, sizeof(zero)));
    return fail(PE_ETIMEOUT, "a bounded tensor-core wait timed out in an earlier launch");
  }
  return PE_OK;
}

template <int D, int H>
static pe_status value_bf16_impl(const pe_net& net, const float* params, const void* obs, int64_t n,
                                 float* value, uint8_t* ws, cudaStream_t st) {
  const int64_t img = NetKind<D, H>::kImgPad;
  int32_t* err = reinterpret_cast<int32_t*>(ws + 2 * img);
  PE_TRY_CUDA(cudaMemsetAsync(err, 0, 4, st));
  pe_status s = make_images<D, H>(params, net.n_actions, ws, st, false);
  if (s != PE_OK) return s;
  return launch_mlp<D, H>(ws + img, params, net.n_actions, 1, obs, n, value, 1, 1, err, st, PE_PROF_MLP_VALUE);
}

pe_status value_bf16(const pe_net& net, const float* params, const void* obs, int64_t n, float* value,
                     void* wsv, cudaStream_t st) {
  uint8_t* ws = reinterpret_cast<uint8_t*>(wsv);
  if (net.obs_dim == 32 && net.hidden == 256) return value_bf16_impl<32, 256>(net, params, obs, n, value, ws, st);
  if (net.obs_dim == 64 && net.hidden == 512) return value_bf16_impl<64, 512>(net, params, obs, n, value, ws, st);
  return fail(PE_EINVAL, "unsupported bf16 value network (D=%d H=%d)", net.obs_dim, net.hidden);
}

// forward of one bf16 network over gathered minibatch rows, saving x, h1 and
// h2 (used by the bf16 PPO update); img must hold the network's weight image
int64_t bf16_image_bytes(const pe_net& net) {
  if (net.obs_dim == 32 && net.hidden == 256) return NetKind<32, 256>::kImgPad;
  if (net.obs_dim == 64 && net.hidden == 512) return NetKind<64, 512>::kImgPad;
  return -1;
}

pe_status bf16_make_images(const pe_net& net, const float* params, uint8_t* two_images, cudaStream_t st) {
  if (net.obs_dim == 32 && net.hidden == 256) return make_images<32, 256>(params, net.n_actions, two_images, st, true);
  if (net.obs_dim == 64 && net.hidden == 512) return make_images<64, 512>(params, net.n_actions, two_images, st, true);
  return fail(PE_EINVAL, "unsupported bf16 network");
}

// forward of both networks over the same gathered minibatch rows with the PPO
// loss in the head: the policy (image at img, loss lp, saving x, h[0], h[1])
// and the value network (image at img + bf16_image_bytes, loss lv, saving
// h[2], h[3]).  The streamed network runs both in one launch, its tiles
// spread over the persistent CTAs together.
pe_status bf16_forward_loss(const pe_net& net, const uint8_t* img, const float* params, const void* obs,
                            const uint32_t* gather, int64_t n, const PpoHead& lp, const PpoHead& lv,
                            __nv_bfloat16* x, __nv_bfloat16* const h[4], int32_t* err, cudaStream_t st) {
  const MlpSave sp{gather, x, h[0], h[1], lp};
  const MlpSave sv{gather, nullptr, h[2], h[3], lv};
  float* out = nullptr;
  if (net.obs_dim == 32 && net.hidden == 256) {
    const uint8_t* img_v = img + NetKind<32, 256>::kImgPad;
    pe_status s = launch_mlp<32, 256>(img, params, net.n_actions, 0, obs, n, out, 0, net.n_actions, err, st,
                                      PE_PROF_PPO_GRAD, sp);
    if (s != PE_OK) return s;
    return launch_mlp<32, 256>(img_v, params, net.n_actions, 1, obs, n, out, 0, 1, err, st, PE_PROF_PPO_GRAD, sv);
  }
  if (net.obs_dim == 64 && net.hidden == 512)
    return launch_mlp<64, 512>(img, params, net.n_actions, 0, obs, n, out, 0, net.n_actions, err, st,
                               PE_PROF_PPO_GRAD, sp, MlpSecond{img + NetKind<64, 512>::kImgPad, sv});
  return fail(PE_EINVAL, "unsupported bf16 network");
}

int64_t value_bf16_ws_bytes(const pe_net& net) {
  if (net.obs_dim == 32 && net.hidden == 256) return bf16_ws_bytes<32, 256>(0);
  if (net.obs_dim == 64 && net.hidden == 512) return bf16_ws_bytes<64, 512>(0);
  return -1;
}

}  // namespace pe
