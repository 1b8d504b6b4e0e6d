// Backward pass of the bf16 policy/value networks (72B: 32-256-256x16,
// Stress: 64-512-512x16) on the tcgen05 tensor cores, for the PPO update
// (Sec. 4.2).  With z = W3 h2 + b3, h2 = tanh(W2 h1 + b2), h1 = tanh(W1 x + b1)
// and dz = dLoss/dz per sample (from the loss kernel), the update needs
//   da2 = bf16(dz W3 (1 - h2^2)),  da1 = bf16(da2 W2 (1 - h1^2))   (per sample)
//   dW2 = da2^T h1, db2 = sum da2, dW1 = da1^T x, db1 = sum da1,
//   dW3 = dz^T h2                                                (over samples)
// with fp32 accumulation everywhere and bf16 at the rounding points the
// oracle emulates (dz, da2 and da1 enter the products as bf16).
//
// Every per-sample operand lives in global memory as a 128-row "tile image",
// byte for byte the swizzled shared-memory layout the kernels use (see
// tc.cuh), so that each operand tile arrives with one bulk copy:
//   x, h1, h2, da2, da1: K-major over features, 128-byte rows, H/64 blocks
//   (x: D = 32 in 64-byte rows); dz: 16 bf16 in 32-byte rows.
// Read with samples as the reduction dimension, the same bytes are the
// MN-major operands of the weight-gradient products.
//
// bwd_data_kernel (Stress, H = 512; one 128-sample tile at a time,
// persistent; the 72B networks compute these products inside the fused
// forward-backward kernel of fused_bf16.cu):
//   dh2 = dz W3 (one MMA per 256 columns, K = 16) -> TMEM; epilogue:
//   da2 = bf16(dh2 (1 - h2^2)) into shared memory (the next A operand) and
//   its tile image; dh1 = da2 W2 with W2^T streamed through a two-slot ring
//   of 32 KB stages by a producer warp; epilogue: da1 = bf16(dh1 (1 - h1^2))
//   to its tile image.  Every step works in 256-column halves so that the
//   MMAs, the epilogues and the copies overlap: a loader warp brings each
//   half of the tile's h2 image into the da2 buffer with one bulk copy (da2
//   then overwrites it in place), the dh1 MMAs over da2's first half start
//   while the epilogue writes its second half, each half of the h1 image
//   lands once the dh1 MMAs have read that half of da2, and each half of the
//   next tile's h2 (and of its dh2 accumulators) follows as soon as the da1
//   epilogue has read that half of h1 (and of TMEM).  A dedicated warp
//   issues the MMAs.  One launch covers both networks: the policy's tiles,
//   then the value's, spread over the CTAs as one list (a CTA that crosses
//   from one to the other reloads W3^T), which balances a tile count that
//   is not a multiple of the SM count.
// wgrad_kernel (split over samples): each CTA owns 128 output rows (one
//   block of layer outputs o) of one network and one 256-column chunk, and
//   accumulates over its share of the minibatch, 64 samples per stage:
//   [dW2 | db2] = da2^T [h1 | 1], and for column chunk 0 also
//   [dW1 | db1] = da1^T [x | 1] and dW3^T = h2^T dz; it writes its fp32
//   accumulators as one partial block.  Column chunk 0's stages bring more
//   bytes, so its groups get proportionally more (shorter) sample shares.
//   wgrad_reduce_kernel sums the partial
//   blocks of every output in a fixed order (deterministic) into the
//   canonical gradient vector.
#include <algorithm>

#include "bf16_layout.cuh"
#include "mlp_f32.cuh"
#include "tc.cuh"

namespace pe {

constexpr int kBwCompute = 512;         // 16 compute warps
constexpr int kBwThreads = kBwCompute + 96;  // + the W2^T producer, the h loader and the MMA issuer warps

int64_t bwd_image_bytes(int H) {
  if (H == 256) return BwdImg<256>::TOTAL;
  if (H == 512) return BwdImg<512>::TOTAL;
  return -1;
}

template <int D, int H>
__global__ void bwd_image_kernel(const float* __restrict__ params, int A, uint8_t* __restrict__ img0,
                                 uint8_t* __restrict__ img1) {
  using I = BwdImg<H>;
  const int value_net = (int)blockIdx.y;  // y = 0 policy, 1 value
  uint8_t* img = value_net ? img1 : img0;
  const MlpLayout Lp = mlp_layout(D, H, A);
  const float* w2 = params + (value_net ? Lp.v2 : Lp.w2);
  const float* w3 = params + (value_net ? Lp.v3 : Lp.w3);
  const int nout = value_net ? 1 : A;
  const int total = H * 16 + H * H;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    if (i < H * 16) {
      const int o = i / 16, a = i % 16;  // W3^T[o][a] = W3[a][o]
      const float v = a < nout ? w3[(int64_t)a * H + o] : 0.0f;
      *reinterpret_cast<__nv_bfloat16*>(img + bwd_img_offset<H>(3, a, o)) = __float2bfloat16_rn(v);
    } else {
      const int j = i - H * 16, o = j / H, c = j % H;  // W2[o][c] = W2^T[c][o]
      *reinterpret_cast<__nv_bfloat16*>(img + bwd_img_offset<H>(2, o, c)) = __float2bfloat16_rn(w2[j]);
    }
  }
}

template <int H>
struct BwdSmem {
  // A operand of dh1 = da2 W2 (K-major SW128), in 256-column halves (K-blocks
  // 0-3 and 4-7).  Each half of a tile's h2 image arrives here first and da2
  // overwrites it in place (da2 is elementwise in h2); once the dh1 MMAs have
  // read a half of da2, that half of the h1 image arrives for the second
  // epilogue; once that epilogue has read it, the next tile's h2 half.
  alignas(1024) uint8_t da2[kBwRows * H * 2];
  alignas(1024) uint8_t ring[2][kBwStage];
  alignas(1024) uint8_t w3t[H * 32];           // B operand of dh2 = dz W3 (K-major SW32)
  alignas(1024) uint8_t dz[kBwRows * 32];      // A operand of dh2 (K-major SW32)
  uint64_t full[2], empty[2], bar_w, fin;
  // one completion per tile each: h2 / h1 half landed (bulk copies), dz
  // written, dh2 N-half done, da2 half written, dh1 N-half 0 done, dh1
  // N-half 1 past K-block 3, dh1 done, da1 half read out of TMEM and h1
  uint64_t h2a, h2b, h1a, h1b, dzin, mdh2a, mdh2b, d2a, d2b, m1a, n1lo, m1b, da, db;
  uint32_t tmem_base;
  int32_t err;
};

// per network (policy, value): one launch covers both, their tiles spread
// over the persistent CTAs together
struct BwdArgs {
  const uint8_t* img[2];  // backward weight image of each network
  const uint8_t* dz[2];   // dz tile images (4 KB per tile)
  const uint8_t* h1[2];   // h1 tile images
  const uint8_t* h2[2];   // h2 tile images
  uint8_t* da2[2];        // out: da2 tile images
  uint8_t* da1[2];        // out: da1 tile images
  int64_t n;              // valid samples (both networks)
  int32_t* err;
};

template <int H>
__global__ void __launch_bounds__(kBwThreads, 1) bwd_data_kernel(BwdArgs g) {
  using I = BwdImg<H>;
  static_assert(H == 512, "two 256-column halves per product");
  constexpr int kTileBytes = kBwRows * H * 2;
  constexpr int kHalfBytes = kTileBytes / 2;  // K-blocks 0-3 or 4-7 of a tile image
  constexpr int KBH = I::KB / 2;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  BwdSmem<H>& s = *reinterpret_cast<BwdSmem<H>*>(base);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s.err = 0;
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.full[i], 1);
      tc::mbar_init(&s.empty[i], 1);
    }
    tc::mbar_init(&s.bar_w, 1);
    tc::mbar_init(&s.fin, 1);
    tc::mbar_init(&s.h2a, 1);
    tc::mbar_init(&s.h2b, 1);
    tc::mbar_init(&s.h1a, 1);
    tc::mbar_init(&s.h1b, 1);
    tc::mbar_init(&s.dzin, kBwCompute / 32);
    tc::mbar_init(&s.mdh2a, 1);
    tc::mbar_init(&s.mdh2b, 1);
    tc::mbar_init(&s.d2a, kBwCompute / 32);
    tc::mbar_init(&s.d2b, kBwCompute / 32);
    tc::mbar_init(&s.m1a, 1);
    tc::mbar_init(&s.n1lo, 1);
    tc::mbar_init(&s.m1b, 1);
    tc::mbar_init(&s.da, kBwCompute / 32);
    tc::mbar_init(&s.db, kBwCompute / 32);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&s.tmem_base, H);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = s.tmem_base;
  const int64_t tiles = (g.n + kBwRows - 1) / kBwRows;  // per network
  const int my_tiles = (int)((2 * tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);
  // this CTA's k-th tile: its network (ni; the policy's tiles come first, so
  // a CTA switches network at most once) and its tile index within it
  auto tile_of = [&](int k, int& ni) -> int64_t {
    const int64_t q = (int64_t)blockIdx.x + (int64_t)k * gridDim.x;
    ni = q >= tiles ? 1 : 0;
    return q - ni * tiles;
  };
  // a bounded wait that is skipped once the CTA has an error
  auto wt = [&](uint64_t* b, uint32_t par) -> bool {
    if (*reinterpret_cast<volatile int32_t*>(&s.err)) return false;
    if (tc::mbar_wait(b, par)) return true;
    atomicExch(&s.err, 1);
    return false;
  };
  int ni0 = 0;
  if (my_tiles > 0) (void)tile_of(0, ni0);
  int last_issued = -1;  // producer: global index of its last issued stage
  int nh[4] = {0, 0, 0, 0};  // loader: copies issued into h2a, h2b, h1a, h1b
  int cur = ni0;         // MMA issuer: network of the W3^T in shared memory
  if (warp == kBwCompute / 32) {
    // producer: the W2^T stages of every tile, in consumption order
    if (lane == 0) {
      int gs = 0;
      bool ok = true;
      for (int t = 0; t < my_tiles && ok; ++t) {
        int ni;
        (void)tile_of(t, ni);
        const uint8_t* img = ni ? g.img[1] : g.img[0];
        for (int st = 0; st < I::STAGES; ++st) {
          const int slot = gs & 1;
          if (gs >= 2 && !wt(&s.empty[slot], ((gs - 2) >> 1) & 1)) {
            ok = false;
            break;
          }
          tc::mbar_expect_tx(&s.full[slot], (uint32_t)kBwStage);
          tc::bulk_g2s(s.ring[slot], img + I::W3T + (int64_t)st * kBwStage, (uint32_t)kBwStage, &s.full[slot]);
          last_issued = gs++;
        }
      }
    }
  } else if (warp == kBwCompute / 32 + 1) {
    // loader: per tile, h1's first half once the dh1 MMAs over da2's first
    // half are done, its second half once all are; then the next tile's h2
    // halves as the second epilogue frees the halves of the buffer
    if (lane == 0) {
      auto copy = [&](int which, uint64_t* bar, const uint8_t* src, int half) {
        tc::mbar_expect_tx(bar, (uint32_t)kHalfBytes);
        tc::bulk_g2s(s.da2 + half * kHalfBytes, src + half * kHalfBytes, (uint32_t)kHalfBytes, bar);
        ++nh[which];
      };
      if (my_tiles > 0) {
        const uint8_t* h2 = (ni0 ? g.h2[1] : g.h2[0]) + tile_of(0, ni0) * (int64_t)kTileBytes;
        copy(0, &s.h2a, h2, 0);
        copy(1, &s.h2b, h2, 1);
      }
      for (int t = 0; t < my_tiles; ++t) {
        const uint32_t par = t & 1;
        int ni;
        const int64_t tl = tile_of(t, ni);
        const uint8_t* h1 = (ni ? g.h1[1] : g.h1[0]) + tl * (int64_t)kTileBytes;
        if (!wt(&s.n1lo, par)) break;
        copy(2, &s.h1a, h1, 0);
        if (!wt(&s.m1b, par)) break;
        copy(3, &s.h1b, h1, 1);
        if (t + 1 < my_tiles) {
          int nn;
          const int64_t nt = tile_of(t + 1, nn);
          const uint8_t* h2 = (nn ? g.h2[1] : g.h2[0]) + nt * (int64_t)kTileBytes;
          if (!wt(&s.da, par)) break;
          copy(0, &s.h2a, h2, 0);
          if (!wt(&s.db, par)) break;
          copy(1, &s.h2b, h2, 1);
        }
      }
    }
  } else if (warp == kBwCompute / 32 + 2) {
    // MMA issuer
    if (lane == 0) {
      tc::mbar_expect_tx(&s.bar_w, (uint32_t)I::W3T);
      tc::bulk_g2s(s.w3t, ni0 ? g.img[1] : g.img[0], (uint32_t)I::W3T, &s.bar_w);
      (void)wt(&s.bar_w, 0);
      const uint32_t da2a = tc::smem_u32(s.da2), dza = tc::smem_u32(s.dz), w3a = tc::smem_u32(s.w3t);
      constexpr uint32_t kIdN = tc::idesc_bf16(kBwRows, 256);
      int gs = 0;
      // dh1 = da2 W2: K-blocks [k0, k1) of da2 into N-half h (TMEM columns 256 h ..)
      auto dh1 = [&](int h, int k0, int k1) {
#pragma unroll 1
        for (int kb = k0; kb < k1; ++kb) {
          const int slot = gs & 1;
          (void)wt(&s.full[slot], (gs >> 1) & 1);
          tc::fence_after();
          const uint32_t ra = tc::smem_u32(s.ring[slot]);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc::mma_bf16(tmem + h * 256, tc::desc_kmajor(da2a + kb * kBwRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                         tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, (kb | kk) != 0);
          tc::mma_commit(&s.empty[slot]);
          ++gs;
        }
      };
      for (int t = 0; t < my_tiles; ++t) {
        const uint32_t par = t & 1;
        int ni;
        (void)tile_of(t, ni);
        (void)wt(&s.dzin, par);
        tc::fence_after();
        if (ni != cur) {
          // the value network's W3^T replaces the policy's (every MMA that
          // read it completed before the previous tile's da2 epilogue)
          cur = ni;
          tc::mbar_expect_tx(&s.bar_w, (uint32_t)I::W3T);
          tc::bulk_g2s(s.w3t, g.img[1], (uint32_t)I::W3T, &s.bar_w);
          (void)wt(&s.bar_w, 1);
          tc::fence_after();
        }
        // dh2 = dz W3, one K = 16 MMA per N-half, each once the previous
        // tile's da1 epilogue has read that half of TMEM
#pragma unroll 1
        for (int h = 0; h < I::NH; ++h) {
          if (t > 0) {
            (void)wt(h ? &s.db : &s.da, par ^ 1);
            tc::fence_after();
          }
          tc::mma_bf16(tmem + h * 256, tc::desc_strided(dza, 16, 256, tc::kLayoutSW32),
                       tc::desc_strided(w3a + h * 256 * 32, 16, 256, tc::kLayoutSW32), kIdN, 0);
          tc::mma_commit(h ? &s.mdh2b : &s.mdh2a);
        }
        (void)wt(&s.d2a, par);
        tc::fence_after();
        dh1(0, 0, KBH);
        (void)wt(&s.d2b, par);
        tc::fence_after();
        dh1(0, KBH, 2 * KBH);
        tc::mma_commit(&s.m1a);
        dh1(1, 0, KBH);
        tc::mma_commit(&s.n1lo);
        dh1(1, KBH, 2 * KBH);
        tc::mma_commit(&s.m1b);
      }
      // every MMA of this CTA completes before TMEM is released
      tc::mma_commit(&s.fin);
      if (!tc::mbar_wait(&s.fin, 0)) atomicExch(&s.err, 1);
    }
  } else {
    const int quad = warp & 3, slice = warp >> 2, row = quad * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    constexpr int NJ = H / 2 / 4 / 16;  // 16-column chunks per thread and half
    // d = bf16(TMEM (1 - h^2)) over this thread's chunks of half hf, h read
    // from the shared buffer at the offsets d is written to (in place when
    // in_place), d also to the tile image outt
    auto epi = [&](int hf, bool valid, uint8_t* outt, bool in_place) {
#pragma unroll 2
      for (int j = 0; j < NJ; ++j) {
        const int c = hf * (H / 2) + slice * (H / 8) + j * 16;
        float v[16];
        tc::tmem_ld16(lane_addr + (uint32_t)c, v);
        const uint32_t o0 = tc::swz_offset<128>(row, c, kBwRows), o1 = tc::swz_offset<128>(row, c + 8, kBwRows);
        const uint4 hb[2] = {*reinterpret_cast<const uint4*>(s.da2 + o0), *reinterpret_cast<const uint4*>(s.da2 + o1)};
        uint32_t pk[8];
        tanh_grad16(v, hb, valid, pk);
        const uint4 lo = make_uint4(pk[0], pk[1], pk[2], pk[3]), hi = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        if (in_place) {
          *reinterpret_cast<uint4*>(s.da2 + o0) = lo;
          *reinterpret_cast<uint4*>(s.da2 + o1) = hi;
        }
        *reinterpret_cast<uint4*>(outt + o0) = lo;
        *reinterpret_cast<uint4*>(outt + o1) = hi;
      }
    };
    auto handover = [&](uint64_t* bar) {
      tc::fence_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
    };
    uint4 dzv = make_uint4(0, 0, 0, 0);
    if (tid < kBwRows * 2 && my_tiles > 0)
      dzv = __ldg(reinterpret_cast<const uint4*>((ni0 ? g.dz[1] : g.dz[0]) + tile_of(0, ni0) * (kBwRows * 32)) + tid);
    for (int t = 0; t < my_tiles; ++t) {
      const uint32_t par = t & 1;
      int ni, nn = 0;
      const int64_t tile = tile_of(t, ni);
      const int64_t ntile = t + 1 < my_tiles ? tile_of(t + 1, nn) : 0;
      const int nr = (int)(g.n - tile * kBwRows < kBwRows ? g.n - tile * kBwRows : kBwRows);
      const bool valid = row < nr;
      if (t + 1 < my_tiles) {
        // the next tile's h1/h2 images asked of L2 a tile ahead (128-byte lines)
        const uint8_t* h2n = (nn ? g.h2[1] : g.h2[0]) + ntile * (int64_t)kTileBytes;
        const uint8_t* h1n = (nn ? g.h1[1] : g.h1[0]) + ntile * (int64_t)kTileBytes;
        for (int64_t off = (int64_t)tid * 128; off < (int64_t)kTileBytes; off += (int64_t)kBwCompute * 128) {
          tc::prefetch_l2(h2n + off);
          tc::prefetch_l2(h1n + off);
        }
      }
      // dz tile (4 KB, already in the SW32 layout; the previous tile's dh2
      // MMAs have read the old one), then the next tile's into registers
      if (tid < kBwRows * 2) {
        reinterpret_cast<uint4*>(s.dz)[tid] = dzv;
        if (t + 1 < my_tiles)
          dzv = __ldg(reinterpret_cast<const uint4*>((nn ? g.dz[1] : g.dz[0]) + ntile * (kBwRows * 32)) + tid);
      }
      handover(&s.dzin);
      uint8_t* const da2o = (ni ? g.da2[1] : g.da2[0]) + tile * (int64_t)kTileBytes;
      uint8_t* const da1o = (ni ? g.da1[1] : g.da1[0]) + tile * (int64_t)kTileBytes;
      // da2 = bf16(dh2 (1 - h2^2)) per half: in place over h2 (the next A
      // operand) and its tile image
      (void)wt(&s.mdh2a, par);
      (void)wt(&s.h2a, par);
      tc::fence_after();
      epi(0, valid, da2o, true);
      handover(&s.d2a);
      (void)wt(&s.mdh2b, par);
      (void)wt(&s.h2b, par);
      tc::fence_after();
      epi(1, valid, da2o, true);
      handover(&s.d2b);
      // da1 = bf16(dh1 (1 - h1^2)) per half, to its tile image
      (void)wt(&s.m1a, par);
      (void)wt(&s.h1a, par);
      tc::fence_after();
      epi(0, valid, da1o, false);
      handover(&s.da);
      (void)wt(&s.m1b, par);
      (void)wt(&s.h1b, par);
      tc::fence_after();
      epi(1, valid, da1o, false);
      handover(&s.db);
    }
  }
  tc::fence_before();
  __syncthreads();
  // on an error, the producer, the loader and the issuer wait (bounded) for
  // the copies they may still have in flight before the CTA leaves
  if (s.err && warp == kBwCompute / 32 && lane == 0)
    for (int q = last_issued - 1; q <= last_issued; ++q)
      if (q >= 0) (void)tc::mbar_wait(&s.full[q & 1], (q >> 1) & 1);
  if (s.err && warp == kBwCompute / 32 + 1 && lane == 0) {
    uint64_t* bars[4] = {&s.h2a, &s.h2b, &s.h1a, &s.h1b};
    for (int k = 0; k < 4; ++k)
      if (nh[k] > 0) (void)tc::mbar_wait(bars[k], (nh[k] - 1) & 1);
  }
  if (s.err && warp == kBwCompute / 32 + 2 && lane == 0) (void)tc::mbar_wait(&s.bar_w, cur != ni0 ? 1 : 0);
  if (tid == 0 && s.err && g.err) atomicExch(g.err, 1);
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, H);
}

// ---------------------------------------------------------------------------
// weight gradients: split over samples, 64 samples per stage
// ---------------------------------------------------------------------------
constexpr int kWgSamples = 64;
constexpr int kWgThreads = 128;
// stage layout (bytes): A da2 | A da1 | A h2 (each 2 blocks of 64 features x
// 64 samples), B h1 (4 blocks: 256 columns), B x (64 samples x D), B dz
constexpr int kWgA = 2 * kWgSamples * 128;  // 16 KB
constexpr int kWgDa2 = 0, kWgDa1 = kWgA, kWgH2 = 2 * kWgA, kWgH1 = 3 * kWgA;
constexpr int kWgX = kWgH1 + 4 * kWgSamples * 128;        // 80 KB
constexpr int kWgDz = kWgX + kWgSamples * 128;            // x takes at most 8 KB
constexpr int kWgStageBytes = kWgDz + kWgSamples * 32;    // 90 KB
constexpr int kWgMaxCols = 256 + 16 + 64 + 16 + 16;       // dW2 | db2 | dW1 | db1 | dW3^T

template <int D>
struct WgCols {  // TMEM / partial-block column of each product
  static constexpr int DW2 = 0, DB2 = 256, DW1 = 272, DB1 = 272 + D, DW3 = 288 + D, NC0 = 304 + D;
};

struct WgSmem {
  alignas(1024) uint8_t st[2][kWgStageBytes];
  alignas(1024) uint8_t ones[512];  // 16 samples x 16 columns of bf16 ones (B of the bias sums)
  uint64_t full[2], empty[2], bar_mma;
  uint32_t tmem_base;
  int32_t err;
};

struct WgNet {
  const uint8_t *da2, *da1, *h1, *h2, *dz;  // tile images
};

struct WgArgs {
  WgNet net[2];
  const uint8_t* x;   // shared input tile images
  int64_t n;          // valid samples
  int nstages;        // ceil(n / 64)
  int spc[2];         // stages per CTA, per column chunk
  int S[2];           // sample chunks (CTAs per group), per column chunk
  float* part;        // one [128][kWgMaxCols] partial block per CTA, in CTA order
  int32_t* err;
};

// CTA b of the weight-gradient launch: its output group and sample chunk.
// Groups are ordered (network, row block, column chunk); the CTAs of one
// (network, row block) are S[0] chunks of column chunk 0, then S[1] of
// column chunk 1 (with one column chunk, S[0] chunks per group).
template <int NCH>
__host__ __device__ __forceinline__ void wg_cta(int b, const int (&S)[2], int& grp, int& chunk) {
  if (NCH == 2) {
    const int per = S[0] + S[1], q = b / per, r = b % per;
    const int nc = r < S[0] ? 0 : 1;
    grp = 2 * q + nc;
    chunk = nc ? r - S[0] : r;
  } else {
    grp = b / S[0];
    chunk = b % S[0];
  }
}

// first CTA (partial block) of group grp
template <int NCH>
__host__ __device__ __forceinline__ int wg_first_cta(int grp, const int (&S)[2]) {
  return NCH == 2 ? (grp >> 1) * (S[0] + S[1]) + ((grp & 1) ? S[0] : 0) : grp * S[0];
}

template <int D, int H>
__global__ void __launch_bounds__(kWgThreads, 1) wgrad_kernel(WgArgs g) {
  using Cn = WgCols<D>;
  constexpr int NCH = H / 256, MB = H / 128;
  constexpr int XB = D * 2;                    // x row bytes (64 or 128)
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  WgSmem& s = *reinterpret_cast<WgSmem*>(base);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int grp, chunk;
  wg_cta<NCH>((int)blockIdx.x, g.S, grp, chunk);
  const int ni = grp / (MB * NCH), mb = (grp / NCH) % MB, nc = grp % NCH;
  const bool first = nc == 0;  // column chunk 0 also takes dW1, db1, dW3^T
  const WgNet& nt = g.net[ni];
  const int spc = nc ? g.spc[1] : g.spc[0];
  const int k0 = chunk * spc, k1 = min(k0 + spc, g.nstages);
  if (tid == 0) {
    s.err = 0;
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.full[i], 1);
      tc::mbar_init(&s.empty[i], 1);
    }
    tc::mbar_init(&s.bar_mma, 1);
    tc::fence_mbar_init();
  }
  for (int i = tid; i < 512 / 4; i += kWgThreads) reinterpret_cast<uint32_t*>(s.ones)[i] = 0x3F803F80u;
  if (warp == 0) tc::tmem_alloc(&s.tmem_base, 512);
  tc::fence_async_smem();
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = s.tmem_base;
  const int64_t hb = (int64_t)kWgSamples * 128;  // bytes of one 64-sample half of a 128-row block
  int last_issued = -1;
  if (warp == 0) {
    if (lane == 0) {
      for (int k = k0; k < k1; ++k) {
        const int j = k - k0, slot = j & 1;
        if (j >= 2 && !tc::mbar_wait(&s.empty[slot], ((j - 2) >> 1) & 1)) {
          atomicExch(&s.err, 1);
          break;
        }
        const int64_t tile = k >> 1, half = k & 1;
        const int64_t tb = tile * (int64_t)(kBwRows * H * 2);  // tile image base of a hidden-width operand
        uint8_t* d = s.st[slot];
        const uint32_t bytes = (uint32_t)(2 * hb + 4 * hb + (first ? 4 * hb + kWgSamples * XB + kWgSamples * 32 : 0));
        tc::mbar_expect_tx(&s.full[slot], bytes);
        for (int q = 0; q < 2; ++q) {
          const int64_t off = tb + (int64_t)(2 * mb + q) * kBwRows * 128 + half * hb;
          tc::bulk_g2s(d + kWgDa2 + q * hb, nt.da2 + off, (uint32_t)hb, &s.full[slot]);
          if (first) {
            tc::bulk_g2s(d + kWgDa1 + q * hb, nt.da1 + off, (uint32_t)hb, &s.full[slot]);
            tc::bulk_g2s(d + kWgH2 + q * hb, nt.h2 + off, (uint32_t)hb, &s.full[slot]);
          }
        }
        for (int q = 0; q < 4; ++q) {
          const int64_t off = tb + (int64_t)(4 * nc + q) * kBwRows * 128 + half * hb;
          tc::bulk_g2s(d + kWgH1 + q * hb, nt.h1 + off, (uint32_t)hb, &s.full[slot]);
        }
        if (first) {
          tc::bulk_g2s(d + kWgX, g.x + tile * (int64_t)(kBwRows * XB) + half * kWgSamples * XB,
                       (uint32_t)(kWgSamples * XB), &s.full[slot]);
          tc::bulk_g2s(d + kWgDz, nt.dz + tile * (int64_t)(kBwRows * 32) + half * kWgSamples * 32,
                       (uint32_t)(kWgSamples * 32), &s.full[slot]);
        }
        last_issued = j;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t onea = tc::smem_u32(s.ones);
      constexpr uint32_t kIdW2 = tc::idesc_bf16_mn(128, 256, 1, 1);
      constexpr uint32_t kId16 = tc::idesc_bf16_mn(128, 16, 1, 1);
      constexpr uint32_t kIdD = tc::idesc_bf16_mn(128, D, 1, 1);
      constexpr uint32_t kXLayout = D == 32 ? tc::kLayoutSW64 : tc::kLayoutSW128;
      constexpr uint32_t kXAtom = D == 32 ? 512 : 1024;
      const uint64_t ones = tc::desc_strided(onea, 16, 256, tc::kLayoutSW32);
      for (int k = k0; k < k1; ++k) {
        const int j = k - k0, slot = j & 1;
        if (!tc::mbar_wait(&s.full[slot], (j >> 1) & 1)) {
          atomicExch(&s.err, 1);
          break;
        }
        tc::fence_after();
        const uint32_t sa = tc::smem_u32(s.st[slot]);
#pragma unroll
        for (int kk = 0; kk < kWgSamples / 16; ++kk) {
          const uint32_t acc = (j | kk) != 0;
          const uint64_t a2 = tc::desc_strided(sa + kWgDa2 + kk * 2048, (uint32_t)hb, 1024, tc::kLayoutSW128);
          tc::mma_bf16(tmem + Cn::DW2, a2, tc::desc_strided(sa + kWgH1 + kk * 2048, (uint32_t)hb, 1024, tc::kLayoutSW128),
                       kIdW2, acc);
          if (first) {
            tc::mma_bf16(tmem + Cn::DB2, a2, ones, kId16, acc);
            const uint64_t a1 = tc::desc_strided(sa + kWgDa1 + kk * 2048, (uint32_t)hb, 1024, tc::kLayoutSW128);
            tc::mma_bf16(tmem + Cn::DW1, a1,
                         tc::desc_strided(sa + kWgX + kk * 16 * XB, 16, kXAtom, kXLayout), kIdD, acc);
            tc::mma_bf16(tmem + Cn::DB1, a1, ones, kId16, acc);
            tc::mma_bf16(tmem + Cn::DW3, tc::desc_strided(sa + kWgH2 + kk * 2048, (uint32_t)hb, 1024, tc::kLayoutSW128),
                         tc::desc_strided(sa + kWgDz + kk * 512, 16, 256, tc::kLayoutSW32), kId16, acc);
          }
        }
        tc::mma_commit(&s.empty[slot]);
      }
      tc::mma_commit(&s.bar_mma);
    }
  }
  // epilogue: the accumulators of this CTA's 128 output rows
  __syncwarp();
  const bool have = k1 > k0;
  if (have && !tc::mbar_wait(&s.bar_mma, 0)) atomicExch(&s.err, 1);
  tc::fence_after();
  __syncthreads();
  {
    const int row = warp * 32 + lane;
    float* prow = g.part + ((int64_t)blockIdx.x * 128 + row) * kWgMaxCols;
    const int ncols = first ? Cn::NC0 : 256;
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
    for (int c = 0; c < ncols; c += 16) {
      float v[16];
      tc::tmem_ld16(lane_addr + (uint32_t)c, v);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        *reinterpret_cast<float4*>(prow + c + 4 * q) =
            (have && !s.err) ? make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3])
                             : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    }
  }
  tc::fence_before();
  __syncthreads();
  if (s.err && warp == 0 && lane == 0 && last_issued >= 0)
    (void)tc::mbar_wait(&s.full[last_issued & 1], (last_issued >> 1) & 1);
  if (tid == 0 && s.err && g.err) atomicExch(g.err, 1);
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// The rest of the minibatch gradient and its squared norm, in one launch of
// kWgReduceBlocks blocks (all orders fixed, so the result is deterministic):
//   - every weight and hidden-bias entry: the sum over the S sample chunks
//     of its partial blocks, in chunk order;
//   - blocks 0 .. 5 + A also sum the loss partial rows, one quantity per
//     block (the five minibatch statistics, then the head-bias gradients
//     from the unrounded dz): thread t takes rows t, t + 512, ... in order,
//     then a fixed shuffle tree and the warps in order;
//   - each block writes the fp32 sum of squares of the entries it wrote
//     (threads in order of a fixed tree), the Adam kernel sums the blocks.
constexpr int kWgReduceBlocks = 256;
constexpr int kWgReduceThreads = 512;  // 27 warps per SM, eight chunk loads in flight per thread
constexpr int kLossPartW = 32;  // loss-kernel partial row: pg, ent, kl, clip, vl, db3[16], dc3

template <int D, int H>
__global__ void __launch_bounds__(kWgReduceThreads) wgrad_reduce_kernel(const float* __restrict__ part, int S0, int S1,
                                                           int A,
                                                           float* __restrict__ grad, const float* __restrict__ lossp,
                                                           int nlb, double* __restrict__ stat5,
                                                           float* __restrict__ sq) {
  using Cn = WgCols<D>;
  constexpr int NCH = H / 256, MB = H / 128;
  __shared__ float red[kWgReduceThreads / 32];
  const MlpLayout Lp = mlp_layout(D, H, A);
  const int64_t total = (int64_t)2 * MB * NCH * 128 * kWgMaxCols;
  float q = 0.0f;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int col = (int)(i % kWgMaxCols);
    const int row = (int)((i / kWgMaxCols) % 128);
    const int grp = (int)(i / ((int64_t)kWgMaxCols * 128));
    const int ni = grp / (MB * NCH), mb = (grp / NCH) % MB, nc = grp % NCH;
    const int o = mb * 128 + row;
    const int nout = ni ? 1 : A;
    int64_t dst = -1;
    if (col < 256) {
      dst = (ni ? Lp.v2 : Lp.w2) + (int64_t)o * H + nc * 256 + col;
    } else if (nc == 0) {
      if (col == Cn::DB2) dst = (ni ? Lp.c2 : Lp.b2) + o;
      else if (col >= Cn::DW1 && col < Cn::DW1 + D) dst = (ni ? Lp.v1 : Lp.w1) + (int64_t)o * D + (col - Cn::DW1);
      else if (col == Cn::DB1) dst = (ni ? Lp.c1 : Lp.b1) + o;
      else if (col >= Cn::DW3 && col < Cn::DW3 + nout) dst = (ni ? Lp.v3 : Lp.w3) + (int64_t)(col - Cn::DW3) * H + o;
    }
    if (dst < 0) continue;
    const int S[2] = {S0, S1};
    const int nch = nc ? S1 : S0;
    const float* p = part + ((int64_t)wg_first_cta<NCH>(grp, S) * 128 + row) * kWgMaxCols + col;
    float acc = 0.0f;
#pragma unroll 8
    for (int k = 0; k < nch; ++k) acc += p[(int64_t)k * 128 * kWgMaxCols];
    grad[dst] = acc;
    q = fmaf(acc, acc, q);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ double redd[kWgReduceThreads / 32];
  const int w = (int)blockIdx.x;  // statistic w (w < 5), then head-bias sum j = w - 5 (policy j < A, then the value's)
  if (w < 5 + A + 1) {
    const int col = w < 5 ? w : (w - 5 < A ? 5 + (w - 5) : 21);
    double t = 0.0;
#pragma unroll 4
    for (int b = threadIdx.x; b < nlb; b += blockDim.x) t += (double)lossp[(int64_t)b * kLossPartW + col];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (lane == 0) redd[warp] = t;
    __syncthreads();
    if (threadIdx.x == 0) {
      double u = 0.0;
      for (int k = 0; k < (int)(blockDim.x >> 5); ++k) u += redd[k];
      if (w < 5) {
        stat5[w] = u;
      } else {
        const int j = w - 5;
        const float g = (float)u;
        grad[j < A ? Lp.b3 + j : Lp.c3] = g;
        q = fmaf(g, g, q);
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) q += __shfl_xor_sync(0xffffffffu, q, off);
  if (lane == 0) red[warp] = q;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];
    sq[blockIdx.x] = t;
  }
}

int wgrad_reduce_blocks() { return kWgReduceBlocks; }

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
// partial blocks for up to kWgMaxCtas CTAs (the launch keeps groups x S below it)
constexpr int kWgMaxCtas = 256;
int64_t wgrad_partial_bytes() { return (int64_t)kWgMaxCtas * 128 * kWgMaxCols * 4; }

template <int D, int H>
static pe_status bwd_images(const float* params, int A, uint8_t* const img[2], cudaStream_t st) {
  {
    ProfScope ps(PE_PROF_PPO_OTHER, st);
    bwd_image_kernel<D, H><<<dim3(128, 2), 256, 0, st>>>(params, A, img[0], img[1]);
  }
  PE_CHECK_LAUNCH("bwd_image_kernel");
  return PE_OK;
}

template <int D, int H>
static pe_status bwd_launch(const float* params, int A, uint8_t* const img[2], const uint8_t* x,
                            const uint8_t* const dz[2], const uint8_t* const h1[2], const uint8_t* const h2[2],
                            uint8_t* const da2[2], uint8_t* const da1[2], int64_t n, float* part, float* grad,
                            const float* lossp, int nlb, double* stat5, float* sq, int32_t* err, bool data_done,
                            cudaStream_t st) {
  int dev = 0, sms = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int64_t tiles = (n + kBwRows - 1) / kBwRows;
  if (data_done) {
    // the backward images and the data products came with the fused forward-backward kernel
  } else if constexpr (H == 256) {
    return fail(PE_EINVAL, "the 72B data products run in the fused forward-backward kernel");
  } else {
    auto kern = bwd_data_kernel<H>;
    const int bytes = (int)sizeof(BwdSmem<H>) + 1024;
    PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    const int grid = (int)std::min<int64_t>(2 * tiles, sms);
    BwdArgs a;
    for (int ni = 0; ni < 2; ++ni) {
      a.img[ni] = img[ni];
      a.dz[ni] = dz[ni];
      a.h1[ni] = h1[ni];
      a.h2[ni] = h2[ni];
      a.da2[ni] = da2[ni];
      a.da1[ni] = da1[ni];
    }
    a.n = n;
    a.err = err;
    ProfScope ps(PE_PROF_PPO_GRAD, st);
    kern<<<grid, kBwThreads, bytes, st>>>(a);
  }
  PE_CHECK_LAUNCH("bwd_data_kernel");
  {
    constexpr int groups = 2 * (H / 128) * (H / 256);
    WgArgs a;
    for (int ni = 0; ni < 2; ++ni) a.net[ni] = WgNet{da2[ni], da1[ni], h1[ni], h2[ni], dz[ni]};
    a.x = x;
    a.n = n;
    a.nstages = (int)((n + kWgSamples - 1) / kWgSamples);
    // CTAs per (network, row block), split between the column chunks in
    // proportion to the bytes a stage brings in: chunk 0 also loads da1, h2,
    // x and dz (for the Stress networks 90 KB per stage against 48 KB), so
    // with equal shares its CTAs would set the launch's length
    constexpr int NCH = H / 256;
    const int cap = std::max(NCH, std::min(sms, kWgMaxCtas) / (groups / NCH));
    int want[2] = {cap, 0};
    if (NCH == 2) {
      const double hb = (double)kWgSamples * 128;
      const double b0 = 10 * hb + kWgSamples * (D * 2 + 32), b1 = 6 * hb;
      want[0] = std::min(cap - 1, std::max(1, (int)std::lround(cap * b0 / (b0 + b1))));
      want[1] = cap - want[0];
    }
    int ctas = 0;
    for (int c = 0; c < 2; ++c) {
      a.spc[c] = a.S[c] = 0;
      if (c >= NCH) continue;
      const int s_want = std::max(1, std::min(want[c], a.nstages));
      a.spc[c] = (a.nstages + s_want - 1) / s_want;
      a.S[c] = (a.nstages + a.spc[c] - 1) / a.spc[c];
      ctas += a.S[c];
    }
    ctas *= groups / NCH;
    a.part = part;
    a.err = err;
    auto kern = wgrad_kernel<D, H>;
    const int bytes = (int)sizeof(WgSmem) + 1024;
    PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    ProfScope ps(PE_PROF_PPO_GRAD, st);
    kern<<<ctas, kWgThreads, bytes, st>>>(a);
    PE_CHECK_LAUNCH("wgrad_kernel");
    wgrad_reduce_kernel<D, H><<<kWgReduceBlocks, kWgReduceThreads, 0, st>>>(part, a.S[0], a.S[1], A, grad, lossp, nlb,
                                                                           stat5, sq);
    PE_CHECK_LAUNCH("wgrad_reduce_kernel");
  }
  return PE_OK;
}

// the whole backward of both networks of a bf16 PPO minibatch step: writes
// every entry of the gradient vector (the head biases from the loss kernel's
// partials), the five minibatch statistics, and kWgReduceBlocks partial sums
// of squares of the gradient
pe_status bf16_backward(const pe_net& net, const float* params, uint8_t* const img[2], const uint8_t* x,
                        const uint8_t* const dz[2], const uint8_t* const h1[2], const uint8_t* const h2[2],
                        uint8_t* const da2[2], uint8_t* const da1[2], int64_t n, float* part, float* grad,
                        const float* lossp, int nlb, double* stat5, float* sq, int32_t* err, bool data_done,
                        cudaStream_t st) {
  if (n <= 0) return PE_OK;
  if (net.obs_dim == 32 && net.hidden == 256)
    return bwd_launch<32, 256>(params, net.n_actions, img, x, dz, h1, h2, da2, da1, n, part, grad, lossp, nlb, stat5,
                               sq, err, data_done, st);
  if (net.obs_dim == 64 && net.hidden == 512)
    return bwd_launch<64, 512>(params, net.n_actions, img, x, dz, h1, h2, da2, da1, n, part, grad, lossp, nlb, stat5,
                               sq, err, data_done, st);
  return fail(PE_EINVAL, "unsupported bf16 network for the backward pass");
}

pe_status bf16_bwd_images(const pe_net& net, const float* params, uint8_t* const img[2], cudaStream_t st) {
  if (net.obs_dim == 32 && net.hidden == 256) return bwd_images<32, 256>(params, net.n_actions, img, st);
  if (net.obs_dim == 64 && net.hidden == 512) return bwd_images<64, 512>(params, net.n_actions, img, st);
  return fail(PE_EINVAL, "unsupported bf16 network for the backward images");
}

}  // namespace pe
