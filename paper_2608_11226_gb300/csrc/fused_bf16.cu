// Fused forward and backward-data pass of the bf16 PPO update (Sec. 4.2) for
// the 72B networks (D = 32, H = 256): per 128-sample tile,
//   x -> h1 = tanh(W1 x + b1) -> h2 = tanh(W2 h1 + b2) -> z = W3 h2 + b3
//     -> loss and dz (the head epilogue) -> dh2 = dz W3 -> da2 = bf16(dh2 (1 - h2^2))
//     -> dh1 = da2 W2 -> da1 = bf16(dh1 (1 - h1^2)),
// in one kernel, with the arithmetic of mlp_bf16_pair_kernel followed by
// the backward data products of bwd_bf16.cu (the same bits).  h2 and dz
// never leave the chip between the two halves: da2 overwrites h2 in place in
// the tile's shared buffer, and dz goes to shared memory beside its tile
// image.  The tile images the weight-gradient kernel reads (x, h1, h2, dz,
// da2, da1) are written as before.
//
// Two tiles are in flight per CTA (slots 0 and 1), each with its own 64 KB
// activation buffer (X, then h1, h2, da2), its dz tile and half of TMEM
// (columns 256 s .. 256 s + 255, used in turn by layer 1, layer 2, the head,
// dh2 and dh1).  Warps 0-15 run the epilogues, warp 16 streams the weights
// that do not stay resident through a two-slot ring of 32 KB stages (per
// tile pair: W1, the four W2 K-blocks of each slot, the four W2^T stages of
// each slot), warp 17 issues the MMAs.  Hand-overs are mbarriers that
// complete once per tile pair:
//   epilogue -> issuer (16 arrivals): xin, h1in, h2in, dzin, d2in;
//   issuer -> epilogue (tcgen05.commit): mma1, mma2, head, mdh2, mdh1.
// The loss epilogue of slot s runs on the four warps of column slice s (one
// per TMEM lane quadrant), so the two slots' losses run side by side.  The
// last epilogue of a tile reads h1 back from the h1 tile image that the same
// thread wrote in the first one (the same rows and columns), from L2.
#include <algorithm>

#include "bf16_layout.cuh"
#include "mlp_f32.cuh"
#include "tc.cuh"

namespace pe {

constexpr int kFuThreads = 576;  // 16 epilogue warps, a ring producer, an MMA issuer

template <int D, int H>
struct FusedSmem {
  alignas(1024) uint8_t act[2][kTcRows * H * 2];  // per slot: X (aliases the start), h1, h2, then da2
  alignas(1024) uint8_t ring[2][kBwStage];         // W1, W2 and W2^T stages
  alignas(1024) uint8_t w3[Img<D, H>::W3];         // B of the head (K-major SW128)
  alignas(1024) uint8_t w3t[BwdImg<H>::W3T];       // B of dh2 = dz W3 (K-major SW32)
  alignas(1024) uint8_t dz[2][kTcRows * 32];       // A of dh2 per slot (K-major SW32)
  float b1[H], b2[H], b3[kHeadN];
  uint64_t bar_w, fin, full[2], empty[2];
  uint64_t mma1[2], mma2[2], head[2], mdh2[2], mdh1[2];
  uint64_t xin[2], h1in[2], h2in[2], dzin[2], d2in[2];
  uint32_t tmem_base;
  int32_t err;
};

struct FusedArgs {
  const uint8_t* img;    // forward weight image of the network (W1 | W2 | W3)
  const uint8_t* bimg;   // backward weight image (W3^T | W2^T stages)
  const float* params;
  int A, value_net;
  const __nv_bfloat16* obs;
  int64_t n;             // valid samples (rows gathered through save.gather)
  MlpSave save;          // gather; x (policy only), h1, h2 tile images; the loss (dz images, partial rows)
  uint8_t* da2;          // out: da2 tile images
  uint8_t* da1;          // out: da1 tile images
  int32_t* err;
};

template <int D, int H>
__global__ void __launch_bounds__(kFuThreads, 1) ppo_fused_pair_kernel(FusedArgs g) {
  using I = Img<D, H>;
  using Bw = BwdImg<H>;
  static_assert(H == 256 && Bw::NH == 1 && Bw::KB == 4, "two tiles in flight need 2 x 256 TMEM columns");
  static_assert(I::W1 <= kBwStage, "W1 travels as one ring stage");
  constexpr int KB2 = H / 64;                    // W2 K-blocks per tile (32 KB each)
  constexpr int CPR = D / 8;                     // 16-byte observation chunks per row
  constexpr int XCH = kTcRows * CPR / kTcThreads;
  constexpr int kTile = kTcRows * H * 2;         // bytes of an h / da tile image
  constexpr int NJ = H / 64;                     // 16-column chunks per epilogue thread
  static_assert(kTcRows * CPR % kTcThreads == 0, "observation chunks per thread");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  FusedSmem<D, H>& s = *reinterpret_cast<FusedSmem<D, H>*>(base);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const MlpLayout Lp = mlp_layout(D, H, g.A);
  const int nout = g.value_net ? 1 : g.A;
  if (tid == 0) {
    s.err = 0;
    tc::mbar_init(&s.bar_w, 1);
    tc::mbar_init(&s.fin, 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&s.full[i], 1);
      tc::mbar_init(&s.empty[i], 1);
      tc::mbar_init(&s.mma1[i], 1);
      tc::mbar_init(&s.mma2[i], 1);
      tc::mbar_init(&s.head[i], 1);
      tc::mbar_init(&s.mdh2[i], 1);
      tc::mbar_init(&s.mdh1[i], 1);
      tc::mbar_init(&s.xin[i], 16);
      tc::mbar_init(&s.h1in[i], 16);
      tc::mbar_init(&s.h2in[i], 16);
      tc::mbar_init(&s.dzin[i], 16);
      tc::mbar_init(&s.d2in[i], 16);
    }
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&s.tmem_base, 512);
  for (int i = tid; i < H; i += blockDim.x) {
    s.b1[i] = __ldg(g.params + (g.value_net ? Lp.c1 : Lp.b1) + i);
    s.b2[i] = __ldg(g.params + (g.value_net ? Lp.c2 : Lp.b2) + i);
  }
  if (tid < kHeadN) s.b3[tid] = tid < nout ? __ldg(g.params + (g.value_net ? Lp.c3 : Lp.b3) + tid) : 0.0f;
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = s.tmem_base;
  const int64_t tiles = (g.n + kTcRows - 1) / kTcRows;
  const int my_tiles = (int)((tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);
  const int npairs = (my_tiles + 1) / 2;
  // a bounded wait that is skipped once the CTA has an error (so that a
  // failed CTA does not spend one time-out per remaining hand-over)
  auto wt = [&](uint64_t* b, uint32_t par) -> bool {
    if (*reinterpret_cast<volatile int32_t*>(&s.err)) return false;
    if (tc::mbar_wait(b, par)) return true;
    atomicExch(&s.err, 1);
    return false;
  };
  int last_issued = -1;
  if (warp == 16) {
    // producer: per tile pair W1, the W2 K-blocks of slot 0 and of slot 1,
    // the W2^T stages of slot 0 and of slot 1, in the issuer's order
    if (lane == 0) {
      int gs = 0;
      auto issue = [&](const uint8_t* src, uint32_t bytes) -> bool {
        const int slot = gs & 1;
        if (gs >= 2 && !wt(&s.empty[slot], ((gs - 2) >> 1) & 1)) return false;
        tc::mbar_expect_tx(&s.full[slot], bytes);
        tc::bulk_g2s(s.ring[slot], src, bytes, &s.full[slot]);
        last_issued = gs++;
        return true;
      };
      bool ok = true;
      for (int p = 0; p < npairs && ok; ++p) {
        ok = issue(g.img, (uint32_t)I::W1);
        for (int sl = 0; sl < 2 && ok; ++sl)
          for (int kb = 0; kb < KB2 && ok; ++kb)
            ok = issue(g.img + I::W1 + (int64_t)kb * kBwStage, (uint32_t)kBwStage);
        for (int sl = 0; sl < 2 && ok; ++sl)
          for (int kb = 0; kb < Bw::KB && ok; ++kb)
            ok = issue(g.bimg + Bw::W3T + (int64_t)kb * kBwStage, (uint32_t)kBwStage);
      }
    }
  } else if (warp == 17) {
    // MMA issuer
    if (lane == 0) {
      tc::mbar_expect_tx(&s.bar_w, (uint32_t)(I::W3 + Bw::W3T));
      tc::bulk_g2s(s.w3, g.img + I::W1 + I::W2, (uint32_t)I::W3, &s.bar_w);
      tc::bulk_g2s(s.w3t, g.bimg, (uint32_t)Bw::W3T, &s.bar_w);
      (void)wt(&s.bar_w, 0);
      const uint32_t w3a = tc::smem_u32(s.w3), w3ta = tc::smem_u32(s.w3t);
      constexpr uint32_t kL1 = I::RB1 == 64 ? tc::kLayoutSW64 : tc::kLayoutSW128;
      constexpr uint32_t kIdN = tc::idesc_bf16(kTcRows, H);
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
      for (int p = 0; p < npairs; ++p) {
        const uint32_t par = p & 1;
        // layer 1 of both slots from one W1 stage
        const uint32_t w1a = stage_in();
        for (int sl = 0; sl < 2; ++sl) {
          (void)wt(&s.xin[sl], par);
          tc::fence_after();
          const uint32_t xa = tc::smem_u32(s.act[sl]);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk)
            tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(xa + kk * 32, 8 * I::RB1, kL1),
                         tc::desc_kmajor(w1a + kk * 32, 8 * I::RB1, kL1), kIdN, kk > 0);
          tc::mma_commit(&s.mma1[sl]);
        }
        stage_out();
        // layer 2, W2 streamed per slot
        for (int sl = 0; sl < 2; ++sl) {
          (void)wt(&s.h1in[sl], par);
          tc::fence_after();
          const uint32_t ha = tc::smem_u32(s.act[sl]);
          for (int kb = 0; kb < KB2; ++kb) {
            const uint32_t ra = stage_in();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(ha + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                           tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, (kb | kk) != 0);
            stage_out();
          }
          tc::mma_commit(&s.mma2[sl]);
        }
        // head (W3 resident)
        for (int sl = 0; sl < 2; ++sl) {
          (void)wt(&s.h2in[sl], par);
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
        // dh2 = dz W3 (W3^T resident): one K = 16 MMA per slot
        for (int sl = 0; sl < 2; ++sl) {
          (void)wt(&s.dzin[sl], par);
          tc::fence_after();
          tc::mma_bf16(tmem + sl * 256, tc::desc_strided(tc::smem_u32(s.dz[sl]), 16, 256, tc::kLayoutSW32),
                       tc::desc_strided(w3ta, 16, 256, tc::kLayoutSW32), kIdN, 0);
          tc::mma_commit(&s.mdh2[sl]);
        }
        // dh1 = da2 W2, W2^T streamed per slot
        for (int sl = 0; sl < 2; ++sl) {
          (void)wt(&s.d2in[sl], par);
          tc::fence_after();
          const uint32_t da = tc::smem_u32(s.act[sl]);
          for (int kb = 0; kb < Bw::KB; ++kb) {
            const uint32_t ra = stage_in();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_bf16(tmem + sl * 256, tc::desc_kmajor(da + kb * kTcRows * 128 + kk * 32, 1024, tc::kLayoutSW128),
                           tc::desc_kmajor(ra + kk * 32, 1024, tc::kLayoutSW128), kIdN, (kb | kk) != 0);
            stage_out();
          }
          tc::mma_commit(&s.mdh1[sl]);
        }
      }
      // every MMA of this CTA completes before TMEM is released
      tc::mma_commit(&s.fin);
      if (!tc::mbar_wait(&s.fin, 0)) atomicExch(&s.err, 1);
      if (s.err) (void)tc::mbar_wait(&s.bar_w, 0);
    }
  } else {
    // epilogue warps: four TMEM lane quadrants x four column slices
    const int quad = warp & 3, slice = warp >> 2, row = quad * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
    auto tile_of = [&](int k) { return (int64_t)blockIdx.x + (int64_t)k * gridDim.x; };
    auto rows_of = [&](int k) {
      if (k >= my_tiles) return 0;
      const int64_t left = g.n - tile_of(k) * kTcRows;
      return (int)(left < kTcRows ? left : kTcRows);
    };
    uint4 xv[2][XCH];
    auto fetch_x = [&](int k, uint4 (&dst)[XCH]) {
      const int64_t tl = tile_of(k);
#pragma unroll
      for (int q = 0; q < XCH; ++q) {
        const int i = tid + q * kTcThreads, r = i / CPR, c = i % CPR;
        const int64_t rr = tl * kTcRows + r;
        dst[q] = make_uint4(0, 0, 0, 0);
        if (k < my_tiles && rr < g.n) {
          const int64_t src = g.save.gather ? (int64_t)__ldg(g.save.gather + rr) : rr;
          dst[q] = __ldg(reinterpret_cast<const uint4*>(g.obs + src * D) + c);
        }
      }
    };
    auto put_x = [&](int sl, int k) {
      const int64_t tl = tile_of(k);
#pragma unroll
      for (int q = 0; q < XCH; ++q) {
        const int i = tid + q * kTcThreads, r = i / CPR, c = i % CPR;
        const uint32_t off = tc::swz_offset<I::RB1>(r, c * 8, kTcRows);
        *reinterpret_cast<uint4*>(s.act[sl] + off) = xv[sl][q];
        if (g.save.x && k < my_tiles)
          *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(g.save.x) + tl * (int64_t)(kTcRows * D * 2) + off) =
              xv[sl][q];
      }
    };
    auto handover = [&](uint64_t* bar) {
      tc::fence_async_smem();
      tc::fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
    };
    // hidden layer: tanh(acc + bias) -> bf16 -> act[sl] and the tile image
    auto hidden = [&](int sl, const float* bias, __nv_bfloat16* gsave, int k) {
      uint8_t* gi = (gsave && k < my_tiles) ? reinterpret_cast<uint8_t*>(gsave) + tile_of(k) * (int64_t)kTile : nullptr;
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        const int c = slice * (H / 4) + j * 16;
        float v[16];
        tc::tmem_ld16(lane_base + (uint32_t)(sl * 256 + c), v);
        uint32_t pk[8];
        tc::tanh16_bf16(v, bias + c, pk);
        const uint32_t o0 = tc::swz_offset<128>(row, c, kTcRows), o1 = tc::swz_offset<128>(row, c + 8, kTcRows);
        const uint4 lo = make_uint4(pk[0], pk[1], pk[2], pk[3]), hi = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        *reinterpret_cast<uint4*>(s.act[sl] + o0) = lo;
        *reinterpret_cast<uint4*>(s.act[sl] + o1) = hi;
        if (gi) {
          *reinterpret_cast<uint4*>(gi + o0) = lo;
          *reinterpret_cast<uint4*>(gi + o1) = hi;
        }
      }
    };
    // head: the PPO loss per row, dz to its tile image and to the slot's
    // shared dz tile (zeros for a slot without a tile); slot s by the four
    // warps of column slice s (one per TMEM lane quadrant), so that the two
    // slots' losses run side by side
    auto head_epi = [&](int sl, int k) {
      if (slice != sl) return;
      if (k < my_tiles) {
        float v[16];
        tc::tmem_ld16(lane_base + (uint32_t)(sl * 256), v);
        ppo_head_row(g.save.loss, g.value_net, g.A, s.b3, g.save.gather, tile_of(k), row, g.n, v, quad, s.dz[sl]);
      } else {
        *reinterpret_cast<uint4*>(s.dz[sl] + row * 32) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(s.dz[sl] + row * 32 + 16) = make_uint4(0, 0, 0, 0);
      }
    };
    // d = bf16(TMEM (1 - h^2)): da2 with h2 from act[sl] (in place), or da1
    // with h1 from registers (hv, loaded from this thread's own h1 writes)
    auto grad_epi = [&](int sl, int k, uint8_t* gout, const uint4 (*hv)[2]) {
      const bool valid = row < rows_of(k);
      uint8_t* outt = k < my_tiles ? gout + tile_of(k) * (int64_t)kTile : nullptr;
#pragma unroll
      for (int j = 0; j < NJ; ++j) {
        const int c = slice * (H / 4) + j * 16;
        float v[16];
        tc::tmem_ld16(lane_base + (uint32_t)(sl * 256 + c), v);
        const uint32_t o0 = tc::swz_offset<128>(row, c, kTcRows), o1 = tc::swz_offset<128>(row, c + 8, kTcRows);
        uint4 hb[2];
        if (hv) {
          hb[0] = hv[j][0];
          hb[1] = hv[j][1];
        } else {
          hb[0] = *reinterpret_cast<const uint4*>(s.act[sl] + o0);
          hb[1] = *reinterpret_cast<const uint4*>(s.act[sl] + o1);
        }
        uint32_t pk[8];
        tanh_grad16(v, hb, valid, pk);
        const uint4 lo = make_uint4(pk[0], pk[1], pk[2], pk[3]), hi = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        if (!hv) {
          *reinterpret_cast<uint4*>(s.act[sl] + o0) = lo;
          *reinterpret_cast<uint4*>(s.act[sl] + o1) = hi;
        }
        if (outt) {
          *reinterpret_cast<uint4*>(outt + o0) = lo;
          *reinterpret_cast<uint4*>(outt + o1) = hi;
        }
      }
    };
    fetch_x(0, xv[0]);
    fetch_x(1, xv[1]);
    for (int sl = 0; sl < 2; ++sl) {
      put_x(sl, sl);
      handover(&s.xin[sl]);
    }
    fetch_x(2, xv[0]);
    fetch_x(3, xv[1]);
    for (int p = 0; p < npairs; ++p) {
      const uint32_t par = p & 1;
      for (int sl = 0; sl < 2; ++sl) {
        (void)wt(&s.mma1[sl], par);
        tc::fence_after();
        hidden(sl, s.b1, g.save.h1, 2 * p + sl);
        handover(&s.h1in[sl]);
      }
      for (int sl = 0; sl < 2; ++sl) {
        (void)wt(&s.mma2[sl], par);
        tc::fence_after();
        hidden(sl, s.b2, g.save.h2, 2 * p + sl);
        handover(&s.h2in[sl]);
      }
      for (int sl = 0; sl < 2; ++sl) {
        (void)wt(&s.head[sl], par);
        tc::fence_after();
        head_epi(sl, 2 * p + sl);
        handover(&s.dzin[sl]);
      }
      for (int sl = 0; sl < 2; ++sl) {
        (void)wt(&s.mdh2[sl], par);
        tc::fence_after();
        grad_epi(sl, 2 * p + sl, g.da2, nullptr);
        handover(&s.d2in[sl]);
      }
      for (int sl = 0; sl < 2; ++sl) {
        const int k = 2 * p + sl;
        // this thread's h1 chunks of the tile, in flight during the dh1 MMAs
        uint4 hv[NJ][2];
        const uint8_t* h1t =
            k < my_tiles ? reinterpret_cast<const uint8_t*>(g.save.h1) + tile_of(k) * (int64_t)kTile : nullptr;
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
          const int c = slice * (H / 4) + j * 16;
          hv[j][0] = make_uint4(0, 0, 0, 0);
          hv[j][1] = make_uint4(0, 0, 0, 0);
          if (h1t) {
            hv[j][0] = __ldcg(reinterpret_cast<const uint4*>(h1t + tc::swz_offset<128>(row, c, kTcRows)));
            hv[j][1] = __ldcg(reinterpret_cast<const uint4*>(h1t + tc::swz_offset<128>(row, c + 8, kTcRows)));
          }
        }
        (void)wt(&s.mdh1[sl], par);
        tc::fence_after();
        grad_epi(sl, k, g.da1, hv);
        // the slot's buffer and TMEM half are free: the next pair's X
        if (p + 1 < npairs) {
          put_x(sl, k + 2);
          handover(&s.xin[sl]);
        }
      }
      fetch_x(2 * p + 4, xv[0]);
      fetch_x(2 * p + 5, xv[1]);
    }
  }
  tc::fence_before();
  __syncthreads();
  // on an error, the producer waits (bounded) for the copies it may still
  // have in flight before the CTA leaves
  if (s.err && warp == 16 && lane == 0)
    for (int q = last_issued - 1; q <= last_issued; ++q)
      if (q >= 0) (void)tc::mbar_wait(&s.full[q & 1], (q >> 1) & 1);
  if (tid == 0 && s.err && g.err) atomicExch(g.err, 1);
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
bool bf16_fused_supported(const pe_net& net) { return net.obs_dim == 32 && net.hidden == 256; }

pe_status bf16_fused_fwd_bwd(const pe_net& net, const uint8_t* img, const uint8_t* bimg, const float* params,
                             int value_net, const void* obs, const uint32_t* gather, int64_t n, const PpoHead& loss,
                             __nv_bfloat16* x, __nv_bfloat16* h1, __nv_bfloat16* h2, uint8_t* da2, uint8_t* da1,
                             int32_t* err, cudaStream_t st) {
  if (!bf16_fused_supported(net)) return fail(PE_EINVAL, "fused PPO forward-backward: 32-256-256 networks only");
  if (n <= 0) return PE_OK;
  int dev = 0, sms = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  PE_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int64_t tiles = (n + kTcRows - 1) / kTcRows;
  const int grid = (int)std::min<int64_t>((tiles + 1) / 2, sms);
  auto kern = ppo_fused_pair_kernel<32, 256>;
  constexpr int bytes = (int)sizeof(FusedSmem<32, 256>) + 1024;
  static_assert(bytes <= 232448, "fused kernel shared memory");
  PE_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
  FusedArgs a;
  a.img = img;
  a.bimg = bimg;
  a.params = params;
  a.A = net.n_actions;
  a.value_net = value_net;
  a.obs = reinterpret_cast<const __nv_bfloat16*>(obs);
  a.n = n;
  a.save = MlpSave{gather, x, h1, h2, loss};
  a.da2 = da2;
  a.da1 = da1;
  a.err = err;
  {
    ProfScope ps(PE_PROF_PPO_GRAD, st);
    kern<<<grid, kFuThreads, bytes, st>>>(a);
  }
  PE_CHECK_LAUNCH("ppo_fused_pair_kernel");
  return PE_OK;
}

}  // namespace pe
