// Blackwell (sm_103a) tensor-core primitives as inline PTX: tcgen05 MMA with
// TMEM accumulators, shared-memory matrix descriptors, TMEM allocation and
// loads, bulk copies and mbarriers.  Every wait is bounded: on timeout it
// returns false and the caller records an error instead of spinning forever.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace pe {
namespace tc {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// Swizzled K-major operand layouts (the byte address bits [4, 4+b) are
// XOR-ed with bits [7, 7+b)):
//   SW128: rows of 128 B (64 bf16), 8-row atoms of 1024 B, b = 3
//   SW64 : rows of  64 B (32 bf16), 8-row atoms of  512 B, b = 2
//   SW32 : rows of  32 B (16 bf16), 8-row atoms of  256 B, b = 1
// Element (r, k) of a tile with R rows and K columns (bf16) lives in K-block
// kb = k / KB (KB = 64, 32 or 16 elements) at byte
//   kb * R * RB + r * RB + (((k % KB) / 8) ^ ((r % 8) >> s)) * 16 + (k % 8) * 2
// with RB the row bytes and s = 0 for SW128, 1 for SW64, 2 for SW32; the atom
// base must be aligned to the atom size.
enum : uint32_t { kLayoutSW128 = 2, kLayoutSW64 = 4, kLayoutSW32 = 6 };

template <int RB>
__host__ __device__ __forceinline__ uint32_t swz_offset(int r, int k, int R) {
  static_assert(RB == 128 || RB == 64 || RB == 32, "row bytes of a swizzled layout");
  constexpr int KB = RB / 2;  // bf16 elements per row of a K-block
  const int kb = k / KB, kk = k % KB;
  const int chunk = kk / 8;
  const int phys = RB == 128 ? (chunk ^ (r & 7)) : RB == 64 ? (chunk ^ ((r >> 1) & 3)) : (chunk ^ ((r >> 2) & 1));
  return (uint32_t)(kb * R * RB + r * RB + phys * 16 + (kk % 8) * 2);
}

// The same bytes serve as an MN-major operand.  A tile stored as above with
// rows = K (samples) and contiguous elements = M or N (features) is the
// canonical MN-major swizzled layout: the 128/64/32-byte rows hold 64/32/16
// consecutive M (or N) elements of one K index, XOR-swizzled within 8-row
// atoms.  Its descriptor takes two strides: LBO = bytes between atoms that
// are adjacent along M/N (the next 64/32/16 elements), SBO = bytes between
// 8-row groups along K.

// tcgen05 shared-memory matrix descriptor, K-major, swizzled:
// start address >> 4 [0,14), leading-dim byte offset >> 4 [16,30) (unused
// for swizzled K-major), stride-dim byte offset >> 4 [32,46) (one 8-row atom),
// fixed 0b001 at [46,49), layout type [61,64).
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t saddr, uint32_t sbo_bytes, uint32_t layout) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1u << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)(layout & 7u) << 61;
  return d;
}

// shared-memory matrix descriptor with both byte strides given (MN-major
// operands, and K-major SW32 tiles): start >> 4 at [0,14), LBO >> 4 at
// [16,30), SBO >> 4 at [32,46), 0b001 at [46,49), layout type at [61,64)
__device__ __forceinline__ uint64_t desc_strided(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes,
                                                 uint32_t layout) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)(layout & 7u) << 61;
  return d;
}

// instruction descriptor for kind::f16 with bf16 A and B, fp32 D, both K-major
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// the same with A and/or B MN-major (bits 15 and 16 of the descriptor)
__host__ __device__ constexpr uint32_t idesc_bf16_mn(int M, int N, int a_mn, int b_mn) {
  return idesc_bf16(M, N) | ((uint32_t)(a_mn & 1) << 15) | ((uint32_t)(b_mn & 1) << 16);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t da, uint64_t db, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t"
      "}\n" ::"r"(tmem_d),
      "l"(da), "l"(db), "r"(idesc), "r"(accumulate));
}

// arrive on an mbarrier once every tcgen05 op issued so far by this thread completed
__device__ __forceinline__ void mma_commit(uint64_t* mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(mbar))
               : "memory");
}

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// generic-proxy shared-memory writes -> visible to the async proxy (MMA, bulk copies)
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// TMEM allocation by one full warp; the base address is written to *slot
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// 16 consecutive fp32 columns of this thread's TMEM lane (32x32b shape: warp
// w reads lanes 32*(w%4) .. +31; taddr carries the lane in bits [16,32))
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// named barrier `id` over `nthreads` threads that also ORs a predicate across
// them: every thread gets the same answer, so a loop can stop uniformly
__device__ __forceinline__ bool bar_any(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t"
      "}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// ask L2 to fetch the 128-byte line holding p (no register result, no wait)
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t"
      "}\n"
      : "=r"(ok)
      : "r"(smem_u32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}

// bounded wait for phase `parity` of the barrier: false after ~`cycles` SM cycles
__device__ __forceinline__ bool mbar_wait(uint64_t* b, uint32_t parity, long long cycles = 4000000000LL) {
  const long long t0 = clock64();
  while (!mbar_try_wait(b, parity)) {
    if (clock64() - t0 > cycles) return false;
  }
  return true;
}

// bulk copy global -> shared (size a multiple of 16 B, both addresses 16-B aligned);
// completion is signalled as transaction bytes on the mbarrier
__device__ __forceinline__ void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes, uint64_t* mbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_u32(mbar))
      : "memory");
}

// tanh of 16 hidden pre-activations (v + bias, one TMEM chunk of a thread's
// row), rounded to bf16 and packed in pairs; the bias is added with the
// packed two-lane fp32 add (the same rounding as two adds).
__device__ __forceinline__ void tanh16_bf16(const float (&v)[16], const float* bias, uint32_t (&pk)[8]) {
#pragma unroll
  for (int i = 0; i < 16; i += 2) {
    const float2 z = __fadd2_rn(make_float2(v[i], v[i + 1]), *reinterpret_cast<const float2*>(bias + i));
    __nv_bfloat162 r = __floats2bfloat162_rn(tanhf(z.x), tanhf(z.y));
    pk[i / 2] = *reinterpret_cast<uint32_t*>(&r);
  }
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

}  // namespace tc
}  // namespace pe
