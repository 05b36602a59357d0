// tc_common.cuh -- Blackwell (sm_100 family) tensor-core building blocks as
// inline PTX: TMEM allocation and access, tcgen05.mma (kind::f16, bf16 in,
// fp32 accumulate), shared-memory matrix descriptors for K-major operands in
// the 128-byte swizzled layout, and mbarrier waits that give up after a time
// limit instead of spinning forever.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace rdn {
namespace tc {

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n"
      "}\n"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// Wait for the phase with the given parity to complete.  Gives up after
// `max_cycles` SM clock cycles (about one second at 2 GHz for 2e9) and
// returns false, so a kernel can record an error and return instead of
// hanging the GPU.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity,
                                          long long max_cycles = 2000000000ll) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > max_cycles) return false;
  }
  return true;
}

// Arm `bar` for `bytes` of asynchronous copies (counts as this thread's arrival).
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// Bulk (untiled, TMA) copy global -> shared; completion is signalled on `bar`
// as transaction bytes.  Both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst_smem, const void *src_gmem, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Tiled (tensor-map) bulk copy global -> shared of a 3-D box at coordinates
// (c0, c1, c2), innermost first; completion is signalled on `bar` as
// transaction bytes.  `map` is the address of a CUtensorMap in kernel
// parameter space (a __grid_constant__ parameter).  The destination is
// 1024-byte aligned for the 128-byte swizzled layout; c0 times the element
// size is a multiple of 16 bytes.
__device__ __forceinline__ void tma_load_3d(void *dst_smem, const void *map, int c0, int c1,
                                            int c2, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst_smem)),
      "l"(map), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
      : "memory");
}

// Hints that bring global memory closer ahead of its use (no completion to
// wait for; the later loads find the lines cached): into L2, a contiguous
// range (16-byte aligned address and size) or the 128-byte line of one address.
__device__ __forceinline__ void prefetch_l2_bulk(const void *src_gmem, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src_gmem), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void prefetch_l2_line(const void *src_gmem) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(src_gmem));
}
// ... and the line of one address into this SM's L1, for loads a few
// thousand cycles later
__device__ __forceinline__ void prefetch_l1_line(const void *src_gmem) {
  asm volatile("prefetch.global.L1 [%0];" ::"l"(src_gmem));
}

// 16 consecutive floats of shared memory at a 16-byte aligned address, by
// four 16-byte loads
__device__ __forceinline__ void lds16(const float *p, float (&v)[16]) {
  const float4 *q = reinterpret_cast<const float4 *>(p);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float4 a = q[k];
    v[4 * k] = a.x;
    v[4 * k + 1] = a.y;
    v[4 * k + 2] = a.z;
    v[4 * k + 3] = a.w;
  }
}

// Two floats as bf16 hi + lo parts, each pair packed in 32 bits (a in the low
// half): hi is a's upper 16 bits (bf16 truncation, exact, no conversion), lo
// the remainder a - hi (exact in fp32) rounded to bf16; hi + lo carries about
// 16 significant bits (relative error below 2^-17).
__device__ __forceinline__ void split_pack_bf16(float a, float b, uint32_t &hi, uint32_t &lo) {
  const uint32_t ua = __float_as_uint(a), ub = __float_as_uint(b);
  hi = __byte_perm(ua, ub, 0x7632);
  const __nv_bfloat162 r = __floats2bfloat162_rn(a - __uint_as_float(ua & 0xFFFF0000u),
                                                 b - __uint_as_float(ub & 0xFFFF0000u));
  lo = *reinterpret_cast<const uint32_t *>(&r);
}

// 16-byte asynchronous copy global -> shared, zero-filled when !valid (the
// source is then not read, but must still be a valid address).  Completes at
// cp_async_wait_all() of the issuing thread; a barrier then publishes it.
__device__ __forceinline__ void cp_async16(void *dst_smem, const void *src_gmem, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst_smem)),
               "l"(src_gmem), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Bulk copy shared -> global, tracked by this thread's bulk groups: issue,
// then bulk_commit(); bulk_wait_read() returns once every committed copy has
// finished reading shared memory, bulk_wait_all() once they are complete.
// Both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_s2g(void *dst_gmem, const void *src_smem, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst_gmem),
               "r"(smem_u32(src_smem)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// ... all but the newest committed group
__device__ __forceinline__ void bulk_wait_read_all_but_last() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// ------------------------------------------------------------------ fences
__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// generic-proxy shared-memory writes -> visible to the async proxy (the MMA)
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// -------------------------------------------------------------------- TMEM
// Called by one full warp.  The allocated column base (lane 0) is written to
// *slot in shared memory.
__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// TMEM address of (lane, column): lane in the upper 16 bits.
__device__ __forceinline__ uint32_t tmem_addr(uint32_t base, uint32_t lane, uint32_t col) {
  return base + (lane << 16) + col;
}

// One warp reads 32 lanes x 16 consecutive 32-bit columns: thread i of the
// warp gets lane (lane_base + i), columns col .. col+15.  Waits for the
// load before returning.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Two such loads with one wait for both (one exposed latency instead of two).
__device__ __forceinline__ void tmem_ld16x2(uint32_t ta, float (&a)[16], uint32_t tb,
                                            float (&b)[16]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%32];\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%33];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
        "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]),
        "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
        "=r"(r[30]), "=r"(r[31])
      : "r"(ta), "r"(tb)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    a[i] = __uint_as_float(r[i]);
    b[i] = __uint_as_float(r[16 + i]);
  }
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n"
      "tcgen05.wait::st.sync.aligned;\n" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}

// --------------------------------------------------------------------- MMA
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major,
// shape M x N (M in {64, 128}; N a multiple of 16 up to 256).
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4)                          // D format: fp32
         | (1u << 7)                        // A format: bf16
         | (1u << 10)                       // B format: bf16
         | ((uint32_t)(N >> 3) << 17)       // N / 8
         | ((uint32_t)(M >> 4) << 24);      // M / 16
}

// Shared-memory descriptor of a K-major operand stored in the 128-byte
// swizzled layout: rows of 64 bf16 (128 bytes), 8-row groups 1024 bytes
// apart, tile base 1024-byte aligned.  Advancing K by 16 elements inside a
// row is +32 bytes on the start address.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1 << 16;             // leading byte offset (unused when swizzled): 16 B
  d |= (uint64_t)(1024 >> 4) << 32;   // stride byte offset: 1024 B per 8 rows
  d |= (uint64_t)1 << 46;             // descriptor version for this architecture
  d |= (uint64_t)2 << 61;             // swizzle mode: 128 B
  return d;
}

// Descriptor of an MN-major operand in the 128-byte swizzled layout: rows are
// the K index (128 bytes = 64 elements of the M or N index each), 8-row
// groups 1024 bytes apart, and consecutive 64-element M/N atoms `lbo` bytes
// apart.  Advancing K by 16 rows is +2048 bytes on the start address.
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;  // stride between M/N atoms
  d |= (uint64_t)(1024 >> 4) << 32;              // stride between 8-row K groups
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// A byte offset as an increment of a descriptor's start-address field (the
// field holds address / 16 in 14 bits; shared-memory addresses stay below
// 256 KB, so an in-range offset never carries out of it).
__device__ __forceinline__ uint64_t desc_off(uint32_t bytes) { return (uint64_t)(bytes >> 4); }

constexpr uint32_t kAMajorMN = 1u << 15, kBMajorMN = 1u << 16;

// D[tmem] (+)= A * B^T for one K = 16 slice, issued by one thread.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "setp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once every MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// D (+)= A * B^T over K = 16 * ksteps, A K-major (64-column blocks a_blk
// apart), B MN-major (K rows, N in 64-wide atoms b_lbo apart).
template <bool kRolled = false>
__device__ __forceinline__ void mma_tile_kmn(uint32_t d_tmem, uint32_t a_base, uint32_t a_blk,
                                             uint32_t b_base, uint32_t b_lbo, int ksteps,
                                             uint32_t idesc, bool accumulate_first) {
  auto step = [&](int kk) {
    const uint32_t a = a_base + (uint32_t)(kk >> 2) * a_blk + (uint32_t)(kk & 3) * 32u;
    mma_bf16(d_tmem, sdesc_sw128(a), sdesc_sw128_mn(b_base + (uint32_t)kk * 2048u, b_lbo),
             idesc | kBMajorMN, (kk > 0 || accumulate_first) ? 1u : 0u);
  };
  if constexpr (kRolled) {
    const uint64_t a0 = sdesc_sw128(a_base), b0 = sdesc_sw128_mn(b_base, b_lbo);
#pragma unroll 1
    for (int kb = 0; kb < ksteps; kb += 4) {
      const uint64_t a = a0 + desc_off((uint32_t)(kb >> 2) * a_blk);
      const uint64_t b = b0 + desc_off((uint32_t)kb * 2048u);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (kb + j < ksteps)
          mma_bf16(d_tmem, a + desc_off(32u * j), b + desc_off(2048u * j), idesc | kBMajorMN,
                   (kb + j > 0 || accumulate_first) ? 1u : 0u);
    }
  } else {
#pragma unroll
    for (int kk = 0; kk < ksteps; ++kk) step(kk);
  }
}

// D (+)= A * B^T over K = 16 * ksteps (<= 4), A MN-major (K rows, M atoms
// a_lbo apart), B K-major in one 64-column block.
template <bool kRolled = false>
__device__ __forceinline__ void mma_tile_mnk(uint32_t d_tmem, uint32_t a_base, uint32_t a_lbo,
                                             uint32_t b_base, int ksteps, uint32_t idesc,
                                             bool accumulate_first) {
  auto step = [&](int kk) {
    mma_bf16(d_tmem, sdesc_sw128_mn(a_base + (uint32_t)kk * 2048u, a_lbo),
             sdesc_sw128(b_base + (uint32_t)kk * 32u), idesc | kAMajorMN,
             (kk > 0 || accumulate_first) ? 1u : 0u);
  };
  if constexpr (kRolled) {  // ksteps <= 4: one group
    const uint64_t a0 = sdesc_sw128_mn(a_base, a_lbo), b0 = sdesc_sw128(b_base);
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < ksteps)
        mma_bf16(d_tmem, a0 + desc_off(2048u * j), b0 + desc_off(32u * j), idesc | kAMajorMN,
                 (j > 0 || accumulate_first) ? 1u : 0u);
  } else {
#pragma unroll
    for (int kk = 0; kk < ksteps; ++kk) step(kk);
  }
}

// D (+)= A * B^T over K = 16 * ksteps with both operands MN-major (K rows;
// M / N atoms a_lbo / b_lbo apart).
template <bool kRolled = false>
__device__ __forceinline__ void mma_tile_mnmn(uint32_t d_tmem, uint32_t a_base, uint32_t a_lbo,
                                              uint32_t b_base, uint32_t b_lbo, int ksteps,
                                              uint32_t idesc, bool accumulate_first) {
  auto step = [&](int kk) {
    mma_bf16(d_tmem, sdesc_sw128_mn(a_base + (uint32_t)kk * 2048u, a_lbo),
             sdesc_sw128_mn(b_base + (uint32_t)kk * 2048u, b_lbo),
             idesc | kAMajorMN | kBMajorMN, (kk > 0 || accumulate_first) ? 1u : 0u);
  };
  if constexpr (kRolled) {
    const uint64_t a0 = sdesc_sw128_mn(a_base, a_lbo), b0 = sdesc_sw128_mn(b_base, b_lbo);
#pragma unroll 1
    for (int kb = 0; kb < ksteps; kb += 4) {
      const uint64_t a = a0 + desc_off((uint32_t)kb * 2048u), b = b0 + desc_off((uint32_t)kb * 2048u);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (kb + j < ksteps)
          mma_bf16(d_tmem, a + desc_off(2048u * j), b + desc_off(2048u * j),
                   idesc | kAMajorMN | kBMajorMN, (kb + j > 0 || accumulate_first) ? 1u : 0u);
    }
  } else {
#pragma unroll
    for (int kk = 0; kk < ksteps; ++kk) step(kk);
  }
}

// Sum a per-thread vector v[64] over the 32 lanes of a warp by halving
// exchanges: afterwards lane l holds the warp sums for tokens
// t = tbase(l) and tbase(l) + 1 in out[0..1], with
// tbase(l) = 32 b4 + 16 b3 + 8 b2 + 4 b1 + 2 b0 for the bits b of l.
__device__ __forceinline__ void warp_transpose_reduce64(const float (&v)[64], float (&out)[2]) {
  const int lane = threadIdx.x & 31;
  float a[32];
  {
    const bool hi = lane & 16;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float send = hi ? v[k] : v[32 + k];
      const float keep = hi ? v[32 + k] : v[k];
      a[k] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
  }
  float b[16];
  {
    const bool hi = lane & 8;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const float send = hi ? a[k] : a[16 + k];
      const float keep = hi ? a[16 + k] : a[k];
      b[k] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
  }
  float c[8];
  {
    const bool hi = lane & 4;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float send = hi ? b[k] : b[8 + k];
      const float keep = hi ? b[8 + k] : b[k];
      c[k] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
  }
  float d[4];
  {
    const bool hi = lane & 2;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float send = hi ? c[k] : c[4 + k];
      const float keep = hi ? c[4 + k] : c[k];
      d[k] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
    }
  }
  {
    const bool hi = lane & 1;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const float send = hi ? d[k] : d[2 + k];
      const float keep = hi ? d[2 + k] : d[k];
      out[k] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
    }
  }
}
// Sum a per-thread vector v[32] over the 32 lanes of a warp by halving
// exchanges: afterwards lane l holds the warp sum of v[l].
__device__ __forceinline__ float warp_transpose_reduce32(const float (&v)[32]) {
  const int lane = threadIdx.x & 31;
  float a[16], b[8], c[4], d[2];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const bool hi = lane & 16;
    a[k] = (hi ? v[16 + k] : v[k]) + __shfl_xor_sync(0xffffffffu, hi ? v[k] : v[16 + k], 16);
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const bool hi = lane & 8;
    b[k] = (hi ? a[8 + k] : a[k]) + __shfl_xor_sync(0xffffffffu, hi ? a[k] : a[8 + k], 8);
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const bool hi = lane & 4;
    c[k] = (hi ? b[4 + k] : b[k]) + __shfl_xor_sync(0xffffffffu, hi ? b[k] : b[4 + k], 4);
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const bool hi = lane & 2;
    d[k] = (hi ? c[2 + k] : c[k]) + __shfl_xor_sync(0xffffffffu, hi ? c[k] : c[2 + k], 2);
  }
  const bool hi = lane & 1;
  return (hi ? d[1] : d[0]) + __shfl_xor_sync(0xffffffffu, hi ? d[0] : d[1], 1);
}

// The same for v[16]: afterwards lanes 2 i and 2 i + 1 hold the warp sum of v[i].
__device__ __forceinline__ float warp_transpose_reduce16(const float (&v)[16]) {
  const int lane = threadIdx.x & 31;
  float a[8], b[4], c[2];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const bool hi = lane & 16;
    a[k] = (hi ? v[8 + k] : v[k]) + __shfl_xor_sync(0xffffffffu, hi ? v[k] : v[8 + k], 16);
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const bool hi = lane & 8;
    b[k] = (hi ? a[4 + k] : a[k]) + __shfl_xor_sync(0xffffffffu, hi ? a[k] : a[4 + k], 8);
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const bool hi = lane & 4;
    c[k] = (hi ? b[2 + k] : b[k]) + __shfl_xor_sync(0xffffffffu, hi ? b[k] : b[2 + k], 4);
  }
  const bool hi = lane & 2;
  const float d = (hi ? c[1] : c[0]) + __shfl_xor_sync(0xffffffffu, hi ? c[0] : c[1], 2);
  return d + __shfl_xor_sync(0xffffffffu, d, 1);
}

__device__ __forceinline__ int transpose_reduce_tbase(int lane) {
  return ((lane >> 4) & 1) * 32 + ((lane >> 3) & 1) * 16 + ((lane >> 2) & 1) * 8 +
         ((lane >> 1) & 1) * 4 + (lane & 1) * 2;
}

// Byte offset of element (r, c), c in [0, 64), in a K-major 128B-swizzled tile
// whose rows are 64 bf16 wide: the 16-byte chunk index is XORed with r mod 8.
__device__ __forceinline__ uint32_t sw128(int r, int c) {
  return (uint32_t)(r * 128 + ((((c >> 3) ^ (r & 7)) & 7) << 4) + (c & 7) * 2);
}

// (kRolled: a loop over groups of 4 K-steps per call site instead of an
// unrolled sequence -- for kernels whose straight-line code would not stay in
// the instruction cache.  The descriptors are built once and advanced by
// adding to their address field, so that the issuing thread keeps up with the
// tensor pipe: rebuilding both per step costs about 90 cycles an MMA.)
// Issue D = A * B^T over K = 16 * ksteps for K-major SW128 tiles A [M][K] and
// B [N][K] stored as consecutive 64-column blocks (a_blk / b_blk bytes apart).
template <bool kRolled = false>
__device__ __forceinline__ void mma_tile(uint32_t d_tmem, uint32_t a_base, uint32_t a_blk,
                                         uint32_t b_base, uint32_t b_blk, int ksteps,
                                         uint32_t idesc, bool accumulate_first) {
  auto step = [&](int kk) {
    const uint32_t off = (uint32_t)(kk & 3) * 32u;
    const uint32_t a = a_base + (uint32_t)(kk >> 2) * a_blk + off;
    const uint32_t b = b_base + (uint32_t)(kk >> 2) * b_blk + off;
    mma_bf16(d_tmem, sdesc_sw128(a), sdesc_sw128(b), idesc,
             (kk > 0 || accumulate_first) ? 1u : 0u);
  };
  if constexpr (kRolled) {
    const uint64_t a0 = sdesc_sw128(a_base), b0 = sdesc_sw128(b_base);
#pragma unroll 1
    for (int kb = 0; kb < ksteps; kb += 4) {
      const uint64_t a = a0 + desc_off((uint32_t)(kb >> 2) * a_blk);
      const uint64_t b = b0 + desc_off((uint32_t)(kb >> 2) * b_blk);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (kb + j < ksteps)
          mma_bf16(d_tmem, a + desc_off(32u * j), b + desc_off(32u * j), idesc,
                   (kb + j > 0 || accumulate_first) ? 1u : 0u);
    }
  } else {
#pragma unroll
    for (int kk = 0; kk < ksteps; ++kk) step(kk);
  }
}

}  // namespace tc

// Host: a tensor map over a token-major bf16 tensor [rows][H][D] (q, k, v, dO:
// rows = B*T tokens) whose box is 64 tokens x 1 head x 64 columns, landing in
// shared memory as a K-major 128-byte swizzled tile of 64 rows (8 KB): the
// layout the tensor-core kernels' operand tiles use.  Out-of-range rows read
// as zero.  Returns false if the driver's encoder is unavailable or refuses.
bool make_tile_map(void *map128, const void *base, int D, int H, long long rows);
}  // namespace rdn
