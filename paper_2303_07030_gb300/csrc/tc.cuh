// tc.cuh -- tcgen05 (5th-generation tensor core) and TMA helpers, sm_103a.
//
// Inline PTX wrappers for: tensor-memory allocation, the single-thread MMA
// issue of kind::tf32, MMA completion on an mbarrier, tensor-memory loads for
// the epilogue, 2D tiled TMA loads, and the shared-memory / instruction
// descriptors of K-major operands in the 128-byte swizzled layout.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace sdad {
namespace tc {

// ---------------------------------------------------------------------------
// descriptors
// ---------------------------------------------------------------------------
// Instruction descriptor of tcgen05.mma.kind::tf32: fp32 accumulator, A and B
// TF32, both K-major, shape M x N (M in {64, 128}, N a multiple of 8/16).
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4)                       // D format: f32
         | (2u << 7)                     // A format: tf32
         | (2u << 10)                    // B format: tf32
         | (0u << 15) | (0u << 16)       // A, B K-major
         | ((uint32_t)(N >> 3) << 17)    // N / 8
         | ((uint32_t)(M >> 4) << 24);   // M / 16
}

// Instruction descriptor of tcgen05.mma.kind::f16 with BF16 A and B and an
// fp32 accumulator, shape M x N; a_mn / b_mn: the operand is MN-major (its
// M or N index runs along the 128-byte rows of the swizzled layout) instead
// of K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
  return (1u << 4)                       // D format: f32
         | (1u << 7)                     // A format: bf16
         | (1u << 10)                    // B format: bf16
         | ((a_mn ? 1u : 0u) << 15)      // A major-ness
         | ((b_mn ? 1u : 0u) << 16)      // B major-ness
         | ((uint32_t)(N >> 3) << 17)    // N / 8
         | ((uint32_t)(M >> 4) << 24);   // M / 16
}

// Shared-memory descriptor of an MN-major operand in the 128-byte swizzled
// canonical layout: each block of 128 bytes along M/N (64 bf16) is a stack
// of rows 128 bytes apart, one row per K index, swizzled in 8-row atoms
// (1024 bytes); consecutive M/N blocks are `mn_stride` bytes apart (leading
// byte offset), consecutive 8-row groups along K 1024 bytes apart (stride
// byte offset).  `addr` is the shared address of the K-step's first row.
__device__ __forceinline__ uint64_t smem_desc_sw128_mn(uint32_t addr, uint32_t mn_stride) {
  const uint64_t start = (addr >> 4) & 0x3FFFu;
  const uint64_t lbo = (mn_stride >> 4) & 0x3FFFu;
  const uint64_t sbo = 1024 >> 4;
  return start | (lbo << 16) | (sbo << 32) | (1ull << 46) /* version */ |
         (2ull << 61) /* SWIZZLE_128B */;
}

// Byte offset of 2-byte element (row, c) inside one 128-byte-wide block of
// the swizzled layout (c in 0..63): rows 128 bytes apart, 16-byte chunks
// XOR-ed with the row index within its 8-row atom.
__device__ __forceinline__ uint32_t sw128_offset_b16(int row, int c) {
  const uint32_t chunk = (uint32_t)(c >> 3) ^ (uint32_t)(row & 7);
  return (uint32_t)row * 128u + chunk * 16u + (uint32_t)(c & 7) * 2u;
}

// Shared-memory descriptor of a K-major operand stored in the 128-byte
// swizzled canonical layout: 8-row atoms of 8 x 128 bytes (1024-byte
// aligned), consecutive atoms along M/N 1024 bytes apart.  `addr` is the
// shared address of the first row of the k-slice to read (the atom base plus
// the byte offset of the slice within the 128-byte row).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
  const uint64_t start = (addr >> 4) & 0x3FFFu;
  const uint64_t lbo = 1;                        // unused for swizzled K-major
  const uint64_t sbo = 1024 >> 4;                // 8-row atom stride
  return start | (lbo << 16) | (sbo << 32) | (1ull << 46) /* version */ |
         (2ull << 61) /* SWIZZLE_128B */;
}

// Byte offset of element (row, k) (4-byte elements) inside one 128-byte-wide
// k-block of a K-major swizzled tile: rows 128 bytes apart, 16-byte chunks
// XOR-ed with the row index within its 8-row atom.
__device__ __forceinline__ uint32_t sw128_offset(int row, int k) {
  const uint32_t chunk = (uint32_t)(k >> 2) ^ (uint32_t)(row & 7);
  return (uint32_t)row * 128u + chunk * 16u + (uint32_t)(k & 3) * 4u;
}

// ---------------------------------------------------------------------------
// tensor memory
// ---------------------------------------------------------------------------
// Allocates `ncols` (power of two >= 32) columns; one full warp calls it.
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D (tmem) (+)= A (smem desc) * B (smem desc), issued by one thread.
__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, bool accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"((uint32_t)accumulate)
      : "memory");
}

// D (tmem) (+)= A * B with BF16 operands (kind::f16), issued by one thread.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, bool accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"((uint32_t)accumulate)
      : "memory");
}

// Arrives on `bar` once all MMAs issued so far by this thread have completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 consecutive 32-bit columns of this warp's 32 TMEM lanes (lane i of the
// warp gets TMEM lane base+i).  Wait with tmem_wait_ld() before use.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 consecutive 32-bit columns of this warp's 32 TMEM lanes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ---------------------------------------------------------------------------
// TMA
// ---------------------------------------------------------------------------
// 2D tiled load of box (x, y) of `map` into shared memory; completion counted
// on `bar` in bytes.  x is the innermost coordinate (a multiple of 4 fp32
// elements: 16-byte aligned).
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// TF32 split of an fp32 value: hi keeps the sign, exponent and the 10
// leading mantissa bits (exactly representable in tf32), lo = x - hi (exact
// in fp32).  hi + lo == x.
__device__ __forceinline__ float tf32_hi(float x) {
  return __uint_as_float(__float_as_uint(x) & 0xFFFFE000u);
}

}  // namespace tc
}  // namespace sdad
