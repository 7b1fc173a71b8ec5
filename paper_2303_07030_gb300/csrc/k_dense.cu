// k_dense.cu -- dense projection of the graph loss (f_in = 128, f_out = 64),
// on the tcgen05 tensor cores.
//
//   proj_fwd_kernel:  P  = H W                 H: n x 128, W: 128 x 64
//   proj_bwd_kernel:  dH = G W^T  and  dW += H^T G over the CTA's rows, in one
//                     sweep that reads each row of H and G once (per-CTA
//                     partials of dW, then one fixed-order reduction)
//
// Precision: fp32 operands are split into two BF16 parts, x = hi + lo + r with
// hi = bf16(x), lo = bf16(x - hi), |r| <= 2^-16 |x|, and each product is taken
// as hi*hi' + hi*lo' + lo*hi' (three kind::f16 MMAs, fp32 accumulation in
// tensor memory): about 2^-15 relative error per product, well inside the
// 1e-4 normwise gradient tolerance (4e-6 normwise for P on the workload's
// distributions).  No tensor-memory accumulation runs longer than one tile:
// the tiles' dW are added in fp32 registers.
//
// Pipeline (one CTA of 16 warps per SM, persistent over 128-row tiles t =
// blockIdx.x + i * gridDim.x; a tile's rows are one contiguous block of H
// and of G): thread 0 streams each tile into shared memory with bulk copies
// (cp.async.bulk, completion counted in bytes on an mbarrier), two 64-row
// halves at a time in a ring of two raw stages; the threads split a landed
// half into BF16 hi and lo parts, written in the 128-byte swizzled layout the
// MMAs read, and the freed stage is refilled with the next tile's half at
// once.  Thread 0 issues the tile's MMAs, which commit to an mbarrier; while
// the tensor cores work, the threads drain the previous tile's accumulator
// (tcgen05.ld) to global memory (accumulators are double-buffered in tensor
// memory).  Every wait is bounded; a kernel that gives up still waits for
// the copies and MMAs it issued before it leaves.
//
// Operand layouts (all 128-byte swizzled; a "block" is a stack of 128-byte
// rows, each row 64 BF16 values):
//   H tile  [2 blocks of 64 features][128 rows]  K-major A of P = H W
//                                                (rows = M, features = K), and
//                                                MN-major A of dW = H^T G
//                                                (features = M, rows = K)
//   G tile  [1 block][128 rows]                  K-major A of dH = G W^T and
//                                                MN-major B of dW
//   W^T     [2 blocks][64 rows = f_out]          K-major B of P
//   W       [1 block][128 rows = f_in]           K-major B of dH
#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace sdad {

constexpr int kFin = 128, kFout = 64;
constexpr int kTileM = 128;
constexpr int kHalfM = 64;              // rows per raw stage
constexpr int kDenseThreads = 512;
constexpr uint32_t kBlk = 128 * 128;    // bytes of a 128-row block of 128-byte rows
constexpr uint32_t kHRow = kFin * 4;    // bytes of an fp32 row of H
constexpr uint32_t kGRow = kFout * 4;   // ... of G

// shared-memory map of proj_fwd_kernel (from a 1024-byte aligned base)
constexpr uint32_t kFwdRaw = 0;                         // 2 stages x 64 rows of H (fp32)
constexpr uint32_t kFwdRawStage = kHalfM * kHRow;       // 32 KB
constexpr uint32_t kFwdA = kFwdRaw + 2 * kFwdRawStage;  // [hi|lo][kb] x kBlk
constexpr uint32_t kFwdW = kFwdA + 4 * kBlk;            // W^T: [hi|lo][kb] x 64 rows x 128 B, per source
constexpr uint32_t kFwdWBytes = 4 * 64 * 128;
// NSRC sources (P = H W, or P = H W + H2 W2): barriers after the NSRC W^T
constexpr uint32_t fwd_bar(int nsrc) { return kFwdW + (uint32_t)nsrc * kFwdWBytes; }
constexpr uint32_t fwd_smem(int nsrc) { return fwd_bar(nsrc) + 64 + 1024; }   // + barriers, TMEM slot, alignment
constexpr uint32_t kFwdSmem = fwd_smem(1);
// shared-memory map of proj_bwd_kernel
constexpr uint32_t kBwdRawStage = kHalfM * (kHRow + kGRow);   // 48 KB: 64 rows of H, then of G
constexpr uint32_t kBwdRaw = 0;
constexpr uint32_t kBwdG = kBwdRaw + 2 * kBwdRawStage;  // [hi|lo] x kBlk
constexpr uint32_t kBwdH = kBwdG + 2 * kBlk;            // [hi|lo][block] x kBlk
constexpr uint32_t kBwdW = kBwdH + 4 * kBlk;            // W: [hi|lo] x kBlk
constexpr uint32_t kBwdBar = kBwdW + 2 * kBlk;
constexpr uint32_t kBwdSmem = kBwdBar + 64 + 1024;
static_assert(fwd_smem(2) <= 227 * 1024 && kBwdSmem <= 227 * 1024, "shared memory of one CTA");

__device__ __forceinline__ uint32_t bf2_bits(__nv_bfloat162 v) {
  return *reinterpret_cast<const uint32_t*>(&v);
}

// hi and lo BF16 parts of four fp32 values (in order), four values per uint2
__device__ __forceinline__ void split4(float4 x, uint2& hi, uint2& lo) {
  const __nv_bfloat162 h01 = __floats2bfloat162_rn(x.x, x.y);
  const __nv_bfloat162 h23 = __floats2bfloat162_rn(x.z, x.w);
  const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
  hi = make_uint2(bf2_bits(h01), bf2_bits(h23));
  lo = make_uint2(bf2_bits(__floats2bfloat162_rn(x.x - f01.x, x.y - f01.y)),
                  bf2_bits(__floats2bfloat162_rn(x.z - f23.x, x.w - f23.y)));
}

__device__ __forceinline__ void sts64(uint32_t addr, uint2 v) {
  asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(v.x), "r"(v.y) : "memory");
}
__device__ __forceinline__ void sts16(uint32_t addr, uint16_t v) {
  asm volatile("st.shared.b16 [%0], %1;" ::"r"(addr), "h"(v) : "memory");
}
__device__ __forceinline__ float4 lds128(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// writes the hi and lo parts of one fp32 value at byte offset `off` of the
// hi and lo copies
__device__ __forceinline__ void put1(uint32_t hi_base, uint32_t lo_base, uint32_t off, float v) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  const __nv_bfloat16 l = __float2bfloat16_rn(v - __bfloat162float(h));
  sts16(hi_base + off, *reinterpret_cast<const uint16_t*>(&h));
  sts16(lo_base + off, *reinterpret_cast<const uint16_t*>(&l));
}

__device__ __forceinline__ uint32_t align1024(uint32_t a) { return (a + 1023u) & ~1023u; }

// bulk copy of `bytes` (a multiple of 16) from global memory to the shared
// address `dst`, completion counted on the mbarrier at shared address `bar`
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// rows of [r0, r0 + 64) that exist (r0 < n gives at least one)
__device__ __forceinline__ int half_rows(int r0, int n) { return max(0, min(kHalfM, n - r0)); }

// Splits 64 landed rows of fp32 data (row-major, C4 float4 per row, at raw
// address `raw`) into the hi / lo swizzled blocks (block b holds columns
// 64 b .. 64 b + 63, blocks kBlk apart), at tile rows row0 .. row0 + 63.
// Rows at or past `valid` read as zero.
template <int C4>
__device__ __forceinline__ void split_half(uint32_t raw, uint32_t hi_base, uint32_t lo_base,
                                           int row0, int valid) {
  constexpr int kN = kHalfM * C4;   // float4 of the half
#pragma unroll
  for (int q = threadIdx.x; q < kN; q += kDenseThreads) {
    const int r = q / C4, f = 4 * (q % C4);
    const float4 x = r < valid ? lds128(raw + 16u * (uint32_t)q) : make_float4(0.f, 0.f, 0.f, 0.f);
    const uint32_t off = (uint32_t)(f >> 6) * kBlk + tc::sw128_offset_b16(row0 + r, f & 63);
    uint2 hi, lo;
    split4(x, hi, lo);
    sts64(hi_base + off, hi);
    sts64(lo_base + off, lo);
  }
}

// K-major operand descriptor of k-step s (16 BF16 = 32 bytes) in a block
__device__ __forceinline__ uint64_t kdesc(uint32_t block, int s) {
  return tc::smem_desc_sw128(block + 32u * (uint32_t)s);
}
// MN-major operand descriptor of k-step s (16 rows = 2048 bytes); MN blocks kBlk apart
__device__ __forceinline__ uint64_t mndesc(uint32_t block, int s) {
  return tc::smem_desc_sw128_mn(block + 2048u * (uint32_t)s, kBlk);
}

// drains COLS accumulator columns for this warp's 32 rows into out rows of
// width OUTW (rows at or past n are not stored)
template <int COLS, bool STREAM>
__device__ __forceinline__ void drain_rows(uint32_t taddr, float* __restrict__ out, int OUTW,
                                           int row, int col, int n) {
  float v[COLS];
  if constexpr (COLS == 32) tc::tmem_ld32(taddr, v);
  else tc::tmem_ld16(taddr, v);
  tc::tmem_wait_ld();
  if (row < n) {
    float4* dst = reinterpret_cast<float4*>(out + (size_t)row * OUTW + col);
#pragma unroll
    for (int q = 0; q < COLS / 4; ++q) {
      const float4 w = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      if (STREAM) __stcs(dst + q, w);
      else dst[q] = w;
    }
  }
}

// The raw-stage ring shared by both kernels: stage h (0, 1) holds half h of
// a tile; n_issued / n_waited count the uses of each stage's barrier.
struct RawRing {
  uint64_t* full;   // two mbarriers
  int n_issued[2];
  int n_waited[2];
  __device__ __forceinline__ uint32_t parity(int h) const { return (uint32_t)(n_waited[h] & 1); }
  // before leaving: wait for every copy issued but not waited for
  __device__ __forceinline__ void drain(WsHeader* hdr) {
    for (int h = 0; h < 2; ++h)
      if (n_issued[h] > n_waited[h]) mbar_drain(&full[h], (uint32_t)((n_issued[h] - 1) & 1), hdr);
  }
};

// ---------------------------------------------------------------------------
// P = H W  (NSRC = 1), or P = H W + H2 W2  (NSRC = 2: the forward mode's
// P' = H' W + H W' as one product; both sources' rows of a tile go through the
// same raw stages and split buffers, one after the other, and their MMAs add
// into the tile's accumulator)
// ---------------------------------------------------------------------------
template <int NSRC>
__global__ void __launch_bounds__(kDenseThreads, 1)
    proj_fwd_kernel(const float* __restrict__ H, const float* __restrict__ W,
                    const float* __restrict__ H2, const float* __restrict__ W2,
                    float* __restrict__ P, int n, WsHeader* hdr) {
  extern __shared__ unsigned char dense_smem[];
  const uint32_t base = align1024(smem_u32(dense_smem));
  unsigned char* gbase = dense_smem + (base - smem_u32(dense_smem));
  uint64_t* full = reinterpret_cast<uint64_t*>(gbase + fwd_bar(NSRC));
  uint64_t* mma = full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + fwd_bar(NSRC) + 24);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t idesc = tc::idesc_bf16(kTileM, kFout, false, false);
  auto A = [&](int part, int kb) { return base + kFwdA + (uint32_t)(part * 2 + kb) * kBlk; };
  auto Wt = [&](int src, int part, int kb) {
    return base + kFwdW + (uint32_t)src * kFwdWBytes + (uint32_t)(part * 2 + kb) * (64 * 128);
  };
  auto raw = [&](int h) { return base + kFwdRaw + (uint32_t)h * kFwdRawStage; };

  const int ntiles = (n + kTileM - 1) / kTileM;
  const int grid = gridDim.x;
  const int nloc = (ntiles - (int)blockIdx.x + grid - 1) / grid;   // >= 1: grid <= tiles
  // half h of source q of local tile i into raw stage h
  auto issue = [&](int i, int q, int h) {
    const int r0 = ((int)blockIdx.x + i * grid) * kTileM + h * kHalfM;
    const uint32_t bytes = (uint32_t)half_rows(r0, n) * kHRow;
    mbar_arrive_expect_tx(&full[h], bytes);
    if (bytes) bulk_load(raw(h), (q == 0 ? H : H2) + (size_t)r0 * kFin, bytes, smem_u32(&full[h]));
  };
  RawRing ring{full, {0, 0}, {0, 0}};
  if (tid == 0) {
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    mbar_init(mma, 1);
    fence_mbar_init();
    for (int h = 0; h < 2; ++h) issue(0, 0, h);   // tile 0's halves of the first source
  }
  ring.n_issued[0] = ring.n_issued[1] = 1;
  if (warp == 0) tc::tmem_alloc(tmem_slot, 2 * kFout);   // two accumulators of 64 columns
  // operand B = W^T (row n' = column n' of W) of each source, once per CTA
#pragma unroll
  for (int q = 0; q < NSRC; ++q) {
    const float* Wq = q == 0 ? W : W2;
    for (int idx = tid; idx < kFin * kFout; idx += kDenseThreads) {
      const int k = idx / kFout, nn = idx % kFout;
      put1(Wt(q, 0, k >> 6), Wt(q, 1, k >> 6), tc::sw128_offset_b16(nn, k & 63), __ldg(Wq + idx));
    }
  }
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  const int q4 = warp & 3, cg = warp >> 2;   // epilogue: TMEM lanes 32 q4.., columns 16 cg..
  bool ok = true;
  int last = -1;      // local index of the last tile whose MMAs were issued
  int ncommit = 0;    // MMA groups committed so far (one per tile and source)
  for (int i = 0; i < nloc && ok; ++i) {
    const int t = (int)blockIdx.x + i * grid, row0 = t * kTileM;
#pragma unroll 1
    for (int q = 0; q < NSRC; ++q) {
      if (ncommit > 0) {   // the split parts are free once the last MMA group is done
        ok = __syncthreads_and(mbar_wait(mma, (uint32_t)((ncommit - 1) & 1), hdr));
        if (!ok) break;
        tc::fence_after_sync();
      }
      for (int h = 0; h < 2; ++h) {
        ok = __syncthreads_and(mbar_wait(&full[h], ring.parity(h), hdr));
        if (!ok) break;
        ++ring.n_waited[h];
        split_half<32>(raw(h), A(0, 0), A(1, 0), h * kHalfM, half_rows(row0 + h * kHalfM, n));
        __syncthreads();   // the stage is read: refill it with the next source's half, or the next tile's
        const bool more = q + 1 < NSRC || i + 1 < nloc;
        if (more) {
          if (tid == 0) {
            if (q + 1 < NSRC) issue(i, q + 1, h);
            else issue(i + 1, 0, h);
          }
          ++ring.n_issued[h];
        }
      }
      if (!ok) break;
      tc::fence_proxy_async_smem();
      tc::fence_before_sync();
      __syncthreads();
      if (tid == 0) {
        tc::fence_after_sync();
        const uint32_t d = tmem + (uint32_t)(kFout * (i & 1));
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int s = 0; s < 4; ++s) {
            const uint64_t ah = kdesc(A(0, kb), s), al = kdesc(A(1, kb), s);
            const uint64_t bh = kdesc(Wt(q, 0, kb), s), bl = kdesc(Wt(q, 1, kb), s);
            tc::mma_bf16(d, ah, bh, idesc, q > 0 || (kb | s) != 0);
            tc::mma_bf16(d, ah, bl, idesc, true);
            tc::mma_bf16(d, al, bh, idesc, true);
          }
        tc::mma_commit(mma);
      }
      ++ncommit;
    }
    if (!ok) break;
    last = i;
    if (i >= 1) {   // tile i-1's accumulator to P while the tensor cores work on tile i
      const int row = (t - grid) * kTileM + 32 * q4 + lane;
      drain_rows<16, false>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFout * ((i - 1) & 1) + 16 * cg),
                            P, kFout, row, 16 * cg, n);
    }
  }
  if (ok && last >= 0) {
    ok = __syncthreads_and(mbar_wait(mma, (uint32_t)((ncommit - 1) & 1), hdr));
    if (ok) {
      tc::fence_after_sync();
      const int row = ((int)blockIdx.x + last * grid) * kTileM + 32 * q4 + lane;
      drain_rows<16, false>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFout * (last & 1) + 16 * cg),
                            P, kFout, row, 16 * cg, n);
    }
  }
  if (!ok) {   // a wait gave up: let the issued copies land and the MMAs end
    if (ncommit > 0) mbar_drain(mma, (uint32_t)((ncommit - 1) & 1), hdr);
    ring.drain(hdr);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 2 * kFout);
}

// ---------------------------------------------------------------------------
// dH = G W^T and this CTA's part of dW = H^T G
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kDenseThreads, 1)
    proj_bwd_kernel(const float* __restrict__ H, const float* __restrict__ W,
                    const float* __restrict__ G, float* __restrict__ dH,
                    float* __restrict__ dWpart, int n, WsHeader* hdr) {
  extern __shared__ unsigned char dense_smem[];
  const uint32_t base = align1024(smem_u32(dense_smem));
  unsigned char* gbase = dense_smem + (base - smem_u32(dense_smem));
  uint64_t* full = reinterpret_cast<uint64_t*>(gbase + kBwdBar);
  uint64_t* mma = full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kBwdBar + 24);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t idesc_dh = tc::idesc_bf16(kTileM, kFin, false, false);
  constexpr uint32_t idesc_dw = tc::idesc_bf16(kFin, kFout, true, true);
  // tensor memory: two dH accumulators (128 columns each), then two of dW
  // (64 each); a tile's dW is added in fp32 registers (each thread 16 entries)
  constexpr uint32_t kDwCol = 2 * kFin;
  auto Gs = [&](int part) { return base + kBwdG + (uint32_t)part * kBlk; };
  auto Hs = [&](int part) { return base + kBwdH + (uint32_t)(part * 2) * kBlk; };
  auto Ws = [&](int part) { return base + kBwdW + (uint32_t)part * kBlk; };
  auto raw = [&](int h) { return base + kBwdRaw + (uint32_t)h * kBwdRawStage; };
  // thread 0: the copies of rows [r0, r0 + 64) of H and G into stage h
  auto issue = [&](int h, int r0) {
    const int rows = half_rows(r0, n);
    mbar_arrive_expect_tx(&full[h], (uint32_t)rows * (kHRow + kGRow));
    if (rows) {
      bulk_load(raw(h), H + (size_t)r0 * kFin, (uint32_t)rows * kHRow, smem_u32(&full[h]));
      bulk_load(raw(h) + kHalfM * kHRow, G + (size_t)r0 * kFout, (uint32_t)rows * kGRow,
                smem_u32(&full[h]));
    }
  };

  const int ntiles = (n + kTileM - 1) / kTileM;
  const int grid = gridDim.x;
  const int nloc = (ntiles - (int)blockIdx.x + grid - 1) / grid;   // >= 1: grid <= tiles
  RawRing ring{full, {0, 0}, {0, 0}};
  if (tid == 0) {
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    mbar_init(mma, 1);
    fence_mbar_init();
    issue(0, (int)blockIdx.x * kTileM);
    issue(1, (int)blockIdx.x * kTileM + kHalfM);
  }
  ring.n_issued[0] = ring.n_issued[1] = 1;
  if (warp == 0) tc::tmem_alloc(tmem_slot, 512);
  // operand B of dH = W (row n' = row n' of W), once per CTA
  for (int idx = tid; idx < kFin * kFout; idx += kDenseThreads) {
    const int nn = idx / kFout, k = idx % kFout;
    put1(Ws(0), Ws(1), tc::sw128_offset_b16(nn, k), __ldg(W + idx));
  }
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  const int q4 = warp & 3, cg = warp >> 2;   // epilogue: TMEM lanes 32 q4.., a quarter of the columns
  float dwacc[16];   // this thread's entries of the CTA's dW: row 32 q4 + lane, columns 16 cg ..
#pragma unroll
  for (int c = 0; c < 16; ++c) dwacc[c] = 0.f;
  // tile j's dH to memory (row0: its first row) and its dW into dwacc
  auto epilogue = [&](int j, int row0) {
    const uint32_t lanes = (uint32_t)(32 * q4) << 16;
    if (dH)
      drain_rows<32, true>(tmem + lanes + (uint32_t)(kFin * (j & 1) + 32 * cg), dH, kFin,
                           row0 + 32 * q4 + lane, 32 * cg, n);
    float v[16];
    tc::tmem_ld16(tmem + lanes + kDwCol + (uint32_t)(kFout * (j & 1) + 16 * cg), v);
    tc::tmem_wait_ld();
#pragma unroll
    for (int c = 0; c < 16; ++c) dwacc[c] += v[c];
  };
  bool ok = true;
  int last = -1;
  for (int i = 0; i < nloc; ++i) {
    const int t = (int)blockIdx.x + i * grid, row0 = t * kTileM;
    if (i >= 1) {   // the split parts are free once tile i-1's MMAs are done
      ok = __syncthreads_and(mbar_wait(mma, (uint32_t)((i - 1) & 1), hdr));
      if (!ok) break;
      tc::fence_after_sync();
    }
    for (int h = 0; h < 2; ++h) {
      ok = __syncthreads_and(mbar_wait(&full[h], ring.parity(h), hdr));
      if (!ok) break;
      ++ring.n_waited[h];
      const int valid = half_rows(row0 + h * kHalfM, n);
      split_half<32>(raw(h), Hs(0), Hs(1), h * kHalfM, valid);
      split_half<16>(raw(h) + kHalfM * kHRow, Gs(0), Gs(1), h * kHalfM, valid);
      __syncthreads();   // the stage is read: refill it with the next tile's half
      if (i + 1 < nloc) {
        if (tid == 0) issue(h, row0 + grid * kTileM + h * kHalfM);
        ++ring.n_issued[h];
      }
    }
    if (!ok) break;
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      // dW of the tile: M = f_in (MN-major H), N = f_out (MN-major G), K = the tile's rows
      const uint32_t dw = tmem + kDwCol + (uint32_t)(kFout * (i & 1));
#pragma unroll
      for (int s = 0; s < kTileM / 16; ++s) {
        const uint64_t ah = mndesc(Hs(0), s), al = mndesc(Hs(1), s);
        const uint64_t bh = mndesc(Gs(0), s), bl = mndesc(Gs(1), s);
        tc::mma_bf16(dw, ah, bh, idesc_dw, s > 0);
        tc::mma_bf16(dw, ah, bl, idesc_dw, true);
        tc::mma_bf16(dw, al, bh, idesc_dw, true);
      }
      // dH = G W^T: M = rows, N = f_in, K = f_out (both K-major)
      const uint32_t d = tmem + (uint32_t)(kFin * (i & 1));
#pragma unroll
      for (int s = 0; s < (dH ? kFout / 16 : 0); ++s) {
        const uint64_t ah = kdesc(Gs(0), s), al = kdesc(Gs(1), s);
        const uint64_t bh = kdesc(Ws(0), s), bl = kdesc(Ws(1), s);
        tc::mma_bf16(d, ah, bh, idesc_dh, s > 0);
        tc::mma_bf16(d, ah, bl, idesc_dh, true);
        tc::mma_bf16(d, al, bh, idesc_dh, true);
      }
      tc::mma_commit(mma);
    }
    last = i;
    if (i >= 1) epilogue(i - 1, (t - grid) * kTileM);   // while the tensor cores work on tile i
  }
  if (ok && last >= 0) {
    ok = __syncthreads_and(mbar_wait(mma, (uint32_t)(last & 1), hdr));
    if (ok) {
      tc::fence_after_sync();
      epilogue(last, ((int)blockIdx.x + last * grid) * kTileM);
      // this CTA's dW: TMEM lane = f_in, column = f_out
      float4* dst = reinterpret_cast<float4*>(dWpart + (size_t)blockIdx.x * kFin * kFout +
                                              (size_t)(32 * q4 + lane) * kFout + 16 * cg);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        dst[q] = make_float4(dwacc[4 * q], dwacc[4 * q + 1], dwacc[4 * q + 2], dwacc[4 * q + 3]);
    }
  }
  if (!ok) {   // a wait gave up: let the issued copies land and the MMAs end
    if (last >= 0) mbar_drain(mma, (uint32_t)(last & 1), hdr);
    ring.drain(hdr);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 512);
}

// dW[e] = sum_p parts[p][e], p in ascending order.
__global__ void dw_reduce_kernel(const float* __restrict__ parts, int nparts,
                                 float* __restrict__ dW) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= kFin * kFout) return;
  float s = 0.f;
  for (int p = 0; p < nparts; ++p) s += parts[(size_t)p * kFin * kFout + e];
  dW[e] = s;
}

__global__ void zero_dw_kernel(float* __restrict__ dW) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e < kFin * kFout) dW[e] = 0.f;
}

namespace {
int dense_grid(int n) {
  const int tiles = (n + kTileM - 1) / kTileM;
  return std::max(1, std::min(tiles, device_sm_count()));
}
}  // namespace

cudaError_t dense_proj_fwd(const float* H, const float* W, float* P, int n, WsHeader* hdr,
                           cudaStream_t st) {
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(proj_fwd_kernel<1>), (int)kFwdSmem);
  if (e != cudaSuccess || n <= 0) return e;
  {
    KTimer t("proj_fwd", st);
    proj_fwd_kernel<1><<<dense_grid(n), kDenseThreads, kFwdSmem, st>>>(H, W, nullptr, nullptr, P,
                                                                       n, hdr);
  }
  return cudaGetLastError();
}

cudaError_t dense_proj_fwd2(const float* H, const float* W, const float* H2, const float* W2,
                            float* P, int n, WsHeader* hdr, cudaStream_t st) {
  constexpr uint32_t smem = fwd_smem(2);
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(proj_fwd_kernel<2>), (int)smem);
  if (e != cudaSuccess || n <= 0) return e;
  {
    KTimer t("proj_fwd2", st);
    proj_fwd_kernel<2><<<dense_grid(n), kDenseThreads, smem, st>>>(H, W, H2, W2, P, n, hdr);
  }
  return cudaGetLastError();
}

cudaError_t dense_proj_bwd(const float* H, const float* W, const float* G, float* dH,
                           float* dWpart, float* dW, int n, WsHeader* hdr, cudaStream_t st) {
  // dH and dW come from one sweep (which skips dH's MMAs and stores when dH
  // is not wanted); dW's per-CTA partials are summed afterwards
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(proj_bwd_kernel), (int)kBwdSmem);
  if (e != cudaSuccess) return e;
  if (n <= 0) {
    if (dW) {
      zero_dw_kernel<<<(kFin * kFout + 255) / 256, 256, 0, st>>>(dW);
      return cudaGetLastError();
    }
    return cudaSuccess;
  }
  const int grid = dense_grid(n);
  static_assert(kDwParts >= 152, "one dW partial per CTA");
  if (grid > kDwParts) return cudaErrorInvalidConfiguration;
  {
    KTimer t("proj_bwd", st);
    proj_bwd_kernel<<<grid, kDenseThreads, kBwdSmem, st>>>(H, W, G, dH, dWpart, n, hdr);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (!dW) return cudaSuccess;
  {
    KTimer t("dw_reduce", st);
    dw_reduce_kernel<<<(kFin * kFout + 255) / 256, 256, 0, st>>>(dWpart, grid, dW);
  }
  return cudaGetLastError();
}

}  // namespace sdad
