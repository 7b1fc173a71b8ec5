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
// distributions).  BF16 parts take half the shared memory of TF32 parts, so a
// CTA holds two tiles and W, and the MMAs issue at the BF16 rate.
//
// Pipeline (one CTA of 16 warps per SM, 128-row tiles t = blockIdx.x + i *
// gridDim.x): the threads load tile i+1 into registers (16-byte streaming
// loads) while the tensor cores work on tile i and the threads drain tile
// i-1's accumulator from tensor memory (tcgen05.ld) to global memory.  The
// next tile is split and written into the other of two shared-memory buffers
// in the 128-byte swizzled layout, and thread 0 issues its MMAs; each tile's
// MMAs commit to the mbarrier of its buffer, which frees the buffer and
// publishes the accumulator.  Accumulators are double-buffered in tensor
// memory.  Every wait is bounded; a kernel that gives up still waits for the
// MMAs it issued before it frees tensor memory.
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
constexpr int kDenseThreads = 512;
constexpr uint32_t kBlk = 128 * 128;   // bytes of a 128-row block

// shared-memory map of proj_fwd_kernel (from a 1024-byte aligned base)
constexpr uint32_t kFwdA = 0;                          // [buf][hi|lo][kb] x kBlk
constexpr uint32_t kFwdW = kFwdA + 8 * kBlk;           // W^T: [hi|lo][kb] x 64 rows x 128 B
constexpr uint32_t kFwdBar = kFwdW + 4 * 64 * 128;
constexpr uint32_t kFwdSmem = kFwdBar + 32 + 1024;     // two barriers, the TMEM slot, alignment
// shared-memory map of proj_bwd_kernel
constexpr uint32_t kBwdG = 0;                          // [buf][hi|lo] x kBlk
constexpr uint32_t kBwdH = kBwdG + 4 * kBlk;           // [buf][hi|lo][block] x kBlk
constexpr uint32_t kBwdW = kBwdH + 8 * kBlk;           // W: [hi|lo] x kBlk
constexpr uint32_t kBwdBar = kBwdW + 2 * kBlk;
constexpr uint32_t kBwdSmem = kBwdBar + 32 + 1024;
static_assert(kBwdSmem <= 227 * 1024, "shared memory of one CTA");

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

// writes the hi and lo parts of one fp32 value at byte offset `off` of the
// hi and lo copies
__device__ __forceinline__ void put1(uint32_t hi_base, uint32_t lo_base, uint32_t off, float v) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  const __nv_bfloat16 l = __float2bfloat16_rn(v - __bfloat162float(h));
  sts16(hi_base + off, *reinterpret_cast<const uint16_t*>(&h));
  sts16(lo_base + off, *reinterpret_cast<const uint16_t*>(&l));
}

__device__ __forceinline__ uint32_t align1024(uint32_t a) { return (a + 1023u) & ~1023u; }

// 16-byte loads of one 128-row tile of a row-major [n x (C4 * 4)] fp32 matrix
// (rows past n read as zero): element j of this thread is float4 q = tid +
// kDenseThreads * j, at row q / C4, column 4 (q % C4).
template <int C4, int NJ>
__device__ __forceinline__ void load_tile(float4 (&R)[NJ], const float* __restrict__ X, int row0,
                                          int n) {
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int q = threadIdx.x + kDenseThreads * j;
    const int r = row0 + q / C4;
    R[j] = r < n ? __ldcs(reinterpret_cast<const float4*>(X + (size_t)r * (C4 * 4)) + (q % C4))
                 : make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

// ... and their hi / lo parts into the swizzled blocks at hi_base / lo_base
// (block b holds columns 64 b .. 64 b + 63; blocks kBlk bytes apart)
template <int C4, int NJ>
__device__ __forceinline__ void store_tile(const float4 (&R)[NJ], uint32_t hi_base,
                                           uint32_t lo_base) {
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const int q = threadIdx.x + kDenseThreads * j;
    const int r = q / C4, f = 4 * (q % C4);
    const uint32_t off = (uint32_t)(f >> 6) * kBlk + tc::sw128_offset_b16(r, f & 63);
    uint2 hi, lo;
    split4(R[j], hi, lo);
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

// drains COLS accumulator columns (starting at column c0 of the tile's
// accumulator) for this warp's 32 rows into out rows of width OUTW
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

// ---------------------------------------------------------------------------
// P = H W
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kDenseThreads, 1)
    proj_fwd_kernel(const float* __restrict__ H, const float* __restrict__ W,
                    float* __restrict__ P, int n, WsHeader* hdr) {
  extern __shared__ unsigned char dense_smem[];
  const uint32_t base = align1024(smem_u32(dense_smem));
  unsigned char* gbase = dense_smem + (base - smem_u32(dense_smem));
  uint64_t* bar = reinterpret_cast<uint64_t*>(gbase + kFwdBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kFwdBar + 16);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t idesc = tc::idesc_bf16(kTileM, kFout, false, false);
  auto A = [&](int b, int part, int kb) { return base + kFwdA + (uint32_t)((b * 2 + part) * 2 + kb) * kBlk; };
  auto Wt = [&](int part, int kb) { return base + kFwdW + (uint32_t)(part * 2 + kb) * (64 * 128); };

  const int ntiles = (n + kTileM - 1) / kTileM;
  const int grid = gridDim.x;
  int t = blockIdx.x;
  float4 R[8];   // the next H tile: 128 rows x 32 float4
  if (t < ntiles) load_tile<32, 8>(R, H, t * kTileM, n);

  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(tmem_slot, 2 * kFout);   // two accumulators of 64 columns
  // operand B = W^T (row n' = column n' of W), once per CTA
  for (int idx = tid; idx < kFin * kFout; idx += kDenseThreads) {
    const int k = idx / kFout, nn = idx % kFout;
    const uint32_t off = tc::sw128_offset_b16(nn, k & 63);
    put1(Wt(0, k >> 6), Wt(1, k >> 6), off, __ldg(W + idx));
  }
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  const int q4 = warp & 3, cg = warp >> 2;   // epilogue: TMEM lanes 32 q4.., columns 16 cg..
  bool ok = true;
  int last = -1;   // local index of the last tile whose MMAs were issued
  int i = 0;
  for (; t < ntiles; ++i, t += grid) {
    const int b = i & 1;
    if (i >= 2) {   // buffer b is free once tile i-2's MMAs are done
      ok = __syncthreads_and(mbar_wait(&bar[b], ((i >> 1) - 1) & 1, hdr));
      if (!ok) break;
    }
    store_tile<32, 8>(R, A(b, 0, 0), A(b, 1, 0));
    if (t + grid < ntiles) load_tile<32, 8>(R, H, (t + grid) * kTileM, n);
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      const uint32_t d = tmem + (uint32_t)(kFout * b);
#pragma unroll
      for (int kb = 0; kb < 2; ++kb)
#pragma unroll
        for (int s = 0; s < 4; ++s) {
          const uint64_t ah = kdesc(A(b, 0, kb), s), al = kdesc(A(b, 1, kb), s);
          const uint64_t bh = kdesc(Wt(0, kb), s), bl = kdesc(Wt(1, kb), s);
          tc::mma_bf16(d, ah, bh, idesc, (kb | s) != 0);
          tc::mma_bf16(d, ah, bl, idesc, true);
          tc::mma_bf16(d, al, bh, idesc, true);
        }
      tc::mma_commit(&bar[b]);
    }
    last = i;
    if (i >= 1) {   // tile i-1's accumulator to P while the tensor cores work on tile i
      ok = __syncthreads_and(mbar_wait(&bar[b ^ 1], ((i - 1) >> 1) & 1, hdr));
      if (!ok) break;
      tc::fence_after_sync();
      const int row = (t - grid) * kTileM + 32 * q4 + lane;
      drain_rows<16, false>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFout * (b ^ 1) + 16 * cg),
                            P, kFout, row, 16 * cg, n);
    }
  }
  if (ok && last >= 0) {
    ok = __syncthreads_and(mbar_wait(&bar[last & 1], (last >> 1) & 1, hdr));
    if (ok) {
      tc::fence_after_sync();
      const int row = (blockIdx.x + last * grid) * kTileM + 32 * q4 + lane;
      drain_rows<16, false>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFout * (last & 1) + 16 * cg),
                            P, kFout, row, 16 * cg, n);
    }
  }
  // a wait gave up: the issued MMAs still write tensor memory; let them end
  if (!ok && last >= 0) mbar_drain(&bar[last & 1], (last >> 1) & 1, hdr);
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
  uint64_t* bar = reinterpret_cast<uint64_t*>(gbase + kBwdBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kBwdBar + 16);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr uint32_t idesc_dh = tc::idesc_bf16(kTileM, kFin, false, false);
  constexpr uint32_t idesc_dw = tc::idesc_bf16(kFin, kFout, true, true);
  // dW of each tile in tensor memory (two accumulators after the two of dH);
  // the tiles' dW are added in registers in fp32 (each thread 16 entries), so
  // no tensor-memory accumulation runs longer than one tile's 8 k-steps
  constexpr uint32_t kDwCol = 2 * kFin;
  auto Gs = [&](int b, int part) { return base + kBwdG + (uint32_t)(b * 2 + part) * kBlk; };
  auto Hs = [&](int b, int part) { return base + kBwdH + (uint32_t)((b * 2 + part) * 2) * kBlk; };
  auto Ws = [&](int part) { return base + kBwdW + (uint32_t)part * kBlk; };

  const int ntiles = (n + kTileM - 1) / kTileM;
  const int grid = gridDim.x;
  int t = blockIdx.x;
  float4 RG[4], RH[8];   // the next tile: G 128 x 16 float4, H 128 x 32 float4
  if (t < ntiles) {
    load_tile<16, 4>(RG, G, t * kTileM, n);
    load_tile<32, 8>(RH, H, t * kTileM, n);
  }

  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(tmem_slot, 512);   // dH: 2 x 128 columns; dW: 2 x 64
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
  // adds tile-buffer bb's dW accumulator to dwacc
  auto add_dw = [&](int bb) {
    float v[16];
    tc::tmem_ld16(tmem + ((uint32_t)(32 * q4) << 16) + kDwCol + (uint32_t)(kFout * bb + 16 * cg), v);
    tc::tmem_wait_ld();
#pragma unroll
    for (int c = 0; c < 16; ++c) dwacc[c] += v[c];
  };
  bool ok = true;
  int last = -1;
  int i = 0;
  for (; t < ntiles; ++i, t += grid) {
    const int b = i & 1;
    if (i >= 2) {
      ok = __syncthreads_and(mbar_wait(&bar[b], ((i >> 1) - 1) & 1, hdr));
      if (!ok) break;
    }
    store_tile<16, 4>(RG, Gs(b, 0), Gs(b, 1));
    store_tile<32, 8>(RH, Hs(b, 0), Hs(b, 1));
    if (t + grid < ntiles) {
      load_tile<16, 4>(RG, G, (t + grid) * kTileM, n);
      load_tile<32, 8>(RH, H, (t + grid) * kTileM, n);
    }
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      // dW += H^T G: M = f_in (MN-major H), N = f_out (MN-major G), K = the tile's rows
#pragma unroll
      for (int s = 0; s < kTileM / 16; ++s) {
        const uint64_t ah = mndesc(Hs(b, 0), s), al = mndesc(Hs(b, 1), s);
        const uint64_t bh = mndesc(Gs(b, 0), s), bl = mndesc(Gs(b, 1), s);
        const uint32_t dw = tmem + kDwCol + (uint32_t)(kFout * b);
        tc::mma_bf16(dw, ah, bh, idesc_dw, s > 0);
        tc::mma_bf16(dw, ah, bl, idesc_dw, true);
        tc::mma_bf16(dw, al, bh, idesc_dw, true);
      }
      // dH = G W^T: M = rows, N = f_in, K = f_out (both K-major)
      const uint32_t d = tmem + (uint32_t)(kFin * b);
#pragma unroll
      for (int s = 0; s < (dH ? kFout / 16 : 0); ++s) {
        const uint64_t ah = kdesc(Gs(b, 0), s), al = kdesc(Gs(b, 1), s);
        const uint64_t bh = kdesc(Ws(0), s), bl = kdesc(Ws(1), s);
        tc::mma_bf16(d, ah, bh, idesc_dh, s > 0);
        tc::mma_bf16(d, ah, bl, idesc_dh, true);
        tc::mma_bf16(d, al, bh, idesc_dh, true);
      }
      tc::mma_commit(&bar[b]);
    }
    last = i;
    if (i >= 1) {   // tile i-1's dH to memory and its dW into dwacc
      ok = __syncthreads_and(mbar_wait(&bar[b ^ 1], ((i - 1) >> 1) & 1, hdr));
      if (!ok) break;
      tc::fence_after_sync();
      const int row = (t - grid) * kTileM + 32 * q4 + lane;
      if (dH)
        drain_rows<32, true>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFin * (b ^ 1) + 32 * cg),
                             dH, kFin, row, 32 * cg, n);
      add_dw(b ^ 1);
    }
  }
  if (ok && last >= 0) {
    ok = __syncthreads_and(mbar_wait(&bar[last & 1], (last >> 1) & 1, hdr));
    if (ok) {
      tc::fence_after_sync();
      const int row = (blockIdx.x + last * grid) * kTileM + 32 * q4 + lane;
      if (dH)
        drain_rows<32, true>(tmem + ((uint32_t)(32 * q4) << 16) + (uint32_t)(kFin * (last & 1) + 32 * cg),
                             dH, kFin, row, 32 * cg, n);
      add_dw(last & 1);
      // this CTA's dW: TMEM lane = f_in, column = f_out
      float4* dst = reinterpret_cast<float4*>(dWpart + (size_t)blockIdx.x * kFin * kFout +
                                              (size_t)(32 * q4 + lane) * kFout + 16 * cg);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        dst[q] = make_float4(dwacc[4 * q], dwacc[4 * q + 1], dwacc[4 * q + 2], dwacc[4 * q + 3]);
    }
  }
  if (!ok && last >= 0) mbar_drain(&bar[last & 1], (last >> 1) & 1, hdr);
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
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(proj_fwd_kernel), (int)kFwdSmem);
  if (e != cudaSuccess || n <= 0) return e;
  {
    KTimer t("proj_fwd", st);
    proj_fwd_kernel<<<dense_grid(n), kDenseThreads, kFwdSmem, st>>>(H, W, P, n, hdr);
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
