// k_dense.cu -- dense projection of the graph loss (f_in = 128, f_out = 64).
//
//   P  = H W        H: n x 128, W: 128 x 64       (tensor cores)
//   dH = G W^T      G: n x 64                      (tensor cores)
//   dW = H^T G      per-CTA partial sums on the CUDA cores (tiles staged by
//                   cp.async, double-buffered), then one fixed-order reduction
//
// Tensor-core kernels: one CTA of 4 warps per SM, 128-row tiles.  The row
// tile arrives by TMA in the 128-byte swizzled K-major layout; the threads
// split it in place into TF32 hi and lo parts, and thread 0 issues
// tcgen05.mma.kind::tf32 with the fp32 accumulator in tensor memory:
//   D = A_hi B_hi + A_hi B_lo + A_lo B_hi      ("3xTF32": about fp32 accuracy)
// The epilogue reads the accumulator with tcgen05.ld (warp w: TMEM lanes
// 32w..32w+31, i.e. tile rows 32w..32w+31) and stores rows.  W (or its
// transpose) is split and swizzled into shared memory once per CTA.
// Waits on mbarriers are bounded (status word in the workspace header).
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace sdad {

constexpr int kFin = 128, kFout = 64;
constexpr int kTileM = 128;
constexpr int kTcThreads = 128;

// ---------------------------------------------------------------------------
// tensor maps (driver entry point obtained through the runtime)
// ---------------------------------------------------------------------------
namespace {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Row-major fp32 matrix [rows x cols] read in boxes of 32 columns x 128 rows
// with the 128-byte swizzle (rows past the end read as zero).
bool make_map(CUtensorMap* map, const float* base, int rows, int cols) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * sizeof(float)};
  const cuuint32_t box[2] = {32, kTileM};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}
}  // namespace

// ---------------------------------------------------------------------------
// shared memory of the tensor-core kernels
// ---------------------------------------------------------------------------
// KA k-blocks (32 fp32 wide) of the A tile (128 rows) and of operand B (NB
// rows), hi and lo copies of both, each k-block 1024-byte aligned.
template <int KA, int NB>
struct TcSmem {
  float a_hi[KA][kTileM * 32];
  float a_lo[KA][kTileM * 32];
  float b_hi[KA][NB * 32];
  float b_lo[KA][NB * 32];
  uint64_t bar_load;
  uint64_t bar_mma;
  uint32_t tmem_base;
};

template <int KA, int NB>
constexpr size_t tc_smem_bytes() {
  return sizeof(TcSmem<KA, NB>) + 1024;   // room to align the base to 1024 bytes
}

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
  const uint32_t a = smem_u32(p);
  return p + ((1024u - (a & 1023u)) & 1023u);
}

// Writes operand B (NB rows x KA*32 columns, K-major, swizzled) split into hi
// and lo.  get(n, k) returns the fp32 value of row n, column k.
template <int KA, int NB, class Get>
__device__ __forceinline__ void stage_b(TcSmem<KA, NB>& S, Get get) {
  for (int idx = threadIdx.x; idx < NB * KA * 32; idx += blockDim.x) {
    const int nn = idx / (KA * 32), k = idx % (KA * 32);
    const float v = get(nn, k);
    const float hi = tc::tf32_hi(v);
    const uint32_t off = tc::sw128_offset(nn, k & 31) / 4;
    S.b_hi[k >> 5][off] = hi;
    S.b_lo[k >> 5][off] = v - hi;
  }
}

// One CTA per SM; each CTA takes the 128-row tiles t = blockIdx.x, +gridDim.x.
// X: [n x KA*32] (read through `map`), B staged from W, out: [n x NB].
//   W_ROWS_ARE_B: operand B row n' is W row n' (dH = G W^T);
//   otherwise operand B row n' is W column n' (P = H W).
template <int KA, int NB, bool W_ROWS_ARE_B>
__global__ void __launch_bounds__(kTcThreads, 1)
    proj_tc_kernel(const __grid_constant__ CUtensorMap map, const float* __restrict__ W,
                   float* __restrict__ out, int n, WsHeader* hdr) {
  extern __shared__ unsigned char raw[];
  TcSmem<KA, NB>& S = *reinterpret_cast<TcSmem<KA, NB>*>(align1024(raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr uint32_t kTileBytes = KA * kTileM * 32 * sizeof(float);
  constexpr uint32_t idesc = tc::idesc_tf32(kTileM, NB);

  if (threadIdx.x == 0) {
    mbar_init(&S.bar_load, 1);
    mbar_init(&S.bar_mma, 1);
    fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&S.tmem_base, NB);   // NB columns of fp32 accumulators
  if (W_ROWS_ARE_B)
    stage_b<KA, NB>(S, [&](int nn, int k) { return __ldg(W + (size_t)nn * (KA * 32) + k); });
  else
    stage_b<KA, NB>(S, [&](int nn, int k) { return __ldg(W + (size_t)k * NB + nn); });
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = S.tmem_base;

  uint32_t ph_load = 0, ph_mma = 0;
  const int ntiles = (n + kTileM - 1) / kTileM;
  for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
    const int row0 = t * kTileM;
    if (threadIdx.x == 0) {
      mbar_arrive_expect_tx(&S.bar_load, kTileBytes);
#pragma unroll
      for (int kb = 0; kb < KA; ++kb) tc::tma_load_2d(S.a_hi[kb], &map, kb * 32, row0, &S.bar_load);
    }
    // all threads take the same decision (a wait that gave up ends the kernel)
    const bool got = __syncthreads_and(mbar_wait(&S.bar_load, ph_load, hdr));
    if (!got) {   // the tile's copy may still be landing: let it, then leave
      mbar_drain(&S.bar_load, ph_load, hdr);
      break;
    }
    ph_load ^= 1;
    // split the tile in place: hi stays, lo goes to the twin buffer
    {
      float4* hi4 = reinterpret_cast<float4*>(&S.a_hi[0][0]);
      float4* lo4 = reinterpret_cast<float4*>(&S.a_lo[0][0]);
      for (int i = threadIdx.x; i < (int)(kTileBytes / 16); i += blockDim.x) {
        const float4 x = hi4[i];
        const float4 h = make_float4(tc::tf32_hi(x.x), tc::tf32_hi(x.y), tc::tf32_hi(x.z),
                                     tc::tf32_hi(x.w));
        hi4[i] = h;
        lo4[i] = make_float4(x.x - h.x, x.y - h.y, x.z - h.z, x.w - h.w);
      }
    }
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (threadIdx.x == 0) {
      tc::fence_after_sync();
#pragma unroll
      for (int s = 0; s < KA * 4; ++s) {   // k-steps of 8 tf32 (32 bytes)
        const int kb = s >> 2;
        const uint32_t off = (uint32_t)(s & 3) * 32u;
        const uint64_t ah = tc::smem_desc_sw128(smem_u32(S.a_hi[kb]) + off);
        const uint64_t al = tc::smem_desc_sw128(smem_u32(S.a_lo[kb]) + off);
        const uint64_t bh = tc::smem_desc_sw128(smem_u32(S.b_hi[kb]) + off);
        const uint64_t bl = tc::smem_desc_sw128(smem_u32(S.b_lo[kb]) + off);
        tc::mma_tf32(tmem, ah, bh, idesc, s > 0);
        tc::mma_tf32(tmem, ah, bl, idesc, true);
        tc::mma_tf32(tmem, al, bh, idesc, true);
      }
      tc::mma_commit(&S.bar_mma);
    }
    const bool done = __syncthreads_and(mbar_wait(&S.bar_mma, ph_mma, hdr));
    if (!done) {   // the MMAs still write tensor memory: let them end before it is freed
      mbar_drain(&S.bar_mma, ph_mma, hdr);
      break;
    }
    ph_mma ^= 1;
    tc::fence_after_sync();
    // epilogue: warp w owns tile rows 32w .. 32w+31 (its TMEM lane quadrant)
    {
      const int row = row0 + warp * 32 + lane;
      const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
      for (int c = 0; c < NB; c += 32) {
        float v[32];
        tc::tmem_ld32(taddr + (uint32_t)c, v);
        tc::tmem_wait_ld();
        if (row < n) {
          float4* dst = reinterpret_cast<float4*>(out + (size_t)row * NB + c);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
      }
    }
    tc::fence_before_sync();
    __syncthreads();
  }
  tc::fence_after_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, NB);
}

// dW partials: dWpart[b] = sum over the CTA's 64-row tiles of H_tile^T G_tile.
// Thread (ta, tb) owns dW[4*ta .. +3][8*tb .. +7] in registers.  The tiles go
// through two shared-memory stages filled by cp.async (16-byte copies; rows
// past n are zero-filled), so the next tile loads while this one is used.
constexpr int kDwRows = 64;
struct DwStage {
  float H[kDwRows * kFin];
  float G[kDwRows * kFout];
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}

// Issues the copies of the tile starting at row r0 into stage S (one group).
__device__ __forceinline__ void dw_load(DwStage& S, const float* __restrict__ H,
                                        const float* __restrict__ G, int r0, int n) {
  for (int i = threadIdx.x; i < kDwRows * kFin / 4; i += blockDim.x) {
    const int rr = i / (kFin / 4);
    const bool ok = r0 + rr < n;
    cp_async16(S.H + 4 * i, ok ? H + (size_t)r0 * kFin + 4 * i : H, ok);
  }
  for (int i = threadIdx.x; i < kDwRows * kFout / 4; i += blockDim.x) {
    const int rr = i / (kFout / 4);
    const bool ok = r0 + rr < n;
    cp_async16(S.G + 4 * i, ok ? G + (size_t)r0 * kFout + 4 * i : G, ok);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

__global__ void __launch_bounds__(256)
    proj_dw_kernel(const float* __restrict__ H, const float* __restrict__ G,
                   float* __restrict__ dWpart, int n) {
  extern __shared__ __align__(16) unsigned char dw_raw[];
  DwStage* st = reinterpret_cast<DwStage*>(dw_raw);   // two stages
  const int tid = threadIdx.x, tb = tid & 7, ta = tid >> 3;   // ta 0..31, tb 0..7
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  const int stride = gridDim.x * kDwRows;
  int r0 = blockIdx.x * kDwRows;
  if (r0 < n) dw_load(st[0], H, G, r0, n);
  for (int it = 0; r0 < n; ++it, r0 += stride) {
    DwStage& cur = st[it & 1];
    const bool more = r0 + stride < n;
    if (more) dw_load(st[(it + 1) & 1], H, G, r0 + stride, n);
    if (more)
      asm volatile("cp.async.wait_group 1;" ::: "memory");   // this tile's group is done
    else
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
#pragma unroll 4
    for (int r = 0; r < kDwRows; ++r) {
      const float4 h = *reinterpret_cast<const float4*>(cur.H + r * kFin + 4 * ta);
      const float4 g0 = *reinterpret_cast<const float4*>(cur.G + r * kFout + 8 * tb);
      const float4 g1 = *reinterpret_cast<const float4*>(cur.G + r * kFout + 8 * tb + 4);
      const float hv[4] = {h.x, h.y, h.z, h.w};
      const float gv[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(hv[i], gv[j], acc[i][j]);
    }
    __syncthreads();   // the stage is refilled two tiles on
  }
  float* dst = dWpart + (size_t)blockIdx.x * kFin * kFout;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float4* d = reinterpret_cast<float4*>(dst + (4 * ta + i) * kFout + 8 * tb);
    d[0] = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
    d[1] = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
  }
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

namespace {

template <int KA, int NB, bool T>
cudaError_t launch_tc(const char* name, const float* X, int xcols, const float* W, float* out,
                      int n, WsHeader* hdr, cudaStream_t st) {
  auto kern = proj_tc_kernel<KA, NB, T>;
  constexpr size_t smem = tc_smem_bytes<KA, NB>();
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kern), (int)smem);
  if (e != cudaSuccess) return e;
  if (n <= 0) return cudaSuccess;
  CUtensorMap map;
  if (!make_map(&map, X, n, xcols)) return cudaErrorInvalidValue;
  const int tiles = (n + kTileM - 1) / kTileM;
  const int grid = std::min(tiles, device_sm_count());
  {
    KTimer t(name, st);
    kern<<<grid, kTcThreads, smem, st>>>(map, W, out, n, hdr);
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t dense_proj_fwd(const float* H, const float* W, float* P, int n, WsHeader* hdr,
                           cudaStream_t st) {
  // P = H W: A = H (K = 128 -> 4 k-blocks), operand B row n' = W column n' (64 rows)
  return launch_tc<4, kFout, false>("proj_fwd", H, kFin, W, P, n, hdr, st);
}

cudaError_t dense_proj_bwd(const float* H, const float* W, const float* G, float* dH,
                           float* dWpart, float* dW, int n, WsHeader* hdr, cudaStream_t st) {
  cudaError_t e;
  if (dH) {
    // dH = G W^T: A = G (K = 64 -> 2 k-blocks), operand B row n' = W row n' (128 rows)
    if ((e = launch_tc<2, kFin, true>("proj_dh", G, kFout, W, dH, n, hdr, st)) != cudaSuccess)
      return e;
  }
  if (!dW) return cudaSuccess;
  {
    e = ensure_dynamic_smem(reinterpret_cast<const void*>(proj_dw_kernel),
                            (int)(2 * sizeof(DwStage)));
    if (e != cudaSuccess) return e;
    KTimer t("proj_dw", st);
    proj_dw_kernel<<<kDwParts, 256, 2 * sizeof(DwStage), st>>>(H, G, dWpart, n);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  {
    KTimer t("dw_reduce", st);
    dw_reduce_kernel<<<(kFin * kFout + 255) / 256, 256, 0, st>>>(dWpart, kDwParts, dW);
  }
  return cudaGetLastError();
}

}  // namespace sdad
