// k_cp.cu -- CP decomposition of a 3-way sparse tensor (rank 32).
//
//   e_n  = T_n - sum_r A_{i r} B_{j r} C_{k r}
//   L    = sum_n e_n^2
//   dA_i = -2 sum_{n: i_n = i} e_n (B_{j_n} * C_{k_n})    (and cyclically for B, C)
//   dT   = 2 e, entry order
//
// Atomic-free path (SDAD_T_CSC / AUTO): one pass per requested factor over the
// tensor sorted by that mode (a residual-weighted MTTKRP).  The pass streams
// the two other indices and the value of each entry through shared memory
// (bulk copies), keeps the segment's own factor row in registers and gathers
// the two other factor rows (128 bytes each; the factors are L2-resident).
// Lane layout: 4 entries per warp step, 8 lanes per entry, one float4 of the
// 32 factor entries per lane.  The first pass also produces the loss and dT.
//
// Atomic path (SDAD_T_ATOMIC): one pass in entry order that scatters all three
// factor gradients with float4 atomic adds into zeroed outputs.
#include <algorithm>

#include "engine.cuh"
#include "internal.h"

namespace sdad {

constexpr int kCpCap = 2048;
constexpr int kCpNS = 2;
constexpr int kCpLong = 256;

__device__ __forceinline__ float4 mul4(const float4& a, const float4& b) {
  return make_float4(a.x * b.x, a.y * b.y, a.z * b.z, a.w * b.w);
}
__device__ __forceinline__ float dot4(const float4& a, const float4& b) {
  return fmaf(a.w, b.w, fmaf(a.z, b.z, fmaf(a.y, b.y, a.x * b.x)));
}
__device__ __forceinline__ void axpy4c(float4& acc, float e, const float4& b) {
  acc.x = fmaf(e, b.x, acc.x);
  acc.y = fmaf(e, b.y, acc.y);
  acc.z = fmaf(e, b.z, acc.z);
  acc.w = fmaf(e, b.w, acc.w);
}
__device__ __forceinline__ float4 xor4(const float4& v, int o) {
  return make_float4(__shfl_xor_sync(FULL_MASK, v.x, o), __shfl_xor_sync(FULL_MASK, v.y, o),
                     __shfl_xor_sync(FULL_MASK, v.z, o), __shfl_xor_sync(FULL_MASK, v.w, o));
}
__device__ __forceinline__ float4 plus4(const float4& a, const float4& b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 scale4(float s, const float4& a) {
  return make_float4(s * a.x, s * a.y, s * a.z, s * a.w);
}

struct CpModeBody {
  const int32_t* __restrict__ ptr;     // segptr of this mode
  const float* __restrict__ own;       // factor of this mode   [dim x 32]
  const float* __restrict__ f1;        // factor of the first other mode
  const float* __restrict__ f2;        // factor of the second other mode
  float* __restrict__ dOwn;            // nullable
  float* __restrict__ dT;              // nullable
  const int32_t* __restrict__ sperm;   // sorted position -> entry number (needed with dT)
  int add_e2;

  template <int CAP>
  __device__ __forceinline__ void chunk(const ChunkView<3, CAP>& v, int warp, int lane,
                                        double& loss) {
    constexpr int U = 4;   // key groups in flight per warp (16 keys)
    const int slot = lane >> 3, sl = lane & 7;
    for_each_part<kCpLong>(v, ptr, warp, [&](int r, int s0, int s1, int ps, int pe, bool single) {
      const float4 u = __ldg(reinterpret_cast<const float4*>(own + (size_t)r * 32) + sl);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int pb = ps; pb < pe; pb += 4 * U) {
        float4 o1[U], o2[U];
        float t[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const int p = pb + 4 * k + slot;
          o1[k] = make_float4(0.f, 0.f, 0.f, 0.f);
          o2[k] = o1[k];
          t[k] = 0.f;
          if (p < pe) {
            const int j1 = v.geti(0, p), j2 = v.geti(1, p);
            t[k] = v.getf(2, p);
            o1[k] = __ldg(reinterpret_cast<const float4*>(f1 + (size_t)j1 * 32) + sl);
            o2[k] = __ldg(reinterpret_cast<const float4*>(f2 + (size_t)j2 * 32) + sl);
          }
        }
#pragma unroll
        for (int k = 0; k < U; ++k) {
          const int p = pb + 4 * k + slot;
          const bool act = p < pe;
          const float4 h = mul4(o1[k], o2[k]);
          const float model = group_sum<8>(dot4(u, h));
          const float e = act ? t[k] - model : 0.f;
          if (act && sl == 0) {
            if (add_e2) loss += (double)e * (double)e;
            if (dT) dT[sperm ? __ldg(sperm + p) : p] = 2.f * e;
          }
          axpy4c(acc, e, h);
        }
      }
      acc = plus4(acc, xor4(acc, 8));
      acc = plus4(acc, xor4(acc, 16));
      if (dOwn && slot == 0) {
        const float4 g = scale4(-2.f, acc);
        float4* dst = reinterpret_cast<float4*>(dOwn + (size_t)r * 32) + sl;
        if (single && !combined_atomically<CAP, kCpLong>(s0, s1)) *dst = g;
        else atomicAdd(dst, g);
      }
    });
  }
};

__global__ void SDAD_PIPE_BOUNDS
    cp_mode_kernel(StreamSrc<3> src, CpModeBody body, WsHeader* hdr, double* partials,
                   int first_slot, int finalize, double* loss_out) {
  extern __shared__ __align__(1024) unsigned char smraw[];
  using Smem = PipeSmem<3, kCpCap, kCpNS>;
  const double cta =
      run_pipeline<true, 3, kCpCap, kCpNS, CpModeBody, kCpLong>(src, body, hdr, smraw);
  if (loss_out)
    publish_loss(cta, hdr, partials, first_slot, finalize != 0, 1.0, loss_out,
                 reinterpret_cast<Smem*>(smraw)->red);
}

// Entry-order pass scattering all three factor gradients (outputs zeroed).
// Eight lanes per entry (four floats each), four entries per warp step;
// kCpAtomicUnroll steps' index and factor loads are issued together.
#ifndef SDAD_CPA_UNROLL
#define SDAD_CPA_UNROLL 2
#endif
// resident CTAs per SM the pass is compiled for: 4 (64 registers) measured
// 0.966 ms on 10^7 entries, against 0.983 ms at 3 (76 registers) and 1.19 ms
// at 5 (spills); the grid is the resident CTAs (1.06 ms with 8 CTAs per SM
// requested and three resident, the rest in a second wave)
#ifndef SDAD_CPA_MINB
#define SDAD_CPA_MINB 4
#endif
constexpr int kCpAtomicUnroll = SDAD_CPA_UNROLL;
__global__ void __launch_bounds__(256, SDAD_CPA_MINB)
    cp_atomic_kernel(int nnz, const int32_t* __restrict__ I, const int32_t* __restrict__ J,
                     const int32_t* __restrict__ K, const float* __restrict__ T,
                     const float* __restrict__ A, const float* __restrict__ B,
                     const float* __restrict__ C, float* dA, float* dB, float* dC, float* dT,
                     WsHeader* hdr, double* partials, double* loss_out) {
  __shared__ double red[8];
  const int lane = threadIdx.x & 31, slot = lane >> 3, sl = lane & 7;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  double loss = 0.0;
  constexpr int U = kCpAtomicUnroll;   // groups of four entries whose loads go together
  for (int pb = gw * 4 * U; pb < nnz; pb += nw * 4 * U) {
    float4 a[U], b[U], c[U];
    float t[U];
    int i[U], j[U], k[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = pb + 4 * u + slot;
      a[u] = b[u] = c[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      t[u] = 0.f;
      i[u] = j[u] = k[u] = 0;
      if (p < nnz) {
        i[u] = __ldg(I + p); j[u] = __ldg(J + p); k[u] = __ldg(K + p); t[u] = __ldg(T + p);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (pb + 4 * u + slot < nnz) {
        a[u] = __ldg(reinterpret_cast<const float4*>(A + (size_t)i[u] * 32) + sl);
        b[u] = __ldg(reinterpret_cast<const float4*>(B + (size_t)j[u] * 32) + sl);
        c[u] = __ldg(reinterpret_cast<const float4*>(C + (size_t)k[u] * 32) + sl);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int p = pb + 4 * u + slot;
      const float model = group_sum<8>(dot4(a[u], mul4(b[u], c[u])));
      if (p >= nnz) continue;
      const float e = t[u] - model;
      if (sl == 0) {
        loss += (double)e * (double)e;
        if (dT) dT[p] = 2.f * e;
      }
      const float m2 = -2.f * e;
      if (dA) atomicAdd(reinterpret_cast<float4*>(dA + (size_t)i[u] * 32) + sl, scale4(m2, mul4(b[u], c[u])));
      if (dB) atomicAdd(reinterpret_cast<float4*>(dB + (size_t)j[u] * 32) + sl, scale4(m2, mul4(a[u], c[u])));
      if (dC) atomicAdd(reinterpret_cast<float4*>(dC + (size_t)k[u] * 32) + sl, scale4(m2, mul4(a[u], b[u])));
    }
  }
  const double cta = block_sum_d(loss, red);
  publish_loss(cta, hdr, partials, 0, true, 1.0, loss_out, red);
}

namespace {
constexpr size_t kCpSmem = pipe_smem_bytes<3, kCpCap, kCpNS>();
}

cudaError_t run_cp3(const sdad_coo3* T, const float* A, const float* B, const float* C,
                    double* loss, float* dA, float* dB, float* dC, float* dT, sdad_tmode tmode,
                    const WsLayout& L, cudaStream_t st) {
  const int sms = device_sm_count();
  const int nnz = (int)T->nnz;
  cudaError_t e;
  const float* fac[3] = {A, B, C};
  float* dfac[3] = {dA, dB, dC};

  if (tmode == SDAD_T_ATOMIC) {
    for (int m = 0; m < 3; ++m)
      if (dfac[m] && (e = zero_f32(dfac[m], (size_t)T->dims[m] * 32, st)) != cudaSuccess) return e;
    // as many CTAs as are resident at once (a grid-stride loop; no second wave)
    int per_sm = 1;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, cp_atomic_kernel, 256, 0)) !=
        cudaSuccess)
      return e;
    const int grid = std::max(1, std::min((nnz + 32 * kCpAtomicUnroll - 1) / (32 * kCpAtomicUnroll),
                                          sms * std::max(per_sm, 1)));
    {
      KTimer t_cp_atomic("cp_atomic", st);
      cp_atomic_kernel<<<grid, 256, 0, st>>>(nnz, T->idx[0], T->idx[1], T->idx[2], T->val, A, B, C,
                                             dA, dB, dC, dT, L.hdr, L.partials, loss);
    }
    return cudaGetLastError();
  }

  e = ensure_dynamic_smem(reinterpret_cast<const void*>(cp_mode_kernel), (int)kCpSmem);
  if (e != cudaSuccess) return e;
  // initialise combined segments of every requested factor gradient
  for (int m = 0; m < 3; ++m) {
    if (!dfac[m]) continue;
    InitSet s{T->segptr[m], T->dims[m], dfac[m], nullptr, 0.f};
    InitSet none{nullptr, 0, nullptr, nullptr, 0.f};
    if ((e = init_combined<kCpCap, kCpLong>(s, none, 32, sms, st)) != cudaSuccess) return e;
  }
  // modes to run: every requested one; mode 0 alone if none is requested
  int modes[3], nm = 0;
  for (int m = 0; m < 3; ++m)
    if (dfac[m]) modes[nm++] = m;
  if (nm == 0) modes[nm++] = 0;
  const int nc = num_chunks<kCpCap>(T->nnz);
  const int grid = std::min(nc, sms * 2);
  for (int t = 0; t < nm; ++t) {
    const int m = modes[t];
    const int o1 = m == 0 ? 1 : 0, o2 = m == 2 ? 1 : 2;
    StreamSrc<3> src;
    src.ptr = T->segptr[m];
    src.arr[0] = T->sidx[m][o1];
    src.arr[1] = T->sidx[m][o2];
    src.arr[2] = T->sval[m];
    src.nseg = T->dims[m];
    src.nnz = nnz;
    src.nchunks = nc;
    const bool first = t == 0;
    CpModeBody body{T->segptr[m], fac[m], fac[o1], fac[o2], dfac[m], first ? dT : nullptr,
                    T->sperm[m], first ? 1 : 0};
    {
      KTimer t_cp_mode("cp_mode", st);
      cp_mode_kernel<<<grid, kPipeThreads, kCpSmem, st>>>(src, body, L.hdr, L.partials, 0, 1,
                                                          first ? loss : nullptr);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace sdad
