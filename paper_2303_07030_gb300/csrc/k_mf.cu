// k_mf.cu -- matrix factorisation on the observed keys of R (k = 64).
//
//   e_ij = R_ij - U_i . V_j                     for (i, j) in keys(R)
//   L    = sum e_ij^2 + lambda (|U|^2 + |V|^2)
//   dU_i = -2 sum_j e_ij V_j + 2 lambda U_i     (row pass over CSR)
//   dV_j = -2 sum_i e_ij U_i + 2 lambda V_j     (column pass over the CSC twin,
//                                                e recomputed; atomic-free for
//                                                whole columns)
//   dR   = 2 e on keys(R), CSR order            (row pass)
//
// Both passes are the same kernel with the roles of (U, rows) and (V, cols)
// swapped.  Lane layout: a warp works on 4 keys at a time, 8 lanes per key,
// each lane holding 8 of the 64 factor entries (two float4).  The segment's
// own factor row stays in registers; the other factor's row is gathered
// (256 bytes per key, L1/L2).  Segment pieces cut by a chunk boundary or
// longer than kMfLong are combined with float4 atomic adds into rows zeroed
// by init_combined.
#include <algorithm>

#include <climits>

#include "engine.cuh"
#include "halfwarp.cuh"
#include "internal.h"

namespace sdad {

constexpr int kMfCap = 2048;
constexpr int kMfNS = 2;
constexpr int kMfLong = 256;

__device__ __forceinline__ float dot8(const float4& a0, const float4& a1, const float4& b0,
                                      const float4& b1) {
  float d = a0.x * b0.x;
  d = fmaf(a0.y, b0.y, d);
  d = fmaf(a0.z, b0.z, d);
  d = fmaf(a0.w, b0.w, d);
  d = fmaf(a1.x, b1.x, d);
  d = fmaf(a1.y, b1.y, d);
  d = fmaf(a1.z, b1.z, d);
  d = fmaf(a1.w, b1.w, d);
  return d;
}

__device__ __forceinline__ void axpy4(float4& acc, float e, const float4& b) {
  acc.x = fmaf(e, b.x, acc.x);
  acc.y = fmaf(e, b.y, acc.y);
  acc.z = fmaf(e, b.z, acc.z);
  acc.w = fmaf(e, b.w, acc.w);
}

__device__ __forceinline__ float4 shfl_xor4(const float4& v, int o) {
  return make_float4(__shfl_xor_sync(FULL_MASK, v.x, o), __shfl_xor_sync(FULL_MASK, v.y, o),
                     __shfl_xor_sync(FULL_MASK, v.z, o), __shfl_xor_sync(FULL_MASK, v.w, o));
}

__device__ __forceinline__ float4 add4(const float4& a, const float4& b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

__device__ __forceinline__ float4 lin4(float a, const float4& x, float b, const float4& y) {
  return make_float4(fmaf(a, x.x, b * y.x), fmaf(a, x.y, b * y.y), fmaf(a, x.z, b * y.z),
                     fmaf(a, x.w, b * y.w));
}

struct MfBody {
  const int32_t* __restrict__ ptr;
  const float* __restrict__ own;     // [nseg x 64]
  const float* __restrict__ other;   // [* x 64]
  float* __restrict__ dOwn;          // nullable
  float* __restrict__ dR;            // nullable; element-order output (row pass only)
  float lam;
  int add_e2;                        // this pass adds sum e^2 to the loss

  template <int CAP>
  __device__ __forceinline__ void chunk(const ChunkView<2, CAP>& v, int warp, int lane,
                                        double& loss) {
    constexpr int U = 4;   // key groups in flight per warp (16 keys, 4 KB of gathers)
    const int slot = lane >> 3, sl = lane & 7;
    for_each_part<kMfLong>(v, ptr, warp, [&](int r, int s0, int s1, int ps, int pe, bool single) {
      const float4* orow = reinterpret_cast<const float4*>(own + (size_t)r * 64) + sl * 2;
      const float4 u0 = __ldg(orow), u1 = __ldg(orow + 1);
      float4 a0 = make_float4(0.f, 0.f, 0.f, 0.f), a1 = a0;
      for (int pb = ps; pb < pe; pb += 4 * U) {
        float4 o0[U], o1[U];
        float val[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int p = pb + 4 * u + slot;
          o0[u] = make_float4(0.f, 0.f, 0.f, 0.f);
          o1[u] = o0[u];
          val[u] = 0.f;
          if (p < pe) {
            const int j = v.geti(0, p);
            val[u] = v.getf(1, p);
            const float4* q = reinterpret_cast<const float4*>(other + (size_t)j * 64) + sl * 2;
            o0[u] = __ldg(q);
            o1[u] = __ldg(q + 1);
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int p = pb + 4 * u + slot;
          const bool act = p < pe;
          const float d = group_sum<8>(dot8(u0, u1, o0[u], o1[u]));
          const float e = act ? val[u] - d : 0.f;
          if (act && sl == 0) {
            if (add_e2) loss += (double)e * (double)e;
            if (dR) dR[p] = 2.f * e;
          }
          axpy4(a0, e, o0[u]);
          axpy4(a1, e, o1[u]);
        }
      }
      // sum the four key slots (lanes sl, sl+8, sl+16, sl+24)
      a0 = add4(a0, shfl_xor4(a0, 8));
      a1 = add4(a1, shfl_xor4(a1, 8));
      a0 = add4(a0, shfl_xor4(a0, 16));
      a1 = add4(a1, shfl_xor4(a1, 16));
      const bool owner = s0 >= v.cs && (single || warp == 0);
      const bool whole = single && !combined_atomically<CAP, kMfLong>(s0, s1);
      if (owner) {
        const float reg = group_sum<8>(dot8(u0, u1, u0, u1));
        if (lane == 0) loss += (double)lam * (double)reg;
      }
      if (dOwn && slot == 0) {
        const float c = owner ? 2.f * lam : 0.f;
        const float4 g0 = lin4(-2.f, a0, c, u0), g1 = lin4(-2.f, a1, c, u1);
        float4* dst = reinterpret_cast<float4*>(dOwn + (size_t)r * 64) + sl * 2;
        if (whole) {
          dst[0] = g0;
          dst[1] = g1;
        } else {
          atomicAdd(dst, g0);
          atomicAdd(dst + 1, g1);
        }
      }
    });
  }
};

__global__ void SDAD_PIPE_BOUNDS
    mf_kernel(StreamSrc<2> src, MfBody body, WsHeader* hdr, double* partials, int first_slot,
              int finalize, double* loss_out) {
  extern __shared__ __align__(1024) unsigned char smraw[];
  using Smem = PipeSmem<2, kMfCap, kMfNS>;
  const double cta = run_pipeline<true, 2, kMfCap, kMfNS, MfBody, kMfLong>(src, body, hdr, smraw);
  publish_loss(cta, hdr, partials, first_slot, finalize != 0, 1.0, loss_out,
               reinterpret_cast<Smem*>(smraw)->red);
}

// lambda * sum of squares of a dense array (used when no column pass runs).
__global__ void __launch_bounds__(256)
    sumsq_kernel(const float4* __restrict__ a, size_t n4, float lam, WsHeader* hdr,
                 double* partials, int first_slot, double* loss_out) {
  __shared__ double red[8];
  double s = 0.0;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4;
       i += (size_t)gridDim.x * blockDim.x) {
    const float4 v = __ldg(a + i);
    s += (double)(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
  }
  const double cta = block_sum_d(s, red);
  publish_loss(cta * (double)lam, hdr, partials, first_slot, true, 1.0, loss_out, red);
}

namespace {
constexpr size_t kMfSmem = pipe_smem_bytes<2, kMfCap, kMfNS>();
}

// ---------------------------------------------------------------------------
// One-pass mode (SDAD_T_ATOMIC): a single sweep over the CSR computes e, the
// loss, dR, dU (row sums in registers) and scatters dV.
//   init:  dU = 2 lambda U, dV = 2 lambda V (every row), loss part
//          lambda (|U|^2 + |V|^2)
//   sweep: one warp per 1024-key chunk, row by row; per batch of 16 keys of
//          a row, half a warp per key: V_j gathered (16-byte loads), the 16
//          dot products U_i . V_j reduced together, e = R_ij - U_i . V_j,
//          dU_i += -2 e V_j in registers, dV_j += -2 e U_i by vector atomic
//          adds.  With ranked column numbering (sdad_csr_rank_columns) the
//          kMfHot most used columns are summed in shared memory first and
//          added to dV once per CTA, so the hottest columns do not serialise
//          on one address.  Rows cut by chunk boundaries leave pieces.
//   fix:   dU of the cut rows from their pieces (chunk order); loss total.
// V rows are gathered once per key instead of twice (row and column pass).
// The order of the atomic adds varies from run to run.
constexpr int kMfaChunk = kMinCap;   // the piece slots are per kMinCap keys
constexpr int kMfaThreads = 256;
constexpr int kMfaWarps = kMfaThreads / 32;
#ifndef SDAD_MFA_HOT
#define SDAD_MFA_HOT 64
#endif
constexpr int kMfHot = SDAD_MFA_HOT;
// key pairs per batch (4 or 8) and resident CTAs per SM the sweep is compiled
// for.  Measured on 5*10^7 keys: 8 pairs at 3 CTAs (79 registers) 2.83 ms;
// 8 pairs unbounded (122 registers, 2 CTAs) 3.72 ms; 4 pairs at 4 CTAs 2.93 ms,
// at 3 CTAs 3.38 ms, unbounded 4.53 ms; 128 hot columns instead of 64: 2.92 ms
#ifndef SDAD_MFA_PAIRS
#define SDAD_MFA_PAIRS 8
#endif
#ifndef SDAD_MFA_MINB
#define SDAD_MFA_MINB 3
#endif
constexpr int kMfaPairs = SDAD_MFA_PAIRS;
static_assert(kMfaPairs == 4 || kMfaPairs == 8, "the dot-product reductions take 4 or 8 pairs");
// after reduce_half over kMfaPairs values: the key offset of the batch whose
// total lane `lane` holds, whether it is the lane that acts on it, and the
// lane holding the total of key offset o
__device__ __forceinline__ int mfa_key_of_lane(int lane) {
  return kMfaPairs == 8 ? batch_key_of_lane(lane) : 2 * (((lane & 15) >> 2) & 3) + (lane >> 4);
}
__device__ __forceinline__ bool mfa_holder(int lane) {
  return kMfaPairs == 8 ? (lane & 1) == 0 : (lane & 3) == 0;
}
__device__ __forceinline__ int mfa_src_lane(int o) {
  return kMfaPairs == 8 ? batch_src_lane(o) : ((o & 1) << 4) | ((o >> 1) << 2);
}
// Shared-memory place of element 4 sl + c of a hot column's dV row (rank r):
// c-major, so the 16 lanes of a half touch 16 consecutive banks, and rotated
// by 16 for odd ranks, so two halves on columns of different parity use
// different banks (4 sl + c directly gave 4-way bank conflicts; measured
// 2.83 -> 2.75 ms on 5*10^7 keys).
#ifndef SDAD_MFA_HOT_SWIZZLE
#define SDAD_MFA_HOT_SWIZZLE 1
#endif
__device__ __forceinline__ int hot_pos(int r, int sl, int c) {
  if (!SDAD_MFA_HOT_SWIZZLE) return 4 * sl + c;
  return (16 * c + sl + 16 * (r & 1)) & 63;
}
// ... and the element kept at place p
__device__ __forceinline__ int hot_elem(int r, int p) {
  if (!SDAD_MFA_HOT_SWIZZLE) return p;
  const int t = (p - 16 * (r & 1)) & 63;
  return 4 * (t & 15) + (t >> 4);
}

__global__ void __launch_bounds__(256)
    mfa_init_kernel(const float* __restrict__ U, const float* __restrict__ V, int m, int n,
                    float lam, float* __restrict__ dU, float* __restrict__ dV, WsHeader* hdr,
                    double* partials) {
  __shared__ double red[8];
  if (blockIdx.x == 0 && threadIdx.x == 0) hdr->work[0] = 0;   // the sweep's chunk counter
  const size_t nu = (size_t)m * 16, nt = nu + (size_t)n * 16;   // float4 counts
  double s = 0.0;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < nt;
       i += (size_t)gridDim.x * blockDim.x) {
    const bool u = i < nu;
    const float4 x = __ldg(reinterpret_cast<const float4*>(u ? U : V) + (u ? i : i - nu));
    s += (double)dot4(x, x);
    const float4 g = make_float4(2.f * lam * x.x, 2.f * lam * x.y, 2.f * lam * x.z, 2.f * lam * x.w);
    if (u) {
      if (dU) reinterpret_cast<float4*>(dU)[i] = g;
    } else if (dV) {
      reinterpret_cast<float4*>(dV)[i - nu] = g;
    }
  }
  const double cta = block_sum_d(s, red);
  publish_loss(cta * (double)lam, hdr, partials, 0, false, 1.0, nullptr, red);
}

struct MfaPieces {
  float* __restrict__ pfirst;   // [chunks x 64]
  float* __restrict__ plast;    // [chunks x 64]
  int* __restrict__ lastseg;
};

__global__ void __launch_bounds__(kMfaThreads, SDAD_MFA_MINB)
    mfa_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
               const int32_t* __restrict__ rcolidx, const int32_t* __restrict__ rankcol,
               const float* __restrict__ val, int m, int n, int nnz, int nchunks,
               const float* __restrict__ U, const float* __restrict__ V, float lam,
               float* __restrict__ dU, float* __restrict__ dV, float* __restrict__ dR,
               MfaPieces pc, WsHeader* hdr, double* partials, int first_slot) {
  __shared__ float hot[kMfHot * 64];
  __shared__ double red[kMfaWarps];
  const int lane = threadIdx.x & 31;
  const int h = lane >> 4, sl = lane & 15;
  const bool ranked = rcolidx != nullptr && dV != nullptr;
  if (ranked) {
    for (int i = threadIdx.x; i < kMfHot * 64; i += blockDim.x) hot[i] = 0.f;
    __syncthreads();
  }
  const int kl = mfa_key_of_lane(lane);   // the key whose dot product this lane ends with
  double loss = 0.0;
  // chunks are handed out one at a time from a counter in the workspace
  // header (reset by mfa_init_kernel): hub rows make chunks very unequal
  while (true) {
    int ch = 0;
    if (lane == 0) ch = (int)atomicAdd(&hdr->work[0], 1u);
    ch = __shfl_sync(FULL_MASK, ch, 0);
    if (ch >= nchunks) break;   // warp-uniform
    const int cs = ch * kMfaChunk, ce = min(cs + kMfaChunk, nnz);
    if (lane == 0) pc.lastseg[ch] = -1;
    __syncwarp();
    if (cs >= ce) continue;
    int r = warp_lower_bound(rowptr, 0, m + 1, cs + 1) - 1;   // the row of key cs
    int s0 = __ldg(rowptr + r), s1 = __ldg(rowptr + r + 1);
    while (true) {
      const int ps = max(s0, cs), pe = min(s1, ce);
      const float4 uv = ld4(U, r, sl);
      float4 acc = zero4();
      for (int pb = ps; pb < pe; pb += 2 * kMfaPairs) {
        const int nk = min(2 * kMfaPairs, pe - pb);
        const bool mine = lane < nk;
        const int jl = mine ? __ldg(colidx + pb + lane) : 0;
        const float al = mine ? __ldg(val + pb + lane) : 0.f;
        const int rk = (ranked && mine) ? __ldg(rcolidx + pb + lane) : INT_MAX;
        float4 x[kMfaPairs];
        float t[kMfaPairs];
#pragma unroll
        for (int u = 0; u < kMfaPairs; ++u) {
          const int kk = 2 * u + h;
          const int j = __shfl_sync(FULL_MASK, jl, kk);
          x[u] = kk < nk ? ld4(V, j, sl) : zero4();
          t[u] = dot4(x[u], uv);
        }
        const float d = reduce_half(t, lane);
        const float e = __shfl_sync(FULL_MASK, al, kl) - d;   // valid in the holder lanes, kl < nk
        if (mfa_holder(lane) && kl < nk) {
          loss += (double)e * (double)e;
          if (dR) dR[pb + kl] = 2.f * e;
        }
#pragma unroll
        for (int u = 0; u < kMfaPairs; ++u) {
          const int kk = 2 * u + h;
          const float eu = __shfl_sync(FULL_MASK, e, mfa_src_lane(kk));
          const int j = __shfl_sync(FULL_MASK, jl, kk);
          const int rank = __shfl_sync(FULL_MASK, rk, kk);
          if (kk < nk) {
            acc = fma4(eu, x[u], acc);
            if (dV) {
              const float c = -2.f * eu;
              const float4 g = make_float4(c * uv.x, c * uv.y, c * uv.z, c * uv.w);
              if (rank < kMfHot) {
                float* q = hot + rank * 64;
                atomicAdd(q + hot_pos(rank, sl, 0), g.x);
                atomicAdd(q + hot_pos(rank, sl, 1), g.y);
                atomicAdd(q + hot_pos(rank, sl, 2), g.z);
                atomicAdd(q + hot_pos(rank, sl, 3), g.w);
              } else {
                atomicAdd(reinterpret_cast<float4*>(dV + (size_t)j * 64) + sl, g);
              }
            }
          }
        }
      }
      const float4 tot = join_halves(acc);
      if (s0 >= cs && s1 <= ce) {   // the whole row lies in this chunk
        if (dU && lane < 16) {
          const float c = 2.f * lam;
          st4(dU, r, sl, make_float4(fmaf(-2.f, tot.x, c * uv.x), fmaf(-2.f, tot.y, c * uv.y),
                                     fmaf(-2.f, tot.z, c * uv.z), fmaf(-2.f, tot.w, c * uv.w)));
        }
      } else if (lane < 16) {       // a piece of a row cut by the chunk's boundaries
        if (s0 < cs) {
          st4(pc.pfirst, ch, sl, tot);
        } else {
          st4(pc.plast, ch, sl, tot);
          if (lane == 0) pc.lastseg[ch] = r;
        }
      }
      if (s1 >= ce) break;
      // the next row with keys: the one holding key s1
      r = warp_gallop_lower_bound(rowptr, r + 1, m + 1, s1 + 1) - 1;
      s0 = __ldg(rowptr + r);
      s1 = __ldg(rowptr + r + 1);
    }
  }
  if (ranked) {   // the hot columns' sums, once per CTA
    __syncthreads();
    for (int i = threadIdx.x; i < kMfHot * 64; i += blockDim.x) {
      const int slot = i >> 6;
      if (slot < n) atomicAdd(dV + (size_t)__ldg(rankcol + slot) * 64 + hot_elem(slot, i & 63), hot[i]);
    }
  }
  const double cta = block_sum_d(loss, red);
  publish_loss(cta, hdr, partials, first_slot, false, 1.0, nullptr, red);
}

// dU of the rows cut by chunk boundaries: one warp per chunk with a cut row
// begun in it, its pieces added in chunk order; the last CTA sums the loss.
__global__ void __launch_bounds__(256)
    mfa_fix_kernel(const int32_t* __restrict__ rowptr, int nchunks, MfaPieces pc,
                   const float* __restrict__ U, float lam, float* __restrict__ dU, WsHeader* hdr,
                   double* partials, int first_slot, double* loss_out) {
  __shared__ double red[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * 8 + warp, nw = gridDim.x * 8;
  for (int ch = gw; ch < nchunks && dU; ch += nw) {
    const int s = __ldg(pc.lastseg + ch);
    if (s < 0) continue;   // warp-uniform
    const int c1 = (__ldg(rowptr + s + 1) - 1) / kMfaChunk;
    float2 t = __ldg(reinterpret_cast<const float2*>(pc.plast + (size_t)ch * 64) + lane);
    for (int cc = ch + 1; cc <= c1; ++cc) {
      const float2 q = __ldg(reinterpret_cast<const float2*>(pc.pfirst + (size_t)cc * 64) + lane);
      t.x += q.x;
      t.y += q.y;
    }
    const float2 u = __ldg(reinterpret_cast<const float2*>(U + (size_t)s * 64) + lane);
    reinterpret_cast<float2*>(dU + (size_t)s * 64)[lane] =
        make_float2(fmaf(-2.f, t.x, 2.f * lam * u.x), fmaf(-2.f, t.y, 2.f * lam * u.y));
  }
  publish_loss(0.0, hdr, partials, first_slot, true, 1.0, loss_out, red);
}

cudaError_t run_mf_atomic(const sdad_csr* R, const float* U, const float* V, float lambda,
                          double* loss, float* dU, float* dV, float* dR, const WsLayout& L,
                          cudaStream_t st) {
  const int sms = device_sm_count();
  const int m = R->m, n = R->n, nnz = (int)R->nnz;
  const int nchunks = nnz <= 0 ? 1 : (nnz + kMfaChunk - 1) / kMfaChunk;
  const size_t n4 = ((size_t)m + (size_t)n) * 16;
  const int gi = (int)std::max<size_t>(1, std::min<size_t>((n4 + 255) / 256, (size_t)sms * 4));
  cudaError_t e;
  {
    KTimer t("mf_init", st);
    mfa_init_kernel<<<gi, 256, 0, st>>>(U, V, m, n, lambda, dU, dV, L.hdr, L.partials);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  int per_sm = 1;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, mfa_kernel, kMfaThreads, 0)) !=
      cudaSuccess)
    return e;
  const int gw = std::max(1, std::min((nchunks + kMfaWarps - 1) / kMfaWarps, sms * std::max(per_sm, 1)));
  const MfaPieces pc{L.pfirst, L.plast, L.lastseg};
  const bool ranked = csr_ranked(R) && R->rcolidx && R->rankcol;
  {
    KTimer t("mf_atomic", st);
    mfa_kernel<<<gw, kMfaThreads, 0, st>>>(R->rowptr, R->colidx, ranked ? R->rcolidx : nullptr,
                                            ranked ? R->rankcol : nullptr, R->val, m, n, nnz,
                                            nchunks, U, V, lambda, dU, dV, dR, pc, L.hdr,
                                            L.partials, gi);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int gf = std::max(1, std::min((nchunks + 7) / 8, sms * 8));
  {
    KTimer t("mf_fix", st);
    mfa_fix_kernel<<<gf, 256, 0, st>>>(R->rowptr, nchunks, pc, U, lambda, dU, L.hdr, L.partials,
                                        gi + gw, loss);
  }
  return cudaGetLastError();
}

cudaError_t run_mf(const sdad_csr* R, const float* U, const float* V, float lambda,
                   double* loss, float* dU, float* dV, float* dR, sdad_tmode tmode,
                   const WsLayout& L, cudaStream_t st) {
  if (tmode == SDAD_T_ATOMIC) return run_mf_atomic(R, U, V, lambda, loss, dU, dV, dR, L, st);
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(mf_kernel), (int)kMfSmem);
  if (e != cudaSuccess) return e;
  const int sms = device_sm_count();
  InitSet rows{R->rowptr, R->m, dU, nullptr, 0.f};
  InitSet cols{R->colptr, R->n, dV, nullptr, 0.f};
  e = init_combined<kMfCap, kMfLong>(rows, cols, 64, sms, st);
  if (e != cudaSuccess) return e;

  StreamSrc<2> rs;
  rs.ptr = R->rowptr;
  rs.arr[0] = R->colidx;
  rs.arr[1] = R->val;
  rs.nseg = R->m;
  rs.nnz = (int)R->nnz;
  rs.nchunks = num_chunks<kMfCap>(R->nnz);
  const int g1 = std::min(rs.nchunks, sms * 2);
  MfBody rb{R->rowptr, U, V, dU, dR, lambda, 1};
  {
    KTimer t_mf_row("mf_row", st);
    mf_kernel<<<g1, kPipeThreads, kMfSmem, st>>>(rs, rb, L.hdr, L.partials, 0, 0, loss);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;

  if (dV) {
    StreamSrc<2> cs;
    cs.ptr = R->colptr;
    cs.arr[0] = R->rowidx;
    cs.arr[1] = R->val_csc;
    cs.nseg = R->n;
    cs.nnz = (int)R->nnz;
    cs.nchunks = num_chunks<kMfCap>(R->nnz);
    const int g2 = std::min(cs.nchunks, sms * 2);
    MfBody cb{R->colptr, V, U, dV, nullptr, lambda, 0};
    {
      KTimer t_mf_col("mf_col", st);
      mf_kernel<<<g2, kPipeThreads, kMfSmem, st>>>(cs, cb, L.hdr, L.partials, g1, 1, loss);
    }
  } else {
    const size_t n4 = (size_t)R->n * 64 / 4;
    const int g2 = (int)std::max<size_t>(1, std::min<size_t>((n4 + 255) / 256, (size_t)sms * 4));
    {
      KTimer t_mf_sumsq("mf_sumsq", st);
      sumsq_kernel<<<g2, 256, 0, st>>>(reinterpret_cast<const float4*>(V), n4, lambda, L.hdr,
                                       L.partials, g1, loss);
    }
  }
  return cudaGetLastError();
}

}  // namespace sdad
