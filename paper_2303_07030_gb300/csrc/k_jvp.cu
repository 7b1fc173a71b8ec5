// k_jvp.cu -- forward mode: a loss with its directional derivative along a
// tangent of its inputs.  Least squares and logistic regression, along a
// tangent (v', A') of the dense vector and of the sparse operand's values (the tensorized forward-mode rules of Sec. 4
// with a real tangent: (a v_j)' = a v_j' + a' v_j, (op e)' = op'(e) e'):
//   z  = A v,  z' = A v' + A' v            (per row)
//   least squares: r = z - y,  L = 1/2 sum r^2,            L' = sum r z'
//   logistic:      L = (1/m) sum softplus(z) - y z,        L' = (1/m) sum (s(z) - y) z'
// One pass over the CSR rows, laid out like the gradient's row pass (eight
// lanes per row, four rows per warp step, six keys per lane issued together,
// z and z' of row r0 + l handed to lane l); both sums are per lane in row
// order, then per CTA and over the CTAs in a fixed order: reproducible.
// Matrix factorisation and CP have their own passes below (mf_jvp_kernel,
// cp3_jvp_kernel), one per key of R / entry of T.
#include <algorithm>

#include "common.cuh"
#include "halfwarp.cuh"
#include "internal.h"

namespace sdad {

constexpr int kJvpThreads = 256;
constexpr int kJvpWarps = kJvpThreads / 32;
constexpr int kJvpLanes = 8;
constexpr int kJvpSlots = 6;

// Both sums of a forward-mode pass: per CTA in a fixed order (partials[b]
// and partials[gridDim.x + b]), then the last CTA adds the CTAs in order and
// writes them scaled.  Called by every thread of the CTA.
__device__ __forceinline__ void publish_pair(double L, double Lt, WsHeader* hdr, double* partials,
                                             double scale, double* loss, double* loss_t,
                                             double* red) {
  __shared__ bool s_last;
  const double cL = block_sum_d(L, red);
  const double cLt = block_sum_d(Lt, red);
  if (threadIdx.x == 0) {
    partials[blockIdx.x] = cL;
    partials[gridDim.x + blockIdx.x] = cLt;
    __threadfence();
    s_last = atomicAdd(&hdr->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const volatile double* pv = partials;
  double sL = 0.0, sLt = 0.0;
  for (int i = threadIdx.x; i < (int)gridDim.x; i += blockDim.x) {
    sL += pv[i];
    sLt += pv[gridDim.x + i];
  }
  const double tL = block_sum_d(sL, red);
  const double tLt = block_sum_d(sLt, red);
  if (threadIdx.x == 0) {
    *loss = tL * scale;
    *loss_t = tLt * scale;
    hdr->ticket = 0;
  }
}

template <bool LOGREG, bool HAS_VT, bool HAS_AT>
__global__ void __launch_bounds__(kJvpThreads)
    jvp_row_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                   const float* __restrict__ val, const float* __restrict__ valt, int m,
                   const float* __restrict__ v, const float* __restrict__ vt,
                   const float* __restrict__ y, WsHeader* hdr, double* partials, double scale,
                   double* loss, double* loss_t) {
  __shared__ double red[kJvpWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = lane / kJvpLanes, gl = lane % kJvpLanes;
  const int nblk = (m + 31) / 32;
  const int gw = blockIdx.x * kJvpWarps + warp, nw = gridDim.x * kJvpWarps;
  const int b0 = (int)(((long long)nblk * gw) / nw);
  const int b1 = (int)(((long long)nblk * (gw + 1)) / nw);
  double L = 0.0, Lt = 0.0;
  for (int b = b0; b < b1; ++b) {
    const int row = b * 32 + lane;
    const bool valid = row < m;
    const int p0 = valid ? __ldg(rowptr + row) : 0;
    const int p1 = valid ? __ldg(rowptr + row + 1) : 0;
    const float yrow = valid ? __ldg(y + row) : 0.f;
    float zrow = 0.f, ztrow = 0.f;
#pragma unroll 1
    for (int sub = 0; sub < 32 / 4; ++sub) {
      const int t = sub * 4 + grp;
      const int rs = __shfl_sync(FULL_MASK, p0, t), re = __shfl_sync(FULL_MASK, p1, t);
      float z = 0.f, zt = 0.f;
      for (int q0 = rs + gl; q0 < re; q0 += kJvpSlots * kJvpLanes) {
        int j[kJvpSlots];
        float a[kJvpSlots], at[kJvpSlots];
#pragma unroll
        for (int u = 0; u < kJvpSlots; ++u) {
          const int q = q0 + u * kJvpLanes;
          const bool in = q < re;
          j[u] = in ? __ldg(colidx + q) : 0;
          a[u] = in ? __ldg(val + q) : 0.f;
          at[u] = (HAS_AT && in) ? __ldg(valt + q) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < kJvpSlots; ++u) {
          const bool in = q0 + u * kJvpLanes < re;
          const float x = in ? __ldg(v + j[u]) : 0.f;
          const float xt = (HAS_VT && in) ? __ldg(vt + j[u]) : 0.f;
          z += a[u] * x;
          if (HAS_VT) zt += a[u] * xt;
          if (HAS_AT) zt += at[u] * x;
        }
      }
      z = group_sum<kJvpLanes>(z);
      zt = group_sum<kJvpLanes>(zt);
      const int src = (lane & 3) * kJvpLanes;   // row sub * 4 + (lane & 3)
      const float zs = __shfl_sync(FULL_MASK, z, src), zts = __shfl_sync(FULL_MASK, zt, src);
      if ((lane >> 2) == sub) {
        zrow = zs;
        ztrow = zts;
      }
    }
    if (valid) {
      if (LOGREG) {
        const float e = expf(-fabsf(zrow));   // in (0, 1]
        const float tail = log1pf(e);
        const float sp_pos = fmaxf(zrow, 0.f) + tail, sp_neg = fmaxf(-zrow, 0.f) + tail;
        L += (double)((1.f - yrow) * sp_pos) + (double)(yrow * sp_neg);
        const float sig = zrow >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
        Lt += (double)(sig - yrow) * (double)ztrow;
      } else {
        const float r = zrow - yrow;
        L += 0.5 * (double)r * (double)r;
        Lt += (double)r * (double)ztrow;
      }
    }
  }
  publish_pair(L, Lt, hdr, partials, scale, loss, loss_t, red);
}

__device__ __forceinline__ float4 ld4(const float* p, size_t row, int width, int part) {
  return __ldg(reinterpret_cast<const float4*>(p + row * (size_t)width) + part);
}
__device__ __forceinline__ float4 ld4z(const float* p, size_t row, int width, int part) {
  return p ? ld4(p, row, width, part) : make_float4(0.f, 0.f, 0.f, 0.f);
}
__device__ __forceinline__ float dot4f(const float4& a, const float4& b) {
  return fmaf(a.w, b.w, fmaf(a.z, b.z, fmaf(a.y, b.y, a.x * b.x)));
}
__device__ __forceinline__ float4 mul4f(const float4& a, const float4& b) {
  return make_float4(a.x * b.x, a.y * b.y, a.z * b.z, a.w * b.w);
}

// Matrix factorisation, k = 64: a warp takes 1024-key chunks of R (CSR), row
// by row; U_i and U'_i are loaded once per row (half a warp holds a row, one
// float4 per lane), and the row's keys go eight at a time, half a warp per
// key: V_j and V'_j gathered, the eight dot products of each kind reduced
// together.  Per key
//   e = R - U_i . V_j,  e' = R' - (U'_i . V_j + U_i . V'_j),  L += e^2, L' += 2 e e'.
// Then the regulariser over the dense factors: lam (|U|^2 + |V|^2) and its
// tangent 2 lam (U . U' + V . V').  Per-lane sums in a fixed order:
// reproducible.
constexpr int kMfJvpChunk = 1024;
constexpr int kMfJvpPairs = 4;   // key pairs per batch
#ifndef SDAD_MFJVP_MINB
#define SDAD_MFJVP_MINB 3
#endif

__global__ void __launch_bounds__(kJvpThreads, SDAD_MFJVP_MINB)
    mf_jvp_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                  const float* __restrict__ val, const float* __restrict__ valt, int m, int n,
                  int nnz, const float* __restrict__ U, const float* __restrict__ V,
                  const float* __restrict__ Ut, const float* __restrict__ Vt, float lam,
                  WsHeader* hdr, double* partials, double* loss, double* loss_t) {
  __shared__ double red[kJvpWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int h = lane >> 4, sl = lane & 15;
  const int gw = blockIdx.x * kJvpWarps + warp, nw = gridDim.x * kJvpWarps;
  const int nchunks = (nnz + kMfJvpChunk - 1) / kMfJvpChunk;
  // after reduce_half over four values: lane (h, sl) with sl % 4 == 0 holds
  // the total of key 2 ((sl >> 2) & 3) + h of the batch
  const int kl = 2 * ((sl >> 2) & 3) + h;
  const bool holder = (sl & 3) == 0;
  double L = 0.0, Lt = 0.0;
  for (int ch = gw; ch < nchunks; ch += nw) {   // warp-uniform
    const int cs = ch * kMfJvpChunk, ce = min(cs + kMfJvpChunk, nnz);
    int r = warp_lower_bound(rowptr, 0, m + 1, cs + 1) - 1;   // the row of key cs
    int s0 = __ldg(rowptr + r), s1 = __ldg(rowptr + r + 1);
    while (true) {
      const int ps = max(s0, cs), pe = min(s1, ce);
      const float4 uv = ld4(U, r, sl);
      const float4 ut = Ut ? ld4(Ut, r, sl) : zero4();
      for (int pb = ps; pb < pe; pb += 2 * kMfJvpPairs) {
        const int nk = min(2 * kMfJvpPairs, pe - pb);
        const bool mine = lane < nk;
        const int jl = mine ? __ldg(colidx + pb + lane) : 0;
        const float al = mine ? __ldg(val + pb + lane) : 0.f;
        const float atl = (mine && valt) ? __ldg(valt + pb + lane) : 0.f;
        float4 x[kMfJvpPairs], xt[kMfJvpPairs];
#pragma unroll
        for (int u = 0; u < kMfJvpPairs; ++u) {
          const int kk = 2 * u + h;
          const int j = __shfl_sync(FULL_MASK, jl, kk);
          x[u] = kk < nk ? ld4(V, j, sl) : zero4();
          xt[u] = (kk < nk && Vt) ? ld4(Vt, j, sl) : zero4();
        }
        float t[kMfJvpPairs], tt[kMfJvpPairs];
#pragma unroll
        for (int u = 0; u < kMfJvpPairs; ++u) {
          t[u] = dot4(x[u], uv);
          tt[u] = dot4(x[u], ut) + dot4(xt[u], uv);
        }
        const float d = reduce_half(t, lane), dt = reduce_half(tt, lane);
        const float e = __shfl_sync(FULL_MASK, al, kl) - d;
        const float et = __shfl_sync(FULL_MASK, atl, kl) - dt;
        if (holder && kl < nk) {
          L += (double)e * (double)e;
          Lt += 2.0 * (double)e * (double)et;
        }
      }
      if (s1 >= ce) break;
      // the next row with keys: the one holding key s1
      r = warp_gallop_lower_bound(rowptr, r + 1, m + 1, s1 + 1) - 1;
      s0 = __ldg(rowptr + r);
      s1 = __ldg(rowptr + r + 1);
    }
  }
  // regulariser
  const long long t0 = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  const long long nt = (long long)gridDim.x * blockDim.x;
  double R = 0.0, Rt = 0.0;
  for (int which = 0; which < 2; ++which) {
    const float* F = which ? V : U;
    const float* Ft = which ? Vt : Ut;
    const long long n4 = (long long)(which ? n : m) * 16;
    for (long long t = t0; t < n4; t += nt) {
      const float4 f = __ldg(reinterpret_cast<const float4*>(F) + t);
      R += (double)dot4f(f, f);
      if (Ft) Rt += 2.0 * (double)dot4f(f, __ldg(reinterpret_cast<const float4*>(Ft) + t));
    }
  }
  publish_pair(L + (double)lam * R, Lt + (double)lam * Rt, hdr, partials, 1.0, loss, loss_t, red);
}

// CP decomposition, rank 32: four entries per warp step, eight lanes per
// entry (four of the 32 factor entries each).  Per entry
//   e = t - sum_r a b c,  e' = t' - sum_r (a' b c + a b' c + a b c'),
//   L += e^2,  L' += 2 e e'.
__global__ void __launch_bounds__(kJvpThreads)
    cp3_jvp_kernel(int nnz, const int32_t* __restrict__ I, const int32_t* __restrict__ J,
                   const int32_t* __restrict__ K, const float* __restrict__ T,
                   const float* __restrict__ Tt, const float* __restrict__ A,
                   const float* __restrict__ B, const float* __restrict__ C,
                   const float* __restrict__ At, const float* __restrict__ Bt,
                   const float* __restrict__ Ct, WsHeader* hdr, double* partials, double* loss,
                   double* loss_t) {
  __shared__ double red[kJvpWarps];
  const int lane = threadIdx.x & 31, slot = lane >> 3, sl = lane & 7;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  double L = 0.0, Lt = 0.0;
  for (int pb = gw * 4; pb < nnz; pb += nw * 4) {   // warp-uniform
    const int p = pb + slot;
    const bool act = p < nnz;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a, c = a, at = a, bt = a, ct = a;
    float t = 0.f, tt = 0.f;
    if (act) {
      const int i = __ldg(I + p), j = __ldg(J + p), k = __ldg(K + p);
      t = __ldg(T + p);
      tt = Tt ? __ldg(Tt + p) : 0.f;
      a = ld4(A, i, 32, sl);
      b = ld4(B, j, 32, sl);
      c = ld4(C, k, 32, sl);
      at = ld4z(At, i, 32, sl);
      bt = ld4z(Bt, j, 32, sl);
      ct = ld4z(Ct, k, 32, sl);
    }
    const float4 bc = mul4f(b, c);
    const float model = group_sum<8>(dot4f(a, bc));
    const float modelt = group_sum<8>(dot4f(at, bc) + dot4f(a, mul4f(bt, c)) +
                                      dot4f(a, mul4f(b, ct)));
    if (act && sl == 0) {
      const float e = t - model, et = tt - modelt;
      L += (double)e * (double)e;
      Lt += 2.0 * (double)e * (double)et;
    }
  }
  publish_pair(L, Lt, hdr, partials, 1.0, loss, loss_t, red);
}

cudaError_t run_mf_jvp(const sdad_csr* R, const float* U, const float* V, float lambda,
                       const float* valt, const float* Ut, const float* Vt, double* loss,
                       double* loss_t, const WsLayout& L, cudaStream_t st) {
  const int nchunks = (int)((R->nnz + kMfJvpChunk - 1) / kMfJvpChunk);
  // as many CTAs as are resident at once (the chunks are strided over the warps)
  int per_sm = 1;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, mf_jvp_kernel,
                                                                kJvpThreads, 0);
  if (e != cudaSuccess) return e;
  const int grid = std::max(1, std::min(std::max((nchunks + kJvpWarps - 1) / kJvpWarps,
                                                 (R->m + R->n + 255) / 256),
                                        std::min(device_sm_count() * std::max(per_sm, 1),
                                                 kMaxPartials / 2)));
  {
    KTimer t("mf_jvp", st);
    mf_jvp_kernel<<<grid, kJvpThreads, 0, st>>>(R->rowptr, R->colidx, R->val, valt, R->m, R->n,
                                                (int)R->nnz, U, V, Ut, Vt, lambda, L.hdr,
                                                L.partials, loss, loss_t);
  }
  return cudaGetLastError();
}

cudaError_t run_cp3_jvp(const sdad_coo3* T, const float* A, const float* B, const float* C,
                        const float* Tt, const float* At, const float* Bt, const float* Ct,
                        double* loss, double* loss_t, const WsLayout& L, cudaStream_t st) {
  const int nnz = (int)T->nnz;
  // as many CTAs as are resident at once (a grid-stride loop over uniform
  // entries: a second wave only lengthens the tail)
  int per_sm = 1;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, cp3_jvp_kernel,
                                                                kJvpThreads, 0);
  if (e != cudaSuccess) return e;
  const int grid = std::max(1, std::min((nnz + 31) / 32,
                                        std::min(device_sm_count() * std::max(per_sm, 1),
                                                 kMaxPartials / 2)));
  {
    KTimer t("cp3_jvp", st);
    cp3_jvp_kernel<<<grid, kJvpThreads, 0, st>>>(nnz, T->idx[0], T->idx[1], T->idx[2], T->val,
                                                 Tt, A, B, C, At, Bt, Ct, L.hdr, L.partials,
                                                 loss, loss_t);
  }
  return cudaGetLastError();
}

cudaError_t run_jvp(int expr, const sdad_csr* A, const float* v, const float* y, const float* vt,
                    const float* valt, double* loss, double* loss_t, const WsLayout& L,
                    cudaStream_t st) {
  const bool lr = expr == SDAD_EXPR_LOGREG;
  const int nblk = (A->m + 31) / 32;
  const int grid = std::max(1, std::min((nblk + kJvpWarps * 2 - 1) / (kJvpWarps * 2),
                                        kMaxPartials / 2));
  const double scale = lr ? 1.0 / (double)A->m : 1.0;
  const bool hv = vt != nullptr, ha = valt != nullptr && A->nnz > 0;
  auto go = [&](auto kern) {
    kern<<<grid, kJvpThreads, 0, st>>>(A->rowptr, A->colidx, A->val, valt, A->m, v, vt, y, L.hdr,
                                       L.partials, scale, loss, loss_t);
  };
  KTimer t(lr ? "logreg_jvp" : "lsq_jvp", st);
#define SDAD_JVP(LR)                                                       \
  (hv ? (ha ? go(jvp_row_kernel<LR, true, true>) : go(jvp_row_kernel<LR, true, false>)) \
      : (ha ? go(jvp_row_kernel<LR, false, true>) : go(jvp_row_kernel<LR, false, false>)))
  if (lr)
    SDAD_JVP(true);
  else
    SDAD_JVP(false);
#undef SDAD_JVP
  return cudaGetLastError();
}

}  // namespace sdad
