// k_gnn_jvp.cu -- forward mode of the graph propagation loss (f_out = 64).
//
// The loss L = 1/2 |A P - Z|^2 with P = H W, and its derivative along a
// tangent (A' on A's keys, H', W'), by the forward rules of Sec. 4 with a
// real tangent: each value carries its tangent through the same steps.
//   P' = H' W + H W'                               (two tensor-core products)
//   Y_i  = sum_p A_ip P_j,   Y'_i = sum_p (A'_ip P_j + A_ip P'_j)
//   D_i  = Y_i - Z_i,        L = 1/2 sum_i |D_i|^2,   L' = sum_i D_i . Y'_i
// Rows without keys add 1/2 |Z_i|^2 to L and nothing to L'.
// Kernel sequence: P (and P') on the tensor cores; the rows without keys; the
// reverse-mode forward walk's machinery carrying a tangent (run_gnn_jvp_walk
// in k_gnn.cu: half a warp per key, P_j and P'_j gathered, chunk groups from
// a work counter in the longest-first order, per-chunk sums of L and L'); a
// fix kernel that completes the rows cut by chunk boundaries and adds the
// per-chunk and per-CTA sums in a fixed order.  Reproducible bit for bit.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdad {

constexpr int kGjChunk = kMinCap;
constexpr int kGjThreads = 256;
constexpr int kGjWarps = kGjThreads / 32;
constexpr int kTangentSlots = kMaxPartials / 2;   // L' partials follow L's

__device__ __forceinline__ float2 gj_ld2(const float* base, int r, int lane) {
  return __ldg(reinterpret_cast<const float2*>(base + (size_t)r * 64) + lane);
}

struct GjPieces {
  float* __restrict__ yfirst;   // [chunks x 64]: parts of Y of a row begun earlier
  float* __restrict__ ylast;    // [chunks x 64]: parts of Y of the row continuing past
  float* __restrict__ tfirst;   // the same for Y'
  float* __restrict__ tlast;
  int* __restrict__ lastseg;
};

// Stores this CTA's (L, L') sums at slot `slot`.
__device__ __forceinline__ void gj_publish(double L, double Lt, double* partials, int slot,
                                           double* red) {
  const double cL = block_sum_d(L, red);
  const double cLt = block_sum_d(Lt, red);
  if (threadIdx.x == 0) {
    partials[slot] = cL;
    partials[kTangentSlots + slot] = cLt;
  }
}

// rows without keys: L += 1/2 |Z_r|^2 (one warp per 32 rows)
__global__ void __launch_bounds__(kGjThreads)
    gnn_jvp_empty_kernel(const int32_t* __restrict__ rowptr, int m, const float* __restrict__ Z,
                         WsHeader* hdr, double* partials) {
  __shared__ double red[kGjWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (blockIdx.x == 0 && threadIdx.x == 0) hdr->work[0] = 0;   // the walk's group counter
  const int gw = blockIdx.x * kGjWarps + warp, nw = gridDim.x * kGjWarps;
  double L = 0.0;
  for (int blk = gw; blk < (m + 31) / 32; blk += nw) {
    const int r = blk * 32 + lane;
    const bool e = r < m && __ldg(rowptr + r) == __ldg(rowptr + r + 1);
    unsigned todo = __ballot_sync(FULL_MASK, e);
    float lf = 0.f;   // this lane's part (elements 2 lane, 2 lane + 1 of each row), in row order
    while (todo) {    // warp-uniform: eight rows' loads in flight at a time
      int rr[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        rr[u] = todo ? __ffs(todo) - 1 : -1;
        if (todo) todo &= todo - 1;
      }
      float2 z[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        z[u] = rr[u] >= 0 ? gj_ld2(Z, blk * 32 + rr[u], lane) : make_float2(0.f, 0.f);
#pragma unroll
      for (int u = 0; u < 8; ++u) lf = fmaf(z[u].x, z[u].x, fmaf(z[u].y, z[u].y, lf));
    }
    L += 0.5 * (double)lf;
  }
  gj_publish(L, 0.0, partials, blockIdx.x, red);
}

// rows cut by chunk boundaries, then the totals: the last CTA adds every
// CTA's sums (slots [0, nslots) of L and of L') in slot order
__global__ void __launch_bounds__(kGjThreads)
    gnn_jvp_fix_kernel(const int32_t* __restrict__ rowptr, int nchunks, GjPieces pc,
                       const float* __restrict__ Z, const double* __restrict__ closs,
                       const double* __restrict__ cltan, WsHeader* hdr, double* partials,
                       int first_slot, double* loss, double* loss_t) {
  __shared__ double red[kGjWarps];
  __shared__ bool s_last;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kGjWarps + warp, nw = gridDim.x * kGjWarps;
  double L = 0.0, Lt = 0.0;
  // the walk's per-chunk sums: this CTA adds its own slice, in order
  for (int ch = blockIdx.x * blockDim.x + threadIdx.x; ch < nchunks; ch += gridDim.x * blockDim.x) {
    L += closs[ch];
    Lt += cltan[ch];
  }
  for (int ch = gw; ch < nchunks; ch += nw) {
    const int s = __ldg(pc.lastseg + ch);
    if (s < 0) continue;   // warp-uniform
    const int c1 = (__ldg(rowptr + s + 1) - 1) / kGjChunk;
    float2 y = gj_ld2(pc.ylast, ch, lane), t = gj_ld2(pc.tlast, ch, lane);
    for (int cc = ch + 1; cc <= c1; ++cc) {
      const float2 a = gj_ld2(pc.yfirst, cc, lane), b = gj_ld2(pc.tfirst, cc, lane);
      y.x += a.x;
      y.y += a.y;
      t.x += b.x;
      t.y += b.y;
    }
    const float2 z = gj_ld2(Z, s, lane);
    const float2 d = make_float2(y.x - z.x, y.y - z.y);
    L += 0.5 * (double)fmaf(d.x, d.x, d.y * d.y);
    Lt += (double)fmaf(d.x, t.x, d.y * t.y);
  }
  gj_publish(L, Lt, partials, first_slot + blockIdx.x, red);
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&hdr->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int nslots = first_slot + gridDim.x;
  const volatile double* pv = partials;
  double a = 0.0, b = 0.0;
  for (int i = threadIdx.x; i < nslots; i += blockDim.x) {
    a += pv[i];
    b += pv[kTangentSlots + i];
  }
  a = block_sum_d(a, red);
  b = block_sum_d(b, red);
  if (threadIdx.x == 0) {
    *loss = a;
    *loss_t = b;
    hdr->ticket = 0;
  }
}

cudaError_t run_gnn_jvp(const sdad_csr* A, const float* H, const float* W, const float* Z,
                        const float* valt, const float* Ht, const float* Wt, double* loss,
                        double* loss_t, const WsLayout& L, cudaStream_t st) {
  const int sms = device_sm_count();
  const int m = A->m, n = A->n, nnz = (int)A->nnz;
  const int nchunks = nnz <= 0 ? 1 : (nnz + kGjChunk - 1) / kGjChunk;
  cudaError_t e;
  // P = H W; P' = H' W + H W' (in the G buffer), one sweep over H' and H
  if ((e = dense_proj_fwd(H, W, L.P, n, L.hdr, st)) != cudaSuccess) return e;
  const float* Pt = nullptr;
  if (Ht && Wt) e = dense_proj_fwd2(Ht, W, H, Wt, L.G, n, L.hdr, st);
  else if (Ht) e = dense_proj_fwd(Ht, W, L.G, n, L.hdr, st);
  else if (Wt) e = dense_proj_fwd(H, Wt, L.G, n, L.hdr, st);
  if (e != cudaSuccess) return e;
  if (Ht || Wt) Pt = L.G;
  const GjPieces pc{L.pfirst, L.plast, L.tfirst, L.tlast, L.lastseg};
  const int ge = std::max(1, std::min((m + 255) / 256, sms * 4));
  {
    KTimer t("gnn_jvp_empty", st);
    gnn_jvp_empty_kernel<<<ge, kGjThreads, 0, st>>>(A->rowptr, m, Z, L.hdr, L.partials);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if ((e = run_gnn_jvp_walk(A, valt, L.P, Pt, Z, L, st)) != cudaSuccess) return e;
  const int gf = std::max(1, std::min((nchunks + kGjWarps - 1) / kGjWarps, sms * 4));
  static_assert(kTangentSlots >= 152 * 8, "partial slots of the empty and fix kernels");
  {
    KTimer t("gnn_jvp_fix", st);
    gnn_jvp_fix_kernel<<<gf, kGjThreads, 0, st>>>(A->rowptr, nchunks, pc, Z, L.closs, L.cltan,
                                                   L.hdr, L.partials, ge, loss, loss_t);
  }
  return cudaGetLastError();
}

}  // namespace sdad
