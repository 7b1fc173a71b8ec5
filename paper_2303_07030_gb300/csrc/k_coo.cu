// k_coo.cu -- least squares over a sparse operand stored as COO, in entry
// order (Sec. 5.3: the same expression over another physical storage of
// the same dictionary; the entries need no sorting and no CSR / CSC twin).
//
//   z_i  = sum over entries e with row i of val_e x_{col_e}   (entries scatter)
//   r_i  = z_i - y_i,  L = 1/2 sum_i r_i^2                    (row pass)
//   dA_e = r_{row_e} x_{col_e}                                (entry order)
//   dx_j = sum over entries e with column j of val_e r_{row_e}
// Entries may repeat a key: their values add (dictionary +=), and each such
// entry gets the key's gradient.  The two entry passes scatter with
// warp-aggregated atomic adds (lanes that hit the same row or column sum
// first), so their order of additions is not fixed; the loss sum is.  An
// entry whose row or column is out of range is skipped and reported as
// SDAD_ERR_INDEX in the workspace status (sdad_check).
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdad {

constexpr int kCooThreads = 256;

__global__ void __launch_bounds__(kCooThreads)
    coo_z_kernel(const int32_t* __restrict__ row, const int32_t* __restrict__ col,
                 const float* __restrict__ val, int64_t nnz, int m, int n,
                 const float* __restrict__ x, float* __restrict__ z, WsHeader* hdr) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  // every lane of a warp runs the same number of steps (aggregated atomics)
  const int64_t base0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
  for (int64_t b = base0; b < nnz; b += stride) {
    const int64_t e = b + (threadIdx.x & 31);
    bool act = e < nnz;
    int i = act ? __ldg(row + e) : -1;
    const int j = act ? __ldg(col + e) : 0;
    if (act && (i < 0 || i >= m || j < 0 || j >= n)) {   // reported, and the entry skipped
      set_status(hdr, SDAD_ERR_INDEX);
      act = false;
      i = -1;
    }
    const float v = act ? __ldg(val + e) * __ldg(x + j) : 0.f;
    agg_atomic_add(z, i, v, FULL_MASK);
  }
}

// r = z - y in place, loss = 1/2 sum r^2 (fixed order: per CTA, then CTAs)
__global__ void __launch_bounds__(kCooThreads)
    coo_rows_kernel(float* __restrict__ z, const float* __restrict__ y, int m, WsHeader* hdr,
                    double* partials, double* loss) {
  __shared__ double red[kCooThreads / 32];
  double s = 0.0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < m; i += gridDim.x * blockDim.x) {
    const float r = z[i] - __ldg(y + i);
    z[i] = r;
    s += 0.5 * (double)r * (double)r;
  }
  const double cta = block_sum_d(s, red);
  publish_loss(cta, hdr, partials, 0, true, 1.0, loss, red);
}

__global__ void __launch_bounds__(kCooThreads)
    coo_grad_kernel(const int32_t* __restrict__ row, const int32_t* __restrict__ col,
                    const float* __restrict__ val, int64_t nnz, int m, int n,
                    const float* __restrict__ x,
                    const float* __restrict__ r, float* __restrict__ dx, float* __restrict__ dA) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t base0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
  for (int64_t b = base0; b < nnz; b += stride) {
    const int64_t e = b + (threadIdx.x & 31);
    bool act = e < nnz;
    const int i = act ? __ldg(row + e) : 0;
    int j = act ? __ldg(col + e) : -1;
    if (act && (i < 0 || i >= m || j < 0 || j >= n)) {   // already reported by coo_z_kernel
      act = false;
      j = -1;
    }
    const float ri = act ? __ldg(r + i) : 0.f;
    if (act && dA) dA[e] = ri * __ldg(x + j);
    if (dx) agg_atomic_add(dx, j, act ? __ldg(val + e) * ri : 0.f, FULL_MASK);
  }
}

cudaError_t run_lsq_coo(const sdad_coo* A, const float* x, const float* y, double* loss,
                        float* dx, float* dA, const WsLayout& L, cudaStream_t st) {
  const int sms = device_sm_count();
  const int64_t nnz = A->nnz;
  const int ge = (int)std::max<int64_t>(1, std::min<int64_t>((nnz + kCooThreads - 1) / kCooThreads,
                                                             (int64_t)sms * 8));
  cudaError_t e;
  if ((e = zero_f32(L.rowvec, (size_t)A->m, st)) != cudaSuccess) return e;
  if (dx && (e = zero_f32(dx, (size_t)A->n, st)) != cudaSuccess) return e;
  if (nnz > 0) {
    KTimer t("coo_z", st);
    coo_z_kernel<<<ge, kCooThreads, 0, st>>>(A->row, A->col, A->val, nnz, A->m, A->n, x,
                                             L.rowvec, L.hdr);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  {
    const int gr = std::max(1, std::min((A->m + kCooThreads - 1) / kCooThreads, sms * 4));
    KTimer t("coo_rows", st);
    coo_rows_kernel<<<gr, kCooThreads, 0, st>>>(L.rowvec, y, A->m, L.hdr, L.partials, loss);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (nnz > 0 && (dx || dA)) {
    KTimer t("coo_grad", st);
    coo_grad_kernel<<<ge, kCooThreads, 0, st>>>(A->row, A->col, A->val, nnz, A->m, A->n, x,
                                                L.rowvec, dx, dA);
  }
  return cudaGetLastError();
}

}  // namespace sdad
