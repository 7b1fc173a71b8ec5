// k_paper.cu -- the paper's matrix kernels (Sec. 7.1), differentiated with
// respect to the operand the paper names:
//
//   SMVM   f = sum_{i,j} A(i,j) X(j)          df/dX   = A^T 1 (column sums)
//   SMMM   f = sum_{i,k,j} A(i,k) B(k,j)      df/dB   = { (k,j) -> sum_i A(i,k) }
//   BATAX  f = beta A^T A X  (a vector)       df/dX   = beta A^T A (a matrix)
//
// The column sums come from the column pass over A's CSC twin without a
// gather; SMMM's row pass over B and BATAX's A X are the row kernel of
// k_scalar.cu with their own finish.  The BATAX Jacobian is a sparse product
// on a pattern built on the host (sdad_csr_gram_pattern): row j of
// beta A^T A is beta sum_{i in column j} A(i,j) A(i,:), taken one row i at a
// time in ascending i, the lanes of a warp over the keys of row i (distinct
// columns, so distinct outputs), into a per-warp accumulator in shared
// memory (gram_kernel says how a key finds its place).
// Every addition order is fixed: the results are bit-reproducible.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sdad {

// f = sum_j x_j y_j in double, per CTA in a fixed order, then over the CTAs.
__global__ void __launch_bounds__(256)
    dot_kernel(const float* __restrict__ x, const float* __restrict__ y, int n, WsHeader* hdr,
               double* partials, double* out) {
  __shared__ double red[8];
  double s = 0.0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    s += (double)__ldg(x + i) * (double)__ldg(y + i);
  const double cta = block_sum_d(s, red);
  publish_loss(cta, hdr, partials, 0, true, 1.0, out, red);
}

constexpr int kGramWarps = 8;
constexpr int kGramBuf = 1024;        // floats of shared memory per warp
constexpr int kGramCap = kGramBuf / 2;  // searched rows: columns + sums in the buffer

// Three ways to place a key (i, k) of A in output row j (columns sorted):
// a row whose columns span at most kGramBuf values keeps a dense
// accumulator over [kmin, kmax] in shared memory (one add per key, the sums
// gathered at the end by column); a longer span with at most kGramCap
// columns binary-searches the columns held in shared memory; a longer row
// searches and accumulates in place in J_val (only this warp writes it).
__global__ void __launch_bounds__(kGramWarps * 32)
    gram_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                const float* __restrict__ val, const int32_t* __restrict__ colptr,
                const int32_t* __restrict__ rowidx, const float* __restrict__ val_csc, int n,
                const int32_t* __restrict__ jrowptr, const int32_t* __restrict__ jcolidx,
                float beta, float* __restrict__ jval) {
  __shared__ float sbuf[kGramWarps][kGramBuf];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = gridDim.x * kGramWarps;
  float* buf = sbuf[warp];
  for (int j = blockIdx.x * kGramWarps + warp; j < n; j += nw) {   // warp-uniform
    const int js = __ldg(jrowptr + j), len = __ldg(jrowptr + j + 1) - js;
    if (len <= 0) continue;
    const int kmin = __ldg(jcolidx + js), span = __ldg(jcolidx + js + len - 1) - kmin + 1;
    const int mode = span <= kGramBuf ? 0 : (len <= kGramCap ? 1 : 2);
    int32_t* scol = reinterpret_cast<int32_t*>(buf);
    const int32_t* cols = mode == 1 ? scol : jcolidx + js;
    float* acc = mode == 0 ? buf : (mode == 1 ? buf + kGramCap : jval + js);
    const int clear = mode == 0 ? span : len;
    for (int t = lane; t < clear; t += 32) {
      if (mode == 1) scol[t] = __ldg(jcolidx + js + t);
      acc[t] = 0.f;
    }
    __syncwarp();
    // the rows i holding column j, ascending, 32 at a time: lane l holds row
    // t = l's start, end and A(i,j); the keys of the rows then go by items
    // of up to 32 (item: keys [base, min(base + 32, e)) of row t), the next
    // item's keys loaded before the current one is added
    const int q1 = __ldg(colptr + j + 1);
    for (int qb = __ldg(colptr + j); qb < q1; qb += 32) {
      const int nq = min(32, q1 - qb);
      int my_s = 0, my_e = 0;
      float my_a = 0.f;
      if (lane < nq) {
        const int i = __ldg(rowidx + qb + lane);
        my_a = __ldg(val_csc + qb + lane);
        my_s = __ldg(rowptr + i);
        my_e = __ldg(rowptr + i + 1);
      }
      int t = 0;
      int base = __shfl_sync(FULL_MASK, my_s, 0), e = __shfl_sync(FULL_MASK, my_e, 0);
      float a = __shfl_sync(FULL_MASK, my_a, 0);
      int k = -1;
      float b = 0.f;
      if (base + lane < e) {
        k = __ldg(colidx + base + lane);
        b = __ldg(val + base + lane);
      }
      while (t < nq) {   // warp-uniform
        int t2 = t, base2 = base + 32, e2 = e;
        float a2 = a;
        if (base2 >= e) t2 = t + 1;   // the next row
        const int ns = __shfl_sync(FULL_MASK, my_s, t2 & 31);
        const int ne = __shfl_sync(FULL_MASK, my_e, t2 & 31);
        const float na = __shfl_sync(FULL_MASK, my_a, t2 & 31);
        if (t2 != t) {
          base2 = ns;
          e2 = ne;
          a2 = na;
        }
        int k2 = -1;
        float b2 = 0.f;
        if (t2 < nq && base2 + lane < e2) {
          k2 = __ldg(colidx + base2 + lane);
          b2 = __ldg(val + base2 + lane);
        }
        if (k >= 0) {
          int at = k - kmin;   // (a key off the row's pattern is dropped)
          if (mode != 0) {     // the place of k among the row's columns
            int lo = 0, hi = len - 1;
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (cols[mid] < k)
                lo = mid + 1;
              else
                hi = mid;
            }
            at = lo;
          }
          if (mode != 0 || (unsigned)at < (unsigned)span) acc[at] += a * b;
        }
        __syncwarp();   // the next row may add to the same places
        t = t2;
        base = base2;
        e = e2;
        a = a2;
        k = k2;
        b = b2;
      }
    }
    for (int t = lane; t < len; t += 32) {
      const int c = mode == 0 ? __ldg(jcolidx + js + t) - kmin : t;
      jval[js + t] = (unsigned)c < (unsigned)(mode == 0 ? span : len) ? beta * acc[c] : 0.f;
    }
    __syncwarp();
  }
}

cudaError_t run_smvm(const sdad_csr* A, const float* X, double* f, float* dX, const WsLayout& L,
                     cudaStream_t st) {
  float* cs = dX ? dX : L.colsum;
  cudaError_t e = col_pass(A, A->nnz, nullptr, cs, L, st);
  if (e != cudaSuccess) return e;
  const int grid = std::max(1, std::min((A->n + 255) / 256, device_sm_count() * 4));
  {
    KTimer t("smvm_dot", st);
    dot_kernel<<<grid, 256, 0, st>>>(X, cs, A->n, L.hdr, L.partials, f);
  }
  return cudaGetLastError();
}

cudaError_t run_smmm(const sdad_csr* A, const sdad_csr* B, double* f, float* dB,
                     const WsLayout& L, cudaStream_t st) {
  cudaError_t e = col_pass(A, A->nnz, nullptr, L.colsum, L, st);
  if (e != cudaSuccess) return e;
  return smmm_rows(B, L.colsum, f, dB, L, st);
}

cudaError_t run_batax(const sdad_csr* A, const float* X, float beta, float* f,
                      const int32_t* jrowptr, const int32_t* jcolidx, float* J_val,
                      const WsLayout& L, cudaStream_t st) {
  cudaError_t e;
  if (f) {   // f = A^T (beta A X)
    if ((e = batax_rows(A, X, beta, L.rowvec, L.sink, L, st)) != cudaSuccess) return e;
    if ((e = col_pass(A, A->nnz, L.rowvec, f, L, st)) != cudaSuccess) return e;
  }
  if (J_val && A->n > 0) {
    // one output row per warp: the rows of A^T A differ in work, and the
    // block scheduler hands a finished SM the next CTA (measured on the consph
    // stand-in: 0.354 ms, against 0.379 ms with 16 CTAs per SM striding over
    // the rows and 0.42 ms with the resident CTAs only)
    const int grid = std::max(1, (A->n + kGramWarps - 1) / kGramWarps);
    KTimer t("batax_gram", st);
    gram_kernel<<<grid, kGramWarps * 32, 0, st>>>(A->rowptr, A->colidx, A->val, A->colptr,
                                                  A->rowidx, A->val_csc, A->n, jrowptr, jcolidx,
                                                  beta, J_val);
  }
  return cudaGetLastError();
}

}  // namespace sdad
