// internal.h -- launchers shared between the C-ABI layer and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "sdad.h"

namespace sdad {

struct WsHeader;

// Number of SMs of the current device (cached per device).
int device_sm_count();
// Raises `func`'s dynamic shared-memory limit to `bytes` on the current
// device, once per (function, device); thread-safe.
cudaError_t ensure_dynamic_smem(const void* func, int bytes);

// Workspace carved into named regions (all 256-byte aligned).
struct WsLayout {
  WsHeader* hdr;
  double* partials;   // kMaxPartials doubles
  float* rowvec;      // scalar per row (lsq, logreg, batax)       [rows]
  float* colsum;      // smvm/smmm: column sums of A               [cols]
  double* sink;       // a double no caller reads (sums of passes that have none)
  float* vr;          // lsq/logreg, ranked columns: x[rankcol]    [cols]   (NULL: no ranking)
  float* vacc;        // lsq/logreg, ranked: A^T r accumulator     [cols]
  float* bP;          // lsq/logreg, blocked CSC: segment sums     [nb x cols] (NULL: none)
  // lsq/logreg, blocked CSC: pieces of segments cut by its chunk boundaries
  // (per blocked chunk, as pfirst/plast/lastseg below)
  float* bpfirst;
  float* bplast;
  int* bfirstseg;
  int* blastseg;
  float* P;           // graph: H W                                [cols x f_out]
  float* D;           // graph: A (H W) - Z                        [rows x f_out]
  float* G;           // graph: A^T D                              [cols x f_out]
  float* dWpart;      // graph: per-CTA partial H^T G              [kDwParts x f_in x f_out]
  double* closs;      // graph: loss terms of the rows finished inside each chunk [chunks]
  int32_t* order;     // graph: the walks' chunk-group order, then its scratch    [4 x chunks]
  double* cltan;      // graph, forward mode: the L' terms of the rows finished inside each chunk
  float* tfirst;      // graph, forward mode: pieces of Y' (as pfirst / plast below)
  float* tlast;
  // pieces of segments cut by chunk boundaries (deterministic combination):
  float* pfirst;      // per chunk: the piece of the segment begun in an earlier chunk
  float* plast;       // per chunk: the piece of the segment that continues past it
  int* lastseg;       // per chunk: that continuing segment (begun in this chunk), or -1
  size_t bytes;
};

constexpr int kMinCap = 1024;        // smallest chunk size of the engine passes (piece slots)
constexpr int kScalarMinCap = 256;   // smallest chunk of the lsq/logreg column pass

constexpr int kDwParts = 304;

// Computes the layout for an expression; ws may be NULL (sizes only).
// ranked_cols: room for the ranked-column path of lsq/logreg.  For lsq/logreg
// a nonzero width is the rb_log2 of a row-blocked CSC twin to make room for.
WsLayout ws_layout(int expr, int32_t rows, int32_t cols, int64_t nnz, int32_t width, void* ws,
                   bool ranked_cols = true);

// The CSR carries the ranked column numbering (sdad_csr_rank_columns).
inline bool csr_ranked(const sdad_csr* A) { return A->rankcol || A->rcolidx; }
// The CSR carries a row-blocked CSC twin (sdad_csr_block_transpose).
inline bool csr_blocked(const sdad_csr* A) { return A->bcsc_log2 > 0; }
// ... of some columns only; the CSC twin then holds the others.
inline bool csr_split(const sdad_csr* A) { return csr_blocked(A) && A->bcsc_cols; }

// lsq/logreg: whether the transposed product runs as a column pass over the
// CSC twin (else it is scattered from the row pass).
bool scalar_uses_csc(const sdad_csr* A, bool want_dvec, sdad_tmode tmode);


cudaError_t run_scalar(int expr, const sdad_csr* A, const float* xin, const float* y,
                       double* loss, float* dvec, float* dA, sdad_tmode tmode,
                       const WsLayout& L, cudaStream_t st);

// Column pass over A's CSC twin holding nnz keys: out = A^T rvec, or the
// column sums when rvec is NULL (out is zeroed first; deterministic).
cudaError_t col_pass(const sdad_csr* A, int64_t nnz, const float* rvec, float* out,
                     const WsLayout& L, cudaStream_t st);
// Row passes of the paper's matrix kernels: SMMM over B (f, dB on B's keys)
// and BATAX's r = beta A X (no scalar; `sink` takes the row kernel's sum).
cudaError_t smmm_rows(const sdad_csr* B, const float* colsum, double* f, float* dB,
                      const WsLayout& L, cudaStream_t st);
cudaError_t batax_rows(const sdad_csr* A, const float* X, float beta, float* r, double* sink,
                       const WsLayout& L, cudaStream_t st);
// Forward mode of least squares / logistic regression (k_jvp.cu): the loss
// and its derivative along the tangent (vt of the dense vector, valt of A's
// values; NULL = zero).
cudaError_t run_jvp(int expr, const sdad_csr* A, const float* v, const float* y, const float* vt,
                    const float* valt, double* loss, double* loss_t, const WsLayout& L,
                    cudaStream_t st);
cudaError_t run_mf_jvp(const sdad_csr* R, const float* U, const float* V, float lambda,
                       const float* valt, const float* Ut, const float* Vt, double* loss,
                       double* loss_t, const WsLayout& L, cudaStream_t st);
cudaError_t run_cp3_jvp(const sdad_coo3* T, const float* A, const float* B, const float* C,
                        const float* Tt, const float* At, const float* Bt, const float* Ct,
                        double* loss, double* loss_t, const WsLayout& L, cudaStream_t st);
// SMVM / SMMM / BATAX (k_paper.cu).
cudaError_t run_smvm(const sdad_csr* A, const float* X, double* f, float* dX, const WsLayout& L,
                     cudaStream_t st);
cudaError_t run_smmm(const sdad_csr* A, const sdad_csr* B, double* f, float* dB,
                     const WsLayout& L, cudaStream_t st);
cudaError_t run_batax(const sdad_csr* A, const float* X, float beta, float* f,
                      const int32_t* jrowptr, const int32_t* jcolidx, float* J_val,
                      const WsLayout& L, cudaStream_t st);

cudaError_t run_mf(const sdad_csr* R, const float* U, const float* V, float lambda,
                   double* loss, float* dU, float* dV, float* dR, sdad_tmode tmode,
                   const WsLayout& L, cudaStream_t st);

cudaError_t run_cp3(const sdad_coo3* T, const float* A, const float* B, const float* C,
                    double* loss, float* dA, float* dB, float* dC, float* dT, sdad_tmode tmode,
                    const WsLayout& L, cudaStream_t st);

cudaError_t run_lsq_coo(const sdad_coo* A, const float* x, const float* y, double* loss,
                        float* dx, float* dA, const WsLayout& L, cudaStream_t st);

cudaError_t run_gnn_jvp(const sdad_csr* A, const float* H, const float* W, const float* Z,
                        const float* valt, const float* Ht, const float* Wt, double* loss,
                        double* loss_t, const WsLayout& L, cudaStream_t st);

cudaError_t run_gnn(const sdad_csr* A, const float* H, const float* W, const float* Z,
                    double* loss, float* dA, float* dH, float* dW, bool atomic,
                    const WsLayout& L, cudaStream_t st);

// The forward-mode walk over the CSR (graph loss): per chunk, the L and L'
// terms of its finished rows (L.closs, L.cltan) and the pieces of Y and Y' of
// its cut rows; hdr->work[0] must be zero on entry.
cudaError_t run_gnn_jvp_walk(const sdad_csr* A, const float* valt, const float* P,
                             const float* Pt, const float* Z, const WsLayout& L, cudaStream_t st);

// Dense projection kernels (graph loss): P = H W;  dH = G W^T and per-CTA
// partials of H^T G;  dW = sum of the partials.
cudaError_t dense_proj_fwd(const float* H, const float* W, float* P, int n, WsHeader* hdr,
                           cudaStream_t st);
// P = H W + H2 W2 in one sweep (the forward mode's P' = H' W + H W')
cudaError_t dense_proj_fwd2(const float* H, const float* W, const float* H2, const float* W2,
                            float* P, int n, WsHeader* hdr, cudaStream_t st);
cudaError_t dense_proj_bwd(const float* H, const float* W, const float* G, float* dH,
                           float* dWpart, float* dW, int n, WsHeader* hdr, cudaStream_t st);

// Brackets the kernel launched in its scope with timing events when
// sdad_timing_enable(1) is in effect.
class KTimer {
 public:
  KTimer(const char* name, cudaStream_t st);
  ~KTimer();
 private:
  int slot_;
  cudaStream_t st_;
};

// Small helpers.
cudaError_t zero_f32(float* p, size_t count, cudaStream_t st);

// Argument checks shared by the entry points.
constexpr int64_t kMaxNnz = (int64_t(1) << 31) - (int64_t(1) << 16);
bool a16(const void* p);
bool a8(const void* p);
sdad_status map_cuda(cudaError_t e);
sdad_status check_csr(const sdad_csr* A, bool need_csc);
sdad_status check_device();   // current device is sm_103

}  // namespace sdad
