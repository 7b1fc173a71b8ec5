/*
 * sdad.h -- loss and full gradient of sparse tensor expressions on one GPU.
 *
 * C ABI of libsdad.so (NVIDIA GB300, sm_103a).  Each entry point evaluates one
 * differentiated expression: it takes sparse operands plus dense factors and
 * returns the loss together with every requested gradient, in one call.
 * Expressions: five losses (least squares, logistic regression, matrix
 * factorisation, CP decomposition, graph propagation), the paper's matrix
 * kernels SMVM, SMMM and BATAX (gradients, and BATAX's Jacobian), and the
 * forward mode of the five losses (the directional derivative along a
 * tangent).
 *
 * Semantics follow Shaikhha, Huot, Hashemian, "Differentiable Programming for
 * Sparse Tensors" (arXiv 2303.07030):
 *   - gradient e x, one call per differentiated expression (Sec. 4.3);
 *   - the gradient with respect to a sparse operand is indexed by that
 *     operand's own keys (onehot[tensor n] x iterates over the keys of x,
 *     Fig. "api"), so it is returned as a value array in the operand's storage
 *     order and is never densified;
 *   - sparse operands are held in the physical formats of the paper's storage
 *     specifications: CSR (len, pos, idx, val), its column-major twin CSC, and
 *     COO (Fig. "storage_spec", Sec. 5.3);
 *   - destination-passing style: the caller owns and passes every output and
 *     the workspace; the library allocates nothing (Sec. 5.5).
 *
 * Conventions shared by all entry points
 *   - Indices are int32, values float32, losses float64.  nnz must be below
 *     2^31 (SDAD_ERR_OVERFLOW otherwise).
 *   - Dense matrices are row-major with the stated widths.
 *   - "device" pointers live in GPU memory of the current device; "host"
 *     pointers in ordinary CPU memory.
 *   - Device entry points check their arguments on the host first; on any
 *     error they return before enqueuing work and touch no output.  Work is
 *     enqueued on `stream` (a cudaStream_t, NULL = legacy default stream) and
 *     runs asynchronously; outputs are valid once the stream reaches that
 *     point.  A condition a kernel detects (a bounded wait that ran out) is
 *     recorded in the workspace and reported by sdad_check().
 *   - Gradient outputs are overwritten, not accumulated.  A NULL gradient
 *     pointer means "not requested"; the loss is always produced.
 *   - Arrays read by the streaming kernels (CSR/CSC index and value arrays,
 *     COO arrays) and every dense factor must start on a 16-byte boundary
 *     (SDAD_ERR_ALIGN otherwise).
 *   - The contents of device index arrays are not re-validated on the GPU:
 *     pointer arrays must be non-decreasing from 0 to nnz and every index in
 *     range, as the host builders below guarantee (they return SDAD_ERR_INDEX
 *     for input that breaks this).  Device arrays that break it give
 *     undefined results.
 */
#ifndef SDAD_H
#define SDAD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t sdad_status;

enum {
  SDAD_OK = 0,
  SDAD_ERR_NULL = -1,        /* a required pointer is NULL                     */
  SDAD_ERR_SHAPE = -2,       /* negative or inconsistent sizes                  */
  SDAD_ERR_INDEX = -3,       /* an index out of range, or unsorted input        */
  SDAD_ERR_ALIGN = -4,       /* a device array not 16-byte aligned              */
  SDAD_ERR_OVERFLOW = -5,    /* a count does not fit in int32                   */
  SDAD_ERR_WORKSPACE = -6,   /* workspace NULL or smaller than required         */
  SDAD_ERR_CUDA = -7,        /* a CUDA runtime call failed                      */
  SDAD_ERR_TIMEOUT = -8,     /* a device-side wait hit its iteration limit      */
  SDAD_ERR_UNSUPPORTED = -9  /* width/rank not supported, or no sm_103 device   */
};

/* Static string naming a status code (never NULL). */
const char* sdad_status_string(sdad_status s);

/* Version of the library as major*10000 + minor*100 + patch. */
int32_t sdad_version(void);

/* ========================================================================
 * Host builders (host memory in, caller-allocated host memory out).
 * Physical formats of Fig. "storage_spec" (Sec. 5.3); a COO with repeated
 * keys denotes the dictionary in which their values add (Sec. 5.5, res[k] += v).
 * ======================================================================== */

/* COO -> CSR.  Sorts by (row, col) and sums the values of duplicate keys
 * (in double precision, in input order, then rounded to float).
 *   m, n        matrix shape; nnz_in entries in row[], col[] (host)
 *   val         host values, or NULL to build the pattern only
 *   rowptr      out, host int32[m+1]
 *   colidx      out, host int32[nnz_in] (first *nnz_out entries written)
 *   val_out     out, host float[nnz_in], or NULL (ignored when val is NULL)
 *   nnz_out     out, number of distinct keys
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX (entry out of range),
 * SDAD_ERR_OVERFLOW (nnz_in >= 2^31). */
sdad_status sdad_csr_from_coo(int32_t m, int32_t n, int64_t nnz_in, const int32_t* row,
                              const int32_t* col, const float* val, int32_t* rowptr,
                              int32_t* colidx, float* val_out, int64_t* nnz_out);

/* CSR pattern -> CSC pattern plus the transpose permutation (the CSC
 * storage of Fig. "storage_spec", Sec. 5.3; a second physical format of the
 * same dictionary).
 *   rowptr[m+1], colidx[nnz] (host, sorted within rows, no duplicates)
 *   colptr      out, host int32[n+1]
 *   rowidx      out, host int32[nnz]; rows ascending within each column
 *   perm        out, host int32[nnz]; CSC slot q holds the key of CSR slot
 *               perm[q], so val_csc[q] = val[perm[q]] (the CSC value array the
 *               transposed kernels read)
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX (column out of range,
 * rowptr not monotone, or columns not strictly increasing within a row). */
sdad_status sdad_csr_transpose(int32_t m, int32_t n, int64_t nnz, const int32_t* rowptr,
                               const int32_t* colidx, int32_t* colptr, int32_t* rowidx,
                               int32_t* perm);

/* Ranking of the columns of a sparse matrix by their number of keys (a
 * further physical numbering of the same dictionary, in the spirit of Sec.
 * 5.3's separation of storage from expression; not in the paper): the
 * columns with most keys get the smallest ranks (equal counts: ascending
 * column).  The ranked ids are an alternative physical column numbering of
 * the same matrix: the key (i, j) at CSR slot p is stored as (i, rank(j)),
 * the slot order is unchanged.  Kernels that gather a dense vector by column
 * (x, w) or accumulate into one (A^T r) then find the most used entries at
 * the start of the vector, where a few cache lines or a shared-memory copy
 * hold them (sdad_csr.rcolidx / rankcol).
 *   n           number of columns; colidx[nnz] host, each in [0, n)
 *   rcolidx     out, host int32[nnz]: rcolidx[p] = rank(colidx[p])
 *   rankcol     out, host int32[n]:   rankcol[rank(j)] = j
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX, SDAD_ERR_OVERFLOW. */
sdad_status sdad_csr_rank_columns(int32_t n, int64_t nnz, const int32_t* colidx,
                                  int32_t* rcolidx, int32_t* rankcol);

/* Row-blocked CSC twin of some or all columns (a blocked storage of the same
 * dictionary, Sec. 5.3; not one of the paper's formats): the keys of those columns
 * sorted by (row block, column, row), where a row block is 2^rb_log2
 * consecutive rows.  Each key is packed in 32 bits as
 *   key = (h << rb_log2) | (row - first row of its block),
 * h the column's position in `cols` (its id when cols is NULL), so a column
 * pass can keep one block of the row vector in shared memory and read column
 * positions without a pointer array.  Each block's keys start at a multiple
 * of SDAD_BCSC_CHUNK; its range is padded to such a multiple with copies of
 * its last key that map to no CSR slot (their value is 0).
 *   rowptr[m+1], colidx[nnz]      host CSR pattern (any column order in a row)
 *   rb_log2   in [SDAD_BCSC_MIN_LOG2, SDAD_BCSC_MAX_LOG2]
 *   ncols, cols  host int32[ncols], strictly ascending column ids in [0, n):
 *             the columns this twin holds; cols NULL: all n columns (ncols
 *             must then be n).  ncols <= 2^(32-rb_log2), so h packs.
 *   blkptr    out, host int32[nb+1], nb = ceil(m / 2^rb_log2): block b holds
 *             keys [blkptr[b], blkptr[b+1])
 *   bkey      out, host uint32[*bnnz]
 *   bperm     out, host int32[*bnnz]: the CSR slot of each key, -1 for padding
 *             (the blocked value array is val[bperm], 0 where bperm < 0)
 *   bnnz      out, the padded key count.  With blkptr, bkey or bperm NULL only
 *             *bnnz is computed (sizes query).
 * With a column list, the keys of the other columns go to a plain CSC twin of
 * their own (sdad_csr_transpose_rest): a column pass then reads the columns
 * with many keys per row block from the blocked twin and the rest from the
 * plain one.
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX (a column out of
 * range, or cols not strictly ascending), SDAD_ERR_OVERFLOW,
 * SDAD_ERR_UNSUPPORTED (rb_log2 out of range, or ncols too large to pack). */
#define SDAD_BCSC_CHUNK 1024
#define SDAD_BCSC_MIN_LOG2 4
#define SDAD_BCSC_MAX_LOG2 15
sdad_status sdad_csr_block_transpose(int32_t m, int32_t n, int64_t nnz, const int32_t* rowptr,
                                     const int32_t* colidx, int32_t rb_log2, int32_t ncols,
                                     const int32_t* cols, int32_t* blkptr, uint32_t* bkey,
                                     int32_t* bperm, int64_t* bnnz);

/* CSC twin (Sec. 5.3) of the keys whose column is NOT in `cols` (the complement of a
 * column-restricted sdad_csr_block_transpose).
 *   rowptr[m+1], colidx[nnz]      host CSR pattern (sorted within rows)
 *   ncols, cols  host int32[ncols], strictly ascending column ids in [0, n)
 *   colptr    out, host int32[n+1]; the listed columns are empty
 *   rowidx    out, host int32[*rnnz]; rows ascending within each column
 *   perm      out, host int32[*rnnz]: the CSR slot of each key
 *   rnnz      out, the number of such keys.  With rowidx or perm NULL only
 *             colptr and *rnnz are computed (sizes query).
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX. */
sdad_status sdad_csr_transpose_rest(int32_t m, int32_t n, int64_t nnz, const int32_t* rowptr,
                                    const int32_t* colidx, int32_t ncols, const int32_t* cols,
                                    int32_t* colptr, int32_t* rowidx, int32_t* perm,
                                    int64_t* rnnz);

/* Mode index of a 3-way COO tensor (the tensor dictionaries of Sec. 3,
 * stored as COO, Sec. 5.3): a stable sort of the entries by their
 * mode-`mode` index.
 *   i, j, k     host int32[nnz]; dims[3] the tensor shape
 *   perm        out, host int32[nnz]: entry numbers, grouped by idx_mode,
 *               ascending entry number inside a group
 *   segptr      out, host int32[dims[mode]+1]: group s is perm[segptr[s] ..
 *               segptr[s+1])
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_INDEX, SDAD_ERR_OVERFLOW. */
sdad_status sdad_coo3_mode_index(int64_t nnz, const int32_t* i, const int32_t* j,
                                 const int32_t* k, const int32_t dims[3], int32_t mode,
                                 int32_t* perm, int32_t* segptr);

/* Device gather of 32-bit words through a permutation: out[q] = src[perm[q]]
 * for q < count, and 0 where perm[q] is outside [0, n_src) (the -1 that
 * sdad_csr_block_transpose writes for padding keys).  It forms, on the
 * device and on `stream`, the value copies that the physical formats hold
 * beside the CSR values (Sec. 5.3: one dictionary, several storages):
 *   val_csc  = gather(val, perm of sdad_csr_transpose / _transpose_rest)
 *   bcsc_val = gather(val, bperm of sdad_csr_block_transpose)
 *   sval[m], sidx[m][c] = gather(val, idx[c]; perm_m of sdad_coo3_mode_index)
 * so a caller whose sparse values change between calls (a step that updates
 * A itself) refreshes the twins without a host round trip.  The index arrays
 * of the twins do not change with the values.
 *   src[n_src], perm[count], out[count]: device, 16-byte aligned; out must not
 *   overlap src or perm.
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE, SDAD_ERR_ALIGN, SDAD_ERR_UNSUPPORTED
 * (not sm_103), SDAD_ERR_CUDA. */
sdad_status sdad_gather_by_perm(const void* src, int64_t n_src, const int32_t* perm,
                                int64_t count, void* out, void* stream);

/* ========================================================================
 * Device operands (non-owning descriptors of device arrays)
 * ======================================================================== */

/* Sparse matrix A (m x n) in CSR, with an optional CSC twin of the same
 * pattern (needed by the transposed paths and by the column passes). */
typedef struct {
  int32_t m, n;
  int64_t nnz;
  const int32_t* rowptr;   /* device int32[m+1]                          */
  const int32_t* colidx;   /* device int32[nnz], 16-byte aligned         */
  const float* val;        /* device float[nnz], 16-byte aligned         */
  const int32_t* colptr;   /* device int32[n+1], or NULL                 */
  const int32_t* rowidx;   /* device int32[nnz], or NULL                 */
  const float* val_csc;    /* device float[nnz] = val[perm[.]], or NULL  */
  /* optional ranked column numbering (sdad_csr_rank_columns), used by the
   * least-squares and logistic passes when present: both arrays, or neither
   * (an array of zero length may be NULL) */
  const int32_t* rcolidx;  /* device int32[nnz], 16-byte aligned, or NULL */
  const int32_t* rankcol;  /* device int32[n], or NULL                    */
  /* optional row-blocked CSC twin (sdad_csr_block_transpose), used by the
   * least-squares and logistic column passes when present: */
  int32_t bcsc_log2;        /* rb_log2 it was built with, or 0 (absent)     */
  int64_t bcsc_nnz;         /* padded key count                            */
  const int32_t* bcsc_ptr;  /* device int32[nb+1]                          */
  const uint32_t* bcsc_key; /* device uint32[bcsc_nnz], 16-byte aligned     */
  const float* bcsc_val;    /* device float[bcsc_nnz] = val[bperm] (0 pad)  */
  /* columns of the blocked twin: bcsc_cols NULL = all n (bcsc_ncols is then
   * ignored).  With a list, the CSC twin above (colptr, rowidx, val_csc)
   * must be the twin of the OTHER columns (sdad_csr_transpose_rest), holding
   * bcsc_rest_nnz keys; the column pass reads both. */
  int32_t bcsc_ncols;
  const int32_t* bcsc_cols; /* device int32[bcsc_ncols], ascending, or NULL */
  int64_t bcsc_rest_nnz;
  /* optional transpose permutation of the CSC twin (sdad_csr_transpose's
   * perm: CSC slot q holds the key of CSR slot csc_perm[q]); with it the
   * graph loss computes dA in its column pass instead of re-reading P */
  const int32_t* csc_perm;  /* device int32[nnz], or NULL */
} sdad_csr;

/* Sparse matrix A (m x n) as COO entries in any order (Sec. 5.3, Fig.
 * "storage_spec": the coordinate format of the same dictionary).  Entries may
 * repeat a key; their values add. */
typedef struct {
  int32_t m, n;
  int64_t nnz;
  const int32_t* row;   /* device int32[nnz], each in [0, m) */
  const int32_t* col;   /* device int32[nnz], each in [0, n) */
  const float* val;     /* device float[nnz]                 */
} sdad_coo;

/* 3-way sparse tensor in COO plus one mode-sorted copy per mode. */
typedef struct {
  int32_t dims[3];
  int64_t nnz;
  const int32_t* idx[3];   /* device int32[nnz] each (entry order)               */
  const float* val;        /* device float[nnz]                                  */
  /* mode-m sorted copy: entries in the order perm_m of sdad_coo3_mode_index */
  const int32_t* sidx[3][3]; /* sidx[m][c] = idx[c][perm_m[.]], device         */
  const float* sval[3];      /* sval[m] = val[perm_m[.]], device                */
  const int32_t* sperm[3];   /* sperm[m] = perm_m (entry number), device        */
  const int32_t* segptr[3];  /* segptr[m] of sdad_coo3_mode_index, device        */
} sdad_coo3;

/* How the transposed product (A^T times a dense operand) is formed. */
typedef enum {
  SDAD_T_AUTO = 0,    /* library's choice, by measured throughput: where both
                         modes are possible, the first AUTO call on an operand
                         (identified by its device, two of its device pointers,
                         its sizes and the outputs asked for) runs both twice,
                         times them with events on the call's stream (it waits
                         for the stream) and keeps the faster; later AUTO calls
                         run the kept one.  Inside a stream capture no timing
                         is done: a choice made earlier, else CSC (ATOMIC for
                         CP).  Where only one mode's arrays are given, that one */
  SDAD_T_CSC = 1,     /* atomic-free column pass over the CSC twin (deterministic) */
  SDAD_T_ATOMIC = 2   /* scattered from the row pass with atomic adds          */
} sdad_tmode;

/* ========================================================================
 * Workspace
 * ======================================================================== */

typedef enum {
  SDAD_EXPR_LSQ = 1,
  SDAD_EXPR_LOGREG = 2,
  SDAD_EXPR_MF = 3,
  SDAD_EXPR_CP3 = 4,
  SDAD_EXPR_GNN = 5,
  SDAD_EXPR_SMVM = 6,
  SDAD_EXPR_SMMM = 7,
  SDAD_EXPR_BATAX = 8
} sdad_expr;

/* Bytes of device workspace one call of `expr` needs for operand shape
 * (rows, cols, nnz) and dense width `width` (MF: k, CP: rank, GNN: f_out;
 * ignored otherwise).  For CP, rows = cols = max(dims).  For SMMM the shape
 * is A's (rows = m, cols = kk, nnz = keys of A).  The workspace must
 * start on a 256-byte boundary and its header must be zero before the first
 * call (sdad_workspace_init).  One workspace serves one call at a time:
 * calls that share it must be ordered (e.g. on one stream).
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE. */
sdad_status sdad_workspace_bytes(int32_t expr, int32_t rows, int32_t cols, int64_t nnz,
                                 int32_t width, size_t* bytes);

/* Zeroes the 256-byte header of a workspace (enqueued on `stream`).  A
 * workspace must start with a zero header before its first use (this call,
 * or any zero fill); the library keeps the header consistent afterwards.
 * Errors: SDAD_ERR_NULL, SDAD_ERR_ALIGN, SDAD_ERR_CUDA. */
sdad_status sdad_workspace_init(void* ws, void* stream);

/* Waits for `stream`, then reads and clears the device status word held in
 * `ws`: SDAD_OK, or SDAD_ERR_TIMEOUT when a bounded device wait gave up
 * (outputs of that call are then unspecified), or SDAD_ERR_CUDA. */
sdad_status sdad_check(void* ws, void* stream);

/* Sets how many times each bounded device wait of the calls that use `ws`
 * polls before it gives up (Sec. 5 of the paper has no counterpart: this is
 * failure detection of the GPU path).  polls < 0 restores the default
 * (2^22 polls); 0 <= polls < 2^32 - 1 sets that limit, 0 meaning that every
 * wait gives up at once.  A wait that gives up records SDAD_ERR_TIMEOUT
 * (read by sdad_check); the kernel still waits, with the default limit, for
 * the copies and tensor-core work it issued itself before it returns.
 * Enqueued on `stream` (a one-thread kernel writes the header field);
 * sdad_workspace_init restores the default.
 * Errors: SDAD_ERR_NULL, SDAD_ERR_ALIGN, SDAD_ERR_SHAPE, SDAD_ERR_CUDA. */
sdad_status sdad_workspace_set_wait_limit(void* ws, int64_t polls, void* stream);

/* ========================================================================
 * Loss + gradient entry points.  All pointers are device pointers.
 * ======================================================================== */

/* Least squares  L = 1/2 ||A x - y||^2   (A: m x n).  One call of
 * `gradient e x` (Sec. 4.3) for each differentiated operand; the gradient
 * w.r.t. A lives on keys(A) (Fig. "api"), exact up to rounding (Sec. 6).
 *   x[n], y[m]       inputs (may be NULL when n = 0, resp. m = 0)
 *   loss             out, one double
 *   dx[n]            out, dL/dx = A^T r with r = A x - y       (nullable)
 *   dA_val[nnz]      out, dL/dA on keys(A) in CSR order:       (nullable)
 *                    dA_val[p] = r_i x_j for the key (i, j) at slot p
 *   tmode            SDAD_T_CSC needs A's CSC twin
 * With ranked columns (A->rcolidx, A->rankcol) the row pass reads rcolidx
 * instead of colidx and gathers from a copy of x in ranked order (most used
 * entries first, so they share cache lines); outputs are in the original
 * column order.  SDAD_T_CSC is bit-reproducible; SDAD_T_ATOMIC adds the
 * transposed product with warp-aggregated float atomics (order not fixed);
 * AUTO is measured (see sdad_tmode), or ATOMIC without a column structure.
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA/UNSUPPORTED. */
sdad_status sdad_lsq_grad(const sdad_csr* A, const float* x, const float* y, double* loss,
                          float* dx, float* dA_val, sdad_tmode tmode, void* ws, size_t ws_bytes,
                          void* stream);

/* Least squares as sdad_lsq_grad over a COO operand in entry order (no CSR,
 * no twins, no sorting): z = A x by an entry scatter, r = z - y and the loss
 * by a row pass, then dA and dx = A^T r by a second entry pass.  dA_val[nnz]
 * is in the entries' order (an entry that repeats a key gets the key's
 * gradient r_i x_j).  The scatters use warp-aggregated float atomics, so dx
 * (and z) are order-dependent within rounding; the loss is summed in a fixed
 * order.  Indices are checked on the device: an entry out of range is skipped
 * and SDAD_ERR_INDEX is recorded for sdad_check.  Workspace: as
 * sdad_lsq_grad (sdad_workspace_bytes(SDAD_EXPR_LSQ, m, n, nnz, 0)).
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA. */
sdad_status sdad_lsq_coo_grad(const sdad_coo* A, const float* x, const float* y, double* loss,
                              float* dx, float* dA_val, void* ws, size_t ws_bytes, void* stream);

/* Logistic regression over m samples (rows of X: m x n), labels y in [0, 1]
 * (gradient on keys as Sec. 4.3 / Fig. "api"; the SMVM-like product of Sec. 7.1):
 *   z = X w,  L = (1/m) sum_i [log(1 + e^{z_i}) - y_i z_i]
 *   dw[n]     out, X^T (sigmoid(z) - y) / m                     (nullable)
 *   dX_val    out, on keys(X) in CSR order: (sigmoid(z_i) - y_i) w_j / m
 *                                                               (nullable)
 * tmode and ranked columns as for sdad_lsq_grad. */
sdad_status sdad_logreg_grad(const sdad_csr* X, const float* w, const float* y, double* loss,
                             float* dw, float* dX_val, sdad_tmode tmode, void* ws,
                             size_t ws_bytes, void* stream);

/* Matrix factorisation on the observed keys of R (m x n) (sums over the
 * dictionary's keys, Sec. 3; dR on keys(R), Sec. 4.3):
 *   L = sum_{(i,j) in keys(R)} (R_ij - U_i . V_j)^2 + lambda (|U|^2 + |V|^2)
 *   U[m x k], V[n x k] inputs; k = 64 in this version
 *   dU[m x k], dV[n x k] out (nullable); dR_val[nnz] out, 2 e_ij in CSR order
 *   (nullable).  dV: SDAD_T_CSC runs a column pass over R's CSC twin
 *   (bit-reproducible); SDAD_T_ATOMIC is one pass over the CSR that gathers
 *   each V row once and scatters dV with vector atomics (with ranked columns,
 *   rcolidx / rankcol, the 64 most used columns are summed in shared memory
 *   first; order of additions not fixed); AUTO is measured (see sdad_tmode),
 *   or ATOMIC when R has no CSC twin. */
sdad_status sdad_mf_grad(const sdad_csr* R, const float* U, const float* V, int32_t k,
                         float lambda, double* loss, float* dU, float* dV, float* dR_val,
                         sdad_tmode tmode, void* ws, size_t ws_bytes, void* stream);

/* CP decomposition of a 3-way tensor T (dims d0 x d1 x d2, nnz entries)
 * (a sum over the tensor dictionary's entries, Sec. 3; dT on its keys, Sec. 4.3):
 *   e_n = T_n - sum_r A_{i r} B_{j r} C_{k r},   L = sum_n e_n^2
 *   A[d0 x R], B[d1 x R], C[d2 x R] inputs; R = 32 in this version
 *   dA, dB, dC out (nullable): dA_i = -2 sum_{n: i_n = i} e_n (B_j * C_k), ...
 *   dT_val[nnz] out, 2 e_n in entry order (nullable)
 *   SDAD_T_CSC: one atomic-free pass per requested factor over that mode's
 *   sorted copy (sidx, sval, segptr; sperm too when dT_val is wanted);
 *   bit-reproducible.
 *   SDAD_T_ATOMIC: one pass over the entry-order arrays (idx, val) that
 *   scatters all three factor gradients with atomic adds (order not fixed).
 *   SDAD_T_AUTO: measured (see sdad_tmode) when both layouts are given,
 *   else the one given. */
sdad_status sdad_cp3_grad(const sdad_coo3* T, const float* A, const float* B, const float* C,
                          int32_t rank, double* loss, float* dA, float* dB, float* dC,
                          float* dT_val, sdad_tmode tmode, void* ws, size_t ws_bytes,
                          void* stream);

/* Graph propagation  Y = A (H W),  L = 1/2 ||Y - Z||^2   (A: m x n graph)
 * (the GNN use case of Sec. 9; dA on keys(A), Sec. 4.3):
 *   H[n x f_in], W[f_in x f_out], Z[m x f_out]; f_in = 128, f_out = 64 here
 *   dA_val[nnz] out, on keys(A): D_i . (H W)_j with D = Y - Z  (nullable)
 *   dH[n x f_in] out, (A^T D) W^T                              (nullable)
 *   dW[f_in x f_out] out, H^T (A^T D)                          (nullable)
 *   G = A^T D (for dH, dW): SDAD_T_CSC walks A's CSC twin (bit-reproducible);
 *   SDAD_T_ATOMIC scatters it from the CSR with vector atomics (no CSC twin
 *   needed; order not fixed); AUTO is measured (see sdad_tmode), or ATOMIC
 *   when A has no CSC twin.
 *   With A->csc_perm (16-byte aligned) and SDAD_T_CSC, dA is computed in the
 *   column pass over the CSC twin, which gathers D anyway; otherwise in the
 *   forward pass with a second gather of (H W) rows. */
sdad_status sdad_gnn_grad(const sdad_csr* A, const float* H, const float* W, const float* Z,
                          int32_t f_in, int32_t f_out, double* loss, float* dA_val, float* dH,
                          float* dW, sdad_tmode tmode, void* ws, size_t ws_bytes, void* stream);

/* Forward mode (the tensorized forward-mode rules of Sec. 4.2 with a real
 * tangent): the loss and its directional derivative along a tangent of the
 * inputs, in one pass over A's rows.
 *   x_t[n]        tangent of x (resp. w)                        (nullable: 0)
 *   A_t_val[nnz]  tangent of A's values, on keys(A) in CSR order (nullable: 0)
 *   loss, loss_t  out, one double each: L and dL[x_t, A_t] = <grad L, tangent>
 * The workspace is sdad_workspace_bytes(SDAD_EXPR_LSQ, resp. SDAD_EXPR_LOGREG,
 * m, n, nnz, 0); A needs no CSC twin.  Reproducible bit for bit.
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA. */
sdad_status sdad_lsq_jvp(const sdad_csr* A, const float* x, const float* y, const float* x_t,
                         const float* A_t_val, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream);
sdad_status sdad_logreg_jvp(const sdad_csr* X, const float* w, const float* y, const float* w_t,
                            const float* X_t_val, double* loss, double* loss_t, void* ws,
                            size_t ws_bytes, void* stream);

/* Forward mode of matrix factorisation (k = 64) and CP (rank 32): the loss
 * and its directional derivative along a tangent of the sparse operand's
 * values (R_t_val on keys(R) in CSR order, T_t_val in entry order) and of the
 * factors (U_t, V_t; A_t, B_t, C_t: same shapes as the factors, 16-byte
 * aligned).  Every tangent is nullable (zero).  One pass over the keys (MF:
 * CSR arrays only; CP: the entry arrays only).  Workspace: as sdad_mf_grad /
 * sdad_cp3_grad.  Reproducible bit for bit.
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA/UNSUPPORTED (k, rank). */
sdad_status sdad_mf_jvp(const sdad_csr* R, const float* U, const float* V, int32_t k,
                        float lambda, const float* R_t_val, const float* U_t, const float* V_t,
                        double* loss, double* loss_t, void* ws, size_t ws_bytes, void* stream);
sdad_status sdad_cp3_jvp(const sdad_coo3* T, const float* A, const float* B, const float* C,
                         int32_t rank, const float* T_t_val, const float* A_t, const float* B_t,
                         const float* C_t, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream);

/* Forward mode of the graph propagation loss (f_in = 128, f_out = 64):
 *   L = 1/2 |A (H W) - Z|^2 and its directional derivative L' along a tangent
 *   of A's values (A_t_val on keys(A), CSR order), of H (H_t, n x 128) and of
 *   W (W_t, 128 x 64), by the tensorized forward rules of Sec. 4.2 with a
 *   real tangent: P' = H' W + H W' (one two-source tensor-core product),
 *   Y' = A' P + A P',
 *   L' = sum_i (Y_i - Z_i) . Y'_i.  Every tangent is nullable (zero); dense
 *   arrays 16-byte aligned.  One pass over the CSR (no CSC twin needed).
 *   Workspace: as sdad_gnn_grad.  Reproducible bit for bit.
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA/UNSUPPORTED (widths). */
sdad_status sdad_gnn_jvp(const sdad_csr* A, const float* H, const float* W, const float* Z,
                         int32_t f_in, int32_t f_out, const float* A_t_val, const float* H_t,
                         const float* W_t, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream);

/* ========================================================================
 * The paper's matrix kernels (Sec. 7.1), each differentiated with respect to
 * the operand the paper names.  All pointers are device pointers; A needs
 * its CSC twin (colptr, val_csc; BATAX also rowidx).  Every result is
 * bit-reproducible (fixed addition orders, no atomics).
 * ======================================================================== */

/* SMVM  f = sum_{i,j} A(i,j) X(j)  (A: m x n).
 *   X[n]      input (may be NULL when n = 0)
 *   f         out, one double
 *   dX[n]     out, df/dX = A^T 1: the column sums of A         (nullable)
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA. */
sdad_status sdad_smvm_grad(const sdad_csr* A, const float* X, double* f, float* dX, void* ws,
                           size_t ws_bytes, void* stream);

/* SMMM  f = sum_{i,k,j} A(i,k) B(k,j)  (A: m x kk with its CSC twin, B: kk x n).
 *   f          out, one double
 *   dB_val     out, df/dB on keys(B) in B's CSR order: the key (k, j) at
 *              slot p gets sum_i A(i,k), the k-th column sum of A (nullable)
 * The workspace is sized for A (SDAD_EXPR_SMMM, rows m, cols kk, nnz of A).
 * Errors: NULL/SHAPE (A->n != B->m)/ALIGN/OVERFLOW/WORKSPACE/CUDA. */
sdad_status sdad_smmm_grad(const sdad_csr* A, const sdad_csr* B, double* f, float* dB_val,
                           void* ws, size_t ws_bytes, void* stream);

/* Pattern of A^T A (host builder, two-phase): the pairs (j, k) of columns
 * that some row of A holds together, whatever the values.  It is the
 * pattern of the BATAX Jacobian beta A^T A.
 *   rowptr[m+1], colidx[nnz]   host CSR pattern of A (sorted within rows)
 *   jrowptr    out, host int32[n+1]
 *   jcolidx    out, host int32[*jnnz], ascending within each row; NULL: only
 *              jrowptr and *jnnz are computed (sizes query)
 *   jnnz       out, the number of pairs
 * Errors: NULL/SHAPE/INDEX/OVERFLOW (more than 2^31 - 1 pairs). */
sdad_status sdad_csr_gram_pattern(int32_t m, int32_t n, int64_t nnz, const int32_t* rowptr,
                                  const int32_t* colidx, int32_t* jrowptr, int32_t* jcolidx,
                                  int64_t* jnnz);

/* BATAX  f(j) = sum_{i,k} beta A(i,j) A(i,k) X(k), i.e. f = beta A^T A X
 * (A: m x n, with its CSC twin).
 *   X[n]       input
 *   f[n]       out (nullable)
 *   jrowptr[n+1], jcolidx[jnnz]   device copies of sdad_csr_gram_pattern(A)
 *   J_val[jnnz] out, df/dX = beta A^T A on that pattern: entry (j, k) =
 *              beta sum_i A(i,j) A(i,k), the terms added in ascending i
 *              (nullable; then the pattern may be NULL)
 * Errors: NULL/SHAPE/ALIGN/OVERFLOW/WORKSPACE/CUDA. */
sdad_status sdad_batax_grad(const sdad_csr* A, const float* X, float beta, float* f,
                            const int32_t* jrowptr, const int32_t* jcolidx, int64_t jnnz,
                            float* J_val, void* ws, size_t ws_bytes, void* stream);

/* Least squares as sdad_lsq_grad, for callers that cannot allocate device
 * memory or pass a workspace (for example code running under a memory
 * allocator it does not own, such as a framework's caching pool or a host
 * that reserves all device memory at start-up).  The paper has no
 * counterpart; this is a deployment convenience.
 *   Layouts: the plain CSR, and in SDAD_T_CSC / AUTO mode with dx the plain
 *   CSC twin (colptr, rowidx, val_csc).  The ranked column numbering and a
 *   row-blocked twin are ignored; a matrix that carries a row-blocked twin
 *   but no plain CSC twin for every column (a split twin, or a blocked twin
 *   alone) is refused in CSC mode with SDAD_ERR_UNSUPPORTED, although
 *   sdad_lsq_grad accepts it.
 *   Scratch: a fixed 8 MiB array compiled into the library, present on every
 *   device that loads it until the process exits.  A problem needs about
 *   66 KiB + 4 m + 12 nnz / 256 bytes of it (each region rounded up to 256
 *   bytes); one that needs more than 8 MiB is rejected with
 *   SDAD_ERR_WORKSPACE before any device work (at 50M keys that leaves room
 *   for about 1.49M rows).
 *   The call allocates nothing (no cudaMalloc/cudaFree).  Its first call on a
 *   device looks up the array's device address (cudaGetSymbolAddress); make
 *   that first call before any stream capture.  Each call clears the part of
 *   the array that must start at zero, on `stream`.
 *   All calls share the array: calls whose work overlaps on the GPU race.
 *   Device-side conditions (a bounded wait that ran out) are not reported.
 * Errors: as sdad_lsq_grad, SDAD_ERR_WORKSPACE as above. */
sdad_status sdad_lsq_grad_noalloc(const sdad_csr* A, const float* x, const float* y,
                                  double* loss, float* dx, float* dA_val, sdad_tmode tmode,
                                  void* stream);

/* ========================================================================
 * Per-kernel timing (benchmarking aid; not thread-safe)
 * When enabled, every kernel an entry point launches is bracketed by two CUDA
 * events recorded on the call's stream (no host synchronisation); records
 * accumulate until sdad_timing_reset().  Off by default.
 * ======================================================================== */
sdad_status sdad_timing_enable(int32_t on);
sdad_status sdad_timing_reset(void);
int32_t sdad_timing_count(void);
/* Kernel name (static string) and duration in milliseconds of record i;
 * waits for the record's end event.  Errors: SDAD_ERR_SHAPE (i out of range),
 * SDAD_ERR_NULL, SDAD_ERR_CUDA. */
sdad_status sdad_timing_get(int32_t i, const char** name, float* ms);

/* Measurement aid (the paper has no counterpart): enqueues a kernel of
 * `blocks` CTAs x 256 threads, each thread running 16 independent FP32 FMA
 * chains `iters` steps long, and stores the FLOPs it performs in *flops
 * (host).  Timed by the caller with events on `stream`, it gives the FP32
 * FMA rate against which the arithmetic-bound kernels are reported.
 *   out[blocks*256]  device, overwritten (keeps the work observable)
 * Errors: SDAD_ERR_NULL, SDAD_ERR_SHAPE (blocks or iters <= 0),
 * SDAD_ERR_UNSUPPORTED (not sm_103), SDAD_ERR_CUDA. */
sdad_status sdad_probe_fma(float* out, int32_t blocks, int32_t iters, double* flops,
                           void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SDAD_H */
