// api.cu -- the C ABI of libsdad: argument checks, workspace layout, launches.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <cstdint>
#include <cstring>
#include <vector>

#include "common.cuh"
#include "internal.h"
#include "sdad.h"

namespace sdad {

// ---------------------------------------------------------------------------
// device facts
// ---------------------------------------------------------------------------
cudaError_t ensure_dynamic_smem(const void* func, int bytes) {
  // (function, device) pairs already raised, under a lock: the attribute
  // belongs to the device, so a process that uses several GPUs sets it on each
  static std::mutex mu;
  static std::vector<std::pair<const void*, int>> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (const auto& d : done)
    if (d.first == func && d.second == dev) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done.emplace_back(func, dev);
  return e;
}

int device_sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (!cache[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
      v = 148;
    cache[dev] = v;
  }
  return cache[dev];
}

sdad_status check_device() {
  static int ok_cache[64] = {0};   // 0 unknown, 1 ok, -1 unsupported
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDAD_ERR_CUDA;
  if (dev < 0 || dev >= 64) return SDAD_ERR_UNSUPPORTED;
  if (!ok_cache[dev]) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return SDAD_ERR_CUDA;
    ok_cache[dev] = (major == 10 && minor == 3) ? 1 : -1;
  }
  return ok_cache[dev] == 1 ? SDAD_OK : SDAD_ERR_UNSUPPORTED;
}

__global__ void set_wait_kernel(WsHeader* h, uint32_t v) { h->wait_polls = v; }

// out[q] = src[perm[q]] for q < count (32-bit words); perm entries outside
// [0, n_src) (the -1 of padding keys) give 0
__global__ void gather32_kernel(const uint32_t* __restrict__ src, int64_t n_src,
                                const int32_t* __restrict__ perm, int64_t count,
                                uint32_t* __restrict__ out) {
  for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < count;
       q += (int64_t)gridDim.x * blockDim.x) {
    const int32_t p = __ldg(perm + q);
    out[q] = (p >= 0 && p < n_src) ? __ldg(src + p) : 0u;
  }
}

__global__ void zero_kernel(float* __restrict__ p, size_t n) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    p[i] = 0.f;
}

cudaError_t zero_f32(float* p, size_t count, cudaStream_t st) {
  if (!count) return cudaSuccess;
  const int grid = (int)std::min<size_t>((count + 255) / 256, (size_t)device_sm_count() * 8);
  {
    KTimer t("zero", st);
    zero_kernel<<<grid, 256, 0, st>>>(p, count);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// per-kernel timing
// ---------------------------------------------------------------------------
namespace {
struct TimingRec {
  const char* name;
  cudaEvent_t a, b;
};
bool g_timing = false;
std::vector<TimingRec> g_recs;   // events are kept and reused across resets
size_t g_used = 0;
constexpr size_t kMaxRecs = 1 << 16;
}  // namespace

KTimer::KTimer(const char* name, cudaStream_t st) : slot_(-1), st_(st) {
  if (!g_timing || g_used >= kMaxRecs) return;
  if (g_used == g_recs.size()) {
    TimingRec r{nullptr, nullptr, nullptr};
    if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return;
    g_recs.push_back(r);
  }
  TimingRec& r = g_recs[g_used];
  r.name = name;
  if (cudaEventRecord(r.a, st) != cudaSuccess) return;
  slot_ = (int)g_used++;
}

KTimer::~KTimer() {
  if (slot_ >= 0) cudaEventRecord(g_recs[(size_t)slot_].b, st_);
}

// ---------------------------------------------------------------------------
// workspace
// ---------------------------------------------------------------------------
static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

WsLayout ws_layout(int expr, int32_t rows, int32_t cols, int64_t nnz, int32_t width,
                   void* ws, bool ranked_cols) {
  WsLayout L;
  std::memset(&L, 0, sizeof(L));
  char* base = static_cast<char*>(ws);
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    char* p = base ? base + off : nullptr;
    off = align256(off + bytes);
    return p;
  };
  L.hdr = reinterpret_cast<WsHeader*>(take(sizeof(WsHeader)));
  L.partials = reinterpret_cast<double*>(take(sizeof(double) * kMaxPartials));
  L.sink = reinterpret_cast<double*>(take(sizeof(double)));
  if (expr == SDAD_EXPR_SMVM || expr == SDAD_EXPR_SMMM)
    L.colsum = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(cols, 1)));
  if (expr == SDAD_EXPR_BATAX)
    L.rowvec = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(rows, 1)));
  if (expr == SDAD_EXPR_LSQ || expr == SDAD_EXPR_LOGREG) {
    L.rowvec = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(rows, 1)));
    if (ranked_cols) {
      const size_t c = (size_t)std::max(cols, 1);
      L.vr = reinterpret_cast<float*>(take(sizeof(float) * c));
      L.vacc = reinterpret_cast<float*>(take(sizeof(float) * c));
    }
  }
  if (expr == SDAD_EXPR_GNN) {
    const size_t f = (size_t)std::max(width, 1);
    L.P = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(cols, 1) * f));
    L.D = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(rows, 1) * f));
    L.G = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max(cols, 1) * f));
    L.dWpart = reinterpret_cast<float*>(take(sizeof(float) * (size_t)kDwParts * 128 * f));
    const size_t nch = (size_t)(std::max<int64_t>(nnz, 0) / kMinCap + 2);
    L.closs = reinterpret_cast<double*>(take(sizeof(double) * nch));
    L.order = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * 4 * nch));
    L.cltan = reinterpret_cast<double*>(take(sizeof(double) * nch));
    L.tfirst = reinterpret_cast<float*>(take(sizeof(float) * nch * f));
    L.tlast = reinterpret_cast<float*>(take(sizeof(float) * nch * f));
  }
  const bool scalar = expr == SDAD_EXPR_LSQ || expr == SDAD_EXPR_LOGREG ||
                      expr == SDAD_EXPR_SMVM || expr == SDAD_EXPR_SMMM || expr == SDAD_EXPR_BATAX;
  if ((expr == SDAD_EXPR_LSQ || expr == SDAD_EXPR_LOGREG) && width > 0) {   // row-blocked CSC twin with 2^width rows per block
    const int64_t nb = ((int64_t)std::max(rows, 0) + (int64_t(1) << width) - 1) >> width;
    L.bP = reinterpret_cast<float*>(take(sizeof(float) * (size_t)std::max<int64_t>(1, nb * std::max(cols, 1))));
    // its chunks: at most nnz / chunk + one partial chunk per block
    const size_t bchunk = (size_t)(std::max<int64_t>(nnz, 0) / SDAD_BCSC_CHUNK + nb + 2);
    L.bpfirst = reinterpret_cast<float*>(take(sizeof(float) * bchunk));
    L.bplast = reinterpret_cast<float*>(take(sizeof(float) * bchunk));
    L.bfirstseg = reinterpret_cast<int*>(take(sizeof(int) * bchunk));
    L.blastseg = reinterpret_cast<int*>(take(sizeof(int) * bchunk));
  }
  {
    const int64_t cap = scalar ? kScalarMinCap : kMinCap;
    const size_t nchunk = (size_t)(std::max<int64_t>(nnz, 0) / cap + 2);
    const size_t w = (size_t)std::max(width, 1);
    L.pfirst = reinterpret_cast<float*>(take(sizeof(float) * nchunk * w));
    L.plast = reinterpret_cast<float*>(take(sizeof(float) * nchunk * w));
    L.lastseg = reinterpret_cast<int*>(take(sizeof(int) * nchunk));
  }
  L.bytes = off;
  return L;
}

}  // namespace sdad

namespace sdad {

bool a16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
bool a8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7) == 0; }

sdad_status map_cuda(cudaError_t e) { return e == cudaSuccess ? SDAD_OK : SDAD_ERR_CUDA; }

// Shape / pointer checks of a CSR operand.  need_csc: the CSC twin is read.
sdad_status check_csr(const sdad_csr* A, bool need_csc) {
  if (!A) return SDAD_ERR_NULL;
  if (A->m < 0 || A->n < 0 || A->nnz < 0) return SDAD_ERR_SHAPE;
  if (A->nnz > kMaxNnz) return SDAD_ERR_OVERFLOW;
  if (!A->rowptr) return SDAD_ERR_NULL;
  if (A->nnz > 0 && (!A->colidx || !A->val)) return SDAD_ERR_NULL;
  if ((A->colidx && !a16(A->colidx)) || (A->val && !a16(A->val))) return SDAD_ERR_ALIGN;
  if (need_csc) {
    if (!A->colptr) return SDAD_ERR_NULL;
    if (A->nnz > 0 && (!A->rowidx || !A->val_csc)) return SDAD_ERR_NULL;
    if ((A->rowidx && !a16(A->rowidx)) || (A->val_csc && !a16(A->val_csc))) return SDAD_ERR_ALIGN;
  }
  return SDAD_OK;
}

sdad_status check_ws(const WsLayout& need, void* ws, size_t ws_bytes) {
  if (!ws) return SDAD_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return SDAD_ERR_ALIGN;
  if (ws_bytes < need.bytes) return SDAD_ERR_WORKSPACE;
  return SDAD_OK;
}

// ---------------------------------------------------------------------------
// SDAD_T_AUTO: the transposed product chosen by measured throughput
// ---------------------------------------------------------------------------
// An operand is identified by its device, expression, two of its device
// pointers, its sizes and the outputs asked for.  The first AUTO call on it
// runs the call in both modes, twice each, times the second run of each with
// events on the call's stream (so it waits for the stream) and keeps the
// faster; later AUTO calls on the same operand run the kept mode only.  A
// call made while the stream is being captured into a graph does no timing:
// it runs `fallback` (a choice made earlier is still used).
struct AutoKey {
  int dev, expr;
  const void* a;
  const void* b;
  int64_t nnz;
  int32_t m, n;
  uint32_t flags;
  bool operator==(const AutoKey& o) const {
    return dev == o.dev && expr == o.expr && a == o.a && b == o.b && nnz == o.nnz && m == o.m &&
           n == o.n && flags == o.flags;
  }
};

namespace {
std::mutex g_auto_mu;
std::vector<std::pair<AutoKey, sdad_tmode>> g_auto;
}  // namespace

template <class Run>
cudaError_t run_auto(AutoKey key, sdad_tmode fallback, cudaStream_t st, Run run) {
  if (cudaGetDevice(&key.dev) != cudaSuccess) return cudaErrorInvalidDevice;
  {
    std::lock_guard<std::mutex> lock(g_auto_mu);
    for (const auto& kv : g_auto)
      if (kv.first == key) return run(kv.second);
  }
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(st, &cap);
  if (e != cudaSuccess) return e;
  if (cap != cudaStreamCaptureStatusNone) return run(fallback);
  cudaEvent_t ev[2];
  if ((e = cudaEventCreate(&ev[0])) != cudaSuccess) return e;
  if ((e = cudaEventCreate(&ev[1])) != cudaSuccess) {
    cudaEventDestroy(ev[0]);
    return e;
  }
  const sdad_tmode modes[2] = {SDAD_T_CSC, SDAD_T_ATOMIC};
  float ms[2] = {0.f, 0.f};
  for (int trial = 0; trial < 2 && e == cudaSuccess; ++trial)
    for (int k = 0; k < 2 && e == cudaSuccess; ++k) {
      if ((e = cudaEventRecord(ev[0], st)) != cudaSuccess) break;
      if ((e = run(modes[k])) != cudaSuccess) break;
      if ((e = cudaEventRecord(ev[1], st)) != cudaSuccess) break;
      if ((e = cudaEventSynchronize(ev[1])) != cudaSuccess) break;
      if (trial == 1) e = cudaEventElapsedTime(&ms[k], ev[0], ev[1]);
    }
  cudaEventDestroy(ev[0]);
  cudaEventDestroy(ev[1]);
  if (e != cudaSuccess) return e;
  // the outputs are those of the last run (ATOMIC), a complete evaluation
  const sdad_tmode pick = ms[0] <= ms[1] ? SDAD_T_CSC : SDAD_T_ATOMIC;
  std::lock_guard<std::mutex> lock(g_auto_mu);
  bool found = false;
  for (const auto& kv : g_auto) found = found || kv.first == key;
  if (!found) g_auto.emplace_back(key, pick);
  return cudaSuccess;
}

}  // namespace sdad

using namespace sdad;

extern "C" {

const char* sdad_status_string(sdad_status s) {
  switch (s) {
    case SDAD_OK: return "ok";
    case SDAD_ERR_NULL: return "a required pointer is NULL";
    case SDAD_ERR_SHAPE: return "negative or inconsistent sizes";
    case SDAD_ERR_INDEX: return "index out of range or unsorted input";
    case SDAD_ERR_ALIGN: return "array not aligned (16 bytes; workspace 256 bytes)";
    case SDAD_ERR_OVERFLOW: return "count does not fit in int32";
    case SDAD_ERR_WORKSPACE: return "workspace missing or too small";
    case SDAD_ERR_CUDA: return "CUDA runtime error";
    case SDAD_ERR_TIMEOUT: return "device wait exceeded its iteration limit";
    case SDAD_ERR_UNSUPPORTED: return "unsupported width/rank or device (needs sm_103)";
    default: return "unknown status";
  }
}

int32_t sdad_version(void) { return 100; }

sdad_status sdad_workspace_bytes(int32_t expr, int32_t rows, int32_t cols, int64_t nnz,
                                 int32_t width, size_t* bytes) {
  if (!bytes) return SDAD_ERR_NULL;
  if (rows < 0 || cols < 0 || nnz < 0 || width < 0) return SDAD_ERR_SHAPE;
  if (expr < SDAD_EXPR_LSQ || expr > SDAD_EXPR_BATAX) return SDAD_ERR_SHAPE;
  *bytes = ws_layout(expr, rows, cols, nnz, width, nullptr).bytes;
  return SDAD_OK;
}

sdad_status sdad_workspace_init(void* ws, void* stream) {
  if (!ws) return SDAD_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return SDAD_ERR_ALIGN;
  return map_cuda(cudaMemsetAsync(ws, 0, sizeof(WsHeader), (cudaStream_t)stream));
}

sdad_status sdad_gather_by_perm(const void* src, int64_t n_src, const int32_t* perm,
                                int64_t count, void* out, void* stream) {
  if (n_src < 0 || count < 0) return SDAD_ERR_SHAPE;
  if (count == 0) return SDAD_OK;
  if (!perm || !out || (n_src > 0 && !src)) return SDAD_ERR_NULL;
  if (!a16(perm) || !a16(out) || (src && !a16(src))) return SDAD_ERR_ALIGN;
  sdad_status s;
  if ((s = check_device())) return s;
  const int grid = (int)std::min<int64_t>((count + 255) / 256, (int64_t)device_sm_count() * 8);
  {
    KTimer t("gather_by_perm", (cudaStream_t)stream);
    gather32_kernel<<<grid, 256, 0, (cudaStream_t)stream>>>(
        static_cast<const uint32_t*>(src), n_src, perm, count, static_cast<uint32_t*>(out));
  }
  return map_cuda(cudaGetLastError());
}

sdad_status sdad_workspace_set_wait_limit(void* ws, int64_t polls, void* stream) {
  if (!ws) return SDAD_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return SDAD_ERR_ALIGN;
  if (polls >= (int64_t)0xFFFFFFFFll) return SDAD_ERR_SHAPE;
  const uint32_t v = polls < 0 ? 0u : (uint32_t)polls + 1u;
  set_wait_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(static_cast<WsHeader*>(ws), v);
  return map_cuda(cudaGetLastError());
}

sdad_status sdad_check(void* ws, void* stream) {
  if (!ws) return SDAD_ERR_NULL;
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaStreamSynchronize(st) != cudaSuccess) return SDAD_ERR_CUDA;
  int32_t code = 0;
  if (cudaMemcpy(&code, ws, sizeof(code), cudaMemcpyDeviceToHost) != cudaSuccess)
    return SDAD_ERR_CUDA;
  if (code != 0) {
    const int32_t zero = 0;
    if (cudaMemcpy(ws, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
      return SDAD_ERR_CUDA;
  }
  return code;
}

static sdad_status scalar_entry(int expr, const sdad_csr* A, const float* xin, const float* y,
                                double* loss, float* dvec, float* dA, sdad_tmode tmode, void* ws,
                                size_t ws_bytes, void* stream) {
  if (tmode < SDAD_T_AUTO || tmode > SDAD_T_ATOMIC) return SDAD_ERR_SHAPE;
  if (!A) return SDAD_ERR_NULL;
  const bool blocked = csr_blocked(A);
  const bool split = csr_split(A);
  // AUTO without a column structure for every column: the atomic scatter
  if (tmode == SDAD_T_AUTO && dvec && (blocked ? split && !A->colptr : !A->colptr))
    tmode = SDAD_T_ATOMIC;
  const bool csc = scalar_uses_csc(A, dvec != nullptr, tmode);
  sdad_status s = check_csr(A, csc && !blocked);
  if (s) return s;
  if (blocked) {
    const int lg = A->bcsc_log2;
    if (lg < SDAD_BCSC_MIN_LOG2 || lg > SDAD_BCSC_MAX_LOG2) return SDAD_ERR_UNSUPPORTED;
    const int64_t H = split ? A->bcsc_ncols : A->n;
    if (H < 0 || H > A->n) return SDAD_ERR_SHAPE;
    if (H > (int64_t(1) << (32 - lg))) return SDAD_ERR_UNSUPPORTED;
    // segment ids (block, column) are int32
    const int64_t nb = ((int64_t)A->m + (int64_t(1) << lg) - 1) >> lg;
    if (nb * std::max<int64_t>(H, 1) > kMaxNnz) return SDAD_ERR_UNSUPPORTED;
    const int64_t rest = split ? A->bcsc_rest_nnz : 0;
    if (rest < 0 || rest > A->nnz) return SDAD_ERR_SHAPE;
    if (A->bcsc_nnz < A->nnz - rest || A->bcsc_nnz % SDAD_BCSC_CHUNK || A->bcsc_nnz > kMaxNnz)
      return SDAD_ERR_SHAPE;
    if (!A->bcsc_ptr || (A->bcsc_nnz > 0 && (!A->bcsc_key || !A->bcsc_val))) return SDAD_ERR_NULL;
    if (!a16(A->bcsc_key) || !a16(A->bcsc_val)) return SDAD_ERR_ALIGN;
    if (split && csc) {   // the other columns' CSC twin
      if (!A->colptr || (rest > 0 && (!A->rowidx || !A->val_csc))) return SDAD_ERR_NULL;
      if ((A->rowidx && !a16(A->rowidx)) || (A->val_csc && !a16(A->val_csc)))
        return SDAD_ERR_ALIGN;
    }
  }
  if (csr_ranked(A)) {   // both arrays, unless empty
    if ((A->n > 0 && !A->rankcol) || (A->nnz > 0 && !A->rcolidx)) return SDAD_ERR_NULL;
    if (A->nnz > 0 && !a16(A->rcolidx)) return SDAD_ERR_ALIGN;
  }
  if ((!xin && A->n > 0) || (!y && A->m > 0) || !loss) return SDAD_ERR_NULL;
  if (expr == SDAD_EXPR_LOGREG && A->m == 0) return SDAD_ERR_SHAPE;
  if (!a8(loss)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(expr, A->m, A->n, A->nnz, blocked ? A->bcsc_log2 : 0, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  const cudaStream_t st = (cudaStream_t)stream;
  auto run = [&](sdad_tmode mode) { return run_scalar(expr, A, xin, y, loss, dvec, dA, mode, L, st); };
  if (tmode == SDAD_T_AUTO && dvec) {
    const uint32_t flags = 1u | (dA ? 2u : 0u) | (blocked ? 4u : 0u) | (split ? 8u : 0u) |
                           (csr_ranked(A) ? 16u : 0u);
    return map_cuda(run_auto(AutoKey{0, expr, A->rowptr, A->colidx, A->nnz, A->m, A->n, flags},
                             SDAD_T_CSC, st, run));
  }
  return map_cuda(run(tmode));
}

sdad_status sdad_lsq_grad(const sdad_csr* A, const float* x, const float* y, double* loss,
                          float* dx, float* dA_val, sdad_tmode tmode, void* ws, size_t ws_bytes,
                          void* stream) {
  return scalar_entry(SDAD_EXPR_LSQ, A, x, y, loss, dx, dA_val, tmode, ws, ws_bytes, stream);
}

sdad_status sdad_lsq_coo_grad(const sdad_coo* A, const float* x, const float* y, double* loss,
                              float* dx, float* dA_val, void* ws, size_t ws_bytes, void* stream) {
  if (!A || !loss) return SDAD_ERR_NULL;
  if (A->m < 0 || A->n < 0 || A->nnz < 0) return SDAD_ERR_SHAPE;
  if (A->nnz > kMaxNnz) return SDAD_ERR_OVERFLOW;
  if (A->nnz > 0 && (!A->row || !A->col || !A->val)) return SDAD_ERR_NULL;
  if ((!x && A->n > 0) || (!y && A->m > 0)) return SDAD_ERR_NULL;
  if (!a8(loss)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_LSQ, A->m, A->n, A->nnz, 0, ws);
  sdad_status s;
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_lsq_coo(A, x, y, loss, dx, dA_val, L, (cudaStream_t)stream));
}

sdad_status sdad_logreg_grad(const sdad_csr* X, const float* w, const float* y, double* loss,
                             float* dw, float* dX_val, sdad_tmode tmode, void* ws,
                             size_t ws_bytes, void* stream) {
  return scalar_entry(SDAD_EXPR_LOGREG, X, w, y, loss, dw, dX_val, tmode, ws, ws_bytes, stream);
}

sdad_status sdad_mf_grad(const sdad_csr* R, const float* U, const float* V, int32_t k,
                         float lambda, double* loss, float* dU, float* dV, float* dR_val,
                         sdad_tmode tmode, void* ws, size_t ws_bytes, void* stream) {
  if (tmode < SDAD_T_AUTO || tmode > SDAD_T_ATOMIC) return SDAD_ERR_SHAPE;
  if (k != 64) return SDAD_ERR_UNSUPPORTED;
  if (!R) return SDAD_ERR_NULL;
  // AUTO without the CSC twin: the one-pass atomic scatter
  if (tmode == SDAD_T_AUTO && dV && !R->colptr) tmode = SDAD_T_ATOMIC;
  sdad_status s = check_csr(R, dV != nullptr && tmode != SDAD_T_ATOMIC);
  if (s) return s;
  if (csr_ranked(R)) {   // used by the atomic scatter (hot columns in shared memory)
    if ((R->n > 0 && !R->rankcol) || (R->nnz > 0 && !R->rcolidx)) return SDAD_ERR_NULL;
    if (R->nnz > 0 && !a16(R->rcolidx)) return SDAD_ERR_ALIGN;
  }
  if (!U || !V || !loss) return SDAD_ERR_NULL;
  if (!a16(U) || !a16(V) || (dU && !a16(dU)) || (dV && !a16(dV)) || !a8(loss))
    return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_MF, R->m, R->n, R->nnz, k, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  const cudaStream_t st = (cudaStream_t)stream;
  auto run = [&](sdad_tmode mode) {
    return run_mf(R, U, V, lambda, loss, dU, dV, dR_val, mode, L, st);
  };
  if (tmode == SDAD_T_AUTO && dV) {
    const uint32_t flags = 1u | (dU ? 2u : 0u) | (dR_val ? 4u : 0u) | (csr_ranked(R) ? 8u : 0u);
    return map_cuda(run_auto(AutoKey{0, SDAD_EXPR_MF, R->rowptr, R->colidx, R->nnz, R->m, R->n,
                                     flags},
                             SDAD_T_CSC, st, run));
  }
  return map_cuda(run(tmode == SDAD_T_ATOMIC ? SDAD_T_ATOMIC : SDAD_T_CSC));
}

sdad_status sdad_cp3_grad(const sdad_coo3* T, const float* A, const float* B, const float* C,
                          int32_t rank, double* loss, float* dA, float* dB, float* dC,
                          float* dT_val, sdad_tmode tmode, void* ws, size_t ws_bytes,
                          void* stream) {
  if (tmode < SDAD_T_AUTO || tmode > SDAD_T_ATOMIC) return SDAD_ERR_SHAPE;
  if (!T) return SDAD_ERR_NULL;
  if (rank != 32) return SDAD_ERR_UNSUPPORTED;
  if (T->nnz < 0 || T->dims[0] < 0 || T->dims[1] < 0 || T->dims[2] < 0) return SDAD_ERR_SHAPE;
  if (T->nnz > kMaxNnz) return SDAD_ERR_OVERFLOW;
  if (!A || !B || !C || !loss) return SDAD_ERR_NULL;
  if (!a16(A) || !a16(B) || !a16(C) || !a8(loss)) return SDAD_ERR_ALIGN;
  float* dfac[3] = {dA, dB, dC};
  for (int m = 0; m < 3; ++m)
    if (dfac[m] && !a16(dfac[m])) return SDAD_ERR_ALIGN;
  // the entry-order arrays (one-pass atomic scatter) ...
  auto check_entries = [&]() -> sdad_status {
    if (T->nnz > 0 && (!T->idx[0] || !T->idx[1] || !T->idx[2] || !T->val)) return SDAD_ERR_NULL;
    return SDAD_OK;
  };
  // ... and the sorted copies of the modes asked for (per-mode passes)
  auto check_sorted = [&]() -> sdad_status {
    int first = -1;
    for (int m = 0; m < 3; ++m) {
      const bool used = dfac[m] != nullptr || (first < 0 && m == 0 && !dA && !dB && !dC);
      if (!used) continue;
      if (first < 0) first = m;
      if (!T->segptr[m]) return SDAD_ERR_NULL;
      const int o1 = m == 0 ? 1 : 0, o2 = m == 2 ? 1 : 2;
      if (T->nnz > 0 && (!T->sidx[m][o1] || !T->sidx[m][o2] || !T->sval[m])) return SDAD_ERR_NULL;
      if (!a16(T->sidx[m][o1]) || !a16(T->sidx[m][o2]) || !a16(T->sval[m])) return SDAD_ERR_ALIGN;
    }
    if (dT_val && T->nnz > 0 && !T->sperm[first]) return SDAD_ERR_NULL;
    return SDAD_OK;
  };
  sdad_status s;
  bool measure = false;
  if (tmode == SDAD_T_AUTO) {
    // both layouts given: chosen by measured throughput; else the one given
    const bool ent = check_entries() == SDAD_OK, srt = check_sorted() == SDAD_OK;
    measure = ent && srt && T->nnz > 0;
    tmode = ent ? SDAD_T_ATOMIC : SDAD_T_CSC;
  }
  if ((s = tmode == SDAD_T_ATOMIC ? check_entries() : check_sorted())) return s;
  const int32_t dmax = std::max(T->dims[0], std::max(T->dims[1], T->dims[2]));
  const WsLayout L = ws_layout(SDAD_EXPR_CP3, dmax, dmax, T->nnz, rank, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  const cudaStream_t st = (cudaStream_t)stream;
  auto run = [&](sdad_tmode mode) {
    return run_cp3(T, A, B, C, loss, dA, dB, dC, dT_val, mode, L, st);
  };
  if (measure) {
    const uint32_t flags = (dA ? 1u : 0u) | (dB ? 2u : 0u) | (dC ? 4u : 0u) | (dT_val ? 8u : 0u);
    return map_cuda(run_auto(AutoKey{0, SDAD_EXPR_CP3, T->idx[0], T->segptr[0], T->nnz,
                                     T->dims[0], T->dims[1], flags ^ ((uint32_t)T->dims[2] << 4)},
                             SDAD_T_ATOMIC, st, run));
  }
  return map_cuda(run(tmode));
}

static sdad_status jvp_entry(int expr, const sdad_csr* A, const float* v, const float* y,
                             const float* vt, const float* valt, double* loss, double* loss_t,
                             void* ws, size_t ws_bytes, void* stream) {
  sdad_status s = check_csr(A, false);
  if (s) return s;
  if ((!v && A->n > 0) || (!y && A->m > 0) || !loss || !loss_t) return SDAD_ERR_NULL;
  if (expr == SDAD_EXPR_LOGREG && A->m == 0) return SDAD_ERR_SHAPE;
  if (!a8(loss) || !a8(loss_t)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(expr, A->m, A->n, A->nnz, 0, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_jvp(expr, A, v, y, vt, valt, loss, loss_t, L, (cudaStream_t)stream));
}

sdad_status sdad_lsq_jvp(const sdad_csr* A, const float* x, const float* y, const float* x_t,
                         const float* A_t_val, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream) {
  return jvp_entry(SDAD_EXPR_LSQ, A, x, y, x_t, A_t_val, loss, loss_t, ws, ws_bytes, stream);
}

sdad_status sdad_logreg_jvp(const sdad_csr* X, const float* w, const float* y, const float* w_t,
                            const float* X_t_val, double* loss, double* loss_t, void* ws,
                            size_t ws_bytes, void* stream) {
  return jvp_entry(SDAD_EXPR_LOGREG, X, w, y, w_t, X_t_val, loss, loss_t, ws, ws_bytes, stream);
}

sdad_status sdad_mf_jvp(const sdad_csr* R, const float* U, const float* V, int32_t k,
                        float lambda, const float* R_t_val, const float* U_t, const float* V_t,
                        double* loss, double* loss_t, void* ws, size_t ws_bytes, void* stream) {
  if (k != 64) return SDAD_ERR_UNSUPPORTED;
  sdad_status s = check_csr(R, false);
  if (s) return s;
  if (!U || !V || !loss || !loss_t) return SDAD_ERR_NULL;
  if (!a16(U) || !a16(V) || (U_t && !a16(U_t)) || (V_t && !a16(V_t)) || !a8(loss) || !a8(loss_t))
    return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_MF, R->m, R->n, R->nnz, k, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_mf_jvp(R, U, V, lambda, R_t_val, U_t, V_t, loss, loss_t, L,
                             (cudaStream_t)stream));
}

sdad_status sdad_cp3_jvp(const sdad_coo3* T, const float* A, const float* B, const float* C,
                         int32_t rank, const float* T_t_val, const float* A_t, const float* B_t,
                         const float* C_t, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream) {
  if (!T) return SDAD_ERR_NULL;
  if (rank != 32) return SDAD_ERR_UNSUPPORTED;
  if (T->nnz < 0 || T->dims[0] < 0 || T->dims[1] < 0 || T->dims[2] < 0) return SDAD_ERR_SHAPE;
  if (T->nnz > kMaxNnz) return SDAD_ERR_OVERFLOW;
  if (T->nnz > 0 && (!T->idx[0] || !T->idx[1] || !T->idx[2] || !T->val)) return SDAD_ERR_NULL;
  if (!A || !B || !C || !loss || !loss_t) return SDAD_ERR_NULL;
  for (const float* f : {A, B, C, A_t, B_t, C_t})
    if (f && !a16(f)) return SDAD_ERR_ALIGN;
  if (!a8(loss) || !a8(loss_t)) return SDAD_ERR_ALIGN;
  const int32_t dmax = std::max(T->dims[0], std::max(T->dims[1], T->dims[2]));
  const WsLayout L = ws_layout(SDAD_EXPR_CP3, dmax, dmax, T->nnz, rank, ws);
  sdad_status s;
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_cp3_jvp(T, A, B, C, T_t_val, A_t, B_t, C_t, loss, loss_t, L,
                              (cudaStream_t)stream));
}

// The CSC twin's pointer array and values (the column sums read no rowidx).
static sdad_status check_csc_values(const sdad_csr* A) {
  if (!A->colptr || (A->nnz > 0 && !A->val_csc)) return SDAD_ERR_NULL;
  if (A->val_csc && !a16(A->val_csc)) return SDAD_ERR_ALIGN;
  return SDAD_OK;
}

sdad_status sdad_smvm_grad(const sdad_csr* A, const float* X, double* f, float* dX, void* ws,
                           size_t ws_bytes, void* stream) {
  sdad_status s = check_csr(A, false);
  if (s || (s = check_csc_values(A))) return s;
  if ((!X && A->n > 0) || !f) return SDAD_ERR_NULL;
  if (!a8(f)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_SMVM, A->m, A->n, A->nnz, 0, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_smvm(A, X, f, dX, L, (cudaStream_t)stream));
}

sdad_status sdad_smmm_grad(const sdad_csr* A, const sdad_csr* B, double* f, float* dB_val,
                           void* ws, size_t ws_bytes, void* stream) {
  sdad_status s = check_csr(A, false);
  if (s || (s = check_csc_values(A)) || (s = check_csr(B, false))) return s;
  if (A->n != B->m) return SDAD_ERR_SHAPE;
  if (!f) return SDAD_ERR_NULL;
  if (!a8(f)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_SMMM, A->m, A->n, A->nnz, 0, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_smmm(A, B, f, dB_val, L, (cudaStream_t)stream));
}

sdad_status sdad_batax_grad(const sdad_csr* A, const float* X, float beta, float* f,
                            const int32_t* jrowptr, const int32_t* jcolidx, int64_t jnnz,
                            float* J_val, void* ws, size_t ws_bytes, void* stream) {
  sdad_status s = check_csr(A, true);
  if (s) return s;
  if (!X && A->n > 0) return SDAD_ERR_NULL;
  if (J_val) {
    if (jnnz < 0) return SDAD_ERR_SHAPE;
    if (jnnz > kMaxNnz) return SDAD_ERR_OVERFLOW;
    if (!jrowptr || (jnnz > 0 && !jcolidx)) return SDAD_ERR_NULL;
  }
  const WsLayout L = ws_layout(SDAD_EXPR_BATAX, A->m, A->n, A->nnz, 0, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(
      run_batax(A, X, beta, f, jrowptr, jcolidx, J_val, L, (cudaStream_t)stream));
}

sdad_status sdad_gnn_grad(const sdad_csr* A, const float* H, const float* W, const float* Z,
                          int32_t f_in, int32_t f_out, double* loss, float* dA_val, float* dH,
                          float* dW, sdad_tmode tmode, void* ws, size_t ws_bytes, void* stream) {
  if (tmode < SDAD_T_AUTO || tmode > SDAD_T_ATOMIC) return SDAD_ERR_SHAPE;
  if (f_in != 128 || f_out != 64) return SDAD_ERR_UNSUPPORTED;
  if (!A) return SDAD_ERR_NULL;
  // AUTO without the CSC twin: G scattered from the CSR
  if (tmode == SDAD_T_AUTO && (dH || dW) && !A->colptr) tmode = SDAD_T_ATOMIC;
  // the column walk runs for dH, dW, and for dA when the permutation is given
  sdad_status s = check_csr(A, tmode != SDAD_T_ATOMIC && (dH || dW || (dA_val && A->csc_perm)));
  if (s) return s;
  if (A->csc_perm && A->nnz > 0 && !a16(A->csc_perm)) return SDAD_ERR_ALIGN;
  if (!H || !W || !Z || !loss) return SDAD_ERR_NULL;
  if (!a16(H) || !a16(W) || !a16(Z) || (dH && !a16(dH)) || !a8(loss)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_GNN, A->m, A->n, A->nnz, f_out, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  const cudaStream_t st = (cudaStream_t)stream;
  auto run = [&](sdad_tmode mode) {
    return run_gnn(A, H, W, Z, loss, dA_val, dH, dW, mode == SDAD_T_ATOMIC, L, st);
  };
  if (tmode == SDAD_T_AUTO && (dH || dW)) {
    const uint32_t flags = (dA_val ? 1u : 0u) | (dH ? 2u : 0u) | (dW ? 4u : 0u) |
                           (A->csc_perm ? 8u : 0u);
    return map_cuda(run_auto(AutoKey{0, SDAD_EXPR_GNN, A->rowptr, A->colidx, A->nnz, A->m, A->n,
                                     flags},
                             SDAD_T_CSC, st, run));
  }
  return map_cuda(run(tmode));
}

sdad_status sdad_gnn_jvp(const sdad_csr* A, const float* H, const float* W, const float* Z,
                         int32_t f_in, int32_t f_out, const float* A_t_val, const float* H_t,
                         const float* W_t, double* loss, double* loss_t, void* ws,
                         size_t ws_bytes, void* stream) {
  if (f_in != 128 || f_out != 64) return SDAD_ERR_UNSUPPORTED;
  sdad_status s = check_csr(A, false);
  if (s) return s;
  if (!H || !W || !Z || !loss || !loss_t) return SDAD_ERR_NULL;
  for (const float* f : {H, W, Z, H_t, W_t})
    if (f && !a16(f)) return SDAD_ERR_ALIGN;
  if (!a8(loss) || !a8(loss_t)) return SDAD_ERR_ALIGN;
  const WsLayout L = ws_layout(SDAD_EXPR_GNN, A->m, A->n, A->nnz, f_out, ws);
  if ((s = check_ws(L, ws, ws_bytes))) return s;
  if ((s = check_device())) return s;
  return map_cuda(run_gnn_jvp(A, H, W, Z, A_t_val, H_t, W_t, loss, loss_t, L,
                              (cudaStream_t)stream));
}

sdad_status sdad_timing_enable(int32_t on) {
  g_timing = on != 0;
  return SDAD_OK;
}

sdad_status sdad_timing_reset(void) {
  g_used = 0;
  return SDAD_OK;
}

int32_t sdad_timing_count(void) { return (int32_t)g_used; }

sdad_status sdad_timing_get(int32_t i, const char** name, float* ms) {
  if (!name || !ms) return SDAD_ERR_NULL;
  if (i < 0 || (size_t)i >= g_used) return SDAD_ERR_SHAPE;
  const TimingRec& r = g_recs[(size_t)i];
  if (cudaEventSynchronize(r.b) != cudaSuccess) return SDAD_ERR_CUDA;
  if (cudaEventElapsedTime(ms, r.a, r.b) != cudaSuccess) return SDAD_ERR_CUDA;
  *name = r.name;
  return SDAD_OK;
}

}  // extern "C"
