// noalloc.cu -- least squares for callers that cannot allocate device memory.
//
// Every other entry point takes a caller-owned workspace.  Some callers
// cannot provide one: code that runs inside a host whose device memory is
// owned by another allocator (a framework's caching pool, an application
// that reserves all device memory at start-up) may not call cudaMalloc and
// has no way to hand the library scratch memory.  sdad_lsq_grad_noalloc
// serves them with a scratch area built into the library: the file-scope
// device array below, kNoAllocBytes in size.  Every GPU on which the library
// is loaded holds that array until the process exits.
//
// The entry point allocates nothing: no cudaMalloc, no cudaFree, no
// allocating library routine.  All calls share the one array, which keeps
// what the previous call left in it; the part that must start at zero (the
// 256-byte header with the status word and the loss ticket) is cleared by
// each call, on the call's stream.  Calls whose work overlaps on the GPU (on
// different streams, without ordering) race on the array.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

#include "common.cuh"
#include "internal.h"
#include "sdad.h"

namespace sdad {
namespace {

constexpr size_t kNoAllocBytes = size_t(8) << 20;   // 8 MiB

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

// Device address of g_noalloc_scratch, per device.  In host code the array's
// name only stands in for the symbol; the address a kernel can use comes from
// cudaGetSymbolAddress with that device current.
std::atomic<void*> g_scratch_addr[64];

sdad_status scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SDAD_ERR_CUDA;
  if (dev < 0 || dev >= 64) return SDAD_ERR_UNSUPPORTED;
  void* p = g_scratch_addr[dev].load();
  if (!p) {
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return SDAD_ERR_CUDA;
    g_scratch_addr[dev].store(p);
  }
  *out = p;
  return SDAD_OK;
}

}  // namespace
}  // namespace sdad

using namespace sdad;

extern "C" sdad_status sdad_lsq_grad_noalloc(const sdad_csr* A, const float* x, const float* y,
                                             double* loss, float* dx, float* dA_val,
                                             sdad_tmode tmode, void* stream) {
  if (tmode < SDAD_T_AUTO || tmode > SDAD_T_ATOMIC) return SDAD_ERR_SHAPE;
  if (!A) return SDAD_ERR_NULL;
  // the ranked column numbering is not used here (its buffers would not fit)
  sdad_csr plain = *A;
  plain.rcolidx = nullptr;
  plain.rankcol = nullptr;
  A = &plain;
  const bool csc = scalar_uses_csc(A, dx != nullptr, tmode);
  // nor the row-blocked twin; a CSC twin that holds only some columns (the
  // rest of a split twin) cannot serve the column pass alone
  if (csc && csr_split(A)) return SDAD_ERR_UNSUPPORTED;
  // a matrix that carries only a row-blocked twin (no plain CSC twin) has no
  // column structure this entry point can read
  if (csc && csr_blocked(A) && !A->colptr) return SDAD_ERR_UNSUPPORTED;
  plain.bcsc_log2 = 0;
  plain.bcsc_cols = nullptr;
  sdad_status s = check_csr(A, csc);
  if (s) return s;
  if ((!x && A->n > 0) || (!y && A->m > 0) || !loss) return SDAD_ERR_NULL;
  if (!a8(loss)) return SDAD_ERR_ALIGN;
  // the scratch this problem needs must fit in the built-in array
  if (ws_layout(SDAD_EXPR_LSQ, A->m, A->n, A->nnz, 0, nullptr, false).bytes > kNoAllocBytes)
    return SDAD_ERR_WORKSPACE;
  if ((s = check_device())) return s;
  void* scratch = nullptr;
  if ((s = scratch_for_current_device(&scratch))) return s;
  const cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemsetAsync(scratch, 0, sizeof(WsHeader), st) != cudaSuccess) return SDAD_ERR_CUDA;
  const WsLayout L = ws_layout(SDAD_EXPR_LSQ, A->m, A->n, A->nnz, 0, scratch, false);
  return map_cuda(run_scalar(SDAD_EXPR_LSQ, A, x, y, loss, dx, dA_val, tmode, L, st));
}
