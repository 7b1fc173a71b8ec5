// common.cuh -- device helpers shared by the sdad kernels (sm_103a).
//
// * PTX wrappers for mbarriers and the bulk (TMA) global->shared copy.
// * Bounded waits: every spin on an mbarrier gives up after a fixed number of
//   polls and records SDAD_ERR_TIMEOUT in the workspace status word.
// * Warp reductions, a warp-parallel lower_bound over CSR pointers, and the
//   deterministic "last CTA sums the partials" loss reduction.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "sdad.h"

namespace sdad {

constexpr unsigned FULL_MASK = 0xffffffffu;

// ---------------------------------------------------------------------------
// workspace header (first 256 bytes of every workspace)
// ---------------------------------------------------------------------------
struct WsHeader {
  int32_t status;       // sticky error code (0 = ok), cleared by sdad_check
  uint32_t ticket;      // last-CTA ticket of the loss reduction, back to 0 after use
  uint32_t wait_polls;  // 0: bounded waits poll kWaitPolls times; v > 0: v - 1 times
  uint32_t work[2];     // work counters of the graph walks (chunk groups handed out)
  uint32_t pad[59];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

constexpr int kMaxPartials = 8192;           // loss partial slots (doubles)
constexpr size_t kPartialsOffset = 256;
constexpr size_t kWsFixedBytes = kPartialsOffset + sizeof(double) * kMaxPartials;

__device__ __forceinline__ void set_status(WsHeader* h, int32_t code) {
  atomicCAS(&h->status, 0, code);
}

// ---------------------------------------------------------------------------
// PTX: shared-memory addresses, mbarriers, bulk copies
// ---------------------------------------------------------------------------
// Shared-memory accesses at a shared-window address: lds_f32 is ordered with
// other memory accesses (read-add-write sequences), ldg-like lds_f32_nc is not.
__device__ __forceinline__ float lds_f32(uint32_t a) {
  float x;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(x) : "r"(a) : "memory");
  return x;
}
__device__ __forceinline__ float lds_f32_nc(uint32_t a) {
  float x;
  asm("ld.shared.f32 %0, [%1];" : "=f"(x) : "r"(a));
  return x;
}
__device__ __forceinline__ void sts_f32(uint32_t a, float x) {
  asm volatile("st.shared.f32 [%0], %1;" ::"r"(a), "f"(x) : "memory");
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(
                   smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Polls at most kWaitPolls times (each poll may suspend the thread for a
// short, hardware-chosen time), then records a timeout and returns false.
// The workspace header can lower the limit (sdad_workspace_set_wait_limit),
// down to no poll at all, so that the timeout path can be exercised.
constexpr uint32_t kWaitPolls = 1u << 22;

__device__ __forceinline__ uint32_t wait_limit(const WsHeader* h) {
  const uint32_t v = *reinterpret_cast<const volatile uint32_t*>(&h->wait_polls);
  return v ? v - 1 : kWaitPolls;
}

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, WsHeader* h) {
  const uint32_t lim = wait_limit(h);
  for (uint32_t it = 0; it < lim; ++it)
    if (mbar_try_wait(bar, parity)) return true;
  set_status(h, SDAD_ERR_TIMEOUT);
  return false;
}

// The wait a kernel makes before it returns, for asynchronous work it issued
// itself (bulk copies into its shared memory, MMAs into its tensor memory):
// always the full kWaitPolls limit, whatever the header asks, so that a
// kernel that gave up on an earlier wait does not leave while its own copies
// are still landing.  Records a timeout if even that runs out.
__device__ __forceinline__ bool mbar_drain(uint64_t* bar, uint32_t parity, WsHeader* h) {
  for (uint32_t it = 0; it < kWaitPolls; ++it)
    if (mbar_try_wait(bar, parity)) return true;
  set_status(h, SDAD_ERR_TIMEOUT);
  return false;
}

// Bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned) from
// global memory into this CTA's shared memory; completion is signalled on
// `bar` as transaction bytes.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Asynchronous 16-byte global->shared copy (cp.async, L2 only): `bytes` of
// the 16 are read (0..16), the rest of the destination is zero-filled.  Both
// addresses 16-byte aligned.  Completion: cp_async_commit / cp_async_wait.
__device__ __forceinline__ void cp_async16_zfill(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// Waits until at most N of this thread's committed groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Hint to bring elements [b, e) of a 4-byte array into L2 (bulk prefetch by
// the copy engine; no registers, no completion).  Only whole 16-byte units
// inside the range are named, so nothing outside the array is touched.
__device__ __forceinline__ void prefetch_l2_range(const void* base, long long b, long long e) {
  const unsigned long long a0 = (reinterpret_cast<unsigned long long>(base) + 4ull * b + 15) & ~15ull;
  const unsigned long long a1 = (reinterpret_cast<unsigned long long>(base) + 4ull * e) & ~15ull;
  if (a1 > a0) {
    const unsigned long long n = a1 - a0;
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a0), "r"((uint32_t)n)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// warp helpers
// ---------------------------------------------------------------------------
template <int G>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(FULL_MASK, v, o);
  return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL_MASK, v, o);
  return v;
}

// base[idx] += v with one atomic per distinct idx among the calling lanes
// (idx < 0: nothing is added for that lane):
// `active` must be exactly the lanes that call it.  Lanes with equal idx
// (found with __match_any_sync) add their values in lane order and the
// lowest of them issues the atomic, so a hot index costs one atomic per warp
// instead of one per lane.  The shuffles run over `peers`, the lanes that
// share an index, all of which execute the same loop.
__device__ __forceinline__ void agg_atomic_add(float* base, int idx, float v, unsigned active) {
  const unsigned peers = __match_any_sync(active, idx);
  const int lane = threadIdx.x & 31;
  if (idx < 0) return;
  if (peers == (1u << lane)) {
    atomicAdd(base + idx, v);
    return;
  }
  float s = 0.f;
  for (unsigned m = peers; m; m &= m - 1) s += __shfl_sync(peers, v, __ffs(m) - 1);
  if (lane == __ffs(peers) - 1) atomicAdd(base + idx, s);
}

// First i in [lo, hi) with ptr[i] >= key, or hi if none.  ptr is
// non-decreasing.  Called by a full warp; every lane gets the answer.
__device__ __forceinline__ int warp_lower_bound(const int32_t* __restrict__ ptr, int lo, int hi,
                                                int key) {
  const int lane = threadIdx.x & 31;
  while (hi - lo > 32) {
    const int step = (hi - lo + 31) >> 5;
    const int i = lo + lane * step;
    const bool p = (i >= hi) || (__ldg(ptr + i) >= key);
    const unsigned b = __ballot_sync(FULL_MASK, p);
    if (b == 0) {
      lo = lo + 31 * step + 1;
    } else {
      const int f = __ffs(b) - 1;
      hi = min(hi, lo + f * step);
      lo = (f == 0) ? lo : lo + (f - 1) * step + 1;
    }
  }
  const int i = lo + lane;
  const bool p = (i >= hi) || (__ldg(ptr + i) >= key);
  const unsigned b = __ballot_sync(FULL_MASK, p);
  return b ? min(hi, lo + __ffs(b) - 1) : hi;
}

// Same result, for a key whose answer is expected just after `lo`: scans
// 32 entries at a time (one coalesced load each) before falling back to the
// binary search.
__device__ __forceinline__ int warp_gallop_lower_bound(const int32_t* __restrict__ ptr, int lo,
                                                       int hi, int key) {
  const int lane = threadIdx.x & 31;
  for (int t = 0; t < 4 && lo < hi; ++t, lo += 32) {
    const int i = lo + lane;
    const bool p = (i >= hi) || (__ldg(ptr + i) >= key);
    const unsigned b = __ballot_sync(FULL_MASK, p);
    if (b) return min(hi, lo + __ffs(b) - 1);
  }
  return warp_lower_bound(ptr, min(lo, hi), hi, key);
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// ---------------------------------------------------------------------------
// loss reduction
// ---------------------------------------------------------------------------
// Sums `v` over the CTA (fixed order) into thread 0's return value.
// `scratch` holds one double per warp.  Must be called by all threads.
__device__ __forceinline__ double block_sum_d(double v, double* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = (blockDim.x + 31) >> 5;
  v = warp_sum_d(v);
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < nw; ++w) s += scratch[w];
  __syncthreads();
  return s;
}

// Writes this CTA's partial into slot `first_slot + blockIdx.x`.  When
// `finalize` is set, the last CTA to finish sums slots [0, first_slot +
// gridDim.x) in slot order, multiplies by `scale` and stores the loss.  The
// order never depends on timing, so the loss is reproducible bit for bit.
__device__ __forceinline__ void publish_loss(double cta_sum, WsHeader* h, double* partials,
                                             int first_slot, bool finalize, double scale,
                                             double* loss_out, double* scratch) {
  __shared__ bool s_last;
  if (threadIdx.x == 0) {
    partials[first_slot + blockIdx.x] = cta_sum;
    s_last = false;
    if (finalize) {
      __threadfence();
      const uint32_t t = atomicAdd(&h->ticket, 1u);
      s_last = (t == gridDim.x - 1);
    }
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int n = first_slot + gridDim.x;
  double v = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) v += ((volatile double*)partials)[i];
  const double tot = block_sum_d(v, scratch);
  if (threadIdx.x == 0) {
    *loss_out = tot * scale;
    h->ticket = 0;
  }
}

}  // namespace sdad
