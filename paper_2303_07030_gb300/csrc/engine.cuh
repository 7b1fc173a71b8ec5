// engine.cuh -- chunked streaming of a compressed sparse structure.
//
// A compressed structure is (ptr[nseg+1], arrays[NARR][nnz]): segment s owns
// elements [ptr[s], ptr[s+1]) (CSR rows, CSC columns, or mode-sorted COO
// segments).  The element arrays are cut into chunks of CAP elements; each
// CTA takes chunks c = blockIdx.x, blockIdx.x + gridDim.x, ...
//
// Per CTA one producer warp and kConsumerWarps consumer warps form a
// pipeline over NS shared-memory stages:
//   producer: waits for stage s to be empty, finds the chunk's segment range
//             (warp-parallel lower_bound on ptr), writes it to the stage's
//             meta slot and issues one bulk copy per array (TMA engine,
//             completion counted on the stage's `full` mbarrier);
//   consumers: wait on `full`, run Body::chunk on the staged elements, then
//             each warp arrives on `empty`.
//
// Two ways to assign segments to chunks:
//   WHOLE: segment s belongs to the chunk holding ptr[s] (empty trailing
//          segments to the last chunk).  The producer stages the whole span
//          of the chunk's segments, [ptr[r_lo], ptr[r_hi]) rounded out to 16
//          bytes, up to STAGE elements; the body sees whole segments, and only
//          elements past a full stage (a segment longer than the slack
//          STAGE - CAP) or in the last < 4 elements of the arrays are read from
//          global memory.
//   SPLIT: every segment intersecting [cs, ce) is visited, clipped to the
//          chunk; empty segments belong to the chunk holding ptr[s].  A
//          segment cut by a chunk boundary ("straddler") is seen in pieces by
//          several chunks (the body combines them, e.g. with atomics).
#pragma once

#include <algorithm>
#include <climits>

#include "common.cuh"
#include "internal.h"

namespace sdad {

constexpr int kConsumerWarps = 8;
constexpr int kPipeThreads = 32 * (kConsumerWarps + 1);
// resident CTAs per SM the engine kernels are compiled for (0: no bound; they
// then take 96 registers, 2 CTAs per SM).  3 CTAs (72 registers, spills)
// measured slower: MF two passes 4.27 -> 4.74 ms, CP mode pass 0.47 -> 0.51 ms.
#ifndef SDAD_PIPE_MINB
#define SDAD_PIPE_MINB 0
#endif
#if SDAD_PIPE_MINB > 0
#define SDAD_PIPE_BOUNDS __launch_bounds__(kPipeThreads, SDAD_PIPE_MINB)
#else
#define SDAD_PIPE_BOUNDS __launch_bounds__(kPipeThreads)
#endif

constexpr int kMaxLong = 32;   // capacity of the per-chunk list of long parts
constexpr int kSegStage = 128; // segments whose pointers (and side values) are staged

struct ChunkMeta {
  int cs, ce, cb;   // chunk [cs, ce); elements [cs, cb) are staged in shared memory
  int r_lo, r_hi;   // segments to visit
  int nlong;        // SPLIT with long parts: number of parts longer than the threshold
  int pad[2];
  int long_r[kMaxLong];      // ... and their segments, ascending
  int sp[kSegStage + 1];     // ptr[r_lo + t], t <= min(r_hi - r_lo, kSegStage)
  float sy[kSegStage];       // side[r_lo + t], t < min(r_hi - r_lo, kSegStage)
};

constexpr int kPtrWin = 256;   // segment pointers the producer holds in shared memory

template <int NARR, int CAP, int NS>
struct PipeSmem {
  uint32_t buf[NS][NARR][CAP];
  ChunkMeta meta[NS];
  uint64_t full[NS];
  uint64_t empty[NS];
  double red[kConsumerWarps + 1];
  int32_t pwin[kPtrWin];         // ptr[wbase .. wbase + kPtrWin), producer only
  float swin[kPtrWin];           // side[wbase .. wbase + kPtrWin), producer only
};

// The producer's view of ptr: a window of kPtrWin consecutive entries in
// shared memory, refilled with one round of coalesced loads (eight per lane)
// when a search runs past it.  lower_bound() answers are identical to a
// search over global memory.
struct PtrWindow {
  const int32_t* __restrict__ ptr;
  int len;        // nseg + 1
  int32_t* win;   // shared memory
  int base;       // first index held; -1 = empty
  const float* __restrict__ side;   // optional per-segment values (nseg of them)
  float* swin;                      // shared memory, parallel to win

  __device__ __forceinline__ void fill(int b, int lane) {
    base = b;
#pragma unroll
    for (int t = 0; t < kPtrWin / 32; ++t) {
      const int i = b + lane + 32 * t;
      win[lane + 32 * t] = i < len ? __ldg(ptr + i) : INT32_MAX;
      if (side) swin[lane + 32 * t] = i < len - 1 ? __ldg(side + i) : 0.f;
    }
    __syncwarp();
  }
  __device__ __forceinline__ float side_value(int i) const {   // i < len - 1
    return (base >= 0 && i >= base && i < base + kPtrWin) ? swin[i - base] : __ldg(side + i);
  }
  __device__ __forceinline__ int32_t at(int i) const {   // i in the window
    return win[i - base];
  }
  // First i in [lo, len) with ptr[i] >= key; keys and lo never decrease
  // between calls of one producer.
  __device__ __forceinline__ int lower_bound(int lo, int key, int lane) {
    for (int round = 0; round < 8; ++round) {
      if (base < 0 || lo < base || lo >= base + kPtrWin) fill(lo, lane);
      // scan the window from lo, 32 entries per step
      for (int j = lo - base; j < kPtrWin; j += 32) {
        const int i = base + j + lane;
        const bool p = (j + lane >= kPtrWin) ? false : (i >= len || win[j + lane] >= key);
        const unsigned b = __ballot_sync(FULL_MASK, p);
        if (b) return min(len, base + j + __ffs(b) - 1);
      }
      lo = base + kPtrWin;
      if (lo >= len) return len;
    }
    return warp_lower_bound(ptr, lo, len, key);
  }
  // ptr[i] for any i < len (window if present, else global).
  __device__ __forceinline__ int32_t value(int i) const {
    return (base >= 0 && i >= base && i < base + kPtrWin) ? win[i - base] : __ldg(ptr + i);
  }
};

template <int NARR>
struct StreamSrc {
  const int32_t* ptr;     // [nseg + 1]
  const void* arr[NARR];  // 4-byte elements, 16-byte aligned bases
  int nseg;
  int nnz;
  int nchunks;
  const float* side = nullptr;   // optional per-segment values staged with the pointers
};

template <int CAP>
__host__ __device__ inline int num_chunks(long long nnz) {
  return nnz <= 0 ? 1 : (int)((nnz + CAP - 1) / CAP);
}

// Per-chunk view handed to the body (scalars live in registers; the list of
// long parts stays in shared memory).
template <int NARR, int CAP>
struct ChunkView {
  const uint32_t* sb[NARR];  // staged elements [cs, cb) in shared memory
  const uint32_t* g[NARR];   // the same arrays in global memory
  int cs, ce, cb, r_lo, r_hi, nlong;
  const int* long_r;         // shared memory
  const int* sp;             // staged ptr[r_lo ..]       (shared memory)
  const float* sy;           // staged side[r_lo ..]      (shared memory)
  const int32_t* gptr;       // ptr in global memory
  const float* gside;        // side values in global memory

  // ptr[r] for r_lo <= r <= r_hi
  __device__ __forceinline__ int seg_ptr(int r) const {
    const int t = r - r_lo;
    return t <= kSegStage ? sp[t] : __ldg(gptr + r);
  }
  // side[r] for r_lo <= r < r_hi
  __device__ __forceinline__ float seg_side(int r) const {
    const int t = r - r_lo;
    return t < kSegStage ? sy[t] : __ldg(gside + r);
  }

  __device__ __forceinline__ uint32_t get(int a, int p) const {
    if (p >= cs && p < cb) return sb[a][p - cs];
    return __ldg(g[a] + p);
  }
  __device__ __forceinline__ int geti(int a, int p) const { return (int)get(a, p); }
  __device__ __forceinline__ float getf(int a, int p) const { return __uint_as_float(get(a, p)); }
};

// Runs the pipeline.  Body must provide
//   __device__ void chunk(const ChunkView<NARR,CAP>& v, int warp, int lane, double& loss);
// Returns the CTA's loss sum (valid in thread 0 only).  All threads return.
// With SPLIT and LONG_T > 0 the producer also lists the segments whose part
// in the chunk is longer than LONG_T elements (at most kMaxLong exist when
// LONG_T >= CAP / kMaxLong); bodies split those parts over all consumer warps.
// With WRITES_STAGE the body may overwrite the staged elements of its chunk
// (generic-proxy stores); a proxy fence then orders those stores before the
// next bulk copy into the stage.  STAGE (>= CAP) is the capacity of a stage in
// elements (the chunks are CAP elements; WHOLE spans may be longer).
// ChunkView fields: cs = first staged element, cb = end of the staged range,
// ce = end of the chunk's elements (SPLIT: the chunk [cs, ce); WHOLE: the end
// of the span of its segments).
template <bool SPLIT, int NARR, int CAP, int NS, class Body, int LONG_T = 0,
          bool WRITES_STAGE = false, int STAGE = CAP>
__device__ __forceinline__ double run_pipeline(const StreamSrc<NARR>& src, Body& body,
                                               WsHeader* hdr, unsigned char* smraw) {
  static_assert(STAGE >= CAP && STAGE % 4 == 0, "stage capacity");
  using Smem = PipeSmem<NARR, STAGE, NS>;
  Smem& sm = *reinterpret_cast<Smem*>(smraw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumerWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();

  double loss = 0.0;
  const int nc = src.nchunks;

  // this CTA's chunks: a contiguous range [c0, c1)
  const int c0 = (int)(((long long)nc * blockIdx.x) / gridDim.x);
  const int c1 = (int)(((long long)nc * (blockIdx.x + 1)) / gridDim.x);

  if (warp == kConsumerWarps) {
    // ---------------- producer ----------------
    PtrWindow pw{src.ptr, src.nseg + 1, sm.pwin, -1, src.side, sm.swin};
    int lb_cs = 0;   // lower_bound(ptr, cs), carried from the previous chunk
    int issued = 0;  // chunks whose stage this warp has filled (copies issued, arrival made)
    for (int c = c0; c < c1; ++c) {
      const int k = c - c0;
      const int s = k % NS;
      if (k >= NS && !mbar_wait(&sm.empty[s], ((k / NS) - 1) & 1, hdr)) break;
      const int cs = c * CAP;
      const int ce = min(cs + CAP, src.nnz);
      int sb = cs, se = cs, ee = ce;   // staged [sb, se); the chunk's elements end at ee
      if (SPLIT) {
        se = cs + ((ce - cs) & ~3);
        const uint32_t bytes = (uint32_t)(se - sb) * 4u;
        if (lane == 0 && bytes) {
          // element data first: the copies run while the segment bounds are found
          mbar_expect_tx(&sm.full[s], bytes * NARR);
#pragma unroll
          for (int a = 0; a < NARR; ++a)
            bulk_g2s(sm.buf[s][a], static_cast<const uint32_t*>(src.arr[a]) + sb, bytes,
                     &sm.full[s]);
        }
      }
      if (k == 0) lb_cs = warp_lower_bound(src.ptr, 0, src.nseg + 1, cs);
      int r_lo = lb_cs;
      if (SPLIT && lb_cs > 0 && pw.value(lb_cs) > cs) r_lo = lb_cs - 1;
      const int lb_ce = (c == nc - 1) ? src.nseg : pw.lower_bound(lb_cs, ce, lane);
      const int r_hi = min(lb_ce, src.nseg);
      if (!SPLIT) {
        // the span of the chunk's segments, 16-byte aligned, at most STAGE
        const int s_lo = r_lo < r_hi ? pw.value(r_lo) : cs;
        ee = r_lo < r_hi ? pw.value(r_hi) : cs;
        sb = s_lo & ~3;
        int cnt = min((ee - sb + 3) & ~3, (src.nnz - sb) & ~3);
        cnt = max(0, min(cnt, STAGE));
        se = sb + cnt;
        const uint32_t bytes = (uint32_t)cnt * 4u;
        if (lane == 0 && bytes) {
          mbar_expect_tx(&sm.full[s], bytes * NARR);
#pragma unroll
          for (int a = 0; a < NARR; ++a)
            bulk_g2s(sm.buf[s][a], static_cast<const uint32_t*>(src.arr[a]) + sb, bytes,
                     &sm.full[s]);
        }
      }
      int nlong = 0;
      if (SPLIT && LONG_T > 0) {
        static_assert(LONG_T <= 0 || LONG_T * kMaxLong >= CAP, "too many long parts possible");
        for (int r0 = r_lo; r0 < r_hi; r0 += 32) {
          const int r = r0 + lane;
          bool lg = false;
          if (r < r_hi) {
            const int ps = max(pw.value(r), cs), pe = min(pw.value(r + 1), ce);
            lg = pe - ps > LONG_T;
          }
          const unsigned b = __ballot_sync(FULL_MASK, lg);
          if (lg) sm.meta[s].long_r[nlong + __popc(b & ((1u << lane) - 1))] = r;
          nlong += __popc(b);
        }
      }
      // stage the segment pointers (and side values) of the chunk
      {
        ChunkMeta& m = sm.meta[s];
        const int nsp = min(r_hi - r_lo, kSegStage);
        for (int t = lane; t <= nsp; t += 32) m.sp[t] = pw.value(r_lo + t);
        if (src.side)
          for (int t = lane; t < nsp; t += 32) m.sy[t] = pw.side_value(r_lo + t);
      }
      __syncwarp();
      if (lane == 0) {
        ChunkMeta& m = sm.meta[s];
        m.cs = sb; m.ce = ee; m.cb = se; m.r_lo = r_lo; m.r_hi = r_hi;
        m.nlong = nlong;
        mbar_arrive(&sm.full[s]);   // release: meta visible with the phase
      }
      __syncwarp();
      lb_cs = lb_ce;
      issued = k + 1;
    }
    // the copies of the last NS stages may still be landing (consumers that
    // gave up on a wait do not consume them): wait for each before leaving
    for (int k = max(0, issued - NS); k < issued; ++k)
      if (!mbar_drain(&sm.full[k % NS], (k / NS) & 1, hdr)) break;
  } else {
    // ---------------- consumers ----------------
    for (int c = c0; c < c1; ++c) {
      const int k = c - c0;
      const int s = k % NS;
      if (!mbar_wait(&sm.full[s], (k / NS) & 1, hdr)) break;
      ChunkView<NARR, STAGE> v;
#pragma unroll
      for (int a = 0; a < NARR; ++a) {
        v.sb[a] = sm.buf[s][a];
        v.g[a] = static_cast<const uint32_t*>(src.arr[a]);
      }
      const ChunkMeta& mt = sm.meta[s];
      v.cs = mt.cs; v.ce = mt.ce; v.cb = mt.cb;
      v.r_lo = mt.r_lo; v.r_hi = mt.r_hi; v.nlong = mt.nlong;
      v.long_r = mt.long_r;
      v.sp = mt.sp;
      v.sy = mt.sy;
      v.gptr = src.ptr;
      v.gside = src.side;
      body.chunk(v, warp, lane, loss);
      if (WRITES_STAGE) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[s]);
    }
  }
  return block_sum_d(loss, sm.red);
}

// SPLIT mode with long parts: calls fn(r, s0, s1, ps, pe, single) for every
// part of the chunk this warp handles, warp-uniformly.  Every warp scans the
// chunk's segments 32 at a time (one lane per segment, coalesced pointer
// look-ups, a ballot of the segments to visit); the segments to visit are
// dealt round robin over the consumer warps by their running rank, so empty
// segments cost almost nothing and heavy ones are spread evenly.  Parts of at
// most LONG_T elements go whole to one warp; longer parts are cut into
// kConsumerWarps pieces, one per warp (single = false).  With SKIP_EMPTY,
// segments without elements are not visited.
template <int LONG_T, bool SKIP_EMPTY = false, int NARR, int CAP, class Fn>
__device__ __forceinline__ void for_each_part(const ChunkView<NARR, CAP>& v,
                                              const int32_t* __restrict__ ptr, int warp,
                                              Fn&& fn) {
  const int lane = threadIdx.x & 31;
  int rank = 0;   // visited segments before this batch (same in every warp)
  for (int b = v.r_lo; b < v.r_hi; b += 32) {
    const int r = b + lane;
    int s0 = 0, s1 = 0;
    bool take = false;
    if (r < v.r_hi) {
      s0 = v.seg_ptr(r);
      s1 = v.seg_ptr(r + 1);
      const int ps = max(s0, v.cs), pe = min(s1, v.ce);
      take = !(LONG_T > 0 && pe - ps > LONG_T) && !(SKIP_EMPTY && s1 == s0);
    }
    const unsigned all = __ballot_sync(FULL_MASK, take);
    // bits of this warp: ranks rank + k with (rank + k) % kConsumerWarps == warp
    unsigned todo = 0;
    {
      unsigned rest = all;
      int k = rank;
      while (rest) {
        const unsigned bit = rest & (0u - rest);
        if (k % kConsumerWarps == warp) todo |= bit;
        rest ^= bit;
        ++k;
      }
    }
    rank += __popc(all);
    while (todo) {
      const int l = __ffs(todo) - 1;
      todo &= todo - 1;
      const int a0 = __shfl_sync(FULL_MASK, s0, l), a1 = __shfl_sync(FULL_MASK, s1, l);
      fn(b + l, a0, a1, max(a0, v.cs), min(a1, v.ce), true);
    }
  }
  for (int t = 0; t < v.nlong; ++t) {
    const int r = v.long_r[t];
    const int s0 = v.seg_ptr(r), s1 = v.seg_ptr(r + 1);
    const int ps = max(s0, v.cs), pe = min(s1, v.ce);
    const long long len = pe - ps;
    const int a = ps + (int)(len * warp / kConsumerWarps);
    const int b = ps + (int)(len * (warp + 1) / kConsumerWarps);
    fn(r, s0, s1, a, b, false);
  }
}

// True when the results of segment [s0, s1) are combined from several pieces
// with atomic adds (it is cut by a chunk boundary, or it is longer than
// LONG_T), so its destination must be initialised before the pass.
template <int CAP, int LONG_T>
__host__ __device__ __forceinline__ bool combined_atomically(int s0, int s1) {
  if (s1 <= s0) return false;
  return (s0 / CAP != (s1 - 1) / CAP) || (LONG_T > 0 && s1 - s0 > LONG_T);
}

template <int NARR, int CAP, int NS>
constexpr size_t pipe_smem_bytes() {
  return sizeof(PipeSmem<NARR, CAP, NS>);
}

}  // namespace sdad

namespace sdad {

// Initialises the destination rows of segments combined atomically (see
// combined_atomically): out[r] = scale * src[r], or 0 when src is NULL.
// Two independent segment sets (e.g. rows and columns) in one launch.
struct InitSet {
  const int32_t* ptr;
  int nseg;
  float* out;          // [nseg x width]; NULL = skip this set
  const float* src;    // [nseg x width] or NULL
  float scale;
};

template <int CAP, int LONG_T>
__global__ void init_combined_kernel(InitSet a, InitSet b, int width) {
  const int total = (a.out ? a.nseg : 0) + (b.out ? b.nseg : 0);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    const bool first = a.out && i < a.nseg;
    const InitSet& s = first ? a : b;
    const int r = first ? i : i - (a.out ? a.nseg : 0);
    if (!combined_atomically<CAP, LONG_T>(__ldg(s.ptr + r), __ldg(s.ptr + r + 1))) continue;
    float4* d = reinterpret_cast<float4*>(s.out + (size_t)r * width);
    const float4* q = s.src ? reinterpret_cast<const float4*>(s.src + (size_t)r * width) : nullptr;
    for (int t = 0; t < width / 4; ++t) {
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (q) {
        v = __ldg(q + t);
        v.x *= s.scale; v.y *= s.scale; v.z *= s.scale; v.w *= s.scale;
      }
      d[t] = v;
    }
  }
}

template <int CAP, int LONG_T>
inline cudaError_t init_combined(const InitSet& a, const InitSet& b, int width, int sms,
                                 cudaStream_t st) {
  const int total = (a.out ? a.nseg : 0) + (b.out ? b.nseg : 0);
  if (total == 0) return cudaSuccess;
  const int grid = std::max(1, std::min((total + 255) / 256, sms * 8));
  {
    KTimer t_init_combined("init_combined", st);
    init_combined_kernel<CAP, LONG_T><<<grid, 256, 0, st>>>(a, b, width);
  }
  return cudaGetLastError();
}

}  // namespace sdad
