// k_gnn.cu -- graph propagation Y = A (H W), L = 1/2 |Y - Z|^2 (f_out = 64).
//
// Kernel sequence of one call:
//   1. P = H W                                           (dense projection)
//   2. the walks' chunk-group order (most segments first); rows without
//      keys: their loss term |Z_r|^2 / 2 (columns without keys: G_c = 0);
//      then the forward walk over the CSR (a warp per group of two 1024-key
//      chunks, groups taken from a work counter): Y_r = sum_p val[p]
//      P[colidx[p]];  rows finished inside the chunk: D_r = Y_r - Z_r,
//      loss += |D_r|^2 / 2, dA[p] = D_r . P[colidx[p]];  rows cut by chunk
//      boundaries: one 64-wide piece per chunk
//   3. fix: D_r of the cut rows from their pieces (chunk order), loss terms
//   4. dA of the cut rows' keys, chunk by chunk (hub rows are spread over many)
//   5. G = A^T D: the same walk over the CSC twin, gathering D; cut columns
//      leave pieces.  With the CSC twin's transpose permutation, dA is
//      computed here instead of in 2 and 4: the column walk gathers D_i
//      anyway and holds P_c for the column, so dA[perm[q]] = D_i . P_c costs
//      a 4-byte store per key instead of a second 256-byte gather of P
//   6. fix of the cut columns
//   7. dH = G W^T and dW = H^T G                          (dense projection)
//
// Lane layout of the walks: a warp takes two keys at a time, one per half
// warp; lane l of half h = l / 16 holds elements 4(l % 16) .. 4(l % 16) + 3
// of the 64-wide rows, so one warp instruction gathers two 256-byte rows with
// 16-byte loads.  A batch of key pairs (four in both walks) is gathered
// before it is used.  Each half keeps its own partial sum of the open segment; a segment
// that ends is closed by adding the two halves (one shuffle of a float4), so
// every sum has a fixed order (chunk structure, lane layout) and the results
// are reproducible.  The forward mode's walk (gnn_jvp_fwd_kernel, near the
// end) is the forward walk carrying a tangent.
#include <algorithm>
#include <climits>

#include "common.cuh"
#include "halfwarp.cuh"
#include "internal.h"

namespace sdad {

constexpr int kWideChunk = kMinCap;   // 1024 keys: the piece slots are per kMinCap keys
constexpr int kWideThreads = 256;
constexpr int kWideWarps = kWideThreads / 32;
// Loading the next row's Z (forward walk) or the next column's P row (column
// walk) one segment ahead measured neutral to slightly slower on the R-MAT
// graph (registers); kept as an option.
// Streamed arrays of the walks (key indices, values, permutation, Z; dA and
// G written) read and written with the evict-first cache hint, so that L2
// keeps more of the gathered P and D rows.
#ifndef SDAD_WALK_STREAM_HINTS
#define SDAD_WALK_STREAM_HINTS 1
#endif
constexpr bool kStreamHints = SDAD_WALK_STREAM_HINTS;
template <class T>
__device__ __forceinline__ T ld_stream(const T* p) {
  return kStreamHints ? __ldcs(p) : __ldg(p);
}
template <class T>
__device__ __forceinline__ void st_stream(T* p, T v) {
  if (kStreamHints) __stcs(p, v);
  else *p = v;
}

#ifndef SDAD_WALK_LOOKAHEAD
#define SDAD_WALK_LOOKAHEAD 0
#endif
constexpr bool kWalkLookahead = SDAD_WALK_LOOKAHEAD;
// Prefetch into L2 the row each upcoming segment reads when it ends (forward
// walk: Z) or begins (column walk: P), for the segments of each window of 32
// pointers the segment search loads.  Measured: forward walk 1.84 -> 1.70 ms
// on the 2^22-vertex R-MAT graph (0.74 -> 0.60 ms on 2^16 vertices, where one
// chunk of light rows sets the time); column walk 2.81 -> 3.00 ms, so off there.
#ifndef SDAD_FWD_PREFETCH
#define SDAD_FWD_PREFETCH 1
#endif
#ifndef SDAD_COL_PREFETCH
#define SDAD_COL_PREFETCH 0
#endif
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}
// lane l of a window of pointers ptr[lo + 1 + l] = pv: prefetches the 256-byte
// row of segment lo + l (l > 0) of X when that segment holds keys and lies past
// *front; then moves *front to the window's end
__device__ __forceinline__ void prefetch_window(const float* X, int lo, int pv, int lane, int* front) {
  const int prev = __shfl_up_sync(FULL_MASK, pv, 1);
  const int r = lo + lane;
  if (lane > 0 && r > *front && pv != INT_MAX && prev < pv) {
    const char* a = reinterpret_cast<const char*>(X + (size_t)r * 64);
    prefetch_l2(a);
    prefetch_l2(a + 128);
  }
  *front = max(*front, lo + 31);
}
// Resident CTAs per SM the walks are compiled for, and the forward walk's
// batch: measured fastest with 4 key pairs per batch at 6 CTAs (40
// registers) for the forward walk, and 4 pairs at 4 CTAs for the column walk
// (which also holds P_c and the batch's dot products).
#ifndef SDAD_FWD_CTAS
#define SDAD_FWD_CTAS 6
#endif
#ifndef SDAD_FWD_PAIRS
#define SDAD_FWD_PAIRS 4
#endif
constexpr int kFwdCtas = SDAD_FWD_CTAS;
#ifndef SDAD_COL_CTAS
#define SDAD_COL_CTAS 4
#endif
constexpr int kColCtas = SDAD_COL_CTAS;
// key pairs gathered per batch by the forward walk (the column walk reduces
// its dot products in batches of kColPairs)
constexpr int kFwdPairs = SDAD_FWD_PAIRS;
// key pairs gathered per batch by the column walk (4 or 8).  Measured on the
// 2^22-vertex R-MAT graph: 8 pairs at 3 CTAs per SM (76 registers) 2.81 ms,
// 4 pairs at 4 CTAs (60 registers) 2.74 ms, 4 pairs at 5 CTAs (spills) 3.17 ms.
#ifndef SDAD_COL_PAIRS
#define SDAD_COL_PAIRS 4
#endif
constexpr int kColPairs = SDAD_COL_PAIRS;
static_assert(kColPairs == 4 || kColPairs == 8, "the dot-product reductions take 4 or 8 pairs");

__device__ __forceinline__ float2 ld2(const float* base, int r, int lane) {
  return __ldg(reinterpret_cast<const float2*>(base + (size_t)r * 64) + lane);
}
__device__ __forceinline__ void st2(float* base, int r, int lane, float2 v) {
  reinterpret_cast<float2*>(base + (size_t)r * 64)[lane] = v;
}

// The segment holding key p, searched from segment `lo` on (ptr[lo] <= p):
// the last s with ptr[s] <= p, with its bounds.  The next 32 pointers are
// read in one coalesced load and the bounds taken from it by shuffles;
// beyond them, a binary search.  Called by the whole warp.
struct Seg {
  int s, s0, s1;
  int after;   // the segment after s that holds keys, when it lies in the same 32 pointers; else -1
};
template <class Vis>
__device__ __forceinline__ Seg next_segment(const int32_t* __restrict__ ptr, int nseg, int lo,
                                            int p, int lane, Vis& vis) {
  // first i in [lo + 1, nseg] with ptr[i] > p; the segment is i - 1
  const int i = lo + 1 + lane;
  const int pv = i <= nseg ? __ldg(ptr + i) : INT_MAX;
  vis.ahead(lo, pv, lane);
  const unsigned b = __ballot_sync(FULL_MASK, pv > p);
  if (b) {
    const int f = __ffs(b) - 1;
    const int s1 = __shfl_sync(FULL_MASK, pv, f);
    const int before = __shfl_sync(FULL_MASK, pv, (f + 31) & 31);
    // the segment holding key s1: the last i with ptr[i] <= s1
    const unsigned b2 = kWalkLookahead ? __ballot_sync(FULL_MASK, pv > s1 && pv != INT_MAX) : 0u;
    const int after = b2 ? lo + __ffs(b2) - 1 : -1;
    // f = 0 would mean p lies in segment lo itself (not so where the walks call this)
    return Seg{lo + f, f ? before : __ldg(ptr + lo), s1, after};
  }
  const int s = warp_lower_bound(ptr, lo + 33, nseg + 1, p + 1) - 1;
  return Seg{s, __ldg(ptr + s), __ldg(ptr + s + 1), -1};
}

// Chunks are handed out to warps dynamically, a few consecutive chunks at a
// time, from a counter in the workspace header (reset by gnn_empty_kernel):
// a warp that meets short rows or few cut segments takes more chunks, so no
// warp of a CTA waits long for the others.  Results do not depend on which
// warp takes a chunk: every chunk's sums go to that chunk's slots.
constexpr int kFwdGrab = 2;   // chunks per grab, measured best for each walk
#ifndef SDAD_COL_GRAB
#define SDAD_COL_GRAB 1
#endif
constexpr int kColGrab = SDAD_COL_GRAB;
__device__ __forceinline__ int next_group(uint32_t* ctr, int lane) {
  int g = 0;
  if (lane == 0) g = (int)atomicAdd(ctr, 1u);
  return __shfl_sync(FULL_MASK, g, 0);
}
// Order of the chunk groups.  A group's walk time grows with the segments it
// meets, not only with its keys: each segment end is a chain of dependent
// loads (the next pointers, the Z row or the P row), while the keys of one
// long segment stream.  On a graph whose light rows lie together (R-MAT
// without a vertex permutation puts them at the high numbers) the groups
// handed out last were the slowest, and a few warps ran on long after the
// others.  So the groups that meet at least four times the mean number of
// segments are handed out first (the forward walk's chunk by chunk, so that
// a group of light rows is walked by two warps), the others after them; both
// keep their matrix order, so the warps in flight still work on neighbouring groups,
// which share more of their gathered rows in L2 (sorting all groups by
// their segment count made the column walk a seventh slower).  The order
// changes no result: every chunk writes its own slots, which the fix kernels
// add in chunk order.
constexpr int kOrderThreads = 1024;
#ifndef SDAD_ORDER_HEAVY
#define SDAD_ORDER_HEAVY 4
#endif
constexpr int kOrderHeavy = SDAD_ORDER_HEAVY;   // heavy: at least this many times the mean

struct GroupWalk {   // one walk's groups, for the order kernels
  const int32_t* ptr;   // segment pointers (rowptr or colptr)
  int nseg, keys, ngroups;
  int thr;              // segments that make a group heavy
  int grab;             // chunks per group
  bool split;           // hand a heavy group out chunk by chunk
  int32_t* order;       // [ngroups + heavy groups when split]: items, see group_place_kernel
  int32_t* nitems;      // the number of items (NULL: ngroups, no split)
};

// CTA b orders groups [1024 b', 1024 b' + 1024) of walk 0 (b' = b) or of walk
// 1 (b' = b - ctas0).  flag[g]: the group is heavy; count[b]: heavy groups of
// the CTA.
__global__ void __launch_bounds__(kOrderThreads)
    group_flag_kernel(GroupWalk w0, GroupWalk w1, int ctas0, int nnz, int8_t* __restrict__ flag,
                      int32_t* __restrict__ count) {
  const bool second = (int)blockIdx.x >= ctas0;
  const GroupWalk& w = second ? w1 : w0;
  const int g = ((int)blockIdx.x - (second ? ctas0 : 0)) * kOrderThreads + threadIdx.x;
  bool heavy = false;
  if (g < w.ngroups) {
    const long long cs = (long long)g * w.keys, ce = std::min<long long>(cs + w.keys, nnz);
    if (cs < ce) {
      // the last s with ptr[s] <= x, for x = cs and x = ce - 1
      auto seg_of = [&](long long x) {
        int lo = 0, hi = w.nseg + 1;   // ptr[lo] <= x < ptr[hi] (ptr[nseg + 1] taken as +inf)
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (__ldg(w.ptr + mid) <= x) lo = mid;
          else hi = mid;
        }
        return lo;
      };
      heavy = seg_of(ce - 1) - seg_of(cs) + 1 >= w.thr;
    }
    flag[(second ? w0.ngroups : 0) + g] = heavy;
  }
  const int c = __syncthreads_count(heavy);
  if (threadIdx.x == 0) count[blockIdx.x] = c;
}

// Places each group: the heavy ones first, then the others, each in matrix order.
__global__ void __launch_bounds__(kOrderThreads)
    group_place_kernel(GroupWalk w0, GroupWalk w1, int ctas0, int ctas1,
                       const int8_t* __restrict__ flag, const int32_t* __restrict__ count) {
  __shared__ int part[kOrderThreads / 32][2];
  __shared__ int tot[2];
  const bool second = (int)blockIdx.x >= ctas0;
  const GroupWalk& w = second ? w1 : w0;
  const int b = (int)blockIdx.x - (second ? ctas0 : 0);
  const int32_t* cnt = count + (second ? ctas0 : 0);
  const int nb = second ? ctas1 : ctas0;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  // heavy groups of the walk before this CTA's, and in all
  int before = 0, all = 0;
  for (int i = t; i < nb; i += kOrderThreads) {
    const int v = __ldg(cnt + i);
    all += v;
    if (i < b) before += v;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    before += __shfl_xor_sync(FULL_MASK, before, o);
    all += __shfl_xor_sync(FULL_MASK, all, o);
  }
  if (lane == 0) { part[warp][0] = before; part[warp][1] = all; }
  __syncthreads();
  if (t < 2) {
    int x = 0;
    for (int i = 0; i < kOrderThreads / 32; ++i) x += part[i][t];
    tot[t] = x;
  }
  __syncthreads();
  const int hbefore = tot[0], hall = tot[1];
  const int g = b * kOrderThreads + t;
  const bool heavy = g < w.ngroups && flag[(second ? w0.ngroups : 0) + g];
  // rank of this group among the CTA's heavy groups
  const unsigned bal = __ballot_sync(FULL_MASK, heavy);
  __syncthreads();
  if (lane == 0) part[warp][0] = __popc(bal);
  __syncthreads();
  int rank = __popc(bal & ((1u << lane) - 1));
  for (int i = 0; i < warp; ++i) rank += part[i][0];
  if (g < w.ngroups) {
    const int hrank = hbefore + rank;                        // heavy groups before g
    if (!w.split) {
      w.order[heavy ? hrank : hall + (g - hrank)] = g;
    } else if (heavy) {   // one item per chunk: -1 - c for chunk c
      const int c0 = g * w.grab;
      for (int u = 0; u < w.grab; ++u) w.order[w.grab * hrank + u] = -1 - (c0 + u);
    } else {
      w.order[w.grab * hall + (g - hrank)] = g;
    }
  }
  if (w.nitems && b == 0 && t == 0) *w.nitems = w.ngroups + (w.split ? (w.grab - 1) * hall : 0);
}

struct ChunkPieces {
  float* __restrict__ pfirst;   // [chunks x 64]: part of a segment begun in an earlier chunk
  float* __restrict__ plast;    // [chunks x 64]: part of the segment that continues past it
  int* __restrict__ lastseg;    // that segment, or -1
  // stores the chunk's part of a cut segment (half 0 of the warp writes the
  // row); returns true for a cut one
  __device__ __forceinline__ bool cut(int ch, int s, int s0, int s1, int cs, int ce, float4 tot,
                                      int lane) const {
    if (s0 >= cs && s1 <= ce) return false;
    if (lane < 16) {
      if (s0 < cs) {
        st4(pfirst, ch, lane, tot);
      } else {
        st4(plast, ch, lane, tot);
        if (lane == 0) lastseg[ch] = s;
      }
    }
    return true;
  }
};

// One chunk [cs, ce) of a compressed structure (ptr, idx, val), walked two
// keys at a time: calls vis.segment(s, s0, s1, tot, cs, ce) for every segment
// whose keys in the chunk are done (tot = sum of val * X[idx] over them,
// 64-wide, float4 per lane, both halves holding the whole row), and
// vis.key(h, x, q) for every key q (x = the gathered row, held by half h) at
// the moment the walk is in q's segment.  Segments without keys are skipped
// (gnn_empty_kernel handles them).  TAN (forward mode): each key also
// gathers Xt[idx] (Xt may be NULL: zero) and the segment's tangent
// ttot = sum of valt * X[idx] + val * Xt[idx] (valt may be NULL: zero) goes
// to vis.segment2(s, s0, s1, tot, ttot, cs, ce) instead.
template <int NP, class Vis, bool TAN = false>
__device__ __forceinline__ void pair_walk(const int32_t* __restrict__ ptr, int nseg,
                                          const int32_t* __restrict__ idx,
                                          const float* __restrict__ val,
                                          const float* __restrict__ X, int cs, int ce, int hint,
                                          int lane, Vis& vis, int* seg_out,
                                          const float* __restrict__ valt = nullptr,
                                          const float* __restrict__ Xt = nullptr) {
  const int h = lane >> 4, sl = lane & 15;
  // the segment holding key cs: the last s with ptr[s] <= cs
  int s = warp_gallop_lower_bound(ptr, hint, nseg + 1, cs + 1) - 1;
  int s0 = __ldg(ptr + s), s1 = __ldg(ptr + s + 1);
  vis.front = s;
  vis.begin(s, -1);
  float4 acc = zero4();
  float4 tacc = zero4();   // TAN only
  auto close = [&]() {
    if constexpr (TAN) vis.segment2(s, s0, s1, join_halves(acc), join_halves(tacc), cs, ce);
    else vis.segment(s, s0, s1, join_halves(acc), cs, ce);
  };
  for (int base = cs; base < ce; base += 32) {
    const int nk = min(32, ce - base);
    const int jl = lane < nk ? ld_stream(idx + base + lane) : 0;
    const float al = lane < nk ? ld_stream(val + base + lane) : 0.f;
    float atl = 0.f;
    if constexpr (TAN) atl = (valt && lane < nk) ? ld_stream(valt + base + lane) : 0.f;
    vis.window(base, nk, lane);
    for (int k0 = 0; k0 < nk; k0 += 2 * NP) {
      float4 x[NP];
      float4 xt[TAN ? NP : 1];
#pragma unroll
      for (int u = 0; u < NP; ++u) {
        const int kk = k0 + 2 * u + h;
        const int j = __shfl_sync(FULL_MASK, jl, kk & 31);
        x[u] = kk < nk ? ld4(X, j, sl) : zero4();
        if constexpr (TAN) xt[u] = (kk < nk && Xt) ? ld4(Xt, j, sl) : zero4();
      }
#pragma unroll
      for (int u = 0; u < NP; ++u) {
        const int kk = k0 + 2 * u;   // this pair: keys kk (half 0) and kk + 1 (half 1)
        const float a = __shfl_sync(FULL_MASK, al, (kk + h) & 31);
        float at = 0.f;
        if constexpr (TAN) at = __shfl_sync(FULL_MASK, atl, (kk + h) & 31);
        if (kk >= nk) break;   // warp-uniform
        auto add = [&]() {
          acc = fma4(a, x[u], acc);
          if constexpr (TAN) tacc = fma4(at, x[u], fma4(a, xt[u], tacc));
        };
        const int p0 = base + kk;
        const bool two = kk + 1 < nk;
        if ((two ? p0 + 1 : p0) < s1) {   // both keys in segment s (the usual case)
          add();                           // an absent second key adds a zero row
          vis.key(h, x[u], kk + h, u);
          continue;
        }
        // a segment ends inside the pair
        if (p0 >= s1) {
          close();
          const Seg g = next_segment(ptr, nseg, s, p0, lane, vis);
          s = g.s; s0 = g.s0; s1 = g.s1;
          vis.begin(s, g.after);
          acc = zero4();
          tacc = zero4();
        }
        if (h == 0) add();
        vis.key_if(h == 0, x[u], kk, u);
        if (two) {
          if (p0 + 1 >= s1) {
            close();
            const Seg g = next_segment(ptr, nseg, s, p0 + 1, lane, vis);
            s = g.s; s0 = g.s0; s1 = g.s1;
            vis.begin(s, g.after);
            acc = zero4();
            tacc = zero4();
          }
          if (h == 1) add();
          vis.key_if(h == 1, x[u], kk + 1, u);
        }
      }
      vis.batch_done(k0, nk, lane);
    }
  }
  close();
  *seg_out = s;
}



// dA[p] = d . P[colidx[p]] for p in [q0, q1): sixteen gathers in flight, the
// sixteen dot products reduced together, 32 results stored together.  d is
// the row's float4 of this lane's elements (the same in both halves).
__device__ __forceinline__ void sddmm_range(const int32_t* __restrict__ colidx,
                                            const float* __restrict__ P, float4 d,
                                            float* __restrict__ dA, int q0, int q1, int lane) {
  const int h = lane >> 4, sl = lane & 15;
  for (int base = q0; base < q1; base += 32) {
    const int nk = min(32, q1 - base);
    const int jl = lane < nk ? __ldg(colidx + base + lane) : 0;
    float mine = 0.f;
    for (int k0 = 0; k0 < nk; k0 += 2 * kPairs) {
      float t[kPairs];
#pragma unroll
      for (int u = 0; u < kPairs; ++u) {
        const int kk = k0 + 2 * u + h;
        const int j = __shfl_sync(FULL_MASK, jl, kk & 31);
        const float4 x = kk < nk ? ld4(P, j, sl) : zero4();
        t[u] = dot4(d, x);
      }
      const float r = reduce_half8(t, lane);
      const float got = __shfl_sync(FULL_MASK, r, batch_src_lane((lane - k0) & 15));
      if (lane >= k0 && lane < k0 + 2 * kPairs) mine = got;
    }
    if (lane < nk) dA[base + lane] = mine;
  }
}

// ---- 2: forward walk -------------------------------------------------------
struct FwdVisit {
  const int32_t* __restrict__ colidx;
  const float* __restrict__ P;
  const float* __restrict__ Z;
  float* __restrict__ D;
  float* __restrict__ dA;
  ChunkPieces pc;
  int ch, lane;
  double loss;   // this lane's part
  float4 zr;     // Z row of the open row (loaded when the row begins)
  float4 znext;  // Z row of row znext_r, loaded one row ahead
  int znext_r;
  int front;     // rows up to this one are prefetched

  __device__ __forceinline__ void ahead(int lo, int pv, int lane_) {
    if (SDAD_FWD_PREFETCH) prefetch_window(Z, lo, pv, lane_, &front);
  }

  __device__ __forceinline__ void begin(int r, int after) {
    if (!kWalkLookahead) return;   // Z is then read when the row ends
    const int sl = lane & 15;
    zr = r == znext_r ? znext : ld_stream(reinterpret_cast<const float4*>(Z + (size_t)r * 64) + sl);
    znext_r = after;
    if (after >= 0) znext = ld4(Z, after, sl);
  }
  __device__ __forceinline__ void window(int, int, int) {}
  __device__ __forceinline__ void key(int, float4, int, int) {}
  __device__ __forceinline__ void key_if(bool, float4, int, int) {}
  __device__ __forceinline__ void batch_done(int, int, int) {}
  __device__ __forceinline__ void segment(int r, int s0, int s1, float4 tot, int cs, int ce) {
    if (pc.cut(ch, r, s0, s1, cs, ce, tot, lane)) return;
    const int sl = lane & 15;
    if (!kWalkLookahead) zr = ld_stream(reinterpret_cast<const float4*>(Z + (size_t)r * 64) + sl);
    const float4 d = make_float4(tot.x - zr.x, tot.y - zr.y, tot.z - zr.z, tot.w - zr.w);
    if (lane < 16) {
      st4(D, r, sl, d);
      loss += 0.5 * (double)dot4(d, d);
    }
    if (dA) sddmm_range(colidx, P, d, dA, s0, s1, lane);
  }
};

// WITH_DA: dA of the rows finished inside a chunk (when no transpose
// permutation lets the column walk compute it); a template parameter so that
// the plain walk does not carry the SDDMM's registers.
template <bool WITH_DA>
__global__ void __launch_bounds__(kWideThreads, kFwdCtas)
    gnn_fwd_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                   const float* __restrict__ val, int m, int nnz, int nchunks,
                   const float* __restrict__ P, const float* __restrict__ Z, float* __restrict__ D,
                   float* __restrict__ dA, ChunkPieces pc, WsHeader* hdr,
                   double* __restrict__ closs,
                   const int32_t* __restrict__ order, const int32_t* __restrict__ order_items) {
  const int lane = threadIdx.x & 31;
  FwdVisit vis{colidx, P, Z, D, WITH_DA ? dA : nullptr, pc, 0, lane, 0.0, zero4(), zero4(), -1, -1};
  const int nitems = __ldg(order_items);
  while (true) {
    const int k = next_group(&hdr->work[0], lane);
    if (k >= nitems) break;   // warp-uniform
    const int e = __ldg(order + k);   // a group, or -1 - c for chunk c alone
    const int c0 = e >= 0 ? e * kFwdGrab : -1 - e;
    const int c1 = e >= 0 ? min(c0 + kFwdGrab, nchunks) : c0 + 1;
    int hint = 0;
    for (int ch = c0; ch < c1; ++ch) {
      const int cs = ch * kWideChunk, ce = min(cs + kWideChunk, nnz);
      if (lane == 0) pc.lastseg[ch] = -1;
      __syncwarp();
      vis.ch = ch;
      vis.loss = 0.0;
      if (cs < ce) pair_walk<kFwdPairs>(rowptr, m, colidx, val, P, cs, ce, hint, lane, vis, &hint);
      const double cl = warp_sum_d(vis.loss);   // this chunk's rows, added in lane order
      if (lane == 0) closs[ch] = cl;
    }
  }
}

// ---- rows and columns without keys -----------------------------------------
// Rows: the loss term |Z_r|^2 / 2 (their D_r = -Z_r is not stored: no key
// gathers it); columns: G_c = 0.  A warp
// takes 32 consecutive rows (columns), finds the empty ones with one ballot
// and handles them two at a time (half a warp each, one float4 per lane),
// eight rows in flight.
__global__ void __launch_bounds__(kWideThreads)
    gnn_empty_kernel(const int32_t* __restrict__ rowptr, int m, const float* __restrict__ Z,
                     const int32_t* __restrict__ colptr, int n,
                     float* __restrict__ G, WsHeader* hdr, double* partials, double* loss_out) {
  __shared__ double red[kWideWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int half = lane >> 4, sl = lane & 15;
  const int gw = blockIdx.x * kWideWarps + warp, nw = gridDim.x * kWideWarps;
  if (blockIdx.x == 0 && threadIdx.x == 0) {   // the walks that follow hand out chunks from 0
    hdr->work[0] = 0;
    hdr->work[1] = 0;
  }
  const int nbr = (m + 31) / 32, nbc = G ? (n + 31) / 32 : 0;
  float lossf = 0.f;   // this lane's part, within 32-row blocks
  double loss = 0.0;
  for (int blk = gw; blk < nbr + nbc; blk += nw) {
    const bool rows = blk < nbr;
    const int r0 = (rows ? blk : blk - nbr) * 32, lim = rows ? m : n;
    const int32_t* ptr = rows ? rowptr : colptr;
    const int r = r0 + lane;
    const bool e = r < lim && __ldg(ptr + r) == __ldg(ptr + r + 1);
    unsigned todo = __ballot_sync(FULL_MASK, e);
    while (todo) {   // warp-uniform
      int rr[8];
#pragma unroll
      for (int u = 0; u < 4; ++u) {   // pick the next eight (two per step)
        const int a = todo ? __ffs(todo) - 1 : -1;
        if (todo) todo &= todo - 1;
        const int b = todo ? __ffs(todo) - 1 : -1;
        if (todo) todo &= todo - 1;
        rr[2 * u] = a;
        rr[2 * u + 1] = b;
      }
      if (rows) {
        float4 z[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = rr[2 * u + half];
          z[u] = k >= 0 ? __ldg(reinterpret_cast<const float4*>(Z + (size_t)(r0 + k) * 64) + sl)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = rr[2 * u + half];
          if (k < 0) continue;
          lossf += 0.5f * (z[u].x * z[u].x + z[u].y * z[u].y + z[u].z * z[u].z + z[u].w * z[u].w);
        }
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = rr[2 * u + half];
          if (k >= 0)
            reinterpret_cast<float4*>(G + (size_t)(r0 + k) * 64)[sl] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
    }
    loss += (double)lossf;
    lossf = 0.f;
  }
  const double cta = block_sum_d(loss, red);
  publish_loss(cta, hdr, partials, 0, false, 1.0, loss_out, red);
}

// ---- 3 and 6: segments cut by chunk boundaries ------------------------------
// One warp per chunk with a cut segment begun in it: the piece of that chunk
// plus the first piece of each later chunk it reaches, in chunk order.  Rows
// (Z != NULL): D_r = sum - Z_r and the loss term; columns: G_c = sum.
__global__ void __launch_bounds__(kWideThreads)
    wide_fix_kernel(const int32_t* __restrict__ ptr, int nchunks, ChunkPieces pc,
                    const float* __restrict__ Z, float* __restrict__ out, WsHeader* hdr,
                    double* partials, int first_slot, const double* __restrict__ closs,
                    double* loss_out) {
  __shared__ double red[kWideWarps];
  __shared__ bool s_last;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kWideWarps + warp, nw = gridDim.x * kWideWarps;
  double loss = 0.0;
  // the forward walk's per-chunk sums: this CTA adds its own slice, in order
  if (closs)
    for (int ch = blockIdx.x * blockDim.x + threadIdx.x; ch < nchunks; ch += gridDim.x * blockDim.x)
      loss += closs[ch];
  for (int ch = gw; ch < nchunks; ch += nw) {
    const int s = __ldg(pc.lastseg + ch);
    if (s < 0) continue;   // warp-uniform
    const int c1 = (__ldg(ptr + s + 1) - 1) / kWideChunk;
    float2 t = ld2(pc.plast, ch, lane);
    for (int cc = ch + 1; cc <= c1; ++cc) {
      const float2 q = ld2(pc.pfirst, cc, lane);
      t.x += q.x;
      t.y += q.y;
    }
    if (Z) {
      const float2 z = ld2(Z, s, lane);
      t = make_float2(t.x - z.x, t.y - z.y);
      loss += 0.5 * (double)fmaf(t.x, t.x, t.y * t.y);
    }
    st2(out, s, lane, t);
  }
  if (!loss_out) return;
  // this CTA's sum in slot first_slot + b; the last CTA adds the slots in order
  const double cta = block_sum_d(loss, red);
  if (threadIdx.x == 0) {
    partials[first_slot + blockIdx.x] = cta;
    __threadfence();
    s_last = atomicAdd(&hdr->ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const volatile double* pv = partials;
  double v = 0.0;
  for (int i = threadIdx.x; i < first_slot + (int)gridDim.x; i += blockDim.x) v += pv[i];
  const double tot = block_sum_d(v, red);
  if (threadIdx.x == 0) {
    *loss_out = tot;
    hdr->ticket = 0;
  }
}

// ---- 4: dA of the cut rows' keys ---------------------------------------------
__global__ void __launch_bounds__(kWideThreads)
    gnn_cut_sddmm_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                         int m, int nnz, int nchunks, const float* __restrict__ P,
                         const float* __restrict__ D, float* __restrict__ dA) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, sl = lane & 15;
  const int gw = blockIdx.x * kWideWarps + warp, nw = gridDim.x * kWideWarps;
  for (int ch = gw; ch < nchunks; ch += nw) {
    const int cs = ch * kWideChunk, ce = min(cs + kWideChunk, nnz);
    if (cs >= ce) continue;
    const int rf = warp_lower_bound(rowptr, 0, m + 1, cs + 1) - 1;       // row of key cs
    const int rl = warp_lower_bound(rowptr, rf, m + 1, ce) - 1;          // row of key ce - 1
    const int f0 = __ldg(rowptr + rf), f1 = __ldg(rowptr + rf + 1);
    if (f0 < cs || f1 > ce)   // the first row is cut
      sddmm_range(colidx, P, ld4(D, rf, sl), dA, cs, min(f1, ce), lane);
    if (rl != rf) {
      const int l1 = __ldg(rowptr + rl + 1);
      if (l1 > ce)   // the last row continues past the chunk
        sddmm_range(colidx, P, ld4(D, rl, sl), dA, __ldg(rowptr + rl), ce, lane);
    }
  }
}

// ---- 5: G = A^T D over the CSC twin ------------------------------------------
// Visitor of the column walk.  With `perm` (the CSC twin's transpose
// permutation) it also computes, for each key q of column c (row i),
// dA[perm[q]] = D_i . P_c, with P_c held by the lanes while the walk is in
// column c -- the D row is the one gathered for G, so dA costs no gather.
// Sixteen dot products are reduced together (reduce_half8).
struct ColVisit {
  float* __restrict__ G;
  ChunkPieces pc;
  const int32_t* __restrict__ perm;   // NULL: no dA
  const float* __restrict__ P;
  float* __restrict__ dA;
  int n, ch, lane;
  int ql;            // perm of this lane's key of the current 32-key window
  float4 pcol;       // P row of the current column (this lane's elements)
  float4 pnext;      // P row of column pnext_c, loaded one column ahead
  int pnext_c;
  float t[kColPairs];   // this lane's parts of the batch's dot products
  int front;         // columns up to this one are prefetched

  __device__ __forceinline__ void ahead(int lo, int pv, int lane_) {
    if (SDAD_COL_PREFETCH && perm) prefetch_window(P, lo, pv, lane_, &front);
  }

  __device__ __forceinline__ void begin(int c, int after) {
    if (!perm) return;
    const int sl = lane & 15;
    if (!kWalkLookahead) {
      pcol = ld4(P, c, sl);
      return;
    }
    pcol = c == pnext_c ? pnext : ld4(P, c, sl);
    pnext_c = after;
    if (after >= 0) pnext = ld4(P, after, sl);
  }
  __device__ __forceinline__ void window(int base, int nk, int lane_) {
    if (perm) ql = lane_ < nk ? ld_stream(perm + base + lane_) : 0;
  }
  __device__ __forceinline__ void key(int, float4 x, int, int u) {
    if (perm) t[u] = dot4(x, pcol);
  }
  __device__ __forceinline__ void key_if(bool mine, float4 x, int, int u) {
    if (perm && mine) t[u] = dot4(x, pcol);
  }
  __device__ __forceinline__ void batch_done(int k0, int nk, int lane_) {
    if (!perm) return;
    const int sl = lane_ & 15;
    const float r = reduce_half(t, lane_);
    // 8 pairs: lane (h, sl) with sl even holds key k0 + 2 ((sl >> 1) & 7) + h;
    // 4 pairs: lane (h, sl) with sl % 4 == 0 holds key k0 + 2 ((sl >> 2) & 3) + h
    const int kk = k0 + (lane_ >> 4) + (kColPairs == 8 ? 2 * ((sl >> 1) & 7) : 2 * ((sl >> 2) & 3));
    const bool holder = kColPairs == 8 ? (sl & 1) == 0 : (sl & 3) == 0;
    const int q = __shfl_sync(FULL_MASK, ql, kk & 31);
    if (holder && kk < nk) st_stream(dA + q, r);
#pragma unroll
    for (int u = 0; u < kColPairs; ++u) t[u] = 0.f;
  }
  __device__ __forceinline__ void segment(int c, int s0, int s1, float4 tot, int cs, int ce) {
    if (pc.cut(ch, c, s0, s1, cs, ce, tot, lane)) return;
    if (lane < 16) st_stream(reinterpret_cast<float4*>(G + (size_t)c * 64) + lane, tot);
  }
};

// perm != NULL: also dA on the keys
__global__ void __launch_bounds__(kWideThreads, kColCtas)
    gnn_col_kernel(const int32_t* __restrict__ colptr, const int32_t* __restrict__ rowidx,
                   const float* __restrict__ val_csc, int n, int nnz, int nchunks,
                   const float* __restrict__ D, float* __restrict__ G, ChunkPieces pc,
                   const int32_t* __restrict__ perm, const float* __restrict__ P,
                   float* __restrict__ dA, WsHeader* hdr,
                   const int32_t* __restrict__ order) {
  const int lane = threadIdx.x & 31;
  ColVisit vis;
  vis.G = G;
  vis.pc = pc;
  vis.perm = perm;
  vis.P = P;
  vis.dA = dA;
  vis.n = n;
  vis.ch = 0;
  vis.lane = lane;
  vis.ql = 0;
  vis.pcol = zero4();
  vis.pnext = zero4();
  vis.pnext_c = -1;
  vis.front = -1;
#pragma unroll
  for (int u = 0; u < kColPairs; ++u) vis.t[u] = 0.f;
  const int ngroups = (nchunks + kColGrab - 1) / kColGrab;
  while (true) {
    const int k = next_group(&hdr->work[1], lane);
    if (k >= ngroups) break;   // warp-uniform
    const int g = __ldg(order + k);
    int hint = 0;
    for (int ch = g * kColGrab; ch < min((g + 1) * kColGrab, nchunks); ++ch) {
      const int cs = ch * kWideChunk, ce = min(cs + kWideChunk, nnz);
      if (lane == 0) pc.lastseg[ch] = -1;
      __syncwarp();
      vis.ch = ch;
      if (cs < ce) pair_walk<kColPairs>(colptr, n, rowidx, val_csc, D, cs, ce, hint, lane, vis, &hint);
    }
  }
}
// ---- 5 (atomic mode): G = A^T D scattered from the CSR ----------------------
// For each key (i, j): G_j += A_ij D_i, with the 64-wide row of D_i held by
// the warp (lane l: elements 2l, 2l+1) while the walk is in row i, added to
// G_j with vector atomics (float2 per lane).  Chunks of 1024 keys come from
// the workspace's second work counter.  No CSC twin is needed; the order of
// the additions is not fixed.
__global__ void __launch_bounds__(kWideThreads)
    gnn_scatter_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                       const float* __restrict__ val, int m, int nnz, int nchunks,
                       const float* __restrict__ D, float* __restrict__ G, WsHeader* hdr) {
  const int lane = threadIdx.x & 31;
  while (true) {
    const int ch = next_group(&hdr->work[1], lane);
    if (ch >= nchunks) break;   // warp-uniform
    const int cs = ch * kWideChunk, ce = min(cs + kWideChunk, nnz);
    if (cs >= ce) continue;
    int r = warp_lower_bound(rowptr, 0, m + 1, cs + 1) - 1;   // the row of key cs
    int s1 = __ldg(rowptr + r + 1);
    float2 d = ld2(D, r, lane);
    for (int base = cs; base < ce; base += 32) {
      const int nk = min(32, ce - base);
      const int jl = lane < nk ? __ldg(colidx + base + lane) : 0;
      const float al = lane < nk ? __ldg(val + base + lane) : 0.f;
      for (int k = 0; k < nk; ++k) {
        const int j = __shfl_sync(FULL_MASK, jl, k);
        const float a = __shfl_sync(FULL_MASK, al, k);
        if (base + k >= s1) {   // the key opens a later row (warp-uniform)
          r = warp_gallop_lower_bound(rowptr, r + 1, m + 1, base + k + 1) - 1;
          s1 = __ldg(rowptr + r + 1);
          d = ld2(D, r, lane);
        }
        atomicAdd(reinterpret_cast<float2*>(G + (size_t)j * 64) + lane, make_float2(a * d.x, a * d.y));
      }
    }
  }
}

// Orders the forward walk's fgroups groups of kFwdGrab chunks (the CSR) and,
// with cgroups > 0, the column walk's (the CSC twin).  Layout in L.order:
// the forward walk's items [2 fgroups at most], the column walk's groups
// [cgroups], the flags, the per-CTA counts, and the forward walk's item count.
struct WalkOrder {
  const int32_t* fwd;     // items: a group g >= 0, or -1 - c for chunk c alone
  const int32_t* nitems;  // ... their number (device)
  const int32_t* col;     // groups of the column walk
};
static cudaError_t group_order(const sdad_csr* A, int fgroups, int cgroups, const WsLayout& L,
                               cudaStream_t st, WalkOrder* out) {
  const int m = A->m, n = A->n, nnz = (int)A->nnz;
  KTimer t("gnn_order", st);
  const int ctas0 = (fgroups + kOrderThreads - 1) / kOrderThreads;
  const int ctas1 = (cgroups + kOrderThreads - 1) / kOrderThreads;
  int32_t* ord0 = L.order;
  int32_t* ord1 = L.order + 2 * (size_t)fgroups;
  int8_t* flag = reinterpret_cast<int8_t*>(ord1 + cgroups);
  int32_t* count = ord1 + cgroups + (fgroups + cgroups + 3) / 4;
  int32_t* nitems = count + ctas0 + ctas1;
  // mean segments per group: about (segments + groups) / groups
  const GroupWalk w0{A->rowptr, m, kFwdGrab * kWideChunk, fgroups,
                     (int)std::min<long long>(INT_MAX, kOrderHeavy * (((long long)m + fgroups + fgroups - 1) / fgroups)),
                     kFwdGrab, true, ord0, nitems};
  const GroupWalk w1{A->colptr, n, kColGrab * kWideChunk, cgroups,
                     (int)std::min<long long>(INT_MAX, kOrderHeavy * (((long long)n + cgroups + std::max(cgroups, 1) - 1) / std::max(cgroups, 1))),
                     kColGrab, false, ord1, nullptr};
  *out = WalkOrder{ord0, nitems, ord1};
  group_flag_kernel<<<ctas0 + ctas1, kOrderThreads, 0, st>>>(w0, w1, ctas0, nnz, flag, count);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  group_place_kernel<<<ctas0 + ctas1, kOrderThreads, 0, st>>>(w0, w1, ctas0, ctas1, flag, count);
  return cudaGetLastError();
}

// ---- forward mode: the walk carrying (Y, Y') --------------------------------
// Y_r = sum_p val[p] P_j and Y'_r = sum_p (valt[p] P_j + val[p] P'_j); a row
// finished inside its chunk adds 1/2 |Y_r - Z_r|^2 to L and (Y_r - Z_r) . Y'_r
// to L' (this chunk's slots); a row cut by chunk boundaries leaves pieces of
// Y (pfirst / plast) and of Y' (tfirst / tlast).  Same walk, group order and
// Z prefetch as the reverse-mode forward walk.
struct JvpVisit {
  const float* __restrict__ Z;
  ChunkPieces pc;
  float* __restrict__ tfirst;
  float* __restrict__ tlast;
  int ch, lane;
  double L, Lt;   // this lane's parts
  int front;

  __device__ __forceinline__ void ahead(int lo, int pv, int lane_) {
    if (SDAD_FWD_PREFETCH) prefetch_window(Z, lo, pv, lane_, &front);
  }
  __device__ __forceinline__ void begin(int, int) {}
  __device__ __forceinline__ void window(int, int, int) {}
  __device__ __forceinline__ void key(int, float4, int, int) {}
  __device__ __forceinline__ void key_if(bool, float4, int, int) {}
  __device__ __forceinline__ void batch_done(int, int, int) {}
  __device__ __forceinline__ void segment2(int r, int s0, int s1, float4 tot, float4 ttot, int cs,
                                           int ce) {
    if (pc.cut(ch, r, s0, s1, cs, ce, tot, lane)) {
      if (lane < 16) st4(s0 < cs ? tfirst : tlast, ch, lane, ttot);
      return;
    }
    const int sl = lane & 15;
    const float4 z = ld_stream(reinterpret_cast<const float4*>(Z + (size_t)r * 64) + sl);
    const float4 d = make_float4(tot.x - z.x, tot.y - z.y, tot.z - z.z, tot.w - z.w);
    if (lane < 16) {
      L += 0.5 * (double)dot4(d, d);
      Lt += (double)dot4(d, ttot);
    }
  }
};

#ifndef SDAD_JVP_CTAS
#define SDAD_JVP_CTAS 4
#endif
constexpr int kJvpCtas = SDAD_JVP_CTAS;
constexpr int kJvpPairs = 4;

__global__ void __launch_bounds__(kWideThreads, kJvpCtas)
    gnn_jvp_fwd_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ colidx,
                       const float* __restrict__ val, const float* __restrict__ valt, int m,
                       int nnz, int nchunks, const float* __restrict__ P,
                       const float* __restrict__ Pt, const float* __restrict__ Z, ChunkPieces pc,
                       float* __restrict__ tfirst, float* __restrict__ tlast, WsHeader* hdr,
                       double* __restrict__ closs, double* __restrict__ cltan,
                       const int32_t* __restrict__ order,
                       const int32_t* __restrict__ order_items) {
  const int lane = threadIdx.x & 31;
  JvpVisit vis{Z, pc, tfirst, tlast, 0, lane, 0.0, 0.0, -1};
  const int nitems = __ldg(order_items);
  while (true) {
    const int k = next_group(&hdr->work[0], lane);
    if (k >= nitems) break;   // warp-uniform
    const int e = __ldg(order + k);   // a group, or -1 - c for chunk c alone
    const int c0 = e >= 0 ? e * kFwdGrab : -1 - e;
    const int c1 = e >= 0 ? min(c0 + kFwdGrab, nchunks) : c0 + 1;
    int hint = 0;
    for (int ch = c0; ch < c1; ++ch) {
      const int cs = ch * kWideChunk, ce = min(cs + kWideChunk, nnz);
      if (lane == 0) pc.lastseg[ch] = -1;
      __syncwarp();
      vis.ch = ch;
      vis.L = vis.Lt = 0.0;
      if (cs < ce)
        pair_walk<kJvpPairs, JvpVisit, true>(rowptr, m, colidx, val, P, cs, ce, hint, lane, vis,
                                             &hint, valt, Pt);
      const double cl = warp_sum_d(vis.L), ct = warp_sum_d(vis.Lt);   // in lane order
      if (lane == 0) {
        closs[ch] = cl;
        cltan[ch] = ct;
      }
    }
  }
}

cudaError_t run_gnn_jvp_walk(const sdad_csr* A, const float* valt, const float* P,
                             const float* Pt, const float* Z, const WsLayout& L, cudaStream_t st) {
  const int nnz = (int)A->nnz;
  const int nchunks = nnz <= 0 ? 1 : (nnz + kWideChunk - 1) / kWideChunk;
  const int fgroups = (nchunks + kFwdGrab - 1) / kFwdGrab;
  WalkOrder wo;
  cudaError_t e = group_order(A, fgroups, 0, L, st, &wo);
  if (e != cudaSuccess) return e;
  const int grid = std::max(1, std::min((fgroups + kWideWarps - 1) / kWideWarps,
                                        device_sm_count() * kJvpCtas));
  const ChunkPieces pc{L.pfirst, L.plast, L.lastseg};
  KTimer t("gnn_jvp_walk", st);
  gnn_jvp_fwd_kernel<<<grid, kWideThreads, 0, st>>>(A->rowptr, A->colidx, A->val, valt, A->m, nnz,
                                                    nchunks, P, Pt, Z, pc, L.tfirst, L.tlast,
                                                    L.hdr, L.closs, L.cltan, wo.fwd, wo.nitems);
  return cudaGetLastError();
}

cudaError_t run_gnn(const sdad_csr* A, const float* H, const float* W, const float* Z,
                    double* loss, float* dA, float* dH, float* dW, bool atomic,
                    const WsLayout& L, cudaStream_t st) {
  const int sms = device_sm_count();
  const int m = A->m, n = A->n, nnz = (int)A->nnz;
  const int nchunks = nnz <= 0 ? 1 : (nnz + kWideChunk - 1) / kWideChunk;
  // the walks: as many CTAs as are resident at once (their warps take chunk
  // groups from a counter until none is left)
  const int fgroups = (nchunks + kFwdGrab - 1) / kFwdGrab;
  const int cgroups = (nchunks + kColGrab - 1) / kColGrab;
  const int gf1 = std::max(1, std::min((fgroups + kWideWarps - 1) / kWideWarps, sms * kFwdCtas));
  const int gc1 = std::max(1, std::min((cgroups + kWideWarps - 1) / kWideWarps, sms * kColCtas));
  const int gfix = std::max(1, std::min((nchunks + kWideWarps - 1) / kWideWarps, sms * 8));
  const ChunkPieces pc{L.pfirst, L.plast, L.lastseg};
  // the column walk runs for dH and dW (and for dA when the transpose
  // permutation is given), unless G is scattered from the CSR (atomic mode)
  const bool back = !atomic && (dH || dW || (dA && A->csc_perm));
  // with the transpose permutation, dA comes from the column walk (which
  // gathers D anyway) instead of a second gather of P in the forward walk
  const bool dA_in_col = !atomic && dA && A->csc_perm;
  cudaError_t e;
  // 1. P = H W
  if ((e = dense_proj_fwd(H, W, L.P, n, L.hdr, st)) != cudaSuccess) return e;
  // the walks' group order
  WalkOrder wo;
  if ((e = group_order(A, fgroups, back ? cgroups : 0, L, st, &wo)) != cudaSuccess) return e;
  // 2a. rows (and columns) without keys
  const int ge = std::max(1, std::min((m + n + 255) / 256, sms * 8));
  {
    KTimer t("gnn_empty", st);
    gnn_empty_kernel<<<ge, kWideThreads, 0, st>>>(A->rowptr, m, Z, A->colptr, n,
                                                  back ? L.G : nullptr, L.hdr, L.partials, loss);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // 2b. forward walk
  {
    KTimer t("gnn_fwd", st);
    auto fwd = (dA && !dA_in_col) ? gnn_fwd_kernel<true> : gnn_fwd_kernel<false>;
    fwd<<<gf1, kWideThreads, 0, st>>>(A->rowptr, A->colidx, A->val, m, nnz, nchunks, L.P, Z, L.D,
                                      dA_in_col ? nullptr : dA, pc, L.hdr, L.closs, wo.fwd,
                                      wo.nitems);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // 3. cut rows (also finalises the loss over every partial slot)
  {
    KTimer t("gnn_fix", st);
    wide_fix_kernel<<<gfix, kWideThreads, 0, st>>>(A->rowptr, nchunks, pc, Z, L.D, L.hdr,
                                                   L.partials, ge, L.closs, loss);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // 4. dA of the cut rows
  if (dA && !dA_in_col && nnz > 0) {
    KTimer t("gnn_cut_sddmm", st);
    gnn_cut_sddmm_kernel<<<gfix, kWideThreads, 0, st>>>(A->rowptr, A->colidx, m, nnz, nchunks,
                                                        L.P, L.D, dA);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (atomic) {   // 5. G = A^T D scattered from the CSR
    if (!dH && !dW) return cudaSuccess;
    if ((e = zero_f32(L.G, (size_t)n * 64, st)) != cudaSuccess) return e;
    if (nnz > 0) {
      const int gs = std::max(1, std::min((nchunks + kWideWarps - 1) / kWideWarps, sms * 8));
      KTimer t("gnn_scatter", st);
      gnn_scatter_kernel<<<gs, kWideThreads, 0, st>>>(A->rowptr, A->colidx, A->val, m, nnz,
                                                       nchunks, L.D, L.G, L.hdr);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return dense_proj_bwd(H, W, L.G, dH, L.dWpart, dW, n, L.hdr, st);
  }
  if (!back) return cudaSuccess;
  // 5-6. G = A^T D
  {
    KTimer t("gnn_col", st);
    gnn_col_kernel<<<gc1, kWideThreads, 0, st>>>(A->colptr, A->rowidx, A->val_csc, n, nnz,
                                                  nchunks, L.D, L.G, pc,
                                                  dA_in_col ? A->csc_perm : nullptr, L.P, dA,
                                                  L.hdr, wo.col);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  {
    KTimer t("gnn_col_fix", st);
    wide_fix_kernel<<<gfix, kWideThreads, 0, st>>>(A->colptr, nchunks, pc, nullptr, L.G, L.hdr,
                                                   L.partials, 0, nullptr, nullptr);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (!dH && !dW) return cudaSuccess;
  // 7. dH = G W^T, dW = H^T G
  return dense_proj_bwd(H, W, L.G, dH, L.dWpart, dW, n, L.hdr, st);
}

}  // namespace sdad
