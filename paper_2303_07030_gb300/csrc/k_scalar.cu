// k_scalar.cu -- least squares and logistic regression: one scalar per row.
//
// Row pass (CSR), per row i of A:
//   z_i = sum_p val[p] * v[colidx[p]]             (v = x or w)
//   least squares:  r_i = z_i - y_i,  loss += r_i^2 / 2
//   logistic:       g_i = (sigmoid(z_i) - y_i) / m,
//                   loss += (1 - y_i) softplus(z_i) + y_i softplus(-z_i)   (times 1/m)
//   dA[p] = r_i * v[colidx[p]]       (gradient on A's own keys, CSR order)
//   transposed product A^T r either scattered there with atomics
//   (SDAD_T_ATOMIC) or left to the column pass below (r_i kept in workspace).
//
// Column pass (CSC twin): out_j = sum_q val_csc[q] r[rowidx[q]]; columns cut
// by a chunk boundary leave one piece per chunk and a small fix kernel adds
// the pieces in chunk order (atomic-free, bit-reproducible).
//
// Ranked columns (sdad_csr.rcolidx / rankcol): the row pass reads the ranked
// column ids and gathers from v' = v[rankcol] (built by a prep kernel), so the
// most used entries of v sit together in a few cache lines; the atomic
// transposed product accumulates in ranked order and a finish kernel stores
// dx[rankcol[c]].
#include <algorithm>

#include <climits>

#include "common.cuh"
#include "internal.h"

namespace sdad {

struct LsqOp {
  const float* __restrict__ x;
  const float* __restrict__ y;
  __device__ __forceinline__ const float* vec() const { return x; }
  __device__ __forceinline__ float gather(int j) const { return __ldg(x + j); }
  __device__ __forceinline__ float pre(int i) const { return __ldg(y + i); }
  __device__ __forceinline__ float finish(float z, float yi, double& term) const {
    const float r = z - yi;
    term = 0.5 * (double)r * (double)r;
    return r;
  }
};

struct LogregOp {
  const float* __restrict__ w;
  const float* __restrict__ y;
  float inv_m;
  __device__ __forceinline__ const float* vec() const { return w; }
  __device__ __forceinline__ float gather(int j) const { return __ldg(w + j); }
  __device__ __forceinline__ float pre(int i) const { return __ldg(y + i); }
  __device__ __forceinline__ float finish(float z, float yy, double& term) const {
    const float e = expf(-fabsf(z));             // in (0, 1]: no overflow for any z
    const float tail = log1pf(e);                // log(1 + e^-|z|)
    const float sp_pos = fmaxf(z, 0.f) + tail;   // softplus(z)
    const float sp_neg = fmaxf(-z, 0.f) + tail;  // softplus(-z) = softplus(z) - z
    // (1 - y) softplus(z) + y softplus(-z): each term to float precision
    term = (double)((1.f - yy) * sp_pos) + (double)(yy * sp_neg);
    const float sig = z >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
    return (sig - yy) * inv_m;
  }
};

// ---------------------------------------------------------------------------
// Row pass: CSR-vector kernel, no staging.  Each warp takes blocks of 32
// consecutive rows (a contiguous range of blocks per warp); a block is handled
// four rows at a time, eight lanes per row: lane l of a group reads the keys
// q = rs + l + 8k straight from global memory (eight consecutive keys per
// group and step: whole 32-byte sectors), all kRowSlots loads of a step in
// flight, and adds val * v[idx] in k order; a fixed butterfly gives z.  The z of row r0 + l is
// handed to lane l, so the finish (exp, log1p, the loss term) runs once for 32
// rows and r, y move with coalesced accesses.  The loss is summed per lane in
// row order, then per CTA in a fixed order: z, r and the loss are
// reproducible.  EMIT: a second sweep over the block's keys writes dA and
// scatters val * r with atomic adds.
// ---------------------------------------------------------------------------
constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kRowLanes = 8;
constexpr int kRowSlots = 6;
constexpr int kRowBlocksPerWarp = 2;
constexpr bool kRowPrefetch = false;  // bulk L2 prefetch of the next block's keys (measured slower)

template <class Op, bool EMIT>
__global__ void __launch_bounds__(kRowThreads)
    scalar_row_kernel(const int32_t* __restrict__ rowptr, const int32_t* __restrict__ cols,
                      const float* __restrict__ val, int m, Op op, float* __restrict__ rvec,
                      float* __restrict__ dA, float* __restrict__ dxa, WsHeader* hdr,
                      double* partials, double scale, double* loss_out) {
  __shared__ double red[kRowWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = lane / kRowLanes, gl = lane % kRowLanes;
  const int nblk = (m + 31) / 32;
  const int gw = blockIdx.x * kRowWarps + warp, nw = gridDim.x * kRowWarps;
  const int b0 = (int)(((long long)nblk * gw) / nw);
  const int b1 = (int)(((long long)nblk * (gw + 1)) / nw);
  double loss = 0.0;
  for (int b = b0; b < b1; ++b) {
    const int row = b * 32 + lane;
    const bool valid = row < m;
    const int p0 = valid ? __ldg(rowptr + row) : 0;
    const int p1 = valid ? __ldg(rowptr + row + 1) : 0;
    if (kRowPrefetch && b + 1 < b1 && lane == 0) {
      // the next block's keys, into L2 while this block is summed
      const int n0 = __ldg(rowptr + min(m, (b + 1) * 32)), n1 = __ldg(rowptr + min(m, (b + 2) * 32));
      prefetch_l2_range(cols, n0, n1);
      prefetch_l2_range(val, n0, n1);
    }
    const float yrow = valid ? op.pre(row) : 0.f;
    float zrow = 0.f;
#pragma unroll 1
    for (int sub = 0; sub < 32 / 4; ++sub) {
      const int t = sub * 4 + grp;
      const int rs = __shfl_sync(FULL_MASK, p0, t), re = __shfl_sync(FULL_MASK, p1, t);
      float z = 0.f;
      // kRowSlots keys per lane per step, all loads issued before the first
      // use (slots past the row end are masked and add zero); a typical row
      // takes one step
      for (int q0 = rs + gl; q0 < re; q0 += kRowSlots * kRowLanes) {
        int j[kRowSlots];
        float a[kRowSlots];
#pragma unroll
        for (int u = 0; u < kRowSlots; ++u) {
          const int q = q0 + u * kRowLanes;
          j[u] = q < re ? __ldg(cols + q) : 0;
          a[u] = q < re ? __ldg(val + q) : 0.f;
        }
        float x[kRowSlots];
#pragma unroll
        for (int u = 0; u < kRowSlots; ++u) x[u] = q0 + u * kRowLanes < re ? op.gather(j[u]) : 0.f;
#pragma unroll
        for (int u = 0; u < kRowSlots; ++u) z += a[u] * x[u];
      }
      z = group_sum<kRowLanes>(z);
      const float zt = __shfl_sync(FULL_MASK, z, (lane & 3) * kRowLanes);   // row sub*4 + (lane&3)
      if ((lane >> 2) == sub) zrow = zt;
    }
    float rr = 0.f;
    if (valid) {
      double term = 0.0;
      rr = op.finish(zrow, yrow, term);
      loss += term;
      if (rvec) rvec[row] = rr;
    }
    if (EMIT) {
#pragma unroll 1
      for (int sub = 0; sub < 32 / 4; ++sub) {
        const int t = sub * 4 + grp;
        const int rs = __shfl_sync(FULL_MASK, p0, t), re = __shfl_sync(FULL_MASK, p1, t);
        const float rt = __shfl_sync(FULL_MASK, rr, t);
        if (!dxa) {
          for (int q = rs + gl; q < re; q += kRowLanes) dA[q] = rt * op.gather(__ldg(cols + q));
          continue;
        }
        // the scatter: every lane runs the longest group's trip count, so the
        // warp-aggregated atomics see the whole warp (inactive lanes: idx -1)
        int trips = (re - rs + kRowLanes - 1) / kRowLanes;
#pragma unroll
        for (int o = 16; o >= kRowLanes; o >>= 1) trips = max(trips, __shfl_xor_sync(FULL_MASK, trips, o));
        for (int it = 0; it < trips; ++it) {
          const int q = rs + gl + it * kRowLanes;
          const bool act = q < re;
          const int jj = act ? __ldg(cols + q) : -1;
          if (dA && act) dA[q] = rt * op.gather(jj);
          agg_atomic_add(dxa, jj, act ? __ldg(val + q) * rt : 0.f, FULL_MASK);
        }
      }
    }
  }
  const double cta = block_sum_d(loss, red);
  publish_loss(cta, hdr, partials, 0, true, scale, loss_out, red);
}

// Sums the pieces of every column cut by chunk boundaries: the piece of the
// chunk where the column begins plus the first piece of each later chunk it
// reaches.  One warp per chunk: lane l adds the pieces of chunks c + 1 + l,
// c + 33 + l, ... in that order, a fixed butterfly adds the lanes, lane 0 adds
// the beginning piece -- a fixed order, so the sum is reproducible.
__global__ void scalar_col_fix(const int32_t* __restrict__ ptr, int nchunks, int cap,
                               const float* __restrict__ pfirst, const float* __restrict__ plast,
                               const int* __restrict__ lastseg, float* __restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int w0 = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int c = w0; c < nchunks; c += nw) {
    const int s = __ldg(lastseg + c);
    if (s < 0) continue;   // warp-uniform
    const int c1 = (__ldg(ptr + s + 1) - 1) / cap;
    float t = 0.f;
    for (int cc = c + 1 + lane; cc <= c1; cc += 32) t += __ldg(pfirst + cc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(FULL_MASK, t, o);
    if (lane == 0) out[s] = __ldg(plast + c) + t;
  }
}

// ---------------------------------------------------------------------------
// Column pass without staging (CSC twin): out_c = sum_q val_csc[q] r[rowidx[q]].
// Each warp takes one chunk (1024 keys; 256 on small matrices, for more warps);
// a chunk is read in windows of 32 keys (lane l: key base + l, coalesced).
// While a window lies inside the current column c (most windows: the long
// columns hold most keys) every lane just adds val * r to its accumulator,
// four windows per step when they all lie in c (four loads in flight).  A window with column
// boundaries finds each key's column (a 5-step shuffle search over 32 entries
// of colptr), closes column c (warp sum of the accumulators), sums the columns
// that start inside the window (segmented scan over the lanes) and stores the
// complete ones; the last one may continue into the next window and becomes c.
// A column cut by a chunk boundary leaves its part in the chunk's piece slots
// (pfirst: begun in an earlier chunk; plast/lastseg: continues past it) and
// scalar_col_fix adds the pieces in chunk order.  Every addition order is
// fixed: the result is reproducible bit for bit.  Columns without keys stay at
// the zero the output was filled with.
// ---------------------------------------------------------------------------
constexpr int kColThreads = 256;
constexpr int kColWarps = kColThreads / 32;
// chunk size: 1024 keys on large matrices, 256 on small ones (more warps);
// the workspace holds piece slots for 256-key chunks
constexpr int kColChunkLarge = 1024, kColChunkSmall = 256;
constexpr bool kColPrefetch = true;   // bulk L2 prefetch of the chunk's keys

struct ColPieces {
  float* __restrict__ out;
  float* __restrict__ pfirst;
  float* __restrict__ plast;
  int* __restrict__ lastseg;
  // stores the part of column c (keys [s0, s1)) that chunk ch = [cs, ce) holds
  __device__ __forceinline__ void put(int c, int s0, int s1, int ch, int cs, int ce,
                                      float t) const {
    if (s0 >= cs && s1 <= ce) {
      out[c] = t;
    } else if (s0 < cs) {
      pfirst[ch] = t;
    } else {
      plast[ch] = t;
      lastseg[ch] = c;
    }
  }
};

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL_MASK, v, o);
  return v;
}

// UNIT: plain column sums (every r_i = 1): rowidx and r are not read.
template <int CAP, bool UNIT>
__global__ void __launch_bounds__(kColThreads)
    scalar_colv_kernel(const int32_t* __restrict__ colptr, const int32_t* __restrict__ rowidx,
                       const float* __restrict__ val, int n, int nnz, int nchunks,
                       const float* __restrict__ rvec, ColPieces pc) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kColWarps + warp, nw = gridDim.x * kColWarps;
  const int ch0 = (int)(((long long)nchunks * gw) / nw);
  const int ch1 = (int)(((long long)nchunks * (gw + 1)) / nw);
  int c = 0;
  for (int ch = ch0; ch < ch1; ++ch) {
    const int cs = ch * CAP, ce = min(cs + CAP, nnz);
    if (lane == 0) pc.lastseg[ch] = -1;
    __syncwarp();
    if (cs >= ce) continue;
    // the column holding key cs: the last c with colptr[c] <= cs
    if (kColPrefetch && lane == 0) {   // the chunk's keys, into L2 ahead of the windows
      prefetch_l2_range(rowidx, cs, ce);
      prefetch_l2_range(val, cs, ce);
    }
    c = warp_gallop_lower_bound(colptr, ch == ch0 ? 0 : c, n + 1, cs + 1) - 1;
    int cbeg = __ldg(colptr + c), cend = __ldg(colptr + c + 1);
    bool open = true;     // column c has keys in this chunk not yet stored
    float acc = 0.f;      // this lane's part of column c
    for (int base = cs; base < ce; base += 32) {
      // four whole windows inside column c: their loads all in flight at once
      if (open && cend >= base + 4 * 32 && ce >= base + 4 * 32) {
        int ri[4];
        float a[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          ri[u] = UNIT ? 0 : __ldg(rowidx + base + 32 * u + lane);
          a[u] = __ldg(val + base + 32 * u + lane);
        }
        float x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) x[u] = UNIT ? 1.f : __ldg(rvec + ri[u]);
#pragma unroll
        for (int u = 0; u < 4; ++u) acc += a[u] * x[u];
        base += 3 * 32;
        continue;
      }
      const int q = base + lane;
      const int wend = min(base + 32, ce);
      const bool act = q < ce;
      float p = 0.f;
      if (act) p = UNIT ? __ldg(val + q) : __ldg(val + q) * __ldg(rvec + __ldg(rowidx + q));
      if (open && cend >= wend) {   // the whole window lies in column c
        acc += p;
        continue;
      }
      // column of each key: c0 + number of boundaries colptr[c0 + 1 + k] <= q
      int col = INT_MAX;
      {
        int c0 = c;   // every key of the window lies in column c or later
        unsigned todo = __ballot_sync(FULL_MASK, act);
        while (todo) {
          const int bi = c0 + 1 + lane;
          const int bnd = bi <= n ? __ldg(colptr + bi) : INT_MAX;
          int k = 0;
#pragma unroll
          for (int step = 16; step > 0; step >>= 1) {
            const int b = __shfl_sync(FULL_MASK, bnd, k + step - 1);
            if (b <= q) k += step;
          }
          const int b31 = __shfl_sync(FULL_MASK, bnd, 31);   // every lane takes part
          if (k == 31 && b31 <= q) k = 32;
          const bool mine = ((todo >> lane) & 1u) && k < 32;
          if (mine) col = c0 + k;
          todo &= ~__ballot_sync(FULL_MASK, mine);
          c0 += 32;
        }
      }
      // close column c
      if (open) {
        if (act && col == c) acc += p;
        const float t = warp_sum_f(acc);
        if (lane == 0) pc.put(c, cbeg, cend, ch, cs, ce, t);
        open = false;
      }
      // columns that start inside the window: segmented scan by column
      const bool later = act && col != c;
      float sv = later ? p : 0.f;
      const int key = later ? col : (act ? -1 : INT_MAX);
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const float v = __shfl_up_sync(FULL_MASK, sv, d);
        const int kd = __shfl_up_sync(FULL_MASK, key, d);
        if (lane >= d && kd == key) sv += v;
      }
      const int knext = __shfl_down_sync(FULL_MASK, key, 1);
      const bool last_lane_of_seg = later && (lane == 31 || knext != key);
      // the window's last column may continue into the next window
      const int lastcol = __shfl_sync(FULL_MASK, col, max(0, min(31, wend - base - 1)));
      if (last_lane_of_seg) {   // colptr entries just read: L1 hits
        const int s0 = __ldg(colptr + col), s1 = __ldg(colptr + col + 1);
        const bool carry = (col == lastcol) && s1 > wend && wend < ce;
        if (!carry) pc.put(col, s0, s1, ch, cs, ce, sv);
      }
      // the window's last column becomes the current one (open if it continues)
      c = lastcol;
      cbeg = __ldg(colptr + lastcol);
      cend = __ldg(colptr + lastcol + 1);
      open = cend > wend && wend < ce;
      acc = (act && col == lastcol && open) ? p : 0.f;
    }
    if (open) {   // the chunk ended inside column c
      const float t = warp_sum_f(acc);
      if (lane == 0) pc.put(c, cbeg, cend, ch, cs, ce, t);
    }
  }
}

// ---------------------------------------------------------------------------
// Column pass over the row-blocked CSC twin (sdad_csr_block_transpose) of H
// columns: keys sorted by (row block, column, row), key = h << lg | row
// within block (h the column's position among the H),
// each block padded to whole SDAD_BCSC_CHUNK chunks.  A CTA takes a contiguous
// range of chunks; for each block the range touches it copies that block's
// part of r (2^lg floats) into shared memory, then its warps take the block's
// chunks round robin.  A warp reads its chunk in batches of kBcolBatch
// windows of 32 keys, every load of a batch issued before the first use: r
// comes from shared memory (no L1 line per key), the column from the key.  A
// batch inside the current segment (block, column) only adds to per-lane
// accumulators; otherwise its windows go one by one: a window with segment
// boundaries closes the current one and sums the next ones by segmented scan
// (the column after a window is read from the next window's registers, or
// from the key after the batch, loaded with it).  Segment
// sums go to P[block * H + h]; a segment cut by a chunk boundary leaves a
// first piece (pfirst/firstseg: begun in an earlier chunk) or a last piece
// (plast/lastseg: continues past the chunk), and bcol_fix adds the pieces in
// chunk order.  bcol_combine then sums P over the blocks, in block order.
// ---------------------------------------------------------------------------
constexpr int kBcolThreads = 1024;
constexpr int kBcolWarps = kBcolThreads / 32;
constexpr int kBcolChunk = SDAD_BCSC_CHUNK;
constexpr int kBcolBatch = 4;   // windows of 32 keys whose loads are issued together
constexpr int kBcolMinBlocks = 1;
constexpr bool kBcolLaneRuns = true;   // lane-sequential runs (else windows of 32 keys)
constexpr int kBcolK = 8;              // consecutive keys per lane and step (a multiple of 4)

struct BcolOut {
  float* __restrict__ P;        // [nb x H], zero-filled
  float* __restrict__ pfirst;   // per chunk
  float* __restrict__ plast;
  int* __restrict__ firstseg;   // segment id b * H + h, or -1
  int* __restrict__ lastseg;
};

// One chunk of the blocked twin, read in windows of 32 keys (lane l: key
// base + l), kBcolBatch windows per batch.
__device__ __forceinline__ void bcol_chunk_windows(int ch, int b, int k0, int k1, int lg, int H,
                                                   uint32_t mask, uint32_t sbase,
                                                   const uint32_t* __restrict__ bkey,
                                                   const float* __restrict__ bval,
                                                   const BcolOut& o, int lane) {
  const int cs = ch * kBcolChunk, ce = cs + kBcolChunk;
  if (lane == 0) {
    prefetch_l2_range(bkey, cs, ce);
    prefetch_l2_range(bval, cs, ce);
    o.firstseg[ch] = -1;
    o.lastseg[ch] = -1;
  }
  const int segbase = b * H;
  int c = (int)(__ldg(bkey + cs) >> lg);
  bool before = cs > k0 && (int)(__ldg(bkey + cs - 1) >> lg) == c;
  bool open = true;     // segment c has keys in this chunk not yet stored
  float acc = 0.f;      // this lane's part of segment c
  for (int base = cs; base < ce; base += 32 * kBcolBatch) {
    // a batch of windows: every load issued before the first use
    uint32_t kk[kBcolBatch];
    float p[kBcolBatch];
#pragma unroll
    for (int u = 0; u < kBcolBatch; ++u) {
      kk[u] = __ldg(bkey + base + 32 * u + lane);
      p[u] = __ldg(bval + base + 32 * u + lane);
    }
    // the column of the key after the batch (one address for the warp)
    const int after = base + 32 * kBcolBatch;
    const int ncol_after = after < k1 ? (int)(__ldg(bkey + after) >> lg) : -1;
#pragma unroll
    for (int u = 0; u < kBcolBatch; ++u) p[u] *= lds_f32_nc(sbase + 4u * (kk[u] & mask));
    const int last = (int)(__shfl_sync(FULL_MASK, kk[kBcolBatch - 1], 31) >> lg);
    if (open && last == c) {   // the whole batch lies in segment c
#pragma unroll
      for (int u = 0; u < kBcolBatch; ++u) acc += p[u];
      continue;
    }
#pragma unroll
    for (int u = 0; u < kBcolBatch; ++u) {
      const int col = (int)(kk[u] >> lg);
      const float pu = p[u];
      const int col31 = __shfl_sync(FULL_MASK, col, 31);
      // column of the first key after this window (every lane takes part)
      const uint32_t knx = __shfl_sync(FULL_MASK, kk[(u + 1) % kBcolBatch], 0);
      const int ncol = u + 1 < kBcolBatch ? (int)(knx >> lg) : ncol_after;
      if (open && col31 == c) {   // the whole window lies in segment c
        acc += pu;
        continue;
      }
      // close segment c
      if (open) {
        if (col == c) acc += pu;
        const float t = warp_sum_f(acc);
        if (lane == 0) {
          if (before) {
            o.pfirst[ch] = t;
            o.firstseg[ch] = segbase + c;
          } else {
            o.P[segbase + c] = t;
          }
        }
        open = false;
        before = false;
      }
      // segments starting inside the window: segmented scan by column
      const bool later = col != c;
      float sv = later ? pu : 0.f;
      const int keyc = later ? col : -1;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const float v = __shfl_up_sync(FULL_MASK, sv, d);
        const int kd = __shfl_up_sync(FULL_MASK, keyc, d);
        if (lane >= d && kd == keyc) sv += v;
      }
      const int knext = __shfl_down_sync(FULL_MASK, keyc, 1);
      // the window's last segment goes on after it (same block only)
      const bool cont = ncol == col31;
      const bool seg_end = later && (lane == 31 || knext != keyc);
      if (seg_end && !(col == col31 && cont)) o.P[segbase + col] = sv;
      c = col31;
      open = cont;
      acc = (cont && col == col31) ? pu : 0.f;
    }
  }
  if (open) {
    const float t = warp_sum_f(acc);
    // continues past the chunk (within the block), or ends exactly at its end
    const bool cont = ce < k1 && (int)(__ldg(bkey + ce) >> lg) == c;
    if (lane == 0) {
      if (before) {
        o.pfirst[ch] = t;
        o.firstseg[ch] = segbase + c;
      } else if (cont) {
        o.plast[ch] = t;
        o.lastseg[ch] = segbase + c;
      } else {
        o.P[segbase + c] = t;
      }
    }
  }
}

// One chunk of the blocked twin, lane by lane: in each step of 32 * kBcolK
// keys lane l takes the kBcolK consecutive keys base + kBcolK * l + i (vector
// loads) and sums their runs of equal column in key order.  A run that
// starts and ends inside the lane is a whole segment and is stored at once;
// the lane's first run (head) and last run (tail) may go on in the lanes
// before and after it, and a segmented scan over the lanes (one per step,
// fixed order) joins them: a tail is stored by the lane where it ends, a head
// that ends inside its lane by that lane.  The segment open after lane 31
// (warp-uniform column and sum) joins lane 0 of the next step.  A step whose
// keys all lie in that open segment (the common case in long columns) only
// adds to per-lane parts, summed into the segment before the next step with
// a boundary.
__device__ __forceinline__ void bcol_chunk_lanes(int ch, int b, int k0, int k1, int lg, int H,
                                                 uint32_t mask, uint32_t sbase,
                                                 const uint32_t* __restrict__ bkey,
                                                 const float* __restrict__ bval,
                                                 const BcolOut& o, int lane) {
  constexpr int K = kBcolK;
  const int cs = ch * kBcolChunk, ce = cs + kBcolChunk;
  if (lane == 0) {
    prefetch_l2_range(bkey, cs, ce);
    prefetch_l2_range(bval, cs, ce);
    o.firstseg[ch] = -1;
    o.lastseg[ch] = -1;
  }
  const int segbase = b * H;
  const int cfirst = (int)(__ldg(bkey + cs) >> lg);
  // the chunk's first segment began in an earlier chunk: its part here is a piece
  const bool before = cs > k0 && (int)(__ldg(bkey + cs - 1) >> lg) == cfirst;
  auto emit = [&](int col, float v) {
    if (before && col == cfirst) {
      o.pfirst[ch] = v;
      o.firstseg[ch] = segbase + col;
    } else {
      o.P[segbase + col] = v;
    }
  };
  int ccol = cfirst;   // the segment open after the keys read so far
  float cval = 0.f;    // and its sum (without acc)
  float acc = 0.f;     // this lane's part of segment ccol from steps that lie inside it
#pragma unroll 2
  for (int base = cs; base < ce; base += 32 * K) {
    uint32_t k[K];
    float p[K];
    const uint4* kq = reinterpret_cast<const uint4*>(bkey + base + K * lane);
    const float4* vq = reinterpret_cast<const float4*>(bval + base + K * lane);
#pragma unroll
    for (int i = 0; i < K / 4; ++i) {
      const uint4 kk = __ldg(kq + i);
      const float4 vv = __ldg(vq + i);
      k[4 * i] = kk.x, k[4 * i + 1] = kk.y, k[4 * i + 2] = kk.z, k[4 * i + 3] = kk.w;
      p[4 * i] = vv.x, p[4 * i + 1] = vv.y, p[4 * i + 2] = vv.z, p[4 * i + 3] = vv.w;
    }
#pragma unroll
    for (int i = 0; i < K; ++i) p[i] *= lds_f32_nc(sbase + 4u * (k[i] & mask));
    // a step inside the open segment (its last key in column ccol; keys are
    // sorted) only adds to the lane's part
    if ((int)(__shfl_sync(FULL_MASK, k[K - 1], 31) >> lg) == ccol) {
#pragma unroll
      for (int i = 0; i < K; ++i) acc += p[i];
      continue;
    }
    cval += warp_sum_f(acc);
    acc = 0.f;
    // runs inside the lane
    const int c0 = (int)(k[0] >> lg);
    int rc = c0;
    float run = p[0], head = 0.f;
    bool whole = true;   // one column over the lane's K keys
#pragma unroll
    for (int i = 1; i < K; ++i) {
      const int ci = (int)(k[i] >> lg);
      if (ci != rc) {
        if (whole) {
          head = run;
          whole = false;
        } else {
          o.P[segbase + rc] = run;   // began and ended inside the lane
        }
        rc = ci;
        run = 0.f;
      }
      run += p[i];
    }
    // the open segment joins lane 0's head, or it ended with the last step
    if (lane == 0) {
      if (c0 == ccol) {
        if (whole)
          run = cval + run;
        else
          head = cval + head;
      } else {
        emit(ccol, cval);
      }
    }
    // tails carried across lanes: segmented inclusive scan, a segment
    // starting at lane l unless l continues lane l - 1's tail with one column
    const int kprev = __shfl_up_sync(FULL_MASK, rc, 1);
    float S = run;
    bool f = lane == 0 || !whole || kprev != c0;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const float Su = __shfl_up_sync(FULL_MASK, S, d);
      const bool fu = __shfl_up_sync(FULL_MASK, f ? 1 : 0, d) != 0;
      if (lane >= d) {
        if (!f) S = Su + S;
        f = f || fu;
      }
    }
    const float Sprev = __shfl_up_sync(FULL_MASK, S, 1);
    const int cnext = __shfl_down_sync(FULL_MASK, c0, 1);
    if (!whole) emit(c0, (lane > 0 && kprev == c0) ? Sprev + head : head);
    if (lane < 31 && cnext != rc) emit(rc, S);
    ccol = __shfl_sync(FULL_MASK, rc, 31);
    cval = __shfl_sync(FULL_MASK, S, 31);
  }
  cval += warp_sum_f(acc);
  // the segment open at the chunk's end: continues past it (within the
  // block), or ends exactly there
  const bool cont = ce < k1 && (int)(__ldg(bkey + ce) >> lg) == ccol;
  if (lane == 0) {
    if (before && ccol == cfirst) {
      o.pfirst[ch] = cval;
      o.firstseg[ch] = segbase + ccol;
    } else if (cont) {
      o.plast[ch] = cval;
      o.lastseg[ch] = segbase + ccol;
    } else {
      o.P[segbase + ccol] = cval;
    }
  }
}

__global__ void __launch_bounds__(kBcolThreads, kBcolMinBlocks)
    scalar_bcol_kernel(const int32_t* __restrict__ blkptr, const uint32_t* __restrict__ bkey,
                       const float* __restrict__ bval, int nb, int lg, int m, int H,
                       int nchunks, const float* __restrict__ rvec, BcolOut o) {
  extern __shared__ __align__(16) float sr[];   // 2^lg floats
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int C0 = (int)(((long long)nchunks * blockIdx.x) / gridDim.x);
  const int C1 = (int)(((long long)nchunks * (blockIdx.x + 1)) / gridDim.x);
  if (C0 >= C1) return;   // CTA-uniform
  const uint32_t mask = (1u << lg) - 1u;
  const uint32_t sbase = smem_u32(sr);
  // the block holding chunk C0: the last b with blkptr[b] <= C0 * chunk
  int b = warp_lower_bound(blkptr, 0, nb + 1, C0 * kBcolChunk + 1) - 1;
  for (int cs_blk = C0; cs_blk < C1;) {
    const int k0 = __ldg(blkptr + b), k1 = __ldg(blkptr + b + 1);
    const int bc0 = max(cs_blk, k0 / kBcolChunk), bc1 = min(C1, k1 / kBcolChunk);
    if (bc0 < bc1) {   // CTA-uniform
      // the block's rows of r (r0 = b * 2^lg is a multiple of 16 rows: the
      // float4 copies are aligned); rows past m are never read
      const int r0 = b << lg;
      const int cnt = min(1 << lg, m - r0);
      const int n4 = cnt >> 2;
      const float4* src = reinterpret_cast<const float4*>(rvec + r0);
#pragma unroll 4
      for (int i = threadIdx.x; i < n4; i += blockDim.x)
        reinterpret_cast<float4*>(sr)[i] = __ldg(src + i);
      for (int i = 4 * n4 + threadIdx.x; i < cnt; i += blockDim.x) sr[i] = __ldg(rvec + r0 + i);
      __syncthreads();
      for (int ch = bc0 + warp; ch < bc1; ch += kBcolWarps) {
        if (kBcolLaneRuns)
          bcol_chunk_lanes(ch, b, k0, k1, lg, H, mask, sbase, bkey, bval, o, lane);
        else
          bcol_chunk_windows(ch, b, k0, k1, lg, H, mask, sbase, bkey, bval, o, lane);
      }
      __syncthreads();   // the block's r stays until every warp is done
    }
    cs_blk = max(cs_blk, bc1);
    ++b;
  }
}

// Pieces of segments cut by chunk boundaries: the last piece of the chunk
// where a segment begins plus the first piece of each following chunk that
// continues it.  One warp per chunk that leaves a last piece; its lanes read
// the following chunks 32 at a time (a segment's chunks are consecutive, so
// the run ends at the first chunk that does not continue it) and the pieces
// are summed in a fixed order: lane-strided, then a butterfly.
__global__ void scalar_bcol_fix(int nchunks, const float* __restrict__ pfirst,
                                const float* __restrict__ plast,
                                const int* __restrict__ firstseg, const int* __restrict__ lastseg,
                                float* __restrict__ P) {
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  for (int c = blockIdx.x * wpb + (threadIdx.x >> 5); c < nchunks; c += gridDim.x * wpb) {
    const int s = __ldg(lastseg + c);   // warp-uniform
    if (s < 0) continue;
    float t = 0.f;
    for (int base = c + 1; base < nchunks; base += 32) {
      const int cc = base + lane;
      int fs = -1;
      float pv = 0.f;
      if (cc < nchunks) {   // both loads in flight together (pv unused off the run)
        fs = __ldg(firstseg + cc);
        pv = __ldg(pfirst + cc);
      }
      const bool in = fs == s;
      if (in) t += pv;
      if (__ballot_sync(FULL_MASK, in) != FULL_MASK) break;   // warp-uniform
    }
    t = warp_sum_f(t);
    if (lane == 0) P[s] = __ldg(plast + c) + t;
  }
}

// out[col(h)] = sum over blocks b of P[b * H + h], b ascending; col(h) =
// cols[h], or h when cols is NULL.
__global__ void scalar_bcol_combine(const float* __restrict__ P, int nb, int H,
                                    const int32_t* __restrict__ cols, float* __restrict__ out) {
  for (int h = blockIdx.x * blockDim.x + threadIdx.x; h < H; h += gridDim.x * blockDim.x) {
    float t = 0.f;
    int b = 0;
    for (; b + 8 <= nb; b += 8) {   // eight loads in flight, added in block order
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldg(P + (size_t)(b + u) * H + h);
#pragma unroll
      for (int u = 0; u < 8; ++u) t += v[u];
    }
    for (; b < nb; ++b) t += __ldg(P + (size_t)b * H + h);
    out[cols ? __ldg(cols + h) : h] = t;
  }
}

// Before the row pass: with ranked columns v'[c] = v[rankcol[c]] and the
// accumulator of the atomic transposed product (ranked order) is zeroed; a
// buffer of the column pass that must start at zero (the blocked twin's
// per-block sums, 16-byte aligned) is cleared in the same launch.
__global__ void rank_prep_kernel(const float* __restrict__ v, const int32_t* __restrict__ rankcol,
                                 int n, float* __restrict__ vr, float* __restrict__ acc,
                                 float* __restrict__ zbuf, long long zn) {
  const int t0 = blockIdx.x * blockDim.x + threadIdx.x, nt = gridDim.x * blockDim.x;
  for (int c = t0; c < n; c += nt) {
    vr[c] = __ldg(v + __ldg(rankcol + c));
    if (acc) acc[c] = 0.f;
  }
  const long long z4 = zn >> 2;
  for (long long i = t0; i < z4; i += nt)
    reinterpret_cast<float4*>(zbuf)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  for (long long i = 4 * z4 + t0; i < zn; i += nt) zbuf[i] = 0.f;
}

// Ranked columns, after an atomic row pass: out[rankcol[c]] = acc[c].
__global__ void rank_finish_kernel(const float* __restrict__ acc,
                                   const int32_t* __restrict__ rankcol, int n,
                                   float* __restrict__ out) {
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < n; c += gridDim.x * blockDim.x)
    out[__ldg(rankcol + c)] = __ldg(acc + c);
}

namespace {

template <class Op, bool EMIT>
cudaError_t launch_rows(const char* name, const Op& op, const sdad_csr* A, const int32_t* cols,
                        double* loss, double scale, float* dA, float* dxa, float* rvec,
                        const WsLayout& L, cudaStream_t st) {
  const int nblk = (A->m + 31) / 32;
  // blocks of 32 rows per warp: two on large matrices; one when that leaves
  // fewer warps than the GPU holds (a small matrix is latency-bound: more
  // warps, fewer dependent round trips each)
  const int bpw = nblk >= device_sm_count() * 64 * kRowBlocksPerWarp ? kRowBlocksPerWarp : 1;
  int grid = std::max(1, (nblk + kRowWarps * bpw - 1) / (kRowWarps * bpw));
  grid = std::min(grid, kMaxPartials);
  {
    KTimer t(name, st);
    scalar_row_kernel<Op, EMIT><<<grid, kRowThreads, 0, st>>>(
        A->rowptr, cols, A->val, A->m, op, rvec, dA, dxa, L.hdr, L.partials, scale, loss);
  }
  return cudaGetLastError();
}

template <class Op>
cudaError_t row_pass(const char* name, const Op& op, const sdad_csr* A, const int32_t* cols,
                     double* loss, double scale, float* dA, float* dxa, float* rvec,
                     const WsLayout& L, cudaStream_t st) {
  if (dA || dxa) return launch_rows<Op, true>(name, op, A, cols, loss, scale, dA, dxa, rvec, L, st);
  return launch_rows<Op, false>(name, op, A, cols, loss, scale, dA, dxa, rvec, L, st);
}

cudaError_t rows_for(int expr, const sdad_csr* A, const float* v, const float* y,
                     const int32_t* cols, double* loss, float* dA, float* dxa, float* rvec,
                     const WsLayout& L, cudaStream_t st) {
  if (expr == SDAD_EXPR_LSQ)
    return row_pass("lsq_row", LsqOp{v, y}, A, cols, loss, 1.0, dA, dxa, rvec, L, st);
  return row_pass("logreg_row", LogregOp{v, y, 1.0f / (float)A->m}, A, cols, loss,
                  1.0 / (double)A->m, dA, dxa, rvec, L, st);
}

}  // namespace

// Column pass over the CSC twin (colptr, rowidx, val_csc) holding nnz keys;
// rvec NULL: the column sums (rowidx is not read).
cudaError_t col_pass(const sdad_csr* A, int64_t nnz, const float* rvec, float* out,
                     const WsLayout& L, cudaStream_t st) {
  const int cap = nnz >= (int64_t(1) << 22) ? kColChunkLarge : kColChunkSmall;
  const int nchunks = nnz <= 0 ? 1 : (int)((nnz + cap - 1) / cap);
  cudaError_t e = zero_f32(out, (size_t)A->n, st);
  if (e != cudaSuccess) return e;
  const int warps = nchunks;   // one chunk per warp
  const int grid = std::max(1, (warps + kColWarps - 1) / kColWarps);
  {
    KTimer t(rvec ? "scalar_col" : "col_sums", st);
    const ColPieces pc{out, L.pfirst, L.plast, L.lastseg};
    auto go = [&](auto kern) {
      kern<<<grid, kColThreads, 0, st>>>(A->colptr, A->rowidx, A->val_csc, A->n, (int)nnz,
                                          nchunks, rvec, pc);
    };
    if (cap == kColChunkLarge)
      rvec ? go(scalar_colv_kernel<kColChunkLarge, false>)
           : go(scalar_colv_kernel<kColChunkLarge, true>);
    else
      rvec ? go(scalar_colv_kernel<kColChunkSmall, false>)
           : go(scalar_colv_kernel<kColChunkSmall, true>);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int fgrid = std::max(1, std::min((nchunks + 7) / 8, device_sm_count() * 16));
  {
    KTimer t("scalar_col_fix", st);
    scalar_col_fix<<<fgrid, 256, 0, st>>>(A->colptr, nchunks, cap, L.pfirst, L.plast, L.lastseg,
                                          out);
  }
  return cudaGetLastError();
}

namespace {

// The per-block sums P of the blocked column pass ([nb x H]).
long long bcol_sums(const sdad_csr* A) {
  const int lg = A->bcsc_log2;
  const long long nb = ((long long)A->m + (1ll << lg) - 1) >> lg;
  return nb * (long long)(csr_split(A) ? A->bcsc_ncols : A->n);
}

// Column pass over the row-blocked CSC twin (P = L.bP is zero on entry: the
// prep kernel clears it); when the twin holds some columns only, the others
// first go through the plain column pass over their CSC twin (which zeroes
// every output entry, the blocked columns' included).
cudaError_t bcol_pass(const sdad_csr* A, const float* rvec, float* out, const WsLayout& L,
                      cudaStream_t st) {
  const int lg = A->bcsc_log2;
  const bool split = csr_split(A);
  const int H = split ? A->bcsc_ncols : A->n;
  const int nb = (int)(((int64_t)A->m + (int64_t(1) << lg) - 1) >> lg);
  const int nchunks = (int)(A->bcsc_nnz / kBcolChunk);
  const size_t smem = sizeof(float) << lg;
  cudaError_t e;
  if (split && (e = col_pass(A, A->bcsc_rest_nnz, rvec, out, L, st)) != cudaSuccess) return e;
  // the limit belongs to the device: raised once per (kernel, device)
  e = ensure_dynamic_smem(reinterpret_cast<const void*>(scalar_bcol_kernel),
                          (int)(sizeof(float) << SDAD_BCSC_MAX_LOG2));
  if (e != cudaSuccess) return e;
  const int sms = device_sm_count();
  if (nchunks > 0) {
    int per_sm = 1;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, scalar_bcol_kernel, kBcolThreads,
                                                      smem);
    if (e != cudaSuccess) return e;
    const int grid = std::min(nchunks, sms * std::max(per_sm, 1));
    {
      KTimer t("scalar_bcol", st);
      scalar_bcol_kernel<<<grid, kBcolThreads, smem, st>>>(
          A->bcsc_ptr, A->bcsc_key, A->bcsc_val, nb, lg, A->m, H, nchunks, rvec,
          BcolOut{L.bP, L.bpfirst, L.bplast, L.bfirstseg, L.blastseg});
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int fgrid = std::max(1, std::min((nchunks + 7) / 8, sms * 8));
    {
      KTimer t("scalar_bcol_fix", st);
      scalar_bcol_fix<<<fgrid, 256, 0, st>>>(nchunks, L.bpfirst, L.bplast, L.bfirstseg,
                                             L.blastseg, L.bP);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (H > 0) {
    const int cgrid = std::max(1, std::min((H + 255) / 256, sms * 4));
    KTimer t("bcol_combine", st);
    scalar_bcol_combine<<<cgrid, 256, 0, st>>>(L.bP, nb, H, split ? A->bcsc_cols : nullptr, out);
  }
  return cudaGetLastError();
}

}  // namespace

bool scalar_uses_csc(const sdad_csr* A, bool want_dvec, sdad_tmode tmode) {
  (void)A;
  return want_dvec && tmode != SDAD_T_ATOMIC;   // AUTO: the deterministic column pass
}

cudaError_t run_scalar(int expr, const sdad_csr* A, const float* xin, const float* y,
                       double* loss, float* dvec, float* dA, sdad_tmode tmode,
                       const WsLayout& L, cudaStream_t st) {
  const bool csc = scalar_uses_csc(A, dvec != nullptr, tmode);
  const bool ranked = csr_ranked(A) && L.vr;
  const bool atomic = dvec && !csc;
  const int n = A->n;
  cudaError_t e;
  const float* v = xin;
  const int32_t* cols = A->colidx;
  float* acc = dvec;
  const bool blocked = csc && csr_blocked(A) && L.bP;
  const long long zn = blocked ? bcol_sums(A) : 0;   // the blocked pass's sums, cleared first
  bool cleared = false;
  if (ranked) {
    if (n > 0 || zn > 0) {
      const long long work = std::max<long long>(n, zn / 4);
      const int grid = (int)std::max<long long>(
          1, std::min<long long>((work + 255) / 256, device_sm_count() * 4));
      KTimer t("rank_prep", st);
      rank_prep_kernel<<<grid, 256, 0, st>>>(xin, A->rankcol, n, L.vr, atomic ? L.vacc : nullptr,
                                             L.bP, zn);
      cleared = true;
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    v = L.vr;
    cols = A->rcolidx;
    acc = L.vacc;
  } else if (atomic) {
    if ((e = zero_f32(dvec, (size_t)n, st)) != cudaSuccess) return e;
  }
  if (zn > 0 && !cleared && (e = zero_f32(L.bP, (size_t)zn, st)) != cudaSuccess) return e;
  e = rows_for(expr, A, v, y, cols, loss, dA, atomic ? acc : nullptr, csc ? L.rowvec : nullptr, L,
               st);
  if (e != cudaSuccess) return e;
  if (csc) {
    if (blocked) return bcol_pass(A, L.rowvec, dvec, L, st);
    return col_pass(A, A->nnz, L.rowvec, dvec, L, st);
  }
  if (ranked && atomic && n > 0) {
    const int grid = std::max(1, std::min((n + 255) / 256, device_sm_count() * 4));
    KTimer t("rank_finish", st);
    rank_finish_kernel<<<grid, 256, 0, st>>>(L.vacc, A->rankcol, n, dvec);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Row passes of the paper's matrix kernels (Sec. 7.1), on the same row kernel.
// ---------------------------------------------------------------------------

// SMMM over B: z_k = sum_j B(k,j); f = sum_k c_k z_k with c the column sums
// of A (one per row of B); df/dB at key (k, j) = c_k.
struct SmmmOp {
  const float* __restrict__ c;
  __device__ __forceinline__ const float* vec() const { return c; }
  __device__ __forceinline__ float gather(int) const { return 1.f; }
  __device__ __forceinline__ float pre(int k) const { return __ldg(c + k); }
  __device__ __forceinline__ float finish(float z, float ck, double& term) const {
    term = (double)ck * (double)z;
    return ck;
  }
};

// BATAX, first half: r_i = beta (A X)_i (no scalar).
struct BataxOp {
  const float* __restrict__ x;
  float beta;
  __device__ __forceinline__ const float* vec() const { return x; }
  __device__ __forceinline__ float gather(int j) const { return __ldg(x + j); }
  __device__ __forceinline__ float pre(int) const { return 0.f; }
  __device__ __forceinline__ float finish(float z, float, double& term) const {
    term = 0.0;
    return beta * z;
  }
};

cudaError_t smmm_rows(const sdad_csr* B, const float* colsum, double* f, float* dB,
                      const WsLayout& L, cudaStream_t st) {
  return row_pass("smmm_row", SmmmOp{colsum}, B, B->colidx, f, 1.0, dB, nullptr, nullptr, L, st);
}

cudaError_t batax_rows(const sdad_csr* A, const float* X, float beta, float* r, double* sink,
                       const WsLayout& L, cudaStream_t st) {
  return row_pass("batax_row", BataxOp{X, beta}, A, A->colidx, sink, 1.0, nullptr, nullptr, r, L,
                  st);
}

}  // namespace sdad
