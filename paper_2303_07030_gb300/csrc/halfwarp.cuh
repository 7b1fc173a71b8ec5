// halfwarp.cuh -- helpers of the kernels that work on 64-wide fp32 rows with
// half a warp per row: lane l of half h = l / 16 holds elements
// 4 (l % 16) .. 4 (l % 16) + 3, so a warp holds two rows (two keys) at once.
#pragma once

#include "common.cuh"

namespace sdad {

constexpr int kPairs = 8;   // key pairs per batch (16 keys)

__device__ __forceinline__ float4 ld4(const float* base, int r, int sl) {
  return __ldg(reinterpret_cast<const float4*>(base + (size_t)r * 64) + sl);
}
__device__ __forceinline__ void st4(float* base, int r, int sl, float4 v) {
  reinterpret_cast<float4*>(base + (size_t)r * 64)[sl] = v;
}
__device__ __forceinline__ float4 zero4() { return make_float4(0.f, 0.f, 0.f, 0.f); }
__device__ __forceinline__ float4 fma4(float a, float4 x, float4 acc) {
  return make_float4(fmaf(a, x.x, acc.x), fmaf(a, x.y, acc.y), fmaf(a, x.z, acc.z),
                     fmaf(a, x.w, acc.w));
}
__device__ __forceinline__ float dot4(float4 a, float4 b) {
  return fmaf(a.w, b.w, fmaf(a.z, b.z, fmaf(a.y, b.y, a.x * b.x)));
}
// the sum of the two halves' partials (every lane gets its elements' total)
__device__ __forceinline__ float4 join_halves(float4 v) {
  return make_float4(v.x + __shfl_xor_sync(FULL_MASK, v.x, 16),
                     v.y + __shfl_xor_sync(FULL_MASK, v.y, 16),
                     v.z + __shfl_xor_sync(FULL_MASK, v.z, 16),
                     v.w + __shfl_xor_sync(FULL_MASK, v.w, 16));
}

// t[u] holds this lane's part of value u of its half (eight values); returns
// the half's total of value (sl >> 1) & 7, sl = lane % 16 (a butterfly that
// halves the values at each of the first three steps: 8 shuffles for the 16
// totals of the warp).
__device__ __forceinline__ float reduce_half8(float (&t)[kPairs], int lane) {
  static_assert(kPairs == 8, "eight values");
  const bool b3 = lane & 8, b2 = lane & 4, b1 = lane & 2;
  float u4[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {   // keep values 4*b3 + i, send the other half
    const float keep = b3 ? t[i + 4] : t[i], send = b3 ? t[i] : t[i + 4];
    u4[i] = keep + __shfl_xor_sync(FULL_MASK, send, 8);
  }
  float w[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {   // keep 2*b2 + i of u4
    const float keep = b2 ? u4[i + 2] : u4[i], send = b2 ? u4[i] : u4[i + 2];
    w[i] = keep + __shfl_xor_sync(FULL_MASK, send, 4);
  }
  const float keep = b1 ? w[1] : w[0], send = b1 ? w[0] : w[1];
  float x = keep + __shfl_xor_sync(FULL_MASK, send, 2);
  x += __shfl_xor_sync(FULL_MASK, x, 1);
  return x;   // value 4*b3 + 2*b2 + b1 = (sl >> 1) & 7
}

// The same for four values: returns the half's total of value (sl >> 2) & 3
// (6 shuffles for the 8 totals of the warp).
__device__ __forceinline__ float reduce_half4(float (&t)[4], int lane) {
  const bool b3 = lane & 8, b2 = lane & 4;
  float u2[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {   // keep values 2*b3 + i, send the other half
    const float keep = b3 ? t[i + 2] : t[i], send = b3 ? t[i] : t[i + 2];
    u2[i] = keep + __shfl_xor_sync(FULL_MASK, send, 8);
  }
  const float keep = b2 ? u2[1] : u2[0], send = b2 ? u2[0] : u2[1];
  float x = keep + __shfl_xor_sync(FULL_MASK, send, 4);
  x += __shfl_xor_sync(FULL_MASK, x, 2);
  x += __shfl_xor_sync(FULL_MASK, x, 1);
  return x;   // value 2*b3 + b2 = (sl >> 2) & 3
}

__device__ __forceinline__ float reduce_half(float (&t)[8], int lane) { return reduce_half8(t, lane); }
__device__ __forceinline__ float reduce_half(float (&t)[4], int lane) { return reduce_half4(t, lane); }

// The lane holding the total of key offset o (0..15) of a 16-key batch after
// reduce_half8: key o is pair o / 2 of half o % 2.
__device__ __forceinline__ int batch_src_lane(int o) { return ((o & 1) << 4) | ((o >> 1) << 1); }
// ... and the key offset whose total lane `lane` holds
__device__ __forceinline__ int batch_key_of_lane(int lane) {
  return 2 * (((lane & 15) >> 1) & 7) + (lane >> 4);
}

}  // namespace sdad
