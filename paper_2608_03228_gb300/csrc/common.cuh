// Shared device helpers of the SAKI CUDA library (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/saki.h"

namespace saki {

constexpr int kD = 128;          // head dimension supported by this build
constexpr int kLdS = kD + 1;     // padded leading dimension of d x d tiles in shared memory

// Device status bits (one int per fitted matrix / head).
enum : int { kStNonFinite = 1, kStNotConverged = 2, kStTimeout = 4 };

// ---------------------------------------------------------------- dtype helpers
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Unpack one 16-byte vector of inputs into floats.  NV = elements per vector.
template <typename T> struct Vec;
template <> struct Vec<float> {
  static constexpr int NV = 4;
  __device__ __forceinline__ static void unpack(const uint4& v, float* x) {
    x[0] = __uint_as_float(v.x); x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z); x[3] = __uint_as_float(v.w);
  }
  __device__ __forceinline__ static float load1(const float* p) { return *p; }
  __device__ __forceinline__ static float store_cvt(float v) { return v; }
};
template <> struct Vec<__nv_bfloat16> {
  static constexpr int NV = 8;
  __device__ __forceinline__ static void unpack(const uint4& v, float* x) {
    x[0] = bf16_lo(v.x); x[1] = bf16_hi(v.x); x[2] = bf16_lo(v.y); x[3] = bf16_hi(v.y);
    x[4] = bf16_lo(v.z); x[5] = bf16_hi(v.z); x[6] = bf16_lo(v.w); x[7] = bf16_hi(v.w);
  }
  __device__ __forceinline__ static float load1(const __nv_bfloat16* p) { return __bfloat162float(*p); }
};

template <typename T> __device__ __forceinline__ T from_float(float v);
template <> __device__ __forceinline__ float from_float<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// Two floats rounded to bf16 (nearest even), packed low element first.
__device__ __forceinline__ uint32_t pack_bf16_pair(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// ---------------------------------------------------------------- ranking keys
// A 64-bit key orders candidates by (score descending, index ascending): the high
// word is an order-preserving image of the float score (with -0 folded onto +0),
// the low word the bit-complement of the key index.  Key 0 is below every real
// candidate and marks an empty slot.
__device__ __forceinline__ uint32_t ord_bits(float s) {
  uint32_t b = __float_as_uint(s);
  if ((b & 0x7fffffffu) == 0) b = 0;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float ord_float(uint32_t o) {
  const uint32_t b = (o & 0x80000000u) ? (o & 0x7fffffffu) : ~o;
  return __uint_as_float(b);
}
__device__ __forceinline__ uint64_t make_key(float s, uint32_t j) {
  return ((uint64_t)ord_bits(s) << 32) | (uint64_t)(0xffffffffu - j);
}
__device__ __forceinline__ int32_t key_index(uint64_t key) {
  return key ? (int32_t)(0xffffffffu - (uint32_t)key) : -1;
}
__device__ __forceinline__ float key_score(uint64_t key) {
  return key ? ord_float((uint32_t)(key >> 32)) : -INFINITY;
}

__device__ __forceinline__ uint64_t shfl_xor_u64(uint64_t v, int m) {
  uint32_t lo = __shfl_xor_sync(0xffffffffu, (uint32_t)v, m);
  uint32_t hi = __shfl_xor_sync(0xffffffffu, (uint32_t)(v >> 32), m);
  return ((uint64_t)hi << 32) | lo;
}
__device__ __forceinline__ uint64_t shfl_u64(uint64_t v, int src) {
  uint32_t lo = __shfl_sync(0xffffffffu, (uint32_t)v, src);
  uint32_t hi = __shfl_sync(0xffffffffu, (uint32_t)(v >> 32), src);
  return ((uint64_t)hi << 32) | lo;
}

// Warp-wide bitonic sort into descending order of 32*E keys held "striped":
// element i = e*32 + lane lives in v[e] of that lane.
template <int E>
__device__ __forceinline__ void warp_sort_desc(uint64_t (&v)[E]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32 * E; size <<= 1) {
#pragma unroll
    for (int j = size >> 1; j > 0; j >>= 1) {
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const int i = e * 32 + lane;
        const bool desc = (i & size) == 0;
        if (j >= 32) {
          const int m = j >> 5;
          if ((e & m) == 0) {
            const int pe = e | m;
            const uint64_t a = v[e], b = v[pe];
            const bool sw = desc ? (a < b) : (a > b);
            v[e] = sw ? b : a;
            v[pe] = sw ? a : b;
          }
        } else {
          const uint64_t o = shfl_xor_u64(v[e], j);
          const bool lower = (lane & j) == 0;
          v[e] = (lower == desc) ? (v[e] > o ? v[e] : o) : (v[e] < o ? v[e] : o);
        }
      }
    }
  }
}

// a (descending, 32*E striped) := the 32*E largest of a and b (both descending),
// in descending order.
template <int E>
__device__ __forceinline__ void warp_merge_top(uint64_t (&a)[E], const uint64_t (&b)[E]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    // element n-1-i of b lives in register E-1-e of lane 31-lane
    const uint64_t br = shfl_u64(b[E - 1 - e], 31 - lane);
    a[e] = a[e] > br ? a[e] : br;
  }
  // a is now bitonic; merge it into descending order
#pragma unroll
  for (int j = 16 * E; j > 0; j >>= 1) {
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (j >= 32) {
        const int m = j >> 5;
        if ((e & m) == 0) {
          const int pe = e | m;
          const uint64_t x = a[e], y = a[pe];
          a[e] = x > y ? x : y;
          a[pe] = x > y ? y : x;
        }
      } else {
        const uint64_t o = shfl_xor_u64(a[e], j);
        const bool lower = (lane & j) == 0;
        a[e] = lower ? (a[e] > o ? a[e] : o) : (a[e] < o ? a[e] : o);
      }
    }
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int m = 16; m > 0; m >>= 1) v += __shfl_xor_sync(0xffffffffu, v, m);
  return v;
}

}  // namespace saki
