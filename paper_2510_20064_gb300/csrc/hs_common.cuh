// hs_common.cuh -- device helpers shared by the libhedgefb kernels.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {

constexpr float kLog2e = 1.4426950408889634f;

// ---- element decode -------------------------------------------------------
// bf16 is the upper half of a binary32, so widening is a shift (exact);
// fp16 widens with the hardware conversion (exact); fp32 is read as is.

template <int DT>
struct Elem;

template <>
struct Elem<HS_BF16> {
  static constexpr int kBytes = 2;
  static constexpr int kVec = 8;  // elements per 16-byte load
  __device__ static __forceinline__ float one(const void* p, int64_t i) {
    return __uint_as_float(uint32_t(__ldg(static_cast<const uint16_t*>(p) + i)) << 16);
  }
  __device__ static __forceinline__ void vec(const void* p, int64_t i, float (&v)[kVec]) {
    uint4 w = __ldg(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p) + i));
    uint32_t a[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[2 * j] = __uint_as_float(a[j] << 16);
      v[2 * j + 1] = __uint_as_float(a[j] & 0xffff0000u);
    }
  }
};

template <>
struct Elem<HS_FP16> {
  static constexpr int kBytes = 2;
  static constexpr int kVec = 8;
  __device__ static __forceinline__ float one(const void* p, int64_t i) {
    return __half2float(__ushort_as_half(__ldg(static_cast<const unsigned short*>(p) + i)));
  }
  __device__ static __forceinline__ void vec(const void* p, int64_t i, float (&v)[kVec]) {
    uint4 w = __ldg(reinterpret_cast<const uint4*>(static_cast<const unsigned short*>(p) + i));
    uint32_t a[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      __half2 h = *reinterpret_cast<__half2*>(&a[j]);
      float2 f = __half22float2(h);
      v[2 * j] = f.x;
      v[2 * j + 1] = f.y;
    }
  }
};

template <>
struct Elem<HS_FP32> {
  static constexpr int kBytes = 4;
  static constexpr int kVec = 4;
  __device__ static __forceinline__ float one(const void* p, int64_t i) {
    return __ldg(static_cast<const float*>(p) + i);
  }
  __device__ static __forceinline__ void vec(const void* p, int64_t i, float (&v)[kVec]) {
    float4 w = __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(p) + i));
    v[0] = w.x; v[1] = w.y; v[2] = w.z; v[3] = w.w;
  }
};

// ---- arithmetic -----------------------------------------------------------

// 2^x on the MUFU unit (flushes subnormal results to 0; those terms are
// below 2^-126 of the row maximum and do not change an fp32 sum).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// max that propagates NaN: once m is NaN it stays NaN.
__device__ __forceinline__ float max_nan(float m, float x) {
  return (x > m || x != x) ? x : m;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max_nan(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = max_nan(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ int warp_min_int(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Record a data error for the caller without overwriting an earlier one.
__device__ __forceinline__ void report(int* dev_status, int code) {
  if (dev_status) atomicCAS(dev_status, HS_OK, code);
}

}  // namespace hs
