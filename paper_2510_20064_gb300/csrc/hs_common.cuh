// hs_common.cuh -- device helpers shared by the libhedgefb kernels.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kMaxDevices = 64;  // devices a host-side launch cache keeps entries for

// ---- programmatic dependent launch ------------------------------------------
// Every kernel here is launched with programmatic stream serialization, so
// that it can be scheduled while the previous kernel of the stream finishes.
// pdl_wait() blocks until that kernel has completed and its memory is
// visible: each kernel calls it before touching global memory another
// kernel may write or read.  pdl_trigger() lets the next kernel be scheduled
// early.  Both are no-ops in a launch without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

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

// ---- vocabulary chunks ------------------------------------------------------
// A chunk of THREADS * UNROLL * kVec consecutive logits of one row: with VEC,
// slot s of thread t is element v0 + ((s / kVec) * THREADS + t) * kVec +
// s % kVec (16-byte loads, coalesced across the block); without VEC (rows
// not 16-byte aligned) it is v0 + s * THREADS + t.  A thread's slots visit
// increasing v either way.

template <int DT, bool VEC, int THREADS>
__device__ __forceinline__ int64_t slot_pos(int64_t v0, int s, int t) {
  constexpr int kV = Elem<DT>::kVec;
  if (VEC) return v0 + (int64_t((s / kV) * THREADS + t)) * kV + (s % kV);
  return v0 + int64_t(s) * THREADS + t;
}

// Load one chunk of a row into x[] (-inf past the end of the row).
template <int DT, bool VEC, int THREADS, int UNROLL>
__device__ __forceinline__ void load_chunk(const void* row, int64_t v0, int V,
                                           float (&x)[UNROLL * Elem<DT>::kVec]) {
  constexpr int kV = Elem<DT>::kVec;
  const int t = threadIdx.x;
#pragma unroll
  for (int u = 0; u < UNROLL; ++u) {
    if (VEC) {
      const int64_t v = v0 + int64_t(u * THREADS + t) * kV;
      float tmp[kV];
      if (v < V) {
        Elem<DT>::vec(row, v, tmp);
      } else {
#pragma unroll
        for (int e = 0; e < kV; ++e) tmp[e] = -INFINITY;
      }
#pragma unroll
      for (int e = 0; e < kV; ++e) x[u * kV + e] = tmp[e];
    } else {
#pragma unroll
      for (int e = 0; e < kV; ++e) {
        const int64_t v = slot_pos<DT, false, THREADS>(v0, u * kV + e, t);
        x[u * kV + e] = v < V ? Elem<DT>::one(row, v) : -INFINITY;
      }
    }
  }
}

template <int DT>
__device__ __forceinline__ const void* row_ptr(const void* base, int64_t row, int V) {
  return static_cast<const char*>(base) + row * int64_t(V) * Elem<DT>::kBytes;
}

// Target row of tile (b,k) = b*P + k: a chain row, or the path node of a
// draft tree (an out-of-range node reads node 0 and sets *bad_path).
template <int DT>
__device__ __forceinline__ const void* target_row(const void* target, const int32_t* path,
                                                  int M, int P, int64_t tile, int V,
                                                  bool* bad_path) {
  if (!path) return row_ptr<DT>(target, tile, V);
  const int64_t b = tile / P;
  int node = path[tile];
  *bad_path = node < 0 || node >= M;
  if (*bad_path) node = 0;
  return row_ptr<DT>(target, b * M + node, V);
}

// Record a data error for the caller without overwriting an earlier one.
__device__ __forceinline__ void report(int* dev_status, int code) {
  if (dev_status) atomicCAS(dev_status, HS_OK, code);
}

}  // namespace hs
