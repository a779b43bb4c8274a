// hs_greedy.cu -- greedy feedback: alpha = [argmax q_i == argmax p]
// (Thm 2 with branching L = 1 under a greedy target), e_len by Thm 3.
//
//   argmax_chunk_kernel     one CTA per (row, 16K-logit chunk): NaN-propagating
//                           max of the stored logits and the first index
//                           holding it; every logit is read once, 8 16-byte
//                           loads in flight per thread
//   greedy_finalize_kernel  one warp per drafter row (i, b, k): combines the
//                           chunk partials of its target and drafter rows in
//                           chunk order (first index wins ties) and compares;
//                           the last of the P warps of (i, b) to finish (an
//                           atomic count the argmax kernel zeroes) forms e_len
// All of it is exact: maxima and indices of the stored values.
#include <math.h>
#include <stdint.h>

#include <climits>

#include "hs_common.cuh"
#include "hs_greedy.h"

namespace hs {
namespace greedy {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 8;

template <int DT>
__host__ __device__ constexpr int64_t chunk_of() {
  return int64_t(kThreads) * kUnroll * Elem<DT>::kVec;
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) argmax_chunk_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M,
    const void* __restrict__ drafter, int B, int P, int V, Part* __restrict__ parts,
    int nchunk, int* __restrict__ counters, int ncounters) {
  pdl_wait();
  if (counters && blockIdx.x == 0 && blockIdx.y == 0)
    for (int x = threadIdx.x; x < ncounters; x += kThreads) counters[x] = 0;
  constexpr int kV = Elem<DT>::kVec;
  constexpr int kS = kUnroll * kV;
  __shared__ float red_m[kWarps];
  __shared__ int red_a[kWarps];
  const int64_t r = blockIdx.x;
  const int j = blockIdx.y;
  const int64_t BP = int64_t(B) * P;
  bool bad_path = false;
  const void* row = r < BP ? target_row<DT>(target, path, M, P, r, V, &bad_path)
                           : row_ptr<DT>(drafter, r - BP, V);
  const int64_t v0 = int64_t(j) * chunk_of<DT>();
  float x[kS];
  load_chunk<DT, VEC, kThreads, kUnroll>(row, v0, V, x);
  // slots visit increasing v, so a strict '>' keeps the first index; a NaN
  // replaces m and then stays
  float m = -INFINITY;
  int arg = INT_MAX;
#pragma unroll
  for (int s = 0; s < kS; ++s) {
    const int64_t v = slot_pos<DT, VEC, kThreads>(v0, s, threadIdx.x);
    if (v < V && (x[s] > m || x[s] != x[s])) {
      m = x[s];
      arg = int(v);
    }
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  const float wm = warp_max_nan(m);
  const int wa = warp_min_int(m == wm ? arg : INT_MAX);
  if (l == 0) {
    red_m[w] = wm;
    red_a[w] = wa;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float bm = red_m[0];
    for (int q = 1; q < kWarps; ++q) bm = max_nan(bm, red_m[q]);
    int ba = INT_MAX;
    for (int q = 0; q < kWarps; ++q)
      if (red_m[q] == bm && red_a[q] < ba) ba = red_a[q];
    parts[r * nchunk + j] = Part{bm, ba};
  }
  pdl_trigger();
}

// Row argmax from its chunk partials, by one warp: (max, first index).
__device__ __forceinline__ void combine(const Part* __restrict__ pr, int nchunk, float& m,
                                        int& arg) {
  const int l = threadIdx.x & 31;
  float lm = -INFINITY;
  int la = INT_MAX;
  for (int j = l; j < nchunk; j += 32) {  // increasing chunk order per lane
    const Part q = pr[j];
    if (q.m > lm || q.m != q.m) {
      lm = q.m;
      la = q.idx;
    }
  }
  m = warp_max_nan(lm);
  arg = warp_min_int(lm == m ? la : INT_MAX);
}

__global__ void greedy_finalize_kernel(const Part* __restrict__ parts, int nchunk,
                                       const int32_t* __restrict__ path, int M, int N, int B,
                                       int P, float* __restrict__ alpha,
                                       float* __restrict__ e_len, int* __restrict__ counters,
                                       int* dev_status) {
  pdl_wait();
  const int64_t r = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;  // row (i, b, k)
  const int64_t BP = int64_t(B) * P;
  if (r >= int64_t(N) * BP) return;  // whole warp
  const int l = threadIdx.x & 31;
  const int64_t tile = r % BP;
  float mt, md;
  int at, ad;
  combine(parts + tile * nchunk, nchunk, mt, at);
  combine(parts + (BP + r) * nchunk, nchunk, md, ad);
  const bool bad_path = path && (path[tile] < 0 || path[tile] >= M);
  int last = 0;
  if (l == 0) {
    float a;
    if (bad_path || !isfinite(mt) || !isfinite(md)) {
      a = __int_as_float(0x7fc00000);
      report(dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
    } else {
      a = (at == ad) ? 1.f : 0.f;
    }
    alpha[r] = a;
    if (e_len) {
      __threadfence();  // alpha[r] before the count
      last = atomicAdd(&counters[r / P], 1) == P - 1;
    }
  }
  // the last warp of (i, b) forms e_len = 1 + sum_{k<K} prod_{j<=k} alpha_j
  if (__shfl_sync(0xffffffffu, last, 0) && l == 0) {
    __threadfence();
    const int64_t ib = r / P;
    float e = 1.f, prod = 1.f;
    for (int k = 0; k < P - 1; ++k) {
      prod *= __ldcg(alpha + ib * P + k);
      e += prod;
    }
    e_len[ib] = e;
  }
}

// Partials, then one counter per (i, b) at the next 256-byte boundary.
size_t parts_bytes(int N, int B, int P, int V, int dtype) {
  const int64_t ch = dtype == HS_FP32 ? chunk_of<HS_FP32>() : chunk_of<HS_BF16>();
  const int64_t nchunk = (V + ch - 1) / ch;
  const size_t bytes = size_t(int64_t(B) * P * (int64_t(N) + 1) * nchunk) * sizeof(Part);
  return (bytes + 255) & ~size_t(255);
}

template <int DT, bool VEC>
hs_status launch_t(const void* target, const int32_t* path, int M, const void* drafter, int N,
                   int B, int P, int V, float* alpha, float* e_len, void* ws, int* dev_status,
                   cudaStream_t s) {
  Part* parts = static_cast<Part*>(ws);
  const int nchunk = int((V + chunk_of<DT>() - 1) / chunk_of<DT>());
  const unsigned rows = unsigned(int64_t(B) * P * (int64_t(N) + 1));
  int* counters = e_len ? reinterpret_cast<int*>(static_cast<char*>(ws) +
                                                  parts_bytes(N, B, P, V, DT))
                        : nullptr;
  if (launch_pdl(argmax_chunk_kernel<DT, VEC>, dim3(rows, unsigned(nchunk)), dim3(kThreads), 0,
                 s, target, path, M, drafter, B, P, V, parts, nchunk, counters,
                 N * B) != cudaSuccess)
    return HS_ERR_CUDA;
  const int64_t threads = int64_t(N) * B * P * 32;
  if (launch_pdl(greedy_finalize_kernel, dim3(unsigned((threads + 255) / 256)), dim3(256), 0, s,
                 parts, nchunk, path, M, N, B, P, alpha, e_len, counters,
                 dev_status) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

template <int DT>
hs_status launch_dt(bool vec, const void* target, const int32_t* path, int M,
                    const void* drafter, int N, int B, int P, int V, float* alpha, float* e_len,
                    void* ws, int* dev_status, cudaStream_t s) {
  if (vec)
    return launch_t<DT, true>(target, path, M, drafter, N, B, P, V, alpha, e_len, ws,
                              dev_status, s);
  return launch_t<DT, false>(target, path, M, drafter, N, B, P, V, alpha, e_len, ws,
                             dev_status, s);
}

}  // namespace

int64_t chunk_elems(int dtype) {
  return dtype == HS_FP32 ? chunk_of<HS_FP32>() : chunk_of<HS_BF16>();
}

size_t workspace_bytes(int N, int B, int P, int V, int dtype) {
  return parts_bytes(N, B, P, V, dtype) + size_t(N) * B * sizeof(int);
}

hs_status launch(bool vec, const void* target, const int32_t* path, int M, const void* drafter,
                 int dtype, int N, int B, int P, int V, float* alpha, float* e_len, void* ws,
                 int* dev_status, cudaStream_t s) {
  switch (dtype) {
    case HS_BF16:
      return launch_dt<HS_BF16>(vec, target, path, M, drafter, N, B, P, V, alpha, e_len, ws,
                                dev_status, s);
    case HS_FP16:
      return launch_dt<HS_FP16>(vec, target, path, M, drafter, N, B, P, V, alpha, e_len, ws,
                                dev_status, s);
    default:
      return launch_dt<HS_FP32>(vec, target, path, M, drafter, N, B, P, V, alpha, e_len, ws,
                                dev_status, s);
  }
}

}  // namespace greedy
}  // namespace hs
