// hs_greedy.cu -- greedy feedback: alpha = [argmax q_i == argmax p]
// (Thm 2 with branching L = 1 under a greedy target), e_len by Thm 3.
//
//   argmax_chunk_kernel     one CTA per (row, 32K-logit chunk): NaN-propagating
//                           max of the stored logits and the first index
//                           holding it; every logit is read once, each thread
//                           issuing its 16 16-byte loads before using any;
//                           slots past the row's end hold -inf, which never
//                           wins, so no slot is checked against V
//   greedy_finalize_kernel  one warp per (drafter i, query b), lane k for
//                           position k: combines the chunk partials of its
//                           target and drafter rows in chunk order (first
//                           index wins ties) and compares; the warp's prefix
//                           products of alpha then give e_len (no atomics)
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
constexpr int kUnroll = 16;

template <int DT>
__host__ __device__ constexpr int64_t chunk_of() {
  return int64_t(kThreads) * kUnroll * Elem<DT>::kVec;
}

// This thread's max of one chunk of a row and the first index holding it
// (INT_MAX when the chunk has no logit above -inf).  FULL: the chunk lies
// inside the row, so no load needs a bounds check.
template <int DT, bool VEC, bool FULL>
__device__ __forceinline__ void chunk_argmax(const void* row, int64_t v0, int V, float& m,
                                             int& arg) {
  constexpr int kV = Elem<DT>::kVec;
  constexpr int kS = kUnroll * kV;
  float x[kS];
  if (VEC && DT != HS_FP32) {  // all 16 loads in flight first, then the widening
    uint4 raw[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t v = v0 + int64_t(u * kThreads + threadIdx.x) * kV;
      raw[u] = FULL || v < V
                   ? __ldg(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(row) + v))
                   : make_uint4(DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u,
                                DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u,
                                DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u,
                                DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint32_t wd[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (DT == HS_BF16) {
          x[u * kV + 2 * q] = __uint_as_float(wd[q] << 16);
          x[u * kV + 2 * q + 1] = __uint_as_float(wd[q] & 0xffff0000u);
        } else {
          x[u * kV + 2 * q] = __half2float(__ushort_as_half(static_cast<unsigned short>(wd[q] & 0xffffu)));
          x[u * kV + 2 * q + 1] = __half2float(__ushort_as_half(static_cast<unsigned short>(wd[q] >> 16)));
        }
      }
    }
  } else {
    load_chunk<DT, VEC, kThreads, kUnroll>(row, v0, V, x);
  }
  // slots visit increasing v, so a strict '>' keeps the first index; a NaN
  // replaces m and then stays; the -inf past the row's end never replaces
  // it.  The winning slot is kept as its (constant) number and turned into
  // an index once.
  m = -INFINITY;
  int best = -1;
#pragma unroll
  for (int s = 0; s < kS; ++s) {
    if (x[s] > m || x[s] != x[s]) {
      m = x[s];
      best = s;
    }
  }
  arg = best < 0 ? INT_MAX : int(slot_pos<DT, VEC, kThreads>(v0, best, threadIdx.x));
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) argmax_chunk_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M,
    const void* __restrict__ drafter, int B, int P, int V, Part* __restrict__ parts,
    int nchunk) {
  pdl_wait();
  __shared__ float red_m[kWarps];
  __shared__ int red_a[kWarps];
  const int64_t r = blockIdx.x;
  const int j = blockIdx.y;
  const int64_t BP = int64_t(B) * P;
  bool bad_path = false;
  const void* row = r < BP ? target_row<DT>(target, path, M, P, r, V, &bad_path)
                           : row_ptr<DT>(drafter, r - BP, V);
  const int64_t v0 = int64_t(j) * chunk_of<DT>();
  float m;
  int arg;
  if (v0 + chunk_of<DT>() <= V)  // every chunk but a ragged last one: no load predicates
    chunk_argmax<DT, VEC, true>(row, v0, V, m, arg);
  else
    chunk_argmax<DT, VEC, false>(row, v0, V, m, arg);
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

// Row argmax from its chunk partials, by one thread, chunks in order: the
// strict '>' keeps the first chunk holding the max (each chunk's index is its
// first); a NaN or +inf max makes the row unusable (checked by the caller).
__device__ __forceinline__ void combine(const Part* __restrict__ pr, int nchunk, float& m,
                                        int& arg) {
  m = -INFINITY;
  arg = INT_MAX;
  for (int j = 0; j < nchunk; ++j) {
    const Part q = pr[j];
    if (q.m > m || q.m != q.m) {
      m = q.m;
      arg = q.idx;
      if (q.m != q.m) break;  // NaN: the row is unusable whatever follows
    }
  }
}

__global__ void greedy_finalize_kernel(const Part* __restrict__ parts, int nchunk,
                                       const int32_t* __restrict__ path, int M, int N, int B,
                                       int P, float* __restrict__ alpha,
                                       float* __restrict__ e_len, int* dev_status) {
  pdl_wait();
  const int64_t ib = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;  // (i, b)
  if (ib >= int64_t(N) * B) return;  // whole warp
  const int l = threadIdx.x & 31;
  const int64_t BP = int64_t(B) * P, i = ib / B, b = ib - i * B;
  // e_len = 1 + sum_{k < P-1} prod_{j <= k} alpha_j, 32 positions at a time:
  // an inclusive prefix product over the lanes, carried between groups
  float e = 1.f, carry = 1.f;
  for (int k0 = 0; k0 < P; k0 += 32) {
    const int k = k0 + l;
    float a = 1.f;
    if (k < P) {
      const int64_t tile = b * P + k;
      float mt, md;
      int at, ad;
      combine(parts + tile * nchunk, nchunk, mt, at);
      combine(parts + (BP + i * BP + tile) * nchunk, nchunk, md, ad);
      const bool bad_path = path && (path[tile] < 0 || path[tile] >= M);
      if (bad_path || !isfinite(mt) || !isfinite(md)) {
        a = __int_as_float(0x7fc00000);
        report(dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
      } else {
        a = (at == ad) ? 1.f : 0.f;
      }
      alpha[ib * P + k] = a;
    }
    float pp = k < P - 1 ? a : 1.f;  // positions from P-1 on enter no product
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float up = __shfl_up_sync(0xffffffffu, pp, o);
      if (l >= o) pp *= up;
    }
    const float term = k < P - 1 ? carry * pp : 0.f;
    e += warp_sum(term);
    carry *= __shfl_sync(0xffffffffu, pp, 31);
  }
  if (e_len && l == 0) e_len[ib] = e;
}

// One partial per (row, chunk).
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
  if (launch_pdl(argmax_chunk_kernel<DT, VEC>, dim3(rows, unsigned(nchunk)), dim3(kThreads), 0,
                 s, target, path, M, drafter, B, P, V, parts, nchunk) != cudaSuccess)
    return HS_ERR_CUDA;
  const int64_t threads = int64_t(N) * B * 32;
  if (launch_pdl(greedy_finalize_kernel, dim3(unsigned((threads + 255) / 256)), dim3(256), 0, s,
                 parts, nchunk, path, M, N, B, P, alpha, e_len, dev_status) != cudaSuccess)
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
  return parts_bytes(N, B, P, V, dtype);
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
