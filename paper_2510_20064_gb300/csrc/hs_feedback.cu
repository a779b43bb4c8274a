// hs_feedback.cu -- hs_feedback / hs_feedback_path: argument checks and the
// choice of kernels, plus the two-pass stochastic kernels.
//
// Greedy rows go to the argmax kernels (hs_greedy.cu).  Stochastic bf16/fp16
// rows with V % 8 == 0, 16-byte-aligned logits and N <= 32 go to the
// single-read cluster kernel (hs_fused.cu) when V <= 153600, else to the
// persistent streaming kernel (hs_stream.cu).  Everything else takes the
// two-pass path below, which reads each logit twice:
//   row_stats_kernel  one CTA per logit row: max and
//                     S = sum_v 2^{(z_v - m) log2e / T}   (Thm 1's softmax)
//   overlap_kernel    one CTA per ((b,k) tile, vocab chunk): p_v built once
//                     and reused for all N drafters, sum_v min(p_v, q_{i,v})
//                     (Thm 1), one partial sum per chunk
//   finalize_kernel   one warp per (i,b): alpha over the P positions from
//                     the partials in a fixed order, then e_len (Thm 3).
#include <math.h>
#include <stdint.h>

#include <climits>

#include "hs_common.cuh"
#include "hs_fused.h"
#include "hs_greedy.h"
#include "hs_stream.h"
#include "hs_topl.h"

namespace hs {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;  // 16-byte vectors per thread per chunk

// argmax < 0 marks a row that cannot be used: -1 non-finite, -2 bad path.
struct RowStat {
  float m;      // max of the stored logits
  float mc;     // m * log2e / T, the exponent offset used for the row
  float inv_s;  // 1 / sum_v 2^{z_v c - mc}
  int argmax;   // first index of m
};

template <int DT, bool VEC>
__device__ __forceinline__ void load_slots(const void* row, int64_t v0, int V,
                                           float (&x)[kUnroll * Elem<DT>::kVec]) {
  load_chunk<DT, VEC, kThreads, kUnroll>(row, v0, V, x);
}

__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < kWarps; ++j) s += red[j];
  return s;
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) row_stats_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M,
    const void* __restrict__ drafter, int B, int P, int V, float c,
    RowStat* __restrict__ stats) {
  pdl_wait();
  constexpr int kV = Elem<DT>::kVec;
  constexpr int kChunk = kThreads * kUnroll * kV;
  __shared__ float red_m[kWarps];
  __shared__ int red_a[kWarps];
  __shared__ float red_s[kWarps];

  const int64_t r = blockIdx.x;
  const int64_t BP = int64_t(B) * P;
  bool bad_path = false;
  const void* row = r < BP ? target_row<DT>(target, path, M, P, r, V, &bad_path)
                           : row_ptr<DT>(drafter, r - BP, V);

  // pass 1: NaN-propagating max and the first index holding it
  float m = -INFINITY;
  int arg = INT_MAX;
  for (int64_t v0 = 0; v0 < V; v0 += kChunk) {
    float x[kUnroll * kV];
    load_slots<DT, VEC>(row, v0, V, x);
    // a thread visits its slots in increasing v, so a strict '>' keeps the
    // first index of the maximum; a NaN replaces m and then stays
#pragma unroll
    for (int s = 0; s < kUnroll * kV; ++s) {
      int64_t v = slot_pos<DT, VEC, kThreads>(v0, s, threadIdx.x);
      if (v < V && (x[s] > m || x[s] != x[s])) {
        m = x[s];
        arg = int(v);
      }
    }
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  float wm = warp_max_nan(m);
  int wa = warp_min_int((m == wm) ? arg : INT_MAX);
  if (l == 0) { red_m[w] = wm; red_a[w] = wa; }
  __syncthreads();
  float rm = red_m[0];
  for (int j = 1; j < kWarps; ++j) rm = max_nan(rm, red_m[j]);
  int ra = INT_MAX;
  for (int j = 0; j < kWarps; ++j)
    if (red_m[j] == rm && red_a[j] < ra) ra = red_a[j];
  const bool valid = isfinite(rm) && !bad_path;

  float inv_s = 0.f, mc = rm * c;
  if (valid) {
    // pass 2: S = sum_v 2^{z_v c - m c}
    float acc = 0.f;
    for (int64_t v0 = 0; v0 < V; v0 += kChunk) {
      float x[kUnroll * kV];
      load_slots<DT, VEC>(row, v0, V, x);
#pragma unroll
      for (int s = 0; s < kUnroll * kV; ++s) acc += ex2(fmaf(x[s], c, -mc));
    }
    inv_s = 1.f / block_sum(acc, red_s);
  }
  if (threadIdx.x == 0) {
    RowStat st;
    st.m = rm;
    st.mc = mc;
    st.inv_s = inv_s;
    st.argmax = valid ? ra : (bad_path ? -2 : -1);
    stats[r] = st;
  }
  pdl_trigger();
}

template <int DT, bool VEC>
__global__ void __launch_bounds__(kThreads) overlap_kernel(
    const void* __restrict__ target, const int32_t* __restrict__ path, int M,
    const void* __restrict__ drafter, int N, int B, int P, int V, float c,
    const RowStat* __restrict__ stats, float* __restrict__ partial, int nchunk) {
  pdl_wait();
  constexpr int kV = Elem<DT>::kVec;
  constexpr int kS = kUnroll * kV;
  constexpr int kChunk = kThreads * kS;
  extern __shared__ float red[];  // [kWarps][N]

  const int64_t tile = blockIdx.x;
  const int j = blockIdx.y;
  const int64_t b = tile / P, k = tile % P;
  const int64_t BP = int64_t(B) * P;
  const int64_t v0 = int64_t(j) * kChunk;
  bool bad_path = false;
  const void* trow = target_row<DT>(target, path, M, P, tile, V, &bad_path);
  const RowStat st = stats[tile];

  float p[kS];
  load_slots<DT, VEC>(trow, v0, V, p);
#pragma unroll
  for (int s = 0; s < kS; ++s) p[s] = ex2(fmaf(p[s], c, -st.mc)) * st.inv_s;

  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  for (int i = 0; i < N; ++i) {
    const int64_t drow = (int64_t(i) * B + b) * P + k;
    const RowStat sd = stats[BP + drow];
    float q[kS];
    load_slots<DT, VEC>(row_ptr<DT>(drafter, drow, V), v0, V, q);
    float acc = 0.f;
#pragma unroll
    for (int s = 0; s < kS; ++s) acc += fminf(p[s], ex2(fmaf(q[s], c, -sd.mc)) * sd.inv_s);
    acc = warp_sum(acc);
    if (l == 0) red[w * N + i] = acc;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < N; i += kThreads) {
    float s = 0.f;
    for (int ww = 0; ww < kWarps; ++ww) s += red[ww * N + i];
    partial[(tile * nchunk + j) * N + i] = s;
  }
  pdl_trigger();
}

// One warp per (i, b): lanes sum the chunk partials of a position in a fixed
// order (lane-strided, then a shuffle tree), so results repeat bit for bit.
__global__ void finalize_kernel(const RowStat* __restrict__ stats,
                                const float* __restrict__ partial, int nchunk, int N,
                                int B, int P, float* __restrict__ alpha,
                                float* __restrict__ e_len, int* dev_status) {
  pdl_wait();
  const int64_t gw = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  if (gw >= int64_t(N) * B) return;  // whole warp
  const int l = threadIdx.x & 31;
  const int64_t i = gw / B, b = gw % B;
  const int64_t BP = int64_t(B) * P;
  float e = 1.f, prod = 1.f;
  int err = HS_OK;
  for (int k = 0; k < P; ++k) {
    const int64_t tile = b * P + k;
    const int64_t drow = (i * B + b) * P + k;
    const RowStat st = stats[tile], sd = stats[BP + drow];
    const float* pp = partial + tile * int64_t(nchunk) * N + i;
    float a = 0.f;
    for (int j = l; j < nchunk; j += 32) a += pp[int64_t(j) * N];
    a = warp_sum(a);
    if (st.argmax < 0 || sd.argmax < 0) {
      a = __int_as_float(0x7fc00000);  // NaN
      if (err == HS_OK) err = (st.argmax == -2) ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE;
    }
    if (l == 0) alpha[drow] = a;
    if (k < P - 1) {
      prod *= a;
      e += prod;
    }
  }
  if (l == 0) {
    if (e_len) e_len[gw] = e;
    if (err != HS_OK) report(dev_status, err);
  }
}

int elem_bytes(int dtype) { return dtype == HS_FP32 ? 4 : 2; }
int vec_elems(int dtype) { return dtype == HS_FP32 ? 4 : 8; }
int64_t chunk_elems(int dtype) { return int64_t(kThreads) * kUnroll * vec_elems(dtype); }

struct Layout {
  int nchunk;
  size_t stats_off, partial_off, total;
};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool sizes_ok(int N, int B, int P, int V) {
  if (N < 1 || B < 1 || P < 1 || V < 1) return false;
  if (V > (1 << 28)) return false;  // vocab chunks index gridDim.y (<= 65535)
  const int64_t rows = int64_t(B) * P * (int64_t(N) + 1);
  if (rows >= (int64_t(1) << 31)) return false;  // one CTA per row
  if (int64_t(N) * B >= (int64_t(1) << 31)) return false;
  return double(rows) * double(V) < 4.6e18;
}

Layout layout(int N, int B, int P, int V, int dtype, int greedy) {
  Layout L;
  if (greedy) {
    L.nchunk = 0;
    L.stats_off = L.partial_off = 0;
    L.total = align256(greedy::workspace_bytes(N, B, P, V, dtype));
    return L;
  }
  const int64_t rows = int64_t(B) * P * (int64_t(N) + 1);
  L.nchunk = int((V + chunk_elems(dtype) - 1) / chunk_elems(dtype));
  L.stats_off = 0;
  L.partial_off = align256(size_t(rows) * sizeof(RowStat));
  const size_t partial = size_t(B) * P * L.nchunk * size_t(N) * sizeof(float);
  L.total = L.partial_off + align256(partial);
  // the streaming kernel's workspace, when it may take the call
  if (stream::eligible_sizes(dtype, N, V, greedy)) {
    const size_t ss = align256(stream::workspace_bytes(N, B, P, V));
    if (ss > L.total) L.total = ss;
  }
  return L;
}

template <int DT, bool VEC>
hs_status launch_two_pass(const void* target, const int32_t* path, int M, const void* drafter,
                          int N, int B, int P, int V, float c, float* alpha, float* e_len,
                          void* ws, const Layout& L, int* dev_status, cudaStream_t stream) {
  RowStat* stats = reinterpret_cast<RowStat*>(static_cast<char*>(ws) + L.stats_off);
  float* partial = reinterpret_cast<float*>(static_cast<char*>(ws) + L.partial_off);
  const unsigned rows = unsigned(int64_t(B) * P * (int64_t(N) + 1));
  if (launch_pdl(row_stats_kernel<DT, VEC>, dim3(rows), dim3(kThreads), 0, stream, target, path,
                 M, drafter, B, P, V, c, stats) != cudaSuccess)
    return HS_ERR_CUDA;
  const size_t smem = size_t(kWarps) * N * sizeof(float);
  dim3 grid(unsigned(int64_t(B) * P), unsigned(L.nchunk));
  if (launch_pdl(overlap_kernel<DT, VEC>, grid, dim3(kThreads), smem, stream, target, path, M,
                 drafter, N, B, P, V, c, stats, partial, L.nchunk) != cudaSuccess)
    return HS_ERR_CUDA;
  const int64_t threads = int64_t(N) * B * 32;
  if (launch_pdl(finalize_kernel, dim3(unsigned((threads + 255) / 256)), dim3(256), 0, stream,
                 stats, partial, L.nchunk, N, B, P, alpha, e_len, dev_status) != cudaSuccess)
    return HS_ERR_CUDA;
  return HS_OK;
}

template <int DT>
hs_status dispatch_vec(bool vec, const void* target, const int32_t* path, int M,
                       const void* drafter, int N, int B, int P, int V, float c, float* alpha,
                       float* e_len, void* ws, const Layout& L, int* dev_status,
                       cudaStream_t stream) {
  if (vec)
    return launch_two_pass<DT, true>(target, path, M, drafter, N, B, P, V, c, alpha, e_len, ws,
                                     L, dev_status, stream);
  return launch_two_pass<DT, false>(target, path, M, drafter, N, B, P, V, c, alpha, e_len, ws, L,
                                    dev_status, stream);
}

constexpr int kMaxFeedbackN = 1024;  // overlap_kernel keeps [8][N] partials in shared memory

hs_status feedback_common(const void* target, const int32_t* path, int M, const void* drafter,
                          int dtype, int N, int B, int P, int V, float temperature, int greedy,
                          float* alpha, float* e_len, void* ws, size_t ws_bytes,
                          int* dev_status, void* stream) {
  if (dtype != HS_BF16 && dtype != HS_FP16 && dtype != HS_FP32) return HS_ERR_INVALID_ARG;
  if (!sizes_ok(N, B, P, V)) return HS_ERR_INVALID_ARG;
  if (N > kMaxFeedbackN) return HS_ERR_UNSUPPORTED;
  if (!target || !drafter || !alpha) return HS_ERR_INVALID_ARG;
  if (!greedy && !(isfinite(temperature) && temperature > 0.f)) return HS_ERR_INVALID_ARG;
  const int esz = elem_bytes(dtype);
  if (reinterpret_cast<uintptr_t>(target) % esz || reinterpret_cast<uintptr_t>(drafter) % esz ||
      reinterpret_cast<uintptr_t>(alpha) % 4 || reinterpret_cast<uintptr_t>(e_len) % 4 ||
      reinterpret_cast<uintptr_t>(dev_status) % 4)
    return HS_ERR_MISALIGNED;
  const Layout L = layout(N, B, P, V, dtype, greedy);
  if (L.total > 0) {
    if (!ws || ws_bytes < L.total) return HS_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return HS_ERR_MISALIGNED;
  }
  const bool vec = (int64_t(V) * esz) % 16 == 0 && reinterpret_cast<uintptr_t>(target) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(drafter) % 16 == 0;
  const float c = greedy ? 0.f : kLog2e / temperature;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (greedy)
    return greedy::launch(vec, target, path, M, drafter, dtype, N, B, P, V, alpha, e_len, ws,
                          dev_status, s);
  if (fused::eligible(target, drafter, dtype, N, V, greedy))
    return fused::launch(target, path, M, drafter, dtype, N, B, P, V, c, alpha, e_len, dev_status,
                         s);
  if (stream::eligible(target, drafter, dtype, N, V, greedy)) {
    // longer rows: the two-pass kernel while the rows are many enough and
    // L2 still holds a good part of their second passes, else streaming
    const int grid = fused::long_row_grid(N, B, P, V);
    if (grid > 0)
      return fused::launch_two_pass(target, path, M, drafter, dtype, N, B, P, V, c, grid, alpha,
                                    e_len, dev_status, s);
    return stream::launch(target, path, M, drafter, dtype, N, B, P, V, c, alpha, e_len, ws,
                          dev_status, s);
  }
  switch (dtype) {
    case HS_BF16:
      return dispatch_vec<HS_BF16>(vec, target, path, M, drafter, N, B, P, V, c, alpha, e_len,
                                   ws, L, dev_status, s);
    case HS_FP16:
      return dispatch_vec<HS_FP16>(vec, target, path, M, drafter, N, B, P, V, c, alpha, e_len,
                                   ws, L, dev_status, s);
    default:
      return dispatch_vec<HS_FP32>(vec, target, path, M, drafter, N, B, P, V, c, alpha, e_len,
                                   ws, L, dev_status, s);
  }
}

// Draft-tree feedback (Thm 2): validation shared by the chain and path entries.
hs_status topl_common(const void* target, const int32_t* path, int M, const void* drafter,
                      int dtype, int N, int B, int P, int V, float temperature, int greedy, int L,
                      const int32_t* keep, float* alpha, float* e_len, void* ws, size_t ws_bytes,
                      int* dev_status, void* stream) {
  if (dtype != HS_BF16 && dtype != HS_FP16 && dtype != HS_FP32) return HS_ERR_INVALID_ARG;
  if (!sizes_ok(N, B, P, V)) return HS_ERR_INVALID_ARG;
  if (L < 1) return HS_ERR_INVALID_ARG;
  if (L > topl::kMaxL) return HS_ERR_UNSUPPORTED;
  if (V >= (1 << 30)) return HS_ERR_UNSUPPORTED;  // token indices live in 32-bit keys
  if (!target || !drafter || !alpha) return HS_ERR_INVALID_ARG;
  if (!greedy && !(isfinite(temperature) && temperature > 0.f)) return HS_ERR_INVALID_ARG;
  const int esz = elem_bytes(dtype);
  if (reinterpret_cast<uintptr_t>(target) % esz || reinterpret_cast<uintptr_t>(drafter) % esz ||
      reinterpret_cast<uintptr_t>(alpha) % 4 || reinterpret_cast<uintptr_t>(e_len) % 4 ||
      reinterpret_cast<uintptr_t>(dev_status) % 4 || reinterpret_cast<uintptr_t>(keep) % 4)
    return HS_ERR_MISALIGNED;
  if (!ws || ws_bytes < topl::workspace_bytes(N, B, P, V)) return HS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(ws) % 256) return HS_ERR_MISALIGNED;
  const float c = kLog2e / (greedy ? 1.f : temperature);
  return topl::launch(target, path, M, drafter, dtype, N, B, P, V, L, keep, greedy, c, alpha,
                      e_len, ws, dev_status, static_cast<cudaStream_t>(stream));
}

}  // namespace
}  // namespace hs

extern "C" size_t hs_feedback_topl_workspace_size(int N, int B, int P, int V) {
  if (!hs::sizes_ok(N, B, P, V)) return 0;
  return hs::align256(hs::topl::workspace_bytes(N, B, P, V));
}

extern "C" int hs_feedback_topl_kernel_count(int N, int B, int P, int V) {
  if (!hs::sizes_ok(N, B, P, V)) return 0;
  return hs::topl::kernel_count(N, B, P, V);
}

extern "C" hs_status hs_feedback_topl(const void* target, const void* drafter, int dtype, int N,
                                      int B, int P, int V, float temperature, int greedy, int L,
                                      float* alpha, float* e_len, void* workspace,
                                      size_t workspace_bytes, int* dev_status, void* stream) {
  return hs::topl_common(target, nullptr, 0, drafter, dtype, N, B, P, V, temperature, greedy, L,
                         nullptr, alpha, e_len, workspace, workspace_bytes, dev_status, stream);
}

extern "C" hs_status hs_feedback_topl_pruned(const void* target, const void* drafter, int dtype,
                                             int N, int B, int P, int V, float temperature,
                                             int greedy, int L, const int32_t* keep, float* alpha,
                                             float* e_len, void* workspace,
                                             size_t workspace_bytes, int* dev_status,
                                             void* stream) {
  if (!keep) return HS_ERR_INVALID_ARG;
  return hs::topl_common(target, nullptr, 0, drafter, dtype, N, B, P, V, temperature, greedy, L,
                         keep, alpha, e_len, workspace, workspace_bytes, dev_status, stream);
}

extern "C" hs_status hs_feedback_topl_path(const void* tree_target, const int32_t* path_idx,
                                           int M, const void* drafter, int dtype, int N, int B,
                                           int P, int V, float temperature, int greedy, int L,
                                           float* alpha, float* e_len, void* workspace,
                                           size_t workspace_bytes, int* dev_status,
                                           void* stream) {
  if (!path_idx || M < 1) return HS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(path_idx) % 4) return HS_ERR_MISALIGNED;
  if (double(B) * double(M) * double(V) >= 4.6e18) return HS_ERR_INVALID_ARG;
  return hs::topl_common(tree_target, path_idx, M, drafter, dtype, N, B, P, V, temperature,
                         greedy, L, nullptr, alpha, e_len, workspace, workspace_bytes, dev_status,
                         stream);
}

extern "C" hs_status hs_feedback_topl_pruned_path(const void* tree_target,
                                                  const int32_t* path_idx, int M,
                                                  const void* drafter, int dtype, int N, int B,
                                                  int P, int V, float temperature, int greedy,
                                                  int L, const int32_t* keep, float* alpha,
                                                  float* e_len, void* workspace,
                                                  size_t workspace_bytes, int* dev_status,
                                                  void* stream) {
  if (!path_idx || M < 1 || !keep) return HS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(path_idx) % 4) return HS_ERR_MISALIGNED;
  if (double(B) * double(M) * double(V) >= 4.6e18) return HS_ERR_INVALID_ARG;
  return hs::topl_common(tree_target, path_idx, M, drafter, dtype, N, B, P, V, temperature,
                         greedy, L, keep, alpha, e_len, workspace, workspace_bytes, dev_status,
                         stream);
}

extern "C" size_t hs_feedback_workspace_size(int N, int B, int P, int V, int dtype, int greedy) {
  if (dtype != HS_BF16 && dtype != HS_FP16 && dtype != HS_FP32) return 0;
  if (!hs::sizes_ok(N, B, P, V)) return 0;
  return hs::layout(N, B, P, V, dtype, greedy).total;
}

extern "C" int hs_feedback_kernel_count(int N, int B, int P, int V, int dtype, int greedy) {
  if (dtype != HS_BF16 && dtype != HS_FP16 && dtype != HS_FP32) return 0;
  if (!hs::sizes_ok(N, B, P, V)) return 0;
  if (hs::fused::eligible_sizes(dtype, N, V, greedy)) return 2;  // 16-byte-aligned logits
  if (hs::stream::eligible_sizes(dtype, N, V, greedy)) return 2;
  return greedy ? 2 : 3;
}

extern "C" hs_status hs_feedback(const void* target, const void* drafter, int dtype, int N, int B,
                                 int P, int V, float temperature, int greedy, float* alpha,
                                 float* e_len, void* workspace, size_t workspace_bytes,
                                 int* dev_status, void* stream) {
  return hs::feedback_common(target, nullptr, 0, drafter, dtype, N, B, P, V, temperature, greedy,
                             alpha, e_len, workspace, workspace_bytes, dev_status, stream);
}

extern "C" hs_status hs_feedback_path(const void* tree_target, const int32_t* path_idx, int M,
                                      const void* drafter, int dtype, int N, int B, int P, int V,
                                      float temperature, int greedy, float* alpha, float* e_len,
                                      void* workspace, size_t workspace_bytes, int* dev_status,
                                      void* stream) {
  if (!path_idx || M < 1) return HS_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(path_idx) % 4) return HS_ERR_MISALIGNED;
  if (double(B) * double(M) * double(V) >= 4.6e18) return HS_ERR_INVALID_ARG;
  return hs::feedback_common(tree_target, path_idx, M, drafter, dtype, N, B, P, V, temperature,
                             greedy, alpha, e_len, workspace, workspace_bytes, dev_status, stream);
}

extern "C" hs_status hs_test_stream_wait_timeout(const void* target, const void* drafter,
                                                 int dtype, int N, int B, int P, int V,
                                                 float temperature, long long wait_cycles,
                                                 float* alpha, float* e_len, void* workspace,
                                                 size_t workspace_bytes, int* dev_status,
                                                 void* stream) {
  if (!hs::sizes_ok(N, B, P, V) || !target || !drafter || !alpha || !dev_status)
    return HS_ERR_INVALID_ARG;
  if (!(isfinite(temperature) && temperature > 0.f) || wait_cycles < 1) return HS_ERR_INVALID_ARG;
  if (!hs::stream::eligible(target, drafter, dtype, N, V, 0)) return HS_ERR_UNSUPPORTED;
  if (reinterpret_cast<uintptr_t>(alpha) % 4 || reinterpret_cast<uintptr_t>(e_len) % 4 ||
      reinterpret_cast<uintptr_t>(dev_status) % 4 || reinterpret_cast<uintptr_t>(workspace) % 256)
    return HS_ERR_MISALIGNED;
  if (!workspace || workspace_bytes < hs::stream::workspace_bytes(N, B, P, V))
    return HS_ERR_INVALID_ARG;
  return hs::stream::launch_wait_test(target, drafter, dtype, N, B, P, V, hs::kLog2e / temperature,
                                      wait_cycles, alpha, e_len, workspace, dev_status,
                                      static_cast<cudaStream_t>(stream));
}
