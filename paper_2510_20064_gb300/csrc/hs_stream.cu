// hs_stream.cu -- single-DRAM-read stochastic feedback (Thm 1) by a
// persistent kernel that re-reads each logit from L2.
//
// alpha needs each row's normaliser before the min, so every logit is used
// twice.  Here the second use reads it from L2 instead of HBM:
//   * work items are (tile (b,k), vocab chunk j of kChunk logits); at step s
//     CTA c does the STATS of item s*G + c -- for the target row and the N
//     drafter rows of the tile, the chunk's max-offset and sum of
//     2^{z c - offset} (c = log2e / T), written to global memory; the CTA
//     then bumps the tile's counter;
//   * in the same step the CTA does the OVERLAP of the item it read one step
//     earlier: once every chunk of that tile has its stats (bounded wait on
//     the counter), it merges them into each row's offset O and normaliser
//     Z, re-reads the chunk (an L2 hit: one step of items is a few tens of
//     MB), builds p_v = 2^{z_v c - O_t} / Z_t in registers and adds
//     sum_v min(p_v, q_{i,v}) for every drafter i;
//   * the last CTA to finish a tile sums the chunk partials in chunk order
//     and writes alpha[:, b, k].
// No overlap ever waits on a later item than the ones its own CTA has
// already passed, and the launch is cooperative (all CTAs resident), so the
// waits always end; each is bounded anyway: a wait that gives up reports
// HS_ERR_TIMEOUT and marks its tile, whose alphas are then written as NaN.
// HBM traffic is one read of every logit; L2 traffic two.
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "hs_common.cuh"
#include "hs_stream.h"

namespace hs {
namespace stream {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kVecs = 4;                         // 16-byte vectors per thread and row
constexpr int kChunk = kThreads * kVecs * 8;     // logits per row chunk (bf16 / fp16)
constexpr int kMaxN = 32;
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second
// A tile's overlap count carries this mark once an overlap of the tile gave
// up waiting for the tile's statistics (chunks per row stay below it).
constexpr int kTimedOut = 1 << 24;

struct Params {
  const void* target;
  const int32_t* path;
  int M;
  const void* drafter;
  int N, B, P, V;
  float c;      // log2(e) / T
  int nchunk;   // chunks per row
  int ntiles;   // B * P
  int nitems;   // ntiles * nchunk
  int lag;      // steps between an item's stats and its overlap
  float2* stats;  // [ntiles][N+1][nchunk] (offset, sum)
  float* apart;   // [ntiles][N][nchunk] alpha partials
  int* cnt;       // [ntiles] chunks with stats
  int* cnt2;      // [ntiles] chunks with overlap
  float* alpha;
  int* dev_status;
  long long wait_limit;  // clock cycles a wait may take (kTimeoutCycles)
  int stall_tile;        // test hook: this tile's statistics count never completes (-1: none)
};

// Order-preserving int key of a float (NaN above +inf): warp max in one redux.
__device__ __forceinline__ int fkey(float f) {
  const int b = __float_as_int(f);
  return (f != f) ? 0x7fffffff : (b >= 0 ? b : b ^ 0x7fffffff);
}
__device__ __forceinline__ float kfloat(int k) {
  return __int_as_float(k >= 0 ? k : k ^ 0x7fffffff);
}
__device__ __forceinline__ float warp_max_key(float f) {
  return kfloat(__reduce_max_sync(0xffffffffu, fkey(f)));
}

template <int DT>
__device__ __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
  uint32_t r;
  if (DT == HS_BF16)
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  else
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
template <int DT>
__device__ __forceinline__ float lo(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w << 16);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xffffu)));
}
template <int DT>
__device__ __forceinline__ float hi(uint32_t w) {
  if (DT == HS_BF16) return __uint_as_float(w & 0xffff0000u);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
}

// (offset, sum) merge: sums rescaled to the larger offset; -inf offset means
// "no finite logit"; NaN propagates.
__device__ __forceinline__ void merge(float& o, float& s, float o2, float s2) {
  const float O = max_nan(o, o2);
  const float a = (o == -INFINITY || O == -INFINITY) ? 0.f : s * ex2(o - O);
  const float b = (o2 == -INFINITY || O == -INFINITY) ? 0.f : s2 * ex2(o2 - O);
  o = O;
  s = a + b;
}

// Global address of row r (0 = target, 1+i = drafter i) of tile t.
template <int DT>
__device__ __forceinline__ const uint4* row_base(const Params& p, int64_t t, int r) {
  const int64_t b = t / p.P, k = t % p.P;
  int64_t row;
  const void* base;
  if (r == 0) {
    if (p.path) {
      const int nd = p.path[t];
      row = b * p.M + ((nd < 0 || nd >= p.M) ? 0 : nd);
    } else {
      row = t;
    }
    base = p.target;
  } else {
    row = (int64_t(r - 1) * p.B + b) * p.P + k;
    base = p.drafter;
  }
  return reinterpret_cast<const uint4*>(static_cast<const char*>(base) + row * int64_t(p.V) * 2);
}

// The thread's kVecs vectors of one row chunk (-inf past the end of the row).
template <int DT>
__device__ __forceinline__ void load_chunk(const uint4* row, int j, int V, uint4 (&v)[kVecs]) {
  const uint32_t neg = (DT == HS_BF16) ? 0xFF80FF80u : 0xFC00FC00u;
#pragma unroll
  for (int u = 0; u < kVecs; ++u) {
    const int64_t e = int64_t(j) * kChunk + (u * kThreads + threadIdx.x) * 8;
    v[u] = e < V ? __ldcg(row + e / 8) : make_uint4(neg, neg, neg, neg);
  }
}

struct Smem {
  float2 red[kMaxN + 1][kWarps];  // per-warp (offset, sum) of each row of an item
  float2 os[kMaxN + 1];           // row (offset O, 1/Z) of the overlap item
  float ap[kMaxN][kWarps];        // per-warp alpha partials
  int flag;                       // 1: this CTA finishes the tile's alpha
  int wait_mark;                  // kTimedOut when this overlap's wait gave up
};

template <int DT>
__device__ void stats_item(const Params& p, Smem& sm, int x) {
  const int64_t t = x / p.nchunk;
  const int j = x % p.nchunk;
  const int R = p.N + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint4 cur[kVecs], nxt[kVecs];
  load_chunk<DT>(row_base<DT>(p, t, 0), j, p.V, cur);
  for (int r = 0; r < R; ++r) {
    if (r + 1 < R) load_chunk<DT>(row_base<DT>(p, t, r + 1), j, p.V, nxt);
    uint32_t m2 = pmax<DT>(pmax<DT>(cur[0].x, cur[0].y), pmax<DT>(cur[0].z, cur[0].w));
#pragma unroll
    for (int u = 1; u < kVecs; ++u)
      m2 = pmax<DT>(m2, pmax<DT>(pmax<DT>(cur[u].x, cur[u].y), pmax<DT>(cur[u].z, cur[u].w)));
    const float m = warp_max_key(max_nan(lo<DT>(m2), hi<DT>(m2)));
    const float o = (m == -INFINITY) ? -INFINITY : m * p.c;
    const float ou = (m == -INFINITY) ? 0.f : o;
    float s0 = 0.f, s1 = 0.f;
#pragma unroll
    for (int u = 0; u < kVecs; ++u) {
      const uint32_t w[4] = {cur[u].x, cur[u].y, cur[u].z, cur[u].w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        s0 += ex2(fmaf(lo<DT>(w[h]), p.c, -ou));
        s1 += ex2(fmaf(hi<DT>(w[h]), p.c, -ou));
      }
    }
    const float s = warp_sum(s0 + s1);
    if (lane == 0) sm.red[r][warp] = make_float2(o, s);
    if (r + 1 < R) {
#pragma unroll
      for (int u = 0; u < kVecs; ++u) cur[u] = nxt[u];
    }
  }
  __syncthreads();
  for (int r = threadIdx.x; r < R; r += kThreads) {
    float o = -INFINITY, s = 0.f;
    for (int w = 0; w < kWarps; ++w) merge(o, s, sm.red[r][w].x, sm.red[r][w].y);
    p.stats[(t * R + r) * p.nchunk + j] = make_float2(o, s);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(p.cnt + t, 1);
  }
}

template <int DT>
__device__ void overlap_item(const Params& p, Smem& sm, int y) {
  const int64_t t = y / p.nchunk;
  const int j = y % p.nchunk;
  const int R = p.N + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // every chunk of tile t has its stats (bounded wait; the test hook asks
  // for one chunk more than exist, so that the wait runs out)
  if (threadIdx.x == 0) {
    const int need = p.nchunk + (t == p.stall_tile ? 1 : 0);
    const long long t0 = clock64();
    int seen;
    sm.wait_mark = 0;
    while (true) {
      asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(seen) : "l"(p.cnt + t) : "memory");
      if (seen >= need) break;
      if (clock64() - t0 > p.wait_limit) {
        report(p.dev_status, HS_ERR_TIMEOUT);
        sm.wait_mark = kTimedOut;
        break;
      }
      __nanosleep(64);
    }
  }
  __syncthreads();
  const int mark = sm.wait_mark;  // rewritten only after this call's later barriers
  // row offsets and normalisers: warp w merges rows w, w + kWarps, ...
  for (int r = warp; r < R; r += kWarps) {
    float o = -INFINITY, s = 0.f;
    for (int q = lane; q < p.nchunk; q += 32) {
      const float2 v = __ldcg(p.stats + (t * R + r) * p.nchunk + q);
      merge(o, s, v.x, v.y);
    }
    const float O = warp_max_key(o);
    float sc = (o == -INFINITY || O == -INFINITY) ? 0.f : s * ex2(o - O);
    sc = warp_sum(sc);
    if (lane == 0) {
      const bool ok = isfinite(O) && sc > 0.f;
      sm.os[r] = make_float2(ok ? O : __int_as_float(0x7fc00000), ok ? 1.f / sc : 0.f);
    }
  }
  __syncthreads();
  // p of the target chunk, in registers
  float pv[kVecs * 8];
  uint4 cur[kVecs], nxt[kVecs];
  load_chunk<DT>(row_base<DT>(p, t, 0), j, p.V, cur);
  load_chunk<DT>(row_base<DT>(p, t, 1), j, p.V, nxt);
  {
    const float2 ot = sm.os[0];
    const float oc = isnan(ot.x) ? 0.f : ot.x;
#pragma unroll
    for (int u = 0; u < kVecs; ++u) {
      const uint32_t w[4] = {cur[u].x, cur[u].y, cur[u].z, cur[u].w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        pv[u * 8 + 2 * h] = ex2(fmaf(lo<DT>(w[h]), p.c, -oc)) * ot.y;
        pv[u * 8 + 2 * h + 1] = ex2(fmaf(hi<DT>(w[h]), p.c, -oc)) * ot.y;
      }
    }
  }
  for (int i = 0; i < p.N; ++i) {
#pragma unroll
    for (int u = 0; u < kVecs; ++u) cur[u] = nxt[u];
    if (i + 1 < p.N) load_chunk<DT>(row_base<DT>(p, t, i + 2), j, p.V, nxt);
    const float2 od = sm.os[i + 1];
    const float oc = isnan(od.x) ? 0.f : od.x;
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int u = 0; u < kVecs; ++u) {
      const uint32_t w[4] = {cur[u].x, cur[u].y, cur[u].z, cur[u].w};
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        a0 += fminf(pv[u * 8 + 2 * h], ex2(fmaf(lo<DT>(w[h]), p.c, -oc)) * od.y);
        a1 += fminf(pv[u * 8 + 2 * h + 1], ex2(fmaf(hi<DT>(w[h]), p.c, -oc)) * od.y);
      }
    }
    const float a = warp_sum(a0 + a1);
    if (lane == 0) sm.ap[i][warp] = a;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < p.N; i += kThreads) {
    float a = 0.f;
    for (int w = 0; w < kWarps; ++w) a += sm.ap[i][w];
    p.apart[(t * p.N + i) * p.nchunk + j] = a;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    // the count of finished overlaps (low bits) and the mark of a wait that
    // gave up (one bit, set before this CTA's count: the tile's last count
    // sees every mark)
    if (mark) atomicOr(p.cnt2 + t, kTimedOut);
    const int before = atomicAdd(p.cnt2 + t, 1);
    sm.flag = ((before & (kTimedOut - 1)) == p.nchunk - 1) ? 1 + ((before | mark) & kTimedOut)
                                                           : 0;
    __threadfence();
  }
  __syncthreads();
  if (!sm.flag) return;
  // this CTA completed tile t: alpha[:, b, k] from the chunk partials (NaN
  // when one of the tile's waits gave up)
  const bool timed_out = (sm.flag & kTimedOut) != 0;
  const int64_t b = t / p.P, k = t % p.P;
  const bool bad_path = p.path && (p.path[t] < 0 || p.path[t] >= p.M);
  const bool t_ok = !isnan(sm.os[0].x);
  for (int i = threadIdx.x; i < p.N; i += kThreads) {
    float a = 0.f;
    for (int q = 0; q < p.nchunk; ++q) a += __ldcg(p.apart + (t * p.N + i) * p.nchunk + q);
    if (timed_out) {
      a = __int_as_float(0x7fc00000);
    } else if (bad_path || !t_ok || isnan(sm.os[i + 1].x)) {
      a = __int_as_float(0x7fc00000);
      report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
    }
    p.alpha[(int64_t(i) * p.B + b) * p.P + k] = a;
  }
}

template <int DT>
__global__ void __launch_bounds__(kThreads) stream_kernel(const Params p) {
  pdl_wait();
  __shared__ Smem sm;
  const int G = gridDim.x;
  const int steps = (p.nitems + G - 1) / G + p.lag;
  for (int s = 0; s < steps; ++s) {
    const int x = s * G + blockIdx.x;
    if (x < p.nitems) stats_item<DT>(p, sm, x);
    const int y = (s - p.lag) * G + blockIdx.x;
    if (s >= p.lag && y < p.nitems) overlap_item<DT>(p, sm, y);
  }
}

__global__ void elen_kernel(const float* __restrict__ alpha, int64_t NB, int P,
                            float* __restrict__ e_len) {
  pdl_wait();
  const int64_t idx = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= NB) return;
  const float* a = alpha + idx * P;
  float e = 1.f, prod = 1.f;
  for (int k = 0; k < P - 1; ++k) {
    prod *= a[k];
    e += prod;
  }
  e_len[idx] = e;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct Layout {
  size_t stats, apart, cnt, total;
};

Layout layout(int N, int B, int P, int V) {
  const int64_t ntiles = int64_t(B) * P;
  const int64_t nchunk = (V + kChunk - 1) / kChunk;
  Layout L;
  L.stats = 0;
  L.apart = L.stats + align256(size_t(ntiles * (N + 1) * nchunk) * sizeof(float2));
  L.cnt = L.apart + align256(size_t(ntiles * N * nchunk) * sizeof(float));
  L.total = L.cnt + align256(size_t(ntiles) * 2 * sizeof(int));
  return L;
}

template <int DT>
hs_status launch_t(const Params& p0, void* ws, cudaStream_t stream) {
  auto kern = stream_kernel<DT>;
  // occupancy and SM count, queried on the first call per device (so that
  // later calls can be captured into CUDA graphs); the mutex lets host
  // threads driving different GPUs call concurrently
  static std::mutex mu;
  static int per_sm_of[kMaxDevices] = {}, nsm_of[kMaxDevices] = {};
  int dev = 0, per_sm = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return HS_ERR_CUDA;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (!per_sm_of[dev]) {
      int ps = 0, n = 0;
      if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
          cudaOccupancyMaxActiveBlocksPerMultiprocessor(&ps, kern, kThreads, 0) != cudaSuccess ||
          ps < 1)
        return HS_ERR_CUDA;
      per_sm_of[dev] = ps;
      nsm_of[dev] = n;
    }
    per_sm = per_sm_of[dev];
    nsm = nsm_of[dev];
  }
  Params p = p0;
  // one step of items must stay in L2 until its overlap: bound the grid so
  // that a step's logits are at most ~40 MB
  const int64_t item_bytes = int64_t(p.N + 1) * kChunk * 2;
  int64_t grid = (40LL << 20) / item_bytes;
  if (grid < nsm) grid = nsm;
  if (grid > int64_t(per_sm) * nsm) grid = int64_t(per_sm) * nsm;
  if (grid > p.nitems) grid = p.nitems;
  if (grid < 1) grid = 1;
  const Layout L = layout(p.N, p.B, p.P, p.V);
  int* cnt = reinterpret_cast<int*>(static_cast<char*>(ws) + L.cnt);
  if (cudaMemsetAsync(cnt, 0, size_t(p.ntiles) * 2 * sizeof(int), stream) != cudaSuccess)
    return HS_ERR_CUDA;
  p.stats = reinterpret_cast<float2*>(static_cast<char*>(ws) + L.stats);
  p.apart = reinterpret_cast<float*>(static_cast<char*>(ws) + L.apart);
  p.cnt = cnt;
  p.cnt2 = cnt + p.ntiles;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.gridDim = dim3(unsigned(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, kern, p) != cudaSuccess) return HS_ERR_CUDA;
  return HS_OK;
}

}  // namespace

bool eligible_sizes(int dtype, int N, int V, int greedy) {
  return !greedy && (dtype == HS_BF16 || dtype == HS_FP16) && N <= kMaxN && V % 8 == 0;
}

bool eligible(const void* target, const void* drafter, int dtype, int N, int V, int greedy) {
  if (reinterpret_cast<uintptr_t>(target) % 16 || reinterpret_cast<uintptr_t>(drafter) % 16)
    return false;
  return eligible_sizes(dtype, N, V, greedy);
}

size_t workspace_bytes(int N, int B, int P, int V) { return layout(N, B, P, V).total; }

hs_status launch_impl(const void* target, const int32_t* path, int M, const void* drafter,
                      int dtype, int N, int B, int P, int V, float c, float* alpha, float* e_len,
                      void* ws, int* dev_status, cudaStream_t stream, int stall_tile,
                      long long wait_limit) {
  Params p = {};
  p.target = target;
  p.path = path;
  p.M = M;
  p.drafter = drafter;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.c = c;
  p.nchunk = (V + kChunk - 1) / kChunk;
  p.ntiles = B * P;
  p.nitems = p.ntiles * p.nchunk;
  p.lag = 1;
  p.alpha = alpha;
  p.dev_status = dev_status;
  p.stall_tile = stall_tile;
  p.wait_limit = wait_limit;
  const hs_status st = dtype == HS_BF16 ? launch_t<HS_BF16>(p, ws, stream)
                                        : launch_t<HS_FP16>(p, ws, stream);
  if (st != HS_OK) return st;
  if (e_len) {
    const int64_t nb = int64_t(N) * B;
    if (launch_pdl(elen_kernel, dim3(unsigned((nb + 255) / 256)), dim3(256), 0, stream, alpha,
                   nb, P, e_len) != cudaSuccess)
      return HS_ERR_CUDA;
  }
  return HS_OK;
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, float* alpha, float* e_len, void* ws,
                 int* dev_status, cudaStream_t stream) {
  return launch_impl(target, path, M, drafter, dtype, N, B, P, V, c, alpha, e_len, ws, dev_status,
                     stream, -1, kTimeoutCycles);
}

hs_status launch_wait_test(const void* target, const void* drafter, int dtype, int N, int B,
                           int P, int V, float c, long long wait_cycles, float* alpha,
                           float* e_len, void* ws, int* dev_status, cudaStream_t stream) {
  return launch_impl(target, nullptr, 0, drafter, dtype, N, B, P, V, c, alpha, e_len, ws,
                     dev_status, stream, 0, wait_cycles);
}

}  // namespace stream
}  // namespace hs
