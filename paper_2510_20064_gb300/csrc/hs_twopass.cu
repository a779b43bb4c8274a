// hs_twopass.cu -- stochastic feedback (Thm 1), two passes per CTA with the
// second served by L2, for shapes where the cluster kernel (hs_fused.cu)
// leaves SMs idle and the working set below fits in L2.
//
// One CTA per SM, one (b,k) tile at a time, no cluster, no tensor memory;
// c = log2(e) / T throughout:
//   A. the target row: offset o_t = c m + log2 sum_v 2^{c z_v - c m}, so that
//      log2 p_v = c z_v - o_t;
//   B. per group of up to kG drafters: pass 1 gives each one's offset o_i
//      the same way; pass 2 walks the rows backwards (the most recently read
//      part first), reading each target chunk once for the whole group, and
//      sums  min(p_v, q_v) = 2^{min(c z_t - o_t, c z_d - o_i)}
//      (2^x is increasing, so the min moves inside: one exp2 per pair).
// One producer warp streams every chunk the consumers need, in their order,
// into a ring of 32 KB shared-memory stages with cp.async.bulk; the target's
// loads ask L2 to keep its lines (the row is read 1 + 2 ceil(N/kG) times per
// tile), pass 2's drafter loads mark theirs as last use.  HBM reads each
// logit once as long as every SM's target row and kG drafter rows, (1 + kG)
// rows per SM, stay in L2; the caller checks that (preferred()).
#include <math.h>
#include <stdint.h>

#include "hs_common.cuh"
#include "hs_twopass.h"

namespace hs {
namespace twopass {
namespace {

constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;       // + the producer warp
constexpr int kStages = 6;                      // ring stages
constexpr int kVecsPerThread = 4;               // 16-byte vectors of a stage per consumer
constexpr int kChunkVecs = kVecsPerThread * kConsumers;
constexpr int kChunkBytes = kChunkVecs * 16;    // 32 KB
constexpr int kG = 2;                           // drafters per pass-2 group
constexpr long long kTimeoutCycles = 1LL << 31;  // about a second

template <int DT>
struct Pair;  // two logits of a 32-bit word as floats

template <>
struct Pair<HS_BF16> {
  __device__ static __forceinline__ float lo(uint32_t w) { return __uint_as_float(w << 16); }
  __device__ static __forceinline__ float hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
};
template <>
struct Pair<HS_FP16> {
  __device__ static __forceinline__ float lo(uint32_t w) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(w & 0xffffu)));
  }
  __device__ static __forceinline__ float hi(uint32_t w) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(w >> 16)));
  }
};

template <int DT>
__device__ __forceinline__ void unpack(uint4 w, float* x) {
  x[0] = Pair<DT>::lo(w.x);
  x[1] = Pair<DT>::hi(w.x);
  x[2] = Pair<DT>::lo(w.y);
  x[3] = Pair<DT>::hi(w.y);
  x[4] = Pair<DT>::lo(w.z);
  x[5] = Pair<DT>::hi(w.z);
  x[6] = Pair<DT>::lo(w.w);
  x[7] = Pair<DT>::hi(w.w);
}

// ---- PTX wrappers ---------------------------------------------------------------

__device__ __forceinline__ uint32_t saddr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(bar), "r"(parity), "r"(1000000u) : "memory");
  return ok != 0;
}
// Bounded wait; false (the CTA's error flag set, a timeout reported) after
// about a second, or at once when another wait of the CTA already gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* error,
                                          int* dev_status) {
  if (mbar_test(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (*error) return false;
    if (mbar_test(bar, parity)) return true;
    if (clock64() - t0 > kTimeoutCycles) {
      *error = 1;
      report(dev_status, HS_ERR_TIMEOUT);
      return false;
    }
  }
}
__device__ __forceinline__ uint64_t make_policy(int kind) {  // 0 normal, 1 keep, 2 last use
  uint64_t p;
  if (kind == 1)
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  else if (kind == 2)
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  else
    asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// One thread: stream `bytes` (a multiple of 16 from a 16-byte-aligned source)
// into a stage, completing its mbarrier's phase, with an L2 policy.
__device__ __forceinline__ void bulk_fill(uint32_t stage, uint32_t bar, const void* src,
                                          uint32_t bytes, uint64_t pol) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               :: "r"(bar), "r"(bytes) : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
               "[%0], [%1], %2, [%3], %4;"
               :: "r"(stage), "l"(src), "r"(bytes), "r"(bar), "l"(pol) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
  return v;
}
// Barrier of the consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" :: "n"(kConsumers) : "memory");
}

// Merge running pairs (m, s): s is relative to m, in 2^{c(.)}.
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2, float c) {
  const float M = max_nan(m, m2);
  const float a = (m == -INFINITY) ? 0.f : s * ex2((m - M) * c);
  const float b = (m2 == -INFINITY) ? 0.f : s2 * ex2((m2 - M) * c);
  m = M;
  s = a + b;
}

struct Shared {
  uint64_t full[kStages], empty[kStages];
  float m[kConsumerWarps], s[kConsumerWarps];
  int bad[kConsumerWarps];
  float acc[kG][kConsumerWarps];
  int error;
};

struct Params {
  const void* target;
  const int32_t* path;
  const void* drafter;
  float* alpha;
  int* dev_status;
  int M, N, B, P, V;
  int t0;  // first tile of this kernel; it takes tiles t0 .. B*P-1 (0: all)
  float c;
};

// ---- consumer warps ---------------------------------------------------------------

// Packed fp32 pairs (two lanes of one 64-bit register pair).
__device__ __forceinline__ uint64_t pack2(float lo, float hi) {
  uint64_t d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
  return d;
}
__device__ __forceinline__ float lo2(uint64_t d) { return __uint_as_float(uint32_t(d)); }
__device__ __forceinline__ float hi2(uint64_t d) { return __uint_as_float(uint32_t(d >> 32)); }
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// The two logits of a stored word as a packed pair.
template <int DT>
__device__ __forceinline__ uint64_t pair_of(uint32_t w) {
  return pack2(Pair<DT>::lo(w), Pair<DT>::hi(w));
}
// NaN-propagating packed max of two stored words, and the max of its pair.
template <int DT>
__device__ __forceinline__ uint32_t pmax(uint32_t a, uint32_t b) {
  uint32_t r;
  if (DT == HS_BF16)
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  else
    asm("max.NaN.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Per tile, in the producer's order: the target row's offset, then per group
// each drafter row's offset, then pass 2.  Every consumer thread runs the
// same control flow (also after a timeout, then on whatever the stages
// hold), so the consumer barriers always meet; a timed-out call reports
// HS_ERR_TIMEOUT and writes NaN.  A thread holds 4 vectors (32 logits) of
// each stage; only a row's last chunk can end early, and only there are the
// vectors past the row's end replaced by -inf.
template <int DT>
__device__ __forceinline__ void consumer(const Params& p, Shared& sh, uint32_t ring0, int nvec,
                                         int nch, int T, float c, volatile int* err) {
  const int t = threadIdx.x, w = t >> 5, l = t & 31;
  uint32_t stage = 0, phase = 0;  // the next stage and its phase parity
  bool ok = true;
  const uint32_t ninf = DT == HS_BF16 ? 0xFF80FF80u : 0xFC00FC00u;
  const uint64_t c2 = pack2(c, c);
  auto take = [&](int ch, uint4 (&v)[kVecsPerThread]) {
    if (!mbar_wait(saddr(&sh.full[stage]), phase, err, p.dev_status)) ok = false;
    const uint32_t base = ring0 + stage * kChunkBytes + uint32_t(t) * 16u;
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) v[u] = lds128(base + uint32_t(u * kConsumers) * 16u);
    if (ch == nch - 1) {
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u)
        if (ch * kChunkVecs + u * kConsumers + t >= nvec) v[u] = make_uint4(ninf, ninf, ninf, ninf);
    }
    __syncwarp();  // the warp's reads of the stage are done: hand it back
    if (l == 0) mbar_arrive(saddr(&sh.empty[stage]));
    if (++stage == kStages) {
      stage = 0;
      phase ^= 1u;
    }
  };
  // a whole row: offset c m + log2 sum 2^{c (z - m)}, NaN for an unusable row
  auto row_offset = [&]() -> float {
    float m = -INFINITY;
    uint64_t s2 = 0ull;  // packed partial sums relative to m
    bool bad = false;
    for (int ch = 0; ch < nch; ++ch) {
      uint4 v[kVecsPerThread];
      take(ch, v);
      uint32_t mw = pmax<DT>(pmax<DT>(v[0].x, v[0].y), pmax<DT>(v[0].z, v[0].w));
#pragma unroll
      for (int u = 1; u < kVecsPerThread; ++u)
        mw = pmax<DT>(mw, pmax<DT>(pmax<DT>(v[u].x, v[u].y), pmax<DT>(v[u].z, v[u].w)));
      const float cm = max_nan(Pair<DT>::lo(mw), Pair<DT>::hi(mw));
      bad |= (cm != cm) || cm == INFINITY;
      if (cm > m) {
        const float r = (m == -INFINITY) ? 0.f : ex2((m - cm) * c);
        s2 = pack2(lo2(s2) * r, hi2(s2) * r);
        m = cm;
      }
      if (m != -INFINITY) {
        const float off = -m * c;
        const uint64_t off2 = pack2(off, off);
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
          const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint64_t e = fma2(pair_of<DT>(wd[q]), c2, off2);
            s2 = add2(s2, pack2(ex2(lo2(e)), ex2(hi2(e))));
          }
        }
      }
    }
    float s = lo2(s2) + hi2(s2);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
      merge_ms(m, s, __shfl_xor_sync(0xffffffffu, m, o), __shfl_xor_sync(0xffffffffu, s, o), c);
    bad = __any_sync(0xffffffffu, bad);
    if (l == 0) {
      sh.m[w] = m;
      sh.s[w] = s;
      sh.bad[w] = bad;
    }
    consumer_sync();
    float M = sh.m[0], S = sh.s[0];
    bool B = sh.bad[0];
    for (int q = 1; q < kConsumerWarps; ++q) {
      merge_ms(M, S, sh.m[q], sh.s[q], c);
      B = B || sh.bad[q];
    }
    consumer_sync();  // the partials are reused by the next reduction
    if (B || M == -INFINITY || !(S > 0.f) || isinf(S)) return __int_as_float(0x7fc00000);
    return fmaf(M, c, __log2f(S));
  };
  for (int tile = p.t0 + blockIdx.x; tile < T; tile += gridDim.x) {
    bool bad_path = false;
    (void)target_row<DT>(p.target, p.path, p.M, p.P, tile, p.V, &bad_path);
    const float ot = row_offset();
    const uint64_t ot2 = pack2(-ot, -ot);
    for (int g0 = 0; g0 < p.N; g0 += kG) {
      const int gn = p.N - g0 < kG ? p.N - g0 : kG;
      float od[kG];
      uint64_t acc[kG];
#pragma unroll
      for (int gi = 0; gi < kG; ++gi) {
        od[gi] = gi < gn ? row_offset() : 0.f;
        acc[gi] = 0ull;
      }
      for (int ch = nch - 1; ch >= 0; --ch) {
        uint4 v[kVecsPerThread];
        take(ch, v);
        float xt[8 * kVecsPerThread];  // log2 p of the thread's 32 logits
#pragma unroll
        for (int u = 0; u < kVecsPerThread; ++u) {
          const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint64_t e = fma2(pair_of<DT>(wd[q]), c2, ot2);
            xt[8 * u + 2 * q] = lo2(e);
            xt[8 * u + 2 * q + 1] = hi2(e);
          }
        }
#pragma unroll
        for (int gi = 0; gi < kG; ++gi) {
          if (gi < gn) {
            take(ch, v);
            const uint64_t od2 = pack2(-od[gi], -od[gi]);
#pragma unroll
            for (int u = 0; u < kVecsPerThread; ++u) {
              const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const uint64_t e = fma2(pair_of<DT>(wd[q]), c2, od2);
                acc[gi] = add2(acc[gi], pack2(ex2(fminf(xt[8 * u + 2 * q], lo2(e))),
                                              ex2(fminf(xt[8 * u + 2 * q + 1], hi2(e)))));
              }
            }
          }
        }
      }
#pragma unroll
      for (int gi = 0; gi < kG; ++gi) {
        const float a = warp_sum(lo2(acc[gi]) + hi2(acc[gi]));
        if (l == 0) sh.acc[gi][w] = a;
      }
      consumer_sync();
      if (t == 0) {
        for (int gi = 0; gi < gn; ++gi) {
          float a = 0.f;
          for (int q = 0; q < kConsumerWarps; ++q) a += sh.acc[gi][q];
          const bool good = ok && !bad_path && !(ot != ot) && !(od[gi] != od[gi]);
          if (!good && ok) report(p.dev_status, bad_path ? HS_ERR_INVALID_ARG : HS_ERR_NONFINITE);
          p.alpha[int64_t(g0 + gi) * T + tile] = good ? a : __int_as_float(0x7fc00000);
        }
      }
      consumer_sync();
    }
  }
}

size_t shared_bytes() {
  return ((sizeof(Shared) + 127) & ~size_t(127)) + size_t(kStages) * kChunkBytes;
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 1) twopass_kernel(const Params p) {
  extern __shared__ __align__(128) unsigned char smem[];
  Shared& sh = *reinterpret_cast<Shared*>(smem);
  const uint32_t ring0 = saddr(smem + ((sizeof(Shared) + 127) & ~size_t(127)));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(saddr(&sh.full[s]), 1);
      mbar_init(saddr(&sh.empty[s]), kConsumerWarps);
    }
    sh.error = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  pdl_wait();  // the set-up above overlaps the previous kernel of the stream
  volatile int* err = &sh.error;
  const int nvec = p.V / 8;
  const int nch = (nvec + kChunkVecs - 1) / kChunkVecs;
  const int T = p.B * p.P;
  const float c = p.c;

  if (warp == kConsumerWarps) {
    // ------------------------------ producer ---------------------------------
    // Streams every chunk in the order the consumers take them: the target
    // row; then per group, each drafter row; then the rows backwards, each
    // target chunk followed by the group's drafter chunks.
    if (lane == 0) {
      const uint64_t normal = make_policy(0), keep = make_policy(1), once = make_policy(2);
      uint32_t k = 0;
      bool ok = true;
      auto put = [&](const char* row, int ch, uint64_t pol) {
        if (!ok) return;
        const uint32_t s = k % kStages;
        if (k >= kStages &&
            !mbar_wait(saddr(&sh.empty[s]), ((k / kStages) - 1) & 1u, err, p.dev_status)) {
          ok = false;
          return;
        }
        const int v0 = ch * kChunkVecs;
        const int nv = nvec - v0 < kChunkVecs ? nvec - v0 : kChunkVecs;
        bulk_fill(ring0 + s * kChunkBytes, saddr(&sh.full[s]), row + int64_t(v0) * 16,
                  uint32_t(nv) * 16u, pol);
        ++k;
      };
      for (int tile = p.t0 + blockIdx.x; tile < T; tile += gridDim.x) {
        bool bad_path = false;
        const char* trow = static_cast<const char*>(
            target_row<DT>(p.target, p.path, p.M, p.P, tile, p.V, &bad_path));
        for (int ch = 0; ch < nch; ++ch) put(trow, ch, keep);
        for (int g0 = 0; g0 < p.N; g0 += kG) {
          const int gn = p.N - g0 < kG ? p.N - g0 : kG;
          for (int gi = 0; gi < gn; ++gi) {
            const char* drow = static_cast<const char*>(
                row_ptr<DT>(p.drafter, int64_t(g0 + gi) * T + tile, p.V));
            for (int ch = 0; ch < nch; ++ch) put(drow, ch, normal);
          }
          for (int ch = nch - 1; ch >= 0; --ch) {
            put(trow, ch, keep);
            for (int gi = 0; gi < gn; ++gi)
              put(static_cast<const char*>(row_ptr<DT>(p.drafter, int64_t(g0 + gi) * T + tile, p.V)),
                  ch, once);
          }
        }
      }
      if (!ok) {
        // the copies already issued must land before the CTA's memory goes
        for (uint32_t j = k > uint32_t(kStages) ? k - kStages : 0; j < k; ++j) {
          const long long t0 = clock64();
          while (!mbar_test(saddr(&sh.full[j % kStages]), (j / kStages) & 1u) &&
                 clock64() - t0 < kTimeoutCycles) {
          }
        }
      }
    }
  } else {
    consumer<DT>(p, sh, ring0, nvec, nch, T, c, err);
  }
}

}  // namespace

bool preferred(int V, int elem_bytes, int tiles, int sms, int cluster_sms, size_t l2_bytes) {
  if (cluster_sms >= sms || tiles < 2 * sms) return false;
  const double working_set = double(1 + kG) * double(V) * elem_bytes * sms;
  return working_set <= 0.9 * double(l2_bytes);
}

hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, int t0, int grid, float* alpha,
                 int* dev_status, cudaStream_t stream) {
  Params p;
  p.target = target;
  p.path = path;
  p.drafter = drafter;
  p.alpha = alpha;
  p.dev_status = dev_status;
  p.M = M;
  p.N = N;
  p.B = B;
  p.P = P;
  p.V = V;
  p.t0 = t0;
  p.c = c;
  const size_t smem = shared_bytes();
  auto kern = dtype == HS_BF16 ? twopass_kernel<HS_BF16> : twopass_kernel<HS_FP16>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) !=
      cudaSuccess)
    return HS_ERR_CUDA;
  return launch_pdl(kern, dim3(unsigned(grid)), dim3(kThreads), smem, stream, p) == cudaSuccess
             ? HS_OK
             : HS_ERR_CUDA;
}

}  // namespace twopass
}  // namespace hs
