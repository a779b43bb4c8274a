// hs_twopass.h -- internal interface of the two-pass-per-CTA stochastic
// kernel (hs_twopass.cu) the cluster kernel's dispatch hands some shapes to.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {
namespace twopass {

// Whether this kernel should take a call: the cluster kernel would leave
// SMs idle (cluster_sms < sms), there are at least two drafter rows per SM,
// and what each SM keeps in L2 between a row's two passes -- two drafter
// rows and the part of the target row tensor memory does not hold (all past
// 256 KB) -- fits in 90% of L2.
bool preferred(int V, int elem_bytes, int tiles, int N, int sms, int cluster_sms,
               size_t l2_bytes);

// The grid for calls with fewer than two drafter rows per SM whose drafters
// pair up within tiles (N even): one CTA per pair of rows, when that keeps
// at least 70% of the SMs busy and the pairs' working set fits in 90% of L2;
// else 0.  (4 drafters x 56 tiles of 151 936 logits: 112 CTAs, 30.1 us per
// call against the cluster kernel's 30.9.)
int pair_grid(int V, int elem_bytes, int tiles, int N, int sms, size_t l2_bytes);

// The grid for rows longer than the cluster kernel holds (V > 153 600): one
// CTA per SM when there are two drafter rows per SM or more and the SMs'
// working sets (as for preferred()) come to at most twice L2 -- the second
// passes then partly miss L2, but measured on V = 200 000 and 262 144 the call
// still took 1.36-1.45x less time than the streaming kernel's -- else
// pair_grid(); 0 leaves the call to the streaming kernel.
int long_row_grid(int V, int elem_bytes, int tiles, int N, int sms, size_t l2_bytes);

// alpha of tiles t0 .. B*P-1 (bf16/fp16, V % 8 == 0, 16-byte-aligned rows)
// over `grid` CTAs (one per SM), each taking an even, contiguous run of the
// drafter rows (tile-major).
hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, int t0, int grid, float* alpha,
                 int* dev_status, cudaStream_t stream);

}  // namespace twopass
}  // namespace hs
