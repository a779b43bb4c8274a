// hs_stream.h -- internal interface of the persistent chunked stochastic
// feedback kernel (hs_stream.cu): every logit read once from HBM, a second
// time from L2.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {
namespace stream {

// Sizes and mode the kernel takes (pointer alignment aside).
bool eligible_sizes(int dtype, int N, int V, int greedy);

// Same, plus the 16-byte alignment of both logit tensors.
bool eligible(const void* target, const void* drafter, int dtype, int N, int V, int greedy);

// Workspace: per-chunk row statistics, per-chunk alpha partials and tile
// counters.
size_t workspace_bytes(int N, int B, int P, int V);

// alpha [N,B,P] (and e_len [N,B] when non-null); c = log2(e) / T.  Clears
// the tile counters, launches the persistent kernel, then one small kernel
// that sums each tile's chunk partials into alpha and forms e_len.
hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, float* alpha, float* e_len, void* ws,
                 int* dev_status, cudaStream_t stream);

// Test hook for the bounded waits: launch() with tile 0's statistics count
// made unreachable (one count more is awaited than exist) and every counter
// wait limited to wait_cycles clock cycles, so that tile 0's waits run out:
// they report HS_ERR_TIMEOUT and tile 0's alphas come out NaN, while every
// other tile completes normally.
hs_status launch_wait_test(const void* target, const void* drafter, int dtype, int N, int B,
                           int P, int V, float c, long long wait_cycles, float* alpha,
                           float* e_len, void* ws, int* dev_status, cudaStream_t stream);

}  // namespace stream
}  // namespace hs
