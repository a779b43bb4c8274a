// hs_fused.h -- internal interface of the single-read cluster kernel
// (hs_fused.cu) used by hs_feedback / hs_feedback_path.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {
namespace fused {

constexpr int kMaxC = 8;   // CTAs per cluster (portable limit)
constexpr int kMaxN = 32;  // drafters per tile the kernel accumulates

// For bf16/fp16 rows the cluster kernel cannot hold (V > 153 600): the
// two-pass kernel's grid (twopass::long_row_grid on this device), 0 for the
// streaming kernel.
int long_row_grid(int N, int B, int P, int V);

// The two-pass kernel on `grid` CTAs, then e_len (when non-null).
hs_status launch_two_pass(const void* target, const int32_t* path, int M, const void* drafter,
                          int dtype, int N, int B, int P, int V, float c, int grid, float* alpha,
                          float* e_len, int* dev_status, cudaStream_t stream);

// Sizes and mode the kernel takes (pointer alignment aside).
bool eligible_sizes(int dtype, int N, int V, int greedy);

// Same, plus the 16-byte alignment of both logit tensors.
bool eligible(const void* target, const void* drafter, int dtype, int N, int V, int greedy);

// alpha [N,B,P] (and e_len [N,B] when non-null) for stochastic feedback;
// c = log2(e) / T.  Launches the cluster kernel and, for e_len, one small
// kernel.
hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, float c, float* alpha, float* e_len,
                 int* dev_status, cudaStream_t stream);

}  // namespace fused
}  // namespace hs
