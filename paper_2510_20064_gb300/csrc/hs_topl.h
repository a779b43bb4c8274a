// hs_topl.h -- internal interface of the draft-tree feedback (Thm 2) kernels
// in hs_topl.cu, used by hs_feedback_topl / hs_feedback_topl_path.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {
namespace topl {

constexpr int kMaxL = 16;  // children per node the kernels rank

// Bytes of workspace launch() needs: the target rows' share statistics, the
// drafter rows' candidate lists, and one counter per (drafter, query).
size_t workspace_bytes(int N, int B, int P, int V);

// Kernels one launch() runs.
int kernel_count(int N, int B, int P, int V);

// alpha [N,B,P] (and e_len [N,B] when non-null); c = log2(e) / T.  keep
// (device [N,B,P] int32, or null for all L): the candidate set of drafter row
// r is the first keep[r] tokens of its top L; a keep outside [0, L] gives NaN
// and HS_ERR_INVALID_ARG in *dev_status.
hs_status launch(const void* target, const int32_t* path, int M, const void* drafter, int dtype,
                 int N, int B, int P, int V, int L, const int32_t* keep, int greedy, float c,
                 float* alpha, float* e_len, void* ws, int* dev_status, cudaStream_t stream);

}  // namespace topl
}  // namespace hs
