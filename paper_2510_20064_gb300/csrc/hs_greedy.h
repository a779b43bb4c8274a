// hs_greedy.h -- internal interface of the greedy feedback kernels
// (hs_greedy.cu) used by hs_feedback / hs_feedback_path.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hedgefb.h"

namespace hs {
namespace greedy {

// Maximum of a chunk of one row and the first index holding it.
struct Part {
  float m;
  int idx;
};

int64_t chunk_elems(int dtype);
size_t workspace_bytes(int N, int B, int P, int V, int dtype);

// alpha [N,B,P] in {0,1} (NaN for unusable rows) and e_len [N,B]; `vec`
// selects 16-byte loads (rows 16-byte aligned).  Two kernel launches.
hs_status launch(bool vec, const void* target, const int32_t* path, int M, const void* drafter,
                 int dtype, int N, int B, int P, int V, float* alpha, float* e_len, void* ws,
                 int* dev_status, cudaStream_t s);

}  // namespace greedy
}  // namespace hs
