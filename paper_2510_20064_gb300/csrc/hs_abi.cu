// hs_abi.cu -- status strings and version of the libhedgefb C ABI.
#include "hedgefb.h"

extern "C" const char* hs_status_string(int status) {
  switch (status) {
    case HS_OK: return "HS_OK";
    case HS_ERR_INVALID_ARG: return "HS_ERR_INVALID_ARG: invalid argument";
    case HS_ERR_UNSUPPORTED: return "HS_ERR_UNSUPPORTED: outside the supported sizes";
    case HS_ERR_MISALIGNED: return "HS_ERR_MISALIGNED: pointer not aligned to its element type";
    case HS_ERR_NONFINITE: return "HS_ERR_NONFINITE: NaN, +inf or all -inf logit row";
    case HS_ERR_CUDA: return "HS_ERR_CUDA: CUDA launch failed";
    case HS_ERR_TIMEOUT: return "HS_ERR_TIMEOUT: a bounded device wait ran out";
    default: return "HS_ERR_UNKNOWN: unknown status code";
  }
}

extern "C" int hs_version(void) { return 100; }
