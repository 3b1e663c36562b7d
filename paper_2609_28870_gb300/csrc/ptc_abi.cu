// C-ABI entry points that belong to no stage.
#include "ptc_internal.h"

extern "C" const char* ptc_strerror(ptc_status s) {
  switch (s) {
    case PTC_OK: return "ok";
    case PTC_ERR_INVALID_ARG: return "invalid argument or malformed device input";
    case PTC_ERR_UNSORTED: return "request timestamps are not non-decreasing";
    case PTC_ERR_OVERFLOW: return "size or cost overflow (N or D >= 2^32-1, or a cost constant >= 2^64)";
    case PTC_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case PTC_ERR_CUDA: return "CUDA runtime error";
    case PTC_ERR_TIMEOUT: return "a bounded device-side wait gave up";
    case PTC_ERR_HASH_COLLISION: return "two different prefixes share one block id";
    case PTC_ERR_NOT_IMPLEMENTED: return "not implemented";
  }
  return "unknown status";
}

extern "C" const char* ptc_version(void) { return "ptc 0.1.0 (sm_103a)"; }
