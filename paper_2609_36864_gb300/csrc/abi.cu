// Library-wide entry points of the C ABI declared in hdl.h.
#include "hdl.h"

extern "C" int32_t hdl_abi_version(void) { return HDL_ABI_VERSION; }

extern "C" const char* hdl_status_string(hdl_status s) {
  switch (s) {
    case HDL_OK: return "HDL_OK";
    case HDL_ERR_INVALID_ARG: return "HDL_ERR_INVALID_ARG";
    case HDL_ERR_UNSUPPORTED: return "HDL_ERR_UNSUPPORTED";
    case HDL_ERR_WORKSPACE: return "HDL_ERR_WORKSPACE";
    case HDL_ERR_CUDA: return "HDL_ERR_CUDA";
    case HDL_ERR_TIMEOUT: return "HDL_ERR_TIMEOUT";
    case HDL_ERR_BAD_TARGET: return "HDL_ERR_BAD_TARGET";
  }
  return "HDL_ERR_UNKNOWN";
}
