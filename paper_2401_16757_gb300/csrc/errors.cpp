// Status strings and the per-thread last-error message of the C ABI.
#include <string>

#include "internal.h"

namespace swapnet {
static thread_local std::string t_last_error;
void set_error(const std::string& msg) {
  try {
    t_last_error = msg;
  } catch (...) {  // no room for the message: leave it empty rather than throw
    t_last_error.clear();
  }
}
}  // namespace swapnet

extern "C" {

const char* swapnet_strerror(int status) {
  switch (status) {
    case SWAPNET_OK: return "ok";
    case SWAPNET_ERR_INVALID_ARG: return "invalid argument";
    case SWAPNET_ERR_INFEASIBLE: return "no partition fits the budget";
    case SWAPNET_ERR_OOM: return "out of memory";
    case SWAPNET_ERR_CUDA: return "CUDA error";
    case SWAPNET_ERR_TIMEOUT: return "device-side wait timed out";
    case SWAPNET_ERR_MISALIGNED: return "misaligned pointer or size";
    case SWAPNET_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case SWAPNET_ERR_IO: return "weights file I/O error";
    case SWAPNET_ERR_INTERNAL: return "unexpected host-side error";
    default: return "unknown status";
  }
}

const char* swapnet_last_error(void) { return swapnet::t_last_error.c_str(); }

}  // extern "C"
