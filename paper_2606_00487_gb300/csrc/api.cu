// Library-wide entry points of the TAPS C ABI (status strings, version).
#include "common.cuh"

extern "C" const char* taps_status_string(int status) {
  switch (status) {
    case TAPS_OK: return "ok";
    case TAPS_ERR_INVALID_ARG: return "invalid argument";
    case TAPS_ERR_UNSUPPORTED: return "unsupported size or option";
    case TAPS_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case TAPS_ERR_CUDA: return "CUDA launch failed";
    case TAPS_ERR_DEVICE: return "device-detected fault";
    default: return "unknown status";
  }
}

extern "C" int taps_version(void) { return 1; }
