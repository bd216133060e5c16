// Library-wide entry points: status names, version, device queries.
#include <cuda_runtime.h>

#include <mutex>

#include "pace_internal.cuh"

namespace pace {

int sm_count() {
  static std::mutex mu;
  static int cached_dev = -1;
  static int cached = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  std::lock_guard<std::mutex> g(mu);
  if (dev != cached_dev) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
      n = 1;
    cached = n;
    cached_dev = dev;
  }
  return cached;
}

uint64_t& launch_counter() {
  thread_local uint64_t n = 0;
  return n;
}

ProfileEvents& profile_events(int kernel) {
  thread_local ProfileEvents ev[2];
  return ev[kernel == PACE_PROFILE_TAG_REDUCE ? 1 : 0];
}

}  // namespace pace

extern "C" pace_status pace_set_profile_events(int32_t kernel, void* begin, void* end) {
  if (kernel != PACE_PROFILE_LMHEAD && kernel != PACE_PROFILE_TAG_REDUCE)
    return PACE_ERR_INVALID_ARG;
  pace::ProfileEvents& e = pace::profile_events(kernel);
  e.begin = static_cast<cudaEvent_t>(begin);
  e.end = static_cast<cudaEvent_t>(end);
  return PACE_OK;
}

extern "C" uint64_t pace_kernel_launches(void) { return pace::launch_counter(); }

extern "C" const char* pace_status_string(pace_status status) {
  switch (status) {
    case PACE_OK: return "PACE_OK";
    case PACE_ERR_INVALID_ARG: return "PACE_ERR_INVALID_ARG";
    case PACE_ERR_VERSION_ORDER: return "PACE_ERR_VERSION_ORDER";
    case PACE_ERR_NAN_INPUT: return "PACE_ERR_NAN_INPUT";
    case PACE_ERR_UNSUPPORTED_SHAPE: return "PACE_ERR_UNSUPPORTED_SHAPE";
    case PACE_ERR_WORKSPACE: return "PACE_ERR_WORKSPACE";
    case PACE_ERR_TIMEOUT: return "PACE_ERR_TIMEOUT";
    case PACE_ERR_CUDA: return "PACE_ERR_CUDA";
  }
  return "PACE_ERR_UNKNOWN";
}

extern "C" int32_t pace_version(void) { return 100; }
