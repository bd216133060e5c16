// Library-wide entry points: status names, version, device queries.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <mutex>

#include "pace_internal.cuh"
#include "pace_tma.cuh"

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

std::atomic<int>& lmhead_split_pref() {
  static std::atomic<int> s{0};
  return s;
}

namespace {

// cuTensorMapEncodeTiled from the driver, looked up through the runtime so the
// library links no driver stub and loads on machines without a GPU.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

}  // namespace

pace_status encode_bf16_2d(CUtensorMap* tm, const void* ptr, int64_t rows, int64_t cols,
                           int64_t ld, int box_inner, int box_outer) {
  auto enc = tensor_map_encoder();
  if (!enc) return PACE_ERR_CUDA;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_outer)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? PACE_OK : PACE_ERR_UNSUPPORTED_SHAPE;
}

ProfileEvents& profile_events(int kernel) {
  thread_local ProfileEvents ev[2];
  return ev[kernel == PACE_PROFILE_TAG_REDUCE ? 1 : 0];
}

namespace {

// One thread waits, with the kernels' bounded wait, on an mbarrier that no
// thread ever arrives on; the wait gives up after limit_ns and the timeout is
// reported exactly as the tensor-core kernels report theirs.
__global__ void wait_timeout_selftest_kernel(uint64_t limit_ns, int32_t* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (!mbar_wait_bounded(&bar, 0, nullptr, limit_ns)) report(status, PACE_ERR_TIMEOUT);
}

}  // namespace

}  // namespace pace

extern "C" pace_status pace_wait_timeout_selftest(uint64_t limit_ns, int32_t* status_dev,
                                                  void* stream) {
  if (!status_dev || limit_ns == 0 || limit_ns > pace::kWaitLimitNs)
    return PACE_ERR_INVALID_ARG;
  pace::wait_timeout_selftest_kernel<<<1, 32, 0, pace::as_stream(stream)>>>(limit_ns, status_dev);
  return pace::last_launch_status();
}

extern "C" pace_status pace_set_profile_events(int32_t kernel, void* begin, void* end) {
  if (kernel != PACE_PROFILE_LMHEAD && kernel != PACE_PROFILE_TAG_REDUCE)
    return PACE_ERR_INVALID_ARG;
  pace::ProfileEvents& e = pace::profile_events(kernel);
  e.begin = static_cast<cudaEvent_t>(begin);
  e.end = static_cast<cudaEvent_t>(end);
  return PACE_OK;
}

extern "C" uint64_t pace_kernel_launches(void) { return pace::launch_counter(); }

extern "C" pace_status pace_set_lmhead_splits(int32_t splits) {
  if (splits < 0 || splits > 8) return PACE_ERR_INVALID_ARG;
  pace::lmhead_split_pref().store(splits);
  return PACE_OK;
}

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

extern "C" int32_t pace_version(void) { return 300; }
