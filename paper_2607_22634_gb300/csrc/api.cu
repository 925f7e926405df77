// Library-wide host entry points: status strings, version, device properties.
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

// One thread waits, with a limit of `limit` SM cycles, for a phase of an mbarrier
// that nothing ever arrives on; the wait runs out and reports PRESTO_DEV_TIMEOUT
// exactly as the kernels' own waits do.  Nothing asynchronous is in flight.
__global__ void wait_selftest_kernel(int32_t* dev_status, long long limit) {
  __shared__ uint64_t bar;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (!mbar_wait(&bar, 0, nullptr, limit)) report(dev_status, PRESTO_DEV_TIMEOUT);
}

}  // namespace

int sm_count() {
  static int counts[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (counts[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    counts[dev] = n;
  }
  return counts[dev];
}

}  // namespace presto

extern "C" const char* presto_status_string(int status) {
  switch (status) {
    case PRESTO_OK:
      return "PRESTO_OK";
    case PRESTO_ERR_INVALID_ARG:
      return "PRESTO_ERR_INVALID_ARG: null pointer, bad size or bad dtype";
    case PRESTO_ERR_UNSUPPORTED:
      return "PRESTO_ERR_UNSUPPORTED: a documented limit is exceeded";
    case PRESTO_ERR_CUDA:
      return "PRESTO_ERR_CUDA: a CUDA call or kernel launch failed";
    case PRESTO_ERR_WORKSPACE:
      return "PRESTO_ERR_WORKSPACE: workspace missing, misaligned or too small";
    default:
      return "PRESTO: unknown status";
  }
}

extern "C" int presto_version(void) { return (1 << 16) | 0; }

extern "C" int presto_build_flags(void) {
#ifdef PRESTO_CHECKS
  return PRESTO_BUILD_CHECKS;
#else
  return 0;
#endif
}

extern "C" int presto_selftest_wait_timeout(int32_t* dev_status, long long wait_cycles,
                                            presto_stream_t stream) {
  PRESTO_CHECK_ARG(dev_status);
  PRESTO_CHECK_ARG(wait_cycles >= 0 && wait_cycles <= presto::kWaitCycles);
  presto::wait_selftest_kernel<<<1, 1, 0, stream>>>(dev_status, wait_cycles);
  return presto::launch_status();
}
