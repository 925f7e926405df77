// Library-wide host entry points: status strings, version, device properties.
#include <mutex>

#include "common.cuh"

namespace presto {

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
