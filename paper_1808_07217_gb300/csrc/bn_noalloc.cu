// lsgd_batchnorm_stats_noalloc: the per-worker BatchNorm statistics without any device allocation.
//
// Some callers cannot let a library allocate device memory mid-run: a framework that has handed
// all free HBM to its own caching pool (so cudaMalloc / cudaMallocAsync would fail, or make the
// pool release cached blocks and stall), or a latency-critical training loop that budgets every
// byte at start-up and treats an allocation in the loop as an error.  This entry point computes the
// same statistics as lsgd_batchnorm_stats, with its chunk partials in a fixed array that is part of
// the library's device image instead of a stream-ordered allocation.
#include <mutex>
#include <string>

#include "../../include/lsgd.h"
#include "lsgd_internal.h"
#include "resnet.h"

namespace {

// Room for G * ceil(P / 1024) * C * 2 partial values, e.g. 16 replicas x 128 chunks x 64 channels.
// Every GPU that loads the library keeps these 4 MiB until the process exits.
constexpr size_t kNoAllocScratchFloats = size_t(1) << 20;
static __device__ __align__(256) float g_bn_noalloc_scratch[kNoAllocScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
float* g_scratch_on_device[kMaxDevices] = {};

}  // namespace

extern "C" lsgd_status lsgd_batchnorm_stats_noalloc(const float* y, int64_t P, int C, int G,
                                                    float* mean, float* rstd, void* stream) {
  if (!y || !mean || !rstd || P < 1 || C < 1 || C > 256 || G < 1 || G > 65535 ||
      (P + 1023) / 1024 > 65535) {
    lsgd::set_last_error("lsgd_batchnorm_stats_noalloc: bad arguments");
    return LSGD_EINVAL;
  }
  const size_t need = lsgd::batchnorm_stats_scratch_floats(P, C, G);
  if (need > kNoAllocScratchFloats) {
    lsgd::set_last_error("lsgd_batchnorm_stats_noalloc: G * ceil(P / 1024) * C * 2 = " +
                         std::to_string(need) + " partial values exceed the fixed scratch of " +
                         std::to_string(kNoAllocScratchFloats) + " (use lsgd_batchnorm_stats)");
    return LSGD_EINVAL;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    lsgd::set_last_error("lsgd_batchnorm_stats_noalloc: no usable current device");
    return LSGD_ECUDA;
  }
  // In host code the array's name is only a host-side stand-in; the kernels need its device
  // address, looked up once per device (with that device current) on the first call.
  float* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_scratch_on_device[dev]) {
      void* p = nullptr;
      const cudaError_t e = cudaGetSymbolAddress(&p, g_bn_noalloc_scratch);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        lsgd::set_last_error(std::string("lsgd_batchnorm_stats_noalloc: cudaGetSymbolAddress: ") +
                             cudaGetErrorString(e));
        return LSGD_ECUDA;
      }
      g_scratch_on_device[dev] = static_cast<float*>(p);
    }
    scratch = g_scratch_on_device[dev];
  }
  // The first pass overwrites every partial value the second pass reads, so nothing has to be
  // cleared between calls.
  const cudaError_t e =
      lsgd::launch_batchnorm_stats(y, P, C, G, mean, rstd, scratch, (cudaStream_t)stream);
  if (e != cudaSuccess) {
    lsgd::set_last_error(std::string("lsgd_batchnorm_stats_noalloc: ") + cudaGetErrorString(e));
    return LSGD_ECUDA;
  }
  return LSGD_OK;
}
