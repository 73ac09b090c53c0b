// Self-test of the bounded pipeline waits: a kernel waits on an mbarrier
// that nothing arrives on, gives up after a short limit through the same wait
// routine the GEMM roles use, records SOLO_FLAG_TIMEOUT and returns.
#include "internal.h"
#include "ptx.cuh"
#include "../../include/solo_readout.h"

namespace solo {
namespace {

__global__ void wait_timeout_selftest_kernel(uint32_t* flags, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbarrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // Phase 0 of a fresh barrier completes only after one arrival; none comes.
    const bool completed = mbar_wait_limit(&bar, 0, &abort_flag, limit_ns);
    atomicOr(flags, completed ? 0u : static_cast<uint32_t>(SOLO_FLAG_TIMEOUT));
  }
}

}  // namespace
}  // namespace solo

extern "C" solo_status_t solo_readout_selftest_wait_timeout(uint32_t* device_flags,
                                                            uint32_t limit_us,
                                                            solo_stream_t stream) {
  if (device_flags == nullptr || limit_us == 0 || limit_us > 1000000u) return SOLO_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(device_flags) & 3u) return SOLO_ERR_MISALIGNED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  solo::wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(device_flags,
                                                      static_cast<uint64_t>(limit_us) * 1000ull);
  return solo::launched() == cudaSuccess ? SOLO_OK : SOLO_ERR_CUDA;
}
