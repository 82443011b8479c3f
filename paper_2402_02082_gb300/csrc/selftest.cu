// Self-test of the kernels' failure path: bounded waits that give up, record
// GLIDE_ERR_DEVICE_TIMEOUT in the workspace and release every other waiter of
// the CTA, leaving the CUDA context usable.  Nothing here faults or hangs: the
// barrier that never completes is waited on with a short, bounded limit.
#include <cuda_runtime.h>

#include "../../include/glide.h"
#include "common.cuh"

namespace {

__global__ void selftest_timeout_kernel(unsigned* status, uint64_t limit_ns) {
  __shared__ uint64_t bar[2];
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    glide::mbar_init(&bar[0], 1);
    glide::mbar_init(&bar[1], 1);
    abort_flag = 0;
    glide::fence_barrier_init();
  }
  __syncthreads();
  // Nothing ever arrives on either barrier.  Warp 0 gives up after limit_ns and
  // raises the abort flag; warp 1 would wait ten times longer, but the flag
  // releases it as soon as warp 0 gives up.
  if (threadIdx.x == 0) glide::mbar_wait(&bar[0], 0, &abort_flag, status, limit_ns);
  if (threadIdx.x == 32) glide::mbar_wait(&bar[1], 0, &abort_flag, status, 10 * limit_ns);
}

}  // namespace

extern "C" glide_status glide_selftest_wait_timeout(void* workspace, uint32_t limit_us, glide_stream_t stream) {
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 15u) || limit_us < 1 || limit_us > 2000000)
    return GLIDE_ERR_INVALID;
  selftest_timeout_kernel<<<1, 64, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<unsigned*>(workspace), (uint64_t)limit_us * 1000ull);
  return cudaGetLastError() == cudaSuccess ? GLIDE_OK : GLIDE_ERR_CUDA;
}
