// Self-test of the bounded device waits (e2s_selftest_bounded_wait).
//
// Every mbarrier wait in the score kernels gives up after a wall-clock limit,
// records E2S_ERR_TIMEOUT in the status word and lets the kernel return, so a
// lost arrival ends the launch with an error the host can read instead of a
// hung GPU.  This kernel exercises exactly that wait (ptx::mbar_wait) on a
// barrier with nothing else in flight: no TMA copy, no MMA, no other thread.
#include <cuda_runtime.h>

#include "sm100_ptx.cuh"

namespace e2s {
namespace {

__global__ void bounded_wait_kernel(int complete, uint64_t limit_ns, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  ptx::mbar_init(&bar, 2);              // phase 0 completes after two arrivals
  ptx::fence_barrier_init();
  ptx::mbar_arrive(&bar);
  if (complete) ptx::mbar_arrive(&bar);
  ptx::mbar_wait(&bar, 0, limit_ns, status);
}

}  // namespace
}  // namespace e2s

extern "C" e2s_status e2s_selftest_bounded_wait(int32_t complete, int64_t limit_ns, void* ws,
                                                void* stream) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return E2S_ERR_WORKSPACE;
  if (limit_ns < 1000000 || limit_ns > 2000000000) return E2S_ERR_INVALID_ARG;
  e2s::bounded_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      complete != 0, static_cast<uint64_t>(limit_ns), static_cast<uint32_t*>(ws));
  return cudaGetLastError() == cudaSuccess ? E2S_OK : E2S_ERR_CUDA;
}
