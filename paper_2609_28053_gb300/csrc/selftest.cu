// selftest.cu -- failure detection without a GPU fault.
//
// Every wait in this library's kernels is a bounded poll of a shared-memory
// mbarrier; when a pipeline stalls, the kernel gives up, writes
// EQB_ERR_CUDA to the caller's error word and returns, and the context stays
// usable.  This kernel exercises that path on purpose: one thread waits on a
// barrier that nothing ever completes, with the same bounded poll, and
// reports the stall.
#include <cuda_runtime.h>
#include <stdint.h>

#include "eqb.h"
#include "eqb_device.cuh"

namespace eqb {
namespace {

__global__ void stalled_wait_kernel(int32_t* err, uint32_t polls) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = saddr(&bar);
  if (threadIdx.x == 0) {
    bar_init(b, 1);  // one arrival expected; none will come
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0 && !bar_wait_bounded(b, 0u, polls)) raise_flag(err, kErrCuda);
}

}  // namespace
}  // namespace eqb

extern "C" eqb_status eqb_selftest_stalled_wait(int32_t* err_flag, int32_t polls, void* stream) {
  if (!err_flag || polls < 1 || polls > (1 << 24)) return EQB_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(err_flag) % 4) != 0) return EQB_ERR_INVALID_ARG;
  eqb::stalled_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      err_flag, static_cast<uint32_t>(polls));
  return cudaGetLastError() == cudaSuccess ? EQB_OK : EQB_ERR_CUDA;
}
