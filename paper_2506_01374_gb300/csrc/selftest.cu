// Self-test of the bounded device waits that every tensor-core kernel uses.
// One thread waits on an mbarrier phase that nothing completes; the wait must
// give up after its limit and record a timeout in the status word instead of
// hanging, and the CUDA context must stay usable afterwards.
#include <cuda_runtime.h>

#include "rc_internal.h"
#include "tc_common.cuh"

namespace {
__global__ void bounded_wait_kernel(int* status, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !tc::mbar_wait_for(&bar, 0, &abort_flag, status, limit_ns))
    tc::record_failure(status, RC_DEV_TIMEOUT_FULL);
}
}  // namespace

extern "C" rc_status rc_selftest_bounded_wait(double wait_ms, void* stream) {
  if (!(wait_ms > 0) || wait_ms > 2000) return rc_fail(RC_ERR_INVALID_ARG, "rc_selftest_bounded_wait: 0 < wait_ms <= 2000");
  int* st = nullptr;
  cudaError_t e = cudaMalloc((void**)&st, sizeof(int));
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "rc_selftest_bounded_wait: %s", cudaGetErrorString(e));
  int h = 0;
  e = cudaMemsetAsync(st, 0, sizeof(int), (cudaStream_t)stream);
  if (e == cudaSuccess) {
    bounded_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(st, (unsigned long long)(wait_ms * 1e6));
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaMemcpy(&h, st, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(st);
  if (e != cudaSuccess) return rc_fail(RC_ERR_CUDA, "rc_selftest_bounded_wait: %s", cudaGetErrorString(e));
  if (h == RC_DEV_TIMEOUT_FULL) return rc_fail(RC_ERR_DEVICE_TIMEOUT, "bounded wait gave up as designed");
  return RC_OK;  // the wait did not give up: the self-test failed
}
