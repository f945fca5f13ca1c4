// Self-test of the bounded mbarrier wait (zl_wait_selftest): one CTA waits, with the same helper every
// tcgen05 kernel uses, on an mbarrier that nothing arrives at. The wait gives up after its limit,
// records ZL_DEVERR_TIMEOUT in the error word and the kernel returns normally.
#include <cuda_runtime.h>

#include <string>

#include "common.cuh"
#include "ops.h"
#include "tcgen05.cuh"
#include "zerolock.h"

namespace {

__global__ void __launch_bounds__(64, 1) wait_selftest_k(unsigned* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    zl::tc::mbar_init(&bar, 1);   // one arrival would complete phase 0; none is ever made
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x < 32) zl::tc::uwait(&bar, 0u, &abort_flag, err);   // warp-uniform, as in the kernels
  __syncthreads();
}

zl_status fail(zl_status st, const std::string& m) {
  zl::set_last_error(m);
  return st;
}

bool sticky(cudaError_t e) {
  return e == cudaErrorIllegalAddress || e == cudaErrorLaunchFailure || e == cudaErrorIllegalInstruction ||
         e == cudaErrorMisalignedAddress || e == cudaErrorHardwareStackError || e == cudaErrorAssert;
}

}  // namespace

extern "C" zl_status zl_wait_selftest(unsigned* bits_out) {
  if (!bits_out) return fail(ZL_ERR_ARG, "NULL argument");
  cudaStream_t s = nullptr;
  unsigned* err = nullptr;
  cudaError_t e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaMallocAsync((void**)&err, sizeof(unsigned), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(err, 0, sizeof(unsigned), s);
  if (e == cudaSuccess) {
    zl::note_launch(1);
    wait_selftest_k<<<1, 64, 0, s>>>(err);
    e = cudaGetLastError();
  }
  unsigned bits = 0;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&bits, err, sizeof(unsigned), cudaMemcpyDeviceToHost, s);
  if (err) cudaFreeAsync(err, s);
  const cudaError_t e2 = s ? cudaStreamSynchronize(s) : cudaSuccess;
  if (e == cudaSuccess) e = e2;
  if (s) cudaStreamDestroy(s);
  if (e != cudaSuccess)
    return fail(sticky(e) ? ZL_ERR_STATE : ZL_ERR_CUDA, std::string("zl_wait_selftest: ") + cudaGetErrorString(e));
  *bits_out = bits;
  return ZL_OK;
}
