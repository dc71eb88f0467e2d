// failure.cu — a check of the failure reporting behind every bounded wait.
//
// Kernels that stream with bulk copies wait on mbarriers with mbar_wait_bounded: a
// wait that runs out writes kDevWaitTimeout into the caller's device error word and
// the kernel returns, so the context stays usable and the host reads the status when
// it chooses.  semkv_debug_wait_timeout runs that same wait on a barrier nothing
// arrives on, with a caller-chosen short poll limit, so a test can make a wait run
// out without faulting or hanging the GPU.
#include "checks.h"
#include "common.cuh"

namespace {

// One CTA: every warp waits on a barrier that expects one arrival which never comes;
// each wait gives up after `polls` polls and the warp records the timeout.
__global__ void wait_timeout_kernel(int32_t* err, uint32_t polls) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0)
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(
                     (uint32_t)__cvta_generic_to_shared(&bar))
                 : "memory");
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  __syncthreads();
  const bool done = semkv::mbar_wait_bounded(&bar, 0u, polls);
  if (!done && (threadIdx.x & 31) == 0) semkv::raise_error(err, semkv::kDevWaitTimeout);
}

}  // namespace

extern "C" semkv_status semkv_debug_wait_timeout(int32_t* dev_error, uint32_t polls,
                                                 void* stream) {
  if (!dev_error || polls < 1 || polls > semkv::kWaitPolls) return SEMKV_EINVAL;
  if (!semkv::aligned(dev_error, 4)) return SEMKV_EALIGN;
  wait_timeout_kernel<<<1, 128, 0, (cudaStream_t)stream>>>(dev_error, polls);
  return cudaGetLastError() == cudaSuccess ? SEMKV_OK : SEMKV_ECUDA;
}
