// Testing hooks for the failure paths (declared in include/tq.h under
// "Testing hooks"): a kernel whose only wait can never be satisfied, so the
// scans' bounded wait runs out and reports through the search status word.
#include <cuda_runtime.h>

#include <cstdint>

#include "tq_internal.h"
#include "tq_kernels.h"
#include "tq_wait.cuh"

namespace tq {
namespace {

__global__ void k_debug_wait(long long budget, int* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(wait_smem_u32(&bar)));
    abort_flag = 0;
  }
  __syncthreads();
  // nothing ever arrives on `bar`: phase 0 never completes
  if (threadIdx.x == 0) bounded_wait(&bar, 0, &abort_flag, status, 99, budget);
}

thread_local int t_fail_allocs = 0;

}  // namespace

int& fail_allocs() { return t_fail_allocs; }

cudaError_t dev_malloc(void** p, size_t bytes) {
  if (t_fail_allocs > 0) {
    --t_fail_allocs;
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(p, bytes);
}

cudaError_t launch_debug_wait(long long budget, int* status, cudaStream_t s) {
  k_debug_wait<<<1, 32, 0, s>>>(budget, status);
  return cudaGetLastError();
}

}  // namespace tq

extern "C" tq_status tq_debug_fail_allocs(int count) {
  if (count < 0) return tq::fail(TQ_EINVAL, "tq_debug_fail_allocs: count %d < 0", count);
  tq::fail_allocs() = count;
  return tq::ok();
}
