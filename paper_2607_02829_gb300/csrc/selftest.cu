// Self-test of the bounded pipeline wait (sr_selftest_wait_timeout): the
// mbarrier wait every tensor-core kernel uses, run on a barrier that nothing
// arrives at, with a short limit.  The wait must give up, set bit 0 of the fault
// word and return, leaving the context usable.  No TMA, no tensor memory.
#include <string>

#include "../../include/sparse_reslim.h"
#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace sr {
void set_error_message(const std::string& msg);
}  // namespace sr

namespace {

using namespace sr::tc;

__global__ void __launch_bounds__(32, 1)
wait_timeout_kernel(unsigned int* fault, unsigned long long limit_ns,
                    unsigned long long* waited_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);          // one arrival would complete phase 0; none comes
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncwarp();
  if (threadIdx.x == 0) {
    const unsigned long long t0 = global_ns();
    const bool completed = mbar_wait(&bar, 0, &abort_flag, fault, limit_ns);
    *waited_ns = global_ns() - t0;
    if (completed) atomicOr(fault, 0x80000000u);   // cannot happen: nothing arrived
  }
}

sr_status reject(sr_status st, const std::string& msg) {
  sr::set_error_message(msg);
  return st;
}

}  // namespace

extern "C" sr_status sr_selftest_wait_timeout(uint32_t* fault, uint32_t limit_us,
                                              uint64_t* waited_ns, void* stream) {
  if (!fault || (reinterpret_cast<uintptr_t>(fault) % 4) != 0)
    return reject(SR_ERR_INVALID_ARG, "fault must be a non-NULL, 4-byte aligned device pointer");
  if (!waited_ns || (reinterpret_cast<uintptr_t>(waited_ns) % 8) != 0)
    return reject(SR_ERR_INVALID_ARG, "waited_ns must be a non-NULL, 8-byte aligned device pointer");
  if (limit_us < 1 || limit_us > 1000000)
    return reject(SR_ERR_INVALID_ARG, "limit_us must lie in 1 .. 1000000");
  wait_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      fault, 1000ull * limit_us, reinterpret_cast<unsigned long long*>(waited_ns));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess)
    return reject(SR_ERR_CUDA, std::string("wait_timeout_kernel: ") + cudaGetErrorString(e));
  return SR_OK;
}
