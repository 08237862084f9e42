// Self-test of the bounded waits that every pipelined kernel uses (no device
// fault, no hang): one block initialises an mbarrier that expects one arrival,
// never arrives, and waits on it with the given limit. The wait gives up,
// records the timeout in the status word it is given (the header of the
// caller's workspace, read and cleared by hsa_check) and the kernel returns,
// leaving the context usable.
#include "tc.cuh"

namespace hsa {
namespace {

__global__ void __launch_bounds__(32) selftest_wait_kernel(unsigned long long limit_ns, unsigned* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncwarp();
  if (threadIdx.x == 0) tc::mbar_wait_for(smem_u32(&bar), 0, limit_ns, &abort_flag, status);
}

}  // namespace

cudaError_t launch_selftest_wait(unsigned long long limit_ns, unsigned* status, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(limit_ns, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace hsa
