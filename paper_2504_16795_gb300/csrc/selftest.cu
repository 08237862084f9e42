// Self-test of the bounded waits that every pipelined kernel uses (no device
// fault, no hang): one block initialises an mbarrier that expects one arrival,
// never arrives, and waits on it with the given limit. The wait gives up,
// records the timeout in this file's status word (read and cleared by
// hsa_device_check) and the kernel returns, leaving the context usable.
#include "tc.cuh"

namespace hsa {
namespace {

__device__ unsigned g_selftest_status;

__global__ void __launch_bounds__(32) selftest_wait_kernel(unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  __syncwarp();
  if (threadIdx.x == 0) tc::mbar_wait_for(smem_u32(&bar), 0, limit_ns, &abort_flag, &g_selftest_status);
}

}  // namespace

cudaError_t launch_selftest_wait(unsigned long long limit_ns, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(limit_ns);
  note_launches(1);
  return cudaGetLastError();
}

unsigned selftest_take_status() {
  unsigned v = 0, zero = 0;
  if (cudaMemcpyFromSymbol(&v, g_selftest_status, sizeof(v)) != cudaSuccess) return ~0u;
  cudaMemcpyToSymbol(g_selftest_status, &zero, sizeof(zero));
  return v;
}

}  // namespace hsa
