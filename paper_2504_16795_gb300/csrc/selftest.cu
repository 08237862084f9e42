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

// The selection's tensor-core score pass on one tile, to measure the rounding
// that its certificate bounds: C [128, 64] = A [128, D] . B [64, D]^T with the
// operands in the layout the selection kernel gives them (K-major, 128-byte
// swizzle, 64-column blocks stacked) and the same instruction sequence (one
// bf16 MMA of K = 16 per step, accumulating in tensor memory in increasing
// K). One block of four warps; thread r reads row r of the accumulator.
template <int D>
__global__ void __launch_bounds__(128, 1) selftest_score_tile_kernel(const uint16_t* __restrict__ A,
                                                                     const uint16_t* __restrict__ B,
                                                                     float* __restrict__ C, unsigned* status) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ uint64_t bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  constexpr int kM = 128, kN = 64, D8 = D / 8;
  const uint32_t abase = smem_u32(smem_raw) + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t bbase = abase + kM * D * 2;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int u = tid; u < kM * D8; u += 128) {
    const int r = u / D8, ch = u % D8;
    const uint4 v = reinterpret_cast<const uint4*>(A + (long long)r * D)[ch];
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(abase + tc::sw128_offset(kM, r, ch * 8)), "r"(v.x),
                 "r"(v.y), "r"(v.z), "r"(v.w));
  }
  for (int u = tid; u < kN * D8; u += 128) {
    const int r = u / D8, ch = u % D8;
    const uint4 v = reinterpret_cast<const uint4*>(B + (long long)r * D)[ch];
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(bbase + tc::sw128_offset(kN, r, ch * 8)), "r"(v.x),
                 "r"(v.y), "r"(v.z), "r"(v.w));
  }
  tc::fence_proxy_async_smem();
  if (tid == 0) {
    tc::mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(smem_u32(&tmem_base), kN);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;
  if (tid == 0) {
    constexpr uint32_t idesc = tc::idesc_bf16(kM, kN);
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint32_t blk = kk >> 2, w = kk & 3;
      tc::mma_bf16_ss(tmem, tc::sdesc_sw128(abase + blk * kM * 128 + w * 32),
                      tc::sdesc_sw128(bbase + blk * kN * 128 + w * 32), idesc, kk > 0);
    }
    tc::mma_commit(smem_u32(&bar));
  }
  __syncwarp();
  const bool ok = tc::mbar_wait(smem_u32(&bar), 0, &abort_flag, status);
  tc::fence_after_sync();
  if (ok) {
#pragma unroll
    for (int h = 0; h < kN / 32; ++h) {
      float x[32];
      tc::tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + h * 32, x);
      tc::tmem_wait_ld();
#pragma unroll
      for (int c = 0; c < 32; ++c) C[(long long)(warp * 32 + lane) * kN + h * 32 + c] = x[c];
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kN);
  }
}

template <int D>
cudaError_t run_score_tile(const void* A, const void* B, float* C, unsigned* status, cudaStream_t st) {
  const size_t smem = (size_t)(128 + 64) * D * 2 + 1024;
  cudaError_t e = cudaFuncSetAttribute(selftest_score_tile_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  selftest_score_tile_kernel<D><<<1, 128, smem, st>>>((const uint16_t*)A, (const uint16_t*)B, C, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_selftest_score_tile(int d, const void* A, const void* B, float* C, unsigned* status,
                                       cudaStream_t st) {
  return d == 64 ? run_score_tile<64>(A, B, C, status, st) : run_score_tile<128>(A, B, C, status, st);
}

cudaError_t launch_selftest_wait(unsigned long long limit_ns, unsigned* status, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(limit_ns, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace hsa
