// Chunk mean pool: K̄_i = (1/S) sum_{s<S} K_{iS+s}  (§3.1 "Chunk Selection";
// Appendix A, Eq. 3). Pure bandwidth: K is read once, K̄ written once.
//
// Thread (b, i, g, e8) owns 8 consecutive elements of the head dimension of one
// chunk summary and walks the chunk's S rows in token order, so a warp reads
// 32 x 16 contiguous bytes per row. The sum is fp32 in token order followed by
// one division by S; the bf16 copy is its round-to-nearest-even.
#include "common.cuh"

namespace hsa {
namespace {

constexpr int kBatch = 16;

__global__ void __launch_bounds__(256) pool_kernel(const uint4* __restrict__ K, float4* __restrict__ kbar32,
                                                   uint4* __restrict__ kbar16, int L, int Hkv, int d8, int S,
                                                   long long total) {
  griddep_wait();
  const long long stride = (long long)gridDim.x * blockDim.x;
  const int Nc = L / S;
  const long long row_vec = (long long)Hkv * d8;  // uint4 per token row
  for (long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
    const long long e8 = u % d8;
    const long long g = (u / d8) % Hkv;
    const long long i = (u / ((long long)d8 * Hkv)) % Nc;
    const long long b = u / ((long long)d8 * Hkv * Nc);
    const uint4* src = K + ((b * L + i * S) * Hkv + g) * d8 + e8;
    float acc[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] = 0.f;
    // kBatch rows in flight per thread: all loads of a batch are issued before
    // its sums, which still run in token order
    for (int s0 = 0; s0 < S; s0 += kBatch) {
      uint4 v[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j)
        if (s0 + j < S) v[j] = __ldg(src + (long long)(s0 + j) * row_vec);
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        if (s0 + j < S) {
          acc[0] = acc[0] + bf16_lo(v[j].x);
          acc[1] = acc[1] + bf16_hi(v[j].x);
          acc[2] = acc[2] + bf16_lo(v[j].y);
          acc[3] = acc[3] + bf16_hi(v[j].y);
          acc[4] = acc[4] + bf16_lo(v[j].z);
          acc[5] = acc[5] + bf16_hi(v[j].z);
          acc[6] = acc[6] + bf16_lo(v[j].w);
          acc[7] = acc[7] + bf16_hi(v[j].w);
        }
      }
    }
    const float fs = (float)S;
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] = __fdiv_rn(acc[c], fs);
    kbar32[u * 2] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    kbar32[u * 2 + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    if (kbar16) {
      uint4 o;
      o.x = pack_bf16x2(acc[0], acc[1]);
      o.y = pack_bf16x2(acc[2], acc[3]);
      o.z = pack_bf16x2(acc[4], acc[5]);
      o.w = pack_bf16x2(acc[6], acc[7]);
      kbar16[u] = o;
    }
  }
}

}  // namespace

cudaError_t launch_pool(const Dims& D, const void* K, float* kbar32, void* kbar16, cudaStream_t st) {
  const int d8 = D.d / 8;
  const long long total = (long long)D.B * D.Nc * D.Hkv * d8;
  if (total == 0) return cudaSuccess;
  const int grid = grid_cap((total + 255) / 256, 152LL * 16);
  (void)launch_dependent(pool_kernel, dim3(grid), dim3(256), 0, st, (const uint4*)K, (float4*)kbar32, (uint4*)kbar16,
                         D.L, D.Hkv, d8, D.S, total);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace hsa
