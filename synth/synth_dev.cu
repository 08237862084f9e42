// Seeded synthetic-input generator, device implementation.
//
// Holds no arithmetic of the attention method: it only writes the seeded
// inputs directly into device memory so that large workloads need no host
// generation and no host-to-device copy. The definitions are the same
// published ones the host implementation (synth_host.c) follows, written here
// independently:
//   * SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): output n of the stream
//     that starts in state s0 is mix64(s0 + (n + 1) * 0x9E3779B97F4A7C15);
//     a seed selects s0 = mix64(seed).
//   * Irwin-Hall(12) normal: element e sums the twelve 16-bit fields of
//     outputs 3e, 3e+1, 3e+2 and returns (2 * sum - 786420) / 2^17.
//   * bf16 = round-to-nearest-even of the fp32 value.
// A test compares the two implementations bit for bit.
#include <cstdint>
#include <cuda_runtime.h>

#include "synth.h"

namespace {

__device__ __forceinline__ uint64_t dev_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

__device__ __forceinline__ float dev_ih12(uint64_t s0, uint64_t e) {
  uint32_t acc = 0;
#pragma unroll
  for (int r = 0; r < 3; ++r) {
    uint64_t x = dev_mix64(s0 + (3ULL * e + r + 1ULL) * 0x9E3779B97F4A7C15ULL);
    acc += (uint32_t)(x & 0xFFFFu) + (uint32_t)((x >> 16) & 0xFFFFu) +
           (uint32_t)((x >> 32) & 0xFFFFu) + (uint32_t)(x >> 48);
  }
  int32_t centred = (int32_t)(2u * acc) - 786420;
  return __int2float_rn(centred) * (1.0f / 131072.0f);
}

__device__ __forceinline__ uint16_t dev_bf16_rne(float x) {
  uint32_t u = __float_as_uint(x);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

__device__ __forceinline__ float dev_bf16_to_f32(uint16_t h) {
  return __uint_as_float(((uint32_t)h) << 16);
}

__global__ void fill_bf16_kernel(uint16_t* __restrict__ out, int64_t n, uint64_t s0, int64_t offset) {
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    out[i] = dev_bf16_rne(dev_ih12(s0, (uint64_t)(offset + i)));
}

__global__ void add_rows_kernel(uint16_t* __restrict__ x, int64_t row_len, const int64_t* __restrict__ rows,
                                const float* __restrict__ vecs, int64_t n_rows, int64_t vec_stride) {
  int64_t total = n_rows * row_len;
  int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    int64_t r = i / row_len, c = i - r * row_len;
    uint16_t* p = x + rows[r] * row_len + c;
    *p = dev_bf16_rne(dev_bf16_to_f32(*p) + vecs[r * vec_stride + c]);
  }
}

__global__ void add_chunk_offsets_kernel(uint16_t* __restrict__ K, int B, int L, int Hkv, int d, int S,
                                         const float* __restrict__ off) {
  const int Nc = L / S;
  const int64_t total = (int64_t)B * Nc * S * Hkv * d;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    // i enumerates (b, t < Nc*S, g, e) in row-major order of K restricted to complete chunks.
    int64_t e = i % d;
    int64_t g = (i / d) % Hkv;
    int64_t t = (i / ((int64_t)d * Hkv)) % ((int64_t)Nc * S);
    int64_t b = i / ((int64_t)d * Hkv * Nc * S);
    int64_t chunk = t / S;
    uint16_t* p = K + ((b * L + t) * Hkv + g) * d + e;
    float o = off[((b * Nc + chunk) * Hkv + g) * d + e];
    *p = dev_bf16_rne(dev_bf16_to_f32(*p) + o);
  }
}

inline int grid_for(int64_t n) {
  int64_t blocks = (n + 255) / 256;
  if (blocks > 152 * 32) blocks = 152 * 32;
  if (blocks < 1) blocks = 1;
  return (int)blocks;
}

inline uint64_t host_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

}  // namespace

extern "C" int synth_dev_fill_bf16(void* out, int64_t n, uint64_t seed, int64_t offset, void* stream) {
  if (n < 0 || (n > 0 && out == nullptr)) return 1;
  if (n == 0) return 0;
  fill_bf16_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream>>>((uint16_t*)out, n, host_mix64(seed), offset);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

extern "C" int synth_dev_add_rows(void* x, int64_t row_len, const int64_t* rows, const float* vecs,
                                  int64_t n_rows, int64_t vec_stride, void* stream) {
  if (row_len <= 0 || n_rows < 0) return 1;
  if (n_rows == 0) return 0;
  if (x == nullptr || rows == nullptr || vecs == nullptr) return 1;
  add_rows_kernel<<<grid_for(n_rows * row_len), 256, 0, (cudaStream_t)stream>>>(
      (uint16_t*)x, row_len, rows, vecs, n_rows, vec_stride);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

extern "C" int synth_dev_add_chunk_offsets(void* K, int B, int L, int Hkv, int d, int S, const float* off,
                                           void* stream) {
  if (B < 0 || L < 0 || Hkv <= 0 || d <= 0 || S <= 0) return 1;
  int64_t total = (int64_t)B * (L / S) * S * Hkv * d;
  if (total == 0) return 0;
  if (K == nullptr || off == nullptr) return 1;
  add_chunk_offsets_kernel<<<grid_for(total), 256, 0, (cudaStream_t)stream>>>((uint16_t*)K, B, L, Hkv, d, S, off);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
