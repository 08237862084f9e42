// Appending tokens to a decode memory (§3.2 "Inference": the memory grows as
// tokens are decoded; only completed chunks are summarised and selectable, and
// each step scans the summaries and reads k chunks).
//
// One launch writes the new rows and pools every chunk they complete. Thread
// (chunk, g, e8) of a newly completed chunk walks the chunk's S rows in token
// order, taking the rows already in the memory from the memory and the others
// from the new rows (which it also stores, with their V rows), and divides the
// fp32 sum by S: the arithmetic and order of hsa_chunk_pool, so a memory built
// by appends holds summaries bit-identical to pooling the whole memory at once.
// Rows of the trailing incomplete chunk are only copied. The memory may sit in
// page-locked host memory; the new rows and the summaries may not alias it
// except that K_new (V_new) may be the memory's own rows n_tokens.. (a prefill
// that wrote its keys in place): every element is then read and written by one
// thread, so the store rewrites the value just read.
#include "common.cuh"

namespace hsa {
namespace {

__global__ void __launch_bounds__(256) append_kernel(const uint4* K_new, const uint4* V_new, uint4* K_mem, uint4* V_mem,
                                                     float4* __restrict__ kbar32, long long T0, long long n_new,
                                                     long long c_lo, long long n_pool, long long tail0, int row_vec,
                                                     int S) {
  const long long stride = (long long)gridDim.x * blockDim.x;
  const long long pool_items = n_pool * row_vec;
  const long long total = pool_items + (T0 + n_new - tail0) * row_vec;
  for (long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
    if (u < pool_items) {
      const long long e = u % row_vec;  // g * d8 + e8
      const long long c = c_lo + u / row_vec;
      const long long t_first = c * S;
      const int s_new = (int)max(0LL, min((long long)S, T0 - t_first));  // rows before s_new are in the memory
      float acc[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = 0.f;
      auto add = [&](const uint4 v) {
        acc[0] = acc[0] + bf16_lo(v.x);
        acc[1] = acc[1] + bf16_hi(v.x);
        acc[2] = acc[2] + bf16_lo(v.y);
        acc[3] = acc[3] + bf16_hi(v.y);
        acc[4] = acc[4] + bf16_lo(v.z);
        acc[5] = acc[5] + bf16_hi(v.z);
        acc[6] = acc[6] + bf16_lo(v.w);
        acc[7] = acc[7] + bf16_hi(v.w);
      };
      for (int s = 0; s < s_new; ++s) add(K_mem[(t_first + s) * row_vec + e]);
#pragma unroll 8
      for (int s = s_new; s < S; ++s) {
        const long long t = t_first + s;
        const uint4 v = K_new[(t - T0) * row_vec + e];
        const uint4 vv = V_new[(t - T0) * row_vec + e];
        K_mem[t * row_vec + e] = v;
        V_mem[t * row_vec + e] = vv;
        add(v);
      }
      const float fs = (float)S;
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = __fdiv_rn(acc[i], fs);
      kbar32[(c * row_vec + e) * 2] = make_float4(acc[0], acc[1], acc[2], acc[3]);
      kbar32[(c * row_vec + e) * 2 + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    } else {
      const long long v = u - pool_items;
      const long long t = tail0 + v / row_vec, e = v % row_vec;
      K_mem[t * row_vec + e] = K_new[(t - T0) * row_vec + e];
      V_mem[t * row_vec + e] = V_new[(t - T0) * row_vec + e];
    }
  }
}

}  // namespace

cudaError_t launch_memory_append(const DecodeDims& D, long long n_tokens, long long n_new, const void* K_new,
                                 const void* V_new, void* K_mem, void* V_mem, float* kbar32, void* index,
                                 cudaStream_t st) {
  if (n_new <= 0) return cudaSuccess;
  const long long S = D.S;
  const long long c_lo = n_tokens / S;             // the chunk the first new row falls in
  const long long c_hi = (n_tokens + n_new) / S;   // chunks below c_hi are complete afterwards
  const long long n_pool = c_hi > c_lo ? c_hi - c_lo : 0;
  const long long tail0 = c_hi * S > n_tokens ? c_hi * S : n_tokens;  // first row only copied
  const int row_vec = D.Hkv * (D.d / 8);
  const long long total = (n_pool + (n_tokens + n_new - tail0)) * row_vec;
  const int grid = grid_cap((total + 255) / 256, 152LL * 16);
  append_kernel<<<grid, 256, 0, st>>>((const uint4*)K_new, (const uint4*)V_new, (uint4*)K_mem, (uint4*)V_mem,
                                      (float4*)kbar32, n_tokens, n_new, c_lo, n_pool, tail0, row_vec, (int)S);
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || index == nullptr || n_pool == 0) return e;
  return launch_index_rows(D, kbar32, index, c_lo, c_hi, st);
}

}  // namespace hsa
