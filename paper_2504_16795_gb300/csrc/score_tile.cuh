// Exact fp32 score tile shared by selection and decode: 64 query rows x 64
// chunk summaries, 256 threads, each thread 4 rows x 4 chunks. Every score is
// the fused multiply-add chain over the head dimension in order, starting
// from 0, so its value does not depend on the tiling.
#pragma once
#include "common.cuh"

namespace hsa {

constexpr int kScoreRows = 64;
constexpr int kScoreCols = 64;

// qs: [64][D + 4] fp32 rows (query), kb: [64][D + 4] fp32 rows (chunk summaries).
// Thread (ty = tid / 16, tx = tid % 16) owns rows ty*4 + i and chunks tx + 16*j.
template <int D>
__device__ __forceinline__ void score_tile(const float (*qs)[D + 4], const float (*kb)[D + 4], int ty, int tx,
                                           float (&acc)[4][4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
#pragma unroll 2
  for (int e = 0; e < D; e += 4) {
    float4 qv[4], kv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) qv[i] = *reinterpret_cast<const float4*>(&qs[ty * 4 + i][e]);
#pragma unroll
    for (int j = 0; j < 4; ++j) kv[j] = *reinterpret_cast<const float4*>(&kb[tx + 16 * j][e]);
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        acc[i][j] = fmaf(qv[i].x, kv[j].x, acc[i][j]);
        acc[i][j] = fmaf(qv[i].y, kv[j].y, acc[i][j]);
        acc[i][j] = fmaf(qv[i].z, kv[j].z, acc[i][j]);
        acc[i][j] = fmaf(qv[i].w, kv[j].w, acc[i][j]);
      }
  }
}

}  // namespace hsa
