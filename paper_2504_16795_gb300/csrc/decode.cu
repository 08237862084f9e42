// Decode against a resident memory (§3.2 "Inference"): every step scans the
// chunk summaries of the whole memory, keeps the k best chunks per query and
// group, then fetches only those k chunks for token-level attention.
//
//   1. q̂ per (query, group) in fp32, head order.
//   2. scan: blocks stride over tiles of 64 summaries; each scores 64 queries x
//      64 chunks exactly (the same fp32 definition as the prefill selection)
//      and keeps running per-query top-k lists; each block writes its k
//      candidates per query.
//   3. merge: one warp per (query, group) reduces the candidates to the final
//      top-k, orders it by decreasing chunk index and forms the softmax
//      chunk weights.
//   4. attend: one block per selected (query, group, chunk) gathers the chunk's
//      K and V rows and computes the chunk-local softmax attention of the
//      group's heads.
//   5. O = sum_j w_j O_j.
#include "score_tile.cuh"

namespace hsa {
namespace {

constexpr int kThreads = 256;

inline int scan_blocks_x(const DecodeDims& D) {
  const long long tiles = (D.Nc + kScoreCols - 1) / kScoreCols;
  const long long n_qt = (D.Bq + kScoreRows - 1) / kScoreRows;
  long long want = (2LL * 152) / (D.Hkv * n_qt);
  if (want < 1) want = 1;
  if (want > tiles) want = tiles;
  if (want < 1) want = 1;
  return (int)want;
}

template <int D>
struct ScanSmem {
  float qs[kScoreRows][D + 4];
  float kb[kScoreCols][D + 4];
  float sc[kScoreRows][kScoreCols + 1];
};

template <int D>
__global__ void dec_qhat_kernel(const uint16_t* __restrict__ q, float* __restrict__ qhat, int Hq, int Hkv, int G) {
  const int bg = blockIdx.x;  // b * Hkv + g
  const int b = bg / Hkv, g = bg % Hkv;
  for (int e = threadIdx.x; e < D; e += blockDim.x) {
    float acc = 0.f;
    for (int hh = 0; hh < G; ++hh)
      acc = acc + bf16_bits_to_f32(q[((long long)b * Hq + (long long)g * G + hh) * D + e]);
    qhat[(long long)bg * D + e] = acc;
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    dec_scan_kernel(const float* __restrict__ qhat, const float* __restrict__ kbar32,
                    unsigned long long* __restrict__ cand, int Bq, int Hkv, long long Nc, int topk, float scale_sel) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  ScanSmem<D>& sm = *reinterpret_cast<ScanSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = blockIdx.y, qt = blockIdx.z;
  const int nx = gridDim.x;
  const long long n_tiles = (Nc + kScoreCols - 1) / kScoreCols;
  constexpr int D4 = D / 4;
  for (int u = tid; u < kScoreRows * D4; u += kThreads) {
    const int r = u / D4, e4 = u % D4;
    const int b = qt * kScoreRows + r;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (b < Bq) v = *reinterpret_cast<const float4*>(qhat + ((long long)b * Hkv + g) * D + e4 * 4);
    *reinterpret_cast<float4*>(&sm.qs[r][e4 * 4]) = v;
  }
  unsigned long long lst[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) lst[i] = 0ull;
  const int ty = tid >> 4, tx = tid & 15;
  for (long long tile = blockIdx.x; tile < n_tiles; tile += nx) {
    const long long cb = tile * kScoreCols;
    __syncthreads();
    for (int u = tid; u < kScoreCols * D4; u += kThreads) {
      const int ci = u / D4, e4 = u % D4;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (cb + ci < Nc) v = __ldg(reinterpret_cast<const float4*>(kbar32 + ((cb + ci) * Hkv + g) * D) + e4);
      *reinterpret_cast<float4*>(&sm.kb[ci][e4 * 4]) = v;
    }
    __syncthreads();
    float acc[4][4];
    score_tile<D>(sm.qs, sm.kb, ty, tx, acc);
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) sm.sc[ty * 4 + i][tx + 16 * j] = acc[i][j] * scale_sel;
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = warp * 8 + i;
      const long long c0 = cb + lane, c1 = cb + lane + 32;
      unsigned long long k0 = c0 < Nc ? rank_key(sm.sc[r][lane], (uint32_t)c0) : 0ull;
      unsigned long long k1 = c1 < Nc ? rank_key(sm.sc[r][lane + 32], (uint32_t)c1) : 0ull;
      warp_topk_offer(lst[i], k0, topk, lane);
      warp_topk_offer(lst[i], k1, topk, lane);
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int b = qt * kScoreRows + warp * 8 + i;
    if (b < Bq && lane < topk) cand[(((long long)b * Hkv + g) * nx + blockIdx.x) * topk + lane] = lst[i];
  }
}

// Final top-k per (query, group) and the chunk weights (softmax or
// stick-breaking). One warp each.
__global__ void dec_merge_kernel(const unsigned long long* __restrict__ cand, int32_t* __restrict__ idx,
                                 float* __restrict__ s_sel, float* __restrict__ w, int rows, int nx, int topk,
                                 int stick) {
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  if (row >= rows) return;
  const unsigned long long* src = cand + (long long)row * nx * topk;
  const int n = nx * topk;
  unsigned long long mine = 0ull;
  for (int base = 0; base < n; base += 32) {
    const unsigned long long x = base + lane < n ? src[base + lane] : 0ull;
    warp_topk_offer(mine, x, topk, lane);
  }
  const long long o = (long long)row * topk;
  warp_emit_selection(mine, topk, lane, idx + o, s_sel + o);
  __syncwarp();
  bool valid = false;
  float s = -INFINITY;
  if (lane < topk) {
    valid = idx[o + lane] >= 0;
    if (valid) s = s_sel[o + lane];
  }
  const float wj = warp_chunk_weight(s, valid, stick != 0);
  if (lane < topk) w[o + lane] = wj;
}

template <int D>
struct AttSmem {
  float K[kChunk][D + 1];
  float V[kChunk][D];
  float q[16][D];
  float P[16][kChunk];
};

// Token-level attention of one (query, group) over one selected chunk.
template <int D>
__global__ void __launch_bounds__(kThreads) dec_attend_kernel(const uint16_t* __restrict__ q,
                                                              const uint16_t* __restrict__ Kmem,
                                                              const uint16_t* __restrict__ Vmem,
                                                              const int32_t* __restrict__ idx, float* __restrict__ Opart,
                                                              int Hq, int Hkv, int G, int topk, float scale_attn,
                                                              int softmax1) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  AttSmem<D>& sm = *reinterpret_cast<AttSmem<D>*>(smem_raw);
  auto& Ks = sm.K;
  auto& Vs = sm.V;
  auto& qsm = sm.q;
  auto& P = sm.P;
  const int slot = blockIdx.x;  // ((b * Hkv + g) * topk + j)
  const int bg = slot / topk;
  const int b = bg / Hkv, g = bg % Hkv;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float* out = Opart + (long long)slot * G * D;
  const int c = idx[slot];
  if (c < 0) {
    for (int u = tid; u < G * D; u += kThreads) out[u] = 0.f;
    return;
  }
  // the chunk's rows in 16-byte pieces, every piece of a thread requested before
  // the first is used (the memory may also sit in host memory, read over the
  // CPU-GPU link, where a round trip costs microseconds)
  constexpr int kPieces = kChunk * (D / 8) / kThreads;
  static_assert(kPieces * kThreads == kChunk * (D / 8), "whole pieces per thread");
  uint4 kv[kPieces], vv[kPieces];
#pragma unroll
  for (int i = 0; i < kPieces; ++i) {
    const int u = tid + i * kThreads;
    const long long r = (((long long)c * kChunk + u / (D / 8)) * Hkv + g) * D + (u % (D / 8)) * 8;
    kv[i] = *reinterpret_cast<const uint4*>(Kmem + r);
    vv[i] = *reinterpret_cast<const uint4*>(Vmem + r);
  }
#pragma unroll
  for (int i = 0; i < kPieces; ++i) {
    const int u = tid + i * kThreads;
    const int s = u / (D / 8), e = (u % (D / 8)) * 8;
    const uint32_t kw[4] = {kv[i].x, kv[i].y, kv[i].z, kv[i].w}, vw[4] = {vv[i].x, vv[i].y, vv[i].z, vv[i].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      Ks[s][e + 2 * j] = bf16_lo(kw[j]);
      Ks[s][e + 2 * j + 1] = bf16_hi(kw[j]);
      Vs[s][e + 2 * j] = bf16_lo(vw[j]);
      Vs[s][e + 2 * j + 1] = bf16_hi(vw[j]);
    }
  }
  for (int u = tid; u < G * D; u += kThreads) {
    const int hh = u / D, e = u % D;
    qsm[hh][e] = bf16_bits_to_f32(q[((long long)b * Hq + (long long)g * G + hh) * D + e]);
  }
  __syncthreads();
  for (int u = tid; u < G * kChunk; u += kThreads) {
    const int hh = u / kChunk, s = u % kChunk;
    float acc = 0.f;
    for (int e = 0; e < D; ++e) acc = fmaf(qsm[hh][e], Ks[s][e], acc);
    P[hh][s] = acc * scale_attn;
  }
  __syncthreads();
  for (int hh = warp; hh < G; hh += kThreads / 32) {
    const float x0 = P[hh][lane], x1 = P[hh][lane + 32];
    const float m = warp_max(fmaxf(x0, x1));
    const float e0 = expf(x0 - m), e1 = expf(x1 - m);
    const float z = warp_sum(e0 + e1) + (softmax1 ? expf(-m) : 0.f);  // softmax-off-by-one: the zero logit
    P[hh][lane] = e0 / z;
    P[hh][lane + 32] = e1 / z;
  }
  __syncthreads();
  for (int u = tid; u < G * D; u += kThreads) {
    const int hh = u / D, e = u % D;
    float acc = 0.f;
    for (int s = 0; s < kChunk; ++s) acc = fmaf(P[hh][s], Vs[s][e], acc);
    out[u] = acc;
  }
}

template <int D>
__global__ void dec_out_kernel(const float* __restrict__ Opart, const float* __restrict__ w, uint16_t* __restrict__ O,
                               int G, int topk) {
  const int bg = blockIdx.x;
  for (int u = threadIdx.x; u < G * D; u += blockDim.x) {
    float acc = 0.f;
    for (int j = 0; j < topk; ++j) acc = fmaf(w[(long long)bg * topk + j], Opart[((long long)bg * topk + j) * G * D + u], acc);
    O[(long long)bg * G * D + u] = f32_to_bf16_bits(acc);
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct DecLayout {
  size_t qhat, cand, opart, total;
  int nx;
};

DecLayout dec_layout(const DecodeDims& D) {
  DecLayout lo{};
  lo.nx = scan_blocks_x(D);
  size_t o = 0;
  lo.qhat = o;
  o = align256(o + sizeof(float) * (size_t)D.Bq * D.Hkv * D.d);
  lo.cand = o;
  o = align256(o + sizeof(unsigned long long) * (size_t)D.Bq * D.Hkv * lo.nx * D.topk);
  lo.opart = o;
  o = align256(o + sizeof(float) * (size_t)D.Bq * D.Hkv * D.topk * D.G * D.d);
  lo.total = o;
  return lo;
}

template <int DD>
cudaError_t run(const DecodeDims& D, const void* q, const void* K, const void* V, const float* kbar32, void* O,
                int32_t* idx, float* s_sel, float* w, void* ws, cudaStream_t st) {
  const DecLayout lo = dec_layout(D);
  char* base = (char*)ws;
  float* qhat = (float*)(base + lo.qhat);
  unsigned long long* cand = (unsigned long long*)(base + lo.cand);
  float* opart = (float*)(base + lo.opart);
  const int rows = D.Bq * D.Hkv;
  cudaError_t e;
  dec_qhat_kernel<DD><<<rows, 128, 0, st>>>((const uint16_t*)q, qhat, D.Hq, D.Hkv, D.G);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (D.Nc > 0) {
    const size_t smem = sizeof(ScanSmem<DD>);
    if ((e = cudaFuncSetAttribute(dec_scan_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
        cudaSuccess)
      return e;
    dim3 grid(lo.nx, D.Hkv, (D.Bq + kScoreRows - 1) / kScoreRows);
    dec_scan_kernel<DD><<<grid, kThreads, smem, st>>>(qhat, kbar32, cand, D.Bq, D.Hkv, D.Nc, D.topk, D.scale_sel);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  } else {
    if ((e = cudaMemsetAsync(cand, 0, sizeof(unsigned long long) * (size_t)rows * lo.nx * D.topk, st)) !=
        cudaSuccess)
      return e;
  }
  dec_merge_kernel<<<(rows + 7) / 8, 256, 0, st>>>(cand, idx, s_sel, w, rows, lo.nx, D.topk, D.stick ? 1 : 0);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const size_t att_smem = sizeof(AttSmem<DD>);
  if ((e = cudaFuncSetAttribute(dec_attend_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)att_smem)) !=
      cudaSuccess)
    return e;
  dec_attend_kernel<DD><<<rows * D.topk, kThreads, att_smem, st>>>((const uint16_t*)q, (const uint16_t*)K,
                                                           (const uint16_t*)V, idx, opart, D.Hq, D.Hkv, D.G, D.topk,
                                                           D.scale_attn, D.softmax1 ? 1 : 0);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  dec_out_kernel<DD><<<rows, 256, 0, st>>>(opart, w, (uint16_t*)O, D.G, D.topk);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

size_t decode_workspace(const DecodeDims& D) { return dec_layout(D).total; }

cudaError_t launch_decode_attend(const DecodeDims& D, const void* q, const void* K, const void* V,
                                 const int32_t* idx, const float* w, void* O, float* opart, cudaStream_t st) {
  const int rows = D.Bq * D.Hkv;
  cudaError_t e;
  if (D.d == 64) {
    if ((e = cudaFuncSetAttribute(dec_attend_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)sizeof(AttSmem<64>))) != cudaSuccess)
      return e;
    dec_attend_kernel<64><<<rows * D.topk, kThreads, sizeof(AttSmem<64>), st>>>(
        (const uint16_t*)q, (const uint16_t*)K, (const uint16_t*)V, idx, opart, D.Hq, D.Hkv, D.G, D.topk, D.scale_attn,
        D.softmax1 ? 1 : 0);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    dec_out_kernel<64><<<rows, 256, 0, st>>>(opart, w, (uint16_t*)O, D.G, D.topk);
  } else {
    if ((e = cudaFuncSetAttribute(dec_attend_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)sizeof(AttSmem<128>))) != cudaSuccess)
      return e;
    dec_attend_kernel<128><<<rows * D.topk, kThreads, sizeof(AttSmem<128>), st>>>(
        (const uint16_t*)q, (const uint16_t*)K, (const uint16_t*)V, idx, opart, D.Hq, D.Hkv, D.G, D.topk, D.scale_attn,
        D.softmax1 ? 1 : 0);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    dec_out_kernel<128><<<rows, 256, 0, st>>>(opart, w, (uint16_t*)O, D.G, D.topk);
  }
  note_launches(1);
  return cudaGetLastError();
}

bool memory_device_readable(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return true;
  return a.type == cudaMemoryTypeHost && a.devicePointer == p;
}

cudaError_t launch_decode(const DecodeDims& D, const void* q, const void* K, const void* V, const float* kbar32,
                          void* O, int32_t* idx, float* s_sel, float* w, void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, q, K, V, kbar32, O, idx, s_sel, w, ws, st)
                   : run<128>(D, q, K, V, kbar32, O, idx, s_sel, w, ws, st);
}

}  // namespace hsa
