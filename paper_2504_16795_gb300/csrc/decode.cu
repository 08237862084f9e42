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
#include "tc.cuh"

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

// K and V rows stay bf16 in shared memory, each row padded by 16 bytes so that
// the lanes of a warp reading 16 bytes of 32 different rows hit distinct banks.
template <int D>
struct AttSmem {
  static constexpr int kRow = D + 8;  // bf16 elements per staged row
  uint16_t K[kChunk * kRow];
  uint16_t V[kChunk * kRow];
  float q[16][D];
  float P[16][kChunk];
};

// Token-level attention of one (query, group) over one selected chunk. The
// block that finishes last for its (query, group) also forms the output
// O = sum_j w_j O_j, in slot order (a per-row counter, zeroed before the launch,
// tells it that the other partials are written). Each product keeps its fused
// multiply-adds in index order (scores over the head dimension, outputs over the
// chunk's tokens); threads hold several of them at once so that one shared-memory
// read feeds several products.
template <int D>
__global__ void __launch_bounds__(kThreads) dec_attend_kernel(
    const uint16_t* __restrict__ q, const uint16_t* __restrict__ Kmem, const uint16_t* __restrict__ Vmem,
    const int32_t* __restrict__ idx, float* Opart, const float* __restrict__ w, uint16_t* __restrict__ O,
    unsigned* __restrict__ counters, int Hq, int Hkv, int G, int topk, float scale_attn, int softmax1) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  AttSmem<D>& sm = *reinterpret_cast<AttSmem<D>*>(smem_raw);
  constexpr int kRow = AttSmem<D>::kRow, D8 = D / 8;
  auto& qsm = sm.q;
  auto& P = sm.P;
  const int slot = blockIdx.x;  // ((b * Hkv + g) * topk + j)
  const int bg = slot / topk;
  const int b = bg / Hkv, g = bg % Hkv;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float* out = Opart + (long long)slot * G * D;
  tc::griddep_wait();  // the selection (idx, w) and the zeroed counters
  const int c = idx[slot];
  if (c < 0) {
    for (int u = tid; u < G * D; u += kThreads) out[u] = 0.f;
  } else {
  // the chunk's rows in 16-byte pieces, every piece of a thread requested before
  // the first is stored (the memory may also sit in host memory, read over the
  // CPU-GPU link, where a round trip costs microseconds)
  constexpr int kPieces = kChunk * D8 / kThreads;
  static_assert(kPieces * kThreads == kChunk * D8, "whole pieces per thread");
  uint4 kv[kPieces], vv[kPieces];
#pragma unroll
  for (int i = 0; i < kPieces; ++i) {
    const int u = tid + i * kThreads;
    const long long r = (((long long)c * kChunk + u / D8) * Hkv + g) * D + (u % D8) * 8;
    kv[i] = *reinterpret_cast<const uint4*>(Kmem + r);
    vv[i] = *reinterpret_cast<const uint4*>(Vmem + r);
  }
#pragma unroll
  for (int i = 0; i < kPieces; ++i) {
    const int u = tid + i * kThreads;
    const int o = (u / D8) * kRow + (u % D8) * 8;
    *reinterpret_cast<uint4*>(&sm.K[o]) = kv[i];
    *reinterpret_cast<uint4*>(&sm.V[o]) = vv[i];
  }
  for (int u = tid; u < G * D; u += kThreads) {
    const int hh = u / D, e = u % D;
    qsm[hh][e] = bf16_bits_to_f32(q[((long long)b * Hq + (long long)g * G + hh) * D + e]);
  }
  __syncthreads();
  {
    // scores: thread (token s, heads hq, hq + 4, ...): one K read serves its heads
    static_assert(kThreads == 4 * kChunk, "four head groups of one thread per token");
    const int s = tid % kChunk, hq = tid / kChunk;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    const uint16_t* krow = &sm.K[s * kRow];
#pragma unroll 4
    for (int e8 = 0; e8 < D8; ++e8) {
      const uint4 kp = *reinterpret_cast<const uint4*>(krow + e8 * 8);
      const float kf[8] = {bf16_lo(kp.x), bf16_hi(kp.x), bf16_lo(kp.y), bf16_hi(kp.y),
                           bf16_lo(kp.z), bf16_hi(kp.z), bf16_lo(kp.w), bf16_hi(kp.w)};
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int hh = hq + 4 * m;
        if (hh < G) {
          const float4 q0 = *reinterpret_cast<const float4*>(&qsm[hh][e8 * 8]);
          const float4 q1 = *reinterpret_cast<const float4*>(&qsm[hh][e8 * 8 + 4]);
          acc[m] = fmaf(q0.x, kf[0], acc[m]);
          acc[m] = fmaf(q0.y, kf[1], acc[m]);
          acc[m] = fmaf(q0.z, kf[2], acc[m]);
          acc[m] = fmaf(q0.w, kf[3], acc[m]);
          acc[m] = fmaf(q1.x, kf[4], acc[m]);
          acc[m] = fmaf(q1.y, kf[5], acc[m]);
          acc[m] = fmaf(q1.z, kf[6], acc[m]);
          acc[m] = fmaf(q1.w, kf[7], acc[m]);
        }
      }
    }
#pragma unroll
    for (int m = 0; m < 4; ++m)
      if (hq + 4 * m < G) P[hq + 4 * m][s] = acc[m] * scale_attn;
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
  // outputs: thread (8 consecutive dimensions, head): one V read serves 8 products
  for (int u = tid; u < G * D8; u += kThreads) {
    const int hh = u / D8, e8 = u % D8;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int t = 0; t < kChunk; ++t) {
      const uint4 vp = *reinterpret_cast<const uint4*>(&sm.V[t * kRow + e8 * 8]);
      const float p = P[hh][t];
      acc[0] = fmaf(p, bf16_lo(vp.x), acc[0]);
      acc[1] = fmaf(p, bf16_hi(vp.x), acc[1]);
      acc[2] = fmaf(p, bf16_lo(vp.y), acc[2]);
      acc[3] = fmaf(p, bf16_hi(vp.y), acc[3]);
      acc[4] = fmaf(p, bf16_lo(vp.z), acc[4]);
      acc[5] = fmaf(p, bf16_hi(vp.z), acc[5]);
      acc[6] = fmaf(p, bf16_lo(vp.w), acc[6]);
      acc[7] = fmaf(p, bf16_hi(vp.w), acc[7]);
    }
    float4* o4 = reinterpret_cast<float4*>(out + hh * D + e8 * 8);
    o4[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    o4[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
  }
  // the last block of the row sums the partials
  __shared__ int last;
  __threadfence();
  __syncthreads();
  if (tid == 0) last = atomicAdd(&counters[bg], 1u) == (unsigned)(topk - 1);
  __syncthreads();
  if (!last) return;
  __threadfence();
  const float* parts = Opart + (long long)bg * topk * G * D;
  for (int u = tid; u < G * D; u += kThreads) {
    float acc = 0.f;
    for (int j = 0; j < topk; ++j) acc = fmaf(w[(long long)bg * topk + j], __ldcg(parts + (long long)j * G * D + u), acc);
    O[(long long)bg * G * D + u] = f32_to_bf16_bits(acc);
  }
  if (tid == 0) counters[bg] = 0u;
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
  o = align256(o + decode_attend_scratch(D));
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
  return launch_decode_attend(D, q, K, V, idx, w, O, base + lo.opart, st);
}

}  // namespace

size_t decode_workspace(const DecodeDims& D) { return dec_layout(D).total; }

size_t decode_attend_scratch(const DecodeDims& D) {
  const size_t rows = (size_t)D.Bq * D.Hkv;
  return align256(sizeof(float) * rows * D.topk * D.G * D.d) + align256(sizeof(unsigned) * rows);
}

unsigned* decode_attend_counters(const DecodeDims& D, void* scratch) {
  const size_t rows = (size_t)D.Bq * D.Hkv;
  return (unsigned*)((char*)scratch + align256(sizeof(float) * rows * D.topk * D.G * D.d));
}

namespace {
template <int DD>
cudaError_t run_attend(const DecodeDims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                   const float* w, void* O, float* opart, unsigned* counters, cudaStream_t st, bool dependent) {
  const int rows = D.Bq * D.Hkv;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(dec_attend_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)sizeof(AttSmem<DD>))) != cudaSuccess)
    return e;
  const float scale = D.scale_attn;
  const int sm1 = D.softmax1 ? 1 : 0;
  if (dependent)
    e = launch_dependent(dec_attend_kernel<DD>, dim3((unsigned)(rows * D.topk)), dim3(kThreads), sizeof(AttSmem<DD>),
                         st, (const uint16_t*)q, (const uint16_t*)K, (const uint16_t*)V, idx, opart, w, (uint16_t*)O,
                         counters, D.Hq, D.Hkv, D.G, D.topk, scale, sm1);
  else
    dec_attend_kernel<DD><<<rows * D.topk, kThreads, sizeof(AttSmem<DD>), st>>>(
        (const uint16_t*)q, (const uint16_t*)K, (const uint16_t*)V, idx, opart, w, (uint16_t*)O, counters, D.Hq,
        D.Hkv, D.G, D.topk, scale, sm1);
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}
}  // namespace

cudaError_t launch_decode_attend(const DecodeDims& D, const void* q, const void* K, const void* V,
                                 const int32_t* idx, const float* w, void* O, void* scratch, cudaStream_t st,
                                 bool counters_zeroed, bool dependent) {
  const int rows = D.Bq * D.Hkv;
  float* opart = (float*)scratch;
  unsigned* counters = decode_attend_counters(D, scratch);
  if (!counters_zeroed) {
    cudaError_t e = cudaMemsetAsync(counters, 0, sizeof(unsigned) * (size_t)rows, st);
    if (e != cudaSuccess) return e;
  }
  return D.d == 64 ? run_attend<64>(D, q, K, V, idx, w, O, opart, counters, st, dependent)
                   : run_attend<128>(D, q, K, V, idx, w, O, opart, counters, st, dependent);
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
