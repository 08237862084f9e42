// Top-k chunk selection per token and GQA group (§3.1 "Chunk Selection").
//
// One block owns the 64 tokens of one query chunk c for one (b, g): they all
// see exactly the chunks 0..c-1, so the block streams those chunk summaries
// through shared memory in tiles of 64, scores the 64 x 64 tile in registers
// and folds it into per-token running top-k lists held by warps. The
// L x (L/S) score matrix never leaves the chip.
//
// Scores follow one fp32 definition, operation for operation:
//   q̂_e  = ((q_{h0,e} + q_{h1,e}) + ...)            head order
//   dot  = fma(q̂_{d-1}, K̄_{d-1}, ... fma(q̂_0, K̄_0, 0))  dimension order
//   s    = dot * c_sel
// so that the top-k decision is reproducible exactly.
#include "score_tile.cuh"

namespace hsa {
namespace {

constexpr int kTok = 64;      // tokens per block (one chunk)
constexpr int kCt = 64;       // chunk summaries per tile
constexpr int kThreads = 256;

template <int D>
struct SelSmem {
  float qs[kTok][D + 4];
  float kb[kCt][D + 4];
  float sc[kTok][kCt + 1];
};

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    select_kernel(const uint16_t* __restrict__ q, const float* __restrict__ kbar32, int32_t* __restrict__ idx,
                  float* __restrict__ s_sel, int B, int L, int Hq, int Hkv, int G, int topk, int Nc, int n_qt,
                  float scale_sel) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  SelSmem<D>& sm = *reinterpret_cast<SelSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int BH = B * Hkv;
  const int qt = n_qt - 1 - (int)(blockIdx.x / BH);  // heavy (late) query chunks first
  const int bg = blockIdx.x % BH;
  const int b = bg / Hkv, g = bg % Hkv;
  const int t0 = qt * kTok;
  const int nvis = qt < Nc ? qt : Nc;

  // ---- group query q̂ for the 64 tokens (fp32, head order)
  constexpr int D8 = D / 8;
  for (int u = tid; u < kTok * D8; u += kThreads) {
    const int tk = u / D8, e8 = u % D8;
    const int t = t0 + tk;
    float acc[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] = 0.f;
    if (t < L) {
      const uint4* src = reinterpret_cast<const uint4*>(q + (((long long)b * L + t) * Hq + (long long)g * G) * D) + e8;
      for (int hh = 0; hh < G; ++hh) {
        uint4 v = __ldg(src + (long long)hh * D8);
        acc[0] = acc[0] + bf16_lo(v.x);
        acc[1] = acc[1] + bf16_hi(v.x);
        acc[2] = acc[2] + bf16_lo(v.y);
        acc[3] = acc[3] + bf16_hi(v.y);
        acc[4] = acc[4] + bf16_lo(v.z);
        acc[5] = acc[5] + bf16_hi(v.z);
        acc[6] = acc[6] + bf16_lo(v.w);
        acc[7] = acc[7] + bf16_hi(v.w);
      }
    }
    float4* dst = reinterpret_cast<float4*>(&sm.qs[tk][e8 * 8]);
    dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }

  // running lists: warp w owns tokens 8w..8w+7, lane l keeps rank l
  unsigned long long lst[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) lst[i] = 0ull;

  const int ty = tid >> 4, tx = tid & 15;  // 16 x 16 threads, 4 tokens x 4 chunks each
  const float* kb_base = kbar32 + ((long long)b * Nc * Hkv + g) * D;
  for (int cb = 0; cb < nvis; cb += kCt) {
    __syncthreads();  // previous tile fully consumed (and q̂ written on the first pass)
    constexpr int D4 = D / 4;
    for (int u = tid; u < kCt * D4; u += kThreads) {
      const int ci = u / D4, e4 = u % D4;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (cb + ci < nvis) v = __ldg(reinterpret_cast<const float4*>(kb_base + (long long)(cb + ci) * Hkv * D) + e4);
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
      const int tk = warp * 8 + i;
      const int c0 = cb + lane, c1 = cb + lane + 32;
      unsigned long long k0 = c0 < nvis ? rank_key(sm.sc[tk][lane], (uint32_t)c0) : 0ull;
      unsigned long long k1 = c1 < nvis ? rank_key(sm.sc[tk][lane + 32], (uint32_t)c1) : 0ull;
      warp_topk_offer(lst[i], k0, topk, lane);
      warp_topk_offer(lst[i], k1, topk, lane);
    }
  }

#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int t = t0 + warp * 8 + i;
    if (t < L) {
      const long long o = (((long long)b * L + t) * Hkv + g) * topk;
      warp_emit_selection(lst[i], topk, lane, idx + o, s_sel + o);
    }
  }
}

template <int D>
cudaError_t run(const Dims& Dm, const void* q, const float* kbar32, int32_t* idx, float* s_sel, cudaStream_t st) {
  const int n_qt = (Dm.L + kTok - 1) / kTok;
  const long long blocks = (long long)n_qt * Dm.B * Dm.Hkv;
  if (blocks == 0) return cudaSuccess;
  if (blocks > 0x7FFFFFFFLL) return cudaErrorInvalidValue;
  const size_t smem = sizeof(SelSmem<D>);
  cudaError_t e = cudaFuncSetAttribute(select_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  select_kernel<D><<<(unsigned)blocks, kThreads, smem, st>>>((const uint16_t*)q, kbar32, idx, s_sel, Dm.B, Dm.L,
                                                             Dm.Hq, Dm.Hkv, Dm.G, Dm.topk, Dm.Nc, n_qt,
                                                             Dm.scale_sel);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_select(const Dims& D, const void* q, const float* kbar32, int32_t* idx, float* s_sel,
                          cudaStream_t st) {
  return D.d == 64 ? run<64>(D, q, kbar32, idx, s_sel, st) : run<128>(D, q, kbar32, idx, s_sel, st);
}

}  // namespace hsa
