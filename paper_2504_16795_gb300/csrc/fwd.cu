// Hierarchical attention forward (§3.1.1 "Hierarchical Attention", Algorithm 1),
// organised chunk-major instead of token-major.
//
// Algorithm 1 gives every token its own program that loads the k selected K/V
// chunks. Here every (b, g, chunk) is one block: the chunk's 64 x d K and V
// tiles are staged in shared memory once, and the block streams the query
// rows of every selection slot that chose the chunk (from the inverse index),
// 128 rows (= 128/G slots of G heads) per step, through two small dense
// tensor-core products: S = Q K^T (128 x 64 x d) and O' = softmax(S) V
// (128 x d x 64). Each chunk is complete, so its softmax needs no online
// rescaling. The normalised per-slot result O' (bf16) goes to a workspace
// and a second kernel forms O_t = sum_j w_j O'_{t,j} with the chunk weights
// w = softmax_j(s_sel) (the "w/o s.b." variant of §4.1), slots in order j.
#include "common.cuh"

namespace hsa {
namespace {

constexpr int kThreads = 256;
constexpr int kRows = 128;  // query rows per step (8 warps x 16)

template <int D>
struct FwdSmem {
  uint16_t K[kChunk * D];
  uint16_t V[kChunk * D];
  uint16_t Q[2][kRows * D];
};

struct FwdArgs {
  const uint16_t* q;
  const uint16_t* K;
  const uint16_t* V;
  const int32_t* offsets;
  const int32_t* entries;
  uint16_t* Opart;  // [slots, G, D]
  int L, Hq, Hkv, G, log2G, topk, Nc;
  float scale_log2;  // c_att * log2(e)
};

template <int D>
__global__ void __launch_bounds__(kThreads, 2) fwd_chunk_kernel(FwdArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  FwdSmem<D>& sm = *reinterpret_cast<FwdSmem<D>*>(smem_raw);
  constexpr int D8 = D / 8;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int key = blockIdx.x;
  const int c = key % a.Nc, bg = key / a.Nc;
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int off = a.offsets[key];
  const int cnt = a.offsets[key + 1] - off;
  if (cnt <= 0) return;
  const int epi = kRows >> a.log2G;  // slots per step
  const int niter = (cnt + epi - 1) / epi;
  const int slot_div = a.Hkv * a.topk;

  {  // chunk K, V tiles
    const long long row0 = ((long long)b * a.L + (long long)c * kChunk) * a.Hkv + g;
    for (int u = tid; u < kChunk * D8; u += kThreads) {
      const int r = u / D8, ch = u % D8;
      const long long src = (row0 + (long long)r * a.Hkv) * D + ch * 8;
      cp_async16(smem_u32(sm.K) + swz<D>(r, ch * 8), a.K + src);
      cp_async16(smem_u32(sm.V) + swz<D>(r, ch * 8), a.V + src);
    }
  }
  auto load_q = [&](int it, int buf) {
    const uint32_t base = smem_u32(sm.Q[buf]);
    for (int u = tid; u < kRows * D8; u += kThreads) {
      const int r = u / D8, ch = u % D8;
      const int e = it * epi + (r >> a.log2G);
      const uint32_t dst = base + swz<D>(r, ch * 8);
      if (e < cnt) {
        const int p = a.entries[off + e];
        const int t = (p / slot_div) % a.L;
        const long long src = (((long long)b * a.L + t) * a.Hq + (long long)g * a.G + (r & (a.G - 1))) * D + ch * 8;
        cp_async16(dst, a.q + src);
      } else {
        asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(dst), "r"(0));
      }
    }
  };
  load_q(0, 0);
  cp_async_commit();

  const uint32_t kb = smem_u32(sm.K), vb = smem_u32(sm.V);
  for (int it = 0; it < niter; ++it) {
    const int buf = it & 1;
    if (it + 1 < niter) load_q(it + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const uint32_t qb = smem_u32(sm.Q[buf]);
    const int r0 = warp * 16;

    // S = Q K^T : 16 rows x 64 keys per warp
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kd = 0; kd < D / 16; ++kd) {
      uint32_t af[4];
      ldsm_x4(af, qb + swz<D>(r0 + (lane & 7) + 8 * ((lane >> 3) & 1), 16 * kd + 8 * (lane >> 4)));
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bf[4];
        ldsm_x4(bf, kb + swz<D>(16 * np + (lane & 7) + 8 * (lane >> 4), 16 * kd + 8 * ((lane >> 3) & 1)));
        mma_bf16(s[2 * np], af, bf[0], bf[1]);
        mma_bf16(s[2 * np + 1], af, bf[2], bf[3]);
      }
    }
    // softmax over the chunk's 64 keys (rows lane/4 and lane/4 + 8)
    float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      s[i][0] *= a.scale_log2;
      s[i][1] *= a.scale_log2;
      s[i][2] *= a.scale_log2;
      s[i][3] *= a.scale_log2;
      m0 = fmaxf(m0, fmaxf(s[i][0], s[i][1]));
      m1 = fmaxf(m1, fmaxf(s[i][2], s[i][3]));
    }
    m0 = fmaxf(m0, __shfl_xor_sync(0xFFFFFFFFu, m0, 1));
    m0 = fmaxf(m0, __shfl_xor_sync(0xFFFFFFFFu, m0, 2));
    m1 = fmaxf(m1, __shfl_xor_sync(0xFFFFFFFFu, m1, 1));
    m1 = fmaxf(m1, __shfl_xor_sync(0xFFFFFFFFu, m1, 2));
    float z0 = 0.f, z1 = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      s[i][0] = exp2f(s[i][0] - m0);
      s[i][1] = exp2f(s[i][1] - m0);
      s[i][2] = exp2f(s[i][2] - m1);
      s[i][3] = exp2f(s[i][3] - m1);
      z0 += s[i][0] + s[i][1];
      z1 += s[i][2] + s[i][3];
    }
    z0 += __shfl_xor_sync(0xFFFFFFFFu, z0, 1);
    z0 += __shfl_xor_sync(0xFFFFFFFFu, z0, 2);
    z1 += __shfl_xor_sync(0xFFFFFFFFu, z1, 1);
    z1 += __shfl_xor_sync(0xFFFFFFFFu, z1, 2);
    const float i0 = 1.f / z0, i1 = 1.f / z1;
    uint32_t pf[4][4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      pf[kk][0] = pack_bf16x2(s[2 * kk][0] * i0, s[2 * kk][1] * i0);
      pf[kk][1] = pack_bf16x2(s[2 * kk][2] * i1, s[2 * kk][3] * i1);
      pf[kk][2] = pack_bf16x2(s[2 * kk + 1][0] * i0, s[2 * kk + 1][1] * i0);
      pf[kk][3] = pack_bf16x2(s[2 * kk + 1][2] * i1, s[2 * kk + 1][3] * i1);
    }
    // O' = P V : 16 rows x D
    float o[D / 8][4];
#pragma unroll
    for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int np = 0; np < D / 16; ++np) {
        uint32_t bf[4];
        ldsm_x4_t(bf, vb + swz<D>(16 * kk + (lane & 7) + 8 * ((lane >> 3) & 1), 16 * np + 8 * (lane >> 4)));
        mma_bf16(o[2 * np], pf[kk], bf[0], bf[1]);
        mma_bf16(o[2 * np + 1], pf[kk], bf[2], bf[3]);
      }
    }
    // stage the warp's 16 rows (bf16) over its own, now dead, query rows
    uint16_t* stage = sm.Q[buf];
    const int rr = lane >> 2, cc = 2 * (lane & 3);
#pragma unroll
    for (int nt = 0; nt < D / 8; ++nt) {
      *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(stage) + swz<D>(r0 + rr, 8 * nt + cc)) =
          pack_bf16x2(o[nt][0], o[nt][1]);
      *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(stage) + swz<D>(r0 + rr + 8, 8 * nt + cc)) =
          pack_bf16x2(o[nt][2], o[nt][3]);
    }
    __syncwarp();
    for (int u = lane; u < 16 * D8; u += 32) {
      const int r = u / D8, ch = u % D8;
      const int R = r0 + r;
      const int e = it * epi + (R >> a.log2G);
      if (e < cnt) {
        const int p = a.entries[off + e];
        const uint4 v = *reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(stage) + swz<D>(R, ch * 8));
        *reinterpret_cast<uint4*>(a.Opart + ((long long)p * a.G + (R & (a.G - 1))) * D + ch * 8) = v;
      }
    }
    __syncthreads();
  }
}

// O_t = sum_j w_j O'_{t,j}; w = softmax over the selected scores. One warp per (b, t, g).
template <int D>
__global__ void __launch_bounds__(256) fwd_merge_kernel(const float* __restrict__ s_sel,
                                                        const int32_t* __restrict__ idx,
                                                        const uint16_t* __restrict__ Opart, uint16_t* __restrict__ O,
                                                        float* __restrict__ w, long long n_rows, int Hkv, int G,
                                                        int topk, int Nc) {
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  bool valid = false;
  float s = -INFINITY;
  if (lane < topk) {
    const int c = idx[p0 + lane];
    valid = c >= 0 && c < Nc;
    if (valid) s = s_sel[p0 + lane];
  }
  const float m = warp_max(s);
  const float ex = valid ? expf(s - m) : 0.f;
  const float z = warp_sum(ex);
  const float wj = valid ? ex / z : 0.f;
  if (lane < topk) w[p0 + lane] = wj;
  const int keff = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int GD8 = G * (D / 8);
  const uint4* src = reinterpret_cast<const uint4*>(Opart) + p0 * GD8;
  uint4* dst = reinterpret_cast<uint4*>(O) + row * GD8;  // heads of group g are contiguous in O
  // every lane runs every iteration (the weight broadcast needs the full warp);
  // lanes past the row's last 16-byte chunk only skip the memory accesses
  for (int base = 0; base < GD8; base += 32) {
    const int ch = base + lane;
    const bool active = ch < GD8;
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    for (int j = 0; j < keff; ++j) {
      const float wb = __shfl_sync(0xFFFFFFFFu, wj, j);
      if (!active) continue;
      const uint4 v = src[(long long)j * GD8 + ch];
      acc[0] += wb * bf16_lo(v.x);
      acc[1] += wb * bf16_hi(v.x);
      acc[2] += wb * bf16_lo(v.y);
      acc[3] += wb * bf16_hi(v.y);
      acc[4] += wb * bf16_lo(v.z);
      acc[5] += wb * bf16_hi(v.z);
      acc[6] += wb * bf16_lo(v.w);
      acc[7] += wb * bf16_hi(v.w);
    }
    if (!active) continue;
    uint4 out;
    out.x = pack_bf16x2(acc[0], acc[1]);
    out.y = pack_bf16x2(acc[2], acc[3]);
    out.z = pack_bf16x2(acc[4], acc[5]);
    out.w = pack_bf16x2(acc[6], acc[7]);
    dst[ch] = out;
  }
}

template <int D>
cudaError_t run(const Dims& Dm, const void* q, const void* K, const void* V, const int32_t* idx, const float* s_sel,
                const int32_t* offsets, const int32_t* entries, void* O, float* w, void* ws, cudaStream_t st) {
  const long long keys = Dm.keys();
  uint16_t* Opart = (uint16_t*)ws;
  if (keys > 0) {
    FwdArgs a;
    a.q = (const uint16_t*)q;
    a.K = (const uint16_t*)K;
    a.V = (const uint16_t*)V;
    a.offsets = offsets;
    a.entries = entries;
    a.Opart = Opart;
    a.L = Dm.L;
    a.Hq = Dm.Hq;
    a.Hkv = Dm.Hkv;
    a.G = Dm.G;
    a.log2G = __builtin_ctz((unsigned)Dm.G);
    a.topk = Dm.topk;
    a.Nc = Dm.Nc;
    a.scale_log2 = Dm.scale_attn * 1.4426950408889634f;
    const size_t smem = sizeof(FwdSmem<D>);
    cudaError_t e = cudaFuncSetAttribute(fwd_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    fwd_chunk_kernel<D><<<(unsigned)keys, kThreads, smem, st>>>(a);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  fwd_merge_kernel<D><<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(s_sel, idx, Opart, (uint16_t*)O, w, rows, Dm.Hkv,
                                                                  Dm.G, Dm.topk, Dm.Nc);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

size_t forward_workspace(const Dims& D) { return (size_t)D.slots() * D.G * D.d * sizeof(uint16_t); }

cudaError_t launch_forward(const Dims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                           const float* s_sel, const int32_t* offsets, const int32_t* entries, void* O, float* w,
                           void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, q, K, V, idx, s_sel, offsets, entries, O, w, ws, st)
                   : run<128>(D, q, K, V, idx, s_sel, offsets, entries, O, w, ws, st);
}

}  // namespace hsa
