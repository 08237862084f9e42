// Backward of the hierarchical attention (Algorithms 2 and 3, §3.1.2) plus the
// chunk-weight chain into the selection scores (Appendix A: because w takes
// part in the forward pass, the scores receive gradient).
//
// Per slot (token t, group g, selected chunk I_j) and head h of the group:
//   P      = softmax(c_att q_h K_I^T)             (recomputed; the chunk is complete)
//   dP'    = dO_h V_I^T
//   D_h    = sum_s P_s dP'_s  = dO_h · O'_{h,j}   (Algorithm 2: rowsum(O' ∘ ∇O'))
//   dw_j   = sum_h D_h                              (Algorithm 2: ∇w)
//   ds_j   = w_j (dw_j - Δ_t),  Δ_t = sum_j w_j dw_j = sum_h dO_h · O_h
//   da     = w_j P ∘ (dP' - D_h)                    (Algorithms 2/3: ∇S)
//   dq_h  += c_att da K_I + c_sel ds_j K̄_I
//   dK_I  += c_att da^T q_h,  dV_I += w_j P^T dO_h  (Algorithm 3)
//   dK̄_I  += c_sel ds_j q̂_t ;  dK_{I,s} += dK̄_I / S  (mean pool)
//
// The mean-pool term reaches every row s of the chunk equally, and q̂_t is
// the sum of the slot's G query rows, so adding c_sel ds_j / S to every
// element of the slot's rows of the dS tile that feeds dK = dS^T Q produces
// dK̄_I / S inside the same tensor-core product.
//
// Chunk-major and deterministic: one block per (b, g, chunk) owns that
// chunk's dK/dV rows, walks the chunk's slots (from the inverse index) in
// increasing token order 128 query rows at a time and accumulates dK, dV and
// dK̄ on chip; no floating-point atomics anywhere. Each slot's dq
// contribution goes to a bf16 workspace row and a second kernel sums the k
// slots of each token in slot order (fp32).
#include "common.cuh"

namespace hsa {
namespace {

constexpr int kThreads = 256;
constexpr int kRows = 128;

template <int D>
struct BwdSmem {
  uint16_t K[kChunk * D];
  uint16_t V[kChunk * D];
  uint16_t Q[2][kRows * D];
  uint16_t dO[2][kRows * D];
  uint16_t P[kRows * kChunk];   // w * P, bf16
  uint16_t dS[kRows * kChunk];  // c_att * w * P∘(dP' - D) + c_sel * ds / S, bf16
  float kbar[D];
  float wslot[2][kRows];
  float delta[2][kRows];
  int pslot[2][kRows];
};

struct BwdArgs {
  const uint16_t* q;
  const uint16_t* K;
  const uint16_t* V;
  const uint16_t* dO;
  const float* kbar32;
  const float* w;
  const float* delta;  // [B, L, Hkv]
  const int32_t* offsets;
  const int32_t* entries;
  uint16_t* dqpart;  // [slots, G, D] bf16
  float* dK;
  float* dV;
  int L, Hq, Hkv, G, log2G, topk, Nc;
  float scale_log2, scale_attn, scale_sel;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1) bwd_chunk_kernel(BwdArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  BwdSmem<D>& sm = *reinterpret_cast<BwdSmem<D>*>(smem_raw);
  constexpr int D8 = D / 8;
  constexpr int NH = D / 2;  // head-dim columns owned per warp for dK/dV
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int key = blockIdx.x;
  const int c = key % a.Nc, bg = key / a.Nc;
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int off = a.offsets[key];
  const int cnt = a.offsets[key + 1] - off;
  const int epi = kRows >> a.log2G;
  const int niter = (cnt + epi - 1) / epi;
  const int slot_div = a.Hkv * a.topk;
  const long long row0 = ((long long)b * a.L + (long long)c * kChunk) * a.Hkv + g;

  // warp-owned dK/dV sub-tile: chunk rows sr0..sr0+15, head dims dc0..dc0+NH-1
  const int sr0 = 16 * (warp & 3), dc0 = NH * (warp >> 2);
  float dv[NH / 8][4], dk[NH / 8][4];
#pragma unroll
  for (int i = 0; i < NH / 8; ++i) dv[i][0] = dv[i][1] = dv[i][2] = dv[i][3] = dk[i][0] = dk[i][1] = dk[i][2] =
      dk[i][3] = 0.f;

  if (cnt > 0) {
    for (int u = tid; u < kChunk * D8; u += kThreads) {
      const int r = u / D8, ch = u % D8;
      const long long src = (row0 + (long long)r * a.Hkv) * D + ch * 8;
      cp_async16(smem_u32(sm.K) + swz<D>(r, ch * 8), a.K + src);
      cp_async16(smem_u32(sm.V) + swz<D>(r, ch * 8), a.V + src);
    }
    for (int u = tid; u < D; u += kThreads) sm.kbar[u] = a.kbar32[(((long long)b * a.Nc + c) * a.Hkv + g) * D + u];
  }
  auto load_tile = [&](int it, int buf) {
    const uint32_t qbase = smem_u32(sm.Q[buf]), obase = smem_u32(sm.dO[buf]);
    for (int u = tid; u < kRows * D8; u += kThreads) {
      const int r = u / D8, ch = u % D8;
      const int e = it * epi + (r >> a.log2G);
      const uint32_t o = swz<D>(r, ch * 8);
      if (e < cnt) {
        const int p = a.entries[off + e];
        const int t = (p / slot_div) % a.L;
        const long long src = (((long long)b * a.L + t) * a.Hq + (long long)g * a.G + (r & (a.G - 1))) * D + ch * 8;
        cp_async16(qbase + o, a.q + src);
        cp_async16(obase + o, a.dO + src);
      } else {
        asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(qbase + o), "r"(0));
        asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(obase + o), "r"(0));
      }
    }
    if (tid < epi) {
      const int e = it * epi + tid;
      if (e < cnt) {
        const int p = a.entries[off + e];
        const int t = (p / slot_div) % a.L;
        sm.pslot[buf][tid] = p;
        sm.wslot[buf][tid] = a.w[p];
        sm.delta[buf][tid] = a.delta[((long long)b * a.L + t) * a.Hkv + g];
      } else {
        sm.pslot[buf][tid] = -1;
        sm.wslot[buf][tid] = 0.f;
        sm.delta[buf][tid] = 0.f;
      }
    }
  };
  if (niter > 0) load_tile(0, 0);
  cp_async_commit();

  const uint32_t kb = smem_u32(sm.K), vb = smem_u32(sm.V);
  const uint32_t pb = smem_u32(sm.P), db = smem_u32(sm.dS);
  const int rr = lane >> 2, cc = 2 * (lane & 3);
  for (int it = 0; it < niter; ++it) {
    const int buf = it & 1;
    if (it + 1 < niter) load_tile(it + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const uint32_t qb = smem_u32(sm.Q[buf]), ob = smem_u32(sm.dO[buf]);
    const int r0 = warp * 16;

    // S = Q K^T and dP' = dO V^T (16 rows x 64 keys per warp)
    float s[8][4], dp[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) s[i][j] = dp[i][j] = 0.f;
#pragma unroll
    for (int kd = 0; kd < D / 16; ++kd) {
      uint32_t aq[4], ad[4];
      const int ar = r0 + (lane & 7) + 8 * ((lane >> 3) & 1), ac = 16 * kd + 8 * (lane >> 4);
      ldsm_x4(aq, qb + swz<D>(ar, ac));
      ldsm_x4(ad, ob + swz<D>(ar, ac));
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bk[4], bv[4];
        const int br = 16 * np + (lane & 7) + 8 * (lane >> 4), bc = 16 * kd + 8 * ((lane >> 3) & 1);
        ldsm_x4(bk, kb + swz<D>(br, bc));
        ldsm_x4(bv, vb + swz<D>(br, bc));
        mma_bf16(s[2 * np], aq, bk[0], bk[1]);
        mma_bf16(s[2 * np + 1], aq, bk[2], bk[3]);
        mma_bf16(dp[2 * np], ad, bv[0], bv[1]);
        mma_bf16(dp[2 * np + 1], ad, bv[2], bv[3]);
      }
    }
    // P = softmax(c_att S) per row
    float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
#pragma unroll
      for (int j = 0; j < 4; ++j) s[i][j] *= a.scale_log2;
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
    float D0 = 0.f, D1 = 0.f;  // D_h = sum_s P_s dP'_s
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      s[i][0] *= i0;
      s[i][1] *= i0;
      s[i][2] *= i1;
      s[i][3] *= i1;
      D0 += s[i][0] * dp[i][0] + s[i][1] * dp[i][1];
      D1 += s[i][2] * dp[i][2] + s[i][3] * dp[i][3];
    }
    D0 += __shfl_xor_sync(0xFFFFFFFFu, D0, 1);
    D0 += __shfl_xor_sync(0xFFFFFFFFu, D0, 2);
    D1 += __shfl_xor_sync(0xFFFFFFFFu, D1, 1);
    D1 += __shfl_xor_sync(0xFFFFFFFFu, D1, 2);
    // dw per slot: sum of D over the G rows of the slot (rows are grouped in
    // runs of G inside each 8-row half of the warp tile; G = 16 spans both)
    float dw0 = D0, dw1 = D1;
    const int gl = a.G < 8 ? a.G : 8;
    for (int o = 4; o < 4 * gl; o <<= 1) {
      dw0 += __shfl_xor_sync(0xFFFFFFFFu, dw0, o);
      dw1 += __shfl_xor_sync(0xFFFFFFFFu, dw1, o);
    }
    if (a.G == 16) dw0 = dw1 = dw0 + dw1;
    const int R0 = r0 + rr, R1 = R0 + 8;
    const int sl0 = R0 >> a.log2G, sl1 = R1 >> a.log2G;
    const float w0 = sm.wslot[buf][sl0], w1 = sm.wslot[buf][sl1];
    const float ds0 = w0 * (dw0 - sm.delta[buf][sl0]);
    const float ds1 = w1 * (dw1 - sm.delta[buf][sl1]);
    const float pool0 = a.scale_sel * ds0 * (1.f / kChunk), pool1 = a.scale_sel * ds1 * (1.f / kChunk);
    // da (scaled by c_att for the products) and w P, to fragments and shared tiles
    const float ca0 = a.scale_attn * w0, ca1 = a.scale_attn * w1;
    uint32_t dsf[4][4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int nt = 2 * kk + h;
        const float g00 = ca0 * s[nt][0] * (dp[nt][0] - D0), g01 = ca0 * s[nt][1] * (dp[nt][1] - D0);
        const float g10 = ca1 * s[nt][2] * (dp[nt][2] - D1), g11 = ca1 * s[nt][3] * (dp[nt][3] - D1);
        dsf[kk][2 * h] = pack_bf16x2(g00, g01);
        dsf[kk][2 * h + 1] = pack_bf16x2(g10, g11);
        const uint32_t p0 = pack_bf16x2(w0 * s[nt][0], w0 * s[nt][1]);
        const uint32_t p1 = pack_bf16x2(w1 * s[nt][2], w1 * s[nt][3]);
        *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(sm.P) + swz<kChunk>(R0, 8 * nt + cc)) = p0;
        *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(sm.P) + swz<kChunk>(R1, 8 * nt + cc)) = p1;
        *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(sm.dS) + swz<kChunk>(R0, 8 * nt + cc)) =
            pack_bf16x2(g00 + pool0, g01 + pool0);
        *reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(sm.dS) + swz<kChunk>(R1, 8 * nt + cc)) =
            pack_bf16x2(g10 + pool1, g11 + pool1);
      }
    }
    // dsf[kk] is already in A-fragment order {row0 keys 0-7, row1 keys 0-7, row0 keys 8-15, row1 keys 8-15}
    // dq rows: (c_att w da-part) K + c_sel ds K̄, written per slot
    const int e0 = it * epi + sl0, e1 = it * epi + sl1;
    const int p0 = e0 < cnt ? sm.pslot[buf][sl0] : -1;
    const int p1 = e1 < cnt ? sm.pslot[buf][sl1] : -1;
    uint16_t* dq0 = p0 >= 0 ? a.dqpart + ((long long)p0 * a.G + (R0 & (a.G - 1))) * D : nullptr;
    uint16_t* dq1 = p1 >= 0 ? a.dqpart + ((long long)p1 * a.G + (R1 & (a.G - 1))) * D : nullptr;
    const float cs0 = a.scale_sel * ds0, cs1 = a.scale_sel * ds1;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      float acc[D / 16][4];
#pragma unroll
      for (int i = 0; i < D / 16; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint32_t af[4] = {dsf[kk][0], dsf[kk][1], dsf[kk][2], dsf[kk][3]};
#pragma unroll
        for (int np = 0; np < D / 32; ++np) {
          uint32_t bf[4];
          const int col = half * (D / 2) + 16 * np;
          ldsm_x4_t(bf, kb + swz<D>(16 * kk + (lane & 7) + 8 * ((lane >> 3) & 1), col + 8 * (lane >> 4)));
          mma_bf16(acc[2 * np], af, bf[0], bf[1]);
          mma_bf16(acc[2 * np + 1], af, bf[2], bf[3]);
        }
      }
#pragma unroll
      for (int nt = 0; nt < D / 16; ++nt) {
        const int col = half * (D / 2) + 8 * nt + cc;
        if (dq0)
          *reinterpret_cast<uint32_t*>(dq0 + col) =
              pack_bf16x2(acc[nt][0] + cs0 * sm.kbar[col], acc[nt][1] + cs0 * sm.kbar[col + 1]);
        if (dq1)
          *reinterpret_cast<uint32_t*>(dq1 + col) =
              pack_bf16x2(acc[nt][2] + cs1 * sm.kbar[col], acc[nt][3] + cs1 * sm.kbar[col + 1]);
      }
    }
    __syncthreads();  // P, dS tiles and ds complete

    // dV += (wP)^T dO,  dK += (c_att w da)^T Q  over the 128 rows of this step
#pragma unroll
    for (int kr = 0; kr < kRows / 16; ++kr) {
      uint32_t ap[4], as[4];
      const int ar = 16 * kr + (lane & 7) + 8 * (lane >> 4), ac = sr0 + 8 * ((lane >> 3) & 1);
      ldsm_x4_t(ap, pb + swz<kChunk>(ar, ac));
      ldsm_x4_t(as, db + swz<kChunk>(ar, ac));
#pragma unroll
      for (int np = 0; np < NH / 16; ++np) {
        uint32_t bo[4], bq[4];
        const int br = 16 * kr + (lane & 7) + 8 * ((lane >> 3) & 1), bcol = dc0 + 16 * np + 8 * (lane >> 4);
        ldsm_x4_t(bo, ob + swz<D>(br, bcol));
        ldsm_x4_t(bq, qb + swz<D>(br, bcol));
        mma_bf16(dv[2 * np], ap, bo[0], bo[1]);
        mma_bf16(dv[2 * np + 1], ap, bo[2], bo[3]);
        mma_bf16(dk[2 * np], as, bq[0], bq[1]);
        mma_bf16(dk[2 * np + 1], as, bq[2], bq[3]);
      }
    }
    __syncthreads();  // buffers of this step free for the prefetch two steps ahead
  }

  // epilogue: dK (attention and mean-pool terms) and dV of every row of the chunk
#pragma unroll
  for (int nt = 0; nt < NH / 8; ++nt) {
    const int col = dc0 + 8 * nt + cc;
    const long long ra = (row0 + (long long)(sr0 + rr) * a.Hkv) * D + col;
    const long long rb = (row0 + (long long)(sr0 + rr + 8) * a.Hkv) * D + col;
    *reinterpret_cast<float2*>(a.dK + ra) = make_float2(dk[nt][0], dk[nt][1]);
    *reinterpret_cast<float2*>(a.dK + rb) = make_float2(dk[nt][2], dk[nt][3]);
    *reinterpret_cast<float2*>(a.dV + ra) = make_float2(dv[nt][0], dv[nt][1]);
    *reinterpret_cast<float2*>(a.dV + rb) = make_float2(dv[nt][2], dv[nt][3]);
  }
}

// Δ_t = sum over the group's heads of dO · O (one warp per (b, t, g)).
template <int D>
__global__ void __launch_bounds__(256) bwd_delta_kernel(const uint16_t* __restrict__ O, const uint16_t* __restrict__ dO,
                                                        float* __restrict__ delta, long long n_rows, int G) {
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const int GD8 = G * (D / 8);
  const uint4* o = reinterpret_cast<const uint4*>(O) + row * GD8;
  const uint4* d = reinterpret_cast<const uint4*>(dO) + row * GD8;
  float acc = 0.f;
  for (int ch = lane; ch < GD8; ch += 32) {
    const uint4 x = o[ch], y = d[ch];
    acc += bf16_lo(x.x) * bf16_lo(y.x) + bf16_hi(x.x) * bf16_hi(y.x) + bf16_lo(x.y) * bf16_lo(y.y) +
           bf16_hi(x.y) * bf16_hi(y.y) + bf16_lo(x.z) * bf16_lo(y.z) + bf16_hi(x.z) * bf16_hi(y.z) +
           bf16_lo(x.w) * bf16_lo(y.w) + bf16_hi(x.w) * bf16_hi(y.w);
  }
  acc = warp_sum(acc);
  if (lane == 0) delta[row] = acc;
}

// dq_t = sum_j dq'_{t,j} in slot order (one warp per (b, t, g)).
template <int D>
__global__ void __launch_bounds__(256) bwd_dq_merge_kernel(const int32_t* __restrict__ idx,
                                                           const uint16_t* __restrict__ dqpart, float* __restrict__ dq,
                                                           long long n_rows, int G, int topk, int Nc) {
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  bool valid = false;
  if (lane < topk) {
    const int c = idx[p0 + lane];
    valid = c >= 0 && c < Nc;
  }
  const int keff = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int GD8 = G * (D / 8);
  const uint4* src = reinterpret_cast<const uint4*>(dqpart) + p0 * GD8;
  float4* dst = reinterpret_cast<float4*>(dq) + row * GD8 * 2;
  for (int ch = lane; ch < GD8; ch += 32) {
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    for (int j = 0; j < keff; ++j) {
      const uint4 v = src[(long long)j * GD8 + ch];
      acc[0] += bf16_lo(v.x);
      acc[1] += bf16_hi(v.x);
      acc[2] += bf16_lo(v.y);
      acc[3] += bf16_hi(v.y);
      acc[4] += bf16_lo(v.z);
      acc[5] += bf16_hi(v.z);
      acc[6] += bf16_lo(v.w);
      acc[7] += bf16_hi(v.w);
    }
    dst[2 * ch] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[2 * ch + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

// dK = dV = 0 on the rows of a trailing partial chunk.
__global__ void zero_tail_kernel(float* __restrict__ dK, float* __restrict__ dV, int B, int L, int tail0,
                                 long long row_elems) {
  const long long per_b = (long long)(L - tail0) * row_elems;
  const long long total = per_b * B;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
    const long long b = u / per_b, r = u % per_b;
    const long long o = (b * L + tail0) * row_elems + r;
    dK[o] = 0.f;
    dV[o] = 0.f;
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

template <int D>
cudaError_t run(const Dims& Dm, const void* q, const void* K, const void* V, const float* kbar32, const int32_t* idx,
                const float* w, const void* O, const void* dO, const int32_t* offsets, const int32_t* entries,
                float* dq, float* dK, float* dV, void* ws, cudaStream_t st) {
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  uint16_t* dqpart = (uint16_t*)ws;
  float* delta = (float*)((char*)ws + align256((size_t)Dm.slots() * Dm.G * D * sizeof(uint16_t)));
  cudaError_t e;
  bwd_delta_kernel<D><<<(unsigned)((rows + 7) / 8), 256, 0, st>>>((const uint16_t*)O, (const uint16_t*)dO, delta,
                                                                  rows, Dm.G);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const long long keys = Dm.keys();
  if (keys > 0) {
    BwdArgs a;
    a.q = (const uint16_t*)q;
    a.K = (const uint16_t*)K;
    a.V = (const uint16_t*)V;
    a.dO = (const uint16_t*)dO;
    a.kbar32 = kbar32;
    a.w = w;
    a.delta = delta;
    a.offsets = offsets;
    a.entries = entries;
    a.dqpart = dqpart;
    a.dK = dK;
    a.dV = dV;
    a.L = Dm.L;
    a.Hq = Dm.Hq;
    a.Hkv = Dm.Hkv;
    a.G = Dm.G;
    a.log2G = __builtin_ctz((unsigned)Dm.G);
    a.topk = Dm.topk;
    a.Nc = Dm.Nc;
    a.scale_log2 = Dm.scale_attn * 1.4426950408889634f;
    a.scale_attn = Dm.scale_attn;
    a.scale_sel = Dm.scale_sel;
    const size_t smem = sizeof(BwdSmem<D>);
    if ((e = cudaFuncSetAttribute(bwd_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
        cudaSuccess)
      return e;
    bwd_chunk_kernel<D><<<(unsigned)keys, kThreads, smem, st>>>(a);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  bwd_dq_merge_kernel<D><<<(unsigned)((rows + 7) / 8), 256, 0, st>>>(idx, dqpart, dq, rows, Dm.G, Dm.topk, Dm.Nc);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int tail0 = Dm.Nc * kChunk;
  if (tail0 < Dm.L && Dm.B > 0) {
    const long long total = (long long)Dm.B * (Dm.L - tail0) * Dm.Hkv * D;
    zero_tail_kernel<<<grid_cap((total + 255) / 256, 152LL * 8), 256, 0, st>>>(dK, dV, Dm.B, Dm.L, tail0,
                                                                               (long long)Dm.Hkv * D);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

size_t backward_workspace(const Dims& D) {
  return align256((size_t)D.slots() * D.G * D.d * sizeof(uint16_t)) +
         align256((size_t)D.B * D.L * D.Hkv * sizeof(float));
}

cudaError_t launch_backward(const Dims& D, const void* q, const void* K, const void* V, const float* kbar32,
                            const int32_t* idx, const float* w, const void* O, const void* dO,
                            const int32_t* offsets, const int32_t* entries, float* dq, float* dK, float* dV,
                            void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq, dK, dV, ws, st)
                   : run<128>(D, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq, dK, dV, ws, st);
}

}  // namespace hsa
