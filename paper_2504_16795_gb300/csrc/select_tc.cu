// Top-k chunk selection on the tensor cores (§3.1 "Chunk Selection"), with
// the same result as the exact fp32 definition:
//   q̂   = fp32 sum of the group's heads in head order
//   s_i = (fused multiply-add chain of q̂ · K̄_i over d, in order) * c_sel
//   top-k by (s desc, chunk index asc) over the chunks i < t/S.
//
// The score matrix q̂ K̄^T is a dense contraction, so it runs as bf16 tcgen05
// MMAs (q̂ and K̄ rounded to bf16, fp32 accumulation in tensor memory). A
// bf16 score a_i differs from the exact dot product by less than
//   eps_i = 2^-7 * |q̂| * |K̄_i|
// (each bf16 rounding moves a factor by at most 2^-9 of itself, so the
// product sum moves by at most about 2^-8 * sum|q̂_e||K̄_ie| <= 2^-8 |q̂||K̄_i|
// by Cauchy-Schwarz; the fp32 accumulation errors of both sides are far
// below the remaining factor of two). So l_i = a_i - eps_i and
// u_i = a_i + eps_i bracket the exact score: if lambda is the k-th largest
// lower bound, the exact k-th score is at least lambda, and a chunk with
// u_i < lambda is strictly below it (with room to spare for the final
// rounding by c_sel, so no tie can be created).
//
// Per block: 128 consecutive tokens of one (b, g) against tiles of 128 chunk
// summaries. Thread r of the four scan warps owns token row r (tensor-memory
// lane r). It keeps the k largest lower bounds in a sorted register list
// (whose last entry is lambda) and, in a shared-memory buffer, the other
// chunks whose upper bound reaches the current lambda (lambda only rises, so
// a chunk dropped once stays out). A row's first 32 scores go through a
// sorting network at once; later ones are filtered against lambda and only
// the few that pass are inserted one by one.
// At the end the candidates (typically k plus a few) are rescored exactly in
// fp32 and the top k emitted. A row whose buffer overflows is handed to an
// exact warp-per-row pass. The L x (L/S) score matrix never leaves the chip.
#include <algorithm>
#include <cstring>

#include "tc.cuh"

namespace hsa {
namespace {

constexpr int kTok = 128;      // token rows per block (MMA M, tensor-memory lanes)
constexpr int kCt = 128;       // chunk summaries per tile (MMA N)
constexpr int kAcc = 4;        // score accumulators in tensor memory (kCt columns each)
constexpr int kThreads = 192;  // warps 0-3 scan (thread = row), 4 loader, 5 MMA
constexpr int kTmemCols = kAcc * kCt;
constexpr float kEpsRel = 1.f / 128.f;
// Absolute floor of eps_i: covers products the tensor core may flush to zero
// (operands below the normal range), far below any score it could reorder.
constexpr float kEpsAbs = 1e-25f;

template <int KT>
constexpr int window_cap() { return KT <= 8 ? 32 : 48; }

__device__ unsigned g_sel_status;

template <int D, int KT>
struct SelTcSmem {
  static constexpr int kStages = KT <= 8 ? 4 : 3;  // chunk-summary tiles in flight
  static constexpr int kCap = window_cap<KT>();
  static constexpr int kCandMax = KT + kCap;
  static constexpr size_t kTileBytes = (size_t)kStages * kCt * D * 2;
  static constexpr size_t kQ32Bytes = (size_t)kTok * D * 4;
  static constexpr size_t kAfterBytes = kQ32Bytes + (size_t)KT * kTok * 8;
  static constexpr size_t kUnionBytes = kTileBytes > kAfterBytes ? kTileBytes : kAfterBytes;
  // barrier slots
  static constexpr int BAR_A = 0, BAR_Q32 = 1, BAR_FULL = 2, BAR_EMPTY = 2 + kStages,
                       BAR_ACC_FULL = 2 + 2 * kStages, BAR_ACC_EMPTY = BAR_ACC_FULL + kAcc,
                       BAR_KN = BAR_ACC_EMPTY + kAcc, kBars = BAR_KN + kAcc;
  uint16_t A[kTok * D];  // q̂ (bf16) of the block's rows, K-major SW128
  // chunk-summary tiles while scanning; afterwards the rows' fp32 q̂ (128-byte
  // swizzled boxes of 32 columns) and the chosen keys [KT][kTok]
  alignas(1024) unsigned char U[kUnionBytes];
  float wv[kCandMax][kTok];  // window buffer (upper bounds u_i); then the candidates' exact scores
  int wi[kCandMax][kTok];    // their chunk indices
  float knt[kAcc][kCt + 4];  // |K̄_i| of the tile in accumulator ab, then the tile's max
  uint64_t bar[kBars];
  uint32_t tmem_base;
  int abort_flag;
};

struct SelTcArgs {
  const float* qh32;      // [B*Hkv*L, D] fp32 q̂
  const float* qn;        // [B*Hkv*L] |q̂|
  const float* kbar32;    // [B, Nc, Hkv, D]
  const float* kn;        // [B*Hkv, Ncp] |K̄_i|
  const float* ktmax;     // [B*Hkv, Ncp/128, 4] max |K̄_i| over each tile of 128 chunks (in [0])
  int32_t* idx;
  float* s_sel;
  unsigned* nflag;        // rows handed to the exact pass
  int32_t* flags;
  int L, Hkv, Nc, Ncp, topk, n_qt, BH;
  float scale_sel;
};

// Register list sorted by decreasing lower bound l (with the entry's upper
// bound u and chunk index); l is known to beat v[KT-1].
template <int KT>
__device__ __forceinline__ void list_insert(float (&v)[KT], float (&vu)[KT], int (&id)[KT], float l, float u, int c) {
#pragma unroll
  for (int i = KT - 1; i > 0; --i) {
    const bool up = l > v[i - 1];
    const bool here = l > v[i];
    v[i] = up ? v[i - 1] : (here ? l : v[i]);
    vu[i] = up ? vu[i - 1] : (here ? u : vu[i]);
    id[i] = up ? id[i - 1] : (here ? c : id[i]);
  }
  if (l > v[0]) {
    v[0] = l;
    vu[0] = u;
    id[0] = c;
  }
}

// x[c] for a run-time c in [0, 32): a five-level select tree.
__device__ __forceinline__ float pick32(const float (&x)[32], int c) {
  float t[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) t[i] = (c & 1) ? x[2 * i + 1] : x[2 * i];
#pragma unroll
  for (int i = 0; i < 8; ++i) t[i] = (c & 2) ? t[2 * i + 1] : t[2 * i];
#pragma unroll
  for (int i = 0; i < 4; ++i) t[i] = (c & 4) ? t[2 * i + 1] : t[2 * i];
#pragma unroll
  for (int i = 0; i < 2; ++i) t[i] = (c & 8) ? t[2 * i + 1] : t[2 * i];
  return (c & 16) ? t[1] : t[0];
}

// Bitonic sorting network, descending by l, carrying u and c along.
template <int N>
__device__ __forceinline__ void sort_desc(float (&l)[N], float (&u)[N], int (&c)[N]) {
#pragma unroll
  for (int size = 2; size <= N; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1)
#pragma unroll
      for (int i = 0; i < N; ++i) {
        const int j = i ^ stride;
        if (j > i) {
          const bool sw = (i & size) == 0 ? (l[i] < l[j]) : (l[i] > l[j]);
          const float tl = sw ? l[j] : l[i], tu = sw ? u[j] : u[i];
          const int tc = sw ? c[j] : c[i];
          l[j] = sw ? l[i] : l[j];
          u[j] = sw ? u[i] : u[j];
          c[j] = sw ? c[i] : c[j];
          l[i] = tl;
          u[i] = tu;
          c[i] = tc;
        }
      }
}

template <int D, int KT>
__global__ void __launch_bounds__(kThreads, 1)
    sel_tc_kernel(SelTcArgs a, const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_q32) {
  extern __shared__ unsigned char smem_raw[];
  using Smem = SelTcSmem<D, KT>;
  constexpr int kStages = Smem::kStages;
  constexpr int BAR_A = Smem::BAR_A, BAR_Q32 = Smem::BAR_Q32, BAR_FULL = Smem::BAR_FULL, BAR_EMPTY = Smem::BAR_EMPTY,
                BAR_ACC_FULL = Smem::BAR_ACC_FULL, BAR_ACC_EMPTY = Smem::BAR_ACC_EMPTY, BAR_KN = Smem::BAR_KN;
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u));
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int qt = a.n_qt - 1 - (int)(blockIdx.x / a.BH);  // late (heavy) token tiles first
  const int bg = (int)(blockIdx.x % a.BH);
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int t0 = qt * kTok;
  const int t_last = min(t0 + kTok, a.L) - 1;
  const int vis_max = min(t_last / kChunk, a.Nc);
  const int ntiles = (vis_max + kCt - 1) / kCt;
  auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
  volatile int* abort_flag = &sm.abort_flag;
  unsigned* status = &g_sel_status;

  if (tid == 0) {
    tc::mbar_init(bar(BAR_A), 1);
    tc::mbar_init(bar(BAR_Q32), 1);
    for (int i = 0; i < kStages; ++i) {
      tc::mbar_init(bar(BAR_FULL + i), 1);
      tc::mbar_init(bar(BAR_EMPTY + i), 1);
    }
    for (int i = 0; i < kAcc; ++i) {
      tc::mbar_init(bar(BAR_ACC_FULL + i), 1);
      tc::mbar_init(bar(BAR_ACC_EMPTY + i), 128);
      tc::mbar_init(bar(BAR_KN + i), 1);
    }
    sm.abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 5) tc::tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t abase = smem_u32(sm.A), ubase = smem_u32(sm.U);
  constexpr uint32_t kStageBytes = kCt * D * 2;

  if (warp == 4) {
    // ---------------------------------------------------------------- loader
    if (lane == 0 && ntiles > 0) {
      tc::mbar_arrive_expect_tx(bar(BAR_A), kTok * D * 2);
#pragma unroll
      for (int kb = 0; kb < D / 64; ++kb)
        tc::tma_load_2d(abase + kb * kTok * 128, &tmap_q, kb * 64, bg * a.L + t0, bar(BAR_A));
      for (int n = 0; n < ntiles; ++n) {
        const int s = n % kStages;
        if (!tc::mbar_wait(bar(BAR_EMPTY + s), ((n / kStages) & 1) ^ 1, abort_flag, status)) break;
        tc::mbar_arrive_expect_tx(bar(BAR_FULL + s), kStageBytes);
#pragma unroll
        for (int kb = 0; kb < D / 64; ++kb)
          tc::tma_load_2d(ubase + s * kStageBytes + kb * kCt * 128, &tmap_k, kb * 64, bg * a.Nc + n * kCt,
                          bar(BAR_FULL + s));
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---------------------------------------------------------------- MMA issue
    if (lane == 0 && ntiles > 0) {
      constexpr uint32_t idesc = tc::idesc_bf16(kTok, kCt);
      bool ok = tc::mbar_wait(bar(BAR_A), 0, abort_flag, status);
      for (int n = 0; ok && n < ntiles; ++n) {
        const int s = n % kStages, ab = n % kAcc;
        if (!tc::mbar_wait(bar(BAR_FULL + s), (n / kStages) & 1, abort_flag, status)) break;
        if (!tc::mbar_wait(bar(BAR_ACC_EMPTY + ab), ((n / kAcc) & 1) ^ 1, abort_flag, status)) break;
        tc::fence_after_sync();
        // the tile's chunk norms travel with its accumulator (the scan has released both)
        tc::mbar_arrive_expect_tx(bar(BAR_KN + ab), (kCt + 4) * 4);
        tc::bulk_load(smem_u32(sm.knt[ab]), a.kn + (long long)bg * a.Ncp + n * kCt, kCt * 4, bar(BAR_KN + ab));
        tc::bulk_load(smem_u32(&sm.knt[ab][kCt]), a.ktmax + ((long long)bg * (a.Ncp / kCt) + n) * 4, 16,
                      bar(BAR_KN + ab));
        const uint32_t bbase = ubase + s * kStageBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t blk = kk >> 2, w = kk & 3;
          tc::mma_bf16_ss(tmem + ab * kCt, tc::sdesc_sw128(abase + blk * kTok * 128 + w * 32),
                          tc::sdesc_sw128(bbase + blk * kCt * 128 + w * 32), idesc, kk > 0);
        }
        tc::mma_commit(bar(BAR_ACC_FULL + ab));
        tc::mma_commit(bar(BAR_EMPTY + s));
      }
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------------- scan (thread = token row)
    const int r = tid;
    const int t = t0 + r;
    const int vis = t < a.L ? min(t / kChunk, a.Nc) : 0;
    constexpr int kCap = Smem::kCap;
    const long long qrow = (long long)bg * a.L + t;
    const float cq = vis > 0 ? kEpsRel * a.qn[qrow] : 0.f;  // eps_i = cq * |K̄_i| + kEpsAbs
    // slots [KT-k, KT) hold the k largest lower bounds (descending); the slots
    // above hold +inf and never move, so v[KT-1] is always lambda
    float v[KT], vu[KT];
    int id[KT];
#pragma unroll
    for (int i = 0; i < KT; ++i) {
      v[i] = i < KT - a.topk ? INFINITY : -INFINITY;
      vu[i] = v[i];
      id[i] = -1;
    }
    float thr = -INFINITY;  // lambda = v[KT-1]
    bool fresh = true;      // no score of this row seen yet
    int wcnt = 0;
    bool overflow = false;

    auto window_append = [&](float x, int c) {
      if (wcnt == kCap) {  // drop entries that fell below the window
        int j = 0;
        for (int i = 0; i < kCap; ++i) {
          const float wx = sm.wv[i][r];
          if (wx >= thr) {
            sm.wv[j][r] = wx;
            sm.wi[j][r] = sm.wi[i][r];
            ++j;
          }
        }
        wcnt = j;
        if (wcnt == kCap) {
          overflow = true;
          thr = INFINITY;
          return;
        }
      }
      sm.wv[wcnt][r] = x;
      sm.wi[wcnt][r] = c;
      ++wcnt;
    };
    auto consider = [&](float x, int c, float knc) {
      const float e = fmaf(cq, knc, kEpsAbs);
      const float u = x + e;
      if (!(u >= thr)) return;
      const float l = x - e;
      if (l > v[KT - 1]) {
        const float eu = vu[KT - 1];
        const int eid = id[KT - 1];
        list_insert<KT>(v, vu, id, l, u, c);
        thr = v[KT - 1];
        if (eid >= 0 && eu >= thr) window_append(eu, eid);
      } else {
        window_append(u, c);
      }
    };

    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    for (int n = 0; n < ntiles; ++n) {
      const int ab = n % kAcc;
      if (!tc::mbar_wait(bar(BAR_ACC_FULL + ab), (n / kAcc) & 1, abort_flag, status)) break;
      if (!tc::mbar_wait(bar(BAR_KN + ab), (n / kAcc) & 1, abort_flag, status)) break;
      tc::fence_after_sync();
      const float* knt = sm.knt[ab];
      // coarse filter of the tile: a_i + eps_i >= lambda needs a_i >= lambda - cq * max_tile |K̄_i| - kEpsAbs
      const float emax = fmaf(cq, knt[kCt], kEpsAbs);
#pragma unroll 1
      for (int h = 0; h < kCt / 32; ++h) {
        float x[32];
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + ab * kCt + h * 32, x);
        tc::tmem_wait_ld();
        const int c0 = n * kCt + h * 32;
        const int lim = vis - c0;
        if (lim <= 0) continue;
        if (fresh) {
          // first 32 scores of the row: bounds, one sort, the top k to the list
          fresh = false;
          float sl[32], su[32];
          int sc[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const float e = fmaf(cq, knt[h * 32 + c], kEpsAbs);
            const bool ok = c < lim;
            sl[c] = ok ? x[c] - e : -INFINITY;
            su[c] = ok ? x[c] + e : -INFINITY;
            sc[c] = ok ? c0 + c : -1;
          }
          sort_desc<32>(sl, su, sc);
#pragma unroll
          for (int j = 0; j < KT; ++j)
            if (j < a.topk && sc[j] >= 0) list_insert<KT>(v, vu, id, sl[j], su[j], sc[j]);
          thr = v[KT - 1];
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (j >= a.topk && sc[j] >= 0 && su[j] >= thr) window_append(su[j], sc[j]);
          continue;
        }
        uint32_t m = 0;
        const float lo = thr - emax;
#pragma unroll
        for (int c = 0; c < 32; ++c) m |= (c < lim && x[c] >= lo) ? (1u << c) : 0u;
        while (m) {
          const int c = __ffs(m) - 1;
          m &= m - 1;
          const float xc = pick32(x, c);
          if (xc >= thr - emax) consider(xc, c0 + c, knt[h * 32 + c]);
        }
      }
      tc::fence_before_sync();
      tc::mbar_arrive(bar(BAR_ACC_EMPTY + ab));
    }

    // ---------------------------------------------------------------- exact rescoring of the candidates
    // Every MMA has completed once the last accumulator was seen, so the
    // stage buffers are free: the rows' fp32 q̂ lands there in one TMA load.
    if (r == 0 && ntiles > 0 && !*abort_flag) {
      tc::mbar_arrive_expect_tx(bar(BAR_Q32), kTok * D * 4);
#pragma unroll
      for (int cb = 0; cb < D / 32; ++cb)
        tc::tma_load_2d(ubase + cb * kTok * 128, &tmap_q32, cb * 32, bg * a.L + t0, bar(BAR_Q32));
    }
    // candidates: the window entries whose upper bound still reaches lambda, then the list
    int nc = 0;
    for (int j = 0; j < wcnt; ++j)
      if (sm.wv[j][r] >= thr) sm.wi[nc++][r] = sm.wi[j][r];
#pragma unroll
    for (int i = 0; i < KT; ++i)
      if (id[i] >= 0) sm.wi[nc++][r] = id[i];
    const bool q_ok = ntiles == 0 || tc::mbar_wait(bar(BAR_Q32), 0, abort_flag, status);
    if (t < a.L && q_ok && !*abort_flag) {
      const long long p = ((long long)b * a.L + t) * a.Hkv + g;
      int32_t* out_i = a.idx + p * a.topk;
      float* out_s = a.s_sel + p * a.topk;
      const int keff = min(a.topk, vis);
      if (overflow) {
        a.flags[atomicAdd(a.nflag, 1u)] = (int32_t)p;
      } else {
        unsigned long long(*chosen)[kTok] = reinterpret_cast<unsigned long long(*)[kTok]>(sm.U + Smem::kQ32Bytes);
        const unsigned char* qrow_s = sm.U + r * 128;
        const float* kb = a.kbar32 + ((long long)b * a.Nc * a.Hkv + g) * D;
        for (int j0 = 0; j0 < nc; j0 += 4) {
          const float4* k4[4];
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int u = 0; u < 4; ++u)
            k4[u] = reinterpret_cast<const float4*>(kb + (long long)sm.wi[j0 + u < nc ? j0 + u : j0][r] * a.Hkv * D);
#pragma unroll 4
          for (int e4 = 0; e4 < D / 4; ++e4) {
            const float4 qv = *reinterpret_cast<const float4*>(qrow_s + (e4 >> 3) * (kTok * 128) +
                                                               (((e4 & 7) ^ (r & 7)) << 4));
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const float4 kv = __ldg(k4[u] + e4);
              acc[u] = fmaf(qv.x, kv.x, acc[u]);
              acc[u] = fmaf(qv.y, kv.y, acc[u]);
              acc[u] = fmaf(qv.z, kv.z, acc[u]);
              acc[u] = fmaf(qv.w, kv.w, acc[u]);
            }
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (j0 + u < nc) sm.wv[j0 + u][r] = acc[u] * a.scale_sel;
        }
        // the keff largest keys (keys are distinct: they carry the chunk index)
        unsigned long long prev = ~0ull;
        for (int s = 0; s < keff; ++s) {
          unsigned long long best = 0ull;
          for (int j = 0; j < nc; ++j) {
            const unsigned long long kj = rank_key(sm.wv[j][r], (uint32_t)sm.wi[j][r]);
            if (kj < prev && kj > best) best = kj;
          }
          chosen[s][r] = best;
          prev = best;
        }
        // emitted by decreasing chunk index
        for (int s = 0; s < keff; ++s) {
          const unsigned long long ks = chosen[s][r];
          const uint32_t cs = key_chunk(ks);
          int pos = 0;
          for (int u = 0; u < keff; ++u) pos += key_chunk(chosen[u][r]) > cs ? 1 : 0;
          out_i[pos] = (int32_t)cs;
          out_s[pos] = key_score(ks);
        }
        for (int s = keff; s < a.topk; ++s) {
          out_i[s] = -1;
          out_s[s] = -INFINITY;
        }
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 5) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// q̂ of every (b, g, t) row: fp32 head-order sum, its bf16 rounding and its norm.
// Threads D/8 per row, each 8 consecutive elements; rows in [b][g][t] order.
template <int D>
__global__ void __launch_bounds__(256) sel_qhat_kernel(const uint16_t* __restrict__ q, uint16_t* __restrict__ qh16,
                                                       float* __restrict__ qh32, float* __restrict__ qn,
                                                       long long rows, int L, int Hq, int Hkv, int G) {
  constexpr int D8 = D / 8;
  const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long row = u / D8;
  const int e8 = (int)(u % D8);
  const bool valid = row < rows;
  float acc[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) acc[c] = 0.f;
  if (valid) {
    const int t = (int)(row % L);
    const long long bg = row / L;
    const int g = (int)(bg % Hkv);
    const long long b = bg / Hkv;
    const uint4* src = reinterpret_cast<const uint4*>(q + ((b * L + t) * Hq + (long long)g * G) * D) + e8;
    for (int hh = 0; hh < G; ++hh) {
      const uint4 w = __ldg(src + (long long)hh * D8);
      acc[0] = acc[0] + bf16_lo(w.x);
      acc[1] = acc[1] + bf16_hi(w.x);
      acc[2] = acc[2] + bf16_lo(w.y);
      acc[3] = acc[3] + bf16_hi(w.y);
      acc[4] = acc[4] + bf16_lo(w.z);
      acc[5] = acc[5] + bf16_hi(w.z);
      acc[6] = acc[6] + bf16_lo(w.w);
      acc[7] = acc[7] + bf16_hi(w.w);
    }
    float4* d32 = reinterpret_cast<float4*>(qh32 + row * D + e8 * 8);
    d32[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    d32[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    *reinterpret_cast<uint4*>(qh16 + row * D + e8 * 8) =
        make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                   pack_bf16x2(acc[6], acc[7]));
  }
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c) ss = fmaf(acc[c], acc[c], ss);
#pragma unroll
  for (int o = D8 / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  if (valid && e8 == 0) qn[row] = sqrtf(ss);
}

// K̄ in bf16 with rows reordered to [b][g][i], |K̄_i| in fp32 ([b*Hkv+g][Ncp])
// and the largest |K̄_i| of every tile of 128 chunks.
template <int D>
__global__ void __launch_bounds__(256) sel_kbar_kernel(const float* __restrict__ kbar32, uint16_t* __restrict__ kb16,
                                                       float* __restrict__ kn, unsigned* __restrict__ ktmax,
                                                       long long rows, int Nc, int Ncp, int Hkv) {
  constexpr int D8 = D / 8;
  const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long row = u / D8;  // input row (b, i, g)
  const int e8 = (int)(u % D8);
  const bool valid = row < rows;
  float x[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) x[c] = 0.f;
  long long bg = 0;
  int i = 0;
  if (valid) {
    const int g = (int)(row % Hkv);
    const long long bi = row / Hkv;
    i = (int)(bi % Nc);
    const long long b = bi / Nc;
    bg = b * Hkv + g;
    const float4* src = reinterpret_cast<const float4*>(kbar32 + row * D + e8 * 8);
    const float4 lo = __ldg(src), hi = __ldg(src + 1);
    x[0] = lo.x, x[1] = lo.y, x[2] = lo.z, x[3] = lo.w, x[4] = hi.x, x[5] = hi.y, x[6] = hi.z, x[7] = hi.w;
    *reinterpret_cast<uint4*>(kb16 + (bg * Nc + i) * D + e8 * 8) = make_uint4(
        pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]), pack_bf16x2(x[4], x[5]), pack_bf16x2(x[6], x[7]));
  }
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c) ss = fmaf(x[c], x[c], ss);
#pragma unroll
  for (int o = D8 / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  if (valid && e8 == 0) {
    const float nrm = sqrtf(ss);
    kn[bg * Ncp + i] = nrm;
    atomicMax(ktmax + (bg * (Ncp / kCt) + i / kCt) * 4, __float_as_uint(nrm));  // non-negative floats order as integers
  }
}

// Exact pass for the rows whose window buffer overflowed: one warp per row,
// lanes over chunks, the exact fp32 score chain and a warp-held top-k list.
template <int D>
__global__ void __launch_bounds__(256) sel_exact_rows_kernel(const float* __restrict__ qh32,
                                                             const float* __restrict__ kbar32,
                                                             const unsigned* __restrict__ nflag,
                                                             const int32_t* __restrict__ flags,
                                                             int32_t* __restrict__ idx, float* __restrict__ s_sel,
                                                             int L, int Hkv, int Nc, int topk, float scale_sel) {
  __shared__ float qs[8][D];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const unsigned n = *nflag;
  for (unsigned f = blockIdx.x * 8u + wib; f < n; f += gridDim.x * 8u) {
    const long long p = flags[f];
    const int g = (int)(p % Hkv);
    const long long bt = p / Hkv;
    const int t = (int)(bt % L);
    const long long b = bt / L;
    const int vis = min(t / kChunk, Nc);
    const float* qrow = qh32 + ((b * Hkv + g) * L + t) * D;
    __syncwarp();
    for (int e = lane; e < D; e += 32) qs[wib][e] = qrow[e];
    __syncwarp();
    unsigned long long lst = 0ull;
    for (int c0 = 0; c0 < vis; c0 += 32) {
      const int c = c0 + lane;
      unsigned long long key = 0ull;
      if (c < vis) {
        const float4* k4 = reinterpret_cast<const float4*>(kbar32 + ((b * Nc + c) * Hkv + g) * D);
        float acc = 0.f;
#pragma unroll 8
        for (int e4 = 0; e4 < D / 4; ++e4) {
          const float4 kv = __ldg(k4 + e4);
          acc = fmaf(qs[wib][4 * e4], kv.x, acc);
          acc = fmaf(qs[wib][4 * e4 + 1], kv.y, acc);
          acc = fmaf(qs[wib][4 * e4 + 2], kv.z, acc);
          acc = fmaf(qs[wib][4 * e4 + 3], kv.w, acc);
        }
        key = rank_key(acc * scale_sel, (uint32_t)c);
      }
      warp_topk_offer(lst, key, topk, lane);
    }
    warp_emit_selection(lst, topk, lane, idx + p * topk, s_sel + p * topk);
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct SelLayout {
  size_t qh16, qh32, qn, kb16, kn, ktmax, nflag, flags, total;
};

inline int padded_chunks(const Dims& D) { return (D.Nc + kCt - 1) / kCt * kCt; }

// Row counts of the two bf16 operand matrices, padded to one full box (the
// padding rows are never selected: they lie past every row's visible range).
inline size_t q_rows(const Dims& D) { return std::max<size_t>((size_t)D.B * D.Hkv * D.L, kTok); }
inline size_t k_rows(const Dims& D) { return std::max<size_t>((size_t)D.B * D.Hkv * D.Nc, kCt); }

SelLayout sel_layout(const Dims& D) {
  const size_t rows = q_rows(D);
  const size_t krows = k_rows(D);
  SelLayout lo{};
  size_t o = 0;
  lo.qh16 = o;
  o = align256(o + rows * D.d * 2);
  lo.qh32 = o;
  o = align256(o + rows * D.d * 4);
  lo.qn = o;
  o = align256(o + rows * 4);
  lo.kb16 = o;
  o = align256(o + krows * D.d * 2);
  const size_t bh = (size_t)D.B * D.Hkv;
  lo.kn = o;
  o = align256(o + bh * padded_chunks(D) * 4);
  lo.ktmax = o;
  o = align256(o + bh * (padded_chunks(D) / kCt) * 16);
  lo.nflag = o;
  o = align256(o + 4);
  lo.flags = o;
  o = align256(o + (size_t)D.B * D.L * D.Hkv * 4);
  lo.total = o;
  return lo;
}

template <int DD, int KT>
cudaError_t run_tc(const Dims& Dm, const void* q, const float* kbar32, int32_t* idx, float* s_sel, void* ws,
                   cudaStream_t st) {
  const SelLayout lo = sel_layout(Dm);
  char* base = (char*)ws;
  uint16_t* qh16 = (uint16_t*)(base + lo.qh16);
  float* qh32 = (float*)(base + lo.qh32);
  float* qn = (float*)(base + lo.qn);
  uint16_t* kb16 = (uint16_t*)(base + lo.kb16);
  float* kn = (float*)(base + lo.kn);
  unsigned* ktmax = (unsigned*)(base + lo.ktmax);
  unsigned* nflag = (unsigned*)(base + lo.nflag);
  int32_t* flags = (int32_t*)(base + lo.flags);
  const long long rows = (long long)Dm.B * Dm.Hkv * Dm.L;
  const long long krows = (long long)Dm.B * Dm.Nc * Dm.Hkv;
  const int BH = Dm.B * Dm.Hkv;
  cudaError_t e;
  // the tile maxima and the flagged-row counter are adjacent: one clear covers both
  if ((e = cudaMemsetAsync(ktmax, 0, lo.flags - lo.ktmax, st)) != cudaSuccess) return e;
  constexpr int D8 = DD / 8;
  sel_qhat_kernel<DD><<<(unsigned)((rows * D8 + 255) / 256), 256, 0, st>>>((const uint16_t*)q, qh16, qh32, qn, rows,
                                                                          Dm.L, Dm.Hq, Dm.Hkv, Dm.G);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int Ncp = padded_chunks(Dm);
  sel_kbar_kernel<DD><<<(unsigned)((krows * D8 + 255) / 256), 256, 0, st>>>(kbar32, kb16, kn, ktmax, krows, Dm.Nc,
                                                                           Ncp, Dm.Hkv);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;

  CUtensorMap tq, tk, tq32;
  memset(&tq, 0, sizeof(tq));
  memset(&tk, 0, sizeof(tk));
  memset(&tq32, 0, sizeof(tq32));
  if (!tc::make_rows_tmap_f32(&tq32, qh32, (unsigned long long)q_rows(Dm), DD, kTok)) return cudaErrorNotSupported;
  if (!tc::make_rows_tmap(&tq, qh16, (unsigned long long)q_rows(Dm), DD, kTok)) return cudaErrorNotSupported;
  if (!tc::make_rows_tmap(&tk, kb16, (unsigned long long)k_rows(Dm), DD, kCt)) return cudaErrorNotSupported;
  SelTcArgs a;
  a.qh32 = qh32;
  a.qn = qn;
  a.kbar32 = kbar32;
  a.kn = kn;
  a.ktmax = (const float*)ktmax;
  a.idx = idx;
  a.s_sel = s_sel;
  a.nflag = nflag;
  a.flags = flags;
  a.L = Dm.L;
  a.Hkv = Dm.Hkv;
  a.Nc = Dm.Nc;
  a.Ncp = Ncp;
  a.topk = Dm.topk;
  a.n_qt = (Dm.L + kTok - 1) / kTok;
  a.BH = BH;
  a.scale_sel = Dm.scale_sel;
  const size_t smem = sizeof(SelTcSmem<DD, KT>) + 1024;
  if ((e = cudaFuncSetAttribute(sel_tc_kernel<DD, KT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
      cudaSuccess)
    return e;
  const long long blocks = (long long)a.n_qt * BH;
  sel_tc_kernel<DD, KT><<<(unsigned)blocks, kThreads, smem, st>>>(a, tq, tk, tq32);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  sel_exact_rows_kernel<DD><<<2 * 152, 256, 0, st>>>(qh32, kbar32, nflag, flags, idx, s_sel, Dm.L, Dm.Hkv, Dm.Nc,
                                                     Dm.topk, Dm.scale_sel);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

bool select_tc_applies(const Dims& D) { return D.topk <= 16 && D.Nc > 0; }

size_t select_tc_workspace(const Dims& D) { return select_tc_applies(D) ? sel_layout(D).total : 0; }

unsigned select_take_status() {
  unsigned v = 0, zero = 0;
  if (cudaMemcpyFromSymbol(&v, g_sel_status, sizeof(v)) != cudaSuccess) return ~0u;
  cudaMemcpyToSymbol(g_sel_status, &zero, sizeof(zero));
  return v;
}

cudaError_t launch_select_tc(const Dims& D, const void* q, const float* kbar32, int32_t* idx, float* s_sel, void* ws,
                             cudaStream_t st) {
  if (D.d == 64) return D.topk <= 8 ? run_tc<64, 8>(D, q, kbar32, idx, s_sel, ws, st)
                                    : run_tc<64, 16>(D, q, kbar32, idx, s_sel, ws, st);
  return D.topk <= 8 ? run_tc<128, 8>(D, q, kbar32, idx, s_sel, ws, st)
                     : run_tc<128, 16>(D, q, kbar32, idx, s_sel, ws, st);
}

}  // namespace hsa
