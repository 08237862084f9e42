// Top-k chunk selection on the tensor cores (§3.1 "Chunk Selection"), with
// the same result as the exact fp32 definition:
//   q̂   = fp32 sum of the group's heads in head order
//   s_i = (fused multiply-add chain of q̂ · K̄_i over d, in order) * c_sel
//   top-k by (s desc, chunk index asc) over the chunks i < t/S.
//
// The score matrix q̂ K̄^T is a dense contraction, so it runs as bf16 tcgen05
// MMAs (q̂ and K̄ rounded to bf16, fp32 accumulation in tensor memory). A
// bf16 score a_i differs from the exact dot product by less than
//   eps_i = 2^-7 * (9/8) * |q̂| * |K̄_i|.
// Rounding to bf16 (8 significant bits, to nearest) moves a factor by at
// most 2^-8 of itself, so the exact product sum moves by at most
// (2^-7 + 2^-16) * sum|q̂_e||K̄_ie|; the products of bf16 factors are exact in
// fp32, and the fp32 sums of both sides (the tensor core's, allowed up to
// 2^-12 relative, and the reference chain's, about 2^-17) add less than
// 2^-11 of the same sum. Cauchy-Schwarz bounds the sum by |q̂||K̄_i|. So
// l_i = a_i - eps_i and u_i = a_i + eps_i bracket the exact score: if lambda
// is the k-th largest lower bound, the exact k-th score is at least lambda,
// and a chunk with u_i < lambda is strictly below it, with margin enough
// (2^-10 |q̂||K̄_i|) that the final rounding by c_sel cannot create a tie.
//
// Per block: 128 consecutive tokens of one (b, g) against tiles of 64 chunk
// summaries, in one sweep over the tiles plus a second visit of its first few.
// Thread r of the four scan warps owns token row r (tensor-memory lane r).
//   Bound: per group of columns, (largest bf16 score - the tile's largest
//   eps) is at most the group's best lower bound; the k-th largest such term
//   seen so far is a lower bound of lambda (min/max only, no branches), and
//   it only grows. Its final value is lam_lo.
//   Collection: once the bound holds 2k terms, every chunk whose upper bound
//   reaches the bound so far goes to a per-row buffer; the tiles swept before
//   that are visited again against lam_lo. The buffer then holds every chunk
//   whose upper bound reaches lam_lo (plus a few below it, typically k plus a
//   few in all), so it holds every chunk whose lower bound reaches lambda,
//   and lambda is the k-th largest lower bound in the buffer.
// The buffer entries whose upper bound reaches lambda are rescored exactly in
// fp32 and the top k emitted. A full buffer keeps the entries with the
// largest upper bounds and remembers the largest upper bound it dropped; a
// row is certified when that value is below its lambda, and otherwise handed to an
// exact warp-per-row pass. The L x (L/S) score matrix never leaves the chip.
#include <algorithm>
#include <cstring>

#include "tc.cuh"

namespace hsa {
namespace {

constexpr int kTok = 128;      // token rows per block (MMA M, tensor-memory lanes)
constexpr int kCt = 64;        // chunk summaries per tile (MMA N)
constexpr int kThreads = 192;  // warps 0-3 scan (thread = row), 4 loader, 5 MMA
constexpr float kEpsRel = 9.f / 1024.f;  // 2^-7 * 9/8
// Absolute floor of eps_i: covers products the tensor core may flush to zero
// (operands below the normal range), far below any score it could reorder.
constexpr float kEpsAbs = 1e-25f;

// Per list size: pipeline depth, buffer capacity and blocks per SM. With
// K_T = 8 two blocks share an SM (about 106 KB of shared memory and 128
// tensor-memory columns each), so one block's waits overlap the other's work.
template <int KT>
struct SelCfg {
  static constexpr int kStages = KT <= 8 ? 2 : 4;  // chunk-summary tiles in flight
  static constexpr int kAcc = KT <= 8 ? 2 : 4;     // score accumulators in tensor memory (kCt columns each)
  static constexpr int kBuf = KT <= 8 ? 24 : 64;   // candidate entries per row (per thread)
  static constexpr int kExport = 2 * kBuf;          // decode: exported entries per row and range (two buffers)
  static constexpr int kBlocksPerSm = KT <= 8 ? 2 : 1;
  static constexpr int kTmemCols = kAcc * kCt;
};

// Decode blocks (DEC) keep no exact keys: the merge rescores their candidates.
template <int D, int KT, bool DEC = false>
struct SelTcSmem {
  using Cfg = SelCfg<KT>;
  static constexpr int kStages = Cfg::kStages, kAcc = Cfg::kAcc, kBuf = Cfg::kBuf;
  // chunk norms of a tile travel in their own ring, requested by the loader as
  // soon as the scan has released the slot (kKn tiles ahead of the scan)
  static constexpr int kKn = 6;
  // barrier slots
  static constexpr int BAR_A = 0, BAR_Q32 = 1, BAR_FULL = 2, BAR_EMPTY = 2 + kStages,
                       BAR_ACC_FULL = 2 + 2 * kStages, BAR_ACC_EMPTY = BAR_ACC_FULL + kAcc,
                       BAR_KN = BAR_ACC_EMPTY + kAcc, BAR_KNE = BAR_KN + kKn, kBars = BAR_KNE + kKn;
  // A and B are adjacent: once every MMA is done they hold the rows' fp32 q̂ ([e][row], 128 * D floats)
  uint16_t A[kTok * D];                  // q̂ (bf16) of the block's rows, K-major SW128
  uint16_t B[kStages][kCt * D];          // chunk-summary tiles, K-major SW128
  float bl[kBuf][kTok];                  // collected entries: lower bounds, later exact scores
  float bu[kBuf][kTok];                  //   upper bounds
  int bi[kBuf][kTok];                    //   chunk indices
  float knt[kKn][kCt + 4];               // |K̄_i| of a tile, then the tile's max (ring of kKn)
  uint64_t bar[kBars];
  float xch[DEC ? 2 : 1][DEC ? 4 : 1][kTok];  // decode pairs: bound terms swapped after each tile
  float xdrop[DEC ? kTok : 1];                 //   and, at the end, the dropped bound
  int xcnt[DEC ? kTok : 1];                    //   and the entry count
  uint32_t tmem_base;
  int abort_flag;
};
// the rescoring stages 32 fp32 K̄ rows per scan warp in A and B (with K_T = 16, a second buffer
// per warp: two more in A and B, two in bu)
static_assert(sizeof(SelTcSmem<128, 16>::A) + sizeof(SelTcSmem<128, 16>::B) >= 6 * 32 * 128 * 4, "staging");
static_assert(sizeof(SelTcSmem<64, 16>::A) + sizeof(SelTcSmem<64, 16>::B) >= 6 * 32 * 64 * 4, "staging");
static_assert(sizeof(SelTcSmem<128, 16>::bu) >= 2 * 32 * 128 * 4, "staging");
static_assert(sizeof(SelTcSmem<64, 16>::bu) >= 2 * 32 * 64 * 4, "staging");
static_assert(sizeof(SelTcSmem<128, 8>::A) + sizeof(SelTcSmem<128, 8>::B) >= 4 * 32 * 128 * 4, "staging");
static_assert(sizeof(SelTcSmem<64, 8>::A) + sizeof(SelTcSmem<64, 8>::B) >= 4 * 32 * 64 * 4, "staging");
// two blocks per SM with K_T = 8 (228 KB of shared memory, 1 KB reserved per block)
static_assert(2 * (sizeof(SelTcSmem<128, 8>) + 2048) <= 233472, "two prefill blocks per SM");
static_assert(2 * (sizeof(SelTcSmem<128, 8, true>) + 2048) <= 233472, "two decode blocks per SM");

struct SelTcArgs {
  const float* qh32t;     // [B*Hkv, D, Lp] fp32 q̂, transposed (tokens adjacent)
  const float* qn;        // [B*Hkv*L] |q̂|
  const float* kbar32;    // [B, Nc, Hkv, D]
  const float* kn;        // [B*Hkv, Ncp] |K̄_i|
  const float* ktmax;     // [B*Hkv, Ncp/64, 4] max |K̄_i| over each tile of 64 chunks (in [0])
  int32_t* idx;
  float* s_sel;
  unsigned* nflag;        // rows handed to the exact pass
  int32_t* flags;
  int L, Lp, Hkv, Nc, Ncp, topk, n_qt, BH;
  int Nrow;  // rows of the bf16 summaries per (b, g): Nc, or a growing memory's capacity
  float scale_sel;
  // decode against a resident memory: rows are query tokens (all chunks
  // visible); block (split, g, query tile) scans chunks [split*range, +range)
  // and exports, per row, the chunks whose upper bound reaches its own lambda
  int Bq, n_split, range;
  float* cand_l;   // [Hkv, Bq, n_split, kExport] lower bounds
  float* cand_u;   //                          upper bounds
  int32_t* cand_c; //                          chunk indices
  int32_t* cand_n; // [Hkv, Bq, n_split] entry count
  float* cand_d;   // [Hkv, Bq, n_split] largest upper bound the row's buffer dropped (-inf: none)
  float4* cand_s;  // [Hkv, Bq, n_split] (lambda of the range, largest exported lower bound, largest upper bound)
  unsigned* status;  // the call's status word (a bounded wait that gives up sets it)
};

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

// Exact rescoring in shared memory. Each lane of a warp names one chunk (c < 0:
// none); the warp copies the 32 fp32 K̄ rows with coalesced 16-byte cp.async
// (lane j brings float4 j of every row) into `stage`, row l at l * D floats
// with float4 j at slot j ^ (l & 7), so that the lanes' reads of their own
// rows below hit distinct banks.
template <int D>
__device__ __forceinline__ void issue_kbar_rows(uint32_t stage, const float* kb, long long row_stride, int c,
                                                int lane) {
#pragma unroll 4
  for (int l = 0; l < 32; ++l) {
    const int cl = __shfl_sync(0xFFFFFFFFu, c, l);
    if (cl >= 0 && lane < D / 4)
      cp_async16(stage + (uint32_t)(l * D + ((lane ^ (l & 7)) << 2)) * 4u, kb + (long long)cl * row_stride + lane * 4);
  }
  cp_async_commit();
}
template <int D>
__device__ __forceinline__ void stage_kbar_rows(uint32_t stage, const float* kb, long long row_stride, int c,
                                                int lane) {
  issue_kbar_rows<D>(stage, kb, row_stride, c, lane);
  cp_async_wait<0>();
  __syncwarp();
}
// The exact chain of the selection score over the lane's staged row: fused
// multiply-adds in element order from 0 (the caller scales by c_sel).
template <int D>
__device__ __forceinline__ float staged_dot(const float (&q)[D], uint32_t stage, int lane) {
  const uint32_t row = stage + (uint32_t)(lane * D) * 4u;
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < D / 4; ++j) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(row + ((uint32_t)(j ^ (lane & 7)) << 4)));
    acc = fmaf(q[4 * j], v.x, acc);
    acc = fmaf(q[4 * j + 1], v.y, acc);
    acc = fmaf(q[4 * j + 2], v.z, acc);
    acc = fmaf(q[4 * j + 3], v.w, acc);
  }
  return acc;
}

// The same chain for a row whose q̂ lives in lane src's registers: element e
// comes over by shuffle (every lane of the warp takes part).
template <int D>
__device__ __forceinline__ float staged_dot_from(const float (&q)[D], int src, uint32_t stage, int lane) {
  const uint32_t row = stage + (uint32_t)(lane * D) * 4u;
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < D / 4; ++j) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(row + ((uint32_t)(j ^ (lane & 7)) << 4)));
    acc = fmaf(__shfl_sync(0xFFFFFFFFu, q[4 * j], src), v.x, acc);
    acc = fmaf(__shfl_sync(0xFFFFFFFFu, q[4 * j + 1], src), v.y, acc);
    acc = fmaf(__shfl_sync(0xFFFFFFFFu, q[4 * j + 2], src), v.z, acc);
    acc = fmaf(__shfl_sync(0xFFFFFFFFu, q[4 * j + 3], src), v.w, acc);
  }
  return acc;
}

template <int D, int KT, bool DEC>
__global__ void __launch_bounds__(kThreads, SelCfg<KT>::kBlocksPerSm)
    sel_tc_kernel(SelTcArgs a, const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_q32t) {
  extern __shared__ unsigned char smem_raw[];
  using Smem = SelTcSmem<D, KT, DEC>;
  constexpr int kStages = Smem::kStages, kAcc = Smem::kAcc, kKn = Smem::kKn, kTmemCols = SelCfg<KT>::kTmemCols;
  constexpr int BAR_A = Smem::BAR_A, BAR_Q32 = Smem::BAR_Q32, BAR_FULL = Smem::BAR_FULL, BAR_EMPTY = Smem::BAR_EMPTY,
                BAR_ACC_FULL = Smem::BAR_ACC_FULL, BAR_ACC_EMPTY = Smem::BAR_ACC_EMPTY, BAR_KN = Smem::BAR_KN,
                BAR_KNE = Smem::BAR_KNE;
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u));
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int qt, bg, split = 0, c_begin = 0, vis_max;
  if constexpr (DEC) {
    split = (int)blockIdx.x;
    bg = (int)blockIdx.y;  // the memory has one batch row: bg = g
    qt = (int)blockIdx.z;
    c_begin = split * a.range;
    vis_max = max(min(c_begin + a.range, a.Nc) - c_begin, 0);
  } else {
    qt = a.n_qt - 1 - (int)(blockIdx.x / a.BH);  // late (heavy) token tiles first
    bg = (int)(blockIdx.x % a.BH);
    vis_max = min((min(qt * kTok + kTok, a.L) - 1) / kChunk, a.Nc);
  }
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int t0 = qt * kTok;
  const int ntiles = (vis_max + kCt - 1) / kCt;
  // Prefill blocks start their sweep at different tiles, so that concurrent
  // blocks of one (b, g) do not all request the same summary lines at once.
  const int rot = (!DEC && ntiles > 0) ? (int)(blockIdx.x % (unsigned)ntiles) : 0;
  auto tile_of = [&](int it) {
    const int j = it < ntiles ? it : it - ntiles;
    return j + rot < ntiles ? j + rot : j + rot - ntiles;
  };
  auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
  volatile int* abort_flag = &sm.abort_flag;
  unsigned* status = a.status;
  // The lower bound of lambda is the k-th largest of (max over a group of
  // columns - the tile's largest eps): each group holds a chunk whose lower
  // bound is at least its term. Groups of 32 or 8 columns, or single columns
  // for short rows, keep at least 2k terms per row.
  const int vis0 = DEC ? vis_max : min(t0 / kChunk, a.Nc);
  const int gsz = vis0 >= 64 * a.topk ? 32 : (vis0 >= 16 * a.topk ? 8 : 1);
  // One sweep over the tiles collects, past the first t_warm tiles, every
  // chunk whose upper bound reaches the bound built so far; the bound only
  // grows, so this is a superset of the chunks reaching the final one. The
  // t_warm tiles are then visited again against the final bound. Decode
  // starts collecting once the bound holds 2k terms; prefill rows (longer, k
  // up to 16, a buffer per thread) once it holds 8k, which keeps the chunks
  // the early bound admits from crowding their buffers.
  const int t_warm = min(ntiles, ((DEC ? 2 : 8) * a.topk * gsz + kCt - 1) / kCt);
  const int n_iter = ntiles + t_warm;

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
    }
    for (int i = 0; i < kKn; ++i) {
      tc::mbar_init(bar(BAR_KN + i), 1);
      tc::mbar_init(bar(BAR_KNE + i), 128);
    }
    sm.abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 5) tc::tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  tc::griddep_wait();  // the kernel before: the query rows and norms (decode), the bf16 summaries (prefill)
  const uint32_t tmem = sm.tmem_base;
  const uint32_t abase = smem_u32(sm.A), ubase = smem_u32(sm.B);
  constexpr uint32_t kStageBytes = kCt * D * 2;

  if (warp == 4) {
    // ---------------------------------------------------------------- loader
    if (lane == 0 && ntiles > 0) {
      tc::mbar_arrive_expect_tx(bar(BAR_A), kTok * D * 2);
#pragma unroll
      for (int kb = 0; kb < D / 64; ++kb)
        tc::tma_load_2d(abase + kb * kTok * 128, &tmap_q, kb * 64, DEC ? (g * a.n_qt + qt) * kTok : bg * a.L + t0,
                        bar(BAR_A));
      for (int it = 0; it < n_iter; ++it) {
        const int n = tile_of(it);
        const int s = it % kStages, kq = it % kKn;
        // the tile's chunk norms (the scan of tile it - kKn has released the slot)
        if (!tc::mbar_wait(bar(BAR_KNE + kq), ((it / kKn) & 1) ^ 1, abort_flag, status)) break;
        tc::mbar_arrive_expect_tx(bar(BAR_KN + kq), (kCt + 4) * 4);
        tc::bulk_load(smem_u32(sm.knt[kq]), a.kn + (long long)bg * a.Ncp + c_begin + n * kCt, kCt * 4,
                      bar(BAR_KN + kq));
        tc::bulk_load(smem_u32(&sm.knt[kq][kCt]),
                      a.ktmax + ((long long)bg * (a.Ncp / kCt) + c_begin / kCt + n) * 4, 16, bar(BAR_KN + kq));
        if (!tc::mbar_wait(bar(BAR_EMPTY + s), ((it / kStages) & 1) ^ 1, abort_flag, status)) break;
        tc::mbar_arrive_expect_tx(bar(BAR_FULL + s), kStageBytes);
#pragma unroll
        for (int kb = 0; kb < D / 64; ++kb)
          tc::tma_load_2d(ubase + s * kStageBytes + kb * kCt * 128, &tmap_k, kb * 64, bg * a.Nrow + c_begin + n * kCt,
                          bar(BAR_FULL + s));
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---------------------------------------------------------------- MMA issue
    if (lane == 0 && ntiles > 0) {
      constexpr uint32_t idesc = tc::idesc_bf16(kTok, kCt);
      bool ok = tc::mbar_wait(bar(BAR_A), 0, abort_flag, status);
      for (int it = 0; ok && it < n_iter; ++it) {
        const int n = tile_of(it);
        const int s = it % kStages, ab = it % kAcc;
        if (!tc::mbar_wait(bar(BAR_FULL + s), (it / kStages) & 1, abort_flag, status)) break;
        if (!tc::mbar_wait(bar(BAR_ACC_EMPTY + ab), ((it / kAcc) & 1) ^ 1, abort_flag, status)) break;
        tc::fence_after_sync();
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
    // Decode blocks of at most 64 rows scan each row with two threads: the
    // rows were stored twice, so tensor-memory lanes 64-127 repeat lanes 0-63.
    // Thread r takes the lower 32 columns of every tile and thread r + 64 the
    // upper 32; after each tile of the sweep they swap their bound terms
    // through shared memory (named barrier 1), so both hold the row's bound.
    // Each keeps its own buffer, and thread r exports both.
    const bool pair = DEC && a.Bq <= kTok / 2 && gsz >= 8;
    constexpr bool kBothHalves = !DEC && KT > 8;
    const int r = tid;
    const int t = t0 + (pair ? (r & (kTok / 2 - 1)) : r);
    const bool row_ok = DEC ? t < a.Bq : t < a.L;
    const int vis = !row_ok ? 0 : (DEC ? vis_max : min(t / kChunk, a.Nc));
    constexpr int kBuf = Smem::kBuf;
    const long long qrow = DEC ? (long long)t * a.Hkv + g : (long long)bg * a.L + t;
    const float cq = vis > 0 ? kEpsRel * a.qn[qrow] : 0.f;  // eps_i = cq * |K̄_i| + kEpsAbs
    const int h_begin = pair ? r / (kTok / 2) : 0, h_end = pair ? h_begin + 1 : kCt / 32;
    const int nterm = gsz == 8 ? 4 : 1;  // terms per 32 columns (gsz >= 8)
    float bm[KT];  // slots [KT-k, KT): the k largest terms (descending); +inf above
#pragma unroll
    for (int i = 0; i < KT; ++i) bm[i] = i < KT - a.topk ? INFINITY : -INFINITY;
    // branch-free insertion: bm keeps the k largest. Slot i of the new list is
    // the larger of the old slot i and min(old slot i-1, v), so every slot is
    // formed independently (no chain through the list).
    auto push = [&](float v) {
#pragma unroll
      for (int i = KT - 1; i > 0; --i) bm[i] = fmaxf(bm[i], fminf(bm[i - 1], v));
      bm[0] = fmaxf(bm[0], v);
    };
    float lam_lo = -INFINITY;  // the final bound (second visits)
    int cnt = 0;  // collected entries
    float u_drop = -INFINITY;  // largest upper bound a full buffer dropped
    auto scan_barrier = [&]() { asm volatile("barrier.sync 1, 128;" ::: "memory"); };

    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    // The candidates of a half tile: each set bit c of m (a column whose score
    // reaches thr - the tile's largest eps) whose own upper bound reaches thr
    // enters the buffer, as chunk cbase + c.
    auto insert_hits = [&](uint32_t m, const float (&xh)[32], const float* knh, int cbase, float thr) {
      while (m) {
        const int c = __ffs(m) - 1;
        m &= m - 1;
        const float xc = pick32(xh, c);
        const float e = fmaf(cq, knh[c], kEpsAbs);
        if (xc + e >= thr) {
          const float lv = xc - e, uv = xc + e;
          int slot = cnt;
          if (cnt < kBuf) {
            ++cnt;
          } else {  // full: replace the entry with the smallest upper bound, if smaller
            float um = sm.bu[0][r];
            slot = 0;
            for (int j = 1; j < kBuf; ++j) {
              const float uj = sm.bu[j][r];
              if (uj < um) um = uj, slot = j;
            }
            if (uv > um) {
              u_drop = fmaxf(u_drop, um);
            } else {
              u_drop = fmaxf(u_drop, uv);
              slot = -1;
            }
          }
          if (slot >= 0) {
            sm.bl[slot][r] = lv;
            sm.bu[slot][r] = uv;
            sm.bi[slot][r] = cbase + c;
          }
        }
      }
    };
    bool dead = false;  // a wait gave up; in pair mode the warp still meets every barrier
    for (int it = 0; it < n_iter; ++it) {
      const bool sweep = it < ntiles;     // first visit: the bound's terms
      const bool collect = it >= t_warm;  // candidates against the bound so far (final on a second visit)
      const int n = tile_of(it);
      const int ab = it % kAcc, kq = it % kKn;
      if (it == ntiles) lam_lo = bm[KT - 1];
      if (!dead) {
        const bool ok = tc::mbar_wait(bar(BAR_ACC_FULL + ab), (it / kAcc) & 1, abort_flag, status) &&
                        tc::mbar_wait(bar(BAR_KN + kq), (it / kKn) & 1, abort_flag, status);
        dead = !__all_sync(0xFFFFFFFFu, ok);
      }
      if (dead && !pair) break;
      if (!dead) tc::fence_after_sync();
      const float* knt = sm.knt[kq];
      const float emax = dead ? 0.f : fmaf(cq, knt[kCt], kEpsAbs);  // the tile's largest eps_i
      if constexpr (kBothHalves) {
        // Long rows (k > 8: one block per SM, registers to spare): both halves
        // of the tile leave tensor memory together and go through the sweep and
        // the candidate mask side by side, so their dependent chains interleave.
        // Half 0's candidates are tested against a bound that already holds half
        // 1's terms: still at most lam_lo, so the collection stays complete.
        float x0[32], x1[32];
        const int c0 = n * kCt, lim0 = vis - c0, lim1 = lim0 - 32;
        __syncwarp();
        tc::tmem_ld32(tmem + lane_base + ab * kCt, x0);
        tc::tmem_ld32(tmem + lane_base + ab * kCt + 32, x1);
        tc::tmem_wait_ld();
        if (sweep && lim0 > 0) {
          if (lim0 < 2 * 32) {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              x0[c] = c < lim0 ? x0[c] : -INFINITY;
              x1[c] = c < lim1 ? x1[c] : -INFINITY;
            }
          }
          if (gsz == 1) {
#pragma unroll
            for (int c = 0; c < 32; ++c) push(x0[c] - emax);
#pragma unroll
            for (int c = 0; c < 32; ++c) push(x1[c] - emax);
          } else {
            float g0[4], g1[4];  // maxima of the groups of 8 columns
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              g0[j] = fmaxf(fmaxf(fmaxf(x0[8 * j], x0[8 * j + 1]), fmaxf(x0[8 * j + 2], x0[8 * j + 3])),
                            fmaxf(fmaxf(x0[8 * j + 4], x0[8 * j + 5]), fmaxf(x0[8 * j + 6], x0[8 * j + 7])));
              g1[j] = fmaxf(fmaxf(fmaxf(x1[8 * j], x1[8 * j + 1]), fmaxf(x1[8 * j + 2], x1[8 * j + 3])),
                            fmaxf(fmaxf(x1[8 * j + 4], x1[8 * j + 5]), fmaxf(x1[8 * j + 6], x1[8 * j + 7])));
            }
            if (gsz == 8) {
#pragma unroll
              for (int j = 0; j < 4; ++j) push(g0[j] - emax);
#pragma unroll
              for (int j = 0; j < 4; ++j) push(g1[j] - emax);
            } else {
              push(fmaxf(fmaxf(g0[0], g0[1]), fmaxf(g0[2], g0[3])) - emax);
              push(fmaxf(fmaxf(g1[0], g1[1]), fmaxf(g1[2], g1[3])) - emax);
            }
          }
        }
        if (collect && lim0 > 0) {
          const float thr = sweep ? bm[KT - 1] : lam_lo;
          const float lo = thr - emax;
          uint32_t m0 = 0, m1 = 0;
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            m0 |= x0[c] >= lo ? (1u << c) : 0u;
            m1 |= x1[c] >= lo ? (1u << c) : 0u;
          }
          if (lim0 < 32) m0 &= (1u << lim0) - 1u;
          if (lim1 < 32) m1 = lim1 > 0 ? m1 & ((1u << lim1) - 1u) : 0u;
          insert_hits(m0, x0, knt, c_begin + c0, thr);
          insert_hits(m1, x1, knt + 32, c_begin + c0 + 32, thr);
        }
      } else {
#pragma unroll 1
      for (int h = h_begin; h < h_end; ++h) {
        float x[32];
        float tv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};  // this half's terms
        const int c0 = n * kCt + h * 32;
        const int lim = vis - c0;
        if (!dead) {
          __syncwarp();
          tc::tmem_ld32(tmem + lane_base + ab * kCt + h * 32, x);
          tc::tmem_wait_ld();
          if (sweep && lim > 0) {
            if (lim < 32) {
#pragma unroll
              for (int c = 0; c < 32; ++c) x[c] = c < lim ? x[c] : -INFINITY;
            }
            if (gsz == 1) {
#pragma unroll
              for (int c = 0; c < 32; ++c) push(x[c] - emax);
            } else {
              float m8[4];
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                m8[j] = fmaxf(fmaxf(fmaxf(x[8 * j], x[8 * j + 1]), fmaxf(x[8 * j + 2], x[8 * j + 3])),
                              fmaxf(fmaxf(x[8 * j + 4], x[8 * j + 5]), fmaxf(x[8 * j + 6], x[8 * j + 7])));
              }
              if (gsz == 8) {
#pragma unroll
                for (int j = 0; j < 4; ++j) tv[j] = m8[j] - emax;
              } else {
                tv[0] = fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])) - emax;
              }
#pragma unroll
              for (int j = 0; j < 4; ++j)
                if (j < nterm) push(tv[j]);
            }
          }
        }
        if (pair && sweep) {  // the partner's terms of this tile
          float(*xo)[kTok] = sm.xch[it & 1];
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (j < nterm) xo[j][r] = tv[j];
          scan_barrier();
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (j < nterm) push(xo[j][r ^ (kTok / 2)]);
        }
        if (!dead && collect && lim > 0) {
          // every chunk whose upper bound reaches the bound
          const float thr = sweep ? bm[KT - 1] : lam_lo;
          uint32_t m = 0;
          const float lo = thr - emax;
#pragma unroll
          for (int c = 0; c < 32; ++c) m |= x[c] >= lo ? (1u << c) : 0u;
          if (lim < 32) m &= (1u << lim) - 1u;
          insert_hits(m, x, knt + h * 32, c_begin + c0, thr);
        }
      }
      }  // one half at a time
      if (!dead) {
        tc::fence_before_sync();
        tc::mbar_arrive(bar(BAR_ACC_EMPTY + ab));
        tc::mbar_arrive(bar(BAR_KNE + kq));
      }
    }
    if (ntiles == 0) cnt = 0;
    int cnt_p = 0;  // pair mode, thread r < 64: the partner's entries
    if constexpr (DEC) {
      if (pair) {
        sm.xcnt[r] = cnt;
        sm.xdrop[r] = u_drop;
        scan_barrier();
        if (r < kTok / 2) {
          cnt_p = sm.xcnt[r + kTok / 2];
          u_drop = fmaxf(u_drop, sm.xdrop[r + kTok / 2]);
        }
      }
    }
    // lambda of the kept entries: at most the row's true lambda (a subset's k-th largest)
#pragma unroll
    for (int i = 0; i < KT; ++i) bm[i] = i < KT - a.topk ? INFINITY : -INFINITY;
    for (int j = 0; j < cnt; ++j) push(sm.bl[j][r]);
    for (int j = 0; j < cnt_p; ++j) push(sm.bl[j][r + kTok / 2]);
    const float lam_keep = bm[KT - 1];

    if constexpr (DEC) {
      // export the entries whose upper bound reaches this range's lambda, and
      // the largest upper bound the buffer dropped (the merge checks it against
      // the lambda of the whole memory)
      if (row_ok && !*abort_flag && (!pair || r < kTok / 2)) {
        constexpr int kExp = SelCfg<KT>::kExport;  // holds both buffers of a pair
        const long long crow = ((long long)g * a.Bq + t) * a.n_split + split;
        int ne = 0;
        float lmax = -INFINITY, umax = -INFINITY;
        auto take = [&](int col, int n_ent) {
          for (int j = 0; j < n_ent; ++j) {
            const float u = sm.bu[j][col];
            if (u >= lam_keep) {
              const float l = sm.bl[j][col];
              a.cand_l[crow * kExp + ne] = l;
              a.cand_u[crow * kExp + ne] = u;
              a.cand_c[crow * kExp + ne] = sm.bi[j][col];
              lmax = fmaxf(lmax, l);
              umax = fmaxf(umax, u);
              ++ne;
            }
          }
        };
        take(r, cnt);
        take(r + kTok / 2, cnt_p);
        a.cand_n[crow] = ne;
        a.cand_d[crow] = u_drop;
        a.cand_s[crow] = make_float4(lam_keep, lmax, umax, 0.f);
      }
    } else {

    // ---------------------------------------------------------------- exact rescoring of the candidates
    // Every MMA has completed once the last accumulator was seen, so A and B
    // are free: the rows' fp32 q̂ lands there in one TMA box ([e][row]).
    if (r == 0 && ntiles > 0 && !*abort_flag) {
      tc::mbar_arrive_expect_tx(bar(BAR_Q32), kTok * D * 4);
      tc::tma_load_2d(abase, &tmap_q32t, t0, bg * D, bar(BAR_Q32));
    }
    // lambda: the k-th largest lower bound among the kept entries (they
    // include every chunk whose lower bound reaches lam_lo, unless the buffer
    // dropped entries, whose upper bounds must then stay below it); the
    // candidates are the entries whose upper bound reaches it
    const bool overflow = u_drop > -INFINITY && !(u_drop < lam_keep);
    int nc = 0;
    if (!overflow)
      for (int j = 0; j < cnt; ++j)
        if (sm.bu[j][r] >= lam_keep) sm.bi[nc++][r] = sm.bi[j][r];
    const bool q_ok = ntiles == 0 || tc::mbar_wait(bar(BAR_Q32), 0, abort_flag, status);
    const bool live = t < a.L && q_ok && !*abort_flag;
    // the row's fp32 q̂ into registers (element e at qs[e * kTok]; a warp's rows
    // are adjacent words), after which the scan warps reuse A and B as staging
    float qr[D];
    {
      const float* qs = reinterpret_cast<const float*>(sm.A) + r;
#pragma unroll
      for (int e = 0; e < D; ++e) qr[e] = qs[e * kTok];
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    {
      // The warp's candidates, listed row after row, are rescored 32 at a
      // time: lane l takes entry base + l, whatever row it belongs to, and
      // reads that row's q̂ from the owning lane by shuffle.
      const int my_n = (live && !overflow) ? nc : 0;
      int incl = my_n;  // inclusive prefix of the entry counts over the warp's lanes
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
      }
      const int total = __shfl_sync(0xFFFFFFFFu, incl, 31);
      const float* kb = a.kbar32 + ((long long)b * a.Nc * a.Hkv + g) * D;
      const uint32_t stage = abase + (uint32_t)(warp * 32 * D) * 4u;  // 32 rows per warp inside A and B
      // lane l's entry of the round starting at base: its row (owning lane src), index j, chunk c (-1: none)
      auto locate = [&](int base, int& src, int& j, int& c) {
        const int e = base + lane;
        src = 0;  // the owning lane: the number of lanes whose prefix ends at or before e
#pragma unroll
        for (int step = 16; step >= 1; step >>= 1) {
          const int v = __shfl_sync(0xFFFFFFFFu, incl, src + step - 1);
          if (v <= e) src += step;
        }
        j = e - (__shfl_sync(0xFFFFFFFFu, incl, src) - __shfl_sync(0xFFFFFFFFu, my_n, src));
        c = e < total ? sm.bi[j][warp * 32 + src] : -1;
      };
      if constexpr (!DEC && KT > 8) {
        // One block per SM leaves room for a second staging buffer per warp (the
        // rest of A and B for warps 0-1, the freed upper bounds for warps 2-3):
        // the next round's K̄ rows are in flight while this round's chains run.
        const uint32_t stage1 = warp < 2 ? abase + (uint32_t)((4 + warp) * 32 * D) * 4u
                                         : smem_u32(&sm.bu[0][0]) + (uint32_t)((warp - 2) * 32 * D) * 4u;
        int src, j, c;
        locate(0, src, j, c);
        if (total > 0) issue_kbar_rows<D>(stage, kb, (long long)a.Hkv * D, c, lane);
        for (int base = 0, round = 0; base < total; base += 32, ++round) {
          const uint32_t cur = (round & 1) ? stage1 : stage;
          int src_n = 0, j_n = 0, c_n = -1;
          if (base + 32 < total) {
            locate(base + 32, src_n, j_n, c_n);
            issue_kbar_rows<D>((round & 1) ? stage : stage1, kb, (long long)a.Hkv * D, c_n, lane);
            cp_async_wait<1>();
          } else {
            cp_async_wait<0>();
          }
          __syncwarp();
          const float v = staged_dot_from<D>(qr, src, cur, lane);
          if (c >= 0) sm.bl[j][warp * 32 + src] = v * a.scale_sel;
          __syncwarp();  // the buffer is refilled two rounds on
          src = src_n;
          j = j_n;
          c = c_n;
        }
      } else {
        for (int base = 0; base < total; base += 32) {
          int src, j, c;
          locate(base, src, j, c);
          stage_kbar_rows<D>(stage, kb, (long long)a.Hkv * D, c, lane);
          const float v = staged_dot_from<D>(qr, src, stage, lane);
          if (c >= 0) sm.bl[j][warp * 32 + src] = v * a.scale_sel;
          __syncwarp();
        }
      }
    }
    if (live) {
      const long long p = ((long long)b * a.L + t) * a.Hkv + g;
      int32_t* out_i = a.idx + p * a.topk;
      float* out_s = a.s_sel + p * a.topk;
      const int keff = min(a.topk, vis);
      if (overflow) {
        a.flags[atomicAdd(a.nflag, 1u)] = (int32_t)p;
      } else {
        // the KT largest keys, in registers (keys are distinct: they carry the
        // chunk index; 0 never beats a real key)
        unsigned long long top[KT];
#pragma unroll
        for (int i = 0; i < KT; ++i) top[i] = 0ull;
        for (int j = 0; j < nc; ++j) {  // insertion with every slot formed independently
          const unsigned long long v = rank_key(sm.bl[j][r], (uint32_t)sm.bi[j][r]);
#pragma unroll
          for (int i = KT - 1; i > 0; --i) {
            const unsigned long long lo = top[i - 1] < v ? top[i - 1] : v;
            top[i] = top[i] > lo ? top[i] : lo;
          }
          top[0] = top[0] > v ? top[0] : v;
        }
        // the keff best, emitted by decreasing chunk index
#pragma unroll
        for (int s = 0; s < KT; ++s) {
          if (s < keff) {
            const uint32_t cs = key_chunk(top[s]);
            int pos = 0;
#pragma unroll
            for (int u = 0; u < KT; ++u) pos += (u < keff && key_chunk(top[u]) > cs) ? 1 : 0;
            out_i[pos] = (int32_t)cs;
            out_s[pos] = key_score(top[s]);
          }
        }
        for (int s = keff; s < a.topk; ++s) {
          out_i[s] = -1;
          out_s[s] = -INFINITY;
        }
      }
    }
    }  // prefill
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 5) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// q̂ of every (b, g, t) row: the fp32 head-order sum (stored transposed,
// [b*Hkv+g][e][t], so that the rows a warp rescores are adjacent in memory),
// its bf16 rounding ([b*Hkv+g][t][e], the MMA operand) and its norm. One
// block per 32 consecutive tokens of one (b, g).
template <int D>
__global__ void __launch_bounds__(256) sel_qhat_kernel(const uint16_t* __restrict__ q, uint16_t* __restrict__ qh16,
                                                       float* __restrict__ qh32t, float* __restrict__ qn, int L,
                                                       int Lp, int Hq, int Hkv, int G) {
  griddep_wait();
  __shared__ float qs[32][D + 1];
  constexpr int D8 = D / 8;
  const int bg = blockIdx.y;
  const int t0 = blockIdx.x * 32;
  const int b = bg / Hkv, g = bg % Hkv;
  // the D8 threads of a row are adjacent lanes of one warp (256 and 32 are multiples of D8)
  for (int u = threadIdx.x; u < 32 * D8; u += 256) {
    const int rr = u / D8, e8 = u % D8;
    const int t = t0 + rr;
    float acc[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] = 0.f;
    if (t < L) {
      const uint4* src = reinterpret_cast<const uint4*>(q + (((long long)b * L + t) * Hq + (long long)g * G) * D) + e8;
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
      *reinterpret_cast<uint4*>(qh16 + ((long long)bg * L + t) * D + e8 * 8) =
          make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                     pack_bf16x2(acc[6], acc[7]));
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) qs[rr][e8 * 8 + c] = acc[c];
    float ss = 0.f;
#pragma unroll
    for (int c = 0; c < 8; ++c) ss = fmaf(acc[c], acc[c], ss);
#pragma unroll
    for (int o = D8 / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
    if (t < L && e8 == 0) qn[(long long)bg * L + t] = sqrtf(ss);
  }
  __syncthreads();
  for (int u = threadIdx.x; u < 32 * D; u += 256) {
    const int e = u / 32, rr = u % 32;
    const int t = t0 + rr;
    if (t < L) qh32t[((long long)bg * D + e) * Lp + t] = qs[rr][e];
  }
}

// K̄ in bf16 with rows reordered to [b][g][i], |K̄_i| in fp32 ([b*Hkv+g][Ncp])
// and the largest |K̄_i| of every tile of 64 chunks. The input holds Nc chunks
// per batch row, chunk c0 first; they land at chunks c0 .. c0+Nc-1 of an
// output laid out for Nrow chunks per (b, g) (c0 = 0, Nrow = Nc for a whole
// memory; a growing memory appends its newly completed chunks).
template <int D>
__global__ void __launch_bounds__(256) sel_kbar_kernel(const float* __restrict__ kbar32, uint16_t* __restrict__ kb16,
                                                       float* __restrict__ kn, unsigned* __restrict__ ktmax,
                                                       long long rows, int Nc, int Ncp, int Hkv, int c0, int Nrow) {
  griddep_wait();
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
    i = c0 + (int)(bi % Nc);
    const long long b = bi / Nc;
    bg = b * Hkv + g;
    const float4* src = reinterpret_cast<const float4*>(kbar32 + row * D + e8 * 8);
    const float4 lo = __ldg(src), hi = __ldg(src + 1);
    x[0] = lo.x, x[1] = lo.y, x[2] = lo.z, x[3] = lo.w, x[4] = hi.x, x[5] = hi.y, x[6] = hi.z, x[7] = hi.w;
    *reinterpret_cast<uint4*>(kb16 + (bg * Nrow + i) * D + e8 * 8) = make_uint4(
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

// Rows whose candidate buffer could not be certified: every visible chunk is
// scored with the exact chain. One block per flagged row (grid-stride); its
// eight warps take 32 chunks at a time, staging the fp32 K̄ rows in shared
// memory with coalesced copies, and keep running top-k lists that warp 0
// merges at the end.
constexpr int kExactWarps = 8;
template <int D>
__global__ void __launch_bounds__(kExactWarps * 32) sel_exact_rows_kernel(
    const float* __restrict__ qh32t, const float* __restrict__ kbar32, const unsigned* __restrict__ nflag,
    const int32_t* __restrict__ flags, int32_t* __restrict__ idx, float* __restrict__ s_sel, int L, int Lp, int Hkv,
    int Nc, int topk, float scale_sel) {
  griddep_wait();
  extern __shared__ __align__(16) unsigned char ex_smem[];
  float* stage_all = reinterpret_cast<float*>(ex_smem);                    // [warps][32 rows][D]
  float* qsh = stage_all + kExactWarps * 32 * D;                             // [D]
  unsigned long long* lists = reinterpret_cast<unsigned long long*>(qsh + D);  // [warps][32]
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const uint32_t stage = smem_u32(stage_all + wib * 32 * D);
  const unsigned n = *nflag;
  for (unsigned f = blockIdx.x; f < n; f += gridDim.x) {
    const long long p = flags[f];
    const int g = (int)(p % Hkv);
    const long long bt = p / Hkv;
    const int t = (int)(bt % L);
    const long long b = bt / L;
    const int vis = min(t / kChunk, Nc);
    const float* qcol = qh32t + (b * Hkv + g) * D * Lp + t;
    for (int e = threadIdx.x; e < D; e += kExactWarps * 32) qsh[e] = qcol[(long long)e * Lp];
    __syncthreads();
    float qr[D];
#pragma unroll
    for (int e = 0; e < D; ++e) qr[e] = qsh[e];
    const float* kb = kbar32 + (b * Nc * Hkv + g) * D;
    unsigned long long lst = 0ull;
    for (int c0 = wib * 32; c0 < vis; c0 += kExactWarps * 32) {
      const int c = c0 + lane < vis ? c0 + lane : -1;
      stage_kbar_rows<D>(stage, kb, (long long)Hkv * D, c, lane);
      const unsigned long long key = c >= 0 ? rank_key(staged_dot<D>(qr, stage, lane) * scale_sel, (uint32_t)c) : 0ull;
      __syncwarp();
      warp_topk_offer(lst, key, topk, lane);
    }
    lists[wib * 32 + lane] = lane < topk ? lst : 0ull;
    __syncthreads();
    if (wib == 0) {
      for (int w = 1; w < kExactWarps; ++w) warp_topk_offer(lst, lists[w * 32 + lane], topk, lane);
      warp_emit_selection(lst, topk, lane, idx + p * topk, s_sel + p * topk);
    }
    __syncthreads();
  }
}

// Decode queries: q̂ in fp32 ([Bq * Hkv, D], head order), in bf16 as the MMA
// operand ([Hkv, n_qt * 128, D], rows past Bq zero) and its norm. Threads
// D/8 per row.
template <int D>
__global__ void __launch_bounds__(256) dtc_qhat_kernel(const uint16_t* __restrict__ q, float* __restrict__ qh32,
                                                       uint16_t* __restrict__ qh16, float* __restrict__ qn, int Bq,
                                                       int Hq, int Hkv, int G, int n_qt) {
  constexpr int D8 = D / 8;
  const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long row = u / D8;  // g * n_qt * 128 + b
  const int e8 = (int)(u % D8);
  const long long rows = (long long)Hkv * n_qt * kTok;
  const int g = (int)(row / ((long long)n_qt * kTok));
  const int b = (int)(row % ((long long)n_qt * kTok));
  const bool in = row < rows;
  const bool valid = in && b < Bq;
  // at most kTok/2 rows: the bf16 rows are stored twice (rows b and b + 64),
  // so that a selection block scans each row with two threads
  const int bs = (Bq <= kTok / 2 && b >= kTok / 2) ? b - kTok / 2 : b;
  float acc[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) acc[c] = 0.f;
  if (in && bs < Bq) {
    const uint4* src = reinterpret_cast<const uint4*>(q + ((long long)bs * Hq + (long long)g * G) * D) + e8;
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
  }
  if (valid) {
    float4* d32 = reinterpret_cast<float4*>(qh32 + ((long long)b * Hkv + g) * D + e8 * 8);
    d32[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    d32[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
  if (in)
    *reinterpret_cast<uint4*>(qh16 + row * D + e8 * 8) =
        make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                   pack_bf16x2(acc[6], acc[7]));
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 8; ++c) ss = fmaf(acc[c], acc[c], ss);
#pragma unroll
  for (int o = D8 / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  if (valid && e8 == 0) qn[(long long)b * Hkv + g] = sqrtf(ss);
}

// Exact score chain of one chunk summary (dot product in dimension order, from 0).
template <int D>
__device__ __forceinline__ float exact_dot(const float* __restrict__ qs, const float* __restrict__ krow) {
  const float4* k4 = reinterpret_cast<const float4*>(krow);
  float acc = 0.f;
#pragma unroll 8
  for (int e4 = 0; e4 < D / 4; ++e4) {
    const float4 kv = __ldg(k4 + e4);
    acc = fmaf(qs[4 * e4], kv.x, acc);
    acc = fmaf(qs[4 * e4 + 1], kv.y, acc);
    acc = fmaf(qs[4 * e4 + 2], kv.z, acc);
    acc = fmaf(qs[4 * e4 + 3], kv.w, acc);
  }
  return acc;
}

// Decode merge: one block (8 warps) per (query, group). lambda = the k-th
// largest lower bound over the entries every scan block exported, at most the
// true lambda. Every range exported its own lambda and the largest lower and
// upper bounds among its entries. lambda is at least the largest range lambda
// (that range alone holds k chunks whose lower bounds reach it) and at least
// the k-th largest of the ranges' largest lower bounds (k ranges hold one such
// chunk each), so only the ranges whose bounds reach that value are read. A block whose
// buffer dropped an entry with upper bound at or above lambda cannot vouch for
// its range: those ranges are scored exactly (rare). The candidates (entries
// with upper bound at or above lambda, and the exactly scored chunks at or
// above it) are ranked by the exact chain, their K̄ rows staged in shared
// memory 32 at a time per warp.
constexpr int kMergeWarps = 8;
constexpr int kMergeCand = 1024;  // listed candidates; any beyond are scored in place
constexpr int kMaxSplit = 320;    // ranges per row (the layout keeps n_split at most 2 * 152)
template <int D>
__global__ void __launch_bounds__(kMergeWarps * 32) dtc_merge_kernel(
    const float* __restrict__ cand_l, const float* __restrict__ cand_u, const int32_t* __restrict__ cand_c,
    const int32_t* __restrict__ cand_n, const float* __restrict__ cand_d, const float4* __restrict__ cand_s, int kbuf,
    const float* __restrict__ qh32, const float* __restrict__ kbar32, int32_t* __restrict__ idx,
    float* __restrict__ s_sel, float* __restrict__ w, int Bq, int Hkv, int Nc, int n_split, int range, int topk,
    float scale_sel, int stick, unsigned* __restrict__ counters) {
  extern __shared__ __align__(16) unsigned char mg_smem[];
  float* stage_all = reinterpret_cast<float*>(mg_smem);  // [warps][32 rows][D]
  float* qs = stage_all + kMergeWarps * 32 * D;           // [D]
  int* cands = reinterpret_cast<int*>(qs + D);            // [kMergeCand]
  __shared__ unsigned long long lists[kMergeWarps][32];
  __shared__ float4 rs[kMaxSplit];  // per range: (lambda, largest lower bound, largest upper bound, dropped bound)
  __shared__ int rn[kMaxSplit];     // per range: exported entries
  __shared__ float red[kMergeWarps];
  __shared__ float lam_s;
  __shared__ int any_unsure, n_cand, n_hit;
  __shared__ int hit[kMaxSplit];      // ranges whose bounds can reach the current threshold
  __shared__ int hpre[kMaxSplit + 1];  // exclusive prefix of their entry counts
  __shared__ unsigned long long rkey[kMaxSplit];  // per range: key of its largest lower bound (0: none)
  __shared__ unsigned long long ranked[32];       // the k best keys of the warp lists, by rank
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int row = blockIdx.x;  // b * Hkv + g
  const int b = row / Hkv, g = row % Hkv;
  const long long cbase = ((long long)g * Bq + b) * n_split;
  const uint32_t stage = smem_u32(stage_all + wib * 32 * D);
  tc::griddep_wait();  // the scan's exported candidates
  if (threadIdx.x == 0) {
    any_unsure = 0, n_cand = 0;
    counters[row] = 0u;  // for the attention kernel that follows (its output sum)
  }
  for (int e = threadIdx.x; e < D; e += kMergeWarps * 32) qs[e] = qh32[(long long)row * D + e];
  // the ranges' summaries into shared memory, and the largest range lambda
  float ls = -INFINITY;
  for (int sp = threadIdx.x; sp < n_split; sp += kMergeWarps * 32) {
    float4 v = cand_s[cbase + sp];
    v.w = cand_d[cbase + sp];
    rs[sp] = v;
    rn[sp] = cand_n[cbase + sp];
    ls = fmaxf(ls, v.x);
  }
  ls = warp_max(ls);
  if (lane == 0) red[wib] = ls;
  auto krow = [&](int c) { return kbar32 + ((long long)c * Hkv + g) * D; };
  // top-k of the warp lists (lane l of each holds its rank-l key, 0: none),
  // in warp 0: every listed key counts the keys above it (keys are distinct)
  auto combine = [&](unsigned long long mine) {
    lists[wib][lane] = mine;
    if (threadIdx.x < 32) ranked[threadIdx.x] = 0ull;
    __syncthreads();
    const int n = kMergeWarps * topk;
    if (threadIdx.x < n) {
      const unsigned long long key = lists[threadIdx.x / topk][threadIdx.x % topk];
      if (key != 0ull) {
        int rank = 0;
        for (int j = 0; j < n; ++j) rank += lists[j / topk][j % topk] > key ? 1 : 0;
        if (rank < topk) ranked[rank] = key;
      }
    }
    __syncthreads();
    return wib == 0 ? ranked[lane] : 0ull;
  };
  // the ranges whose bound `field` reaches t, listed in shared memory (any
  // order), with the exclusive prefix of their entry counts; returns the
  // number of listed entries
  auto list_ranges = [&](int field, float t) {
    if (threadIdx.x == 0) n_hit = 0;
    __syncthreads();
    for (int sp = threadIdx.x; sp < n_split; sp += kMergeWarps * 32) {
      const float4 v = rs[sp];
      if ((field == 1 ? v.y : v.z) >= t) hit[atomicAdd(&n_hit, 1)] = sp;
    }
    __syncthreads();
    if (wib == 0) {  // lane l sums a run of the listed ranges, then a warp scan
      const int nh = n_hit, per = (nh + 31) / 32, h0 = min(lane * per, nh), h1 = min(h0 + per, nh);
      int sum = 0;
      for (int h = h0; h < h1; ++h) sum += rn[hit[h]];
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
      }
      int run = incl - sum;
      for (int h = h0; h < h1; ++h) {
        hpre[h] = run;
        run += rn[hit[h]];
      }
      if (lane == 31) hpre[nh] = incl;
    }
    __syncthreads();
    return hpre[n_hit];
  };
  // entry e of the listed ranges: (range, slot) through the prefix
  auto entry_at = [&](int e, int& sp, int& j) {
    int lo = 0, hi = n_hit;  // the last h with hpre[h] <= e
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (hpre[mid] <= e) lo = mid; else hi = mid;
    }
    sp = hit[lo];
    j = e - hpre[lo];
  };
  for (int sp = threadIdx.x; sp < n_split; sp += kMergeWarps * 32)
    rkey[sp] = rs[sp].y > -INFINITY ? ((unsigned long long)order_bits(rs[sp].y) << 32) | (uint32_t)sp : 0ull;
  if (threadIdx.x == 0) lam_s = -INFINITY;
  __syncthreads();
  // the k-th largest of the ranges' largest lower bounds: each range key
  // counts the range keys above it
  for (int sp = threadIdx.x; sp < n_split; sp += kMergeWarps * 32) {
    const unsigned long long key = rkey[sp];
    if (key != 0ull) {
      int rank = 0;
      for (int j = 0; j < n_split; ++j) rank += rkey[j] > key ? 1 : 0;
      if (rank == topk - 1) lam_s = rs[sp].y;
    }
  }
  __syncthreads();
  float lam_star = lam_s;
#pragma unroll
  for (int k = 0; k < kMergeWarps; ++k) lam_star = fmaxf(lam_star, red[k]);
  __syncthreads();  // lam_s is written again below
  // ---- lambda over the entries (at or above lam_star) of the ranges that can
  // hold them: the entries of the listed ranges, one per thread
  unsigned long long lst = 0ull;
  {
    const int ne = list_ranges(1, lam_star);
    for (int base = wib * 32; base < ne; base += kMergeWarps * 32) {
      const int e = base + lane;
      unsigned long long key = 0ull;
      if (e < ne) {
        int sp, j;
        entry_at(e, sp, j);
        const float l = cand_l[(cbase + sp) * kbuf + j];
        if (l >= lam_star) key = ((unsigned long long)order_bits(l) << 32) | (uint32_t)(sp * kbuf + j);
      }
      warp_topk_offer(lst, key, topk, lane);
    }
  }
  {
    const unsigned long long all = combine(lst);
    if (wib == 0) {
      const unsigned long long kth = __shfl_sync(0xFFFFFFFFu, all, topk - 1);
      if (lane == 0) lam_s = kth != 0ull ? order_bits_to_float((uint32_t)(kth >> 32)) : -INFINITY;
    }
    __syncthreads();
  }
  const float lam = lam_s;
  for (int sp = threadIdx.x; sp < n_split; sp += kMergeWarps * 32)
    if (rs[sp].w >= lam) any_unsure = 1;
  // ---- the candidates: entries with upper bound at or above lambda, listed
  // (past the list's capacity they are scored here, one per lane)
  unsigned long long fin = 0ull;
  {
    const int ne = list_ranges(2, lam);
    for (int base = wib * 32; base < ne; base += kMergeWarps * 32) {
      const int e = base + lane;
      unsigned long long key = 0ull;
      if (e < ne) {
        int sp, j;
        entry_at(e, sp, j);
        if (cand_u[(cbase + sp) * kbuf + j] >= lam) {
          const int c = cand_c[(cbase + sp) * kbuf + j];
          const int pos = atomicAdd(&n_cand, 1);
          if (pos < kMergeCand)
            cands[pos] = c;
          else
            key = rank_key(exact_dot<D>(qs, krow(c)) * scale_sel, (uint32_t)c);
        }
      }
      warp_topk_offer(fin, key, topk, lane);
    }
  }
  __syncthreads();
  const bool unsure = any_unsure != 0;
  {
    float qr[D];
#pragma unroll
    for (int e = 0; e < D; ++e) qr[e] = qs[e];
    const int nlist = min(n_cand, kMergeCand);
    // each warp rescores an equal share (up to 32 rows at a time)
    const int per = min(32, (nlist + kMergeWarps - 1) / kMergeWarps);
    for (int base = wib * per; base < nlist; base += kMergeWarps * per) {
      const int i = base + lane;
      const int c = (lane < per && i < nlist) ? cands[i] : -1;
      stage_kbar_rows<D>(stage, kbar32 + (long long)g * D, (long long)Hkv * D, c, lane);
      const unsigned long long key =
          c >= 0 ? rank_key(staged_dot<D>(qr, stage, lane) * scale_sel, (uint32_t)c) : 0ull;
      __syncwarp();
      warp_topk_offer(fin, key, topk, lane);
    }
  }
  for (int sp = 0; unsure && sp < n_split; ++sp) {
    if (!(rs[sp].w >= lam)) continue;  // uniform across the block
    // this range's exported entries are scored again below the whole range:
    // skip them there to keep every chunk once
    const int cb = sp * range, ce = min(cb + range, Nc);
    const int n = rn[sp];
    for (int c0 = cb + wib * 32; c0 < ce; c0 += kMergeWarps * 32) {
      const int c = c0 + lane;
      unsigned long long key = 0ull;
      if (c < ce) {
        bool exported = false;
        for (int j = 0; j < n; ++j) exported |= cand_c[(cbase + sp) * kbuf + j] == c && cand_u[(cbase + sp) * kbuf + j] >= lam;
        const float dot = exact_dot<D>(qs, krow(c));
        if (!exported && dot >= lam) key = rank_key(dot * scale_sel, (uint32_t)c);
      }
      warp_topk_offer(fin, key, topk, lane);
    }
  }
  const unsigned long long all = combine(fin);
  if (wib != 0) return;
  const long long o = (long long)row * topk;
  warp_emit_selection(all, topk, lane, idx + o, s_sel + o);
  __syncwarp();
  bool valid = false;
  float sv = -INFINITY;
  if (lane < topk) {
    valid = idx[o + lane] >= 0;
    if (valid) sv = s_sel[o + lane];
  }
  const float wj = warp_chunk_weight(sv, valid, stick != 0);
  if (lane < topk) w[o + lane] = wj;
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct SelLayout {
  size_t qh16, qh32, qn, kb16, kn, ktmax, nflag, flags, total;
};

inline int padded_chunks(const Dims& D) { return (D.Nc + kCt - 1) / kCt * kCt; }
// Row length of the transposed fp32 q̂ (a multiple of 4 tokens: TMA row strides are multiples of 16 bytes).
inline int padded_tokens(const Dims& D) { return (D.L + 3) / 4 * 4; }

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
  o = align256(o + (size_t)D.B * D.Hkv * D.d * padded_tokens(D) * 4);
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
  const long long krows = (long long)Dm.B * Dm.Nc * Dm.Hkv;
  const int BH = Dm.B * Dm.Hkv;
  cudaError_t e;
  // the tile maxima and the flagged-row counter are adjacent: one clear covers both
  if ((e = cudaMemsetAsync(ktmax, 0, lo.flags - lo.ktmax, st)) != cudaSuccess) return e;
  constexpr int D8 = DD / 8;
  const int Lp = padded_tokens(Dm);
  (void)launch_dependent(sel_qhat_kernel<DD>, dim3((unsigned)((Dm.L + 31) / 32), (unsigned)BH), dim3(256), 0, st,
                         (const uint16_t*)q, qh16, qh32, qn, Dm.L, Lp, Dm.Hq, Dm.Hkv, Dm.G);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int Ncp = padded_chunks(Dm);
  (void)launch_dependent(sel_kbar_kernel<DD>, dim3((unsigned)((krows * D8 + 255) / 256)), dim3(256), 0, st, kbar32,
                         kb16, kn, ktmax, krows, Dm.Nc, Ncp, Dm.Hkv, 0, Dm.Nc);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;

  CUtensorMap tq, tk, tq32t;
  memset(&tq, 0, sizeof(tq));
  memset(&tk, 0, sizeof(tk));
  memset(&tq32t, 0, sizeof(tq32t));
  if (!tc::make_plain_tmap_f32(&tq32t, qh32, (unsigned long long)BH * DD, Lp, kTok, DD)) return cudaErrorNotSupported;
  if (!tc::make_rows_tmap(&tq, qh16, (unsigned long long)q_rows(Dm), DD, kTok)) return cudaErrorNotSupported;
  if (!tc::make_rows_tmap(&tk, kb16, (unsigned long long)k_rows(Dm), DD, kCt)) return cudaErrorNotSupported;
  SelTcArgs a{};
  a.status = Dm.status;
  a.qh32t = qh32;
  a.qn = qn;
  a.kbar32 = kbar32;
  a.kn = kn;
  a.ktmax = (const float*)ktmax;
  a.idx = idx;
  a.s_sel = s_sel;
  a.nflag = nflag;
  a.flags = flags;
  a.L = Dm.L;
  a.Lp = Lp;
  a.Hkv = Dm.Hkv;
  a.Nc = Dm.Nc;
  a.Ncp = Ncp;
  a.Nrow = Dm.Nc;
  a.topk = Dm.topk;
  a.n_qt = (Dm.L + kTok - 1) / kTok;
  a.BH = BH;
  a.scale_sel = Dm.scale_sel;
  const size_t smem = sizeof(SelTcSmem<DD, KT>) + 1024;
  if ((e = cudaFuncSetAttribute(sel_tc_kernel<DD, KT, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem)) != cudaSuccess)
    return e;
  const long long blocks = (long long)a.n_qt * BH;
  (void)launch_dependent(sel_tc_kernel<DD, KT, false>, dim3((unsigned)blocks), dim3(kThreads), smem, st, a, tq, tk,
                         tq32t);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const size_t ex_smem = ((size_t)kExactWarps * 32 * DD + DD) * 4 + (size_t)kExactWarps * 32 * 8;
  if ((e = cudaFuncSetAttribute(sel_exact_rows_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)ex_smem)) != cudaSuccess)
    return e;
  (void)launch_dependent(sel_exact_rows_kernel<DD>, dim3(152), dim3(kExactWarps * 32), ex_smem, st, qh32, kbar32, nflag,
                         flags, idx, s_sel, Dm.L, Lp, Dm.Hkv, Dm.Nc, Dm.topk, Dm.scale_sel);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

// ---------------------------------------------------------------- decode against a resident memory
namespace {

struct DecIndexLayout {
  size_t kb16, kn, ktmax, total;
};

// Laid out for the memory's capacity (D.cap chunks per head), so that a growing
// memory keeps every offset as chunks are appended.
DecIndexLayout dec_index_layout(const DecodeDims& D) {
  const size_t ncp = (size_t)((D.cap + kCt - 1) / kCt * kCt);
  const size_t krows = std::max<size_t>((size_t)D.Hkv * D.cap, kCt);
  DecIndexLayout lo{};
  size_t o = 0;
  lo.kb16 = o;
  o = align256(o + krows * D.d * 2);
  lo.kn = o;
  o = align256(o + (size_t)D.Hkv * ncp * 4);
  lo.ktmax = o;
  o = align256(o + (size_t)D.Hkv * (ncp / kCt) * 16);
  lo.total = o;
  return lo;
}

struct DecTcLayout {
  size_t qh32, qh16, qn, cl, cu, cc, cn, cd, cs, opart, total;
  int n_qt, n_split, range;
};

template <int KT>
DecTcLayout dec_tc_layout(const DecodeDims& D) {
  DecTcLayout lo{};
  lo.n_qt = (D.Bq + kTok - 1) / kTok;
  const long long want = (2LL * 152) / ((long long)D.Hkv * lo.n_qt);
  lo.n_split = (int)std::max<long long>(1, std::min<long long>(want, (D.Nc + kCt - 1) / kCt));
  const long long per = (D.Nc + lo.n_split - 1) / lo.n_split;
  lo.range = (int)((per + kCt - 1) / kCt * kCt);
  lo.n_split = (int)((D.Nc + lo.range - 1) / lo.range);
  const size_t rows = (size_t)D.Bq * D.Hkv;
  const size_t nc = rows * lo.n_split * SelCfg<KT>::kExport;
  size_t o = 0;
  lo.qh32 = o;
  o = align256(o + rows * D.d * 4);
  lo.qh16 = o;
  o = align256(o + (size_t)D.Hkv * lo.n_qt * kTok * D.d * 2);
  lo.qn = o;
  o = align256(o + rows * 4);
  lo.cl = o;
  o = align256(o + nc * 4);
  lo.cu = o;
  o = align256(o + nc * 4);
  lo.cc = o;
  o = align256(o + nc * 4);
  lo.cn = o;
  o = align256(o + rows * lo.n_split * 4);
  lo.cd = o;
  o = align256(o + rows * lo.n_split * 4);
  lo.cs = o;
  o = align256(o + rows * lo.n_split * 16);
  lo.opart = o;
  o = align256(o + decode_attend_scratch(D));
  lo.total = o;
  return lo;
}

template <int DD, int KT>
cudaError_t run_decode_tc(const DecodeDims& Dm, const void* q, const void* K, const void* V, const float* kbar32,
                          const void* index, void* O, int32_t* idx, float* s_sel, float* w, void* ws,
                          cudaStream_t st) {
  const DecTcLayout lo = dec_tc_layout<KT>(Dm);
  const DecIndexLayout ix = dec_index_layout(Dm);
  char* base = (char*)ws;
  float* qh32 = (float*)(base + lo.qh32);
  uint16_t* qh16 = (uint16_t*)(base + lo.qh16);
  float* qn = (float*)(base + lo.qn);
  const char* ib = (const char*)index;
  cudaError_t e;
  constexpr int D8 = DD / 8;
  const long long qrows = (long long)Dm.Hkv * lo.n_qt * kTok;
  dtc_qhat_kernel<DD><<<(unsigned)((qrows * D8 + 255) / 256), 256, 0, st>>>((const uint16_t*)q, qh32, qh16, qn, Dm.Bq,
                                                                           Dm.Hq, Dm.Hkv, Dm.G, lo.n_qt);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  CUtensorMap tq, tk, unused;
  memset(&tq, 0, sizeof(tq));
  memset(&tk, 0, sizeof(tk));
  memset(&unused, 0, sizeof(unused));
  const unsigned long long krows = std::max<unsigned long long>((unsigned long long)Dm.Hkv * Dm.cap, kCt);
  if (!tc::make_rows_tmap(&tq, qh16, (unsigned long long)qrows, DD, kTok)) return cudaErrorNotSupported;
  if (!tc::make_rows_tmap(&tk, ib + ix.kb16, krows, DD, kCt)) return cudaErrorNotSupported;
  SelTcArgs a{};
  a.status = Dm.status;
  a.qn = qn;
  a.kbar32 = kbar32;
  a.kn = (const float*)(ib + ix.kn);
  a.ktmax = (const float*)(ib + ix.ktmax);
  a.L = 1;
  a.Hkv = Dm.Hkv;
  a.Nc = (int)Dm.Nc;
  a.Ncp = (int)((Dm.cap + kCt - 1) / kCt * kCt);
  a.Nrow = (int)Dm.cap;
  a.topk = Dm.topk;
  a.n_qt = lo.n_qt;
  a.BH = Dm.Hkv;
  a.scale_sel = Dm.scale_sel;
  a.Bq = Dm.Bq;
  a.n_split = lo.n_split;
  a.range = lo.range;
  a.cand_l = (float*)(base + lo.cl);
  a.cand_u = (float*)(base + lo.cu);
  a.cand_c = (int32_t*)(base + lo.cc);
  a.cand_n = (int32_t*)(base + lo.cn);
  a.cand_d = (float*)(base + lo.cd);
  a.cand_s = (float4*)(base + lo.cs);
  const size_t smem = sizeof(SelTcSmem<DD, KT, true>) + 1024;
  if ((e = cudaFuncSetAttribute(sel_tc_kernel<DD, KT, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem)) != cudaSuccess)
    return e;
  // the scan, the merge and the attention each start as programmatic dependents
  // of the kernel before (their setup overlaps its tail)
  e = launch_dependent(sel_tc_kernel<DD, KT, true>, dim3((unsigned)lo.n_split, (unsigned)Dm.Hkv, (unsigned)lo.n_qt),
                       dim3(kThreads), smem, st, a, tq, tk, unused);
  note_launches(1);
  if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
  const int rows = Dm.Bq * Dm.Hkv;
  if (lo.n_split > kMaxSplit) return cudaErrorNotSupported;
  const size_t mg_smem = ((size_t)kMergeWarps * 32 * DD + DD) * 4 + (size_t)kMergeCand * 4;
  if ((e = cudaFuncSetAttribute(dtc_merge_kernel<DD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)mg_smem)) !=
      cudaSuccess)
    return e;
  unsigned* counters = decode_attend_counters(Dm, base + lo.opart);
  e = launch_dependent(dtc_merge_kernel<DD>, dim3((unsigned)rows), dim3(kMergeWarps * 32), mg_smem, st,
                       (const float*)a.cand_l, (const float*)a.cand_u, (const int32_t*)a.cand_c,
                       (const int32_t*)a.cand_n, (const float*)a.cand_d, (const float4*)a.cand_s,
                       (int)SelCfg<KT>::kExport, (const float*)qh32, kbar32, idx, s_sel, w, Dm.Bq, Dm.Hkv, (int)Dm.Nc,
                       lo.n_split, lo.range, Dm.topk, Dm.scale_sel, Dm.stick ? 1 : 0, counters);
  note_launches(1);
  if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
  return launch_decode_attend(Dm, q, K, V, idx, w, O, base + lo.opart, st, true, true);
}

}  // namespace

bool decode_index_applies(const DecodeDims& D) {
  return D.topk <= 16 && D.cap > 0 && D.cap * (long long)D.Hkv < (1LL << 31);
}

bool decode_tc_applies(const DecodeDims& D) { return decode_index_applies(D) && D.Nc > 0; }

size_t decode_index_bytes(const DecodeDims& D) { return decode_index_applies(D) ? dec_index_layout(D).total : 0; }

cudaError_t launch_index_rows(const DecodeDims& Dm, const float* kbar32, void* index, long long c0, long long c1,
                              cudaStream_t st) {
  if (c1 <= c0) return cudaSuccess;
  const DecIndexLayout ix = dec_index_layout(Dm);
  char* base = (char*)index;
  const int Ncp = (int)((Dm.cap + kCt - 1) / kCt * kCt);
  const long long krows = (c1 - c0) * Dm.Hkv;  // input rows (i, g) of the one-batch memory, chunk c0 first
  const float* src = kbar32 + c0 * Dm.Hkv * Dm.d;
  if (Dm.d == 64)
    (void)launch_dependent(sel_kbar_kernel<64>, dim3((unsigned)((krows * 8 + 255) / 256)), dim3(256), 0, st, src,
                           (uint16_t*)(base + ix.kb16), (float*)(base + ix.kn), (unsigned*)(base + ix.ktmax), krows,
                           (int)(c1 - c0), Ncp, Dm.Hkv, (int)c0, (int)Dm.cap);
  else
    (void)launch_dependent(sel_kbar_kernel<128>, dim3((unsigned)((krows * 16 + 255) / 256)), dim3(256), 0, st, src,
                           (uint16_t*)(base + ix.kb16), (float*)(base + ix.kn), (unsigned*)(base + ix.ktmax), krows,
                           (int)(c1 - c0), Ncp, Dm.Hkv, (int)c0, (int)Dm.cap);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_decode_index(const DecodeDims& Dm, const float* kbar32, void* index, cudaStream_t st) {
  // every byte starts at zero (rows and norms of chunks not yet in the memory,
  // tile maxima before the atomic max), then the Nc chunks present are written
  cudaError_t e = cudaMemsetAsync(index, 0, dec_index_layout(Dm).total, st);
  if (e != cudaSuccess) return e;
  return launch_index_rows(Dm, kbar32, index, 0, Dm.Nc, st);
}

size_t decode_tc_workspace(const DecodeDims& D) {
  if (!decode_tc_applies(D) || D.Bq == 0) return 0;
  return D.topk <= 8 ? dec_tc_layout<8>(D).total : dec_tc_layout<16>(D).total;
}

cudaError_t launch_decode_tc(const DecodeDims& D, const void* q, const void* K, const void* V, const float* kbar32,
                             const void* index, void* O, int32_t* idx, float* s_sel, float* w, void* ws,
                             cudaStream_t st) {
  if (D.d == 64) return D.topk <= 8 ? run_decode_tc<64, 8>(D, q, K, V, kbar32, index, O, idx, s_sel, w, ws, st)
                                    : run_decode_tc<64, 16>(D, q, K, V, kbar32, index, O, idx, s_sel, w, ws, st);
  return D.topk <= 8 ? run_decode_tc<128, 8>(D, q, K, V, kbar32, index, O, idx, s_sel, w, ws, st)
                     : run_decode_tc<128, 16>(D, q, K, V, kbar32, index, O, idx, s_sel, w, ws, st);
}

bool select_tc_applies(const Dims& D) { return D.topk <= 16 && D.Nc > 0; }

size_t select_tc_workspace(const Dims& D) { return select_tc_applies(D) ? sel_layout(D).total : 0; }


cudaError_t launch_select_tc(const Dims& D, const void* q, const float* kbar32, int32_t* idx, float* s_sel, void* ws,
                             cudaStream_t st) {
  if (D.d == 64) return D.topk <= 8 ? run_tc<64, 8>(D, q, kbar32, idx, s_sel, ws, st)
                                    : run_tc<64, 16>(D, q, kbar32, idx, s_sel, ws, st);
  return D.topk <= 8 ? run_tc<128, 8>(D, q, kbar32, idx, s_sel, ws, st)
                     : run_tc<128, 16>(D, q, kbar32, idx, s_sel, ws, st);
}

}  // namespace hsa
