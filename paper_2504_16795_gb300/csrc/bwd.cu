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
// dK̄_I / S inside the same tensor-core product. The same tile also yields the
// selection term of dq: K̄_I is the mean of the chunk's S key rows, so
// (da c_att + c_sel ds_j / S) K_I = c_att da K_I + c_sel ds_j K̄_I.
//
// Chunk-major and deterministic: one block per (b, g, chunk) owns that
// chunk's dK/dV rows, walks the chunk's slots (from the inverse index) in
// increasing token order 128 query rows at a time and accumulates dK^T and
// dV^T in tensor memory; no floating-point atomics anywhere. Each slot's dq
// contribution goes to a bf16 workspace row and a second kernel sums the k
// slots of each token in slot order (fp32).
//
// Per 128-row step on the 5th-generation tensor core (one issuing thread):
//   S = Q K^T, dP' = dO V^T            (M = 128 rows, N = 64, K = d)
//   dV^T += dO^T (wP), dK^T += Q^T dSk (M = d, N = 64, K = 128 rows; the
//                                       row-major tiles read MN-major)
//   dq' = dSk K                        (K read as an MN-major operand)
// The dK/dV products come first, so the Q/dO stage is released before the
// dq product runs. Warps 0-3 and 12-15 (two threads per row) turn S, dP'
// into P and dSk; warps 4-7 store dq' and finally dK, dV; warps 8, 10 and 11 gather the
// Q and dO rows of the next tiles; one thread of warp 9 issues the MMAs.
#include <cstring>

#include "tc.cuh"

namespace hsa {
namespace {

constexpr int kRows = 128;     // query rows per step (tensor-core M)
constexpr int kThreads = 512;  // warps 0-3 and 12-15 softmax/gradients, 4-7 epilogue, 8, 10, 11 loaders, 9 MMA
constexpr int kLoaders = 3;
constexpr int kTmemCols = 512;

template <int D>
struct BwdSmem {
  uint16_t Q[2][kRows * D];       // gathered query rows (grouped K-major SW128, tc::grp_offset)
  uint16_t dO[2][kRows * D];      // gathered output gradients (same layout)
  uint16_t K[kChunk * D];         // chunk keys [s][d]
  uint16_t V[kChunk * D];         // chunk values [s][d]
  uint16_t P[kRows * kChunk];     // w * P
  uint16_t dSk[kRows * kChunk];   // c_att * w * P∘(dP' - D) + c_sel * ds / S  (feeds dK and dq)
  uint16_t dqstage[kRows * 64];   // TMA path: 64 columns of dq' (8-row atoms, 128-byte swizzle; 4 KB per warp)
  int slot_row[2][kRows];         // first q row of each slot (-1: past the list)
  int slot_p[2][kRows];
  float slot_w[2][kRows];
  float slot_delta[2][kRows];
  int row_p[3][kRows];            // softmax -> epilogue: the row's slot id (-1: none)
  float xch[3][2][kRows];         // softmax halves: row maximum, sum and D of each half
  uint64_t bar[16];
  uint32_t tmem_base;
  int abort_flag;
};

// one block per SM: the layout plus the 1024-byte alignment slack must fit the 227 KB opt-in limit
static_assert(sizeof(BwdSmem<128>) + 1024 <= 232448, "shared memory layout too large");

enum {
  BAR_QD_FULL = 0,   // 2: Q and dO tiles landed
  BAR_QD_EMPTY = 2,  // 2: every MMA reading the tiles finished (commit)
  BAR_S_FULL = 4,    // 2: S and dP' ready (commit)
  BAR_S_EMPTY = 6,   // 2: S and dP' read (256 arrivals)
  BAR_P_FULL = 8,    // P, dSk written (256 arrivals)
  BAR_P_EMPTY = 9,   // P, dSq, dSk consumed (commit)
  BAR_DQ_FULL = 10,  // dq accumulator ready (commit)
  BAR_DQ_EMPTY = 11, // dq read (128 arrivals)
  BAR_ACC_DONE = 12, // last dK^T / dV^T update finished (commit)
  BAR_DS_FULL = 13   // 3: row_p of a step written (128 arrivals)
};

struct BwdArgs {
  const uint16_t* q;
  const uint16_t* K;
  const uint16_t* V;
  const uint16_t* dO;
  const float* w;
  const float* delta;  // [B, L, Hkv]
  const int32_t* offsets;
  const int32_t* entries;
  uint16_t* dqpart;  // [slots, G, D] bf16
  float* dK;
  float* dV;
  int L, Hq, Hkv, G, log2G, topk, Nc;
  int n_rows;   // B * L * Hq (a row index past it reads zeros)
  long long n_slots;  // B * L * Hkv * topk (slot ids; debug builds check offsets and entries against it)
  int use_tma;  // G >= 8: each slot's G rows arrive as one swizzled TMA box
  float scale_log2, scale_attn, scale_sel;
  int softmax1;   // softmax-off-by-one inside the chunk
  int dw_mode;    // write dw per slot and leave the selection terms to later passes
                  // (stick-breaking weights, or the attention-only backward)
  float* dw_out;  // [slots] (dw_mode only)
  unsigned* status;  // the call's status word (a bounded wait that gives up sets it)
};

// TMEM columns
template <int D>
struct Cols {
  static constexpr uint32_t S = 0;            // 2 x 64
  static constexpr uint32_t dP = 128;         // 2 x 64
  static constexpr uint32_t dq = 256;         // D
  static constexpr uint32_t dVt = 256 + D;    // 64 (rows = head dim)
  static constexpr uint32_t dKt = 320 + D;    // 64
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_chunk_kernel(BwdArgs a, const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_do,
                     const __grid_constant__ CUtensorMap tmap_dq) {
  griddep_wait();
  extern __shared__ unsigned char smem_raw[];
  BwdSmem<D>& sm = *reinterpret_cast<BwdSmem<D>*>(smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u));
  constexpr int D8 = D / 8;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int c, bg;
  block_key(a.Nc, (int)(gridDim.x / (unsigned)a.Nc), c, bg);
  const int key = bg * a.Nc + c;
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int off = a.offsets[key];
  int cnt = a.offsets[key + 1] - off;
  if (!(bounds_ok(off, 0, a.n_slots + 1, a.status) && bounds_ok(off + cnt, off, a.n_slots + 1, a.status)))
    cnt = 0;  // debug: a list outside the entries is skipped
  const long long row0 = ((long long)b * a.L + (long long)c * kChunk) * a.Hkv + g;
  if (cnt <= 0) {  // a chunk nobody selected: no gradient
    for (int u = tid; u < kChunk * D; u += kThreads) {
      const long long o = (row0 + (long long)(u / D) * a.Hkv) * D + (u % D);
      a.dK[o] = 0.f;
      a.dV[o] = 0.f;
    }
    return;
  }
  const int epi = kRows >> a.log2G;
  const int niter = (cnt + epi - 1) / epi;
  const int slot_div = a.Hkv * a.topk;
  auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
  volatile int* abort_flag = &sm.abort_flag;
  unsigned* status = a.status;

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(bar(BAR_QD_FULL + i), a.use_tma ? kLoaders : 32);
      tc::mbar_init(bar(BAR_QD_EMPTY + i), 1);
      tc::mbar_init(bar(BAR_S_FULL + i), 1);
      tc::mbar_init(bar(BAR_S_EMPTY + i), 256);
    }
    for (int i = 0; i < 3; ++i) tc::mbar_init(bar(BAR_DS_FULL + i), 128);
    tc::mbar_init(bar(BAR_P_FULL), 256);
    tc::mbar_init(bar(BAR_P_EMPTY), 1);
    tc::mbar_init(bar(BAR_DQ_FULL), 1);
    tc::mbar_init(bar(BAR_DQ_EMPTY), 128);
    tc::mbar_init(bar(BAR_ACC_DONE), 1);
    sm.abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 9) tc::tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sm.tmem_base;
  // chunk K and V (rows s), once per block, by warps 0-7 while the loaders
  // already gather the first tiles; the MMA warp meets them at named barrier
  // 5 before its first product
  if (warp < 8) {
    for (int u = tid; u < kChunk * D8; u += 256) {
      const int srow = u / D8, ch = u % D8;
      const long long src = (row0 + (long long)srow * a.Hkv) * D + ch * 8;
      cp_async16(smem_u32(sm.K) + tc::sw128_offset(kChunk, srow, ch * 8), a.K + src);
      cp_async16(smem_u32(sm.V) + tc::sw128_offset(kChunk, srow, ch * 8), a.V + src);
    }
    cp_async_commit();
    cp_async_wait<0>();
    tc::fence_proxy_async_smem();
    asm volatile("bar.arrive 5, 288;" ::: "memory");
  }

  if (warp == 8 || warp == 10 || warp == 11) {
    // ---------------------------------------------------------------- loader warps
    // TMA path: a tile's 2 * epi gathers (item s < epi: the q rows of slot s;
    // item epi + s: the dO rows of slot s) are spread over warps 8, 10 and 11,
    // lane l of loader li taking item li + 3 l, since a TMA issue costs the
    // issuing warp tens of nanoseconds per box. Warp 8 also fills the slot
    // tables and runs the cp.async path alone. Slot data is fetched in two
    // stages ahead of use: the slot ids two tiles ahead, the token, weight and
    // Δ one tile ahead, so no dependent global load sits on the critical path.
    const int li = warp == 8 ? 0 : warp - 9;
    const int item = li + kLoaders * lane;
    const bool has_item = a.use_tma && item < 2 * epi;
    const int islot = item < epi ? item : item - epi;
    const uint32_t item_bytes = (uint32_t)((2 * epi - li + kLoaders - 1) / kLoaders) * a.G * D * 2;
    const uint64_t keep = tc::l2_evict_last();
    auto checked = [&](int p) { return p < 0 || bounds_ok(p, 0, a.n_slots, status) ? p : -1; };
    auto load_ip = [&](int i) {
      const int e = i * epi + islot;
      return checked((has_item && e < cnt) ? a.entries[off + e] : -1);
    };
    auto row_of = [&](int p) {  // past the list: rows past the tensor read zeros
      return p < 0 ? a.n_rows : ((b * a.L + (p / slot_div) % a.L) * a.Hq) + g * a.G;
    };
    auto load_p = [&](int i) {  // warp 8's slot tables: lane l holds slot l
      const int e = i * epi + lane;
      return checked((li == 0 && epi <= 32 && lane < epi && e < cnt) ? a.entries[off + e] : -1);
    };
    int n_row = -1, n_p = -1;
    float n_w = 0.f, n_dl = 0.f;
    auto resolve = [&](int p) {  // slot id -> query row, weight, Δ (loads issued, used an iteration later)
      n_p = p, n_row = -1, n_w = 0.f, n_dl = 0.f;
      if (p >= 0) {
        const int t = (p / slot_div) % a.L;
        n_row = ((b * a.L + t) * a.Hq) + g * a.G;
        n_w = a.w[p];
        n_dl = a.delta[((long long)b * a.L + t) * a.Hkv + g];
      }
    };
    if (li == 0 || a.use_tma) {
      int ip_cur = load_ip(0), ip_next = load_ip(1);
      resolve(load_p(0));
      int p_ahead = load_p(1);
      for (int i = 0; i < niter; ++i) {
        const int st = i & 1;
        const int yi = row_of(ip_cur);
        ip_cur = ip_next;
        ip_next = load_ip(i + 2);
        const int c_row = n_row, c_p = n_p;
        const float c_w = n_w, c_dl = n_dl;
        resolve(p_ahead);
        p_ahead = load_p(i + 2);
        // cp.async path: publish tile i-1 before waiting for tile i's stage (that
        // stage is freed by the dK/dV products of step i-2, which the MMA thread
        // issues only after S/dP' of step i-1, which needs tile i-1)
        if (i >= 1 && !a.use_tma) {
          cp_async_wait<0>();
          tc::fence_proxy_async_smem();
          tc::mbar_arrive(bar(BAR_QD_FULL + ((i - 1) & 1)));
        }
        tc::mbar_wait(bar(BAR_QD_EMPTY + st), ((i >> 1) & 1) ^ 1, abort_flag, status);
        if (li == 0) {
          if (epi <= 32) {
            if (lane < epi) {
              sm.slot_row[st][lane] = c_row;
              sm.slot_p[st][lane] = c_p;
              sm.slot_w[st][lane] = c_w;
              sm.slot_delta[st][lane] = c_dl;
            }
          } else {
            for (int sl = lane; sl < epi; sl += 32) {
              const int e = i * epi + sl;
              int row = -1, p = -1;
              float wv = 0.f, dl = 0.f;
              if (e < cnt) p = checked(a.entries[off + e]);
              if (p >= 0) {
                const int t = (p / slot_div) % a.L;
                row = ((b * a.L + t) * a.Hq) + g * a.G;
                wv = a.w[p];
                dl = a.delta[((long long)b * a.L + t) * a.Hkv + g];
              }
              sm.slot_row[st][sl] = row;
              sm.slot_p[st][sl] = p;
              sm.slot_w[st][sl] = wv;
              sm.slot_delta[st][sl] = dl;
            }
          }
        }
        const uint32_t qb = smem_u32(sm.Q[st]), ob = smem_u32(sm.dO[st]);
        if (a.use_tma) {
          // one box per 8-row group of the lane's item; each loader's expected
          // arrival carries its byte count (warp 8's also publishes the tables)
          if (has_item) {
            const uint32_t dst = (item < epi ? qb : ob) + islot * (a.G >> 3) * (16 * D);
            const CUtensorMap* m = item < epi ? &tmap_q : &tmap_do;
            for (int j = 0; j < (a.G >> 3); ++j)
              tc::tma_load_3d_hint(dst + j * (16 * D), m, 0, yi + 8 * j, 0, bar(BAR_QD_FULL + st), keep);
          }
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_expect_tx(bar(BAR_QD_FULL + st), item_bytes);
          continue;
        }
        __syncwarp();
        for (int u = lane; u < kRows * D8; u += 32) {
          const int r = u / D8, ch = u % D8;
          const int row = sm.slot_row[st][r >> a.log2G];
          const uint32_t o = tc::grp_offset(D, r, ch * 8);
          if (row >= 0) {
            const long long src = ((long long)(row + (r & (a.G - 1)))) * D + ch * 8;
            cp_async16(qb + o, a.q + src);
            cp_async16(ob + o, a.dO + src);
          } else {
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(qb + o), "r"(0));
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(ob + o), "r"(0));
          }
        }
        cp_async_commit();
      }
      if (!a.use_tma) {
        cp_async_wait<0>();
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(bar(BAR_QD_FULL + ((niter - 1) & 1)));
      }
    }
  } else if (warp == 9) {
    // ---------------------------------------------------------------- MMA issue (one thread)
    asm volatile("bar.sync 5, 288;" ::: "memory");  // K and V staged (the whole warp takes part)
    if (lane == 0) {
      constexpr uint32_t idSP = tc::idesc_bf16(kRows, kChunk);                // S, dP': Q K^T, dO V^T
      constexpr uint32_t idDQ = tc::idesc_bf16(kRows, D, false, true);        // dq = dSq K   (K as MN-major B)
      constexpr uint32_t idKV = tc::idesc_bf16(kRows, kChunk, true, true);    // dV^T, dK^T  (both MN-major)
      // head-dim operands of M = 128 from the grouped Q / dO tiles: the second
      // 64-block of a group sits 1024 bytes further, 8-row groups 16 * D apart;
      // with D = 64 it repeats the first block (rows 64..127 are unused)
      constexpr uint32_t kMnQ = D == 128 ? 1024u : 0u;
      constexpr uint32_t kGrp = 16 * D;
      constexpr uint32_t kMnK = (uint32_t)kChunk * 128;
      const uint32_t kbase = smem_u32(sm.K), vbase = smem_u32(sm.V);
      const uint32_t pbase = smem_u32(sm.P), dsk = smem_u32(sm.dSk);
      tc::fence_after_sync();
      auto issue_SdP = [&](int i) {
        const int st = i & 1, sb = i & 1;
        tc::fence_after_sync();
        const uint32_t qb = smem_u32(sm.Q[st]), ob = smem_u32(sm.dO[st]);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t blk = kk >> 2, wq = kk & 3;
          const uint32_t ao = blk * 1024 + wq * 32, bo = blk * kChunk * 128 + wq * 32;
          tc::mma_bf16_ss(tmem + Cols<D>::S + sb * kChunk, tc::sdesc_sw128_sbo(qb + ao, kGrp),
                          tc::sdesc_sw128(kbase + bo), idSP, kk > 0);
          tc::mma_bf16_ss(tmem + Cols<D>::dP + sb * kChunk, tc::sdesc_sw128_sbo(ob + ao, kGrp),
                          tc::sdesc_sw128(vbase + bo), idSP, kk > 0);
        }
        tc::mma_commit(bar(BAR_S_FULL + sb));
      };
      auto issue_KV = [&](int i) {
        const int st = i & 1;
        tc::fence_after_sync();
        // dV^T += dO^T (wP), dK^T += Q^T dSk : M = head dim, N = 64, K = 128 rows
        const uint32_t qb = smem_u32(sm.Q[st]), ob = smem_u32(sm.dO[st]);
#pragma unroll
        for (int kk = 0; kk < kRows / 16; ++kk) {
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          tc::mma_bf16_ss(tmem + Cols<D>::dVt, tc::sdesc_sw128_mn(ob + kk * 2 * kGrp, kMnQ, kGrp),
                          tc::sdesc_sw128_mn(pbase + kk * 2048, 0), idKV, acc);
          tc::mma_bf16_ss(tmem + Cols<D>::dKt, tc::sdesc_sw128_mn(qb + kk * 2 * kGrp, kMnQ, kGrp),
                          tc::sdesc_sw128_mn(dsk + kk * 2048, 0), idKV, acc);
        }
        tc::mma_commit(bar(BAR_QD_EMPTY + st));
      };
      auto issue_DQ = [&]() {
        // dq' = dSk K : M = 128 rows, N = D, K = 64 chunk rows
#pragma unroll
        for (int kk = 0; kk < kChunk / 16; ++kk)
          tc::mma_bf16_ss(tmem + Cols<D>::dq, tc::sdesc_sw128(dsk + kk * 32),
                          tc::sdesc_sw128_mn(kbase + kk * 2048, kMnK), idDQ, kk > 0);
        tc::mma_commit(bar(BAR_DQ_FULL));
        tc::mma_commit(bar(BAR_P_EMPTY));
      };
      // Event loop: issue whichever is ready — S/dP' of step nS (tile landed,
      // accumulator buffer read), dK/dV of step nK (P tiles written) or dq of
      // step nQ (dq accumulator read). Neither barrier can run a phase past the
      // one polled before the corresponding issue, so parity polling is exact.
      int nS = 0, nK = 0, nQ = 0;
      tc::SpinLimit spin;
      while (nQ < niter) {
        bool progressed = false;
        if (nS < niter && nS < nQ + 2 && tc::mbar_test_wait(bar(BAR_QD_FULL + (nS & 1)), (nS >> 1) & 1) &&
            tc::mbar_test_wait(bar(BAR_S_EMPTY + (nS & 1)), ((nS >> 1) & 1) ^ 1)) {
          issue_SdP(nS++);
          progressed = true;
        }
        if (nK < nS && tc::mbar_test_wait(bar(BAR_P_FULL), nK & 1)) {
          issue_KV(nK++);
          progressed = true;
        }
        if (nQ < nK && tc::mbar_test_wait(bar(BAR_DQ_EMPTY), (nQ & 1) ^ 1)) {
          issue_DQ();
          ++nQ;
          progressed = true;
        }
        if (progressed) {
          spin.busy();
        } else if (!spin.idle(abort_flag, status)) {
          break;
        }
      }
      tc::mma_commit(bar(BAR_ACC_DONE));
    }
    __syncwarp();
  } else if (warp < 4 || warp >= 12) {
    // ---------------------------------------------------------------- softmax / gradient rows
    // Two threads per row: warps 0-3 take chunk positions 0-31 and warps
    // 12-15 positions 32-63 of the same rows (tensor-memory lanes); the row
    // maximum, sum and D are combined through shared memory, each pair of
    // warps meeting at its own named barrier.
    const int hf = warp >= 12 ? 1 : 0;
    const int r = (warp & 3) * 32 + lane;
    const int c0 = hf * 32;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const float inv_S = 1.f / (float)kChunk;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + (warp & 3)) : "memory"); };
    for (int i = 0; i < niter; ++i) {
      const int sb = i & 1, st = i & 1;
      tc::mbar_wait(bar(BAR_S_FULL + sb), (i >> 1) & 1, abort_flag, status);
      tc::fence_after_sync();
      float x[32], y[32];
      tc::tmem_ld32(tmem + lane_base + Cols<D>::S + sb * kChunk + c0, x);
      tc::tmem_ld32(tmem + lane_base + Cols<D>::dP + sb * kChunk + c0, y);
      tc::tmem_wait_ld();
      tc::fence_before_sync();
      tc::mbar_arrive(bar(BAR_S_EMPTY + sb));
      // the loader's slot tables of this tile (released with BAR_QD_FULL, whose
      // phase cannot advance before this thread has produced the step's P)
      tc::mbar_wait(bar(BAR_QD_FULL + st), (i >> 1) & 1, abort_flag, status);
      const int slot = r >> a.log2G;
      const float wv = sm.slot_w[st][slot], dl = sm.slot_delta[st][slot];
      const int pv = sm.slot_p[st][slot];
      float mx[8], zz[8], dd[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx[u] = x[u];
#pragma unroll
      for (int k = 8; k < 32; ++k) mx[k & 7] = fmaxf(mx[k & 7], x[k]);
      sm.xch[0][hf][r] =
          fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      pair_sync();
      const float ms = fmaxf(sm.xch[0][0][r], sm.xch[0][1][r]) * a.scale_log2;
#pragma unroll
      for (int u = 0; u < 8; ++u) zz[u] = 0.f;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        x[k] = exp2f(fmaf(x[k], a.scale_log2, -ms));
        zz[k & 7] += x[k];
      }
      sm.xch[1][hf][r] = ((zz[0] + zz[1]) + (zz[2] + zz[3])) + ((zz[4] + zz[5]) + (zz[6] + zz[7]));
      pair_sync();
      const float inv = 1.f / ((sm.xch[1][0][r] + sm.xch[1][1][r]) + (a.softmax1 ? exp2f(-ms) : 0.f));
#pragma unroll
      for (int u = 0; u < 8; ++u) dd[u] = 0.f;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        x[k] *= inv;
        dd[k & 7] = fmaf(x[k], y[k], dd[k & 7]);
      }
      sm.xch[2][hf][r] = ((dd[0] + dd[1]) + (dd[2] + dd[3])) + ((dd[4] + dd[5]) + (dd[6] + dd[7]));
      pair_sync();
      const float Drow = sm.xch[2][0][r] + sm.xch[2][1][r];
      float dw = Drow;  // sum over the G rows of the slot (consecutive lanes)
      for (int o = 1; o < a.G; o <<= 1) dw += __shfl_xor_sync(0xFFFFFFFFu, dw, o);
      // softmax weights: ds = w (dw - Δ), folded in here; stick-breaking weights
      // need every slot's dw first, so the slot's dw goes out and a later pass
      // adds the selection terms
      const float dsv = a.dw_mode ? 0.f : wv * (dw - dl);
      if (a.dw_mode && hf == 0 && (r & (a.G - 1)) == 0 && pv >= 0) a.dw_out[pv] = dw;
      // hand the slot id to the epilogue warps (three buffers: step i+3 runs
      // after S of step i+3, which the MMA thread issues only after the dq
      // product of step i+1, which waits for the epilogue of step i to have
      // read the dq accumulator, and so its slot ids)
      if (hf == 0) {
        sm.row_p[i % 3][r] = pv;
        tc::mbar_arrive(bar(BAR_DS_FULL + i % 3));
      }
      const float ca = a.scale_attn * wv, pool = a.scale_sel * dsv * inv_S;
      tc::mbar_wait(bar(BAR_P_EMPTY), (i & 1) ^ 1, abort_flag, status);
      const uint32_t prow = smem_u32(sm.P), krow = smem_u32(sm.dSk);
#pragma unroll
      for (int c16 = 0; c16 < 4; ++c16) {
        const uint32_t o = tc::sw128_offset(kRows, r, c0 + c16 * 8);
        uint32_t pp[4], gk[4];
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const int k0 = 8 * c16 + 2 * h;
          pp[h] = pack_bf16x2(wv * x[k0], wv * x[k0 + 1]);
          gk[h] = pack_bf16x2(fmaf(ca * x[k0], y[k0] - Drow, pool), fmaf(ca * x[k0 + 1], y[k0 + 1] - Drow, pool));
        }
        asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(prow + o), "r"(pp[0]), "r"(pp[1]), "r"(pp[2]),
                     "r"(pp[3]));
        asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(krow + o), "r"(gk[0]), "r"(gk[1]), "r"(gk[2]),
                     "r"(gk[3]));
      }
      tc::fence_proxy_async_smem();
      tc::mbar_arrive(bar(BAR_P_FULL));
    }
  } else {
    // ---------------------------------------------------------------- epilogue (thread = row, then head dim)
    const int r = tid - 128;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint64_t stream = tc::l2_evict_first();
    for (int j = 0; j < niter; ++j) {
      tc::mbar_wait(bar(BAR_DS_FULL + j % 3), (j / 3) & 1, abort_flag, status);
      const int pj = sm.row_p[j % 3][r];
      tc::mbar_wait(bar(BAR_DQ_FULL), j & 1, abort_flag, status);
      tc::fence_after_sync();
      uint16_t* dst = (!a.use_tma && pj >= 0) ? a.dqpart + ((long long)pj * a.G + (r & (a.G - 1))) * D : nullptr;
      // dq' in 64-column halves: each is read from tensor memory, written to the
      // staging atoms (one 1 KB atom per 8 rows, 128-byte swizzle) and stored by
      // the first lane of every 8-row group with one TMA box; the accumulator
      // is released once the last half has been read
      const uint32_t atom = smem_u32(sm.dqstage) + (warp & 3) * 4096 + (lane >> 3) * 1024;
      const uint32_t row = atom + (lane & 7) * 128, swz = lane & 7;
      const bool issuer = (lane & 7) == 0 && pj >= 0;
#pragma unroll
      for (int h = 0; h < D / 64; ++h) {
        float v[64];
        tc::tmem_ld32(tmem + lane_base + Cols<D>::dq + h * 64, *reinterpret_cast<float(*)[32]>(&v[0]));
        tc::tmem_ld32(tmem + lane_base + Cols<D>::dq + h * 64 + 32, *reinterpret_cast<float(*)[32]>(&v[32]));
        tc::tmem_wait_ld();
        if (h == D / 64 - 1) {
          tc::fence_before_sync();
          tc::mbar_arrive(bar(BAR_DQ_EMPTY));
        }
        if (a.use_tma) {
          if ((lane & 7) == 0) tc::bulk_wait_read();  // the previous round's boxes have left the atoms
          __syncwarp();
#pragma unroll
          for (int c8 = 0; c8 < 8; ++c8) {
            const float* o = &v[8 * c8];
            asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(row + ((c8 ^ swz) << 4)),
                         "r"(pack_bf16x2(o[0], o[1])), "r"(pack_bf16x2(o[2], o[3])), "r"(pack_bf16x2(o[4], o[5])),
                         "r"(pack_bf16x2(o[6], o[7])));
          }
          tc::fence_proxy_async_smem();
          __syncwarp();
          if (issuer) {
            tc::tma_store_2d_hint(&tmap_dq, h * 64, pj * a.G + (r & (a.G - 1)), atom, stream);
            tc::bulk_commit();
          }
        } else if (dst) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + h * 64);
#pragma unroll
          for (int q8 = 0; q8 < 8; ++q8) {
            const float* o = &v[8 * q8];
            d4[q8] = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]),
                                pack_bf16x2(o[6], o[7]));
          }
        }
      }
    }
    if (a.use_tma && (lane & 7) == 0) tc::bulk_wait_all();
    // dK, dV of the chunk: TMEM lane = head dim, column = chunk row
    tc::mbar_wait(bar(BAR_ACC_DONE), 0, abort_flag, status);
    tc::fence_after_sync();
    if ((warp & 3) * 32 < D) {
      const int dcol = r;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float dv[32], dk[32];
        tc::tmem_ld32(tmem + lane_base + Cols<D>::dVt + h * 32, dv);
        tc::tmem_ld32(tmem + lane_base + Cols<D>::dKt + h * 32, dk);
        tc::tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const long long o = (row0 + (long long)(h * 32 + k) * a.Hkv) * D + dcol;
          a.dV[o] = dv[k];
          a.dK[o] = dk[k];
        }
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 9) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// Δ_t = sum over the group's heads of dO · O (one warp per (b, t, g)).
template <int D>
__global__ void __launch_bounds__(256) bwd_delta_kernel(const uint16_t* __restrict__ O, const uint16_t* __restrict__ dO,
                                                        float* __restrict__ delta, long long n_rows, int G) {
  griddep_wait();
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

// Stick-breaking weights (§3.1.1): w_j = b_j R_j with R_j = prod_{i<j} (1 - b_i)
// = 1 - sum_{i<j} w_i, so b_j = w_j / R_j and
//   ds_j = (1 - b_j) w_j dw_j - b_j sum_{k>j} w_k dw_k = (w_j / R_j) (R_{j+1} dw_j - U_j),
// U_j = sum_{k>j} w_k dw_k. One thread per (b, t, g) row; R in double (a
// slot that finds almost no stick left has almost no weight, and its ds stays
// small whatever R's rounding).
//
// Softmax weights (the attention-only backward): ds_j = w_j (dw_j - sum_k w_k dw_k).
// accumulate: ds += (layers sharing one selection add their score gradients).
__global__ void __launch_bounds__(256) bwd_ds_kernel(const int32_t* __restrict__ idx, const float* __restrict__ w,
                                                     const float* __restrict__ dw, float* __restrict__ ds,
                                                     long long n_rows, int topk, int Nc, int stick, int accumulate,
                                                     unsigned* __restrict__ status) {
  griddep_wait();
  const long long row = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  int keff = 0;
  while (keff < topk) {
    const int c = idx[p0 + keff];
    if (c >= 0) bounds_ok(c, 0, Nc, status);  // debug: a chunk id past the sequence is reported
    if (c < 0 || c >= Nc) break;
    ++keff;
  }
  auto put = [&](int j, float v) { ds[p0 + j] = accumulate ? ds[p0 + j] + v : v; };
  for (int j = topk - 1; j >= keff; --j) put(j, 0.f);
  if (!stick) {
    double wdw = 0.0;
    for (int j = 0; j < keff; ++j) wdw += (double)w[p0 + j] * dw[p0 + j];
    for (int j = 0; j < keff; ++j) put(j, (float)(w[p0 + j] * (dw[p0 + j] - wdw)));
    return;
  }
  double R[32];
  double rest = 1.0;
  for (int j = 0; j < keff; ++j) {
    R[j] = rest;
    rest -= (double)w[p0 + j];
  }
  double U = 0.0;
  for (int j = keff - 1; j >= 0; --j) {
    const double wj = w[p0 + j], dwj = dw[p0 + j];
    put(j, R[j] > 0.0 ? (float)((wj / R[j]) * ((R[j] - wj) * dwj - U)) : 0.f);
    U += wj * dwj;
  }
}

// Selection chain into the group query: dq_sel[t, h] = c_sel sum_j ds_j K̄_{I_j}
// for every head h of the group (one warp per (b, t, g); every element written).
template <int D>
__global__ void __launch_bounds__(256) sel_dq_kernel(const int32_t* __restrict__ idx, const float* __restrict__ ds,
                                                     const float* __restrict__ kbar32, float* __restrict__ dq,
                                                     long long n_rows, int G, int topk, int Nc, int L, int Hkv,
                                                     float scale_sel, unsigned* __restrict__ status) {
  griddep_wait();
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  bool valid = false;
  int cl = 0;
  float sl = 0.f;
  if (lane < topk) {  // lane j holds slot j's chunk and scaled score gradient
    cl = idx[p0 + lane];
    valid = cl >= 0 && cl < Nc;
    if (cl >= 0) bounds_ok(cl, 0, Nc, status);
    sl = valid ? scale_sel * ds[p0 + lane] : 0.f;
  }
  const int keff = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const long long b = row / ((long long)L * Hkv);
  const int g = (int)(row % Hkv);
  float4* dst = reinterpret_cast<float4*>(dq) + row * G * (D / 4);
  for (int ch0 = 0; ch0 < G * (D / 8); ch0 += 32) {
    const int ch = ch0 + lane;
    const int e8 = ch % (D / 8);
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    for (int j = 0; j < keff; ++j) {
      const float sj = __shfl_sync(0xFFFFFFFFu, sl, j);
      const int cj = __shfl_sync(0xFFFFFFFFu, cl, j);
      if (ch >= G * (D / 8)) continue;
      const float4* kb = reinterpret_cast<const float4*>(kbar32 + ((b * Nc + cj) * Hkv + g) * D) + e8 * 2;
      const float4 k0 = kb[0], k1 = kb[1];
      acc[0] = fmaf(sj, k0.x, acc[0]);
      acc[1] = fmaf(sj, k0.y, acc[1]);
      acc[2] = fmaf(sj, k0.z, acc[2]);
      acc[3] = fmaf(sj, k0.w, acc[3]);
      acc[4] = fmaf(sj, k1.x, acc[4]);
      acc[5] = fmaf(sj, k1.y, acc[5]);
      acc[6] = fmaf(sj, k1.z, acc[6]);
      acc[7] = fmaf(sj, k1.w, acc[7]);
    }
    if (ch >= G * (D / 8)) continue;
    dst[2 * ch] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[2 * ch + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

// q̂ rows for the chunk-summary gradient: [b, t, g][e] = head-order fp32 sum
// of the group's query rows (the selection's group query).
template <int D>
__global__ void __launch_bounds__(256) bwd_qhat_kernel(const uint16_t* __restrict__ q, float* __restrict__ qhat,
                                                       long long n_rows, int G) {
  griddep_wait();
  constexpr int D8 = D / 8;
  const long long u = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= n_rows * D8) return;
  const long long row = u / D8;
  const int e8 = (int)(u % D8);
  const uint4* src = reinterpret_cast<const uint4*>(q) + row * G * D8 + e8;
  float acc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.f;
  for (int h = 0; h < G; ++h) {
    const uint4 v = src[(long long)h * D8];
    acc[0] += bf16_lo(v.x);
    acc[1] += bf16_hi(v.x);
    acc[2] += bf16_lo(v.y);
    acc[3] += bf16_hi(v.y);
    acc[4] += bf16_lo(v.z);
    acc[5] += bf16_hi(v.z);
    acc[6] += bf16_lo(v.w);
    acc[7] += bf16_hi(v.w);
  }
  float4* dst = reinterpret_cast<float4*>(qhat) + row * (D / 4) + e8 * 2;
  dst[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
  dst[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
}

// The chunk-summary gradient dK̄_i = c_sel sum over the slots that chose chunk
// i (from the inverse index) of ds * q̂_t, spread over the chunk's S key rows
// (mean pool): dK_{iS+s} += dK̄_i / S. Block per (b, g, chunk), in the chunk
// kernels' order (long lists first): kDkbarGroups groups of D threads (thread =
// dimension) take the entries n = group, group + kDkbarGroups, ... with eight
// loads in flight each, and the group sums are added in group order
// (deterministic).
constexpr int kDkbarGroups = 4;
template <int D>
__global__ void __launch_bounds__(D * kDkbarGroups, 2) bwd_stick_dkbar_kernel(const int32_t* __restrict__ offsets,
                                                                           const int32_t* __restrict__ entries,
                                                                           const float* __restrict__ ds,
                                                                           const float* __restrict__ qhat,
                                                                           float* __restrict__ dK, int L, int Hkv,
                                                                           int topk, int Nc, float scale_sel,
                                                                           long long n_slots,
                                                                           unsigned* __restrict__ status) {
  griddep_wait();
  __shared__ float part[kDkbarGroups][D];
  int c, bg;
  block_key(Nc, (int)(gridDim.x / (unsigned)Nc), c, bg);
  const int key = bg * Nc + c;
  const int b = bg / Hkv, g = bg % Hkv;
  const int off = offsets[key];
  int cnt = offsets[key + 1] - off;
  if (!(bounds_ok(off, 0, n_slots + 1, status) && bounds_ok(off + cnt, off, n_slots + 1, status)))
    cnt = 0;  // debug: a list outside the entries is skipped
  if (cnt <= 0) return;
  const int e = threadIdx.x % D, grp = threadIdx.x / D;
  const int slot_div = Hkv * topk;
  constexpr int kStep = kDkbarGroups;
  float acc = 0.f;
  int n = grp;
  for (; n + 7 * kStep < cnt; n += 8 * kStep) {  // eight slots' loads in flight
    int p[8];
    float dv[8], qv[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) p[u] = entries[off + n + u * kStep];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const bool ok = bounds_ok(p[u], 0, n_slots, status);  // debug: a slot id out of range adds nothing
      dv[u] = ok ? ds[p[u]] : 0.f;
      qv[u] = ok ? qhat[((long long)(p[u] / slot_div) * Hkv + g) * D + e] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) acc = fmaf(dv[u], qv[u], acc);
  }
  for (; n < cnt; n += kStep) {
    const int p = entries[off + n];
    if (bounds_ok(p, 0, n_slots, status)) acc = fmaf(ds[p], qhat[((long long)(p / slot_div) * Hkv + g) * D + e], acc);
  }
  part[grp][e] = acc;
  __syncthreads();
  if (grp != 0) return;
  float sum = part[0][e];
#pragma unroll
  for (int k = 1; k < kDkbarGroups; ++k) sum += part[k][e];
  const float add = scale_sel * sum / (float)kChunk;
  const long long row0 = ((long long)b * L + (long long)c * kChunk) * Hkv + g;
  for (int s = 0; s < kChunk; ++s) dK[(row0 + (long long)s * Hkv) * D + e] += add;
}

// dq_t = sum_j dq'_{t,j} in slot order (one warp per (b, t, g)); with
// stick-breaking weights also the selection term c_sel sum_j ds_j K̄_{I_j}
// for every head of the group.
template <int D>
__global__ void __launch_bounds__(256) bwd_dq_merge_kernel(const int32_t* __restrict__ idx,
                                                           const uint16_t* __restrict__ dqpart, float* __restrict__ dq,
                                                           long long n_rows, int G, int topk, int Nc,
                                                           const float* __restrict__ ds,
                                                           const float* __restrict__ kbar32, int L, int Hkv,
                                                           float scale_sel, unsigned* __restrict__ status) {
  griddep_wait();
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  bool valid = false;
  int cl = 0;
  float sl = 0.f;
  if (lane < topk) {  // lane j holds slot j's chunk (and, for the selection term, scaled ds)
    cl = idx[p0 + lane];
    valid = cl >= 0 && cl < Nc;
    if (cl >= 0) bounds_ok(cl, 0, Nc, status);
    if (ds != nullptr && valid) sl = scale_sel * ds[p0 + lane];
  }
  const int keff = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int GD8 = G * (D / 8);
  const uint4* src = reinterpret_cast<const uint4*>(dqpart) + p0 * GD8;
  float4* dst = reinterpret_cast<float4*>(dq) + row * GD8 * 2;
  for (int ch0 = 0; ch0 < GD8; ch0 += 32) {  // every lane runs every round (the slot broadcasts need the warp)
    const int ch = ch0 + lane;
    const bool active = ch < GD8;
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    for (int j = 0; j < keff && active; ++j) {
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
    if (ds != nullptr) {  // stick-breaking: c_sel sum_j ds_j K̄_{I_j}, dims [8 e8, 8 e8 + 8) of this head
      const int e8 = ch % (D / 8);
      const long long b = row / ((long long)L * Hkv);
      const int g = (int)(row % Hkv);
      for (int j = 0; j < keff; ++j) {
        const float sj = __shfl_sync(0xFFFFFFFFu, sl, j);
        const int cj = __shfl_sync(0xFFFFFFFFu, cl, j);
        if (!active) continue;
        const float4* kb = reinterpret_cast<const float4*>(kbar32 + ((b * Nc + cj) * Hkv + g) * D) + e8 * 2;
        const float4 k0 = kb[0], k1 = kb[1];
        acc[0] = fmaf(sj, k0.x, acc[0]);
        acc[1] = fmaf(sj, k0.y, acc[1]);
        acc[2] = fmaf(sj, k0.z, acc[2]);
        acc[3] = fmaf(sj, k0.w, acc[3]);
        acc[4] = fmaf(sj, k1.x, acc[4]);
        acc[5] = fmaf(sj, k1.y, acc[5]);
        acc[6] = fmaf(sj, k1.z, acc[6]);
        acc[7] = fmaf(sj, k1.w, acc[7]);
      }
    }
    if (!active) continue;
    dst[2 * ch] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    dst[2 * ch + 1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

// dK = dV = 0 on the rows of a trailing partial chunk.
__global__ void zero_tail_kernel(float* __restrict__ dK, float* __restrict__ dV, int B, int L, int tail0,
                                 long long row_elems) {
  griddep_wait();
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

// Workspace of a backward call: bf16 dq partials [slots, G, d]; the full
// backward with softmax weights Δ [rows]; whenever the chunk pass writes dw
// (stick-breaking weights, attention-only backward) dw [slots]; the full
// backward with stick-breaking weights also ds [slots] and q̂ [rows, d] fp32.
enum class BwdMode { kFull, kAttention };
struct BwdLayout {
  size_t dqpart, delta, dw, ds, qhat, total;
};
BwdLayout bwd_layout(const Dims& D, BwdMode mode) {
  const size_t rows = (size_t)D.B * D.L * D.Hkv;
  const bool full = mode == BwdMode::kFull;
  BwdLayout lo{};
  size_t o = 0;
  lo.dqpart = o;
  o = align256(o + (size_t)D.slots() * D.G * D.d * sizeof(uint16_t));
  if (full && !D.stick) {
    lo.delta = o;
    o = align256(o + rows * sizeof(float));
  }
  if (!full || D.stick) {
    lo.dw = o;
    o = align256(o + (size_t)D.slots() * sizeof(float));
  }
  if (full && D.stick) {
    lo.ds = o;
    o = align256(o + (size_t)D.slots() * sizeof(float));
    lo.qhat = o;
    o = align256(o + rows * D.d * sizeof(float));
  }
  lo.total = o;
  return lo;
}

template <int D>
cudaError_t launch_dkbar(const Dims& Dm, const void* q, const int32_t* offsets, const int32_t* entries, const float* ds,
                         float* qhat, float* dK, cudaStream_t st) {
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  cudaError_t e;
  (void)launch_dependent(bwd_qhat_kernel<D>, dim3((unsigned)((rows * (D / 8) + 255) / 256)), dim3(256), 0, st,
                         (const uint16_t*)q, qhat, rows, Dm.G);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const long long keys = Dm.keys();
  if (keys > 0) {
    (void)launch_dependent(bwd_stick_dkbar_kernel<D>, dim3((unsigned)keys), dim3(D * kDkbarGroups), 0, st, offsets,
                           entries, ds, qhat, dK, Dm.L, Dm.Hkv, Dm.topk, Dm.Nc, Dm.scale_sel, Dm.slots(), Dm.status);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// kFull: dq, dK, dV including the selection chain (q and K are also the
// selection's inputs). kAttention: dq, dK, dV of the attention alone, and the
// slots' score gradients added into ds_acc.
template <int D>
cudaError_t run(const Dims& Dm, BwdMode mode, const void* q, const void* K, const void* V, const float* kbar32,
                const int32_t* idx, const float* w, const void* O, const void* dO, const int32_t* offsets,
                const int32_t* entries, float* dq, float* dK, float* dV, float* ds_acc, void* ws, cudaStream_t st) {
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  const bool full = mode == BwdMode::kFull;
  const bool dw_mode = !full || Dm.stick;
  const BwdLayout lo = bwd_layout(Dm, mode);
  uint16_t* dqpart = (uint16_t*)((char*)ws + lo.dqpart);
  float* delta = full && !Dm.stick ? (float*)((char*)ws + lo.delta) : nullptr;
  float* dwb = dw_mode ? (float*)((char*)ws + lo.dw) : nullptr;
  float* dsb = full && Dm.stick ? (float*)((char*)ws + lo.ds) : ds_acc;
  float* qhat = full && Dm.stick ? (float*)((char*)ws + lo.qhat) : nullptr;
  cudaError_t e;
  if (delta != nullptr) {  // Δ_t = sum_j w_j dw_j = dO · O feeds the softmax weights' ds inside the chunk kernel
    (void)launch_dependent(bwd_delta_kernel<D>, dim3((unsigned)((rows + 7) / 8)), dim3(256), 0, st, (const uint16_t*)O,
                           (const uint16_t*)dO, delta, rows, Dm.G);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  const long long keys = Dm.keys();
  if (keys > 0) {
    BwdArgs a;
    a.q = (const uint16_t*)q;
    a.K = (const uint16_t*)K;
    a.V = (const uint16_t*)V;
    a.dO = (const uint16_t*)dO;
    a.w = w;
    a.delta = delta != nullptr ? delta : w;  // read by the loader; unused when dw_mode
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
    a.softmax1 = Dm.softmax1 ? 1 : 0;
    a.dw_mode = dw_mode ? 1 : 0;
    a.dw_out = dwb;
    a.status = Dm.status;
    const size_t smem = sizeof(BwdSmem<D>) + 1024;
    if ((e = cudaFuncSetAttribute(bwd_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
        cudaSuccess)
      return e;
    CUtensorMap tq, tdo, tdq;
    memset(&tq, 0, sizeof(tq));
    memset(&tdo, 0, sizeof(tdo));
    memset(&tdq, 0, sizeof(tdq));
    a.n_rows = Dm.B * Dm.L * Dm.Hq;
    a.n_slots = Dm.slots();
    a.use_tma = Dm.G >= 8 ? 1 : 0;
    if (a.use_tma && (!tc::make_group8_tmap(&tq, q, (unsigned long long)a.n_rows, D) ||
                      !tc::make_group8_tmap(&tdo, dO, (unsigned long long)a.n_rows, D) ||
                      !tc::make_rows_tmap(&tdq, dqpart, (unsigned long long)Dm.slots() * Dm.G, D, 8)))
      return cudaErrorNotSupported;
    (void)launch_dependent(bwd_chunk_kernel<D>, dim3((unsigned)keys), dim3(kThreads), smem, st, a, tq, tdo, tdq);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (dw_mode) {
    (void)launch_dependent(bwd_ds_kernel, dim3((unsigned)((rows + 255) / 256)), dim3(256), 0, st, idx, w, dwb, dsb,
                           rows, Dm.topk, Dm.Nc, Dm.stick ? 1 : 0, full ? 0 : 1, Dm.status);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (full && (e = launch_dkbar<D>(Dm, q, offsets, entries, dsb, qhat, dK, st)) != cudaSuccess) return e;
  }
  const bool sel_term = full && Dm.stick;
  (void)launch_dependent(bwd_dq_merge_kernel<D>, dim3((unsigned)((rows + 7) / 8)), dim3(256), 0, st, idx, dqpart, dq,
                         rows, Dm.G, Dm.topk, Dm.Nc, sel_term ? dsb : nullptr, kbar32, Dm.L, Dm.Hkv, Dm.scale_sel,
                         Dm.status);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int tail0 = Dm.Nc * kChunk;
  if (tail0 < Dm.L && Dm.B > 0) {
    const long long total = (long long)Dm.B * (Dm.L - tail0) * Dm.Hkv * D;
    (void)launch_dependent(zero_tail_kernel, dim3(grid_cap((total + 255) / 256, 152LL * 8)), dim3(256), 0, st, dK, dV,
                           Dm.B, Dm.L, tail0, (long long)Dm.Hkv * D);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// The selection chain for a given score gradient: dq_sel (every element), dK_sel
// (zeroed, then the mean-pool share of dK̄ on every complete chunk's rows).
template <int D>
cudaError_t run_select_backward(const Dims& Dm, const void* q_sel, const float* kbar_sel, const int32_t* idx,
                                const float* ds, const int32_t* offsets, const int32_t* entries, float* dq_sel,
                                float* dK_sel, void* ws, cudaStream_t st) {
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  cudaError_t e;
  if ((e = cudaMemsetAsync(dK_sel, 0, (size_t)rows * D * sizeof(float), st)) != cudaSuccess) return e;
  (void)launch_dependent(sel_dq_kernel<D>, dim3((unsigned)((rows + 7) / 8)), dim3(256), 0, st, idx, ds, kbar_sel,
                         dq_sel, rows, Dm.G, Dm.topk, Dm.Nc, Dm.L, Dm.Hkv, Dm.scale_sel, Dm.status);
  note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  return launch_dkbar<D>(Dm, q_sel, offsets, entries, ds, (float*)ws, dK_sel, st);
}

}  // namespace

size_t backward_workspace(const Dims& D) { return bwd_layout(D, BwdMode::kFull).total; }
size_t backward_attention_workspace(const Dims& D) { return bwd_layout(D, BwdMode::kAttention).total; }
size_t select_backward_workspace(const Dims& D) { return align256((size_t)D.B * D.L * D.Hkv * D.d * sizeof(float)); }

cudaError_t launch_backward(const Dims& D, const void* q, const void* K, const void* V, const float* kbar32,
                            const int32_t* idx, const float* w, const void* O, const void* dO,
                            const int32_t* offsets, const int32_t* entries, float* dq, float* dK, float* dV,
                            void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, BwdMode::kFull, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq, dK, dV, nullptr,
                             ws, st)
                   : run<128>(D, BwdMode::kFull, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq, dK, dV,
                              nullptr, ws, st);
}

cudaError_t launch_backward_attention(const Dims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                                      const float* w, const void* dO, const int32_t* offsets,
                                      const int32_t* entries, float* dq, float* dK, float* dV, float* ds_acc,
                                      void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, BwdMode::kAttention, q, K, V, nullptr, idx, w, nullptr, dO, offsets, entries, dq, dK,
                             dV, ds_acc, ws, st)
                   : run<128>(D, BwdMode::kAttention, q, K, V, nullptr, idx, w, nullptr, dO, offsets, entries, dq,
                              dK, dV, ds_acc, ws, st);
}

cudaError_t launch_select_backward(const Dims& D, const void* q_sel, const float* kbar_sel, const int32_t* idx,
                                   const float* ds, const int32_t* offsets, const int32_t* entries, float* dq_sel,
                                   float* dK_sel, void* ws, cudaStream_t st) {
  return D.d == 64 ? run_select_backward<64>(D, q_sel, kbar_sel, idx, ds, offsets, entries, dq_sel, dK_sel, ws, st)
                   : run_select_backward<128>(D, q_sel, kbar_sel, idx, ds, offsets, entries, dq_sel, dK_sel, ws, st);
}

}  // namespace hsa
