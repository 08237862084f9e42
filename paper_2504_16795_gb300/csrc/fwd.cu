// Hierarchical attention forward (§3.1.1 "Hierarchical Attention", Algorithm 1),
// organised chunk-major instead of token-major.
//
// Algorithm 1 gives every token its own program that loads the k selected K/V
// chunks. Here every (b, g, chunk) is one block: the chunk's 64 x d K and V
// tiles are staged in shared memory once, and the block streams the query
// rows of every selection slot that chose the chunk (from the inverse index),
// 128 rows (= 128/G slots of G heads) per step, through two small dense
// tensor-core products: S = Q K^T (128 x 64 x d) and O' = softmax(S) V
// (128 x d x 64), the probabilities going back into tensor memory as the A
// operand of the second product (no shared-memory round trip). Each chunk is complete, so its softmax needs no online
// rescaling. The normalised per-slot result O' (bf16) goes to a workspace
// and a second kernel forms O_t = sum_j w_j O'_{t,j} with the chunk weights
// w = softmax_j(s_sel) (the "w/o s.b." variant of §4.1) or, with the
// stick-breaking flag, the paper's stick-breaking weights over I' (§3.1.1),
// slots in order j. The softmax-off-by-one flag (§3.1.2) adds the zero logit
// to every chunk-local softmax.
//
// A chunk that many tokens selected (a chunk every needle query selects has
// thousands of slots) would make one block run for milliseconds while the
// other SMs idle. Each slot's result is independent of the others, so a
// chunk's slot list is cut into segments of at most kSegTiles steps and every
// segment is its own block (the chunk's K and V are staged by each of them).
// A one-block pass lists the segments in the chunk order of block_key.
#include <cstring>

#include "tc.cuh"

namespace hsa {
namespace {

constexpr int kRows = 128;     // query rows per step (tensor-core M)
constexpr int kQStages = 3;    // gathered query tiles in flight
constexpr int kThreads = 384;  // warps 0-3 softmax, 4-7 epilogue, 8, 10, 11 loaders, 9 MMA
constexpr int kLoaders = 3;    // a TMA issue costs the issuing warp tens of ns per box: spread the boxes
constexpr int kTmemCols = 512;
constexpr int kSegTiles = 128;  // longest segment of a chunk's slot list, in 128-row steps

template <int D>
struct FwdSmem {
  uint16_t Q[kQStages][kRows * D];  // gathered query rows, grouped K-major SW128 (tc::grp_offset)
  uint16_t K[kChunk * D];           // chunk keys [s][d]
  uint16_t V[kChunk * D];           // chunk values [s][d] (read MN-major by the second product)
  uint16_t Ostage[2][kRows * D];    // TMA path: a step's O' rows (grouped layout) on their way out, two steps
  int slot_row[kQStages][kRows];    // cp.async path: first q row of each slot (-1: past the list)
  uint64_t bar[16];
  uint32_t tmem_base;
  int abort_flag;
};

// one block per SM: the layout plus the 1024-byte alignment slack must fit the 227 KB opt-in limit
static_assert(sizeof(FwdSmem<128>) + 1024 <= 232448, "shared memory layout too large");

enum {
  BAR_Q_FULL = 0,   // 3: tile landed
  BAR_Q_EMPTY = 3,  // 3: S MMA of the tile finished (commit)
  BAR_S_FULL = 6,   // 2: S accumulator ready (commit)
  BAR_S_EMPTY = 8,  // 2: S read by the softmax warps (128 arrivals)
  BAR_P_FULL = 10,  // 2: P written to tensor memory (128 arrivals)
  BAR_O_FULL = 12,  // 2: O accumulator ready (commit)
  BAR_O_EMPTY = 14  // 2: O read by the epilogue warps (128 arrivals)
};

struct FwdArgs {
  const uint16_t* q;
  const uint16_t* K;
  const uint16_t* V;
  const int4* segs;  // per block: (key, first entry, end entry, 0)
  const int* nseg;   // number of segments (blocks past it exit)
  const int32_t* entries;
  uint16_t* Opart;  // [slots, G, D]
  int L, Hq, Hkv, G, log2G, topk, Nc;
  int n_rows;   // B * L * Hq (query rows; a row index past it reads zeros)
  long long n_slots;  // B * L * Hkv * topk (slot ids; debug builds check entries against it)
  int use_tma;  // G >= 8: each slot's G rows arrive as one swizzled TMA box
  float scale_log2;  // c_att * log2(e)
  int softmax1;      // softmax-off-by-one inside the chunk
  unsigned* status;  // the call's status word (a bounded wait that gives up sets it)
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    fwd_chunk_kernel(FwdArgs a, const __grid_constant__ CUtensorMap tmap_q, const __grid_constant__ CUtensorMap tmap_o) {
  griddep_wait();
  extern __shared__ unsigned char smem_raw[];
  FwdSmem<D>& sm = *reinterpret_cast<FwdSmem<D>*>(smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u));
  constexpr int D8 = D / 8;
  constexpr uint32_t kColP = 2 * kChunk + 2 * D;  // tensor memory: S x2 | O' x2 | P x2 (32 columns each)
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if ((int)blockIdx.x >= *a.nseg) return;
  const int4 seg = a.segs[blockIdx.x];
  const int key = seg.x;
  const int bg = key / a.Nc, c = key % a.Nc;
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int off = seg.y;
  const int cnt = seg.z - seg.y;
  if (cnt <= 0) return;
  const int epi = kRows >> a.log2G;  // slots per step
  const int niter = (cnt + epi - 1) / epi;
  const int slot_div = a.Hkv * a.topk;
  auto bar = [&](int i) { return smem_u32(&sm.bar[i]); };
  volatile int* abort_flag = &sm.abort_flag;
  unsigned* status = a.status;

  if (tid == 0) {
    for (int i = 0; i < 3; ++i) {
      tc::mbar_init(bar(BAR_Q_FULL + i), a.use_tma ? kLoaders : 32);
      tc::mbar_init(bar(BAR_Q_EMPTY + i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(bar(BAR_S_FULL + i), 1);
      tc::mbar_init(bar(BAR_S_EMPTY + i), 128);
      tc::mbar_init(bar(BAR_P_FULL + i), 128);
      tc::mbar_init(bar(BAR_O_FULL + i), 1);
      tc::mbar_init(bar(BAR_O_EMPTY + i), 128);
    }
    sm.abort_flag = 0;
    tc::fence_mbar_init();
  }
  if (warp == 9) tc::tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sm.tmem_base;
  // chunk K and V ([s][d], 128-byte swizzle), once per block, by warps 0-7
  // while the loaders already gather the first query tiles; the MMA warp
  // meets them at named barrier 1 before its first product
  if (warp < 8) {
    const long long row0 = ((long long)b * a.L + (long long)c * kChunk) * a.Hkv + g;
    for (int u = tid; u < kChunk * D8; u += 256) {
      const int srow = u / D8, ch = u % D8;
      const long long src = (row0 + (long long)srow * a.Hkv) * D + ch * 8;
      cp_async16(smem_u32(sm.K) + tc::sw128_offset(kChunk, srow, ch * 8), a.K + src);
      cp_async16(smem_u32(sm.V) + tc::sw128_offset(kChunk, srow, ch * 8), a.V + src);
    }
    cp_async_commit();
    cp_async_wait<0>();
    tc::fence_proxy_async_smem();
    asm volatile("bar.arrive 1, 288;" ::: "memory");
  }

  if (warp == 8 || warp >= 10) {
    // ---------------------------------------------------------------- loader warps
    // TMA path: loader li (warps 8, 10, 11) gathers the slots li, li + 3, ...
    // of every tile, lane l slot li + 3 l. The slot ids of a tile are loaded
    // two tiles ahead and turned into query rows one tile ahead, so no
    // dependent global load sits on the loader's critical path. The cp.async
    // path runs on warp 8 alone.
    const int li = warp == 8 ? 0 : warp - 9;
    if (li == 0 || a.use_tma) {
      const int my_slot = li + kLoaders * lane;
      const int my_slots = (epi - li + kLoaders - 1) / kLoaders;
      const uint64_t keep = tc::l2_evict_last();
      auto load_p = [&](int i) {
        const int e = i * epi + my_slot;
        const int p = (a.use_tma && my_slot < epi && e < cnt) ? a.entries[off + e] : -1;
        return p < 0 || bounds_ok(p, 0, a.n_slots, status) ? p : -1;
      };
      auto row_of = [&](int p) {  // past the list: rows past the tensor read zeros
        return p < 0 ? a.n_rows : ((b * a.L + (p / slot_div) % a.L) * a.Hq) + g * a.G;
      };
      int p_cur = load_p(0), p_next = load_p(1);
      for (int i = 0; i < niter; ++i) {
        const int st = i % kQStages;
        const int y = row_of(p_cur);
        p_cur = p_next;
        p_next = load_p(i + 2);
        tc::mbar_wait(bar(BAR_Q_EMPTY + st), ((i / kQStages) & 1) ^ 1, abort_flag, status);
        const uint32_t base = smem_u32(sm.Q[st]);
        if (a.use_tma) {
          // one box per 8-row group of the lane's slot; each loader's expected
          // arrival carries its byte count
          if (my_slot < epi) {
            for (int j = 0; j < (a.G >> 3); ++j)
              tc::tma_load_3d_hint(base + (my_slot * (a.G >> 3) + j) * (16 * D), &tmap_q, 0, y + 8 * j, 0,
                                   bar(BAR_Q_FULL + st), keep);
          }
          if (lane == 0) tc::mbar_arrive_expect_tx(bar(BAR_Q_FULL + st), my_slots * a.G * D * 2);
          continue;
        }
        for (int sl = lane; sl < epi; sl += 32) {
          const int e = i * epi + sl;
          int row = -1;
          if (e < cnt) {
            const int p = a.entries[off + e];
            if (bounds_ok(p, 0, a.n_slots, status)) {
              const int t = (p / slot_div) % a.L;
              row = ((b * a.L + t) * a.Hq) + g * a.G;
            }
          }
          sm.slot_row[st][sl] = row;
        }
        __syncwarp();
        for (int u = lane; u < kRows * D8; u += 32) {
          const int r = u / D8, ch = u % D8;
          const int row = sm.slot_row[st][r >> a.log2G];
          const uint32_t dst = base + tc::grp_offset(D, r, ch * 8);
          if (row >= 0) {
            cp_async16(dst, a.q + ((long long)(row + (r & (a.G - 1)))) * D + ch * 8);
          } else {
            asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};\n" ::"r"(dst), "r"(0));
          }
        }
        cp_async_commit();
        if (i >= 1) {
          cp_async_wait<1>();
          tc::fence_proxy_async_smem();
          tc::mbar_arrive(bar(BAR_Q_FULL + (i - 1) % kQStages));
        }
      }
      if (!a.use_tma) {
        cp_async_wait<0>();
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(bar(BAR_Q_FULL + (niter - 1) % kQStages));
      }
    }
  } else if (warp == 9) {
    // ---------------------------------------------------------------- MMA issue (one thread)
    asm volatile("bar.sync 1, 288;" ::: "memory");  // K and V staged (the whole warp takes part)
    if (lane == 0) {
      constexpr uint32_t idS = tc::idesc_bf16(kRows, kChunk);
      constexpr uint32_t idO = tc::idesc_bf16(kRows, D, false, true);  // V as the MN-major B operand
      constexpr uint32_t kMnV = (uint32_t)kChunk * 128;                  // 64-column blocks of V
      const uint32_t kbase = smem_u32(sm.K), vbase = smem_u32(sm.V);
      tc::fence_after_sync();
      auto issue_S = [&](int i) {
        const int st = i % kQStages, sb = i & 1;
        tc::fence_after_sync();
        const uint32_t qbase = smem_u32(sm.Q[st]);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t blk = kk >> 2, w = kk & 3;
          tc::mma_bf16_ss(tmem + sb * kChunk, tc::sdesc_sw128_sbo(qbase + blk * 1024 + w * 32, 16 * D),
                          tc::sdesc_sw128(kbase + blk * kChunk * 128 + w * 32), idS, kk > 0);
        }
        tc::mma_commit(bar(BAR_S_FULL + sb));
        tc::mma_commit(bar(BAR_Q_EMPTY + st));
      };
      auto issue_O = [&](int i) {
        const int pb = i & 1;
        tc::fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kChunk / 16; ++kk)
          tc::mma_bf16_ts(tmem + 2 * kChunk + pb * D, tmem + kColP + pb * (kChunk / 2) + kk * 8,
                          tc::sdesc_sw128_mn(vbase + kk * 2048, kMnV), idO, kk > 0);
        tc::mma_commit(bar(BAR_O_FULL + pb));
      };
      // Event loop: issue S of step nS (tile landed, S buffer read) or O of step
      // nO (P written, O buffer read), whichever is ready. Neither barrier can
      // run a phase past the polled one before the corresponding issue.
      int nS = 0, nO = 0;
      tc::SpinLimit spin;
      while (nO < niter) {
        bool progressed = false;
        if (nS < niter && nS < nO + 2 && tc::mbar_test_wait(bar(BAR_Q_FULL + nS % kQStages), (nS / kQStages) & 1) &&
            tc::mbar_test_wait(bar(BAR_S_EMPTY + (nS & 1)), ((nS >> 1) & 1) ^ 1)) {
          issue_S(nS++);
          progressed = true;
        }
        if (nO < nS && tc::mbar_test_wait(bar(BAR_P_FULL + (nO & 1)), (nO >> 1) & 1) &&
            tc::mbar_test_wait(bar(BAR_O_EMPTY + (nO & 1)), ((nO >> 1) & 1) ^ 1)) {
          issue_O(nO++);
          progressed = true;
        }
        if (progressed) {
          spin.busy();
        } else if (!spin.idle(abort_flag, status)) {
          break;
        }
      }
    }
    __syncwarp();
  } else if (warp < 4) {
    // ---------------------------------------------------------------- softmax (thread = row)
    const int r = tid;
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    for (int i = 0; i < niter; ++i) {
      const int sb = i & 1;
      tc::mbar_wait(bar(BAR_S_FULL + sb), (i >> 1) & 1, abort_flag, status);
      tc::fence_after_sync();
      float x[64];
      tc::tmem_ld32(tmem + lane_base + sb * kChunk, *reinterpret_cast<float(*)[32]>(&x[0]));
      tc::tmem_ld32(tmem + lane_base + sb * kChunk + 32, *reinterpret_cast<float(*)[32]>(&x[32]));
      tc::tmem_wait_ld();
      tc::fence_before_sync();
      tc::mbar_arrive(bar(BAR_S_EMPTY + sb));
      float mx[8], zz[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx[u] = x[u];
#pragma unroll
      for (int k = 8; k < 64; ++k) mx[k & 7] = fmaxf(mx[k & 7], x[k]);
      const float m = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])), fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      const float ms = m * a.scale_log2;
#pragma unroll
      for (int u = 0; u < 8; ++u) zz[u] = 0.f;
#pragma unroll
      for (int k = 0; k < 64; ++k) {
        x[k] = exp2f(fmaf(x[k], a.scale_log2, -ms));
        zz[k & 7] += x[k];
      }
      // softmax-off-by-one: the zero logit adds exp(0 - max) to the denominator
      const float inv = 1.f / ((((zz[0] + zz[1]) + (zz[2] + zz[3])) + ((zz[4] + zz[5]) + (zz[6] + zz[7]))) +
                               (a.softmax1 ? exp2f(-ms) : 0.f));
      // P into tensor memory: the row's 64 probabilities as 32 bf16 pairs
      uint32_t pk[kChunk / 2];
#pragma unroll
      for (int k2 = 0; k2 < kChunk / 2; ++k2) pk[k2] = pack_bf16x2(x[2 * k2] * inv, x[2 * k2 + 1] * inv);
      tc::tmem_st32(tmem + lane_base + kColP + sb * (kChunk / 2), pk);
      tc::tmem_wait_st();
      tc::fence_before_sync();
      tc::mbar_arrive(bar(BAR_P_FULL + sb));
    }
  } else {
    // ---------------------------------------------------------------- epilogue (thread = row)
    const int r = tid - 128;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    // TMA path (G >= 8): each warp writes its 32 rows into the staging tile
    // (swizzled, conflict-free) and the first lane of every slot stores the
    // slot's G rows with one TMA box per 8 rows. Otherwise rows go out directly.
    const bool issuer = a.use_tma && (r & (a.G - 1)) == 0;
    const uint64_t stream = tc::l2_evict_first();
    auto entry = [&](int e) {  // slot id of list entry e (-1 past the list, or out of range)
      const int p = e < cnt ? a.entries[off + e] : -1;
      return p < 0 || bounds_ok(p, 0, a.n_slots, status) ? p : -1;
    };
    int p_next = entry(r >> a.log2G);
    for (int j = 0; j < niter; ++j) {
      const int pj = p_next;
      const int en = (j + 1) * epi + (r >> a.log2G);
      p_next = entry(en);  // prefetch the next step's slot
      const int ob = j & 1;
      const uint32_t stage = smem_u32(sm.Ostage[ob]);
      if (a.use_tma) {  // the stores of step j-2 have read this warp's part of the staging tile
        if (issuer) tc::bulk_wait_read_but1();
        __syncwarp();
      }
      tc::mbar_wait(bar(BAR_O_FULL + ob), (j >> 1) & 1, abort_flag, status);
      tc::fence_after_sync();
      uint16_t* dst = (!a.use_tma && pj >= 0) ? a.Opart + ((long long)pj * a.G + (r & (a.G - 1))) * D : nullptr;
#pragma unroll
      for (int h = 0; h < D / 64; ++h) {  // 64 columns per tensor-memory wait
        float o[64];
        tc::tmem_ld32(tmem + lane_base + 2 * kChunk + ob * D + h * 64, *reinterpret_cast<float(*)[32]>(&o[0]));
        tc::tmem_ld32(tmem + lane_base + 2 * kChunk + ob * D + h * 64 + 32, *reinterpret_cast<float(*)[32]>(&o[32]));
        tc::tmem_wait_ld();
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
          const uint4 v = make_uint4(pack_bf16x2(o[8 * q4], o[8 * q4 + 1]), pack_bf16x2(o[8 * q4 + 2], o[8 * q4 + 3]),
                                     pack_bf16x2(o[8 * q4 + 4], o[8 * q4 + 5]),
                                     pack_bf16x2(o[8 * q4 + 6], o[8 * q4 + 7]));
          if (a.use_tma) {
            asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(stage + tc::grp_offset(D, r, h * 64 + 8 * q4)),
                         "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w));
          } else if (dst) {
            reinterpret_cast<uint4*>(dst + h * 64)[q4] = v;
          }
        }
      }
      tc::fence_before_sync();
      tc::mbar_arrive(bar(BAR_O_EMPTY + ob));
      if (a.use_tma) {
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (issuer) {  // one bulk group per step, empty past the list, so "all but the last" means step j-2
          if (pj >= 0)
            for (int jj = 0; jj < (a.G >> 3); ++jj)
              tc::tma_store_3d_hint(&tmap_o, 0, pj * a.G + 8 * jj, 0, stage + ((r >> 3) + jj) * (16 * D), stream);
          tc::bulk_commit();
        }
      }
    }
    if (issuer) tc::bulk_wait_all();
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 9) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// The segments of every chunk's slot list, chunks in the order of block_key
// (key i of that order = the key block i would take), each list cut into
// pieces of seg_slots entries. One block of 1024 threads, one scan: thread t
// takes the run of keys [t * per, (t + 1) * per) of that order, counts their
// segments, and after a block-wide exclusive scan writes them.
__device__ __forceinline__ int key_in_order(int i, int Nc, int n_bg) {
  const int head = min(kHeadChunks, Nc);
  int c, bg;
  if (i < head * n_bg) {
    c = i / n_bg;
    bg = i % n_bg;
  } else {
    const int r = i - head * n_bg, rest = Nc - head;
    bg = r / rest;
    c = head + r % rest;
  }
  return bg * Nc + c;
}
__global__ void __launch_bounds__(1024) fwd_segments_kernel(const int32_t* __restrict__ offsets, int Nc, int n_bg,
                                                            int seg_slots, int4* __restrict__ segs,
                                                            int* __restrict__ nseg, long long n_slots,
                                                            unsigned* __restrict__ status) {
  griddep_wait();
  __shared__ int warp_sum[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int keys = Nc * n_bg;
  const int per = (keys + 1023) / 1024;
  const int i0 = min(tid * per, keys), i1 = min(i0 + per, keys);
  int n = 0;
  for (int i = i0; i < i1; ++i) {
    const int key = key_in_order(i, Nc, n_bg);
    int o0 = offsets[key], o1 = offsets[key + 1];
    if (!(bounds_ok(o0, 0, n_slots + 1, status) && bounds_ok(o1, o0, n_slots + 1, status))) o1 = o0;  // debug: skip
    const int len = o1 - o0;
    n += len > 0 ? (len + seg_slots - 1) / seg_slots : 0;
  }
  int x = n;  // inclusive scan within the warp
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int v = warp_sum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, v, o);
      if (lane >= o) v += y;
    }
    warp_sum[lane] = v;  // inclusive over warps
  }
  __syncthreads();
  int pos = (warp > 0 ? warp_sum[warp - 1] : 0) + x - n;
  for (int i = i0; i < i1; ++i) {
    const int key = key_in_order(i, Nc, n_bg);
    int o0 = offsets[key], o1 = offsets[key + 1];
    if (!(bounds_ok(o0, 0, n_slots + 1, nullptr) && bounds_ok(o1, o0, n_slots + 1, nullptr))) o1 = o0;
    for (int e = o0; e < o1; e += seg_slots) segs[pos++] = make_int4(key, e, min(e + seg_slots, o1), 0);
  }
  if (tid == 1023) *nseg = warp_sum[31];
}

// O_t = sum_j w_j O'_{t,j}; w = softmax over the selected scores or stick-breaking. One warp per (b, t, g).
template <int D>
__global__ void __launch_bounds__(256, 4) fwd_merge_kernel(const float* __restrict__ s_sel,
                                                        const int32_t* __restrict__ idx,
                                                        const uint16_t* __restrict__ Opart, uint16_t* __restrict__ O,
                                                        float* __restrict__ w, long long n_rows, int Hkv, int G,
                                                        int topk, int Nc, int stick, unsigned* __restrict__ status) {
  griddep_wait();
  const int lane = threadIdx.x & 31;
  const long long row = (long long)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const long long p0 = row * topk;
  bool valid = false;
  float s = -INFINITY;
  if (lane < topk) {
    const int c = idx[p0 + lane];
    valid = c >= 0 && c < Nc;
    if (c >= 0) bounds_ok(c, 0, Nc, status);  // debug: a chunk id past the memory is reported
    if (valid) s = s_sel[p0 + lane];
  }
  const float wj = warp_chunk_weight(s, valid, stick != 0);
  if (lane < topk) w[p0 + lane] = wj;
  const int keff = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int GD8 = G * (D / 8);
  const uint4* src = reinterpret_cast<const uint4*>(Opart) + p0 * GD8;
  uint4* dst = reinterpret_cast<uint4*>(O) + row * GD8;  // heads of group g are contiguous in O
  // every lane runs every iteration (the weight broadcast needs the full warp);
  // lanes past the row's last 16-byte chunk only skip the memory accesses.
  // Slots go in batches of kMergeBatch: their weights are broadcast first, then
  // all their partial rows are requested, then summed in slot order.
  constexpr int kMergeBatch = 4;
  for (int base = 0; base < GD8; base += 32) {
    const int ch = base + lane;
    const bool active = ch < GD8;
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    for (int j0 = 0; j0 < keff; j0 += kMergeBatch) {
      float wb[kMergeBatch];
      uint4 v[kMergeBatch];
#pragma unroll
      for (int u = 0; u < kMergeBatch; ++u) {
        const int j = j0 + u;
        wb[u] = __shfl_sync(0xFFFFFFFFu, wj, j & 31);
        v[u] = (active && j < keff) ? src[(long long)j * GD8 + ch] : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kMergeBatch; ++u) {
        if (j0 + u < keff) {
          acc[0] += wb[u] * bf16_lo(v[u].x);
          acc[1] += wb[u] * bf16_hi(v[u].x);
          acc[2] += wb[u] * bf16_lo(v[u].y);
          acc[3] += wb[u] * bf16_hi(v[u].y);
          acc[4] += wb[u] * bf16_lo(v[u].z);
          acc[5] += wb[u] * bf16_hi(v[u].z);
          acc[6] += wb[u] * bf16_lo(v[u].w);
          acc[7] += wb[u] * bf16_hi(v[u].w);
        }
      }
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

inline size_t align256f(size_t x) { return (x + 255) & ~(size_t)255; }

// Forward workspace: the bf16 partials [slots, G, d], then the segment list
// (at most one segment per key plus one per seg_slots entries) and its count.
struct FwdLayout {
  size_t segs, nseg, total;
  long long max_segs;
};
FwdLayout fwd_layout(const Dims& D) {
  FwdLayout lo{};
  const long long seg_slots = (long long)kSegTiles * (kRows / D.G);
  lo.max_segs = D.keys() + (D.slots() + seg_slots - 1) / seg_slots;
  size_t o = align256f((size_t)D.slots() * D.G * D.d * sizeof(uint16_t));
  lo.segs = o;
  o = align256f(o + (size_t)lo.max_segs * sizeof(int4));
  lo.nseg = o;
  o = align256f(o + sizeof(int));
  lo.total = o;
  return lo;
}

template <int D>
cudaError_t run(const Dims& Dm, const void* q, const void* K, const void* V, const int32_t* idx, const float* s_sel,
                const int32_t* offsets, const int32_t* entries, void* O, float* w, void* ws, cudaStream_t st) {
  const long long keys = Dm.keys();
  const FwdLayout lo = fwd_layout(Dm);
  uint16_t* Opart = (uint16_t*)ws;
  if (keys > 0) {
    int4* segs = (int4*)((char*)ws + lo.segs);
    int* nseg = (int*)((char*)ws + lo.nseg);
    const int seg_slots = kSegTiles * (kRows / Dm.G);
    (void)launch_dependent(fwd_segments_kernel, dim3(1), dim3(1024), 0, st, offsets, Dm.Nc, Dm.B * Dm.Hkv, seg_slots,
                           segs, nseg, Dm.slots(), Dm.status);
    note_launches(1);
    cudaError_t e0 = cudaGetLastError();
    if (e0 != cudaSuccess) return e0;
    FwdArgs a;
    a.q = (const uint16_t*)q;
    a.K = (const uint16_t*)K;
    a.V = (const uint16_t*)V;
    a.segs = segs;
    a.nseg = nseg;
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
    a.softmax1 = Dm.softmax1 ? 1 : 0;
    a.status = Dm.status;
    const size_t smem = sizeof(FwdSmem<D>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(fwd_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    CUtensorMap tq, to;
    memset(&tq, 0, sizeof(tq));
    memset(&to, 0, sizeof(to));
    a.n_rows = Dm.B * Dm.L * Dm.Hq;
    a.n_slots = Dm.slots();
    a.use_tma = Dm.G >= 8 ? 1 : 0;
    if (a.use_tma && !tc::make_group8_tmap(&tq, q, (unsigned long long)a.n_rows, D)) return cudaErrorNotSupported;
    if (a.use_tma && !tc::make_group8_tmap(&to, Opart, (unsigned long long)Dm.slots() * Dm.G, D))
      return cudaErrorNotSupported;
    (void)launch_dependent(fwd_chunk_kernel<D>, dim3((unsigned)lo.max_segs), dim3(kThreads), smem, st, a, tq, to);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  const long long rows = (long long)Dm.B * Dm.L * Dm.Hkv;
  (void)launch_dependent(fwd_merge_kernel<D>, dim3((unsigned)((rows + 7) / 8)), dim3(256), 0, st, s_sel, idx, Opart,
                         (uint16_t*)O, w, rows, Dm.Hkv, Dm.G, Dm.topk, Dm.Nc, Dm.stick ? 1 : 0, Dm.status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

size_t forward_workspace(const Dims& D) { return fwd_layout(D).total; }

cudaError_t launch_forward(const Dims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                           const float* s_sel, const int32_t* offsets, const int32_t* entries, void* O, float* w,
                           void* ws, cudaStream_t st) {
  return D.d == 64 ? run<64>(D, q, K, V, idx, s_sel, offsets, entries, O, w, ws, st)
                   : run<128>(D, q, K, V, idx, s_sel, offsets, entries, O, w, ws, st);
}

}  // namespace hsa
