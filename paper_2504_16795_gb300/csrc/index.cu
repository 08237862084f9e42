// Inverse selection index: for every (b, g, chunk) the selection slots that
// chose it. This replaces the dense mask M and rank R of the paper's backward
// (§3.1.2, Algorithm 3 scans every token for every chunk) with a CSR of the
// slots sorted stably by key (b*Hkv + g)*Nc + chunk, so each key's list comes
// out in increasing slot (token) order, deterministically.
//
// When one batch row's keys (Hkv * Nc) fit in shared memory, one counting pass:
//   count:  per tile of tokens (all groups and slots of those tokens, one b),
//           the count of every key, written key-major: hist[(key, tile)]
//   scan:   exclusive scan of hist = where each (key, tile) run starts
//   place:  per tile, each warp takes a contiguous share of the tile's slots:
//           its counts per key, a prefix over the warps, then its slots in
//           order, 32 at a time (equal keys ranked by lane), so the order
//           within a key is tile, warp, round, lane = slot order
// Otherwise a stable LSD radix sort of the keys, 8 bits per pass:
//   pass p (8-bit digit p):   per-tile digit histogram -> exclusive scan over
//                             (digit, tile) -> stable scatter within each tile
//   offsets:                  from the sorted keys: offsets[k] = first position
//                             whose key is >= k (one pass, no atomics)
// Padded slots (idx = -1) are never listed: the radix sort gives them the
// sentinel key B*Hkv*Nc, which sorts last; the counting pass skips them.
#include <algorithm>

#include "common.cuh"

namespace hsa {
namespace {

constexpr int kThreads = 256;
constexpr int kItems = 8;  // per thread
constexpr int kTile = kThreads * kItems;
constexpr int kScanThreads = 1024;
constexpr int kScanItems = 4;
constexpr int kScanTile = kScanThreads * kScanItems;

struct KeyMap {
  const int32_t* idx;
  int L, Hkv, topk, Nc;
  uint32_t sentinel;
  unsigned* status;  // the call's status word (debug builds report chunk ids past the sequence)
  __device__ __forceinline__ uint32_t key(long long p) const {
    const int c = idx[p];
    if (c >= 0) bounds_ok(c, 0, Nc, status);
    if (c < 0 || c >= Nc) return sentinel;  // padding (or an out-of-range index) is never listed
    const long long g = (p / topk) % Hkv;
    const long long b = p / ((long long)topk * Hkv * L);
    return (uint32_t)((b * Hkv + g) * Nc + c);
  }
};

// Digit histogram of one tile, written digit-major: hist[digit * n_tiles + tile].
__global__ void __launch_bounds__(kThreads) radix_hist_kernel(KeyMap km, const uint32_t* __restrict__ keys_in,
                                                              long long n, int shift, uint32_t* __restrict__ hist,
                                                              int n_tiles) {
  griddep_wait();
  __shared__ uint32_t h[256];
  h[threadIdx.x] = 0;
  __syncthreads();
  const long long base = (long long)blockIdx.x * kTile;
#pragma unroll
  for (int r = 0; r < kItems; ++r) {
    const long long p = base + r * kThreads + threadIdx.x;
    if (p < n) {
      const uint32_t k = keys_in ? keys_in[p] : km.key(p);
      atomicAdd(&h[(k >> shift) & 255u], 1u);
    }
  }
  __syncthreads();
  hist[(long long)threadIdx.x * n_tiles + blockIdx.x] = h[threadIdx.x];
}

// Stable scatter: items are visited in their input order (round r covers
// items base + r*256 .. base + r*256 + 255 in thread order); the rank of an
// item among equal digits is (items of that digit in earlier rounds) +
// (in earlier warps of this round) + (in earlier lanes of this warp).
__global__ void __launch_bounds__(kThreads) radix_scatter_kernel(KeyMap km, const uint32_t* __restrict__ keys_in,
                                                                 const int32_t* __restrict__ vals_in, long long n,
                                                                 int shift, const uint32_t* __restrict__ base_off,
                                                                 int n_tiles, uint32_t* __restrict__ keys_out,
                                                                 int32_t* __restrict__ vals_out) {
  griddep_wait();
  __shared__ uint32_t run[256];
  __shared__ uint32_t cnt[kThreads / 32][256];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  run[tid] = base_off[(long long)tid * n_tiles + blockIdx.x];
  const long long base = (long long)blockIdx.x * kTile;
  for (int r = 0; r < kItems; ++r) {
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) cnt[w][tid] = 0;
    __syncthreads();
    const long long p = base + r * kThreads + tid;
    const bool valid = p < n;
    uint32_t k = 0;
    int32_t v = 0;
    if (valid) {
      k = keys_in ? keys_in[p] : km.key(p);
      v = vals_in ? vals_in[p] : (int32_t)p;
    }
    const uint32_t dig = valid ? ((k >> shift) & 255u) : 256u;
    const unsigned peers = __match_any_sync(0xFFFFFFFFu, dig);
    const int before = __popc(peers & ((1u << lane) - 1u));
    const int leader = 31 - __clz(peers);
    if (valid && lane == leader) cnt[warp][dig] = __popc(peers);
    __syncthreads();
    if (valid) {
      uint32_t pos = run[dig] + before;
      for (int w = 0; w < warp; ++w) pos += cnt[w][dig];
      vals_out[pos] = v;
      if (keys_out) keys_out[pos] = k;
    }
    __syncthreads();
    uint32_t add = 0;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) add += cnt[w][tid];
    run[tid] += add;
    __syncthreads();
  }
}

// offsets[k] = first position of the sorted key array with key >= k, for
// k = 0..n_keys (the sentinel key n_keys sorts last). Position i writes the
// keys in (key[i-1], key[i]]; position n closes the range up to n_keys.
__global__ void offsets_from_sorted_kernel(const uint32_t* __restrict__ sorted, long long n, long long n_keys,
                                           int32_t* __restrict__ offsets) {
  griddep_wait();
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i <= n; i += stride) {
    const long long cur = i < n ? (long long)sorted[i] : n_keys;
    const long long prev = i > 0 ? (long long)sorted[i - 1] : -1;
    const long long hi = cur < n_keys ? cur : n_keys;
    for (long long k = prev + 1; k <= hi; ++k) offsets[k] = (int32_t)i;
  }
}

// ---- counting pass (one batch row's keys in shared memory)
constexpr int kMaxRowKeys = 4096;   // Hkv * Nc of one batch row
constexpr int kTileSlots = 8192;    // slots per tile (a whole number of tokens)
constexpr int kPlaceWarps = 8;
constexpr int kBatch = 16;          // keys a thread reads before it counts them
static_assert(kMaxRowKeys <= 32767, "row-local keys are staged as int16");
static_assert(kPlaceWarps * kMaxRowKeys * 4 + kTileSlots * 2 <= 227 * 1024, "placement shared memory");

struct CountGeom {
  int L, Hkv, topk, Nc, HN;  // HN = Hkv * Nc keys per batch row
  int tile_tokens, n_tiles;  // tiles of each batch row
  __device__ __forceinline__ long long slot0(int b, int tile) const {
    return ((long long)b * L + (long long)tile * tile_tokens) * Hkv * topk;
  }
  __device__ __forceinline__ int tile_slots(int tile) const {
    return min(tile_tokens, L - tile * tile_tokens) * Hkv * topk;
  }
  // the key of slot p within its batch row (g * Nc + chunk), -1 if the slot is not listed
  __device__ __forceinline__ int local_key(const int32_t* idx, long long p, unsigned* status) const {
    const int c = idx[p];
    if (c >= 0) bounds_ok(c, 0, Nc, status);
    if (c < 0 || c >= Nc) return -1;
    return (int)((p / topk) % Hkv) * Nc + c;
  }
};

// Counts of every key of batch row b in one tile: hist[(b*HN + key) * n_tiles + tile].
__global__ void __launch_bounds__(1024) count_keys_kernel(CountGeom cg, const int32_t* __restrict__ idx,
                                                          uint32_t* __restrict__ hist, unsigned* status) {
  griddep_wait();
  extern __shared__ uint32_t cnt[];
  const int tile = (int)blockIdx.x, b = (int)blockIdx.y;
  for (int k = threadIdx.x; k < cg.HN; k += blockDim.x) cnt[k] = 0;
  __syncthreads();
  const long long p0 = cg.slot0(b, tile);
  const int n = cg.tile_slots(tile);
  // kBatch keys per thread are read before they are counted (one memory latency per batch)
  for (int i0 = 0; i0 < n; i0 += kBatch * 1024) {
    int k[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int i = i0 + j * 1024 + (int)threadIdx.x;
      k[j] = i < n ? cg.local_key(idx, p0 + i, status) : -1;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j)
      if (k[j] >= 0) atomicAdd(&cnt[k[j]], 1u);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < cg.HN; k += blockDim.x)
    hist[((long long)b * cg.HN + k) * cg.n_tiles + tile] = cnt[k];
}

// Places the slots of one tile. start[] holds, per key, where the tile's run
// begins (the scanned hist); warp w's counters become where its share's run of
// each key begins, then advance as it writes. The first tile of a batch row
// writes the row's offsets; the last tile of the last row writes the total.
__global__ void __launch_bounds__(kPlaceWarps * 32) place_keys_kernel(CountGeom cg, const int32_t* __restrict__ idx,
                                                                      const uint32_t* __restrict__ start,
                                                                      int32_t* __restrict__ entries,
                                                                      int32_t* __restrict__ offsets, int B,
                                                                      unsigned* status) {
  griddep_wait();
  extern __shared__ uint32_t wc[];  // [kPlaceWarps][HN], then the tile's keys
  const int tile = (int)blockIdx.x, b = (int)blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int HN = cg.HN;
  int16_t* keys = reinterpret_cast<int16_t*>(wc + kPlaceWarps * HN);  // row-local key per slot (-1: not listed)
  for (int k = tid; k < kPlaceWarps * HN; k += blockDim.x) wc[k] = 0;
  __syncthreads();
  const long long p0 = cg.slot0(b, tile);
  const int n = cg.tile_slots(tile);
  const int share = (((n + kPlaceWarps - 1) / kPlaceWarps) + 31) & ~31;
  const int i0 = min(warp * share, n), i1 = min(i0 + share, n);
  uint32_t* mine = wc + warp * HN;
  for (int ib = i0; ib < i1; ib += kBatch * 32) {
    int k[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int i = ib + j * 32 + lane;
      k[j] = i < i1 ? cg.local_key(idx, p0 + i, status) : -1;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int i = ib + j * 32 + lane;
      if (i < i1) keys[i] = (int16_t)k[j];
      if (k[j] >= 0) atomicAdd(&mine[k[j]], 1u);
    }
  }
  __syncthreads();
  for (int k = tid; k < HN; k += blockDim.x) {
    uint32_t run = start[((long long)b * HN + k) * cg.n_tiles + tile];
    if (tile == 0) offsets[(long long)b * HN + k] = (int32_t)run;
#pragma unroll
    for (int w = 0; w < kPlaceWarps; ++w) {
      const uint32_t c = wc[w * HN + k];
      wc[w * HN + k] = run;
      run += c;
    }
  }
  __syncthreads();
  for (int base = i0; base < i1; base += 32) {
    const int i = base + lane;
    const int k = i < i1 ? (int)keys[i] : -1;
    const unsigned peers = __match_any_sync(0xFFFFFFFFu, k);
    const uint32_t pos = k >= 0 ? mine[k] + __popc(peers & ((1u << lane) - 1u)) : 0u;
    if (k >= 0) entries[pos] = (int32_t)(p0 + i);
    __syncwarp();
    if (k >= 0 && lane == 31 - __clz(peers)) mine[k] += __popc(peers);
    __syncwarp();
  }
  if (b == B - 1 && tile == cg.n_tiles - 1) {
    __syncthreads();
    // the end of the last key's run in the last warp's share is the number of listed slots
    if (tid == 0) offsets[(long long)B * HN] = (int32_t)wc[(kPlaceWarps - 1) * HN + HN - 1];
  }
}

// ---- exclusive scan of uint32 (in place), up to kScanTile^2 elements
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_sums, uint32_t& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t s = lane < (int)(blockDim.x / 32) ? warp_sums[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint32_t y = __shfl_up_sync(0xFFFFFFFFu, s, o);
      if (lane >= o) s += y;
    }
    warp_sums[lane] = s;  // inclusive over warps
  }
  __syncthreads();
  total = warp_sums[blockDim.x / 32 - 1];
  const uint32_t warp_base = warp > 0 ? warp_sums[warp - 1] : 0u;
  __syncthreads();
  return warp_base + x - v;
}

__global__ void __launch_bounds__(kScanThreads) scan_tiles_kernel(uint32_t* __restrict__ a, long long n,
                                                                  uint32_t* __restrict__ tile_sums) {
  griddep_wait();
  __shared__ uint32_t ws[32];
  const long long base = (long long)blockIdx.x * kScanTile + (long long)threadIdx.x * kScanItems;
  uint32_t v[kScanItems], s = 0;
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    v[i] = base + i < n ? a[base + i] : 0u;
    s += v[i];
  }
  uint32_t total;
  uint32_t ex = block_exclusive_scan(s, ws, total);
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    if (base + i < n) a[base + i] = ex;
    ex += v[i];
  }
  if (threadIdx.x == 0 && tile_sums) tile_sums[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanThreads) add_tile_base_kernel(uint32_t* __restrict__ a, long long n,
                                                                     const uint32_t* __restrict__ tile_base) {
  griddep_wait();
  const long long base = (long long)blockIdx.x * kScanTile + (long long)threadIdx.x * kScanItems;
  const uint32_t add = tile_base[blockIdx.x];
#pragma unroll
  for (int i = 0; i < kScanItems; ++i)
    if (base + i < n) a[base + i] += add;
}

// Exclusive scan of a[0..n) in place (tile_sums: scratch for the tile totals).
cudaError_t exclusive_scan(uint32_t* a, long long n, uint32_t* tile_sums, cudaStream_t st) {
  const long long tiles = (n + kScanTile - 1) / kScanTile;
  if (tiles <= 1) {
    (void)launch_dependent(scan_tiles_kernel, dim3(1), dim3(kScanThreads), 0, st, a, n, nullptr);
    note_launches(1);
    return cudaGetLastError();
  }
  if (tiles > kScanTile) return cudaErrorInvalidValue;
  (void)launch_dependent(scan_tiles_kernel, dim3((unsigned)tiles), dim3(kScanThreads), 0, st, a, n, tile_sums);
  note_launches(1);
  (void)launch_dependent(scan_tiles_kernel, dim3(1), dim3(kScanThreads), 0, st, tile_sums, tiles, nullptr);
  note_launches(1);
  (void)launch_dependent(add_tile_base_kernel, dim3((unsigned)tiles), dim3(kScanThreads), 0, st, a, n, tile_sums);
  note_launches(1);
  return cudaGetLastError();
}

struct IndexLayout {
  long long n, n_tiles, hist_len, keys;
  int passes;
  size_t off_keys_a, off_keys_b, off_vals_a, off_vals_b, off_hist, off_sums, total;
  bool counting;  // the one-pass counting sort (one batch row's keys fit in shared memory)
  CountGeom cg;
};

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

IndexLayout layout(const Dims& D) {
  IndexLayout lo{};
  lo.n = D.slots();
  lo.keys = D.keys();
  const long long HN = (long long)D.Hkv * D.Nc;
  const long long per_token = (long long)D.Hkv * D.topk;
  if (HN > 0 && HN <= kMaxRowKeys && per_token > 0 && per_token <= kTileSlots) {
    CountGeom cg{};
    cg.L = D.L;
    cg.Hkv = D.Hkv;
    cg.topk = D.topk;
    cg.Nc = D.Nc;
    cg.HN = (int)HN;
    cg.tile_tokens = (int)std::min<long long>(kTileSlots / per_token, D.L);
    cg.n_tiles = (int)((D.L + cg.tile_tokens - 1) / cg.tile_tokens);
    const long long hist_len = (long long)D.B * HN * cg.n_tiles;
    if ((hist_len + kScanTile - 1) / kScanTile <= kScanTile && cg.n_tiles <= 65535 && D.B <= 65535) {
      lo.counting = true;
      lo.cg = cg;
      lo.hist_len = hist_len;
      size_t o = 0;
      lo.off_hist = o;
      o = align256(o + sizeof(uint32_t) * (size_t)hist_len);
      lo.off_sums = o;
      o = align256(o + sizeof(uint32_t) * (size_t)((hist_len + kScanTile - 1) / kScanTile + 1));
      lo.total = o;
      return lo;
    }
  }
  lo.n_tiles = (lo.n + kTile - 1) / kTile;
  lo.hist_len = 256 * lo.n_tiles;
  int bits = 1;
  while ((1ull << bits) <= (unsigned long long)lo.keys) ++bits;  // sentinel = keys must fit
  lo.passes = (bits + 7) / 8;
  size_t o = 0;
  lo.off_keys_a = o;
  o = align256(o + sizeof(uint32_t) * (size_t)lo.n);
  lo.off_keys_b = o;
  o = align256(o + sizeof(uint32_t) * (size_t)lo.n);
  lo.off_vals_a = o;
  o = align256(o + sizeof(int32_t) * (size_t)lo.n);
  lo.off_vals_b = o;
  o = align256(o + sizeof(int32_t) * (size_t)lo.n);
  lo.off_hist = o;
  const long long scan_len = lo.hist_len;
  o = align256(o + sizeof(uint32_t) * (size_t)scan_len);
  lo.off_sums = o;
  o = align256(o + sizeof(uint32_t) * (size_t)((scan_len + kScanTile - 1) / kScanTile + 1));
  lo.total = o;
  return lo;
}

}  // namespace

size_t index_workspace(const Dims& D) { return layout(D).total; }

cudaError_t launch_index(const Dims& D, const int32_t* idx, int32_t* offsets, int32_t* entries, void* ws,
                         cudaStream_t st) {
  const IndexLayout lo = layout(D);
  if (lo.n == 0) return cudaSuccess;
  if ((lo.hist_len + kScanTile - 1) / kScanTile > kScanTile) return cudaErrorInvalidValue;
  char* w = (char*)ws;
  if (lo.counting) {
    uint32_t* hist = (uint32_t*)(w + lo.off_hist);
    uint32_t* sums = (uint32_t*)(w + lo.off_sums);
    const dim3 grid((unsigned)lo.cg.n_tiles, (unsigned)D.B);
    cudaError_t e;
    (void)launch_dependent(count_keys_kernel, grid, dim3(1024), sizeof(uint32_t) * lo.cg.HN, st, lo.cg, idx, hist,
                           D.status);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = exclusive_scan(hist, lo.hist_len, sums, st)) != cudaSuccess) return e;
    const size_t place_smem = sizeof(uint32_t) * (size_t)kPlaceWarps * lo.cg.HN + sizeof(int16_t) * kTileSlots;
    if ((e = cudaFuncSetAttribute(place_keys_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)place_smem)) !=
        cudaSuccess)
      return e;
    (void)launch_dependent(place_keys_kernel, grid, dim3(kPlaceWarps * 32), place_smem, st, lo.cg, idx,
                           (const uint32_t*)hist, entries, offsets, D.B, D.status);
    note_launches(1);
    return cudaGetLastError();
  }
  uint32_t* keys_buf[2] = {(uint32_t*)(w + lo.off_keys_a), (uint32_t*)(w + lo.off_keys_b)};
  int32_t* vals_buf[2] = {(int32_t*)(w + lo.off_vals_a), (int32_t*)(w + lo.off_vals_b)};
  uint32_t* hist = (uint32_t*)(w + lo.off_hist);
  uint32_t* sums = (uint32_t*)(w + lo.off_sums);
  KeyMap km{idx, D.L, D.Hkv, D.topk, D.Nc, (uint32_t)lo.keys, D.status};
  cudaError_t e;
  const uint32_t* kin = nullptr;
  const int32_t* vin = nullptr;
  for (int pass = 0; pass < lo.passes; ++pass) {
    const bool last = pass == lo.passes - 1;
    uint32_t* kout = keys_buf[pass & 1];
    int32_t* vout = last ? entries : vals_buf[pass & 1];
    (void)launch_dependent(radix_hist_kernel, dim3((unsigned)lo.n_tiles), dim3(kThreads), 0, st, km, kin, lo.n,
                           8 * pass, hist, (int)lo.n_tiles);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = exclusive_scan(hist, lo.hist_len, sums, st)) != cudaSuccess) return e;
    (void)launch_dependent(radix_scatter_kernel, dim3((unsigned)lo.n_tiles), dim3(kThreads), 0, st, km, kin, vin, lo.n,
                           8 * pass, hist, (int)lo.n_tiles, kout, vout);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    kin = kout;
    vin = vout;
  }
  // offsets from the sorted keys of the last pass
  (void)launch_dependent(offsets_from_sorted_kernel, dim3(grid_cap((lo.n + 256) / 256, 152LL * 8)), dim3(256), 0, st,
                         kin, lo.n, lo.keys, offsets);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace hsa
