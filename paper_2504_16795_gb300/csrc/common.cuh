// Internal helpers shared by the HSA CUDA kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hsa.h"

namespace hsa {

constexpr int kChunk = 64;  // S: the only chunk size the kernels are built for

// Bits of a call's device status word (the head of its workspace, read and
// cleared by hsa_check): a bounded wait gave up; an index read from an input
// array lay outside its range (checked only in builds with HSA_DEBUG_BOUNDS).
enum : unsigned { kStatusTimeout = 1u, kStatusBounds = 2u };
#ifdef HSA_DEBUG_BOUNDS
constexpr bool kDebugBounds = true;
#else
constexpr bool kDebugBounds = false;
#endif
// Debug builds: whether lo <= v < hi, recording an out-of-range value in the
// status word, so that the caller skips the access it would have made. Other
// builds: true (the check compiles away).
__device__ __forceinline__ bool bounds_ok(long long v, long long lo, long long hi, unsigned* status) {
  if constexpr (kDebugBounds) {
    if (v < lo || v >= hi) {
      if (status) atomicOr(status, kStatusBounds);
      return false;
    }
  }
  return true;
}

// Block order of the chunk kernels. A chunk's list holds the slots of every
// later token that chose it, so early chunks carry the longest lists. The
// first kHeadChunks chunks of every (b, g) run first, chunk-major across the
// pairs, so that no long list starts near the end of the grid; the rest run
// pair by pair in chunk order, so that the blocks in flight gather query rows
// of one (b, g) and share them in L2.
constexpr int kHeadChunks = 16;
__device__ __forceinline__ void block_key(int Nc, int n_bg, int& c, int& bg) {
  const int head = min(kHeadChunks, Nc);
  const int b = (int)blockIdx.x;
  if (b < head * n_bg) {
    c = b / n_bg;
    bg = b % n_bg;
  } else {
    const int r = b - head * n_bg, rest = Nc - head;
    bg = r / rest;
    c = head + r % rest;
  }
}
constexpr int kWarp = 32;

// Every workspace starts with this header: the status word that the
// pipelined kernels of a call set when one of their bounded waits gives up
// (read and cleared by hsa_check). The rest of the workspace follows it.
constexpr size_t kStatusBytes = 256;

// Resolved shape shared by host launchers.
struct Dims {
  int B, L, Hq, Hkv, d, S, topk, G, Nc;
  float scale_sel, scale_attn;
  bool softmax1, stick;  // variants: softmax-off-by-one inside chunks, stick-breaking chunk weights
  unsigned* status = nullptr;  // the call's status word (device memory, the workspace header)
  long long slots() const { return (long long)B * L * Hkv * topk; }
  long long keys() const { return (long long)B * Hkv * Nc; }
};

// Chunk weights of one selection row held by a warp, lane j = slot j (the
// first keff slots valid, in I' order: latest chunk first): softmax over the
// scores, or stick-breaking (§3.1.1 "Chunk Weights") — slot j takes
// sigmoid(s_j) of what the earlier slots left, w_j = b_j prod_{i<j} (1 - b_i).
// Lanes past keff get 0.
__device__ __forceinline__ float warp_chunk_weight(float s, bool valid, bool stick) {
  if (stick) {
    // 1 - sigmoid(s) = sigmoid(-s), exact for large scores
    const float b = valid ? 1.f / (1.f + expf(-s)) : 0.f;
    const float keep = valid ? 1.f / (1.f + expf(s)) : 1.f;
    const int lane = threadIdx.x & 31;
    float r = __shfl_up_sync(0xFFFFFFFFu, keep, 1);  // exclusive product: prod over earlier lanes
    if (lane == 0) r = 1.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float v = __shfl_up_sync(0xFFFFFFFFu, r, o);
      if (lane >= o) r *= v;
    }
    return valid ? b * r : 0.f;
  }
  float m = s;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
  const float ex = valid ? expf(s - m) : 0.f;
  float z = ex;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xFFFFFFFFu, z, o);
  return valid ? ex / z : 0.f;
}

// ------------------------------------------------------------------ bf16
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }
__device__ __forceinline__ float bf16_bits_to_f32(uint16_t v) { return __uint_as_float(((uint32_t)v) << 16); }
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ uint16_t f32_to_bf16_bits(float x) {
  __nv_bfloat16 h = __float2bfloat16_rn(x);
  return *reinterpret_cast<uint16_t*>(&h);
}

// ------------------------------------------------------------------ ranking keys
// A 64-bit key whose unsigned order is the rank order of the paper's top-k:
// larger score first, equal scores by lower chunk index. 0 never beats a real key.
__device__ __forceinline__ uint32_t order_bits(float s) {
  uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float order_bits_to_float(uint32_t o) {
  uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(u);
}
__device__ __forceinline__ unsigned long long rank_key(float s, uint32_t chunk) {
  return ((unsigned long long)order_bits(s) << 32) | (unsigned long long)(0xFFFFFFFFu - chunk);
}
__device__ __forceinline__ uint32_t key_chunk(unsigned long long k) {
  return 0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull);
}
__device__ __forceinline__ float key_score(unsigned long long k) { return order_bits_to_float((uint32_t)(k >> 32)); }

// A warp holds a running top-k list, lane l keeping the key of rank l (l < k,
// descending). Insert x (already known to beat the current k-th key).
__device__ __forceinline__ void warp_topk_insert(unsigned long long& mine, unsigned long long x, int k, int lane) {
  unsigned above = __ballot_sync(0xFFFFFFFFu, lane < k && mine > x);
  int pos = __popc(above);
  unsigned long long up = __shfl_up_sync(0xFFFFFFFFu, mine, 1);
  if (lane < k) {
    if (lane == pos) mine = x;
    else if (lane > pos) mine = up;
  }
}

// Offer one candidate per lane to the running list; threshold = current k-th key.
__device__ __forceinline__ void warp_topk_offer(unsigned long long& mine, unsigned long long cand, int k, int lane) {
  unsigned long long thr = __shfl_sync(0xFFFFFFFFu, mine, k - 1);
  unsigned m = __ballot_sync(0xFFFFFFFFu, cand > thr);
  while (m) {
    int src = __ffs(m) - 1;
    unsigned long long x = __shfl_sync(0xFFFFFFFFu, cand, src);
    warp_topk_insert(mine, x, k, lane);
    thr = __shfl_sync(0xFFFFFFFFu, mine, k - 1);
    m &= ~(1u << src);
    m &= __ballot_sync(0xFFFFFFFFu, cand > thr);
  }
}

// Write a finished list (ranks 0..k-1, valid where key != 0) as idx/s_sel
// ordered by decreasing chunk index, padding with -1 / -inf.
__device__ __forceinline__ int warp_emit_selection(unsigned long long mine, int k, int lane, int32_t* idx_out,
                                                   float* s_out) {
  bool valid = lane < k && mine != 0ull;
  unsigned vm = __ballot_sync(0xFFFFFFFFu, valid);
  int keff = __popc(vm);  // valid entries occupy lanes 0..keff-1
  uint32_t c = valid ? key_chunk(mine) : 0u;
  int rank = 0;
  for (int l = 0; l < keff; ++l) {
    uint32_t other = __shfl_sync(0xFFFFFFFFu, c, l);
    rank += (other > c) ? 1 : 0;
  }
  if (valid) {
    idx_out[rank] = (int32_t)c;
    s_out[rank] = key_score(mine);
  } else if (lane < k) {
    idx_out[lane] = -1;
    s_out[lane] = -__int_as_float(0x7f800000);
  }
  return keff;
}

// ------------------------------------------------------------------ programmatic dependent launch
// A kernel launched with launch_dependent (below) is set up while the previous
// kernel in its stream finishes: griddep_wait returns once that grid has
// completed and its writes are visible (for a kernel launched the ordinary way
// it returns at once). Every such kernel calls it before it reads or writes
// global memory. No kernel signals its dependents early: letting the next
// grid's blocks onto the SMs during a chunk kernel's last wave made the
// backward slower.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ------------------------------------------------------------------ async copies / tensor-core fragments
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
// D = A(16x16, row) * B(16x8, col) + D, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of element (row, col) in a shared tile of bf16 rows of `cols`
// elements, with the 16-byte chunks of each row XOR-swizzled by (row & 7) so
// that ldmatrix reads of 8 consecutive rows hit distinct banks.
template <int COLS>
__device__ __forceinline__ uint32_t swz(int row, int col) {
  return (uint32_t)(row * (COLS * 2) + ((((col >> 3) ^ (row & 7))) << 4) + ((col & 7) << 1));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// ------------------------------------------------------------------ host helpers
// Number of kernels this library has launched since it was loaded.
void note_launches(unsigned long long n);

inline int grid_cap(long long blocks, long long cap = 152LL * 64) {
  if (blocks < 1) return 1;
  return (int)(blocks < cap ? blocks : cap);
}

}  // namespace hsa

// Launchers implemented in the kernel translation units; all return cudaError_t.
namespace hsa {
cudaError_t launch_pool(const Dims& D, const void* K, float* kbar32, void* kbar16, cudaStream_t st);
// Tensor-core selection with exact rescoring (topk <= 16); needs select_tc_workspace bytes.
bool select_tc_applies(const Dims& D);
size_t select_tc_workspace(const Dims& D);
cudaError_t launch_select_tc(const Dims& D, const void* q, const float* kbar32, int32_t* idx, float* s_sel, void* ws,
                             cudaStream_t st);
cudaError_t launch_select(const Dims& D, const void* q, const float* kbar32, int32_t* idx, float* s_sel,
                          cudaStream_t st);
size_t index_workspace(const Dims& D);
cudaError_t launch_index(const Dims& D, const int32_t* idx, int32_t* offsets, int32_t* entries, void* ws,
                         cudaStream_t st);
size_t forward_workspace(const Dims& D);
cudaError_t launch_forward(const Dims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                           const float* s_sel, const int32_t* offsets, const int32_t* entries, void* O, float* w,
                           void* ws, cudaStream_t st);
size_t backward_workspace(const Dims& D);
size_t backward_attention_workspace(const Dims& D);
cudaError_t launch_backward_attention(const Dims& D, const void* q, const void* K, const void* V, const int32_t* idx,
                                      const float* w, const void* dO, const int32_t* offsets,
                                      const int32_t* entries, float* dq, float* dK, float* dV, float* ds_acc,
                                      void* ws, cudaStream_t st);
size_t select_backward_workspace(const Dims& D);
cudaError_t launch_select_backward(const Dims& D, const void* q_sel, const float* kbar_sel, const int32_t* idx,
                                   const float* ds, const int32_t* offsets, const int32_t* entries, float* dq_sel,
                                   float* dK_sel, void* ws, cudaStream_t st);
// Self-test of the bounded waits: one block waits on a barrier nothing arrives at
// and records the timeout in `status`.
cudaError_t launch_selftest_wait(unsigned long long limit_ns, unsigned* status, cudaStream_t st);
// The selection's tensor-core score pass on one 128 x 64 tile (rounding measurements).
cudaError_t launch_selftest_score_tile(int d, const void* A, const void* B, float* C, unsigned* status,
                                       cudaStream_t st);
cudaError_t launch_backward(const Dims& D, const void* q, const void* K, const void* V, const float* kbar32,
                            const int32_t* idx, const float* w, const void* O, const void* dO,
                            const int32_t* offsets, const int32_t* entries, float* dq, float* dK, float* dV,
                            void* ws, cudaStream_t st);
struct DecodeDims {
  int Bq, Hq, Hkv, d, S, topk, G;
  long long Nc;
  float scale_sel, scale_attn;
  bool softmax1, stick;  // variants as in Dims
  long long cap;         // chunks the memory and its index are laid out for (>= Nc)
  unsigned* status = nullptr;  // as in Dims
};
// Launch `kernel` as a programmatic dependent of the previous kernel in `st`
// (it must call griddep_wait before it touches global memory).
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                             Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}
size_t decode_workspace(const DecodeDims& D);
// True when a kernel of the current device may read p at that address: device or
// managed memory, or page-locked host memory mapped at the same address (a decode
// memory kept in host memory). Pageable or unknown memory gives false.
bool memory_device_readable(const void* p);
cudaError_t launch_decode(const DecodeDims& D, const void* q, const void* K, const void* V, const float* kbar32,
                          void* O, int32_t* idx, float* s_sel, float* w, void* ws, cudaStream_t st);
// Token-level attention over the selected chunks and the weighted sum (the last two decode steps);
// scratch: decode_attend_scratch(D) bytes, 256-byte aligned (partials, then one counter per row).
size_t decode_attend_scratch(const DecodeDims& D);
unsigned* decode_attend_counters(const DecodeDims& D, void* scratch);
// counters_zeroed: the kernel before has zeroed the per-row counters (no memset);
// dependent: launched as a programmatic dependent of that kernel.
cudaError_t launch_decode_attend(const DecodeDims& D, const void* q, const void* K, const void* V,
                                 const int32_t* idx, const float* w, void* O, void* scratch, cudaStream_t st,
                                 bool counters_zeroed = false, bool dependent = false);
// Decode over a memory index (bf16 summaries, norms): tensor-core scan with exact rescoring (topk <= 16).
bool decode_index_applies(const DecodeDims& D);  // topk <= 16: the memory has an index
bool decode_tc_applies(const DecodeDims& D);     // ... and at least one chunk
size_t decode_index_bytes(const DecodeDims& D);
cudaError_t launch_decode_index(const DecodeDims& D, const float* kbar32, void* index, cudaStream_t st);
// Index rows of chunks [c0, c1) from kbar32 (the memory's [cap, Hkv, d] summaries).
cudaError_t launch_index_rows(const DecodeDims& D, const float* kbar32, void* index, long long c0, long long c1,
                              cudaStream_t st);
// Append n_new tokens (K_new, V_new [n_new, Hkv, d]) to a memory holding n_tokens:
// rows written, newly completed chunks pooled into kbar32 and, when index is not
// null, entered in the decode index.
cudaError_t launch_memory_append(const DecodeDims& D, long long n_tokens, long long n_new, const void* K_new,
                                 const void* V_new, void* K_mem, void* V_mem, float* kbar32, void* index,
                                 cudaStream_t st);
size_t decode_tc_workspace(const DecodeDims& D);
cudaError_t launch_decode_tc(const DecodeDims& D, const void* q, const void* K, const void* V, const float* kbar32,
                             const void* index, void* O, int32_t* idx, float* s_sel, float* w, void* ws,
                             cudaStream_t st);
// The decode shape check of hsa_decode, shared with the entry point that owns its scratch.
hsa_status_t resolve_decode_shape(const hsa_decode_shape_t* s, DecodeDims* out);
}  // namespace hsa
