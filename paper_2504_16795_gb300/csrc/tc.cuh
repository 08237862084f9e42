// Blackwell (sm_103a) building blocks: mbarriers with bounded waits, the
// 5th-generation tensor core (tcgen05.mma with accumulators in tensor memory),
// tensor-memory allocation and loads, and the shared-memory operand layout.
//
// Operand layout used everywhere: K-major, 128-byte swizzle. A tile of R rows
// and 64 bf16 columns is R x 128 bytes; 8-row groups form 1024-byte atoms and
// the 16-byte chunk c of row r is stored at chunk (c ^ (r % 8)). Wider tiles
// are stacked 64-column blocks. Tile bases are 1024-byte aligned.
#pragma once
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"

namespace hsa {
namespace tc {

// ------------------------------------------------------------------ status
// Every wait below gives up after kWaitLimitNs: it records the failure in the
// block's abort flag and in a device status word, and returns false, so a
// broken pipeline ends the kernel instead of hanging the GPU.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s

// Programmatic dependent launch (common.cuh): the work a kernel does before
// griddep_wait (barrier setup, tensor-memory allocation) overlaps the previous
// grid's tail.
using ::hsa::griddep_wait;

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking poll: mbarrier.try_wait may suspend the thread until the phase
// completes or an implementation-defined time passes, so a thread that polls
// several barriers in turn (an event loop) uses test_wait, which returns at once.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with the given parity to complete, for at most
// `limit_ns`: on giving up it sets the block's abort flag and the status word
// and returns false. The clock is first read after 256 unsuccessful polls, so
// a wait that ends soon pays nothing for the bound.
__device__ __forceinline__ bool mbar_wait_for(uint32_t bar, uint32_t parity, unsigned long long limit_ns,
                                              volatile int* abort_flag, unsigned* status) {
  unsigned long long t0 = 0;
  for (unsigned it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 255u) {
      if (*abort_flag) return false;
      const unsigned long long now = globaltimer();
      if (it == 255u) {
        t0 = now;
      } else if (now - t0 > limit_ns) {
        *abort_flag = 1;
        if (status) atomicOr(status, kStatusTimeout);
        return false;
      }
    }
  }
}
// The pipelines' wait: bounded by kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned* status) {
  return mbar_wait_for(bar, parity, kWaitLimitNs, abort_flag, status);
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n" ::"r"(bar),
               "r"(bytes)
               : "memory");
}

// ------------------------------------------------------------------ TMA
// 2-D tiled bulk copy global -> shared (async proxy); completion is counted
// in bytes on `bar`. x (the innermost coordinate) must be a multiple of 8
// bf16 elements; rows beyond the tensor are filled with zeros.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}
// 3-D tiled bulk copy shared -> global (async proxy), tracked by the issuing
// thread's bulk group: commit with bulk_commit, and before the shared source
// is written again wait with bulk_wait_read.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, int x, int y, int z, uint32_t src) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(src)
               : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, uint32_t src) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src)
               : "memory");
}
// L2 eviction priorities for bulk copies: data read again soon (gathered
// query rows) is kept with evict_last; streamed results written once
// (partials) go out with evict_first, so they do not push the former out.
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                                 uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, %3, "
      "%4}], [%5], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void tma_store_3d_hint(const CUtensorMap* map, int x, int y, int z, uint32_t src,
                                                  uint64_t policy) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group.L2::cache_hint [%0, {%1, %2, %3}], [%4], %5;" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(src), "l"(policy)
               : "memory");
}
__device__ __forceinline__ void tma_store_2d_hint(const CUtensorMap* map, int x, int y, uint32_t src, uint64_t policy) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group.L2::cache_hint [%0, {%1, %2}], [%3], %4;" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(src), "l"(policy)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// The shared sources of all committed bulk groups have been read.
// Every bulk group but the most recent one has finished reading its shared source.
__device__ __forceinline__ void bulk_wait_read_but1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// All committed bulk groups have completed (writes visible).
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// Plain (untiled) bulk copy global -> shared, completion counted in bytes on
// `bar`. Both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}

// Bound for an event loop that polls several barriers: call busy() after a
// pass that issued work and idle() after one that did not; idle() returns
// false (setting the abort flag and the status word) once no work has been
// issued for the wait limit. Reading %globaltimer is slow, so the clock is
// read only every 1024 idle passes, never on the way to the next issue.
struct SpinLimit {
  unsigned n = 0;
  unsigned long long t0 = 0;
  __device__ __forceinline__ void busy() { n = 0; }
  __device__ __forceinline__ bool idle(volatile int* abort_flag, unsigned* status) {
    if ((++n & 1023u) != 0) return true;
    if (*abort_flag) return false;
    const unsigned long long now = globaltimer();
    if (n == 1024u) {
      t0 = now;
    } else if (now - t0 > kWaitLimitNs) {
      *abort_flag = 1;
      if (status) atomicOr(status, kStatusTimeout);
      return false;
    }
    return true;
  }
};


// ------------------------------------------------------------------ proxies
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ------------------------------------------------------------------ tensor memory
// Executed by one full warp. Writes the base address to *dst (shared memory).
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// Address of (lane, column) in tensor memory.
__device__ __forceinline__ uint32_t tmem_addr(uint32_t base, uint32_t lane, uint32_t col) {
  return base + (lane << 16) + col;
}

// 32 lanes x 32 bits, 32 consecutive columns: thread i of the warp gets lane
// (32 * (warp % 4) + i), columns col..col+31.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// Store 32 consecutive 32-bit columns of the thread's lane (32x32b.x32).
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,"
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
        "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
        "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// ------------------------------------------------------------------ MMA
// Instruction descriptor of kind::f16 with bf16 A and B, fp32 accumulator,
// shape M x N; a_mn / b_mn select the MN-major (instead of K-major) operand.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn = false, bool b_mn = false) {
  return (1u << 4)                      // accumulator format: f32
         | (1u << 7)                    // A format: bf16
         | (1u << 10)                   // B format: bf16
         | ((a_mn ? 1u : 0u) << 15)     // A major-ness
         | ((b_mn ? 1u : 0u) << 16)     // B major-ness
         | ((uint32_t)(N >> 3) << 17)   // N / 8
         | ((uint32_t)(M >> 4) << 24);  // M / 16
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row atoms
// 1024 bytes apart. `addr` is the shared address of the first element this
// instruction reads (the K offset inside a 128-byte row is part of it).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t addr) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4)  // start address
         | ((uint64_t)1 << 16)               // leading byte offset (unused by swizzled K-major)
         | ((uint64_t)(1024 >> 4) << 32)     // stride byte offset: next 8-row atom
         | ((uint64_t)1 << 46)               // descriptor version
         | ((uint64_t)2 << 61);              // 128-byte swizzle
}

// MN-major, 128-byte swizzle: each 128-byte row holds 64 consecutive M (or N)
// elements of one K index; 8 K-rows form a 1024-byte atom (stride 1024 along
// K) and the next 64 M/N elements start `mn_block_bytes` further on. A
// K-major tile [k-row][64 columns] read this way is its own transpose, so
// the same shared tile serves both operand orientations.
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t addr, uint32_t mn_block_bytes, uint32_t k8_bytes = 1024) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4)                     // start address
         | ((uint64_t)((mn_block_bytes >> 4) & 0x3FFFu) << 16)  // leading byte offset: next 64 M/N elements
         | ((uint64_t)((k8_bytes >> 4) & 0x3FFFu) << 32)        // stride byte offset: next 8 K-rows
         | ((uint64_t)1 << 46)                                  // descriptor version
         | ((uint64_t)2 << 61);                                 // 128-byte swizzle
}

// D[tmem] (+)= A[smem] * B[smem]^T over one K=16 slice; issued by one thread.
__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// The same with A read from tensor memory: lanes = the M rows, K packed two
// bf16 per 32-bit column (lower K index in the low half), so one K = 16 step
// spans 8 columns; B from shared memory as above.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on `bar` when every MMA this thread issued so far has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// K-major, 128-byte swizzle, 8-row groups `sbo` bytes apart (the start
// address gives the 64-column block inside a group).
__device__ __forceinline__ uint64_t sdesc_sw128_sbo(uint32_t addr, uint32_t sbo) {
  return (uint64_t)((addr & 0x3FFFFu) >> 4)      // start address
         | ((uint64_t)1 << 16)                   // leading byte offset (unused by swizzled K-major)
         | ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32)  // stride byte offset: next 8-row group
         | ((uint64_t)1 << 46)                   // descriptor version
         | ((uint64_t)2 << 61);                  // 128-byte swizzle
}

// Grouped layout of a gathered tile of `cols` bf16 columns: rows in groups of
// 8, group j at j * 16 * cols bytes, holding one 1024-byte swizzled atom
// (8 rows x 64 columns) per 64-column block. One TMA box of 8 rows x all
// columns fills one group. For cols = 64 it is the plain stacked layout.
__device__ __forceinline__ uint32_t grp_offset(int cols, int row, int col) {
  return (uint32_t)((row >> 3) * 16 * cols + (col >> 6) * 1024 + (row & 7) * 128 +
                    ((((col >> 3) & 7) ^ (row & 7)) << 4) + ((col & 7) << 1));
}

// Byte offset of (row, col) in a K-major 128-byte-swizzled tile of `rows` rows
// (bf16 elements; col may exceed 63: 64-column blocks are stacked).
__device__ __forceinline__ uint32_t sw128_offset(int rows, int row, int col) {
  return (uint32_t)((col >> 6) * rows * 128 + row * 128 + ((((col >> 3) & 7) ^ (row & 7)) << 4) + ((col & 7) << 1));
}

// ------------------------------------------------------------------ host: tensor maps
// A bf16 matrix of `rows` x `cols` (row pitch cols * 2 bytes) read in boxes of
// 64 columns x box_rows rows with the 128-byte swizzle of the operand layout.
inline PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  if (encode == nullptr) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
      return nullptr;
    encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  return encode;
}

inline bool make_rows_tmap(CUtensorMap* map, const void* base, unsigned long long rows, int cols, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (encode == nullptr) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A bf16 matrix of `rows` x `cols` read 8 rows at a time into the grouped
// layout (grp_offset): a 3-D view {64 columns, rows, cols/64 blocks} with box
// {64, 8, cols/64} and the 128-byte swizzle.
inline bool make_group8_tmap(CUtensorMap* map, const void* base, unsigned long long rows, int cols) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (encode == nullptr) return false;
  const cuuint64_t dims[3] = {64u, (cuuint64_t)rows, (cuuint64_t)(cols / 64)};
  const cuuint64_t strides[2] = {(cuuint64_t)cols * 2, 128u};
  const cuuint32_t box[3] = {64u, 8u, (cuuint32_t)(cols / 64)};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A bf16 matrix of `rows` x `cols` written (or read) in boxes of 32 columns
// (64 bytes) x 8 rows with the 64-byte swizzle: in shared memory the 16-byte
// chunk c of box row r sits at chunk (c ^ ((r >> 1) & 3)).
inline bool make_rows32_sw64_tmap(CUtensorMap* map, const void* base, unsigned long long rows, int cols) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (encode == nullptr) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {32u, 8u};
  const cuuint32_t estr[2] = {1u, 1u};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same for an fp32 matrix: boxes of 32 columns (128 bytes) x box_rows rows.
// In shared memory, element (r, c) of a box sits in 16-byte chunk
// ((c / 4) ^ (r % 8)) of the box's 128-byte row r.
inline bool make_rows_tmap_f32(CUtensorMap* map, const void* base, unsigned long long rows, int cols, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (encode == nullptr) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 4};
  const cuuint32_t box[2] = {32u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// An fp32 matrix of `rows` x `cols` (row pitch cols * 4 bytes, cols a
// multiple of 4) read in plain (unswizzled) boxes of box_cols x box_rows.
inline bool make_plain_tmap_f32(CUtensorMap* map, const void* base, unsigned long long rows, int cols, int box_cols,
                                int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
  if (encode == nullptr) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 4};
  const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace tc
}  // namespace hsa
