/*
 * hsa.h — C ABI of the Hierarchical Sparse Attention (HSA) hot path on GB300
 * (sm_103a). HSA: arXiv 2504.16795, "Hardware-aligned Hierarchical Sparse
 * Attention for Efficient Long-term Memory Access".
 *
 * The operator (one GQA group g of query heads [g*G, (g+1)*G) sharing KV head g):
 *   K̄_i      = (1/S) sum_{s<S} K_{iS+s}                        chunk summaries
 *   s_{t,i}  = c_sel * (sum_{h in g} q_{t,h}) · K̄_i,  i < floor(t/S)
 *   I_t      = top-k of s_{t,.} (ties: lower chunk index), listed by decreasing index
 *   w_{t,j}  = softmax_j(s_{t,I_j})                              chunk weights
 *   O_{t,h}  = sum_j w_{t,j} softmax(c_att q_{t,h} K_{I_j}^T) V_{I_j}
 * and its gradients into q, K, V (through w also into the scores, K̄ and K).
 *
 * Conventions for every call
 *   Layout   Row-major, head dimension contiguous:
 *              q, O, dO, dq    [B, L, Hq, d]
 *              K, V, dK, dV    [B, L, Hkv, d]
 *              K̄ (kbar32/16)   [B, L/S, Hkv, d]   (complete chunks only)
 *              idx, s_sel, w   [B, L, Hkv, topk]
 *            Query head h belongs to group h / (Hq/Hkv).
 *   Types    q, K, V, O, dO, kbar16: bf16 (passed as void*); scores, weights,
 *            kbar32 and every gradient: fp32; indices: int32.
 *   Memory   Every pointer is device memory owned by the caller, 16-byte
 *            aligned. The library never allocates or frees memory and keeps
 *            no state between calls; scratch comes from the caller's
 *            workspace (size from hsa_workspace_size), which starts with the
 *            call's status word (see hsa_check). The one exception is
 *            hsa_decode_noalloc, whose scratch is a fixed array inside the
 *            library.
 *   Streams  All work is enqueued on `stream`; nothing synchronises the host.
 *   Errors   Arguments are validated before any launch: a bad argument returns
 *            HSA_ERR_INVALID_ARG, a shape outside the supported set
 *            HSA_ERR_UNSUPPORTED, a short workspace HSA_ERR_WORKSPACE, and
 *            nothing is launched in these cases. A failed launch returns
 *            HSA_ERR_CUDA. Empty problems (B, L or Bq zero) return HSA_OK and
 *            launch nothing.
 *   Support  d in {64, 128}; S = 64; Hq a multiple of Hkv with
 *            G = Hq/Hkv in {1, 2, 4, 8, 16}; 1 <= topk <= 32;
 *            B * L * Hkv * topk < 2^31 and B * L * Hq < 2^31.
 *   Causality Token t (0-indexed) sees the completed chunks before its own
 *            chunk (i < t/S); a trailing partial chunk is never selectable.
 *            Fewer visible chunks than topk: all are selected and the rest of
 *            the row is padded with idx = -1, s_sel = -inf, w = 0. No visible
 *            chunk: O = 0 and no gradient.
 */
#ifndef HSA_H
#define HSA_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    HSA_OK = 0,
    HSA_ERR_INVALID_ARG = 1,
    HSA_ERR_UNSUPPORTED = 2,
    HSA_ERR_WORKSPACE = 3,
    HSA_ERR_CUDA = 4,
    HSA_ERR_TIMEOUT = 5,
    HSA_ERR_BOUNDS = 6
} hsa_status_t;

/* Variant flags (hsa_shape_t.flags, hsa_decode_shape_t.flags); 0 selects the
 * defaults: plain softmax inside a chunk, softmax chunk weights.
 *   HSA_FLAG_SOFTMAX1        softmax-off-by-one inside a chunk (§3.1.2 "Kernel
 *                            Design"): a zero logit joins every denominator.
 *   HSA_FLAG_STICK_BREAKING  stick-breaking chunk weights over I' (§3.1.1 "Chunk
 *                            Weights"): slot k (k-th latest selected chunk) gets
 *                            sigmoid(s_k) * prod_{i<k} (1 - sigmoid(s_i)).
 * Any other bit: HSA_ERR_UNSUPPORTED. */
#define HSA_FLAG_SOFTMAX1 1
#define HSA_FLAG_STICK_BREAKING 2

typedef struct {
    int B, L, Hq, Hkv, d, S, topk;
    float scale_sel;  /* c_sel; <= 0 selects 1/sqrt((Hq/Hkv) * d) */
    float scale_attn; /* c_att; <= 0 selects 1/sqrt(d) */
    int flags;        /* HSA_FLAG_*; 0: defaults */
} hsa_shape_t;

typedef struct {
    int Bq, Hq, Hkv, d, S, topk;
    long long n_chunks; /* complete chunks in the memory: the memory holds n_chunks * S tokens */
    float scale_sel;    /* <= 0 selects 1/sqrt((Hq/Hkv) * d) */
    float scale_attn;   /* <= 0 selects 1/sqrt(d) */
    int flags;          /* HSA_FLAG_*; 0: defaults */
    long long capacity_chunks; /* chunks the memory and its decode index are laid
                                  out for (a growing memory, see hsa_memory_append);
                                  0 selects n_chunks; otherwise >= n_chunks */
} hsa_decode_shape_t;

typedef enum {
    HSA_OP_SELECT = 1,
    HSA_OP_INDEX = 2,
    HSA_OP_FORWARD = 3,
    HSA_OP_BACKWARD = 4,
    HSA_OP_BACKWARD_ATTENTION = 5,
    HSA_OP_SELECT_BACKWARD = 6
} hsa_op_t;

/* Human-readable name of a status code (static storage). */
const char* hsa_status_string(hsa_status_t status);

/* Library version: major * 10000 + minor * 100 + patch. */
int hsa_version(void);

/* Number of CUDA kernels this library has launched since it was loaded (a
 * diagnostic for launch accounting; counts launches, not their completion). */
unsigned long long hsa_kernel_launches(void);

/* Bytes of the status header at the start of every workspace (256). */
size_t hsa_status_bytes(void);

/* Device-side health of the calls that used one workspace. The pipelined
 * kernels (selection on the tensor cores, forward, backward, the indexed
 * decode) give up on any internal wait that lasts longer than 2 s, instead
 * of hanging the GPU, and record it in the status word that heads the
 * workspace of their call (its first hsa_status_bytes() bytes, counted in
 * every workspace size). The library keeps no status of its own, so calls
 * on different workspaces (different streams, different threads) are
 * checked separately.
 *   ws, ws_bytes  a workspace given to earlier calls (device memory,
 *                 16-byte aligned, ws_bytes >= hsa_status_bytes()).
 * Waits for `stream` (the stream of those calls), reads and clears the
 * word, and returns HSA_ERR_TIMEOUT if a wait gave up in a call that used
 * this workspace since the word was last cleared (the results of those
 * calls are then invalid), HSA_ERR_BOUNDS if such a call found an input
 * index out of range (only a library built with the debug bounds checks,
 * see below, looks), HSA_ERR_CUDA if the stream reports an error,
 * HSA_OK otherwise; HSA_ERR_INVALID_ARG for a bad workspace.
 * Debug-bounds build (compiled with -DHSA_DEBUG_BOUNDS): every index the
 * forward, backward and index kernels read from an input array (the chunk
 * ids of idx, the offsets and slot ids of the inverse index) is checked
 * against its range before use; an out-of-range value sets the status word
 * and the access it would have made is skipped (no trap, no fault), so
 * hsa_check then returns HSA_ERR_BOUNDS. Other builds skip the checks
 * (out-of-range chunk ids still count as no selection there).
 * The word is sticky until checked, so a new workspace must start with it
 * cleared: zero its first hsa_status_bytes() bytes after allocating it (or
 * call hsa_check once and ignore the result).
 * Synchronising: not for use inside a timed region or a stream capture. */
hsa_status_t hsa_check(void* ws, size_t ws_bytes, cudaStream_t stream);

/* Self-test of that bound: launches one block that waits on a barrier nothing
 * ever completes, for at most limit_ns (1 ns to 1 s). The wait gives up, sets
 * the status word of `ws` (a workspace of at least hsa_status_bytes() bytes)
 * and the block returns, so the next hsa_check of that workspace reports
 * HSA_ERR_TIMEOUT once; the context stays usable. No device fault and no
 * hang is involved. Asynchronous on `stream`; HSA_ERR_INVALID_ARG for a limit
 * outside the range, HSA_ERR_WORKSPACE for a bad workspace. */
hsa_status_t hsa_selftest_wait_timeout(unsigned long long limit_ns, void* ws, size_t ws_bytes,
                                       cudaStream_t stream);

/* Diagnostic (no counterpart in the paper): the tensor-core score pass of
 * hsa_select_topk and hsa_decode_indexed on one tile, so that the rounding of
 * its fp32 accumulation, which the selection certificate bounds (see
 * hsa_select_topk), can be measured on the device.
 *   d      64 or 128 (else HSA_ERR_UNSUPPORTED).
 *   A      [128, d] bf16, row-major (query rows); B [64, d] bf16, row-major
 *          (chunk summaries); device memory, 16-byte aligned.
 *   C      [128, 64] fp32, output: C[r][c] = sum_e A[r][e] B[c][e] as the
 *          selection computes it (the same operand layout and the same
 *          sequence of bf16 MMAs of K = 16, accumulated in tensor memory).
 *   ws     a workspace of at least hsa_status_bytes() bytes (its status word
 *          records a wait that gave up; see hsa_check).
 * One block; asynchronous on `stream`. */
hsa_status_t hsa_selftest_score_tile(int d, const void* A, const void* B, float* C, void* ws, size_t ws_bytes,
                                     cudaStream_t stream);

/* Workspace bytes that `op` needs for `shape`: the status header (see
 * hsa_check) and the op's scratch. 0 for an empty problem (B or L zero),
 * whose call launches nothing and takes no workspace, and for an invalid
 * shape (the call itself then reports the error). */
size_t hsa_workspace_size(int op, const hsa_shape_t* shape);

/* Workspace bytes of hsa_decode for `shape`. */
size_t hsa_decode_workspace_size(const hsa_decode_shape_t* shape);

/*
 * Chunk mean pool (§3.1 "Chunk Selection": K̄_i is the mean-pooled chunk
 * representation; Appendix A, Eq. 3: q·K̄_c equals the mean of the chunk's
 * token logits).
 *   K      [B, L, Hkv, d] bf16, input.
 *   kbar32 [B, L/S, Hkv, d] fp32, output: fp32 sum in token order, divided by S.
 *   kbar16 [B, L/S, Hkv, d] bf16, output (may be NULL): round-to-nearest-even of kbar32.
 * Rows of a trailing partial chunk are not read.
 */
hsa_status_t hsa_chunk_pool(const hsa_shape_t* shape, const void* K, float* kbar32, void* kbar16,
                            cudaStream_t stream);

/*
 * Top-k chunk selection per token and GQA group (§3.1 "Chunk Selection": the
 * score q̂·K̂/sqrt(d_g) over visible chunks and I = {i : rank(s_i) < k}; §3.1.1
 * "Chunk Weights": I' lists the chosen chunks by decreasing index).
 *   q      [B, L, Hq, d] bf16, input.
 *   kbar32 [B, L/S, Hkv, d] fp32, input (from hsa_chunk_pool).
 *   idx    [B, L, Hkv, topk] int32, output: chosen chunks, decreasing index, -1 padded.
 *   s_sel  [B, L, Hkv, topk] fp32, output: their scores, -inf padded.
 * Scores are fp32: q̂ = fp32 sum of the group's heads in head order,
 * dot = fused multiply-add chain over d in order, s = dot * c_sel. The score
 * matrix is never written to memory. For topk <= 16 the scan runs as bf16
 * tensor-core products whose rounding error is bounded per score; only the
 * chunks the bound cannot rule out are rescored with the fp32 chain, so idx
 * and s_sel are exactly those of the definition above. Needs workspace
 * HSA_OP_SELECT (for topk > 16, where every score is computed with the fp32
 * chain, only its status header).
 */
hsa_status_t hsa_select_topk(const hsa_shape_t* shape, const void* q, const float* kbar32, int32_t* idx,
                             float* s_sel, void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * Inverse selection index (replaces the mask M and rank R of §3.1.2, used by
 * Algorithm 3): for every (b, g, chunk i) the list of selection slots that
 * chose it, as a CSR over keys key = (b * Hkv + g) * (L/S) + i:
 *   offsets [B*Hkv*(L/S) + 1] int32, output: entries of key k are
 *           entries[offsets[k] .. offsets[k+1]).
 *   entries [B*L*Hkv*topk] int32, output (capacity): the flat slot index
 *           p = ((b*L + t)*Hkv + g)*topk + j of idx, in increasing p (so in
 *           increasing token order) within each key. Positions from
 *           offsets[B*Hkv*(L/S)] on are unspecified.
 * Deterministic (a stable counting sort when Hkv*(L/S) <= 4096, else a stable
 * radix sort); needs workspace HSA_OP_INDEX.
 */
hsa_status_t hsa_build_index(const hsa_shape_t* shape, const int32_t* idx, int32_t* offsets, int32_t* entries,
                             void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * Hierarchical attention forward (§3.1.1 "Hierarchical Attention", Algorithm
 * 1; chunk weights by softmax over the selected scores, the "w/o s.b."
 * variant of §4.1).
 *   q [B,L,Hq,d], K, V [B,L,Hkv,d] bf16; idx, s_sel from hsa_select_topk;
 *   offsets, entries from hsa_build_index (same idx).
 *   O [B,L,Hq,d] bf16, output.  w [B,L,Hkv,topk] fp32, output (0 at padded slots).
 * Needs workspace HSA_OP_FORWARD. Chunk-major: each (b, g, chunk) tile of K
 * and V is read once and shared by every query head that selected it.
 */
hsa_status_t hsa_forward(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                         const int32_t* idx, const float* s_sel, const int32_t* offsets, const int32_t* entries,
                         void* O, float* w, void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * Backward (Algorithm 2: dq and the chunk-weight gradient; Algorithm 3: dK,
 * dV per chunk; Appendix A: the chunk weights carry gradient into the
 * selection scores, hence into q, K̄ and, through the mean pool, K).
 *   Inputs as in hsa_forward plus kbar32, the forward's w and O, and dO [B,L,Hq,d] bf16.
 *   dq [B,L,Hq,d], dK, dV [B,L,Hkv,d] fp32, outputs (fully written).
 * Deterministic: every dK/dV row is owned by one thread block that walks its
 * chunk's entries in index order; no floating-point atomics.
 * Variants (shape->flags): softmax-off-by-one recomputes P with the zero
 * logit; with stick-breaking weights the score gradient of a slot depends on
 * the later slots' dw (ds_j = (1 - b_j) w_j dw_j - b_j sum_{k>j} w_k dw_k,
 * b = sigmoid(s)), so the chunk pass writes dw per slot and three more passes
 * add the selection terms (ds from w and dw; c_sel ds K̄ into dq; the mean-pool
 * share of dK̄ into dK, per chunk in index order). b is recovered from w
 * (b_j = w_j / (1 - sum_{i<j} w_i)), so s_sel is not an input.
 * Needs workspace HSA_OP_BACKWARD (larger with stick-breaking weights).
 */
hsa_status_t hsa_backward(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                          const float* kbar32, const int32_t* idx, const float* w, const void* O, const void* dO,
                          const int32_t* offsets, const int32_t* entries, float* dq, float* dK, float* dV,
                          void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * Layers that share one selection (the paper shares K, V and the retrieved
 * chunks across its HSA layers, §3.1, and may select with its own q_sel and
 * K^slc): each layer's backward is hsa_backward_attention, which adds that
 * layer's score gradient into ds_accum; the selection chain then runs once,
 * hsa_select_backward, on the summed ds. hsa_backward equals
 * hsa_backward_attention followed by hsa_select_backward with q_sel = q and
 * K^slc = K (outputs added).
 *
 * hsa_backward_attention (Algorithms 2 and 3 without the selection chain):
 *   Inputs as in hsa_backward, without kbar32 and O.
 *   dq [B,L,Hq,d], dK, dV [B,L,Hkv,d] fp32: the attention's gradients (fully written).
 *   ds_accum [B,L,Hkv,topk] fp32, in/out: ds of every slot is added (padding
 *     slots add 0); ds_j = w_j (dw_j - sum_k w_k dw_k) for softmax weights, the
 *     stick-breaking form for HSA_FLAG_STICK_BREAKING (see hsa_backward).
 *   Needs workspace HSA_OP_BACKWARD_ATTENTION.
 */
hsa_status_t hsa_backward_attention(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                                    const int32_t* idx, const float* w, const void* dO, const int32_t* offsets,
                                    const int32_t* entries, float* dq, float* dK, float* dV, float* ds_accum,
                                    void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * hsa_select_backward (Appendix A: the selection scores s = c_sel q̂_sel·K̄_sel
 * receive gradient through the chunk weights):
 *   shape    the selection problem: B, L, S, topk, Hkv, Hq and d of q_sel
 *            (d_sel in {64, 128}), scale_sel; flags and scale_attn unused.
 *   q_sel    [B,L,Hq,d] bf16; kbar_sel [B,L/S,Hkv,d] fp32 (hsa_chunk_pool of K^slc);
 *   idx, offsets, entries: the shared selection and its inverse index;
 *   ds       [B,L,Hkv,topk] fp32 (summed over the layers).
 *   dq_sel   [B,L,Hq,d] fp32 = c_sel sum_j ds_j K̄_sel[I_j] for every head of the
 *            group (fully written).
 *   dK_sel   [B,L,Hkv,d] fp32: dK̄_sel / S on the S rows of every complete
 *            chunk, dK̄_sel[i] = c_sel sum over the slots that chose i of ds q̂_sel
 *            (in index order); 0 elsewhere (fully written).
 *   Needs workspace HSA_OP_SELECT_BACKWARD.
 */
hsa_status_t hsa_select_backward(const hsa_shape_t* shape, const void* q_sel, const float* kbar_sel,
                                 const int32_t* idx, const float* ds, const int32_t* offsets, const int32_t* entries,
                                 float* dq_sel, float* dK_sel, void* ws, size_t ws_bytes, cudaStream_t stream);

/*
 * Decode against a resident memory (§3.2 "Inference": only the chunk
 * summaries are scanned on every step, then the k selected chunks are
 * fetched). One query token per batch row; all n_chunks chunks are visible.
 *   K_mem, V_mem [n_chunks*S, Hkv, d] bf16 (the memory). Device memory, or
 *          page-locked host memory that the device reads at the same address
 *          (cudaHostAlloc, cudaMallocHost, or cudaHostRegister with
 *          cudaHostRegisterMapped): a memory larger than HBM then stays in
 *          host memory and only the k selected chunks per query cross the
 *          CPU-GPU link, with results identical to a device-resident memory.
 *          Pageable or unknown memory returns HSA_ERR_INVALID_ARG before any
 *          launch (checked with cudaPointerGetAttributes on every call).
 *   kbar32 [n_chunks, Hkv, d] fp32 (hsa_chunk_pool of K_mem with B = 1),
 *          device memory.
 *   q, O [Bq, Hq, d] bf16, idx, s_sel, w [Bq, Hkv, topk]: device memory.
 * Needs workspace hsa_decode_workspace_size.
 */
hsa_status_t hsa_decode(const hsa_decode_shape_t* shape, const void* q, const void* K_mem, const void* V_mem,
                        const float* kbar32, void* O, int32_t* idx, float* s_sel, float* w, void* ws,
                        size_t ws_bytes, cudaStream_t stream);

/*
 * Decode index of a resident memory, built once per memory and reused by
 * every hsa_decode_indexed call (§3.2 "Inference": the chunk summaries are
 * what each decoding step scans). It holds the summaries rounded to bf16 in
 * [Hkv][C][d] order, |K̄_i| per chunk and its maximum over every 64 chunks,
 * laid out for C = capacity_chunks (n_chunks when 0) chunks; the n_chunks
 * present are written and every other byte is zeroed, so that
 * hsa_memory_append can enter chunks as they complete. Size from
 * hsa_decode_index_size (0 when topk > 16 or C = 0: hsa_decode_indexed then
 * needs no index). Only shape's Hkv, d, n_chunks, capacity_chunks and topk
 * matter; Bq may be 0.
 *   kbar32 [n_chunks, Hkv, d] fp32 (hsa_chunk_pool of the memory, B = 1);
 *          may be NULL when n_chunks = 0.
 *   index  device memory, caller-owned, 16-byte aligned.
 */
size_t hsa_decode_index_size(const hsa_decode_shape_t* shape);
hsa_status_t hsa_decode_index(const hsa_decode_shape_t* shape, const float* kbar32, void* index, size_t index_bytes,
                              cudaStream_t stream);

/* Workspace bytes of hsa_decode_indexed for `shape`. */
size_t hsa_decode_indexed_workspace_size(const hsa_decode_shape_t* shape);

/*
 * hsa_decode with the memory index: same arguments and results (idx and s_sel
 * identical, O and w to fp32 rounding), with the scan of the summaries on the
 * tensor cores. Blocks over ranges of the memory score bf16 summaries against
 * the group query; per query and range, the scores' rounding error is bounded
 * (|error| < 2^-7 * 9/8 * |q̂| |K̄_i|), so only the chunks that bound cannot rule out
 * are kept, and those are rescored with the fp32 chain of hsa_select_topk
 * before the top-k is taken. For topk > 16 it falls back to hsa_decode's scan
 * (index may then be NULL).
 */
hsa_status_t hsa_decode_indexed(const hsa_decode_shape_t* shape, const void* q, const void* K_mem, const void* V_mem,
                                const float* kbar32, const void* index, void* O, int32_t* idx, float* s_sel, float* w,
                                void* ws, size_t ws_bytes, cudaStream_t stream);

/* Size of the scratch array behind hsa_decode_noalloc (one per device): 8 MiB. */
#define HSA_DECODE_NOALLOC_SCRATCH_BYTES (8u << 20)

/*
 * hsa_decode without a workspace argument: the paper has no counterpart; this
 * is a calling convention for callers that cannot allocate device memory when
 * they decode (a host that embeds the decoder under a device-memory budget
 * fixed at start-up, or a serving loop that must stay out of the allocator,
 * whose cudaMalloc/cudaFree may synchronise the device, between tokens).
 *   Arguments, results and numerics as in hsa_decode (same kernels). The
 *   library allocates nothing: its scratch is a fixed device array of
 *   HSA_DECODE_NOALLOC_SCRATCH_BYTES compiled into the library, one per device.
 *   Limit: a shape whose hsa_decode_workspace_size exceeds that size returns
 *   HSA_ERR_WORKSPACE before any launch (the decode of 64 queries, 8 heads in
 *   one group, d = 128, k = 8 needs about 3.4 MB at any memory length).
 *   First call on each device: looks up the array's address on the current
 *   device (cudaGetSymbolAddress) and caches it; make that first call before
 *   any stream capture on that device.
 *   Nothing in the array needs to start at zero.
 *   Races: every call on a device uses the same array, so calls that can
 *   overlap on one device (different streams, different host threads) corrupt
 *   each other's results; the caller serialises them.
 */
hsa_status_t hsa_decode_noalloc(const hsa_decode_shape_t* shape, const void* q, const void* K_mem,
                                const void* V_mem, const float* kbar32, void* O, int32_t* idx, float* s_sel,
                                float* w, cudaStream_t stream);

/*
 * Append tokens to a growing decode memory (§3.2 "Inference": the memory grows
 * as tokens are decoded, a chunk is summarised once its S tokens are present,
 * and only completed chunks are selectable). One launch stores the new rows of
 * K and V and pools every chunk they complete (the fp32 token-order sum and
 * division of hsa_chunk_pool: summaries bit-identical to pooling the final
 * memory at once); a second enters those chunks in the decode index (rows
 * bit-identical to hsa_decode_index of the final memory with the same
 * capacity).
 *   shape    Hkv, d, S, topk, flags and capacity C = capacity_chunks (or
 *            n_chunks when 0); Bq and Hq are unused but must be valid.
 *   n_tokens tokens already in the memory (rows 0 .. n_tokens-1 written);
 *            n_new tokens are appended: n_tokens + n_new <= C * S, else
 *            HSA_ERR_INVALID_ARG.
 *   K_new, V_new [n_new, Hkv, d] bf16. K_new may be the memory's own rows
 *            from n_tokens on (a prefill that wrote them in place); otherwise
 *            no argument may overlap another.
 *   K_mem, V_mem [C*S, Hkv, d] bf16: device memory, or mapped page-locked host
 *            memory as in hsa_decode (checked the same way, as are K_new, V_new).
 *   kbar32   [C, Hkv, d] fp32, device memory: the summaries of the chunks that
 *            the append completes are written; the rest is untouched.
 *   index    the decode index (hsa_decode_index_size of shape, index_bytes at
 *            least that, else HSA_ERR_WORKSPACE) built by hsa_decode_index with
 *            the same capacity, before the first append (any n_chunks <= C,
 *            including 0) and kept by every append since; or NULL when the
 *            memory is only decoded with hsa_decode. A non-null index with
 *            topk > 16 returns HSA_ERR_UNSUPPORTED.
 * After the call, decode with n_chunks = floor((n_tokens + n_new) / S) and the
 * same capacity_chunks. The trailing incomplete chunk's rows are stored but
 * not selectable until an append completes it. Enqueued on `stream`.
 */
hsa_status_t hsa_memory_append(const hsa_decode_shape_t* shape, long long n_tokens, long long n_new,
                               const void* K_new, const void* V_new, void* K_mem, void* V_mem, float* kbar32,
                               void* index, size_t index_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* HSA_H */
