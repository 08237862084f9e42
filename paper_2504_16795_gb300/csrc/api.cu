// C ABI of the HSA hot path: argument validation, workspace sizing and
// dispatch to the kernels. Nothing here allocates device memory; every check
// runs before the first launch.
#include <atomic>
#include <cmath>
#include <cstdint>

#include "common.cuh"

namespace hsa {
static std::atomic<unsigned long long> g_launches{0};
void note_launches(unsigned long long n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace hsa

namespace {

using hsa::Dims;

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

bool pow2_group(int G) { return G == 1 || G == 2 || G == 4 || G == 8 || G == 16; }

// Validates a prefill shape; fills Dims on success.
hsa_status_t resolve(const hsa_shape_t* s, Dims* out) {
  if (s == nullptr) return HSA_ERR_INVALID_ARG;
  if (s->B < 0 || s->L < 0 || s->Hq <= 0 || s->Hkv <= 0 || s->d <= 0 || s->S <= 0 || s->topk <= 0)
    return HSA_ERR_INVALID_ARG;
  if (s->Hq % s->Hkv != 0) return HSA_ERR_INVALID_ARG;
  if (std::isnan(s->scale_sel) || std::isnan(s->scale_attn) || std::isinf(s->scale_sel) ||
      std::isinf(s->scale_attn))
    return HSA_ERR_INVALID_ARG;
  const int G = s->Hq / s->Hkv;
  if (!pow2_group(G)) return HSA_ERR_UNSUPPORTED;
  if (s->d != 64 && s->d != 128) return HSA_ERR_UNSUPPORTED;
  if (s->S != hsa::kChunk) return HSA_ERR_UNSUPPORTED;
  if (s->topk > 32) return HSA_ERR_UNSUPPORTED;
  if (s->flags & ~(HSA_FLAG_SOFTMAX1 | HSA_FLAG_STICK_BREAKING)) return HSA_ERR_UNSUPPORTED;
  const long long slots = (long long)s->B * s->L * s->Hkv * s->topk;
  if (slots >= (1LL << 31)) return HSA_ERR_UNSUPPORTED;
  const long long rows = (long long)s->B * s->L * s->Hq;  // query rows are indexed in int32
  if (rows >= (1LL << 31)) return HSA_ERR_UNSUPPORTED;
  Dims D;
  D.B = s->B;
  D.L = s->L;
  D.Hq = s->Hq;
  D.Hkv = s->Hkv;
  D.d = s->d;
  D.S = s->S;
  D.topk = s->topk;
  D.G = G;
  D.Nc = s->L / s->S;
  D.scale_sel = s->scale_sel > 0.f ? s->scale_sel : (float)(1.0 / std::sqrt((double)G * s->d));
  D.scale_attn = s->scale_attn > 0.f ? s->scale_attn : (float)(1.0 / std::sqrt((double)s->d));
  D.softmax1 = (s->flags & HSA_FLAG_SOFTMAX1) != 0;
  D.stick = (s->flags & HSA_FLAG_STICK_BREAKING) != 0;
  *out = D;
  return HSA_OK;
}

bool empty(const Dims& D) { return D.B == 0 || D.L == 0; }

hsa_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? HSA_OK : HSA_ERR_CUDA; }

#define HSA_REQUIRE_PTR(p)                          \
  do {                                              \
    if ((p) == nullptr || !aligned16(p)) return HSA_ERR_INVALID_ARG; \
  } while (0)

using hsa::kStatusBytes;

// A caller workspace is the status header followed by `body` bytes of scratch:
// checks its size and alignment and returns the two parts.
hsa_status_t split_ws(void* ws, size_t ws_bytes, size_t body, unsigned** status, void** scratch) {
  if (ws == nullptr || !aligned16(ws) || ws_bytes < kStatusBytes + body) return HSA_ERR_WORKSPACE;
  *status = (unsigned*)ws;
  *scratch = (char*)ws + kStatusBytes;
  return HSA_OK;
}

}  // namespace

extern "C" {

const char* hsa_status_string(hsa_status_t status) {
  switch (status) {
    case HSA_OK: return "HSA_OK";
    case HSA_ERR_INVALID_ARG: return "HSA_ERR_INVALID_ARG: null, misaligned or inconsistent argument";
    case HSA_ERR_UNSUPPORTED: return "HSA_ERR_UNSUPPORTED: shape outside the supported set";
    case HSA_ERR_WORKSPACE: return "HSA_ERR_WORKSPACE: workspace missing or too small";
    case HSA_ERR_CUDA: return "HSA_ERR_CUDA: a kernel launch failed";
    case HSA_ERR_TIMEOUT: return "HSA_ERR_TIMEOUT: a device-side wait gave up (results invalid)";
    case HSA_ERR_BOUNDS: return "HSA_ERR_BOUNDS: an input index was out of range (debug-bounds build; results invalid)";
  }
  return "HSA_ERR_UNKNOWN";
}

int hsa_version(void) { return 100; }

unsigned long long hsa_kernel_launches(void) { return hsa::g_launches.load(std::memory_order_relaxed); }

hsa_status_t hsa_check(void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (ws == nullptr || !aligned16(ws) || ws_bytes < kStatusBytes) return HSA_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return HSA_ERR_CUDA;
  unsigned v = 0;
  if (cudaMemcpyAsync(&v, ws, sizeof(v), cudaMemcpyDeviceToHost, stream) != cudaSuccess ||
      cudaMemsetAsync(ws, 0, sizeof(v), stream) != cudaSuccess || cudaStreamSynchronize(stream) != cudaSuccess)
    return HSA_ERR_CUDA;
  return (v & hsa::kStatusTimeout) ? HSA_ERR_TIMEOUT : (v ? HSA_ERR_BOUNDS : HSA_OK);
}

size_t hsa_status_bytes(void) { return kStatusBytes; }

hsa_status_t hsa_selftest_wait_timeout(unsigned long long limit_ns, void* ws, size_t ws_bytes,
                                       cudaStream_t stream) {
  if (limit_ns == 0 || limit_ns > 1000000000ull) return HSA_ERR_INVALID_ARG;
  unsigned* status = nullptr;
  void* scratch = nullptr;
  hsa_status_t st = split_ws(ws, ws_bytes, 0, &status, &scratch);
  if (st != HSA_OK) return st;
  return hsa::launch_selftest_wait(limit_ns, status, stream) == cudaSuccess ? HSA_OK : HSA_ERR_CUDA;
}

hsa_status_t hsa_selftest_score_tile(int d, const void* A, const void* B, float* C, void* ws, size_t ws_bytes,
                                     cudaStream_t stream) {
  if (d != 64 && d != 128) return HSA_ERR_UNSUPPORTED;
  HSA_REQUIRE_PTR(A);
  HSA_REQUIRE_PTR(B);
  HSA_REQUIRE_PTR(C);
  unsigned* status = nullptr;
  void* scratch = nullptr;
  hsa_status_t st = split_ws(ws, ws_bytes, 0, &status, &scratch);
  if (st != HSA_OK) return st;
  return cuda_status(hsa::launch_selftest_score_tile(d, A, B, C, status, stream));
}

size_t hsa_workspace_size(int op, const hsa_shape_t* shape) {
  Dims D;
  if (resolve(shape, &D) != HSA_OK) return 0;
  if (empty(D)) return 0;
  switch (op) {
    case HSA_OP_SELECT: return kStatusBytes + (hsa::select_tc_applies(D) ? hsa::select_tc_workspace(D) : 0);
    case HSA_OP_INDEX: return kStatusBytes + hsa::index_workspace(D);
    case HSA_OP_FORWARD: return kStatusBytes + hsa::forward_workspace(D);
    case HSA_OP_BACKWARD: return kStatusBytes + hsa::backward_workspace(D);
    case HSA_OP_BACKWARD_ATTENTION: return kStatusBytes + hsa::backward_attention_workspace(D);
    case HSA_OP_SELECT_BACKWARD: return kStatusBytes + hsa::select_backward_workspace(D);
  }
  return 0;
}

hsa_status_t hsa_chunk_pool(const hsa_shape_t* shape, const void* K, float* kbar32, void* kbar16,
                            cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D) || D.Nc == 0) return HSA_OK;
  HSA_REQUIRE_PTR(K);
  HSA_REQUIRE_PTR(kbar32);
  if (kbar16 != nullptr && !aligned16(kbar16)) return HSA_ERR_INVALID_ARG;
  return cuda_status(hsa::launch_pool(D, K, kbar32, kbar16, stream));
}

hsa_status_t hsa_select_topk(const hsa_shape_t* shape, const void* q, const float* kbar32, int32_t* idx,
                             float* s_sel, void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(s_sel);
  if (D.Nc > 0) HSA_REQUIRE_PTR(kbar32);
  const bool tc = hsa::select_tc_applies(D);
  void* scratch = nullptr;
  st = split_ws(ws, ws_bytes, tc ? hsa::select_tc_workspace(D) : 0, &D.status, &scratch);
  if (st != HSA_OK) return st;
  if (tc) return cuda_status(hsa::launch_select_tc(D, q, kbar32, idx, s_sel, scratch, stream));
  return cuda_status(hsa::launch_select(D, q, kbar32, idx, s_sel, stream));
}

hsa_status_t hsa_build_index(const hsa_shape_t* shape, const int32_t* idx, int32_t* offsets, int32_t* entries,
                             void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  HSA_REQUIRE_PTR(offsets);
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(entries);
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::index_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  return cuda_status(hsa::launch_index(D, idx, offsets, entries, scratch, stream));
}

hsa_status_t hsa_forward(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                         const int32_t* idx, const float* s_sel, const int32_t* offsets, const int32_t* entries,
                         void* O, float* w, void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(K);
  HSA_REQUIRE_PTR(V);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(s_sel);
  HSA_REQUIRE_PTR(offsets);
  HSA_REQUIRE_PTR(entries);
  HSA_REQUIRE_PTR(O);
  HSA_REQUIRE_PTR(w);
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::forward_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  return cuda_status(hsa::launch_forward(D, q, K, V, idx, s_sel, offsets, entries, O, w, scratch, stream));
}

hsa_status_t hsa_backward(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                          const float* kbar32, const int32_t* idx, const float* w, const void* O, const void* dO,
                          const int32_t* offsets, const int32_t* entries, float* dq, float* dK, float* dV,
                          void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(K);
  HSA_REQUIRE_PTR(V);
  if (D.Nc > 0) HSA_REQUIRE_PTR(kbar32);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(w);
  HSA_REQUIRE_PTR(O);
  HSA_REQUIRE_PTR(dO);
  HSA_REQUIRE_PTR(offsets);
  HSA_REQUIRE_PTR(entries);
  HSA_REQUIRE_PTR(dq);
  HSA_REQUIRE_PTR(dK);
  HSA_REQUIRE_PTR(dV);
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::backward_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  return cuda_status(
      hsa::launch_backward(D, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq, dK, dV, scratch, stream));
}

hsa_status_t hsa_backward_attention(const hsa_shape_t* shape, const void* q, const void* K, const void* V,
                                    const int32_t* idx, const float* w, const void* dO, const int32_t* offsets,
                                    const int32_t* entries, float* dq, float* dK, float* dV, float* ds_accum,
                                    void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(K);
  HSA_REQUIRE_PTR(V);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(w);
  HSA_REQUIRE_PTR(dO);
  HSA_REQUIRE_PTR(offsets);
  HSA_REQUIRE_PTR(entries);
  HSA_REQUIRE_PTR(dq);
  HSA_REQUIRE_PTR(dK);
  HSA_REQUIRE_PTR(dV);
  HSA_REQUIRE_PTR(ds_accum);
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::backward_attention_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  return cuda_status(hsa::launch_backward_attention(D, q, K, V, idx, w, dO, offsets, entries, dq, dK, dV, ds_accum,
                                                    scratch, stream));
}

hsa_status_t hsa_select_backward(const hsa_shape_t* shape, const void* q_sel, const float* kbar_sel,
                                 const int32_t* idx, const float* ds, const int32_t* offsets, const int32_t* entries,
                                 float* dq_sel, float* dK_sel, void* ws, size_t ws_bytes, cudaStream_t stream) {
  Dims D;
  hsa_status_t st = resolve(shape, &D);
  if (st != HSA_OK) return st;
  if (empty(D)) return HSA_OK;
  HSA_REQUIRE_PTR(q_sel);
  if (D.Nc > 0) HSA_REQUIRE_PTR(kbar_sel);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(ds);
  HSA_REQUIRE_PTR(offsets);
  HSA_REQUIRE_PTR(entries);
  HSA_REQUIRE_PTR(dq_sel);
  HSA_REQUIRE_PTR(dK_sel);
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::select_backward_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  return cuda_status(
      hsa::launch_select_backward(D, q_sel, kbar_sel, idx, ds, offsets, entries, dq_sel, dK_sel, scratch, stream));
}

namespace {
hsa_status_t resolve_decode(const hsa_decode_shape_t* s, hsa::DecodeDims* out) {
  if (s == nullptr) return HSA_ERR_INVALID_ARG;
  if (s->Bq < 0 || s->Hq <= 0 || s->Hkv <= 0 || s->d <= 0 || s->S <= 0 || s->topk <= 0 || s->n_chunks < 0)
    return HSA_ERR_INVALID_ARG;
  if (s->Hq % s->Hkv != 0) return HSA_ERR_INVALID_ARG;
  if (std::isnan(s->scale_sel) || std::isnan(s->scale_attn) || std::isinf(s->scale_sel) ||
      std::isinf(s->scale_attn))
    return HSA_ERR_INVALID_ARG;
  const int G = s->Hq / s->Hkv;
  if (!pow2_group(G)) return HSA_ERR_UNSUPPORTED;
  if (s->d != 64 && s->d != 128) return HSA_ERR_UNSUPPORTED;
  if (s->S != hsa::kChunk) return HSA_ERR_UNSUPPORTED;
  if (s->topk > 32) return HSA_ERR_UNSUPPORTED;
  if (s->n_chunks >= (1LL << 31)) return HSA_ERR_UNSUPPORTED;
  if (s->capacity_chunks < 0 || (s->capacity_chunks > 0 && s->capacity_chunks < s->n_chunks))
    return HSA_ERR_INVALID_ARG;
  if (s->capacity_chunks >= (1LL << 31)) return HSA_ERR_UNSUPPORTED;
  if (s->flags & ~(HSA_FLAG_SOFTMAX1 | HSA_FLAG_STICK_BREAKING)) return HSA_ERR_UNSUPPORTED;
  if ((long long)s->Bq * s->Hkv * s->topk >= (1LL << 31)) return HSA_ERR_UNSUPPORTED;
  hsa::DecodeDims D;
  D.Bq = s->Bq;
  D.Hq = s->Hq;
  D.Hkv = s->Hkv;
  D.d = s->d;
  D.S = s->S;
  D.topk = s->topk;
  D.G = G;
  D.Nc = s->n_chunks;
  D.cap = s->capacity_chunks > 0 ? s->capacity_chunks : s->n_chunks;
  D.scale_sel = s->scale_sel > 0.f ? s->scale_sel : (float)(1.0 / std::sqrt((double)G * s->d));
  D.scale_attn = s->scale_attn > 0.f ? s->scale_attn : (float)(1.0 / std::sqrt((double)s->d));
  D.softmax1 = (s->flags & HSA_FLAG_SOFTMAX1) != 0;
  D.stick = (s->flags & HSA_FLAG_STICK_BREAKING) != 0;
  *out = D;
  return HSA_OK;
}
}  // namespace

size_t hsa_decode_workspace_size(const hsa_decode_shape_t* shape) {
  hsa::DecodeDims D;
  if (resolve_decode(shape, &D) != HSA_OK || D.Bq == 0) return 0;
  return kStatusBytes + hsa::decode_workspace(D);
}

hsa_status_t hsa_decode(const hsa_decode_shape_t* shape, const void* q, const void* K_mem, const void* V_mem,
                        const float* kbar32, void* O, int32_t* idx, float* s_sel, float* w, void* ws,
                        size_t ws_bytes, cudaStream_t stream) {
  hsa::DecodeDims D;
  hsa_status_t st = resolve_decode(shape, &D);
  if (st != HSA_OK) return st;
  if (D.Bq == 0) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(O);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(s_sel);
  HSA_REQUIRE_PTR(w);
  if (D.Nc > 0) {
    HSA_REQUIRE_PTR(K_mem);
    HSA_REQUIRE_PTR(V_mem);
    HSA_REQUIRE_PTR(kbar32);
  }
  void* scratch = nullptr;
  if ((st = split_ws(ws, ws_bytes, hsa::decode_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  if (D.Nc > 0 && !(hsa::memory_device_readable(K_mem) && hsa::memory_device_readable(V_mem)))
    return HSA_ERR_INVALID_ARG;
  return cuda_status(hsa::launch_decode(D, q, K_mem, V_mem, kbar32, O, idx, s_sel, w, scratch, stream));
}

size_t hsa_decode_index_size(const hsa_decode_shape_t* shape) {
  hsa::DecodeDims D;
  if (resolve_decode(shape, &D) != HSA_OK) return 0;
  return hsa::decode_index_bytes(D);
}

hsa_status_t hsa_decode_index(const hsa_decode_shape_t* shape, const float* kbar32, void* index, size_t index_bytes,
                              cudaStream_t stream) {
  hsa::DecodeDims D;
  hsa_status_t st = resolve_decode(shape, &D);
  if (st != HSA_OK) return st;
  if (!hsa::decode_index_applies(D)) return D.cap == 0 ? HSA_OK : HSA_ERR_UNSUPPORTED;
  if (D.Nc > 0) HSA_REQUIRE_PTR(kbar32);
  const size_t need = hsa::decode_index_bytes(D);
  if (index_bytes < need || index == nullptr || !aligned16(index)) return HSA_ERR_WORKSPACE;
  return cuda_status(hsa::launch_decode_index(D, kbar32, index, stream));
}

size_t hsa_decode_indexed_workspace_size(const hsa_decode_shape_t* shape) {
  hsa::DecodeDims D;
  if (resolve_decode(shape, &D) != HSA_OK || D.Bq == 0) return 0;
  return kStatusBytes + (hsa::decode_tc_applies(D) ? hsa::decode_tc_workspace(D) : hsa::decode_workspace(D));
}

hsa_status_t hsa_decode_indexed(const hsa_decode_shape_t* shape, const void* q, const void* K_mem, const void* V_mem,
                                const float* kbar32, const void* index, void* O, int32_t* idx, float* s_sel, float* w,
                                void* ws, size_t ws_bytes, cudaStream_t stream) {
  hsa::DecodeDims D;
  hsa_status_t st = resolve_decode(shape, &D);
  if (st != HSA_OK) return st;
  if (D.Bq == 0) return HSA_OK;
  HSA_REQUIRE_PTR(q);
  HSA_REQUIRE_PTR(O);
  HSA_REQUIRE_PTR(idx);
  HSA_REQUIRE_PTR(s_sel);
  HSA_REQUIRE_PTR(w);
  if (D.Nc > 0) {
    HSA_REQUIRE_PTR(K_mem);
    HSA_REQUIRE_PTR(V_mem);
    HSA_REQUIRE_PTR(kbar32);
  }
  void* scratch = nullptr;
  if (!hsa::decode_tc_applies(D)) {  // k > 16 or an empty memory: the CUDA-core scan of hsa_decode
    if ((st = split_ws(ws, ws_bytes, hsa::decode_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
    if (D.Nc > 0 && !(hsa::memory_device_readable(K_mem) && hsa::memory_device_readable(V_mem)))
      return HSA_ERR_INVALID_ARG;
    return cuda_status(hsa::launch_decode(D, q, K_mem, V_mem, kbar32, O, idx, s_sel, w, scratch, stream));
  }
  HSA_REQUIRE_PTR(index);
  if ((st = split_ws(ws, ws_bytes, hsa::decode_tc_workspace(D), &D.status, &scratch)) != HSA_OK) return st;
  if (!(hsa::memory_device_readable(K_mem) && hsa::memory_device_readable(V_mem))) return HSA_ERR_INVALID_ARG;
  return cuda_status(hsa::launch_decode_tc(D, q, K_mem, V_mem, kbar32, index, O, idx, s_sel, w, scratch, stream));
}

hsa_status_t hsa_memory_append(const hsa_decode_shape_t* shape, long long n_tokens, long long n_new,
                               const void* K_new, const void* V_new, void* K_mem, void* V_mem, float* kbar32,
                               void* index, size_t index_bytes, cudaStream_t stream) {
  hsa::DecodeDims D;
  hsa_status_t st = resolve_decode(shape, &D);
  if (st != HSA_OK) return st;
  if (n_tokens < 0 || n_new < 0 || n_tokens > D.cap * D.S - n_new) return HSA_ERR_INVALID_ARG;
  if (n_new == 0) return HSA_OK;
  HSA_REQUIRE_PTR(K_new);
  HSA_REQUIRE_PTR(V_new);
  HSA_REQUIRE_PTR(K_mem);
  HSA_REQUIRE_PTR(V_mem);
  HSA_REQUIRE_PTR(kbar32);
  if (index != nullptr) {
    if (!hsa::decode_index_applies(D)) return HSA_ERR_UNSUPPORTED;
    if (index_bytes < hsa::decode_index_bytes(D) || !aligned16(index)) return HSA_ERR_WORKSPACE;
  }
  const void* rows[] = {K_new, V_new, K_mem, V_mem};
  for (const void* p : rows)
    if (!hsa::memory_device_readable(p)) return HSA_ERR_INVALID_ARG;
  return cuda_status(
      hsa::launch_memory_append(D, n_tokens, n_new, K_new, V_new, K_mem, V_mem, kbar32, index, stream));
}

}  // extern "C"

hsa_status_t hsa::resolve_decode_shape(const hsa_decode_shape_t* s, hsa::DecodeDims* out) {
  return resolve_decode(s, out);
}
