// Decode with scratch owned by the library (hsa_decode_noalloc).
//
// Some callers cannot hand the library a workspace: a host that embeds the
// decoder under a device-memory budget fixed when it starts, or a serving loop
// that must not enter the allocator between tokens (cudaMalloc and cudaFree may
// synchronise the device). For them this entry point runs the same kernels as
// hsa_decode with its scratch in a fixed array compiled into the library, one
// per device, and allocates nothing.
//
// Set-up: the first call on a device looks up that device's copy of the array
// (cudaGetSymbolAddress, with the device current) and caches the address
// together with the device's current context; that first call should come
// before any stream capture on the device. A call whose stream belongs to
// another device than the current one is refused. After a device reset the
// context differs, so the address is looked up again. Calls that may overlap
// on one device share the array and race on it; callers serialise them.
// Nothing in the array has to start at zero: each call writes every byte it
// later reads.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"

namespace {

constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[HSA_DECODE_NOALLOC_SCRATCH_BYTES];

std::mutex g_scratch_mu;
struct Cached {
  CUcontext ctx;
  void* ptr;
};
Cached g_scratch[kMaxDevices] = {};

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// The calling thread's current driver context (null if it cannot be queried).
CUcontext current_context() {
  static PFN_cuCtxGetCurrent_v4000 get = nullptr;
  if (get == nullptr) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 4000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
      return nullptr;
    get = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(fn);
  }
  CUcontext ctx = nullptr;
  return get(&ctx) == CUDA_SUCCESS ? ctx : nullptr;
}

// Device address of the scratch array on the stream's device, which must be
// the current device; looked up once per device and context.
hsa_status_t device_scratch(cudaStream_t stream, void** out) {
  int dev = -1, sdev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return HSA_ERR_CUDA;
  if (cudaStreamGetDevice(stream, &sdev) != cudaSuccess || sdev != dev) return HSA_ERR_INVALID_ARG;
  if (dev < 0 || dev >= kMaxDevices) return HSA_ERR_UNSUPPORTED;
  const CUcontext ctx = current_context();
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  Cached& c = g_scratch[dev];
  if (c.ptr == nullptr || ctx == nullptr || c.ctx != ctx) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return HSA_ERR_CUDA;
    c.ptr = p;
    c.ctx = ctx;
  }
  *out = c.ptr;
  return HSA_OK;
}

}  // namespace

extern "C" {

hsa_status_t hsa_decode_noalloc(const hsa_decode_shape_t* shape, const void* q, const void* K_mem,
                                const void* V_mem, const float* kbar32, void* O, int32_t* idx, float* s_sel,
                                float* w, cudaStream_t stream) {
  hsa::DecodeDims D;
  hsa_status_t st = hsa::resolve_decode_shape(shape, &D);
  if (st != HSA_OK) return st;
  if (D.Bq == 0) return HSA_OK;
  const void* need_ptrs[] = {q, O, idx, s_sel, w};
  for (const void* p : need_ptrs)
    if (p == nullptr || !aligned16(p)) return HSA_ERR_INVALID_ARG;
  if (D.Nc > 0) {
    const void* mem_ptrs[] = {K_mem, V_mem, kbar32};
    for (const void* p : mem_ptrs)
      if (p == nullptr || !aligned16(p)) return HSA_ERR_INVALID_ARG;
  }
  if (hsa::decode_workspace(D) > (size_t)HSA_DECODE_NOALLOC_SCRATCH_BYTES) return HSA_ERR_WORKSPACE;
  if (D.Nc > 0 && !(hsa::memory_device_readable(K_mem) && hsa::memory_device_readable(V_mem)))
    return HSA_ERR_INVALID_ARG;
  void* scratch = nullptr;
  if ((st = device_scratch(stream, &scratch)) != HSA_OK) return st;
  return hsa::launch_decode(D, q, K_mem, V_mem, kbar32, O, idx, s_sel, w, scratch, stream) == cudaSuccess
             ? HSA_OK
             : HSA_ERR_CUDA;
}

}  // extern "C"
