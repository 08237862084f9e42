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
// (cudaGetSymbolAddress, with the device current) and caches the address; that
// first call should come before any stream capture on the device. Calls that
// may overlap on one device share the array and race on it; callers serialise
// them. Nothing in the array has to start at zero: each call writes every byte
// it later reads.
#include <mutex>

#include "common.cuh"

namespace {

constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[HSA_DECODE_NOALLOC_SCRATCH_BYTES];

std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Device address of the current device's scratch array, looked up once per device.
hsa_status_t device_scratch(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return HSA_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return HSA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return HSA_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
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
  if ((st = device_scratch(&scratch)) != HSA_OK) return st;
  return hsa::launch_decode(D, q, K_mem, V_mem, kbar32, O, idx, s_sel, w, scratch, stream) == cudaSuccess
             ? HSA_OK
             : HSA_ERR_CUDA;
}

}  // extern "C"
