// capi_noalloc.cu -- hscale_rtn_scales_noalloc: the global scale and RTN codes without a
// caller-supplied workspace and without any allocation.
//
// Some callers of this library cannot allocate device memory: a plugin or callback that
// is handed only its input and output tensors by a host framework, or a service whose
// device memory is owned by a framework pool it has no handle to.  They cannot provide
// the small workspace hscale_rtn_scales needs for its amax word.  This entry point keeps
// that word in a fixed array of this file that lives in every GPU's memory from the
// moment the library is loaded there until the process exits.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/hscale.h"
#include "hscale_internal.h"

namespace hscale {

// Unique id of the calling thread's current context, or 0 when it has none yet.  A
// context destroyed and created again (cudaDeviceReset) gets a new id; its module, and
// with it the array below, may then sit at another address, and its streams and events
// are gone.
cudaError_t current_context_id(unsigned long long* id) {
  using CtxGetCurrentFn = CUresult (*)(CUcontext*);
  using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);
  static std::once_flag once;
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (get_current == nullptr || get_id == nullptr) return cudaErrorNotSupported;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  *id = 0;
  if (ctx == nullptr) return cudaSuccess;
  return get_id(ctx, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorDeviceUninitialized;
}

}  // namespace hscale

namespace {

using hscale::current_context_id;

// The fixed scratch of hscale_rtn_scales_noalloc (HSCALE_NOALLOC_SCRATCH_BYTES bytes per
// GPU).  Host code must not pass this name to a kernel: on the host it is only a stand-in
// for the symbol, so its device address is looked up once per device below.
static __device__ __align__(256) uint8_t g_noalloc_scratch[HSCALE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of g_noalloc_scratch in the current device's context, resolved on the
// first call in that context (with that device current) and cached per device together
// with the context's id: a call in a new context of the same device (after
// cudaDeviceReset) resolves it again instead of using a stale address.
cudaError_t scratch_address(uint32_t** out) {
  static std::mutex mu;
  static void* addr[kMaxDevices] = {nullptr};
  static unsigned long long ctx_of[kMaxDevices] = {0};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  unsigned long long id = 0;
  err = current_context_id(&id);
  if (err != cudaSuccess) return err;
  if (id == 0 || addr[dev] == nullptr || ctx_of[dev] != id) {
    // the lookup also makes the runtime bind the device's primary context to the thread
    // when it has none yet, so the context id is read (again) after it
    void* p = nullptr;
    err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (err != cudaSuccess) return err;
    if (p == nullptr) return cudaErrorInvalidSymbol;
    err = current_context_id(&id);
    if (err != cudaSuccess) return err;
    if (id == 0) return cudaErrorDeviceUninitialized;
    addr[dev] = p;
    ctx_of[dev] = id;
  }
  *out = static_cast<uint32_t*>(addr[dev]);
  return cudaSuccess;
}

}  // namespace

extern "C" int hscale_rtn_scales_noalloc(const void* w_bf16, int64_t m, int64_t n,
                                         float* global_scale, uint8_t* codes, void* stream) {
  if (m < 0 || n < 0 || n % 16 != 0) return HSCALE_ERR_SHAPE;
  if (m > 0 && n > 0 && (m > INT64_MAX / n || n / 16 > INT32_MAX)) return HSCALE_ERR_SHAPE;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (w_bf16 == nullptr || global_scale == nullptr) return HSCALE_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(w_bf16) & 15) != 0) return HSCALE_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(global_scale) & 3) != 0) return HSCALE_ERR_ALIGN;
  // the work needs hscale_rtn_workspace_bytes() of scratch, which does not depend on m or n;
  // refuse if it ever outgrows the fixed array
  if (hscale_rtn_workspace_bytes() > (size_t)HSCALE_NOALLOC_SCRATCH_BYTES) return HSCALE_ERR_WORKSPACE;
  uint32_t* amax = nullptr;
  if (scratch_address(&amax) != cudaSuccess) return HSCALE_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the amax word keeps the previous call's value: clear it first
  if (cudaMemsetAsync(amax, 0, sizeof(uint32_t), s) != cudaSuccess) return HSCALE_ERR_CUDA;
  if (hscale::launch_amax(w_bf16, m * n, amax, s) != cudaSuccess) return HSCALE_ERR_CUDA;
  return hscale::launch_rtn_codes(w_bf16, m, n, amax, global_scale, codes, s) == cudaSuccess
             ? HSCALE_OK
             : HSCALE_ERR_CUDA;
}
