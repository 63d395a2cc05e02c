// hscale_internal.h -- host-side launchers shared by the C ABI translation unit.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

namespace hscale {

struct DeviceInfo {
  int device = -1;
  int sm_count = 0;
};

// SM count of the current device (cached per device).
cudaError_t current_device_info(DeviceInfo* out);

// h[j] += sum_t x[t, j]^2.  Arguments already validated; tokens, n > 0.  x_ready: nothing
// that may still be running writes X, so the kernel may read it before the previous
// kernel on the stream has finished.
cudaError_t launch_hessian(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* h, bool x_ready,
                           cudaStream_t stream);

// h[j] = sum of the parts' partial sums p_r[j] (row r at partials + r * ld) in rank order.
cudaError_t launch_sum_partials(const float* partials, int64_t parts, int64_t n, int64_t ld, float* h,
                                cudaStream_t stream);

// amax over W into *amax_bits (16-bit |bf16| pattern, zero-extended); *amax_bits must be 0.
cudaError_t launch_amax(const void* w, int64_t count, uint32_t* amax_bits, cudaStream_t stream);

// s_g from *amax_bits into *global_scale, and (if codes != nullptr) the RTN codes.
cudaError_t launch_rtn_codes(const void* w, int64_t m, int64_t n, const uint32_t* amax_bits,
                             float* global_scale, uint8_t* codes, cudaStream_t stream);

// W [m, n] with rows ld_w elements apart (ld_w % 8 == 0), initial codes with rows ld_init
// bytes apart, codes with rows ld_codes bytes apart, nibbles with rows ld_packed bytes
// apart (ld_packed % 8 == 0).  ctas_per_sm > 0
// caps the grid at that many resident CTAs per SM (room for a concurrent kernel); 0 fills
// every SM.  fourover6: the initial codes are Algorithm 2's, decided in the search kernel
// (init_codes is then ignored).  share_counter: 4 bytes of device memory for the
// work-shared schedule of long contiguous searches (zeroed on the stream first), or
// nullptr for the static deal; the results are the same either way.
cudaError_t launch_refine(const void* w, int64_t ld_w, const float* h, int64_t m, int64_t n,
                          const float* global_scale, const uint8_t* init_codes, int64_t ld_init, int down,
                          int up, uint8_t* codes_out, int64_t ld_codes, uint8_t* packed_out, int64_t ld_packed,
                          int ctas_per_sm, bool fourover6, unsigned* share_counter, cudaStream_t stream);

// Algorithm 2's initial codes (the better of the anchors m/4, m/6 by plain MSE).
cudaError_t launch_fourover6(const void* w, int64_t m, int64_t n, const float* global_scale,
                             uint8_t* codes, cudaStream_t stream);

// cuTensorMapEncodeTiled, looked up once through the runtime's driver entry point.
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
cudaError_t encode_tiled_fn(EncodeTiledFn* out);

// Unique id of the calling thread's current context (0 when it has none yet); a context
// created again after cudaDeviceReset gets a new id.
cudaError_t current_context_id(unsigned long long* id);

// The library's second stream and its events in the current device context, for calls that
// work ahead on it (created on first use and kept).  The lease holds the library's mutex:
// release it (destroy the lease) only after the call has enqueued all its work.  side is
// null when they do not exist yet and `stream` is being captured (they may not be created
// then): the call then runs on `stream` alone.
constexpr int kLookAheadEvents = 10;
struct LookAheadLease {
  std::unique_lock<std::mutex> lock;
  cudaStream_t side = nullptr;
  cudaEvent_t ev[kLookAheadEvents] = {};
};
cudaError_t acquire_look_ahead(cudaStream_t stream, LookAheadLease* lease);

// cudaFuncAttributeMaxDynamicSharedMemorySize = bytes and the maximum shared-memory
// carveout for kernel `func` on the current device, set once per (kernel, device) and
// remembered, so that every GPU of a process gets it (a function attribute belongs to one
// device's context).
cudaError_t ensure_dynamic_smem(const void* func, int bytes);

// dW = W - W_hat of packed NVFP4 weights as a bf16 pair [hi | lo] per row, rows of ld
// elements: hi in [0, n_pad), lo in [n_pad, 2 n_pad), zero padding, n_pad = 64 * ceil(n / 64).
cudaError_t launch_residual(const void* w, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* codes, const uint8_t* packed, void* dw2, int64_t ld_dw2,
                            cudaStream_t stream);

// *out += ||X dW^T||_F^2 on the tensor cores; partials holds one double per 128 x 256 tile.
int64_t output_error_tiles(int64_t tokens, int64_t m);
cudaError_t launch_output_error(const void* x, int64_t tokens, int64_t n, int64_t ld_x, const void* dw2,
                                int64_t ld_dw2, int64_t m, double* out, double* partials,
                                cudaStream_t stream);

// H[n, n] (row stride ld_h) += X^T X on the tensor cores; xt is scratch for X^T
// (n rows of hessian_full_ld(tokens) bf16).
int64_t hessian_full_ld(int64_t tokens);
cudaError_t launch_hessian_full(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* H, int64_t ld_h,
                                void* xt, cudaStream_t stream);

// Algorithm 3 (GPTQ + H-Scale).  The factor's workspace (bytes) and the factor itself; U is
// also used as scratch for the damped copy of H.
int64_t gptq_factor_padded(int64_t n);
size_t gptq_factor_workspace(int64_t n);
cudaError_t launch_gptq_factor(const float* H, int64_t n, int64_t ld_h, float damp, float* U, uint8_t* dead,
                               int32_t* info, void* workspace, cudaStream_t stream);
// C[m, nn] (row stride ld_c, fp32) += A B^T on the tensor cores, with A [m, k] and B [nn, k]
// bf16, rows of k elements contiguous (k % 8 == 0, 16-byte aligned bases); every tile.
// programmatic: launched with programmatic dependent launch (the kernel waits for the
// previous kernel on the stream before its first load, and lets the next one be scheduled).
cudaError_t launch_gemm_accumulate(const void* a, const void* b, int64_t m, int64_t nn, int64_t k, float* C,
                                   int64_t ld_c, cudaStream_t stream, bool programmatic = false);

cudaError_t launch_gptq_hscale(const void* w, int64_t m, int64_t n, const float* U, const float* h,
                               const float* global_scale, const uint8_t* dead, int block, int down, int up,
                               uint8_t* codes, uint8_t* packed, float* Wf, uint16_t* A6, uint16_t* B6,
                               cudaStream_t stream);

// Sticky device error flags of each translation unit (bit 0: a bounded wait ran out);
// cleared on read.
cudaError_t read_hessian_device_error(uint32_t* flags);
cudaError_t read_output_error_device_error(uint32_t* flags);
cudaError_t read_selftest_device_error(uint32_t* flags);

// One CTA waits at most `polls` polls on an mbarrier that nothing arrives on.
cudaError_t launch_bounded_wait_selftest(uint32_t polls, cudaStream_t stream);

cudaError_t launch_pack(const void* w, int64_t m, int64_t n, const float* global_scale,
                        const uint8_t* codes, uint8_t* packed_out, cudaStream_t stream);

}  // namespace hscale
