// capi.cu -- the extern "C" boundary declared in include/hscale.h.
//
// Every entry point validates its arguments on the host before enqueueing anything,
// then calls the launchers in hessian.cu / scales.cu.  No exception crosses the ABI.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/hscale.h"
#include "hscale_internal.h"

namespace hscale {

cudaError_t current_device_info(DeviceInfo* out) {
  static std::mutex mu;
  static int sms[64] = {0};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (sms[dev] == 0) {
    int v = 0;
    err = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    sms[dev] = v;
  }
  out->device = dev;
  out->sm_count = sms[dev];
  return cudaSuccess;
}

}  // namespace hscale

namespace {

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

inline int from_cuda(cudaError_t e) { return e == cudaSuccess ? HSCALE_OK : HSCALE_ERR_CUDA; }

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

// common checks of a weight matrix argument
inline int check_weight(const void* w, int64_t m, int64_t n) {
  if (m < 0 || n < 0) return HSCALE_ERR_SHAPE;
  if (n % 16 != 0) return HSCALE_ERR_SHAPE;
  if (m > 0 && n > 0 && (m > INT64_MAX / n || n / 16 > INT32_MAX)) return HSCALE_ERR_SHAPE;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (w == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(w, 16)) return HSCALE_ERR_ALIGN;
  return HSCALE_OK;
}

}  // namespace

extern "C" {

const char* hscale_status_string(int status) {
  switch (status) {
    case HSCALE_OK: return "ok";
    case HSCALE_ERR_NULL: return "a required pointer is NULL";
    case HSCALE_ERR_SHAPE: return "invalid shape (negative size, n not a multiple of 16/8, ld < n, or too large)";
    case HSCALE_ERR_ALIGN: return "misaligned pointer or leading dimension";
    case HSCALE_ERR_ARG: return "scalar argument out of range";
    case HSCALE_ERR_CUDA: return "CUDA runtime error";
    case HSCALE_ERR_WORKSPACE: return "workspace missing or too small";
    default: return "unknown status";
  }
}

int hscale_abi_version(void) { return 4; }

int hscale_device_error_flags(uint32_t* flags) {
  if (flags == nullptr) return HSCALE_ERR_NULL;
  uint32_t a = 0, b = 0, c = 0;
  cudaError_t err = hscale::read_hessian_device_error(&a);
  if (err == cudaSuccess) err = hscale::read_output_error_device_error(&b);
  if (err == cudaSuccess) err = hscale::read_selftest_device_error(&c);
  *flags = a | b | c;
  return from_cuda(err);
}

int hscale_selftest_bounded_wait(uint32_t polls, void* stream) {
  return from_cuda(hscale::launch_bounded_wait_selftest(polls, as_stream(stream)));
}

int hscale_hessian_diag_accumulate(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x,
                                   float* h, void* stream) {
  return hscale_hessian_diag_accumulate_ex(x_bf16, tokens, n, ld_x, h, 0u, stream);
}

int hscale_hessian_diag_accumulate_ex(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x,
                                      float* h, uint32_t flags, void* stream) {
  if ((flags & ~(uint32_t)HSCALE_HESSIAN_X_READY) != 0) return HSCALE_ERR_ARG;
  if (tokens < 0 || n < 0 || ld_x < n) return HSCALE_ERR_SHAPE;
  if (n % 8 != 0) return HSCALE_ERR_SHAPE;
  if (n > (int64_t)65535 * 64) return HSCALE_ERR_SHAPE;  // 64-channel tiles on grid.y
  if (tokens == 0 || n == 0) return HSCALE_OK;
  if (x_bf16 == nullptr || h == nullptr) return HSCALE_ERR_NULL;
  if (ld_x % 8 != 0) return HSCALE_ERR_ALIGN;
  if (!aligned(x_bf16, 16) || !aligned(h, 4)) return HSCALE_ERR_ALIGN;
  if (tokens > INT32_MAX || tokens > INT64_MAX / ld_x) return HSCALE_ERR_SHAPE;
  return from_cuda(hscale::launch_hessian(x_bf16, tokens, n, ld_x, h, (flags & HSCALE_HESSIAN_X_READY) != 0,
                                          as_stream(stream)));
}

int hscale_hessian_sum_partials(const float* partials, int64_t parts, int64_t n, int64_t ld, float* h,
                                void* stream) {
  if (parts < 0 || n < 0 || (parts > 0 && ld < n)) return HSCALE_ERR_SHAPE;
  if (parts == 0 || n == 0) return HSCALE_OK;
  if (parts > 1 && ld > INT64_MAX / parts) return HSCALE_ERR_SHAPE;
  if (partials == nullptr || h == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(partials, 4) || !aligned(h, 4)) return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_sum_partials(partials, parts, n, ld, h, as_stream(stream)));
}

int hscale_amax_bits(const void* w_bf16, int64_t m, int64_t n, uint32_t* amax_bits, void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (amax_bits == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(amax_bits, 4)) return HSCALE_ERR_ALIGN;
  cudaStream_t s = as_stream(stream);
  // an empty matrix has amax 0: the word is cleared either way
  if (cudaMemsetAsync(amax_bits, 0, sizeof(uint32_t), s) != cudaSuccess) return HSCALE_ERR_CUDA;
  if (m == 0 || n == 0) return HSCALE_OK;
  return from_cuda(hscale::launch_amax(w_bf16, m * n, amax_bits, s));
}

int hscale_global_scale_from_amax(const uint32_t* amax_bits, float* global_scale, void* stream) {
  if (amax_bits == nullptr || global_scale == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(amax_bits, 4) || !aligned(global_scale, 4)) return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_rtn_codes(nullptr, 0, 16, amax_bits, global_scale, nullptr, as_stream(stream)));
}

size_t hscale_rtn_workspace_bytes(void) { return 256; }

int hscale_rtn_scales(const void* w_bf16, int64_t m, int64_t n, float* global_scale,
                      uint8_t* codes, void* workspace, size_t workspace_bytes, void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (global_scale == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(global_scale, 4)) return HSCALE_ERR_ALIGN;
  if (workspace == nullptr || workspace_bytes < hscale_rtn_workspace_bytes()) return HSCALE_ERR_WORKSPACE;
  if (!aligned(workspace, 4)) return HSCALE_ERR_ALIGN;
  cudaStream_t s = as_stream(stream);
  uint32_t* amax = static_cast<uint32_t*>(workspace);
  cudaError_t err = cudaMemsetAsync(amax, 0, sizeof(uint32_t), s);
  if (err != cudaSuccess) return HSCALE_ERR_CUDA;
  err = hscale::launch_amax(w_bf16, m * n, amax, s);
  if (err != cudaSuccess) return HSCALE_ERR_CUDA;
  return from_cuda(hscale::launch_rtn_codes(w_bf16, m, n, amax, global_scale, codes, s));
}

int hscale_refine_scales(const void* w_bf16, const float* h, int64_t m, int64_t n,
                         const float* global_scale, const uint8_t* init_codes, int32_t down,
                         int32_t up, uint8_t* codes_out, uint8_t* packed_out, void* stream) {
  return hscale_refine_scales_ex(w_bf16, h, m, n, global_scale, init_codes, down, up, codes_out,
                                 packed_out, 0, stream);
}

int hscale_refine_scales_ex(const void* w_bf16, const float* h, int64_t m, int64_t n,
                            const float* global_scale, const uint8_t* init_codes, int32_t down,
                            int32_t up, uint8_t* codes_out, uint8_t* packed_out,
                            int32_t ctas_per_sm, void* stream) {
  return hscale_refine_scales_strided(w_bf16, n, h, m, n, global_scale, init_codes, n / 16, 0, down, up,
                                      codes_out, n / 16, packed_out, n / 2, ctas_per_sm, stream);
}

int hscale_refine_scales_4over6(const void* w_bf16, const float* h, int64_t m, int64_t n,
                                const float* global_scale, int32_t down, int32_t up, uint8_t* codes_out,
                                uint8_t* packed_out, int32_t ctas_per_sm, void* stream) {
  return hscale_refine_scales_strided(w_bf16, n, h, m, n, global_scale, nullptr, 0, 1, down, up, codes_out,
                                      n / 16, packed_out, n / 2, ctas_per_sm, stream);
}

namespace {

// Argument checks and launch shared by the refine entry points.
int refine_checked(const void* w_bf16, int64_t ld_w, const float* h, int64_t m, int64_t n,
                   const float* global_scale, const uint8_t* init_codes, int64_t ld_init, int32_t fourover6,
                   int32_t down, int32_t up, uint8_t* codes_out, int64_t ld_codes, uint8_t* packed_out,
                   int64_t ld_packed, int32_t ctas_per_sm, unsigned* share_counter, void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (down < 0 || up < 0 || down > 125 || up > 125) return HSCALE_ERR_ARG;
  if (ctas_per_sm < 0 || (fourover6 != 0 && fourover6 != 1)) return HSCALE_ERR_ARG;
  if (fourover6 && init_codes != nullptr) return HSCALE_ERR_ARG;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (ld_w < n || ld_codes < n / 16 || (packed_out != nullptr && ld_packed < n / 2) ||
      (init_codes != nullptr && ld_init < n / 16))
    return HSCALE_ERR_SHAPE;
  if (ld_w > INT64_MAX / m || ld_codes > INT64_MAX / m || (packed_out != nullptr && ld_packed > INT64_MAX / m) ||
      (init_codes != nullptr && ld_init > INT64_MAX / m))
    return HSCALE_ERR_SHAPE;
  if (ld_w % 8 != 0) return HSCALE_ERR_ALIGN;
  if (global_scale == nullptr || codes_out == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(global_scale, 4)) return HSCALE_ERR_ALIGN;
  if (h != nullptr && !aligned(h, 16)) return HSCALE_ERR_ALIGN;
  if (packed_out != nullptr && (!aligned(packed_out, 8) || ld_packed % 8 != 0)) return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_refine(w_bf16, ld_w, h, m, n, global_scale, init_codes,
                                         init_codes ? ld_init : 0, down, up, codes_out, ld_codes, packed_out,
                                         packed_out ? ld_packed : 0, ctas_per_sm, fourover6 != 0, share_counter,
                                         as_stream(stream)));
}

}  // namespace

int hscale_refine_scales_strided(const void* w_bf16, int64_t ld_w, const float* h, int64_t m, int64_t n,
                                 const float* global_scale, const uint8_t* init_codes, int64_t ld_init,
                                 int32_t fourover6, int32_t down, int32_t up, uint8_t* codes_out,
                                 int64_t ld_codes, uint8_t* packed_out, int64_t ld_packed, int32_t ctas_per_sm,
                                 void* stream) {
  return refine_checked(w_bf16, ld_w, h, m, n, global_scale, init_codes, ld_init, fourover6, down, up, codes_out,
                        ld_codes, packed_out, ld_packed, ctas_per_sm, nullptr, stream);
}

size_t hscale_refine_workspace_bytes(void) { return 16; }

int hscale_refine_scales_ws(const void* w_bf16, const float* h, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* init_codes, int32_t fourover6, int32_t down, int32_t up,
                            uint8_t* codes_out, uint8_t* packed_out, int32_t ctas_per_sm, void* workspace,
                            size_t workspace_bytes, void* stream) {
  if (workspace != nullptr) {
    if (workspace_bytes < hscale_refine_workspace_bytes()) return HSCALE_ERR_WORKSPACE;
    if (!aligned(workspace, 16)) return HSCALE_ERR_ALIGN;
  }
  return refine_checked(w_bf16, n, h, m, n, global_scale, init_codes, n / 16, fourover6, down, up, codes_out,
                        n / 16, packed_out, n / 2, ctas_per_sm, static_cast<unsigned*>(workspace), stream);
}

int hscale_fourover6_codes(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                           uint8_t* codes, void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (global_scale == nullptr || codes == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(global_scale, 4)) return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_fourover6(w_bf16, m, n, global_scale, codes, as_stream(stream)));
}

int hscale_dequant_residual(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* codes, const uint8_t* packed, void* dw2_bf16, int64_t ld_dw2,
                            void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (m == 0 || n == 0) return HSCALE_OK;
  const int64_t n_pad = (n + 63) / 64 * 64;
  if (ld_dw2 < 2 * n_pad || m > INT64_MAX / ld_dw2) return HSCALE_ERR_SHAPE;
  if (global_scale == nullptr || codes == nullptr || packed == nullptr || dw2_bf16 == nullptr)
    return HSCALE_ERR_NULL;
  if (!aligned(global_scale, 4) || !aligned(packed, 8) || !aligned(dw2_bf16, 16) || ld_dw2 % 8 != 0)
    return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_residual(w_bf16, m, n, global_scale, codes, packed, dw2_bf16, ld_dw2,
                                           as_stream(stream)));
}

size_t hscale_output_error_workspace_bytes(int64_t tokens, int64_t m) {
  if (tokens <= 0 || m <= 0) return 0;
  const int64_t tiles = hscale::output_error_tiles(tokens, m);
  return (size_t)((tiles * 8 + 255) / 256 * 256);
}

int hscale_output_error(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x, const void* dw2_bf16,
                        int64_t ld_dw2, int64_t m, double* out_sum, void* workspace, size_t workspace_bytes,
                        void* stream) {
  if (tokens < 0 || n < 0 || m < 0 || ld_x < n) return HSCALE_ERR_SHAPE;
  if (n % 16 != 0) return HSCALE_ERR_SHAPE;
  const int64_t n_pad = (n + 63) / 64 * 64;
  if (ld_dw2 < 2 * n_pad) return HSCALE_ERR_SHAPE;
  if (tokens == 0 || n == 0 || m == 0) return HSCALE_OK;
  if (tokens > INT32_MAX || m > INT32_MAX || tokens > INT64_MAX / ld_x || m > INT64_MAX / ld_dw2)
    return HSCALE_ERR_SHAPE;
  if (hscale::output_error_tiles(tokens, m) > INT32_MAX) return HSCALE_ERR_SHAPE;
  if (x_bf16 == nullptr || dw2_bf16 == nullptr || out_sum == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(x_bf16, 16) || !aligned(dw2_bf16, 16) || !aligned(out_sum, 8) || ld_x % 8 != 0 ||
      ld_dw2 % 8 != 0)
    return HSCALE_ERR_ALIGN;
  if (workspace == nullptr || workspace_bytes < hscale_output_error_workspace_bytes(tokens, m) ||
      !aligned(workspace, 8))
    return HSCALE_ERR_WORKSPACE;
  return from_cuda(hscale::launch_output_error(x_bf16, tokens, n, ld_x, dw2_bf16, ld_dw2, m, out_sum,
                                               static_cast<double*>(workspace), as_stream(stream)));
}

size_t hscale_hessian_full_workspace_bytes(int64_t tokens, int64_t n) {
  if (tokens <= 0 || n <= 0) return 0;
  return (size_t)((n * hscale::hessian_full_ld(tokens) * 2 + 255) / 256 * 256);
}

int hscale_hessian_full_accumulate(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x, float* H,
                                   int64_t ld_h, void* workspace, size_t workspace_bytes, void* stream) {
  if (tokens < 0 || n < 0 || ld_x < n || ld_h < n) return HSCALE_ERR_SHAPE;
  if (tokens == 0 || n == 0) return HSCALE_OK;
  if (tokens > INT32_MAX || n > INT32_MAX || tokens > INT64_MAX / ld_x || n > INT64_MAX / ld_h) return HSCALE_ERR_SHAPE;
  if (x_bf16 == nullptr || H == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(x_bf16, 2) || !aligned(H, 4)) return HSCALE_ERR_ALIGN;
  // X with 16-byte aligned rows is read as it is; other X is transposed into the workspace
  const bool direct = aligned(x_bf16, 16) && ld_x % 8 == 0;
  if (!direct && (workspace == nullptr || workspace_bytes < hscale_hessian_full_workspace_bytes(tokens, n) ||
                  !aligned(workspace, 256)))
    return HSCALE_ERR_WORKSPACE;
  return from_cuda(hscale::launch_hessian_full(x_bf16, tokens, n, ld_x, H, ld_h, workspace, as_stream(stream)));
}

size_t hscale_gptq_factor_workspace_bytes(int64_t n) {
  if (n <= 0 || n > 65536) return 0;
  return hscale::gptq_factor_workspace(n);
}

int hscale_gptq_factor(const float* H, int64_t n, int64_t ld_h, float damp, float* U, uint8_t* dead,
                       int32_t* info, void* workspace, size_t workspace_bytes, void* stream) {
  if (n < 0 || ld_h < n || n > 65536) return HSCALE_ERR_SHAPE;
  if (!(damp >= 0.0f)) return HSCALE_ERR_ARG;
  if (n == 0) return HSCALE_OK;
  if (H == nullptr || U == nullptr || info == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(H, 4) || !aligned(U, 4) || !aligned(info, 4)) return HSCALE_ERR_ALIGN;
  if (workspace == nullptr || workspace_bytes < hscale_gptq_factor_workspace_bytes(n) || !aligned(workspace, 256))
    return HSCALE_ERR_WORKSPACE;
  return from_cuda(hscale::launch_gptq_factor(H, n, ld_h, damp, U, dead, info, workspace, as_stream(stream)));
}

namespace {
inline int64_t round256(int64_t bytes) { return (bytes + 255) / 256 * 256; }
}  // namespace

// running weights (fp32 m x n) and two buffers each of the bf16 split operands of the
// update GEMM: A' (m x 6 block) and B' (n x 6 block)
size_t hscale_gptq_workspace_bytes(int64_t m, int64_t n, int32_t block) {
  if (m <= 0 || n <= 0 || block <= 0) return 0;
  const int64_t b = block;
  return (size_t)(round256(m * n * 4) + round256(2 * m * 6 * b * 2) + round256(2 * n * 6 * b * 2));
}

int hscale_gptq_hscale(const void* w_bf16, int64_t m, int64_t n, const float* U, const float* h,
                       const float* global_scale, const uint8_t* dead, int32_t block, int32_t down, int32_t up,
                       uint8_t* codes_out, uint8_t* packed_out, void* workspace, size_t workspace_bytes,
                       void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (block <= 0 || block % 16 != 0 || (n > 0 && n % block != 0)) return HSCALE_ERR_SHAPE;
  if (down < 0 || up < 0 || down > 125 || up > 125) return HSCALE_ERR_ARG;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (U == nullptr || h == nullptr || global_scale == nullptr || codes_out == nullptr || packed_out == nullptr)
    return HSCALE_ERR_NULL;
  if (!aligned(U, 16) || !aligned(h, 16) || !aligned(global_scale, 4) || !aligned(packed_out, 8))
    return HSCALE_ERR_ALIGN;
  if (workspace == nullptr || workspace_bytes < hscale_gptq_workspace_bytes(m, n, block) || !aligned(workspace, 256))
    return HSCALE_ERR_WORKSPACE;
  uint8_t* base = static_cast<uint8_t*>(workspace);
  const int64_t b = block;
  float* Wf = reinterpret_cast<float*>(base);
  uint16_t* A6 = reinterpret_cast<uint16_t*>(base + round256(m * n * 4));
  uint16_t* B6 = reinterpret_cast<uint16_t*>(base + round256(m * n * 4) + round256(2 * m * 6 * b * 2));
  return from_cuda(hscale::launch_gptq_hscale(w_bf16, m, n, U, h, global_scale, dead, block, down, up, codes_out,
                                              packed_out, Wf, A6, B6, as_stream(stream)));
}

int hscale_pack_nvfp4(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                      const uint8_t* codes, uint8_t* packed_out, void* stream) {
  int st = check_weight(w_bf16, m, n);
  if (st != HSCALE_OK) return st;
  if (m == 0 || n == 0) return HSCALE_OK;
  if (global_scale == nullptr || codes == nullptr || packed_out == nullptr) return HSCALE_ERR_NULL;
  if (!aligned(global_scale, 4)) return HSCALE_ERR_ALIGN;
  if (!aligned(packed_out, 8)) return HSCALE_ERR_ALIGN;
  return from_cuda(hscale::launch_pack(w_bf16, m, n, global_scale, codes, packed_out,
                                       as_stream(stream)));
}

}  // extern "C"
