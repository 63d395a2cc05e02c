// hscale_internal.h -- host-side launchers shared by the C ABI translation unit.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace hscale {

struct DeviceInfo {
  int device = -1;
  int sm_count = 0;
};

// SM count of the current device (cached per device).
cudaError_t current_device_info(DeviceInfo* out);

// h[j] += sum_t x[t, j]^2.  Arguments already validated; tokens, n > 0.
cudaError_t launch_hessian(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* h,
                           cudaStream_t stream);

// amax over W into *amax_bits (16-bit |bf16| pattern, zero-extended); *amax_bits must be 0.
cudaError_t launch_amax(const void* w, int64_t count, uint32_t* amax_bits, cudaStream_t stream);

// s_g from *amax_bits into *global_scale, and (if codes != nullptr) the RTN codes.
cudaError_t launch_rtn_codes(const void* w, int64_t m, int64_t n, const uint32_t* amax_bits,
                             float* global_scale, uint8_t* codes, cudaStream_t stream);

// ctas_per_sm > 0 caps the grid at that many resident CTAs per SM (room for a concurrent
// kernel); 0 fills every SM.
cudaError_t launch_refine(const void* w, const float* h, int64_t m, int64_t n,
                          const float* global_scale, const uint8_t* init_codes, int down, int up,
                          uint8_t* codes_out, uint8_t* packed_out, int ctas_per_sm, cudaStream_t stream);

// Algorithm 2's initial codes (the better of the anchors m/4, m/6 by plain MSE).
cudaError_t launch_fourover6(const void* w, int64_t m, int64_t n, const float* global_scale,
                             uint8_t* codes, cudaStream_t stream);

// Sticky device error flags of this library (bit 0: a bounded wait ran out); cleared on read.
cudaError_t read_and_clear_device_error(uint32_t* flags);

cudaError_t launch_pack(const void* w, int64_t m, int64_t n, const float* global_scale,
                        const uint8_t* codes, uint8_t* packed_out, cudaStream_t stream);

}  // namespace hscale
