// hscale_device.cuh -- device helpers shared by the H-Scale kernels (sm_103a).
//
// Number formats are handled with fp32 bit arithmetic, never tables:
//   * E4M3 (OCP E4M3FN, exponent bias 7): the fp32 whose bit pattern is (code << 20)
//     equals E4M3(code) * 2^-120, because shifting the 3-bit mantissa into fp32's top
//     mantissa bits and the 4-bit exponent into fp32's exponent field lines E4M3's
//     subnormal boundary up with fp32's.  The ladder L+ of Eq. 8 is codes 1..126.
//   * E2M1 (bias 1): the fp32 with bit pattern (code << 22) equals E2M1(code) * 2^-126,
//     for the same reason.  So rounding a value to the E2M1 grid is rounding the bit
//     pattern of (value * 2^-126) to a multiple of 2^22, and saturating at 6 is an
//     integer min against the pattern of 6 * 2^-126.
// These identities need denormals kept (no flush-to-zero), so the library is built
// without --use_fast_math.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace hscale {

// ---------------------------------------------------------------- loads
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

__device__ __forceinline__ uint4 ld_nc_v4(const void* p) {
  uint4 r;
  asm("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

// ---------------------------------------------------------------- bf16
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// ---------------------------------------------------------------- formats
constexpr uint32_t kE4M3MaxCode = 126;          // 448, top of the ladder (M of Eq. 8)
constexpr uint32_t kE2M1SixRaw = 7u << 22;      // bit pattern of 6 * 2^-126
constexpr uint32_t kE2M1Half = 1u << 21;        // half a grid step in the raw encoding
constexpr uint32_t kE2M1Keep = 0xFFC00000u;     // keeps exponent + 1 mantissa bit

// E4M3 magnitude of code c in [0, 127]; exact.
__device__ __forceinline__ float e4m3_mag(uint32_t c) {
  return __fmul_rn(__uint_as_float(c << 20), 0x1p120f);
}

// E2M1 magnitude of raw pattern q (q = code << 22); exact for any code.
__device__ __forceinline__ float e2m1_from_raw(uint32_t q) {
  return __fmul_rn(__uint_as_float(q), 0x1p126f);
}

// fast reciprocal (relative error <= 2^-22), used only where the result is checked
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// ---------------------------------------------------------------- scaled domain
// All scale arithmetic runs on w * 2^-K and s_g * 2^-K with K chosen so that
// s_g * 2^-K lies in [2^-12, 2^-11): then every effective scale s' = s_g l 2^-K is at
// most 448 * 2^-11, s' * 2^126 cannot overflow, 2^-126 / s' is a normal number, and
// every comparison keeps its sign (scaling by a power of two is exact).
struct ScaleDomain {
  float sg;    // s_g
  float sgk;   // s_g * 2^-K
  float pw;    // 2^-K
};

__device__ __forceinline__ ScaleDomain make_scale_domain(float sg) {
  ScaleDomain d;
  int e = (int)((__float_as_uint(sg) >> 23) & 0xFFu) - 127;
  int K = e + 12;
  if (K > 126) K = 126;
  if (K < -126) K = -126;
  d.sg = sg;
  d.pw = __uint_as_float((uint32_t)(127 - K) << 23);
  d.sgk = __fmul_rn(sg, d.pw);
  return d;
}

// ---------------------------------------------------------------- RTN code (Eq. 7)
// code = max(1, RNE_E4M3_sat(amax_g / (c s_g))) for an anchor c = 2 * half_c (6 for the
// max-abs RTN scale of Eq. 7; 4 and 6 for the 4over6 anchors of Algorithm 2), decided
// exactly.  amax_k = amax_g * 2^-K, inv_raw = 2^-120 / (c sgk).  An fp32 estimate of the
// quotient picks a code within one step; the two midpoints next to it are then checked
// exactly: c * mu has <= 7 significant bits and one FMA rounds once, so the sign of
// fma(-c mu, sgk, amax_k) is the sign of amax_g - c mu s_g.  Ties go to the even code.
__device__ __forceinline__ uint32_t anchored_code(float amax_k, float sgk, float inv_raw, float half_c) {
  const float r_raw = __fmul_rn(amax_k, inv_raw);  // ~ amax_g / (c s_g) * 2^-120
  uint32_t c = (__float_as_uint(r_raw) + (1u << 19)) >> 20;
  c = min(c, kE4M3MaxCode);
  if (c < kE4M3MaxCode) {
    const float muc = __fmul_rn(half_c, __fadd_rn(e4m3_mag(c), e4m3_mag(c + 1)));
    const float t = __fmaf_rn(-muc, sgk, amax_k);
    if (t > 0.0f || (t == 0.0f && ((c + 1) & 1u) == 0)) c += 1;
  }
  if (c > 0) {
    const float muc = __fmul_rn(half_c, __fadd_rn(e4m3_mag(c - 1), e4m3_mag(c)));
    const float t = __fmaf_rn(-muc, sgk, amax_k);
    if (t < 0.0f || (t == 0.0f && ((c - 1) & 1u) == 0)) c -= 1;
  }
  return c < 1 ? 1u : c;
}

__device__ __forceinline__ uint32_t rtn_code(float amax_k, float sgk, float inv6_raw) {
  return anchored_code(amax_k, sgk, inv6_raw, 3.0f);
}

// ~2^-120 / (c sgk): the factor anchored_code multiplies amax_k by (a normal number).  Only
// an estimate is needed (anchored_code checks both neighbouring midpoints exactly), so it is
// the correctly rounded reciprocal of the rounded product (c sgk) 2^120, within 2^-23.
__device__ __forceinline__ float anchor_inv_raw(float sgk, float c) {
  return __frcp_rn(__fmul_rn(__fmul_rn(c, sgk), 0x1p120f));
}
__device__ __forceinline__ float rtn_inv6_raw(float sgk) { return anchor_inv_raw(sgk, 6.0f); }

// ---------------------------------------------------------------- E2M1 projection (Eq. 12)
// Fast rounding of y_raw = (|w| / s) * 2^-126 to the E2M1 grid: round-half-up on the
// raw bit pattern, then saturate.  Exact except when the true quotient lies within a
// few ulps of a midpoint; e2m1_uncertain() flags exactly those patterns.
__device__ __forceinline__ uint32_t e2m1_round_raw(float y_raw) {
  return min((__float_as_uint(y_raw) + kE2M1Half) & kE2M1Keep, kE2M1SixRaw);
}

// True when y_raw's discarded 22 bits are within 16 units of the half point, i.e. the
// quotient is within 16 ulps of an E2M1 midpoint.  The fast y_raw is within 4 units of
// the exact quotient (reciprocal 2^-22, two roundings of 2^-24, or half a denormal
// unit), so outside this window the fast rounding is the exact one.
__device__ __forceinline__ bool e2m1_uncertain(float y_raw) {
  return ((__float_as_uint(y_raw) - 0x1FFFF0u) & 0x3FFFFFu) <= 0x20u;
}

// Exact round-to-nearest-even magnitude code of a_k / (l sgk) for an uncertain y_raw:
// the midpoint between the two grid points bracketing y_raw is compared exactly with
// one FMA (mid * l has <= 7 significant bits).
__device__ __forceinline__ uint32_t e2m1_exact_code(float y_raw, float a_k, float l, float sgk) {
  const uint32_t zt = __float_as_uint(y_raw) & kE2M1Keep;
  const uint32_t klo = zt >> 22;
  const float vlo = e2m1_from_raw(zt);
  const float vhi = e2m1_from_raw(zt + (1u << 22));
  const float mid = __fmul_rn(0.5f, __fadd_rn(vlo, vhi));
  const float t = __fmaf_rn(-__fmul_rn(mid, l), sgk, a_k);
  uint32_t k;
  if (t > 0.0f) k = klo + 1;
  else if (t < 0.0f) k = klo;
  else k = (klo & 1u) ? klo + 1 : klo;  // tie: even code
  return min(k, 7u);
}

// Exact round-to-nearest-even magnitude code of a_k / (l sgk) (a_k >= 0) when the quotient
// is known to lie between the grid points of codes klo and klo + 1 (klo < 7): the midpoint
// is compared exactly with one FMA; a tie goes to the even code.
__device__ __forceinline__ uint32_t e2m1_code_between(float a_k, uint32_t klo, float l, float sgk) {
  const float vlo = e2m1_from_raw(klo << 22);
  const float vhi = e2m1_from_raw((klo + 1) << 22);
  const float mid = __fmul_rn(0.5f, __fadd_rn(vlo, vhi));
  const float t = __fmaf_rn(-__fmul_rn(mid, l), sgk, a_k);
  if (t > 0.0f) return klo + 1;
  if (t < 0.0f) return klo;
  return (klo & 1u) ? klo + 1 : klo;
}

// Exact magnitude code of a_k / (l sgk): fast path plus the exact fix when flagged.
__device__ __forceinline__ uint32_t e2m1_code(float a_k, float inv_raw, float l, float sgk) {
  const float y = __fmul_rn(a_k, inv_raw);
  uint32_t k = e2m1_round_raw(y) >> 22;
  if (e2m1_uncertain(y)) k = e2m1_exact_code(y, a_k, l, sgk);
  return k;
}

// 2^-126 / s' for s' = l * sgk (fast reciprocal; every use is either checked or bounded).
__device__ __forceinline__ float inv_raw_of(float sp) {
  return __fmul_rn(rcp_approx(sp), 0x1p-126f);
}

}  // namespace hscale
