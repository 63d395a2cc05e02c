// scales.cu -- global scale, RTN codes, H-Scale search and NVFP4 packing on sm_103a.
//
//   amax_kernel         amax|W| (integer max of |bf16| bit patterns; order-free)
//   rtn_codes_kernel    s_g = amax / 2688 and the RTN code of every group (Eq. 7)
//   refine_*_kernel     Algorithm 1: per group, every distinct E4M3 code in the window
//                       (Eqs. 8-11) is scored by sum_j h_j (|w_j| - s q_j)^2 (Eqs. 6, 12,
//                       13); the best code is re-quantized exactly and packed.  Their
//                       4over6 instances decide Algorithm 2's initial code in place.  One
//                       per-group body (search_unit) under four deals of the units:
//                         refine_kernel         2-D views, ragged rows (static)
//                         refine_linear_kernel  contiguous W, static (a search beside
//                                               another kernel, or a tiny one)
//                         refine_sm_kernel      contiguous W alone on the GPU: one CTA per
//                                               SM, units shared through shared memory
//                         refine_shared_kernel  contiguous W, long searches: units shared
//                                               through a counter in a caller workspace
//   fourover6_codes_kernel  Algorithm 2's initial codes as a separate pass
//   pack_kernel         exact FP4 quantization with given codes (Eq. 2)
//
// The search (one group per thread, no shuffles in the hot loop)
//   A candidate scale s' = l sgk is scored as E = s'^2 sum_j h_j (q_j - y_j)^2 with
//   y_j = a_j / s' (one packed multiply by a tabulated reciprocal) and q_j = RNE_sat(y_j)
//   from the hardware E2M1 conversion (saturation included) converted back to f16; the
//   residual q - y is one mixed f16/f32 subtract.  That is five lane operations per
//   element and candidate.  The tabulated reciprocal is correctly rounded, so y (one more
//   rounding) is within a relative eps = 2^-23 (+ 2^-48) of the exact quotient y*, and
//   every element's term differs from its exact-decision term by at most
//   4 eps y* |q* - y*| + 8 eps^2 y*^2 (also where a midpoint falls between y and y*:
//   both distances to the grid are then within eps y* of half the grid gap), so by
//   Cauchy-Schwarz the fast score is within
//        4 eps sqrt(A E*) + 8 eps^2 A + 14 * 2^-24 E*    (A = sum_j h_j a_j^2)
//   of the exact score E*; in terms of the fast score E that is at most
//   4.01 * 2^-23 sqrt(A E) + 33 * 2^-46 A + 15 * 2^-24 E.  When
//        runner-up - best > 2^-18 E2 + 2^-19 sqrt(A E2) + 2^-35 A
//   (more than the two errors together, with at least 2x slack on every term) and
//   E2 >= 2^-36 A (so the bound grows slower than the score for every other candidate),
//   the fast winner is the exact winner; the kernel puts an upper bound of A in its place
//   (the fp32 sum times 1 + 2^-19; a larger A only widens the margin).  (A quotient
//   below the normal range carries an absolute error of half a denormal unit instead;
//   such an element rounds to zero under every candidate, and a group made only of them
//   has scores within rounding of A under every candidate, which the 2^-18 E2 term sends
//   to the exact rescoring.)
//   Otherwise the group is "ambiguous" and the whole warp rescores it cooperatively with
//   exact rounding decisions (16 lanes per candidate, one element each, a fixed
//   pairwise shuffle tree per error: relative error <= 8 * 2^-24), applying the tie
//   rule (smaller error, then smaller |shift|, then smaller shift).  The winner's
//   nibbles are always produced with exact round-to-nearest-even decisions.
#include <algorithm>
#include <atomic>

#include "hscale_device.cuh"
#include "hscale_internal.h"
#include "tma.cuh"

namespace hscale {
namespace {

constexpr int kRefineThreads = 128;
constexpr int kWarpsPerRefineBlock = kRefineThreads / 32;
constexpr float kInf = __builtin_huge_valf();

// ---------------------------------------------------------------- amax
__global__ void __launch_bounds__(256) amax_kernel(const uint4* __restrict__ w, int64_t nvec,
                                                   uint32_t* __restrict__ amax_bits) {
  __shared__ uint32_t warp_max[8];
  uint32_t m2 = 0;  // two packed 16-bit maxima
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    const uint4 v = ld_stream_v4(w + i);
    m2 = __vmaxu2(m2, v.x & 0x7FFF7FFFu);
    m2 = __vmaxu2(m2, v.y & 0x7FFF7FFFu);
    m2 = __vmaxu2(m2, v.z & 0x7FFF7FFFu);
    m2 = __vmaxu2(m2, v.w & 0x7FFF7FFFu);
  }
  uint32_t m = max(m2 & 0xFFFFu, m2 >> 16);
  m = __reduce_max_sync(0xFFFFFFFFu, m);
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x < 32) {
    m = threadIdx.x < (blockDim.x >> 5) ? warp_max[threadIdx.x] : 0u;
    m = __reduce_max_sync(0xFFFFFFFFu, m);
    if (threadIdx.x == 0 && m) atomicMax(amax_bits, m);
  }
}

__device__ __forceinline__ float global_scale_of(uint32_t amax_bits) {
  const float amax = __uint_as_float(amax_bits << 16);
  return amax == 0.0f ? 1.0f : __fdiv_rn(amax, 2688.0f);  // 6 * 448
}

// max(|x|, |y|) of two bf16 pairs, half by half (the sign of each half is the product of
// the inputs' signs; finite inputs).  One of the inputs' magnitudes is returned exactly.
__device__ __forceinline__ uint32_t bf16x2_absmax(uint32_t x, uint32_t y) {
  uint32_t r;
  asm("max.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(x), "r"(y));
  return r;
}

// The 16-bit |bf16| pattern of the group's largest magnitude (for finite values the order
// of magnitudes is the order of their patterns).
__device__ __forceinline__ uint32_t group_abs_max_bits(const uint4& a, const uint4& b) {
  const uint32_t m = bf16x2_absmax(bf16x2_absmax(bf16x2_absmax(a.x, a.y), bf16x2_absmax(a.z, a.w)),
                                   bf16x2_absmax(bf16x2_absmax(b.x, b.y), bf16x2_absmax(b.z, b.w)));
  return bf16x2_absmax(m, __byte_perm(m, 0, 0x1032)) & 0x7FFFu;
}

// ---------------------------------------------------------------- RTN codes
__global__ void __launch_bounds__(256) rtn_codes_kernel(const uint4* __restrict__ w, int64_t groups,
                                                        const uint32_t* __restrict__ amax_bits,
                                                        float* __restrict__ global_scale,
                                                        uint8_t* __restrict__ codes) {
  const float sg = global_scale_of(*amax_bits);
  if (blockIdx.x == 0 && threadIdx.x == 0) *global_scale = sg;
  if (codes == nullptr) return;
  const ScaleDomain d = make_scale_domain(sg);
  const float inv6 = rtn_inv6_raw(d.sgk);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += stride) {
    const uint4 a = ld_stream_v4(w + 2 * g);
    const uint4 b = ld_stream_v4(w + 2 * g + 1);
    const float amax_k = __fmul_rn(__uint_as_float(group_abs_max_bits(a, b) << 16), d.pw);
    codes[g] = (uint8_t)rtn_code(amax_k, d.sgk, inv6);
  }
}

// ---------------------------------------------------------------- search helpers
// a_j keeps the sign of w_j.  Every score is even in a_j (round-to-nearest-even and
// saturation are symmetric, and only squares of residuals enter), so the search pays
// nothing for the sign, and the pack converts the signed quotients directly.
struct Group {
  float2 a[8];     // w * 2^-K, elements (2i, 2i+1)
};

// The group's 16 bf16 values, given as two 16-byte words (element 2i in the low half of
// word i), unpacked and scaled.
__device__ __forceinline__ void unpack_group(const uint4& p, const uint4& q, float pw, Group& G) {
  const uint32_t wb[8] = {p.x, p.y, p.z, p.w, q.x, q.y, q.z, q.w};
#pragma unroll
  for (int i = 0; i < 8; ++i)
    G.a[i] = __fmul2_rn(make_float2(bf16_lo(wb[i]), bf16_hi(wb[i])), make_float2(pw, pw));
}

// The group whose 16 bf16 values start at wg (16-byte aligned).
__device__ __forceinline__ void load_group_at(const uint4* wg, float pw, Group& G) {
  unpack_group(ld_stream_v4(wg), ld_stream_v4(wg + 1), pw, G);
}

__device__ __forceinline__ void load_group(const uint4* w, int64_t g, float pw, Group& G) {
  load_group_at(w + 2 * g, pw, G);
}

// Per-block table of the candidate constants of every E4M3 code c (1..126), filled once
// per CTA and stored pre-splatted for the packed arithmetic: x = y = s'^2 and
// z = w = 1 / s' (correctly rounded), with s' = l(c) * sgk in [2^-21, 2^-2], so both are
// normal numbers.  One 16-byte shared load per candidate replaces a decode, a multiply
// and a reciprocal on the candidate's critical path.
__device__ __forceinline__ float4 candidate_constants(uint32_t c, float sgk) {
  const float sp = __fmul_rn(e4m3_mag(c), sgk);
  const float s2 = __fmul_rn(sp, sp), inv = c ? __frcp_rn(sp) : 0.0f;
  return make_float4(s2, s2, inv, inv);
}

// q - y for a pair of quotients y (real units): q = RNE_sat(y) by the hardware E2M1
// conversion, back to f16 (exact), and one mixed f16 - f32 subtract per element.
__device__ __forceinline__ float2 e2m1_residual2(float2 y) {
  float d0, d1;
  asm("{\n\t.reg .b8 c;\n\t.reg .b32 q;\n\t.reg .f16 lo, hi;\n\t"
      "cvt.rn.satfinite.e2m1x2.f32 c, %3, %2;\n\t"
      "cvt.rn.f16x2.e2m1x2 q, c;\n\t"
      "mov.b32 {lo, hi}, q;\n\t"
      "sub.rn.f32.f16 %0, lo, %2;\n\t"
      "sub.rn.f32.f16 %1, hi, %3;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(y.x), "f"(y.y));
  return make_float2(d0, d1);
}

// Fast score of one candidate from its table entry t (see the file comment): per pair of
// elements one packed multiply for the quotients, the hardware rounding and residuals,
// a packed square and a packed FMA into the h-weighted sum (one chain per half of the
// pair: the candidates scored side by side give the independent work); then the halves'
// sum and one multiply by s'^2.
__device__ __forceinline__ float fast_score(const Group& G, const float2 (&hv2)[8], float4 t) {
  const float2 inv2 = make_float2(t.z, t.w);
  float2 acc = make_float2(0.f, 0.f);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 d = e2m1_residual2(__fmul2_rn(G.a[i], inv2));
    acc = __ffma2_rn(hv2[i], __fmul2_rn(d, d), acc);
  }
  return __fmul_rn(t.x, __fadd_rn(acc.x, acc.y));
}

// Running best (e1, best) and runner-up e2 (e1 <= e2); branch-free: a select and three
// min/max.  A tie with the best makes e2 = e1 (the margin test then fails); NaN scores
// are ignored.
__device__ __forceinline__ void keep_best(float e, int c, float& e1, float& e2, int& best) {
  best = e < e1 ? c : best;
  e2 = fminf(e2, fmaxf(e1, e));
  e1 = fminf(e1, e);
}

// Scores the codes [a, b) two at a time (independent chains interleave).
__device__ __forceinline__ void score_range(const Group& G, const float2 (&hv2)[8],
                                            const float4* tab, int a, int b, float& e1, float& e2,
                                            int& best) {
  int c = a;
  for (; c + 1 < b; c += 2) {
    const float4 t0 = tab[c], t1 = tab[c + 1];
    const float ea = fast_score(G, hv2, t0);
    const float eb = fast_score(G, hv2, t1);
    keep_best(ea, c, e1, e2, best);
    keep_best(eb, c + 1, e1, e2, best);
  }
  if (c < b) keep_best(fast_score(G, hv2, tab[c]), c, e1, e2, best);
}

// Upper bound of A = sum_j h_j a_j^2, the scale of the fast-score error bound:
// (sum_j h_j) * max_j a_j^2.  Two multiplies instead of a pass over the group; a larger A
// only widens the margin (the rounding of the bound, a relative 2^-20 at most, is far
// inside the margin's 2x slack).
__device__ __forceinline__ float energy_bound(float hsum, float amax_k) {
  return __fmul_rn(hsum, __fmul_rn(amax_k, amax_k));
}

// A = sum_j h_j a_j^2 itself (scaled domain), for the search's margin test.  (sum h) amax^2
// can exceed it many times over (one large weight, or h concentrated on small ones), and
// the margin's dominant term grows with sqrt(A), so the tighter value sends several times
// fewer groups to the exact rescoring.  The fp32 sum of non-negative terms is within a
// relative 12 * 2^-24 of A; the factor 1 + 2^-19 makes the result an upper bound.
__device__ __forceinline__ float group_energy(const Group& G, const float2 (&hv2)[8]) {
  float2 acc = __fmul2_rn(hv2[0], __fmul2_rn(G.a[0], G.a[0]));
#pragma unroll
  for (int i = 1; i < 8; ++i) acc = __ffma2_rn(hv2[i], __fmul2_rn(G.a[i], G.a[i]), acc);
  return __fmul_rn(__fadd_rn(acc.x, acc.y), 1.0f + 0x1p-19f);
}

// A sufficient condition for fast_winner_certain that costs six operations: a relative
// gap above 2^-9 with A <= 2^18 E2 (A_bound any upper bound of A, here (sum h) amax^2)
// gives a margin of at most (2^-18 + 2^-19 2^9 + 2^-35 2^18) E2 < 2^-9 E2, and
// E2 >= 2^-36 A.  (The fp32 rounding of the gap and of A_bound is a few units of 2^-24,
// far inside the factor of two between 2^-9 and the margin.)  The scores' error bound
// holds for results in the normal range, so a runner-up below 2^-100 is left to
// fast_winner_certain (which sends denormal ones to the exact rescoring); a zero,
// infinite or NaN runner-up fails it too.
__device__ __forceinline__ bool fast_winner_clear(float e1, float e2, float A_bound) {
  return e2 >= 0x1p-100f && __fsub_rn(e2, e1) > __fmul_rn(0x1p-9f, e2) && A_bound <= __fmul_rn(0x1p18f, e2);
}

// tie rule of the search: smaller error, then smaller |shift|, then smaller shift
__device__ __forceinline__ bool better(float e, int c, float be, int bc, int c0) {
  if (e != be) return e < be;
  const int s = c - c0, bs = bc - c0;
  const int as = s < 0 ? -s : s, abs_ = bs < 0 ? -bs : bs;
  return as < abs_ || (as == abs_ && s < bs);
}

// Exact-decision score of one element under code c (scaled domain, one rounding in the
// residual: q * l is exact and the FMA rounds once).
__device__ __forceinline__ float exact_term(float a_k, float hj, uint32_t c, float sgk) {
  const float l = e4m3_mag(c);
  const float inv = inv_raw_of(__fmul_rn(l, sgk));
  const uint32_t k = e2m1_code(a_k, inv, l, sgk);
  const float ql = __fmul_rn(e2m1_from_raw(k << 22), l);
  const float r = __fmaf_rn(-ql, sgk, a_k);
  return __fmul_rn(hj, __fmul_rn(r, r));
}

// The whole warp rescores the group of lane `owner` with exact rounding decisions and
// returns its winning code (in every lane).  Lanes 0-15 take the candidates lo, lo+2,
// ..., lanes 16-31 lo+1, lo+3, ...; lane j of each half scores element j & 15.
__device__ __noinline__ int warp_exact_search(int owner, const uint16_t* wg_own, const float* h,
                                 int64_t hcol_own, int c0, int lo, int hi, float sgk, float pw) {
  const int lane = threadIdx.x & 31;
  const int j = lane & 15, half = lane >> 4;
  const uint16_t wb = wg_own[j];
  const float a_k = __fmul_rn(fabsf(__uint_as_float((uint32_t)wb << 16)), pw);
  const float hj = h ? h[hcol_own * 16 + j] : 1.0f;
  const unsigned mask = 0xFFFFu << (16 * half);
  float be = kInf;
  int bc = -1;
  for (int c = lo + half; c <= hi; c += 2) {
    float e = exact_term(a_k, hj, (uint32_t)c, sgk);
    e = __fadd_rn(e, __shfl_xor_sync(mask, e, 1));
    e = __fadd_rn(e, __shfl_xor_sync(mask, e, 2));
    e = __fadd_rn(e, __shfl_xor_sync(mask, e, 4));
    e = __fadd_rn(e, __shfl_xor_sync(mask, e, 8));
    if (bc < 0 || better(e, c, be, bc, c0)) { be = e; bc = c; }
  }
  __syncwarp();
  const float oe = __shfl_xor_sync(0xFFFFFFFFu, be, 16);
  const int oc = __shfl_xor_sync(0xFFFFFFFFu, bc, 16);
  if (oc >= 0 && (bc < 0 || better(oe, oc, be, bc, c0))) { be = oe; bc = oc; }
  (void)owner;
  return bc;
}

// Hardware E2M1 conversion of two fp32 values (round-to-nearest-even, saturating at
// +-6, sign kept, also for a result of zero): one byte, `hi` in the upper nibble.
__device__ __forceinline__ uint32_t cvt_e2m1x2(float hi, float lo) {
  uint32_t r;
  asm("{\n\t.reg .b8 t;\n\tcvt.rn.satfinite.e2m1x2.f32 t, %1, %2;\n\tcvt.u32.u8 %0, t;\n\t}"
      : "=r"(r)
      : "f"(hi), "f"(lo));
  return r;
}

// The anchored code of Eq. 7 (anchor c = 2 * half_c; RTN is c = 6), decided by the hardware
// E4M3 conversion (round-to-nearest-even, saturating at 448) of two bracketing quotients
// r_lo = amax_k * inv_lo and r_hi = amax_k * inv_hi, with inv_lo and inv_hi the reciprocal
// 1 / (c sgk) (relative error <= 2^-23) scaled by 1 -+ 2^-20: r_lo lies below the exact
// quotient amax_g / (c s_g) and r_hi above it, so where the two conversions (one
// instruction for the pair) agree, that code is the exact rounding; otherwise an E4M3
// midpoint lies between them and the exact midpoint tests of anchored_code() decide.
// Quotients below the fp32 normal range convert to code 0 under both.  Code 0 is clamped
// to 1.
__device__ __forceinline__ uint32_t anchored_code_fast(float amax_k, float sgk, float inv_lo, float inv_hi,
                                                       float inv_raw, float half_c) {
  const float rl = __fmul_rn(amax_k, inv_lo), rh = __fmul_rn(amax_k, inv_hi);
  uint32_t p;
  asm("{\n\t.reg .b16 t;\n\tcvt.rn.satfinite.e4m3x2.f32 t, %1, %2;\n\tcvt.u32.u16 %0, t;\n\t}"
      : "=r"(p)
      : "f"(rh), "f"(rl));
  uint32_t c = p & 0xFFu;
  if (c != (p >> 8)) c = anchored_code(amax_k, sgk, inv_raw, half_c);
  return c < 1u ? 1u : c;
}

// Bracketing factors of a reciprocal (see quantize_pack): 1 -+ 2^-20.
constexpr float kBracketLo = 1.0f - 0x1p-20f;
constexpr float kBracketHi = 1.0f + 0x1p-20f;

// Exact final re-quantization of one group under code c: 8 bytes of packed nibbles.
// inv ~ 1 / s' is the correctly rounded reciprocal of s' = l(c) sgk (the candidate
// table's), so y = a * inv is within a relative 2^-23 (+ 2^-48) of the exact quotient
// y* = a / s'.  The quotients are formed under two bracketing reciprocals,
// inv (1 - 2^-20) and inv (1 + 2^-20), each rounded once more: the one is below |y*| and
// the other above it by at least 2^-21 |y*| - 4 * 2^-24 |y*| > 0.  Round-to-nearest-even
// is monotone, so where the hardware conversions (RNE, saturation, sign kept also for a
// zero) of the two agree, that is the exact rounding of y*; the two differ only where a
// midpoint of the grid lies between them (an exact tie among them), and those elements are
// decided exactly with the one-FMA midpoint test of e2m1_exact_code, reading the weight back
// from `wg` (the group's 16 bf16 values): the lower conversion gives the lower of the two
// grid points.  A quotient below the normal range is far below the first midpoint 0.25 and
// converts to a signed zero under both reciprocals.
// Four element pairs (real-unit quotients) converted to E2M1 nibble pairs and packed into
// one 32-bit word, pair i in byte i.
__device__ __forceinline__ uint32_t cvt_e2m1x8(float2 y0, float2 y1, float2 y2, float2 y3) {
  uint32_t r;
  asm("{\n\t.reg .b8 b0, b1, b2, b3;\n\t"
      "cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n\t"
      "cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n\t"
      "cvt.rn.satfinite.e2m1x2.f32 b2, %6, %5;\n\t"
      "cvt.rn.satfinite.e2m1x2.f32 b3, %8, %7;\n\t"
      "mov.b32 %0, {b0, b1, b2, b3};\n\t}"
      : "=r"(r)
      : "f"(y0.x), "f"(y0.y), "f"(y1.x), "f"(y1.y), "f"(y2.x), "f"(y2.y), "f"(y3.x), "f"(y3.y));
  return r;
}

// Bit 4j of the result is set iff nibble j of x is non-zero.
__device__ __forceinline__ uint32_t nonzero_nibbles(uint32_t x) {
  x |= x >> 1;
  x |= x >> 2;
  return x & 0x11111111u;
}

__device__ __forceinline__ uint2 quantize_pack(const Group& G, uint32_t c, float inv, float sgk, float pw,
                                               const uint16_t* wg) {
  const float ilo = __fmul_rn(inv, kBracketLo), ihi = __fmul_rn(inv, kBracketHi);
  const float2 il2 = make_float2(ilo, ilo), ih2 = make_float2(ihi, ihi);
  uint32_t lo[2], hi[2];
#pragma unroll
  for (int wd = 0; wd < 2; ++wd) {
    const float2* a = G.a + 4 * wd;
    lo[wd] = cvt_e2m1x8(__fmul2_rn(a[0], il2), __fmul2_rn(a[1], il2), __fmul2_rn(a[2], il2), __fmul2_rn(a[3], il2));
    hi[wd] = cvt_e2m1x8(__fmul2_rn(a[0], ih2), __fmul2_rn(a[1], ih2), __fmul2_rn(a[2], ih2), __fmul2_rn(a[3], ih2));
  }
  if ((lo[0] ^ hi[0]) | (lo[1] ^ hi[1])) {
    const float l = e4m3_mag(c);
#pragma unroll
    for (int wd = 0; wd < 2; ++wd) {
      uint32_t flagged = nonzero_nibbles(lo[wd] ^ hi[wd]);
      while (flagged) {
        const int sh = __ffs(flagged) - 1;  // 4 * (element index within the word)
        flagged &= flagged - 1;
        const uint32_t nib = (lo[wd] >> sh) & 0xFu;  // the lower magnitude code, with the sign
        const float a = __fmul_rn(__uint_as_float(((uint32_t)wg[8 * wd + (sh >> 2)] & 0x7FFFu) << 16), pw);
        const uint32_t k = e2m1_code_between(a, nib & 7u, l, sgk);
        lo[wd] = (lo[wd] & ~(0xFu << sh)) | (((nib & 8u) | k) << sh);
      }
    }
  }
  return make_uint2(lo[0], lo[1]);
}

// ---------------------------------------------------------------- 4over6 scores (Algorithm 2)
// Plain-MSE error of one group under code c with exact rounding decisions: one rounding
// in each residual (q * l is exact inside the FMA), the square, and a fixed pairwise
// 16-term sum; relative error <= 7 * 2^-24.
__device__ __forceinline__ float exact_group_mse(const Group& G, uint32_t c, float sgk) {
  const float l = e4m3_mag(c);
  const float inv = inv_raw_of(__fmul_rn(l, sgk));
  float t[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float a = fabsf((j & 1) ? G.a[j >> 1].y : G.a[j >> 1].x);
    const uint32_t k = e2m1_code(a, inv, l, sgk);
    const float r = __fmaf_rn(-__fmul_rn(e2m1_from_raw(k << 22), l), sgk, a);
    t[j] = __fmul_rn(r, r);
  }
#pragma unroll
  for (int step = 1; step < 16; step <<= 1)
#pragma unroll
    for (int j = 0; j + step < 16; j += 2 * step) t[j] = __fadd_rn(t[j], t[j + step]);
  return t[0];
}

// Fast plain-MSE score of one candidate (fast_score with every h_j = 1).
__device__ __forceinline__ float fast_mse(const Group& G, float4 t) {
  const float2 inv2 = make_float2(t.z, t.w);
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 d = e2m1_residual2(__fmul2_rn(G.a[i], inv2));
    if (i & 1) acc1 = __ffma2_rn(d, d, acc1);
    else acc0 = __ffma2_rn(d, d, acc0);
  }
  const float2 t2 = __fadd2_rn(acc0, acc1);
  return __fmul_rn(t.x, __fadd_rn(t2.x, t2.y));
}

// Is the fast winner (fast score e1) certainly ahead of the runner-up (e2), given the
// energy A = sum_j h_j a_j^2 of the group (or an upper bound of it)?  The test of the file comment, in units of e2
// (no underflow or overflow for 2^-36 A <= e2 <= A-ish):
//   g = (e2 - e1) / e2 - 2^-18 - 2^-35 A / e2 > 2^-19 sqrt(A / e2), tested on squares.
// A zero, denormal or non-finite e2 makes the reciprocal infinite or NaN and g fails.
__device__ __forceinline__ bool fast_winner_certain(float e1, float e2, float A) {
  const float r = rcp_approx(e2);
  const float ratio = __fmul_rn(A, r);
  const float g = __fsub_rn(__fsub_rn(__fmul_rn(__fsub_rn(e2, e1), r), 0x1p-18f), __fmul_rn(0x1p-35f, ratio));
  const bool certain = g > 0.0f && __fmul_rn(g, g) > __fmul_rn(0x1p-38f, ratio);
  return certain && ratio <= 0x1p36f && A > 0.0f;
}

// The anchor choice of Algorithm 2 for one group with exact rounding decisions (the
// group is read back from global memory); the anchor 4 code c4 wins an exact tie.  Kept
// out of line: the search calls it only when the fast scores cannot order the anchors.
__device__ __noinline__ uint32_t fourover6_exact_pick(const uint4* wg, float pw, uint32_t c4, uint32_t c6,
                                                      float sgk) {
  Group G;
  load_group_at(wg, pw, G);
  return exact_group_mse(G, c6, sgk) < exact_group_mse(G, c4, sgk) ? c6 : c4;
}

// Algorithm 2's initial code of one group, decided in the search kernel: the two
// anchored codes, their fast plain-MSE scores from the candidate table and, only when
// the margin test cannot order them, the exact comparison.  When the test passes, the
// fast order is the order of the exact errors, and the exact fp32 sums (relative error
// <= 7 * 2^-24, far inside the margin) order them the same way; so the result is always
// the code fourover6_codes_kernel writes.
__device__ __forceinline__ int fourover6_init_code(const Group& G, const uint4* wg, const float4* tab,
                                                   float amax_k, float sgk, float pw, float inv4, float inv6,
                                                   const float2& b4, const float2& b6) {
  const uint32_t c4 = anchored_code_fast(amax_k, sgk, b4.x, b4.y, inv4, 2.0f);
  const uint32_t c6 = anchored_code_fast(amax_k, sgk, b6.x, b6.y, inv6, 3.0f);
  if (c4 == c6) return (int)c4;
  const float e4 = fast_mse(G, tab[c4]);
  const float e6 = fast_mse(G, tab[c6]);
  if (fast_winner_certain(fminf(e4, e6), fmaxf(e4, e6), energy_bound(16.0f, amax_k)))
    return (int)(e6 < e4 ? c6 : c4);
  return (int)fourover6_exact_pick(wg, pw, c4, c6, sgk);
}

// ---------------------------------------------------------------- refine (Algorithm 1)
// 16-byte asynchronous copy global -> shared (L1 bypassed), and the wait for all but the
// latest `n` groups of this thread's copies.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem)), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

// Reciprocal 1 / (c sgk) scaled by the bracketing factors (lo, hi) of anchored_code_fast.
__device__ __forceinline__ float2 anchor_brackets(float sgk, float c) {
  const float r = __frcp_rn(__fmul_rn(c, sgk));
  return make_float2(__fmul_rn(r, kBracketLo), __fmul_rn(r, kBracketHi));
}

// Work unit: one warp, 32 consecutive groups of one row (a "row chunk", 1 KB of W); warps
// stride over (row, chunk) units so the h slice of a lane is reloaded only when its chunk
// changes.  Each lane copies its group of the warp's next unit into a per-warp staging
// buffer in shared memory (cp.async, two buffers) while the current unit is scored, so the
// scoring never waits for W; a lane reads back only what it copied itself.  7 resident
// CTAs of 4 warps per SM; the rarely taken warp-cooperative rescoring is a separate call so
// it does not raise the register count.
// kFourOverSix: the initial codes are Algorithm 2's, decided in place (init_codes unused).
// W, the codes and the nibbles are 2-D views: row r starts at element r * ld_w of w, byte
// r * ld_i of the initial codes, byte r * ld_c of the codes and 8-byte word r * ld_p of the
// nibbles.
template <bool kFourOverSix>
__global__ void __launch_bounds__(kRefineThreads, 7)
refine_kernel(const uint4* __restrict__ w, int64_t ld_w, const float* __restrict__ h, int64_t m, int ng,
              const float* __restrict__ global_scale, const uint8_t* init_codes, int64_t ld_i,
              int down, int up, uint8_t* codes_out, int64_t ld_c, uint2* __restrict__ packed_out, int64_t ld_p) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int64_t warp_global = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t warps_total = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int chunks = (ng + 31) / 32;
  const int64_t units = m * chunks;

  __shared__ float4 tab[128];
  // per warp, two buffers of one unit: the first 16 bytes of every lane's group, then the
  // second 16 bytes (consecutive lanes, consecutive 16-byte words: conflict-free)
  __shared__ __align__(16) uint4 stage[kWarpsPerRefineBlock][2][64];
  const ScaleDomain d = make_scale_domain(*global_scale);
  const float inv6 = rtn_inv6_raw(d.sgk);
  const float inv4 = kFourOverSix ? anchor_inv_raw(d.sgk, 4.0f) : 0.0f;
  const float2 b6 = anchor_brackets(d.sgk, 6.0f);
  const float2 b4 = kFourOverSix ? anchor_brackets(d.sgk, 4.0f) : make_float2(0.f, 0.f);
  for (int c = threadIdx.x; c < 128; c += blockDim.x) tab[c] = candidate_constants((uint32_t)c, d.sgk);

  int cur_chunk = -1;
  float2 hv2[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) hv2[j] = make_float2(1.0f, 1.0f);

  // (row, chunk) of unit u, advanced by warps_total units per step without a division
  const int row_step = (int)(warps_total / chunks);
  const int chunk_step = (int)(warps_total - (int64_t)row_step * chunks);
  int64_t row = warp_global / chunks;
  int chunk = (int)(warp_global - row * chunks);

  // the copy of unit (r, ch), if it exists, into buffer `buf`; always one commit group
  auto stage_unit = [&](int64_t uu, int64_t r, int ch, int buf) {
    const int gc = ch * 32 + lane;
    if (uu < units && gc < ng) {
      const uint4* src = w + (r * ld_w + (int64_t)gc * 16) / 8;
      cp_async16(&stage[warp][buf][lane], src);
      cp_async16(&stage[warp][buf][32 + lane], src + 1);
    }
    cp_async_commit();
  };
  stage_unit(warp_global, row, chunk, 0);
  __syncthreads();  // the candidate table

  int buf = 0;
  for (int64_t u = warp_global; u < units; u += warps_total, buf ^= 1) {
    const int gcol = chunk * 32 + lane;
    const bool active = gcol < ng;
    const int64_t wofs = row * ld_w + (int64_t)gcol * 16;  // first element of the group
    // (row, chunk) of the warp's next unit, whose copy starts now
    int64_t nrow = row + row_step;
    int nchunk = chunk + chunk_step;
    if (nchunk >= chunks) {
      nchunk -= chunks;
      ++nrow;
    }
    stage_unit(u + warps_total, nrow, nchunk, buf ^ 1);

    if (chunk != cur_chunk) {
      cur_chunk = chunk;
      if (h != nullptr && active) {
        const float4* hp = reinterpret_cast<const float4*>(h + (int64_t)gcol * 16);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 t = hp[i];
          hv2[2 * i] = make_float2(t.x, t.y);
          hv2[2 * i + 1] = make_float2(t.z, t.w);
        }
      }
    }

    Group G;
    int c0 = 1, lo = 1, hi = 1;
    float amax_k = 0.0f;
    cp_async_wait_1();  // this lane's copy of the current unit has landed
    if (active) {
      const uint4 p = stage[warp][buf][lane];
      const uint4 q = stage[warp][buf][32 + lane];
      amax_k = __fmul_rn(__uint_as_float(group_abs_max_bits(p, q) << 16), d.pw);
      unpack_group(p, q, d.pw, G);
      if (!kFourOverSix && init_codes != nullptr) {
        c0 = init_codes[row * ld_i + gcol] & 0x7F;
        c0 = c0 < 1 ? 1 : (c0 > (int)kE4M3MaxCode ? (int)kE4M3MaxCode : c0);
      } else {
        c0 = kFourOverSix ? fourover6_init_code(G, w + wofs / 8, tab, amax_k, d.sgk, d.pw, inv4, inv6, b4, b6)
                          : (int)anchored_code_fast(amax_k, d.sgk, b6.x, b6.y, inv6, 3.0f);
      }
      lo = max(1, c0 - down);
      hi = min((int)kE4M3MaxCode, c0 + up);
    }

    // ---- fast scores of every distinct candidate (the same trip count in every lane
    // unless the window is clipped at the ends of the ladder)
    float e1 = kInf, e2 = kInf;
    int best = c0;
    if (active) score_range(G, hv2, tab, lo, hi + 1, e1, e2, best);

    // ---- is the fast winner certain?
    bool ambiguous = false;
    if (active && hi > lo) ambiguous = !fast_winner_certain(e1, e2, group_energy(G, hv2));
    unsigned amb = __ballot_sync(0xFFFFFFFFu, ambiguous);
    while (amb) {
      const int owner = __ffs(amb) - 1;
      amb &= amb - 1;
      const int64_t wofs_own = __shfl_sync(0xFFFFFFFFu, wofs, owner);
      const int gcol_own = __shfl_sync(0xFFFFFFFFu, gcol, owner);
      const int c0o = __shfl_sync(0xFFFFFFFFu, c0, owner);
      const int loo = __shfl_sync(0xFFFFFFFFu, lo, owner);
      const int hio = __shfl_sync(0xFFFFFFFFu, hi, owner);
      const int bc = warp_exact_search(owner, reinterpret_cast<const uint16_t*>(w) + wofs_own, h, gcol_own,
                                       c0o, loo, hio, d.sgk, d.pw);
      if (lane == owner) best = bc;
    }

    if (active) {
      codes_out[row * ld_c + gcol] = (uint8_t)best;
      if (packed_out != nullptr)
        packed_out[row * ld_p + gcol] = quantize_pack(G, (uint32_t)best, tab[best].z, d.sgk, d.pw,
                                                      reinterpret_cast<const uint16_t*>(w) + wofs);
    }
    row = nrow;
    chunk = nchunk;
  }
}

// Constants of one search call shared by every group.
struct SearchConsts {
  float inv6, inv4;  // anchored_code's reciprocals for the anchors 6 and 4
  float2 b6, b4;     // their bracketing pairs (anchored_code_fast)
};

__device__ __forceinline__ SearchConsts search_consts(const ScaleDomain& d, bool fourover6) {
  SearchConsts k;
  k.inv6 = rtn_inv6_raw(d.sgk);
  k.inv4 = fourover6 ? anchor_inv_raw(d.sgk, 4.0f) : 0.0f;
  k.b6 = anchor_brackets(d.sgk, 6.0f);
  k.b4 = fourover6 ? anchor_brackets(d.sgk, 4.0f) : make_float2(0.f, 0.f);
  return k;
}

// One unit of the contiguous layout: every lane searches its group g (index `go`, whose 16
// bf16 values are p, q and sit at wg in W; h slice hv2 of column group hcol = chunk * 32 +
// lane) and writes code byte go and nibble word go.  All 32 lanes take part (the warp
// rescores ambiguous groups together).
template <bool kFourOverSix>
__device__ __forceinline__ void search_unit(const uint4& p, const uint4& q, const uint4* wg, int64_t go, int64_t chunk,
                                            const float2 (&hv2)[8], float hsum, const uint4* __restrict__ w,
                                            const float* __restrict__ h, const float4* tab, const ScaleDomain& d,
                                            const SearchConsts& k, const uint8_t* init_codes, int down, int up,
                                            uint8_t* codes_out, uint2* __restrict__ packed_out) {
  const int lane = threadIdx.x & 31;
  const float amax_k = __fmul_rn(__uint_as_float(group_abs_max_bits(p, q) << 16), d.pw);
  Group G;
  unpack_group(p, q, d.pw, G);
  int c0;
  if (!kFourOverSix && init_codes != nullptr) {
    c0 = init_codes[go] & 0x7F;
    c0 = c0 < 1 ? 1 : (c0 > (int)kE4M3MaxCode ? (int)kE4M3MaxCode : c0);
  } else {
    c0 = kFourOverSix ? fourover6_init_code(G, wg, tab, amax_k, d.sgk, d.pw, k.inv4, k.inv6, k.b4, k.b6)
                      : (int)anchored_code_fast(amax_k, d.sgk, k.b6.x, k.b6.y, k.inv6, 3.0f);
  }
  const int lo = max(1, c0 - down);
  const int hi = min((int)kE4M3MaxCode, c0 + up);

  float e1 = kInf, e2 = kInf;
  int best = c0;
  score_range(G, hv2, tab, lo, hi + 1, e1, e2, best);

  // the cheap sufficient test with the loose energy bound first; the exact energy and the
  // full test only for the groups it cannot clear
  bool ambiguous = hi > lo && !fast_winner_clear(e1, e2, energy_bound(hsum, amax_k));
  if (ambiguous) ambiguous = !fast_winner_certain(e1, e2, group_energy(G, hv2));
  unsigned amb = __ballot_sync(0xFFFFFFFFu, ambiguous);
  while (amb) {
    const int owner = __ffs(amb) - 1;
    amb &= amb - 1;
    const int64_t g_own = __shfl_sync(0xFFFFFFFFu, go, owner);
    const int c0o = __shfl_sync(0xFFFFFFFFu, c0, owner);
    const int loo = __shfl_sync(0xFFFFFFFFu, lo, owner);
    const int hio = __shfl_sync(0xFFFFFFFFu, hi, owner);
    const int bc = warp_exact_search(owner, reinterpret_cast<const uint16_t*>(w) + g_own * 16, h,
                                     chunk * 32 + owner, c0o, loo, hio, d.sgk, d.pw);
    if (lane == owner) best = bc;
  }

  codes_out[go] = (uint8_t)best;
  if (packed_out != nullptr)
    packed_out[go] = quantize_pack(G, (uint32_t)best, tab[best].z, d.sgk, d.pw,
                                   reinterpret_cast<const uint16_t*>(wg));
}

// Loads the h slice of column chunk `chunk` (this lane's 16 values) and its sum.
__device__ __forceinline__ void load_h_slice(const float* __restrict__ h, int64_t chunk, float2 (&hv2)[8],
                                             float& hsum) {
  const int lane = threadIdx.x & 31;
  const float4* hp = reinterpret_cast<const float4*>(h + (chunk * 32 + lane) * 16);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 t = hp[i];
    hv2[2 * i] = make_float2(t.x, t.y);
    hv2[2 * i + 1] = make_float2(t.z, t.w);
  }
  float2 s2 = __fadd2_rn(__fadd2_rn(hv2[0], hv2[1]), __fadd2_rn(hv2[2], hv2[3]));
  s2 = __fadd2_rn(s2, __fadd2_rn(__fadd2_rn(hv2[4], hv2[5]), __fadd2_rn(hv2[6], hv2[7])));
  hsum = __fadd_rn(s2.x, s2.y);
}

// The search over a contiguous W [m, n] with n a multiple of 512 (every unit a full row
// chunk) and contiguous outputs: the same work as refine_kernel per group, with the walk
// reduced to pointer increments.  Unit u is groups [32 u, 32 u + 32), i.e. the 1 KB of W at
// uint4 offset 64 u, code bytes [32 u, 32 u + 32) and nibble words [32 u, 32 u + 32); every
// lane of every unit is active.  Warps take every warps_total-th unit (a static deal).
template <bool kFourOverSix>
__global__ void __launch_bounds__(kRefineThreads, 7)
refine_linear_kernel(const uint4* __restrict__ w, const float* __restrict__ h, int64_t units, int chunks,
                     const float* __restrict__ global_scale, const uint8_t* init_codes, int down, int up,
                     uint8_t* codes_out, uint2* __restrict__ packed_out) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int64_t warp_global = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t warps_total = ((int64_t)gridDim.x * blockDim.x) >> 5;

  __shared__ float4 tab[128];
  __shared__ __align__(16) uint4 stage[kWarpsPerRefineBlock][2][64];
  const ScaleDomain d = make_scale_domain(*global_scale);
  const SearchConsts k = search_consts(d, kFourOverSix);
  for (int c = threadIdx.x; c < 128; c += blockDim.x) tab[c] = candidate_constants((uint32_t)c, d.sgk);

  // this lane's group of unit u: uint4 words 64 u + 2 lane and the one after
  const int64_t wstep = warps_total * 64;
  const uint4* wp = w + warp_global * 64 + 2 * lane;
  const int64_t ostep = warps_total * 32;
  int64_t go = warp_global * 32 + lane;  // this lane's group index
  // the grid holds at most 2^31 warps, so 32-bit remainders suffice
  int chunk = (int)((uint32_t)warp_global % (uint32_t)chunks);
  const int chunk_step = (int)((uint32_t)warps_total % (uint32_t)chunks);
  uint4* const st0 = &stage[warp][0][lane];
  uint4* const st1 = &stage[warp][1][lane];

  if (warp_global < units) {
    cp_async16(st0, wp);
    cp_async16(st0 + 32, wp + 1);
  }
  cp_async_commit();
  __syncthreads();  // the candidate table

  float2 hv2[8];
  float hsum = 16.0f;  // sum of the lane's 16 h values (h = 1 without h)
  int cur_chunk = -1;
#pragma unroll
  for (int j = 0; j < 8; ++j) hv2[j] = make_float2(1.0f, 1.0f);

  int buf = 0;
  for (int64_t u = warp_global; u < units; u += warps_total, buf ^= 1) {
    // the copy of the warp's next unit starts now
    if (u + warps_total < units) {
      uint4* dst = buf ? st0 : st1;
      cp_async16(dst, wp + wstep);
      cp_async16(dst + 32, wp + wstep + 1);
    }
    cp_async_commit();

    if (h != nullptr && chunk != cur_chunk) {
      cur_chunk = chunk;
      load_h_slice(h, chunk, hv2, hsum);
    }

    cp_async_wait_1();  // this lane's copy of the current unit has landed
    const uint4* cur = buf ? st1 : st0;
    search_unit<kFourOverSix>(cur[0], cur[32], wp, go, chunk, hv2, hsum, w, h, tab, d, k, init_codes, down, up,
                              codes_out, packed_out);
    wp += wstep;
    go += ostep;
    chunk += chunk_step;
    if (chunk >= chunks) chunk -= chunks;
  }
}

// Units per batch of the work-shared search.
constexpr uint32_t kShareBatch = 2;

// The same search with the units shared out at run time.  The warp schedulers favour the
// warps of the CTAs that became resident first, so with a static deal those warps finish
// early and the last CTAs to arrive run on alone at the end of a long call (on a
// 28672 x 8192 matrix, k = 4, warps finished between 246 and 489 us).  Here warps take
// batches of kShareBatch units from a counter in global memory (*next, zero at launch), so
// the faster warps simply take more of them.  Batches run down the rows of one column chunk
// (unit v is row v % m of chunk v / m), so a warp's h slice mostly stays put.  The first
// batch of each warp is its index; the counter hands out the rest, one batch ahead, so the
// atomic's latency stays hidden.  Same per-group work and bytes as refine_linear_kernel.
template <bool kFourOverSix>
__global__ void __launch_bounds__(kRefineThreads, 7)
refine_shared_kernel(const uint4* __restrict__ w, const float* __restrict__ h, uint32_t m, uint32_t units,
                     int64_t row_words, int64_t ng, const float* __restrict__ global_scale,
                     const uint8_t* init_codes, int down, int up, uint8_t* codes_out,
                     uint2* __restrict__ packed_out, unsigned* __restrict__ next) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t warp_global = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;

  __shared__ float4 tab[128];
  __shared__ __align__(16) uint4 stage[kWarpsPerRefineBlock][2][64];
  const ScaleDomain d = make_scale_domain(*global_scale);
  const SearchConsts k = search_consts(d, kFourOverSix);
  for (int c = threadIdx.x; c < 128; c += blockDim.x) tab[c] = candidate_constants((uint32_t)c, d.sgk);

  // the current unit v = (row, chunk) and the end of its batch; lane 0 holds the index of
  // the warp's following batch
  uint32_t v = warp_global * kShareBatch;
  uint32_t vend = min(v + kShareBatch, units);
  uint32_t chunk = v < units ? v / m : 0, row = v - chunk * m;
  uint32_t batch_after = 0;
  if (lane == 0) batch_after = warps_total + atomicAdd(next, 1u);
  auto group_of = [&](uint32_t r, uint32_t c) { return w + (int64_t)r * row_words + (int64_t)c * 64 + 2 * lane; };
  uint4* const st0 = &stage[warp][0][lane];
  uint4* const st1 = &stage[warp][1][lane];
  if (v < units) {
    const uint4* s = group_of(row, chunk);
    cp_async16(st0, s);
    cp_async16(st0 + 32, s + 1);
  }
  cp_async_commit();
  __syncthreads();  // the candidate table

  float2 hv2[8];
  float hsum = 16.0f;
  uint32_t cur_chunk = 0xFFFFFFFFu;
#pragma unroll
  for (int j = 0; j < 8; ++j) hv2[j] = make_float2(1.0f, 1.0f);

  int buf = 0;
  while (v < units) {
    // the warp's next unit: the next row of this batch, else the first of the next batch;
    // its copy starts now
    uint32_t v2 = v + 1, row2 = row + 1, chunk2 = chunk;
    if (row2 == m) {
      row2 = 0;
      ++chunk2;
    }
    if (v2 >= vend) {
      const uint32_t b = __shfl_sync(0xFFFFFFFFu, batch_after, 0);
      if (lane == 0) batch_after = warps_total + atomicAdd(next, 1u);
      v2 = b < units / kShareBatch + 1 ? b * kShareBatch : units;
      vend = min(v2 + kShareBatch, units);
      if (v2 < units) {
        chunk2 = v2 / m;
        row2 = v2 - chunk2 * m;
      }
    }
    if (v2 < units) {
      uint4* dst = buf ? st0 : st1;
      const uint4* s = group_of(row2, chunk2);
      cp_async16(dst, s);
      cp_async16(dst + 32, s + 1);
    }
    cp_async_commit();

    if (h != nullptr && chunk != cur_chunk) {
      cur_chunk = chunk;
      load_h_slice(h, chunk, hv2, hsum);
    }

    cp_async_wait_1();  // this lane's copy of the current unit has landed
    const uint4* cur = buf ? st1 : st0;
    search_unit<kFourOverSix>(cur[0], cur[32], group_of(row, chunk), (int64_t)row * ng + (int64_t)chunk * 32 + lane,
                              chunk, hv2, hsum, w, h, tab, d, k, init_codes, down, up, codes_out, packed_out);
    v = v2;
    row = row2;
    chunk = chunk2;
    buf ^= 1;
  }
}

// Warps of refine_sm_kernel's CTA: 7 x 4, the search warps one SM holds at 72 registers.
constexpr int kSmWarps = 28;

// The search of a matrix alone on the GPU, one CTA per SM: the CTA takes an equal share
// of the (column-major) units and its warps share them out through a counter in shared
// memory, one unit at a time.  Warps of one CTA all became resident together, but the
// schedulers still favour some of them; here the favoured ones simply take more units, so
// every warp of the SM finishes within about one unit of the others.  The SMs' shares are
// equal, which suits a search that has the GPU to itself (refine_shared_kernel's global
// counter balances the SMs as well, for long searches).  Same per-group work and bytes as
// refine_linear_kernel.
template <bool kFourOverSix>
__global__ void __launch_bounds__(kSmWarps * 32, 1)
refine_sm_kernel(const uint4* __restrict__ w, const float* __restrict__ h, uint32_t m, uint32_t units,
                 int64_t row_words, int64_t ng, const float* __restrict__ global_scale,
                 const uint8_t* init_codes, int down, int up, uint8_t* codes_out,
                 uint2* __restrict__ packed_out) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  __shared__ float4 tab[128];
  __shared__ __align__(16) uint4 stage[kSmWarps][2][64];
  __shared__ unsigned next_unit;
  const ScaleDomain d = make_scale_domain(*global_scale);
  const SearchConsts k = search_consts(d, kFourOverSix);
  for (int c = threadIdx.x; c < 128; c += blockDim.x) tab[c] = candidate_constants((uint32_t)c, d.sgk);

  // this CTA's units [vbeg, vlim); unit v is row v % m of column chunk v / m
  const uint32_t vbeg = (uint32_t)(((uint64_t)units * blockIdx.x) / gridDim.x);
  const uint32_t vlim = (uint32_t)(((uint64_t)units * (blockIdx.x + 1)) / gridDim.x);
  if (threadIdx.x == 0) next_unit = vbeg + kSmWarps;  // the first kSmWarps units go to warps in order
  auto group_of = [&](uint32_t r, uint32_t c) { return w + (int64_t)r * row_words + (int64_t)c * 64 + 2 * lane; };
  uint4* const st0 = &stage[warp][0][lane];
  uint4* const st1 = &stage[warp][1][lane];
  uint32_t v = vbeg + warp;
  uint32_t chunk = v < vlim ? v / m : 0, row = v - chunk * m;
  if (v < vlim) {
    const uint4* s = group_of(row, chunk);
    cp_async16(st0, s);
    cp_async16(st0 + 32, s + 1);
  }
  cp_async_commit();
  __syncthreads();  // the candidate table and the counter

  float2 hv2[8];
  float hsum = 16.0f;
  uint32_t cur_chunk = 0xFFFFFFFFu;
#pragma unroll
  for (int j = 0; j < 8; ++j) hv2[j] = make_float2(1.0f, 1.0f);

  int buf = 0;
  while (v < vlim) {
    // the warp's next unit (counter values grow, so its chunk is at or after this one's;
    // a division only when it leaves this chunk); its copy starts now
    uint32_t v2 = 0;
    if (lane == 0) v2 = atomicAdd(&next_unit, 1u);
    v2 = __shfl_sync(0xFFFFFFFFu, v2, 0);
    uint32_t chunk2 = chunk, row2 = 0;
    if (v2 < vlim) {
      row2 = v2 - chunk * m;
      if (row2 >= m) {
        chunk2 = v2 / m;
        row2 = v2 - chunk2 * m;
      }
      uint4* dst = buf ? st0 : st1;
      const uint4* s = group_of(row2, chunk2);
      cp_async16(dst, s);
      cp_async16(dst + 32, s + 1);
    }
    cp_async_commit();

    if (h != nullptr && chunk != cur_chunk) {
      cur_chunk = chunk;
      load_h_slice(h, chunk, hv2, hsum);
    }

    cp_async_wait_1();  // this lane's copy of the current unit has landed
    const uint4* cur = buf ? st1 : st0;
    search_unit<kFourOverSix>(cur[0], cur[32], group_of(row, chunk), (int64_t)row * ng + (int64_t)chunk * 32 + lane,
                              chunk, hv2, hsum, w, h, tab, d, k, init_codes, down, up, codes_out, packed_out);
    v = v2;
    row = row2;
    chunk = chunk2;
    buf ^= 1;
  }
}

// ---------------------------------------------------------------- pack with given codes
__global__ void __launch_bounds__(256) pack_kernel(const uint4* __restrict__ w, int64_t groups,
                                                   const float* __restrict__ global_scale,
                                                   const uint8_t* __restrict__ codes,
                                                   uint2* __restrict__ packed_out) {
  const ScaleDomain d = make_scale_domain(*global_scale);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += stride) {
    Group G;
    load_group(w, g, d.pw, G);
    uint32_t c = codes[g] & 0x7Fu;
    c = c < 1 ? 1u : (c > kE4M3MaxCode ? kE4M3MaxCode : c);
    packed_out[g] = quantize_pack(G, c, __frcp_rn(__fmul_rn(e4m3_mag(c), d.sgk)), d.sgk, d.pw,
                                  reinterpret_cast<const uint16_t*>(w) + g * 16);
  }
}

// Resident CTAs per SM of a kernel, queried once per kernel and device (the query is
// not repeated under stream capture).
// ---------------------------------------------------------------- 4over6 init (Algorithm 2)
// Initial codes of Algorithm 2: for m = max|w| of the group, the E4M3 codes of m / (4 s_g)
// and m / (6 s_g) (each as in Eq. 7), and the one whose group has the smaller plain MSE;
// the anchor 4 (first in C = {4, 6}) wins an exact tie.
__global__ void __launch_bounds__(256) fourover6_codes_kernel(const uint4* __restrict__ w, int64_t groups,
                                                              const float* __restrict__ global_scale,
                                                              uint8_t* __restrict__ codes) {
  const ScaleDomain d = make_scale_domain(*global_scale);
  const float inv4 = anchor_inv_raw(d.sgk, 4.0f);
  const float inv6 = anchor_inv_raw(d.sgk, 6.0f);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += stride) {
    Group G;
    const uint4 p = ld_stream_v4(w + 2 * g), q = ld_stream_v4(w + 2 * g + 1);
    unpack_group(p, q, d.pw, G);
    const float amax_k = __fmul_rn(__uint_as_float(group_abs_max_bits(p, q) << 16), d.pw);
    const uint32_t c4 = anchored_code(amax_k, d.sgk, inv4, 2.0f);
    const uint32_t c6 = anchored_code(amax_k, d.sgk, inv6, 3.0f);
    uint32_t c = c4;
    if (c6 != c4 && exact_group_mse(G, c6, d.sgk) < exact_group_mse(G, c4, d.sgk)) c = c6;
    codes[g] = (uint8_t)c;
  }
}

// Resident blocks per SM of kKernel at `threads` threads, queried once per device (a race
// between threads only repeats the query: the cached value is the same either way).
// First the kernel is given the whole shared-memory carveout.  An SM keeps the split of
// its on-chip memory that its first resident CTA asked for, and the default split for
// these small-shared-memory kernels leaves no room for a Hessian CTA (68 KB) beside them,
// so a Hessian pass launched alongside a search would wait for the whole search (measured:
// a 4096-channel pass beside a 14336 x 4096 search took 0.29 ms instead of 0.20; the
// search itself is within 2 % either way, a 196 KB split gave the same times).
template <auto kKernel>
int occupancy_blocks(int threads) {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  int blocks = cache[dev].load(std::memory_order_relaxed);
  if (blocks == 0) {
    cudaFuncSetAttribute(kKernel, cudaFuncAttributePreferredSharedMemoryCarveout, (int)cudaSharedmemCarveoutMaxShared);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, kKernel, threads, 0) != cudaSuccess ||
        blocks < 1)
      blocks = 1;
    cache[dev].store(blocks, std::memory_order_relaxed);
  }
  return blocks;
}

}  // namespace

cudaError_t launch_amax(const void* w, int64_t count, uint32_t* amax_bits, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t nvec = count / 8;
  int64_t blocks = (nvec + 255) / 256;
  blocks = std::min<int64_t>(blocks, (int64_t)info.sm_count * occupancy_blocks<amax_kernel>(256));
  amax_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4*>(w), nvec, amax_bits);
  return cudaGetLastError();
}

cudaError_t launch_rtn_codes(const void* w, int64_t m, int64_t n, const uint32_t* amax_bits,
                             float* global_scale, uint8_t* codes, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t groups = m * (n / 16);
  int64_t blocks = codes ? (groups + 255) / 256 : 1;
  blocks = std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)info.sm_count * occupancy_blocks<rtn_codes_kernel>(256)));
  rtn_codes_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4*>(w), groups,
                                                          amax_bits, global_scale, codes);
  return cudaGetLastError();
}

cudaError_t launch_refine(const void* w, int64_t ld_w, const float* h, int64_t m, int64_t n,
                          const float* global_scale, const uint8_t* init_codes, int64_t ld_init, int down,
                          int up, uint8_t* codes_out, int64_t ld_codes, uint8_t* packed_out, int64_t ld_packed,
                          int ctas_per_sm, bool fourover6, unsigned* share_counter, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int ng = (int)(n / 16);
  const int64_t units = m * ((ng + 31) / 32);
  // contiguous W and outputs with whole row chunks: the pointer-walk kernel
  const bool linear = ld_w == n && ng % 32 == 0 && ld_codes == ng && (packed_out == nullptr || ld_packed == n / 2) &&
                      (init_codes == nullptr || ld_init == ng);
  int per_sm = linear ? (fourover6 ? occupancy_blocks<refine_linear_kernel<true>>(kRefineThreads)
                                   : occupancy_blocks<refine_linear_kernel<false>>(kRefineThreads))
                      : (fourover6 ? occupancy_blocks<refine_kernel<true>>(kRefineThreads)
                                   : occupancy_blocks<refine_kernel<false>>(kRefineThreads));
  if (ctas_per_sm > 0) per_sm = std::min(per_sm, ctas_per_sm);
  const int64_t resident = (int64_t)info.sm_count * per_sm;
  const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((units + kWarpsPerRefineBlock - 1) / kWarpsPerRefineBlock, resident));
  // Work sharing pays once a warp's static share is long (its spread in finishing times
  // grows with it): from about 512 units x candidates per warp on (measured on 1 GB300:
  // a 28672 x 8192 matrix gains 5 % at k = 4 and 12 % at k = 16, a 14336 x 4096 one nothing
  // at k = 4 and 7 % at k = 16, and 4096 x 4096 matrices lose to the counter's cost).
  const int64_t candidates = std::min(down + up + 1, (int)kE4M3MaxCode);
  if (linear && share_counter != nullptr && units < (int64_t(1) << 30) && m < (int64_t(1) << 30) &&
      units * candidates >= 512 * (resident * kWarpsPerRefineBlock)) {
    err = cudaMemsetAsync(share_counter, 0, sizeof(unsigned), stream);
    if (err != cudaSuccess) return err;
    auto sk = fourover6 ? refine_shared_kernel<true> : refine_shared_kernel<false>;
    const int64_t batches = (units + kShareBatch - 1) / kShareBatch;
    const int64_t sblocks =
        std::max<int64_t>(1, std::min<int64_t>((batches + kWarpsPerRefineBlock - 1) / kWarpsPerRefineBlock, resident));
    sk<<<(unsigned)sblocks, kRefineThreads, 0, stream>>>(static_cast<const uint4*>(w), h, (uint32_t)m,
                                                         (uint32_t)units, n / 8, ng, global_scale,
                                                         fourover6 ? nullptr : init_codes, down, up, codes_out,
                                                         reinterpret_cast<uint2*>(packed_out), share_counter);
    return cudaGetLastError();
  }
  // A search alone on the GPU with at least two units per warp: one CTA per SM sharing its
  // units out in shared memory (1 GB300, k = 4: 14336 x 4096 127.6 -> 115.4 us, 4096 x 4096
  // 41.6 -> 39.6 us; 1024 x 4096, one or two units per warp, keeps the static deal).
  if (linear && ctas_per_sm == 0 && units >= 2 * (int64_t)info.sm_count * kSmWarps && units < (int64_t(1) << 30) &&
      m < (int64_t(1) << 30)) {
    auto qk = fourover6 ? refine_sm_kernel<true> : refine_sm_kernel<false>;
    const int fits = fourover6 ? occupancy_blocks<refine_sm_kernel<true>>(kSmWarps * 32)
                               : occupancy_blocks<refine_sm_kernel<false>>(kSmWarps * 32);
    if (fits >= 1) {
      qk<<<(unsigned)info.sm_count, kSmWarps * 32, 0, stream>>>(static_cast<const uint4*>(w), h, (uint32_t)m,
                                                               (uint32_t)units, n / 8, ng, global_scale,
                                                               fourover6 ? nullptr : init_codes, down, up, codes_out,
                                                               reinterpret_cast<uint2*>(packed_out));
      return cudaGetLastError();
    }
  }
  if (linear) {
    auto lk = fourover6 ? refine_linear_kernel<true> : refine_linear_kernel<false>;
    lk<<<(unsigned)blocks, kRefineThreads, 0, stream>>>(static_cast<const uint4*>(w), h, units, (ng + 31) / 32,
                                                         global_scale, fourover6 ? nullptr : init_codes, down, up,
                                                         codes_out, reinterpret_cast<uint2*>(packed_out));
    return cudaGetLastError();
  }
  auto kernel = fourover6 ? refine_kernel<true> : refine_kernel<false>;
  kernel<<<(unsigned)blocks, kRefineThreads, 0, stream>>>(static_cast<const uint4*>(w), ld_w, h, m, ng, global_scale,
                                                          fourover6 ? nullptr : init_codes, ld_init, down, up,
                                                          codes_out, ld_codes, reinterpret_cast<uint2*>(packed_out),
                                                          ld_packed / 8);
  return cudaGetLastError();
}

cudaError_t launch_fourover6(const void* w, int64_t m, int64_t n, const float* global_scale,
                             uint8_t* codes, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t groups = m * (n / 16);
  int64_t blocks = (groups + 255) / 256;
  blocks = std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)info.sm_count * occupancy_blocks<fourover6_codes_kernel>(256)));
  fourover6_codes_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4*>(w), groups,
                                                                global_scale, codes);
  return cudaGetLastError();
}

cudaError_t launch_pack(const void* w, int64_t m, int64_t n, const float* global_scale,
                        const uint8_t* codes, uint8_t* packed_out, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t groups = m * (n / 16);
  int64_t blocks = (groups + 255) / 256;
  blocks = std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)info.sm_count * occupancy_blocks<pack_kernel>(256)));
  pack_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4*>(w), groups,
                                                     global_scale, codes,
                                                     reinterpret_cast<uint2*>(packed_out));
  return cudaGetLastError();
}

}  // namespace hscale
