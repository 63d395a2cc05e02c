/*
 * hscale.h -- C ABI of the GB300 (sm_103a) H-Scale hot path.
 *
 * H-Scale ("Hessian-Guided Scale Refinement for NVFP4 Sub-Byte LLM Inference")
 * picks each 16-element NVFP4 group's E4M3 local scale by a windowed search that
 * minimises a diagonal-Hessian weighted reconstruction error.  The data-parallel
 * hot path has two parts, both exposed here:
 *
 *   1. hscale_hessian_diag_accumulate   h_j += sum_t x_tj^2 over a token chunk
 *                                       (Sec. 3.2, Eq. 4: h = diag(X^T X));
 *                                       _ex: the same, overlapping the previous kernel
 *                                       when X is known to be complete
 *   2. hscale_rtn_scales                global scale s_g and the RTN local-scale codes
 *                                       (Sec. 3.3 "Initialization", Eq. 7)
 *      hscale_refine_scales             Algorithm 1: walk the E4M3 ladder around the
 *                                       initial code (Eqs. 8-10), quantize the group to
 *                                       E2M1 under each candidate (Eqs. 11-12), keep the
 *                                       code with the smallest sum_j h_j (w_j - s q_j)^2
 *                                       (Eqs. 6, 13), then re-quantize and pack
 *      hscale_refine_scales_ex          the same with a cap on resident CTAs per SM
 *      hscale_pack_nvfp4                final FP4 quantization with given codes
 *                                       (Sec. 3.3 "Final re-quantization", Eq. 2)
 *      hscale_fourover6_codes           the 4over6 initial codes of Algorithm 2, an
 *                                       alternative start for the refinement (Sec. 3.5)
 *      hscale_refine_scales_4over6      Algorithm 2 in one pass: those codes decided
 *                                       inside the search
 *      hscale_refine_scales_strided     the search on 2-D views (column blocks, slices)
 *      hscale_refine_scales_ws          the search with its units shared out at run time
 *                                       (a 16-byte workspace; same results)
 *      hscale_dequant_residual          dW = W - W_hat of the packed weights (Eqs. 1-3)
 *      hscale_output_error              ||X dW^T||_F^2 on the tensor cores (Eq. 3)
 *      hscale_hessian_full_accumulate   H += X^T X on the tensor cores (Algorithm 3)
 *      hscale_gptq_factor               damped inverse-Cholesky factor (Algorithm 3)
 *      hscale_gptq_hscale               GPTQ with H-Scale as local quantizer (Algorithm 3)
 *
 * Equation numbers count the paper's displayed equations in order (Eq. 1 is the
 * effective scale s = s_g * l).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All pointers except `stream` are DEVICE pointers owned by the caller; the
 *   library allocates and frees no memory (hscale_gptq_hscale keeps one stream and a
 *   few events per device context, see there).  Work is enqueued on `stream` (a
 *   cudaStream_t passed as void*, NULL = legacy default stream) and nothing
 *   synchronises: results are ready when the stream reaches them.
 * - Matrices are row-major.  W is [m, n] bfloat16 with contiguous rows; groups of 16
 *   run along n (the input-channel axis), so n must be a multiple of 16.
 * - Local-scale codes are E4M3 bytes in [1, 126] (the index iota of Algorithm 1 is
 *   the byte itself), stored [m, n/16] row-major, one byte per group.
 * - Packed FP4 is [m, n/2] bytes: element 2j of a row in the low nibble of byte j,
 *   element 2j+1 in the high nibble.  A nibble is sign<<3 | E2M1 magnitude code; the
 *   sign is the sign bit of w, also when the magnitude rounds to zero.
 * - The effective scale of a group is s_g * E4M3(code); dequantized weight =
 *   E2M1(nibble) * s_g * E4M3(code).
 * - Rounding is round-to-nearest-even on the exact real quotients w / (s_g * l) and
 *   amax_group / (6 s_g), decided exactly in the kernels; E2M1 saturates at 6, E4M3
 *   at 448.
 * - Inputs are assumed finite; NaN or Inf in W, X or h gives unspecified codes.
 *   s_g must be a positive normal fp32 number.
 * - Zero-sized inputs (m, n or tokens == 0) return HSCALE_OK and launch nothing.
 * - Every argument is checked before anything is enqueued; a failed check returns
 *   its status and enqueues nothing.  A launch failure returns HSCALE_ERR_CUDA
 *   (cudaGetLastError after the launch).  No C++ exception crosses the ABI.
 * - Results are deterministic: the same inputs on the same GPU model give the same
 *   bits on every run.
 */
#ifndef HSCALE_H
#define HSCALE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum hscale_status {
  HSCALE_OK = 0,
  HSCALE_ERR_NULL = 1,      /* a required pointer is NULL                            */
  HSCALE_ERR_SHAPE = 2,     /* negative size, n not a multiple of 16, ld < n, ...    */
  HSCALE_ERR_ALIGN = 3,     /* a pointer or leading dimension breaks the alignment   */
  HSCALE_ERR_ARG = 4,       /* an out-of-range scalar argument (window half-widths)  */
  HSCALE_ERR_CUDA = 5,      /* the CUDA runtime reported an error for a launch       */
  HSCALE_ERR_WORKSPACE = 6  /* workspace missing or smaller than the query says      */
} hscale_status;

/* Static, NUL-terminated description of a status code (unknown codes included). */
const char* hscale_status_string(int status);

/* ABI version of this header (incremented on any signature change). */
int hscale_abi_version(void);

/*
 * Device-side failure report.  Kernels never hang: every wait on an asynchronous copy
 * is bounded, and a wait that runs out sets a sticky flag on the current device (and
 * the affected h entries become NaN).  This call synchronises with the device, stores
 * the flags in *flags (0 = no failure; bit 0 = a bounded wait ran out) and clears them.
 */
int hscale_device_error_flags(uint32_t* flags);

/*
 * Self-test of that failure path (the paper has no counterpart): one CTA waits, at most
 * `polls` polls, on an mbarrier that nothing arrives on, so the wait runs out and sets
 * bit 0 of the device error flags the way a stalled copy pipeline would, without a fault
 * or a hang.  The kernel then ends normally and the context stays usable.
 */
int hscale_selftest_bounded_wait(uint32_t polls, void* stream);

/*
 * Hessian diagonal, one token chunk (Sec. 3.2, Eq. 4).
 *
 *   h[j] += sum_{t < tokens} x[t * ld_x + j]^2      for j < n
 *
 * x      [tokens, ld_x] bfloat16, 16-byte aligned; only the first n columns are read;
 *        tokens < 2^31.
 * h      [n] fp32, read and written (accumulated in place).  Zero it before the first
 *        chunk; streaming a calibration set is one call per chunk on the same h.
 * n      multiple of 8; ld_x >= n and a multiple of 8.
 * Arithmetic: x^2 is exact in fp32; the squares are summed on the tensor cores in fp32
 * over runs of 1024 tokens (their accumulation is measured low by about 0.9 units in the
 * last place per 16 tokens, so about 2^-18 relative per run at most), then the runs'
 * sums and a thread-block cluster's partial sums meet in fp32 round-to-nearest adds in
 * a fixed order.  Every run of a call gives the same bits.
 * Nothing else is touched: the call needs no workspace.  The call's kernel is launched
 * with programmatic dependent launch; it waits for the kernel before it on the stream
 * to finish (and for its writes to be visible) before it reads X, so X may be the output
 * of any earlier work on the stream, including a kernel that lets its dependents start
 * early.  hscale_hessian_diag_accumulate_ex lets a caller whose X is already complete
 * skip that wait.
 */
int hscale_hessian_diag_accumulate(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x,
                                   float* h, void* stream);

/*
 * hscale_hessian_diag_accumulate with flags (the paper has no counterpart: a scheduling
 * option of the library).  Same arguments, results and status codes, plus:
 *
 * flags  0, or HSCALE_HESSIAN_X_READY: the caller guarantees that X is complete, i.e.
 *        nothing that may still be running on the GPU when this call's kernel starts
 *        writes X (for instance calibration chunks resident in device memory, streamed
 *        by successive calls).  The kernel then starts streaming X while the previous
 *        kernel on the stream finishes, and waits for it only before it reads and
 *        updates h; successive chunk calls overlap.  Without the guarantee this flag can
 *        read stale or partly written X.  Other bits return HSCALE_ERR_ARG.
 */
#define HSCALE_HESSIAN_X_READY 1u
int hscale_hessian_diag_accumulate_ex(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x,
                                      float* h, uint32_t flags, void* stream);

/*
 * Rank-order sum of partial Hessian diagonals (Sec. 3.2, Eq. 4, with the calibration tokens
 * split across ranks: h = sum over the ranks' token shares of sum_t x_tj^2).  The paper has
 * no counterpart; it is the reduction step of a token-sharded calibration pass.
 *
 *   h[j] = (((p_0[j] + p_1[j]) + p_2[j]) + ...) + p_{parts-1}[j]      for j < n
 *
 * partials  [parts, ld] fp32 device array, row r = rank r's partial h (its own
 *           hscale_hessian_diag_accumulate calls into a zeroed vector); ld >= n.
 * h         [n] fp32, written (not accumulated).  The adds are fp32 round-to-nearest in rank
 *           order, so every rank that sums the same gathered partials gets the same bits,
 *           and repeated runs give the same bits; against one rank's pass over every token,
 *           the result differs only by the order of the additions (relative error of the
 *           same bound).
 * parts = 0 or n = 0 is a no-op.
 */
int hscale_hessian_sum_partials(const float* partials, int64_t parts, int64_t n, int64_t ld, float* h,
                                void* stream);

/*
 * The global amax of W as an integer word, for a global scale over a matrix whose rows are
 * split across ranks (the paper has no counterpart).  The global scale of Sec. 3.3 needs the
 * amax of the whole matrix: each rank computes the word of its rows, the ranks take the
 * maximum of the words (an all-reduce with MAX on a 32-bit integer), and
 * hscale_global_scale_from_amax turns the result into s_g.
 *
 * amax_bits  device uint32, written: the bf16 bit pattern of max|w| over the m x n bf16
 *            matrix w (16-byte aligned, n % 16 == 0), zero-extended; 0 for an empty or all-zero
 *            matrix.  Bit patterns of non-negative bf16 values order as the values do, so the
 *            maximum of the ranks' words is the word of the whole matrix.
 */
int hscale_amax_bits(const void* w_bf16, int64_t m, int64_t n, uint32_t* amax_bits, void* stream);

/*
 * s_g = fl32(amax / (6 * 448)) from an amax word of hscale_amax_bits (1.0 when it is 0):
 * the global scale hscale_rtn_scales writes for a matrix of that amax, bit for bit.
 * amax_bits and global_scale are device pointers (4-byte aligned).
 */
int hscale_global_scale_from_amax(const uint32_t* amax_bits, float* global_scale, void* stream);

/*
 * Global scale and RTN local-scale codes (Sec. 3.3 "Initialization", Eq. 7).
 *
 *   s_g      = fl32(amax|W| / (6 * 448))          (1.0 when W is all zero)
 *   codes[g] = max(1, RNE_E4M3_sat(amax_g / (6 s_g)))   for every group g
 *
 * w             [m, n] bfloat16, 16-byte aligned, n % 16 == 0.
 * global_scale  device fp32 scalar, written.
 * codes         [m, n/16] bytes, written; may be NULL to compute only s_g.
 * workspace     at least hscale_rtn_workspace_bytes() bytes of device memory, 4-byte
 *               aligned; its contents on entry do not matter (the call clears it on
 *               the stream before use).
 */
size_t hscale_rtn_workspace_bytes(void);
int hscale_rtn_scales(const void* w_bf16, int64_t m, int64_t n, float* global_scale,
                      uint8_t* codes, void* workspace, size_t workspace_bytes, void* stream);

/*
 * hscale_rtn_scales without a workspace and without any allocation.  (The paper has no
 * counterpart: this is a convenience of the library.)
 *
 * Same inputs, outputs and results as hscale_rtn_scales, for callers that cannot
 * allocate device memory, such as a plugin or callback that is handed only its input and
 * output tensors, or a service whose device memory belongs to a framework pool it cannot
 * reach.  The call allocates nothing (no cudaMalloc, no cudaFree, no allocating library
 * routine); its scratch is a fixed array of HSCALE_NOALLOC_SCRATCH_BYTES bytes compiled
 * into the library, which every GPU that loads the library holds until the process exits.
 *
 * - The first call on each device looks up that array's device address (a synchronous
 *   runtime query) and caches it with the id of the device's context; make that first
 *   call before any stream capture.  A call in a new context of the device (after
 *   cudaDeviceReset) looks the address up again, so it is then a first call too.
 * - Every call on a device shares the array: each call clears the part it uses on its
 *   stream before use, and calls whose work overlaps on the GPU (different streams,
 *   different threads) race with each other.  Serialise them.
 * - The scratch this work needs does not grow with m or n, so no input size is refused
 *   for lack of scratch; HSCALE_ERR_WORKSPACE would mean the work needs more than
 *   HSCALE_NOALLOC_SCRATCH_BYTES.
 */
#define HSCALE_NOALLOC_SCRATCH_BYTES 256
int hscale_rtn_scales_noalloc(const void* w_bf16, int64_t m, int64_t n, float* global_scale,
                              uint8_t* codes, void* stream);

/*
 * 4over6 initial codes (Algorithm 2, the part before HScaleGroupQuantize), to be refined
 * by hscale_refine_scales as its init_codes.
 *
 * For every group with m = max|w|, the anchors c in C = {4, 6} give the codes
 * max(1, RNE_E4M3_sat(m / (c s_g))) (each as in Eq. 7); the code whose group has the
 * smaller plain weight MSE sum_j (|w_j| - q_j s)^2 (exact E2M1 round-to-nearest-even
 * decisions) is written.  The anchor 4, first in C, wins an exact tie; errors within about
 * 1e-6 relative may be ordered either way (fp32 sums).
 *
 * w             [m, n] bfloat16, 16-byte aligned, n % 16 == 0.
 * global_scale  device fp32 scalar s_g (e.g. from hscale_rtn_scales with codes = NULL).
 * codes         [m, n/16] bytes, written.
 */
int hscale_fourover6_codes(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                           uint8_t* codes, void* stream);

/*
 * H-Scale refinement, Algorithm 1 (Eqs. 6-13), fused with the final re-quantization.
 *
 * For every group with initial code c (init_codes[g] with its sign bit cleared and
 * clamped to [1, 126]; or, when init_codes is NULL, the RTN code of Eq. 7 computed in
 * place), the candidates are the distinct codes clip(c + delta, 1, 126) for
 * delta = -down .. up; each candidate's error is sum_j h_j (|w_j| - s q_j)^2 with
 * s = s_g * E4M3(code) and q_j the E2M1 round-to-nearest-even of |w_j| / s.  The code
 * with the smallest error wins; exact ties keep the smaller |delta|, then the smaller
 * delta.  Codes whose errors differ by less than about 1e-6 relative may be ordered
 * either way (fp32 error sums).
 *
 * w             [m, n] bfloat16, 16-byte aligned, n % 16 == 0.
 * h             [n] fp32, 16-byte aligned; NULL means h = 1 (plain weight MSE search).
 * global_scale  device fp32 scalar s_g (e.g. from hscale_rtn_scales).
 * init_codes    [m, n/16] bytes or NULL.
 * down, up      window half-widths, 0 <= down, up <= 125 (the paper's default is
 *               down = 9, up = 6, i.e. K = 16 candidates).
 * codes_out     [m, n/16] bytes, written; may alias init_codes.
 * packed_out    [m, n/2] bytes, 8-byte aligned, written; may be NULL.
 */
int hscale_refine_scales(const void* w_bf16, const float* h, int64_t m, int64_t n,
                         const float* global_scale, const uint8_t* init_codes, int32_t down,
                         int32_t up, uint8_t* codes_out, uint8_t* packed_out, void* stream);

/*
 * hscale_refine_scales with an explicit launch shape; the results are identical.
 * The paper has no counterpart: this is a scheduling knob for callers that run the
 * search alongside another kernel (e.g. the next input space's Hessian pass on another
 * stream).  ctas_per_sm = 0 fills every SM as hscale_refine_scales does (a search with at
 * least two 32-group units per warp then runs as one CTA of 28 warps per SM whose warps
 * share its units at run time; a smaller one as up to 7 CTAs of 4 warps per SM); k > 0
 * keeps at most k of the search's CTAs (128 threads, 72 registers each) resident per SM,
 * leaving the rest of the register file to concurrent work.  Negative values return
 * HSCALE_ERR_ARG.
 */
int hscale_refine_scales_ex(const void* w_bf16, const float* h, int64_t m, int64_t n,
                            const float* global_scale, const uint8_t* init_codes, int32_t down,
                            int32_t up, uint8_t* codes_out, uint8_t* packed_out,
                            int32_t ctas_per_sm, void* stream);

/*
 * 4over6 + H-Scale, Algorithm 2 in one pass: the 4over6 initial codes are decided inside
 * the search, group by group, and the window is searched around them.
 *
 * The results equal hscale_fourover6_codes followed by hscale_refine_scales_ex with those
 * codes as init_codes, bit for bit, in one read of W and one launch, and with no
 * intermediate codes array.  The anchors are ordered by fast plain-MSE scores (the
 * hardware E2M1 conversion) whenever a margin test shows that the fast order is the exact
 * one; the few other groups take the exact comparison of hscale_fourover6_codes.
 *
 * Arguments as for hscale_refine_scales_ex without init_codes: w [m, n] bfloat16
 * (16-byte aligned, n % 16 == 0); h [n] fp32 (16-byte aligned) or NULL for h = 1;
 * global_scale a device fp32 scalar; 0 <= down, up <= 125; codes_out [m, n/16] bytes,
 * written; packed_out [m, n/2] bytes (8-byte aligned) or NULL; ctas_per_sm >= 0 (0 fills
 * every SM).  The same status codes as hscale_refine_scales_ex.
 */
int hscale_refine_scales_4over6(const void* w_bf16, const float* h, int64_t m, int64_t n,
                                const float* global_scale, int32_t down, int32_t up, uint8_t* codes_out,
                                uint8_t* packed_out, int32_t ctas_per_sm, void* stream);

/*
 * Bytes of device workspace hscale_refine_scales_ws takes: 16.
 */
size_t hscale_refine_workspace_bytes(void);

/*
 * hscale_refine_scales_ex (fourover6 = 0) or hscale_refine_scales_4over6 (fourover6 = 1)
 * with the units of long searches shared out at run time; the results are identical.
 * The paper has no counterpart: this is a schedule.  The GPU's warp schedulers favour the
 * warps that became resident first, so when every warp is dealt an equal share up front,
 * the late ones run on alone at the end of a long call; here warps take small batches of
 * units from a counter in `workspace` instead.  The library uses it when each warp would
 * otherwise get at least about 512 units x candidates (e.g. a 28672 x 8192 matrix at
 * k = 4, or a 14336 x 4096 one at k = 16); shorter searches take the static deal.
 *
 * w, h, m, n, global_scale, init_codes, down, up, codes_out, packed_out, ctas_per_sm as for
 * hscale_refine_scales_ex; fourover6 as for hscale_refine_scales_strided (0 or 1; 1 with
 * init_codes returns HSCALE_ERR_ARG).
 * workspace        device memory of at least hscale_refine_workspace_bytes() bytes,
 *                  16-byte aligned, owned by the caller; or NULL (no work sharing through
 *                  it).  When the call shares units through it, it zeroes the first 4 bytes
 *                  on `stream` before the kernel and the kernel counts in them, so calls
 *                  that may run at the same time on the GPU need distinct workspaces; a
 *                  short search leaves it untouched.  Nothing needs to persist between
 *                  calls.
 * workspace_bytes  its size; below hscale_refine_workspace_bytes() returns
 *                  HSCALE_ERR_WORKSPACE (a misaligned workspace returns HSCALE_ERR_ALIGN).
 * The other status codes are those of hscale_refine_scales_strided.
 */
int hscale_refine_scales_ws(const void* w_bf16, const float* h, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* init_codes, int32_t fourover6, int32_t down, int32_t up,
                            uint8_t* codes_out, uint8_t* packed_out, int32_t ctas_per_sm, void* workspace,
                            size_t workspace_bytes, void* stream);

/*
 * The search on 2-D views: hscale_refine_scales_ex / hscale_refine_scales_4over6 on a
 * block of columns (or rows) of larger arrays.  The paper has no counterpart: it lets a
 * caller search a column block of W as soon as h of those channels is final, while the
 * Hessian pass of the next block runs, or quantize one slice of a fused matrix.
 *
 * w             [m, n] bfloat16 view; row r starts at element r * ld_w.  w 16-byte
 *               aligned, ld_w >= n, ld_w % 8 == 0 (every row 16-byte aligned).
 * h             [n] fp32 of the view's columns, 16-byte aligned; NULL means h = 1.
 * global_scale  device fp32 scalar s_g (of the whole matrix the view belongs to).
 * init_codes    NULL, or [m, n/16] bytes with rows ld_init bytes apart, ld_init >= n/16
 *               (used only when fourover6 = 0; ld_init is ignored when it is NULL).
 * fourover6     0: initial codes from init_codes, or RTN (Eq. 7) when it is NULL;
 *               1: Algorithm 2's 4over6 codes decided in place (init_codes must be NULL).
 *               Other values and fourover6 = 1 with init_codes return HSCALE_ERR_ARG.
 * codes_out     [m, n/16] bytes with rows ld_codes bytes apart (ld_codes >= n/16), written.
 * packed_out    NULL, or [m, n/2] bytes with rows ld_packed bytes apart: 8-byte aligned,
 *               ld_packed >= n/2 and ld_packed % 8 == 0.
 * down, up, ctas_per_sm as for hscale_refine_scales_ex.
 *
 * Every group's result depends only on its 16 weights, its 16 h values, s_g and the
 * window, so a view gives exactly the bytes the whole-matrix call writes there.
 */
int hscale_refine_scales_strided(const void* w_bf16, int64_t ld_w, const float* h, int64_t m, int64_t n,
                                 const float* global_scale, const uint8_t* init_codes, int64_t ld_init,
                                 int32_t fourover6, int32_t down, int32_t up, uint8_t* codes_out,
                                 int64_t ld_codes, uint8_t* packed_out, int64_t ld_packed, int32_t ctas_per_sm,
                                 void* stream);

/*
 * Final FP4 quantization with given codes (Sec. 3.3 "Final re-quantization", Eq. 2):
 * packed nibble of w = sign(w) << 3 | RNE_E2M1_sat(|w| / (s_g * E4M3(code))).
 *
 * w             [m, n] bfloat16, 16-byte aligned, n % 16 == 0.
 * codes         [m, n/16] bytes; the sign bit is ignored and a code is read as
 *               clamp(code, 1, 126), the clip of Eq. 10.
 * packed_out    [m, n/2] bytes, 8-byte aligned, written.
 */
int hscale_pack_nvfp4(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                      const uint8_t* codes, uint8_t* packed_out, void* stream);

/*
 * Quantization residual dW = W - W_hat of packed NVFP4 weights (the dW of Eq. 3), for the
 * layer-output evaluation below.  W_hat = sign * s_g * E4M3(code) * E2M1(magnitude) per
 * nibble (Eqs. 1-2); dW is w - s_g * (l q) rounded once to fp32, then split into bf16
 * hi = RN(dW) and lo = RN(dW - hi), so hi + lo equals dW to a relative 2^-17.
 *
 * w          [m, n] bfloat16, 16-byte aligned, n % 16 == 0.
 * codes      [m, n/16] bytes (sign bit ignored, clamped to [1, 126] as in the pack).
 * packed     [m, n/2] bytes, 8-byte aligned (the layout hscale_refine_scales writes).
 * dw2        [m, ld_dw2] bfloat16, 16-byte aligned, written: with n_pad = 64 * ceil(n/64),
 *            columns [0, n) hold hi, [n_pad, n_pad + n) hold lo, and [n, n_pad) and
 *            [n_pad + n, 2 n_pad) are zero.  ld_dw2 >= 2 n_pad, ld_dw2 % 8 == 0.
 */
int hscale_dequant_residual(const void* w_bf16, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* codes, const uint8_t* packed, void* dw2_bf16, int64_t ld_dw2,
                            void* stream);

/*
 * Layer-output error of a quantization (Eq. 3): *out_sum += ||X dW^T||_F^2 over this chunk
 * of calibration tokens, computed on the tensor cores as C = X hi^T + X lo^T (bf16
 * operands, fp32 accumulation) with the sum of squares of C fused into the GEMM.  Tiles of
 * 128 tokens x 256 outputs each give one fp64 partial; the partials are added in a fixed
 * order, so the result is deterministic.
 *
 * x          [tokens, ld_x] bfloat16 row-major (first n columns used), 16-byte aligned,
 *            ld_x % 8 == 0, tokens < 2^31.
 * dw2        the [m, ld_dw2] output of hscale_dequant_residual for the same n.
 * out_sum    device fp64 scalar, accumulated (the caller zeroes it once).
 * workspace  device buffer of hscale_output_error_workspace_bytes(tokens, m) bytes.
 */
size_t hscale_output_error_workspace_bytes(int64_t tokens, int64_t m);
int hscale_output_error(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x, const void* dw2_bf16,
                        int64_t ld_dw2, int64_t m, double* out_sum, void* workspace, size_t workspace_bytes,
                        void* stream);

/*
 * GPTQ with H-Scale as its local quantizer (Algorithm 3), in three calls.
 *
 * 1. hscale_hessian_full_accumulate: H[n, n] (fp32, row stride ld_h) += X^T X over a chunk
 *    of calibration tokens, on the tensor cores (bf16 products, fp32 accumulation); its
 *    diagonal is the h of Eq. 4.  The tokens are taken in segments of 2048, each
 *    accumulated from zero and added into a running sum with fp32 round-to-nearest adds,
 *    and the sum is added into H: the error stays that of a 2048-token accumulation
 *    whatever the call size (|dH| <= 1e-5 sqrt(H_ii H_jj)), and a call over T tokens into
 *    a zeroed H equals successive 2048-token calls bit for bit.  Large calls are faster.  H is symmetric and only its upper triangle (j >= i) is
 *    accumulated and read later: 128 x 256 tiles wholly below the diagonal are not
 *    written, those crossing it are written in full.  x is [tokens, ld_x] bf16 row-major
 *    (2-byte aligned).  When x is 16-byte aligned and ld_x a multiple of 8 the tensor
 *    cores read X as it is (MN-major operand tiles) and the workspace may be NULL; other X
 *    is first transposed into the workspace (hscale_hessian_full_workspace_bytes, 256-byte
 *    aligned), which then must be given.
 *
 * 2. hscale_gptq_factor: the damped inverse-Cholesky factor, formed as GPTQ forms it.
 *    Only the upper triangle of H (j >= i) is read.  Channels with H_jj = 0 are dead (dead[j] = 1 if dead is not NULL; their weights are
 *    zeroed in step 3) and get H_jj = 1; the diagonal gets damp * mean(diag H) (GPTQ uses
 *    damp = 0.01); U [n, n] (fp32, row stride n) is upper triangular with
 *    U^T U = (H + damp I)^-1, formed from the Cholesky factor of the reversed matrix and
 *    its triangular inverse (no explicit inverse of H), by the library's own kernels: a
 *    blocked Cholesky in 128-wide block columns with the triangular inverse built in the same
 *    sweep, the diagonal blocks on CUDA cores and the trailing updates on the tensor cores
 *    with fp32-level accuracy (three-way bf16 splits).  info is a device int32[3]: info[0] the
 *    status of the factorization (0 = success; > 0: a pivot was not positive, the damped
 *    matrix is not positive definite, and U is unspecified), info[1] = info[2] = 0.  The
 *    workspace (hscale_gptq_factor_workspace_bytes, 256-byte aligned) holds the reversed
 *    matrix and the inverse side by side (2 n_pad^2 floats, n_pad = 128 ceil(n / 128)) and
 *    the split operands of the updates.  U is written only at the end of the call.
 *    n <= 65536.
 *
 * 3. hscale_gptq_hscale: for each block of `block` columns (a multiple of 16 dividing n)
 *    of the running fp32 weights (W with dead columns zeroed): the RTN codes of Eq. 7 of
 *    the current block weights, the H-Scale search over the window (down, up) with the
 *    diagonal proxy h [n] (16-byte aligned) and the global scale s_g of the original W
 *    (U as written by hscale_gptq_factor, 16-byte aligned),
 *    with exact E2M1 decisions and the tie rule of hscale_refine_scales; then
 *    E = (W_b - W_hat_b) / diag(U_b) and W[:, i+B:] -= E U[i:i+B, i+B:] with fp32-level
 *    accuracy (on the tensor cores: three-way bf16 splits of E and U, the six products
 *    above 2^-24 relative, fp32 accumulation).  Writes codes_out [m, n/16] and packed_out
 *    [m, n/2] (8-byte aligned) as hscale_refine_scales does.  The workspace
 *    (hscale_gptq_workspace_bytes) holds the running weights and two buffers of each
 *    split operand.  With more than one block the call works ahead: the update of the
 *    next block's columns runs on `stream` and the rest of each update on a second stream
 *    of the library, alongside the next block's quantization; events order the two, every
 *    weight receives its updates in block order (the same bits on every run), and the
 *    call's work on `stream` ends after all of it.  The library creates that stream and
 *    its events on the first such call in each device context and keeps them; a first
 *    call made while `stream` is being captured (which may not create them) runs every
 *    block on `stream` instead, with the same results.  Calls are enqueued one at a time.
 */
size_t hscale_hessian_full_workspace_bytes(int64_t tokens, int64_t n);
int hscale_hessian_full_accumulate(const void* x_bf16, int64_t tokens, int64_t n, int64_t ld_x, float* H,
                                   int64_t ld_h, void* workspace, size_t workspace_bytes, void* stream);
size_t hscale_gptq_factor_workspace_bytes(int64_t n);
int hscale_gptq_factor(const float* H, int64_t n, int64_t ld_h, float damp, float* U, uint8_t* dead,
                       int32_t* info, void* workspace, size_t workspace_bytes, void* stream);
size_t hscale_gptq_workspace_bytes(int64_t m, int64_t n, int32_t block);
int hscale_gptq_hscale(const void* w_bf16, int64_t m, int64_t n, const float* U, const float* h,
                       const float* global_scale, const uint8_t* dead, int32_t block, int32_t down, int32_t up,
                       uint8_t* codes_out, uint8_t* packed_out, void* workspace, size_t workspace_bytes,
                       void* stream);

#ifdef __cplusplus
}
#endif

#endif /* HSCALE_H */
