// factor.cu -- the damped inverse-Cholesky factor of GPTQ (Algorithm 3) on sm_103a.
//
// U is upper triangular with U^T U = A^-1 for the damped Hessian A = H + damp * mean(diag H) I
// (dead channels, H_jj = 0, get H_jj = 1 first).  With J the order-reversing permutation and
// B = J A J = L L^T (L lower, Cholesky), A = (J L J)(J L^T J), so U = (J L J)^-1 = J L^-1 J:
// upper triangular with a positive diagonal, hence the Cholesky factor of A^-1.  No inverse of
// A is formed.
//
// B is padded to n_pad = 128 * ceil(n / 128) with an identity block, whose factor and inverse
// are the identity.  B (then L, lower) and X (R, then X = L^-1, lower) sit side by side in one
// [n_pad, 2 n_pad] buffer, so that the two updates of a step are one GEMM over contiguous
// columns.  The sweep takes 128-wide block columns j = 0, 1, ...  (right-looking):
//   diag     the CTA of factor_diag_kernel factors the (updated) diagonal block,
//            B_jj = L_jj L_jj^T, in shared memory and inverts it, Z_jj = L_jj^-1, into the
//            inverse's diagonal block (32-wide tiles: one warp factors and inverts each 32 x 32
//            tile on the diagonal, the CTA's warps update the other tiles);
//   strips   panel L_ij = B_ij Z_jj^T (i > j) and the inverse's row X_j,c = Z_jj R_j,c (c < j),
//            in 64-wide strips on CUDA cores (factor_strip_kernel);
//   updates  B_ik -= L_ij L_kj^T over the trailing square, and R_ic -= L_ij X_jc for i > j,
//            c <= j: for the rows below the diagonal block, the columns from the trailing
//            square's first to the inverse's block j are contiguous in the buffer, n_pad of
//            them, and both updates are one product -L_:j [L_:j ; X_j,:]^T.  It runs on the
//            tensor cores: the tcgen05 GEMM with three-way bf16 splits of both operands (the
//            six products above 2^-24 relative, one GEMM over K = 6 * 128), which carries
//            fp32-level accuracy.
// X = L^-1 is built alongside: row blocks below the diagonal accumulate
// R_ic = -sum_k L_ik X_kc as the sweep passes, and X_ic = Z_ii R_ic once row block i is reached.
// A last kernel writes U_ij = X_{n-1-i, n-1-j}.
//
// A pivot that is not positive (the damped matrix is then not positive definite) is recorded
// in info[0] as its 1-based order in B and replaced by 1, so the sweep ends with finite values;
// U is then unspecified.
#include <cuda_bf16.h>

#include <algorithm>

#include "hscale_internal.h"
#include "tma.cuh"

namespace hscale {
namespace {

constexpr int kNb = 128;                  // block of the sweep
constexpr int kSub = 32;                  // sub-block of the diagonal factor (one warp)
constexpr int kLd = kNb + 4;              // padded shared-memory row (16-byte multiple)
constexpr int kDiagThreads = 512;
constexpr int kDiagSmemBytes = (2 * kNb * kLd + kSub * kLd + 4 * kSub) * 4;
constexpr int kStripRows = 32;            // rows (or columns) of one strip
constexpr int kStripThreads = 256;
constexpr int kStripSmemBytes = (kNb * (kNb + 4) + kNb * (kStripRows + 4)) * 4;
constexpr int kSplitK = 6 * kNb;          // K of the split update GEMMs

// ---------------------------------------------------------------- set-up
// One block: dead channels (H_jj = 0) and the damped diagonal dd_j = d_j + damp * mean(d),
// d_j = H_jj, or 1 for a dead channel (fp32; the mean in fp64).
__global__ void __launch_bounds__(1024) damp_diagonal_kernel(const float* __restrict__ H, int64_t n, int64_t ld_h,
                                                             float damp, uint8_t* __restrict__ dead,
                                                             float* __restrict__ dd) {
  __shared__ double part[1024];
  double s = 0.0;
#pragma unroll 4
  for (int64_t j = threadIdx.x; j < n; j += blockDim.x) {
    float d = H[j * ld_h + j];
    const bool is_dead = (d == 0.0f);
    if (is_dead) d = 1.0f;
    if (dead) dead[j] = (uint8_t)is_dead;
    dd[j] = d;
    s += (double)d;
  }
  part[threadIdx.x] = s;
  __syncthreads();
  for (int step = 512; step > 0; step >>= 1) {
    if ((int)threadIdx.x < step) part[threadIdx.x] += part[threadIdx.x + step];
    __syncthreads();
  }
  const float add = (float)((double)damp * part[0] / (double)n);
  for (int64_t j = threadIdx.x; j < n; j += blockDim.x) dd[j] = dd[j] + add;
}

// W2 [n_pad, 2 n_pad]: the left half B_ij = A_{n-1-i, n-1-j} for i, j < n, A the damped H
// (read from H's upper triangle, row stride ld_h, and the damped diagonal dd), the identity
// beyond n; the right half (X) zero where the sweep accumulates into it, strictly below the
// 128-block diagonal (nothing reads X above it).  One 32 x 32 tile of each half per block.
// Every read and write runs along a row: a tile of B below the diagonal reads H's rows
// (reversed), a tile above it reads the mirrored tile of H and transposes it in shared
// memory, and a tile on the diagonal reads the entries on and below it and takes the rest
// from its own transpose.
__global__ void __launch_bounds__(256) reverse_pad_kernel(const float* __restrict__ H, int64_t n, int64_t ld_h,
                                                          const float* __restrict__ dd, int64_t n_pad,
                                                          float* __restrict__ W2) {
  __shared__ float t[32][33];
  const int bi = (int)blockIdx.y, bj = (int)blockIdx.x;
  const int64_t i0 = 32 * (int64_t)bi, j0 = 32 * (int64_t)bj, ld = 2 * n_pad;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  if (bi < bj) {
    // B_ij = A_{n-1-j, n-1-i}: t[jj][ii]
    for (int jj = ty; jj < 32; jj += 8) {
      const int64_t j = j0 + jj, i = i0 + tx;
      t[jj][tx] = (i < n && j < n) ? H[(n - 1 - j) * ld_h + (n - 1 - i)] : 0.0f;
    }
    __syncthreads();
    for (int ii = ty; ii < 32; ii += 8) W2[(i0 + ii) * ld + j0 + tx] = t[tx][ii];  // i < j: 0 beyond n
  } else {
    // B_ij = A_{n-1-i, n-1-j} for i >= j: t[ii][jj]
    for (int ii = ty; ii < 32; ii += 8) {
      const int64_t i = i0 + ii, j = j0 + tx;
      t[ii][tx] = (i < n && j < n && i >= j) ? H[(n - 1 - i) * ld_h + (n - 1 - j)] : 0.0f;
    }
    __syncthreads();
    for (int ii = ty; ii < 32; ii += 8) {
      const int64_t i = i0 + ii, j = j0 + tx;
      float v;
      if (i < n && j < n)
        v = i == j ? dd[n - 1 - i] : (i > j ? t[ii][tx] : t[tx][ii]);
      else
        v = i == j ? 1.0f : 0.0f;
      W2[i * ld + j] = v;
    }
  }
  if (bi / (kNb / 32) > bj / (kNb / 32))
    for (int ii = ty; ii < 32; ii += 8) W2[(i0 + ii) * ld + n_pad + j0 + tx] = 0.0f;
}

// U_ij = X_{n-1-i, n-1-j} for j >= i, 0 below the diagonal (U row stride n; X row stride ld);
// rows i = blockIdx.y, + gridDim.y, ...
__global__ void __launch_bounds__(256) reverse_out_kernel(const float* __restrict__ Xw, int64_t ld, int64_t n,
                                                          float* __restrict__ U) {
  const int64_t j = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (j >= n) return;
#pragma unroll 4
  for (int64_t i = blockIdx.y; i < n; i += gridDim.y) U[i * n + j] = j >= i ? Xw[(n - 1 - i) * ld + (n - 1 - j)] : 0.0f;
}

// ---------------------------------------------------------------- diagonal block
__device__ __forceinline__ void record_failure(int32_t* info, int32_t order) {
  atomicCAS(reinterpret_cast<int*>(info), 0, order);
}

__device__ __forceinline__ float rsqrt_approx(float x) {
  float r;
  asm("rsqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// One warp factors the 32 x 32 block at A (row stride kLd, lower triangle) in place,
// A = L L^T, and writes Z = L^-1 (lower, zeros above) at Zo (row stride kLd); col is a 128-float scratch (two 64-float buffers).  Lane i holds row i of
// the block in registers (every loop has a constant trip count and every register index is a
// constant, so the row stays in registers; kept out of line: inlined into the block kernel,
// the compiler moves the row to local memory).  Two columns are eliminated per step: the
// 2 x 2 pivot block gives L_jj, L_j+1,j and L_j+1,j+1, every lane scales its two entries, the
// pairs (L_kj, L_k,j+1) go to shared memory and come back four rows per 16-byte broadcast
// load, and each lane updates its row.  Entries above the diagonal are updated too
// (harmlessly) and zeroed at the end.  The square roots come from the approximate hardware
// instruction (relative error about 2^-22), which keeps the serial chain of pivots short.
// The inverse is built in the same sweep: lane c also holds column c of Z, as partial sums
// s_i = delta_ic - sum_{m < j} L_im Z_mc over the rows not yet final.  When columns j and
// j + 1 of L are known, Z_jc = s_j / L_jj and Z_j+1,c = (s_j+1 - L_j+1,j Z_jc) / L_j+1,j+1
// (forward substitution), and the later rows take s_k -= L_kj Z_jc + L_k,j+1 Z_j+1,c with
// the same broadcast loads as the factor's update, so no second serial pass is needed.
// Each step updates the next pivot pair's two rows first and computes that pair's pivots
// before the rest of its update, so the serial chain of the next step can run alongside this
// step's bulk of independent FMAs; the pivot columns alternate between the two scratch
// buffers, so one __syncwarp per step orders them.  A pivot that is not positive is kept in a
// register (the first one) and recorded once at the end, so no step branches.  Every value
// takes the same operations in the same order as a plain right-looking sweep.

// The pivot pair (j, j + 1) from the current rows (the 2 x 2 block comes from lanes j and
// j + 1): this lane's entries v0 = L_lane,j and v1 = L_lane,j+1 (zero above the diagonal),
// rows j and j + 1 of Z in this lane's column (1 / L_jj = ra, 1 / L_j+1,j+1 = rc), all four
// written back into r and z.
__device__ __forceinline__ void pivot_pair(float (&r)[kSub], float (&z)[kSub], const int j, int lane,
                                           int32_t base, int32_t& fail, float& v0, float& v1, float& zj,
                                           float& zj1) {
  const unsigned full = 0xFFFFFFFFu;
  float a = __shfl_sync(full, r[j], j);
  const float b = __shfl_sync(full, r[j], j + 1);
  const float c = __shfl_sync(full, r[j + 1], j + 1);
  const bool bad_a = !(a > 0.0f);
  fail = (fail == 0 && bad_a) ? base + j + 1 : fail;
  a = bad_a ? 1.0f : a;
  const float ra = rsqrt_approx(a);
  const float l00 = __fmul_rn(a, ra), l10 = __fmul_rn(b, ra);
  float c2 = __fmaf_rn(-l10, l10, c);
  const bool bad_c = !(c2 > 0.0f);
  fail = (fail == 0 && bad_c) ? base + j + 2 : fail;
  c2 = bad_c ? 1.0f : c2;
  const float rc = rsqrt_approx(c2);
  const float l11 = __fmul_rn(c2, rc);
  const float x0 = __fmul_rn(r[j], ra);
  const float x1 = __fmul_rn(__fmaf_rn(-x0, l10, r[j + 1]), rc);
  v0 = lane == j ? l00 : (lane == j + 1 ? l10 : (lane > j + 1 ? x0 : 0.0f));
  v1 = lane == j + 1 ? l11 : (lane > j + 1 ? x1 : 0.0f);
  r[j] = v0;
  r[j + 1] = v1;
  zj = __fmul_rn(z[j], ra);
  zj1 = __fmul_rn(__fmaf_rn(-l10, zj, z[j + 1]), rc);
  z[j] = zj;
  z[j + 1] = zj1;
}

// Rows k and k + 1 of this lane's row and Z column take the pivot pair's update; cb holds
// the pairs (L_kj, L_k,j+1) of every row.
__device__ __forceinline__ void update_pair(float (&r)[kSub], float (&z)[kSub], const int k, const float* cb,
                                            float v0, float v1, float zj, float zj1) {
  const float4 q = *reinterpret_cast<const float4*>(cb + 2 * k);  // (L_kj, L_k,j+1, L_k+1,j, L_k+1,j+1)
  r[k] = __fmaf_rn(-v0, q.x, __fmaf_rn(-v1, q.y, r[k]));
  r[k + 1] = __fmaf_rn(-v0, q.z, __fmaf_rn(-v1, q.w, r[k + 1]));
  z[k] = __fmaf_rn(-q.x, zj, __fmaf_rn(-q.y, zj1, z[k]));
  z[k + 1] = __fmaf_rn(-q.z, zj, __fmaf_rn(-q.w, zj1, z[k + 1]));
}

__device__ __noinline__ void factor_sub32(float* A, float* Zo, float* col, int lane, int32_t* info,
                                          int32_t base) {
  float r[kSub], z[kSub];
#pragma unroll
  for (int k = 0; k < kSub; k += 4) {
    const float4 a = *reinterpret_cast<const float4*>(A + lane * kLd + k);
    r[k] = a.x;
    r[k + 1] = a.y;
    r[k + 2] = a.z;
    r[k + 3] = a.w;
  }
#pragma unroll
  for (int k = 0; k < kSub; ++k) z[k] = k == lane ? 1.0f : 0.0f;
  int32_t fail = 0;
  float v0, v1, zj, zj1;
  pivot_pair(r, z, 0, lane, base, fail, v0, v1, zj, zj1);
#pragma unroll
  for (int j = 0; j + 2 < kSub; j += 2) {
    float* cb = col + ((j >> 1) & 1) * (2 * kSub);
    reinterpret_cast<float2*>(cb)[lane] = make_float2(v0, v1);
    __syncwarp();
    update_pair(r, z, j + 2, cb, v0, v1, zj, zj1);
    float n0, n1, nz0, nz1;
    pivot_pair(r, z, j + 2, lane, base, fail, n0, n1, nz0, nz1);
#pragma unroll
    for (int k = j + 4; k < kSub; k += 2) update_pair(r, z, k, cb, v0, v1, zj, zj1);
    v0 = n0;
    v1 = n1;
    zj = nz0;
    zj1 = nz1;
  }
  if (fail != 0 && lane == 0) record_failure(info, fail);
#pragma unroll
  for (int k = 0; k < kSub; k += 4)
    *reinterpret_cast<float4*>(A + lane * kLd + k) =
        make_float4(k <= lane ? r[k] : 0.0f, k + 1 <= lane ? r[k + 1] : 0.0f, k + 2 <= lane ? r[k + 2] : 0.0f,
                    k + 3 <= lane ? r[k + 3] : 0.0f);
  // lane c holds column c of Z: row i is zero above the diagonal (i < c)
#pragma unroll
  for (int i = 0; i < kSub; ++i) Zo[i * kLd + lane] = i >= lane ? z[i] : 0.0f;
}

// Warp-tile products on 32 x 32 tiles in shared memory (row stride kLd = 4 mod 32 words, a
// multiple of 4).  A warp computes 16 rows of the output tile: lane (h = lane / 16,
// cl = lane % 16) holds rows h + 2 r (r < 8) and columns cl, cl + 16 in acc[r][0..1]
// (independent accumulators).  Per four m, A's rows are read as 16-byte words (two rows per
// warp, four banks apart: one wavefront), and B either row by row (kNT false: B[m][c] at
// B + m kLd + c; consecutive lanes, consecutive words) or, for a transposed operand, in place
// from its rows (kNT true: B[m][c] at B + c kLd + m; lanes cl read rows cl and cl + 16 as
// 16-byte words, four banks apart: two wavefronts each), so no transposed copy is needed.
//   acc[r][q] += sum_m A[h + 2 r][m] B[m][cl + 16 q]   (-= with kNeg), over m in order
template <bool kNT, bool kNeg = false>
__device__ __forceinline__ void tile_mma(float (&acc)[8][2], const float* A, const float* B, int lane) {
  const int h = lane >> 4, cl = lane & 15;
#pragma unroll 2
  for (int m = 0; m < kSub; m += 4) {
    float b[4][2];
    if (kNT) {
      const float4 u = *reinterpret_cast<const float4*>(B + cl * kLd + m);
      const float4 v = *reinterpret_cast<const float4*>(B + (cl + 16) * kLd + m);
      b[0][0] = u.x; b[1][0] = u.y; b[2][0] = u.z; b[3][0] = u.w;
      b[0][1] = v.x; b[1][1] = v.y; b[2][1] = v.z; b[3][1] = v.w;
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        b[q][0] = B[(m + q) * kLd + cl];
        b[q][1] = B[(m + q) * kLd + cl + 16];
      }
    }
    if (kNeg) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        b[q][0] = -b[q][0];
        b[q][1] = -b[q][1];
      }
    }
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const float4 a = *reinterpret_cast<const float4*>(A + (h + 2 * r) * kLd + m);
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        acc[r][q] = __fmaf_rn(a.x, b[0][q], acc[r][q]);
        acc[r][q] = __fmaf_rn(a.y, b[1][q], acc[r][q]);
        acc[r][q] = __fmaf_rn(a.z, b[2][q], acc[r][q]);
        acc[r][q] = __fmaf_rn(a.w, b[3][q], acc[r][q]);
      }
    }
  }
}
__device__ __forceinline__ void tile_zero(float (&acc)[8][2]) {
#pragma unroll
  for (int r = 0; r < 8; ++r) acc[r][0] = acc[r][1] = 0.0f;
}
__device__ __forceinline__ void tile_load(float (&acc)[8][2], const float* T, int lane) {
  const int h = lane >> 4, cl = lane & 15;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    acc[r][0] = T[(h + 2 * r) * kLd + cl];
    acc[r][1] = T[(h + 2 * r) * kLd + cl + 16];
  }
}
__device__ __forceinline__ void tile_store(const float (&acc)[8][2], float* T, int lane, float sign) {
  const int h = lane >> 4, cl = lane & 15;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    T[(h + 2 * r) * kLd + cl] = sign * acc[r][0];
    T[(h + 2 * r) * kLd + cl + 16] = sign * acc[r][1];
  }
}

constexpr int kHalf = kSub / 2;           // rows of a tile per warp (two warps per tile)

// Factor the 128 x 128 diagonal block at (j0, j0) of Bw and invert the factor: Z_jj = L_jj^-1
// into Xw's diagonal block (zeros above the diagonal).  The block is a 4 x 4 grid of 32 x 32
// tiles, taken in tile columns p = 0..3:
//   (a) warp 0 factors the tile on the diagonal and inverts it (factor_sub32);
//   (b) the tiles below it: L_ip = B_ip Z_p^T, two warps per tile;
//   (c) the tiles of the rest of the block: B_ik -= L_ip L_kp^T, two warps per tile (at most
//       six tiles: one round of the sixteen warps).
// Z_p^T and L_kp^T are read in place (the transposed form of the tile product).  The inverse
// of the block is built by tile rows q = 1..3, X_qr = -Z_q T_qr with
// T_qr = sum_{m=r}^{q-1} L_qm X_mr (r < q), on six warps while warp 0 runs (a): T_qr needs
// only the tile columns m < q, and X_qr only Z_q besides, so during (a) of step p they form
// row p - 1 (its X) and then row p (its T); row 3's X follows the sweep.  Those six warps
// (2, 3, 6, 7, 10, 11) sit on the two schedulers that warp 0 does not use: sharing warp 0's
// scheduler, they slowed its serial sweep (n = 4096: 1.69 against 1.65 ms).
__global__ void __launch_bounds__(kDiagThreads, 1)
factor_diag_kernel(const float* __restrict__ Bw, int64_t ld, int64_t j0, float* __restrict__ Xw,
                   int32_t* __restrict__ info) {
  extern __shared__ __align__(16) float sm[];
  float* S = sm;                 // [128][kLd] the block, then L (lower)
  float* X = S + kNb * kLd;      // [128][kLd] the inverse (lower)
  float* T = X + kNb * kLd;      // [32][kLd] the T tiles of the inverse's current row
  float* col = T + kSub * kLd;   // [128] the pivot columns of factor_sub32
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int h0 = kHalf * (warp & 1);  // the first of a warp's 16 rows within its tile
  const int pair = warp >> 1;         // which tile a warp works on (of up to eight at a time)

  // programmatic dependent launch: the strips may be scheduled now; the previous step's update
  // must have finished before the block is read
  pdl_launch_dependents();
  pdl_wait_primary();
  const float* blk = Bw + j0 * ld + j0;
  // independent 16-byte loads per thread in flight
#pragma unroll 4
  for (int t = 0; t < kNb * kNb / 4 / kDiagThreads; ++t) {
    const int e = tid + t * kDiagThreads;
    const int r = e >> 5, c = (e & 31) * 4;
    *reinterpret_cast<float4*>(S + r * kLd + c) = *reinterpret_cast<const float4*>(blk + r * ld + c);
    *reinterpret_cast<float4*>(X + r * kLd + c) = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  __syncthreads();

  for (int p = 0; p < kNb / kSub; ++p) {
    const int c0 = p * kSub;
    if (warp == 0) {
      factor_sub32(S + c0 * kLd + c0, X + c0 * kLd + c0, col, lane, info, (int32_t)(j0 + c0));
    } else if ((warp & 2) != 0 && warp < 12 && p >= 1) {
      // warps 2, 3, 6, 7, 10, 11: the schedulers that warp 0 does not use
      const int u = warp >> 2;        // the tile column r = u of the inverse's row
      if (p >= 2) {
        // X_qr = -Z_q T_qr for q = p - 1
        const int q0 = (p - 1) * kSub;
        if (u < p - 1) {
          float acc[8][2];
          tile_zero(acc);
          tile_mma<false>(acc, X + (q0 + h0) * kLd + q0, T + u * kSub, lane);
          tile_store(acc, X + (q0 + h0) * kLd + u * kSub, lane, -1.0f);
        }
        asm volatile("bar.sync 1, 192;" ::: "memory");  // these six warps: X_q done, T tiles free
      }
      // T_pr = sum_{m=r}^{p-1} L_pm X_mr
      if (u < p) {
        float acc[8][2];
        tile_zero(acc);
        for (int m = u; m < p; ++m)
          tile_mma<false>(acc, S + (c0 + h0) * kLd + m * kSub, X + m * kSub * kLd + u * kSub, lane);
        tile_store(acc, T + h0 * kLd + u * kSub, lane, 1.0f);
      }
    }
    __syncthreads();
    // (b) tiles below: L_ip = B_ip Z_p^T
    const int below = kNb / kSub - 1 - p;
    if (below == 0) break;
    if (pair < below) {
      const int r0 = c0 + kSub * (1 + pair) + h0;  // this warp's first row
      float acc[8][2];
      tile_zero(acc);
      tile_mma<true>(acc, S + r0 * kLd + c0, X + c0 * kLd + c0, lane);
      __syncwarp();
      tile_store(acc, S + r0 * kLd + c0, lane, 1.0f);
    }
    __syncthreads();
    // (c) tiles (i, k), p < k <= i: B_ik -= L_ip L_kp^T
    {
      int t = pair, i = p + 1;
      while (i < kNb / kSub && t > i - (p + 1)) {
        t -= i - p;
        ++i;
      }
      if (i < kNb / kSub) {
        const int k0 = (p + 1 + t) * kSub, r0 = i * kSub + h0;
        float acc[8][2];
        tile_load(acc, S + r0 * kLd + k0, lane);
        tile_mma<true, true>(acc, S + r0 * kLd + c0, S + k0 * kLd + c0, lane);
        tile_store(acc, S + r0 * kLd + k0, lane, 1.0f);
      }
    }
    __syncthreads();
  }

  // the inverse's last tile row: X_3r = -Z_3 T_3r
  if (pair < kNb / kSub - 1) {
    const int q0 = kNb - kSub;
    float acc[8][2];
    tile_zero(acc);
    tile_mma<false>(acc, X + (q0 + h0) * kLd + q0, T + pair * kSub, lane);
    tile_store(acc, X + (q0 + h0) * kLd + pair * kSub, lane, -1.0f);
  }
  __syncthreads();

  // write-out: Z into Xw's diagonal block (16-byte words).  L_jj itself is not needed again:
  // the panel uses Z_jj, and the rest of the sweep reads only the blocks below the diagonal.
  float* xo = Xw + j0 * ld + j0;
#pragma unroll 4
  for (int t = 0; t < kNb * kNb / 4 / kDiagThreads; ++t) {
    const int e = tid + t * kDiagThreads;
    const int r = e >> 5, c = (e & 31) * 4;
    *reinterpret_cast<float4*>(xo + r * ld + c) = *reinterpret_cast<const float4*>(X + r * kLd + c);
  }
}

// ---------------------------------------------------------------- strips (CUDA cores)
// Blocks [0, panel_strips): the panel below the diagonal block, 32 rows each:
//   P[i][c] = sum_{m <= c} B[i][j0 + m] Z[c][m]        (L_ij = B_ij Z_jj^T, rows i of B)
// written to P (row stride 128, rows relative to r_first).
// Blocks [panel_strips, ...): the inverse's row j, 32 columns each, in place in Xw:
//   X[j0 + r][c] = sum_{m <= r} Z[r][m] R[j0 + m][c]   (X_jc = Z_jj R_jc, c < j0)
// Z = Z_jj is Xw's diagonal block.  256 threads; each computes 4 x 4 outputs over K = 128 from
// shared memory, reading four consecutive m per 16-byte load: the panel's columns
// c = tx + 32 k take Z's rows 132 words apart (each load spans every bank in four
// wavefronts), the shared operand of a warp is a broadcast, and the row's columns are one
// 16-byte word.  The sums run over m in order.  The staging loads are unrolled so that each
// thread has several in flight.
__global__ void __launch_bounds__(kStripThreads)
factor_strip_kernel(const float* __restrict__ Bw, float* __restrict__ Xw, int64_t ld, int64_t j0,
                    float* __restrict__ P, int panel_strips, int64_t r_first) {
  // launched in stream order (scheduled early, beside the diagonal block's CTA, the strips ran
  // slower); lets the split kernel be scheduled
  pdl_launch_dependents();
  extern __shared__ __align__(16) float sm[];
  constexpr int kZl = kNb + 4;       // row-major Z (16-byte rows; rows 4 banks apart)
  constexpr int kRl = kStripRows + 4;
  const int tid = threadIdx.x;
  const bool panel = (int)blockIdx.x < panel_strips;
  const int sb = panel ? (int)blockIdx.x : (int)blockIdx.x - panel_strips;
  float* Zs = sm;                    // 128 x kZl
  float* Ss = sm + kNb * kZl;        // panel: B rows (i, m), 32 x kZl; row: R (m, c), 128 x kRl
  const float* zsrc = Xw + j0 * ld + j0;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;
#pragma unroll 16
  for (int e = tid; e < kNb * kNb / 4; e += kStripThreads) {
    const int r = e >> 5, c = (e & 31) * 4;
    *reinterpret_cast<float4*>(Zs + r * kZl + c) = *reinterpret_cast<const float4*>(zsrc + r * ld + c);
  }
  // Both products run over m in order, four m per step: 16-byte loads of four consecutive m
  // (the same address across a warp where the operand is shared: a broadcast).
  if (panel) {
    const int64_t row0 = r_first + (int64_t)sb * kStripRows;
#pragma unroll 4
    for (int e = tid; e < kStripRows * kNb / 4; e += kStripThreads) {
      const int i = e >> 5, m = (e & 31) * 4;
      *reinterpret_cast<float4*>(Ss + i * kZl + m) = *reinterpret_cast<const float4*>(Bw + (row0 + i) * ld + j0 + m);
    }
    __syncthreads();
    // outputs 32 rows x 128 columns: rows 4 ty .. +3, columns tx + 32 k (k < 4); Z's rows
    // tx + 32 k are read four m at a time (lanes 4 banks apart: four wavefronts per load)
    const int ty = tid >> 5, tx = tid & 31;
#pragma unroll 2
    for (int m = 0; m < kNb; m += 4) {
      float4 bv[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) bv[k] = *reinterpret_cast<const float4*>(Zs + (tx + 32 * k) * kZl + m);
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float4 av = *reinterpret_cast<const float4*>(Ss + (4 * ty + a) * kZl + m);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          acc[a][k] = __fmaf_rn(av.x, bv[k].x, acc[a][k]);
          acc[a][k] = __fmaf_rn(av.y, bv[k].y, acc[a][k]);
          acc[a][k] = __fmaf_rn(av.z, bv[k].z, acc[a][k]);
          acc[a][k] = __fmaf_rn(av.w, bv[k].w, acc[a][k]);
        }
      }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int k = 0; k < 4; ++k) P[((int64_t)sb * kStripRows + 4 * ty + a) * kNb + tx + 32 * k] = acc[a][k];
  } else {
    const int64_t col0 = (int64_t)sb * kStripRows;
#pragma unroll 4
    for (int e = tid; e < kNb * kStripRows / 4; e += kStripThreads) {
      const int m = e >> 3, c = (e & 7) * 4;
      *reinterpret_cast<float4*>(Ss + m * kRl + c) = *reinterpret_cast<const float4*>(Xw + (j0 + m) * ld + col0 + c);
    }
    __syncthreads();
    // outputs 128 rows x 32 columns: rows 4 ty .. +3, columns 4 tx .. +3
    const int ty = tid >> 3, tx = tid & 7;
#pragma unroll 2
    for (int m = 0; m < kNb; m += 4) {
      float4 av[4], bv[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) av[a] = *reinterpret_cast<const float4*>(Zs + (4 * ty + a) * kZl + m);
#pragma unroll
      for (int q = 0; q < 4; ++q) bv[q] = *reinterpret_cast<const float4*>(Ss + (m + q) * kRl + 4 * tx);
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float am[4] = {av[a].x, av[a].y, av[a].z, av[a].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          acc[a][0] = __fmaf_rn(am[q], bv[q].x, acc[a][0]);
          acc[a][1] = __fmaf_rn(am[q], bv[q].y, acc[a][1]);
          acc[a][2] = __fmaf_rn(am[q], bv[q].z, acc[a][2]);
          acc[a][3] = __fmaf_rn(am[q], bv[q].w, acc[a][3]);
        }
      }
    }
    // R was staged into shared memory before the first barrier, so the outputs may overwrite it
#pragma unroll
    for (int a = 0; a < 4; ++a)
      *reinterpret_cast<float4*>(Xw + (j0 + 4 * ty + a) * ld + col0 + 4 * tx) =
          make_float4(acc[a][0], acc[a][1], acc[a][2], acc[a][3]);
  }
}

// ---------------------------------------------------------------- three-way bf16 splits
// x = x1 + x2 + x3 with bf16 parts, each difference exact in fp32: the parts carry x to
// about 2^-24 relative.
__device__ __forceinline__ void split3(float x, uint16_t (&p)[3]) {
  const __nv_bfloat16 a = __float2bfloat16_rn(x);
  const float r1 = __fsub_rn(x, __bfloat162float(a));
  const __nv_bfloat16 b = __float2bfloat16_rn(r1);
  const float r2 = __fsub_rn(r1, __bfloat162float(b));
  const __nv_bfloat16 c = __float2bfloat16_rn(r2);
  p[0] = __bfloat16_as_ushort(a);
  p[1] = __bfloat16_as_ushort(b);
  p[2] = __bfloat16_as_ushort(c);
}

// Both split operands of a step's update in one launch.  Blocks [0, panel_blocks): the panel
// P [rows, 128] (fp32) into its place in Bw (rows r_first.., columns j0..) and as the two
// operands of the updates: An = [-P1 | -P1 | -P2 | -P1 | -P2 | -P3] and
// Bp = [P1 | P2 | P1 | P3 | P2 | P1] (rows of 6 * 128 bf16), so that An Bp^T = -P P^T to fp32
// accuracy (the six products E1U1, E1U2, E2U1, E1U3, E2U2, E3U1).  The blocks after them: the
// inverse's row block j (Xw rows j0..j0+127, columns 0..cols-1) transposed, as the B operand
// of the R update: Bx[c] = [X1 | X2 | X1 | X3 | X2 | X1] of column c of the row block, one
// 32 x 32 tile per block (4 tiles per 32 columns) through shared memory (coalesced reads
// along c, writes along the row index).  The two parts are independent.
__global__ void __launch_bounds__(256) factor_split_kernel(const float* __restrict__ P, int64_t rows,
                                                           float* __restrict__ Bw, const float* __restrict__ Xw,
                                                           int64_t ld, int64_t r_first, int64_t j0, int64_t cols,
                                                           int panel_blocks, uint16_t* __restrict__ An,
                                                           uint16_t* __restrict__ Bp, uint16_t* __restrict__ Bx) {
  pdl_launch_dependents();
  pdl_wait_primary();  // the strips' panel and row (programmatic dependent launch)
  if ((int)blockIdx.x < panel_blocks) {
    const int64_t total = rows * kNb;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
         e += (int64_t)panel_blocks * blockDim.x) {
      const int64_t i = e >> 7;
      const int k = (int)(e & (kNb - 1));
      const float x = P[e];
      Bw[(r_first + i) * ld + j0 + k] = x;
      uint16_t p[3], q[3];
      split3(x, p);
      split3(-x, q);
      uint16_t* a = An + i * kSplitK + k;
      uint16_t* b = Bp + i * kSplitK + k;
      a[0] = q[0]; a[kNb] = q[0]; a[2 * kNb] = q[1]; a[3 * kNb] = q[0]; a[4 * kNb] = q[1]; a[5 * kNb] = q[2];
      b[0] = p[0]; b[kNb] = p[1]; b[2 * kNb] = p[0]; b[3 * kNb] = p[2]; b[4 * kNb] = p[1]; b[5 * kNb] = p[0];
    }
    return;
  }
  __shared__ float t[32][33];
  const int rb = (int)blockIdx.x - panel_blocks;
  const int64_t c0 = (int64_t)(rb >> 2) * 32;
  const int m0 = (rb & 3) * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int mm = ty; mm < 32; mm += 8) t[mm][tx] = c0 + tx < cols ? Xw[(j0 + m0 + mm) * ld + c0 + tx] : 0.0f;
  __syncthreads();
  for (int cc = ty; cc < 32; cc += 8) {
    const int64_t c = c0 + cc;
    if (c >= cols) continue;
    uint16_t p[3];
    split3(t[tx][cc], p);
    uint16_t* b = Bx + c * kSplitK + m0 + tx;
    b[0] = p[0]; b[kNb] = p[1]; b[2 * kNb] = p[0]; b[3 * kNb] = p[2]; b[4 * kNb] = p[1]; b[5 * kNb] = p[0];
  }
}

inline int64_t round256(int64_t bytes) { return (bytes + 255) / 256 * 256; }

// The diagonal block, split and update kernels are launched with programmatic dependent launch:
// the kernel before each lets it be scheduled as soon as it starts, and it waits for that
// kernel's writes before its first read, so those launches do not each wait out a launch's
// latency (n = 4096: 1.92 -> 1.88 ms).  The strips are launched in stream order: scheduled
// early, beside the diagonal block, they made the sweep 4 % slower.
template <typename... KArgs, typename... Args>
cudaError_t launch_chained(void (*kernel)(KArgs...), unsigned grid, unsigned block, int smem, cudaStream_t stream,
                           Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(block, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t err = cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

}  // namespace

int64_t gptq_factor_padded(int64_t n) { return (n + kNb - 1) / kNb * kNb; }

// W2 = [B | X] (n_pad x 2 n_pad fp32), the panel (n_pad x 128 fp32) and the split operands (A: n_pad x 768 bf16; B: [L_:j ; X_j,:], n_pad x 768 bf16), each region
// 256-byte aligned.
size_t gptq_factor_workspace(int64_t n) {
  const int64_t np = gptq_factor_padded(n);
  return (size_t)(round256(2 * np * np * 4) + round256(np * kNb * 4) + 2 * round256(np * kSplitK * 2));
}

cudaError_t launch_gptq_factor(const float* H, int64_t n, int64_t ld_h, float damp, float* Uo, uint8_t* dead,
                               int32_t* info, void* workspace, cudaStream_t stream) {
  DeviceInfo dinfo;
  cudaError_t err = current_device_info(&dinfo);
  if (err != cudaSuccess) return err;
  const int64_t np = gptq_factor_padded(n);
  const int64_t ld = 2 * np;
  uint8_t* base = static_cast<uint8_t*>(workspace);
  float* Bw = reinterpret_cast<float*>(base);  // left half of W2; X = Bw + np
  float* Xw = Bw + np;
  float* P = reinterpret_cast<float*>(base + round256(2 * np * np * 4));
  uint8_t* ops = base + round256(2 * np * np * 4) + round256(np * kNb * 4);
  uint16_t* An = reinterpret_cast<uint16_t*>(ops);
  uint16_t* Bo = reinterpret_cast<uint16_t*>(ops + round256(np * kSplitK * 2));

  if ((err = cudaMemsetAsync(info, 0, 3 * sizeof(int32_t), stream)) != cudaSuccess) return err;
  // the damped diagonal, in the panel's buffer until the sweep writes the first panel
  float* dd = P;
  damp_diagonal_kernel<<<1, 1024, 0, stream>>>(H, n, ld_h, damp, dead, dd);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  reverse_pad_kernel<<<dim3((unsigned)(np / 32), (unsigned)(np / 32)), 256, 0, stream>>>(H, n, ld_h, dd, np, Bw);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  if ((err = ensure_dynamic_smem(reinterpret_cast<const void*>(factor_diag_kernel), kDiagSmemBytes)) != cudaSuccess)
    return err;
  if ((err = ensure_dynamic_smem(reinterpret_cast<const void*>(factor_strip_kernel), kStripSmemBytes)) != cudaSuccess)
    return err;

  const int64_t nblk = np / kNb;
  for (int64_t jb = 0; jb < nblk; ++jb) {
    const int64_t j0 = jb * kNb;
    const int64_t r_first = j0 + kNb;          // first row below the diagonal block
    const int64_t rows = np - r_first;         // rows of the panel
    if ((err = launch_chained(factor_diag_kernel, 1, kDiagThreads, kDiagSmemBytes, stream, (const float*)Bw, ld, j0,
                              Xw, info)) != cudaSuccess)
      return err;
    const int panel_strips = (int)(rows / kStripRows);
    const int row_strips = (int)(j0 / kStripRows);
    if (panel_strips + row_strips > 0) {
      factor_strip_kernel<<<(unsigned)(panel_strips + row_strips), kStripThreads, kStripSmemBytes, stream>>>(
          Bw, Xw, ld, j0, P, panel_strips, r_first);
      if ((err = cudaGetLastError()) != cudaSuccess) return err;
    }
    if (rows == 0) break;
    const int sblocks = (int)std::max<int64_t>(1, std::min<int64_t>((rows * kNb + 255) / 256,
                                                                    (int64_t)dinfo.sm_count * 8));
    const int64_t xcols = j0 + kNb;            // columns of the inverse's row block j, diagonal included
    const int64_t rblocks = (xcols + 31) / 32 * (kNb / 32);
    if ((err = launch_chained(factor_split_kernel, (unsigned)(sblocks + rblocks), 256, 0, stream, (const float*)P, rows,
                              Bw, (const float*)Xw, ld, r_first, j0, xcols, sblocks, An, Bo, Bo + rows * kSplitK)) !=
        cudaSuccess)
      return err;
    // rows below the diagonal block, columns r_first .. np + xcols of W2 (rows + xcols = np):
    // the trailing square and the inverse's rows, -= L_:j [L_:j ; X_j,:]^T
    if ((err = launch_gemm_accumulate(An, Bo, rows, rows + xcols, kSplitK, Bw + r_first * ld + r_first, ld, stream,
                                      true)) != cudaSuccess)
      return err;
  }
  // 256 columns per block, rows strided over 512 blocks (several independent rows per thread)
  reverse_out_kernel<<<dim3((unsigned)((n + 255) / 256), (unsigned)std::min<int64_t>(n, 512)), 256, 0, stream>>>(
      Xw, ld, n, Uo);
  return cudaGetLastError();
}

}  // namespace hscale
