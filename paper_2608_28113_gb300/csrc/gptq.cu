// gptq.cu -- GPTQ with H-Scale as the local quantizer (Algorithm 3) on sm_103a.
//
//   factor            the damped inverse-Cholesky factor U of GPTQ: dead channels (H_jj = 0)
//                     get H_jj = 1, the diagonal gets damp * mean(diag), and U is upper
//                     triangular with U^T U = (H + damp I)^-1 = A^-1.  It is formed without
//                     A^-1: with J the order-reversing permutation and J A J = L L^T (L lower,
//                     Cholesky), A = (J L J)(J L^T J), so U = (J L J)^-1 = J L^-1 J, an
//                     upper-triangular matrix with a positive diagonal, hence the Cholesky
//                     factor.  cuSOLVER does the Cholesky and cuBLAS the triangular solve
//                     L^T Y = I (both loaded at run time) on column-major storage: Y = L^-T
//                     in column-major order is (J Y J)^T = U^T after reversing the array,
//                     i.e. row-major U.
//   block_kernel      four lanes per 16-element group of a block of B columns of the running
//                     fp32 weights: the RTN code (Eq. 7) of the current weights, the exact
//                     H-Scale search over the window (Algorithm 1, exact E2M1 decisions, the
//                     tie rule of the search), the codes and packed nibbles, and the
//                     propagated errors E = (W - W_hat) / U_jj
//   update            W[:, i+B:] -= E U[i:i+B, i+B:] with fp32-level accuracy on the tensor
//                     cores (three-way bf16 splits, six products, one GEMM)
#include <dlfcn.h>

#include <algorithm>
#include <cstdio>
#include <mutex>
#include <vector>

#include <cublas_v2.h>
#include <cuda_bf16.h>
#include <cusolverDn.h>

#include "hscale_device.cuh"
#include "hscale_internal.h"

namespace hscale {
namespace {

// ---------------------------------------------------------------- cuSOLVER at run time
struct Solver {
  decltype(&cusolverDnCreate) create = nullptr;
  decltype(&cusolverDnSetStream) set_stream = nullptr;
  decltype(&cusolverDnSpotrf_bufferSize) potrf_size = nullptr;
  decltype(&cusolverDnSpotrf) potrf = nullptr;
  decltype(&cublasCreate_v2) blas_create = nullptr;
  decltype(&cublasSetStream_v2) blas_set_stream = nullptr;
  decltype(&cublasStrsm_v2) trsm = nullptr;
  bool ok = false;
};

const Solver& solver() {
  static Solver s;
  static std::once_flag once;
  std::call_once(once, [] {
    void* lib = nullptr;
    for (const char* name : {"libcusolver.so.12", "libcusolver.so.11", "libcusolver.so"}) {
      lib = dlopen(name, RTLD_NOW | RTLD_LOCAL);
      if (lib) break;
    }
    if (!lib) return;
    s.create = reinterpret_cast<decltype(s.create)>(dlsym(lib, "cusolverDnCreate"));
    s.set_stream = reinterpret_cast<decltype(s.set_stream)>(dlsym(lib, "cusolverDnSetStream"));
    s.potrf_size = reinterpret_cast<decltype(s.potrf_size)>(dlsym(lib, "cusolverDnSpotrf_bufferSize"));
    s.potrf = reinterpret_cast<decltype(s.potrf)>(dlsym(lib, "cusolverDnSpotrf"));
    void* blas = nullptr;
    for (const char* name : {"libcublas.so.13", "libcublas.so.12", "libcublas.so"}) {
      blas = dlopen(name, RTLD_NOW | RTLD_LOCAL);
      if (blas) break;
    }
    if (!blas) return;
    s.blas_create = reinterpret_cast<decltype(s.blas_create)>(dlsym(blas, "cublasCreate_v2"));
    s.blas_set_stream = reinterpret_cast<decltype(s.blas_set_stream)>(dlsym(blas, "cublasSetStream_v2"));
    s.trsm = reinterpret_cast<decltype(s.trsm)>(dlsym(blas, "cublasStrsm_v2"));
    s.ok = s.create && s.set_stream && s.potrf_size && s.potrf && s.blas_create && s.blas_set_stream && s.trsm;
  });
  return s;
}

// one handle of each library per device, created on first use
cusolverDnHandle_t solver_handle() {
  static std::mutex mu;
  static cusolverDnHandle_t handles[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!handles[dev] && solver().create(&handles[dev]) != CUSOLVER_STATUS_SUCCESS) handles[dev] = nullptr;
  return handles[dev];
}

cublasHandle_t blas_handle() {
  static std::mutex mu;
  static cublasHandle_t handles[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!handles[dev] && solver().blas_create(&handles[dev]) != CUBLAS_STATUS_SUCCESS) handles[dev] = nullptr;
  return handles[dev];
}

// ---------------------------------------------------------------- factor helpers
// One block: dead channels, the mean of the diagonal, and the damping added to it.
__global__ void __launch_bounds__(1024) damp_diagonal_kernel(float* A, int64_t n, float damp, uint8_t* dead) {
  __shared__ double part[1024];
  double s = 0.0;
  for (int64_t j = threadIdx.x; j < n; j += blockDim.x) {
    float d = A[j * n + j];
    const bool is_dead = (d == 0.0f);
    if (is_dead) A[j * n + j] = d = 1.0f;
    if (dead) dead[j] = (uint8_t)is_dead;
    s += (double)d;
  }
  part[threadIdx.x] = s;
  __syncthreads();
  for (int step = 512; step > 0; step >>= 1) {
    if ((int)threadIdx.x < step) part[threadIdx.x] += part[threadIdx.x + step];
    __syncthreads();
  }
  const float add = (float)((double)damp * part[0] / (double)n);
  for (int64_t j = threadIdx.x; j < n; j += blockDim.x) A[j * n + j] += add;
}

// B[i][j] = A[p][q] with (p, q) = (n-1-i, n-1-j) taken in the upper triangle (p <= q) of
// row-major A: B = J A J, complete and symmetric, from A's upper triangle.
__global__ void __launch_bounds__(256) reverse_symmetric_kernel(const float* __restrict__ A, int64_t n,
                                                                float* __restrict__ B) {
  const int64_t total = n * n;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = e / n, j = e - i * n;
    const int64_t p = n - 1 - i, q = n - 1 - j;
    B[e] = p <= q ? A[p * n + q] : A[q * n + p];
  }
}

// Reverses the n*n array A in place (A[e] <-> A[n*n - 1 - e]) and zeroes what lands below
// the diagonal of row-major A.
__global__ void __launch_bounds__(256) reverse_upper_kernel(float* A, int64_t n) {
  const int64_t total = n * n, half = total / 2;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < half; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t f = total - 1 - e;
    const float a = A[e], b = A[f];
    const int64_t re = e / n, rf = f / n;
    A[e] = re > e - re * n ? 0.0f : b;
    A[f] = rf > f - rf * n ? 0.0f : a;
  }
}

// the n x n identity
__global__ void __launch_bounds__(256) identity_kernel(float* X, int64_t n) {
  const int64_t total = n * n;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / n;
    X[e] = (e - r * n == r) ? 1.0f : 0.0f;
  }
}

// ---------------------------------------------------------------- block quantizer
__device__ __forceinline__ bool better_code(float e, int c, float be, int bc, int c0) {
  if (e != be) return e < be;
  const int s = c - c0, bs = bc - c0;
  const int as = s < 0 ? -s : s, abs_ = bs < 0 ? -bs : bs;
  return as < abs_ || (as == abs_ && s < bs);
}

// sum_j h_j (a_j - s' q_j)^2 with exact E2M1 decisions, one rounding per residual and a
// fixed pairwise sum (relative error <= 8 * 2^-24)
__device__ float exact_group_score(const float (&a)[16], const float (&hj)[16], uint32_t c, float sgk) {
  const float l = e4m3_mag(c);
  const float inv = inv_raw_of(__fmul_rn(l, sgk));
  float t[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint32_t k = e2m1_code(a[j], inv, l, sgk);
    const float r = __fmaf_rn(-__fmul_rn(e2m1_from_raw(k << 22), l), sgk, a[j]);
    t[j] = __fmul_rn(hj[j], __fmul_rn(r, r));
  }
#pragma unroll
  for (int step = 1; step < 16; step <<= 1)
#pragma unroll
    for (int j = 0; j + step < 16; j += 2 * step) t[j] = __fadd_rn(t[j], t[j + step]);
  return t[0];
}

// Four lanes (a quad) per group: each scores every fourth candidate of the window with exact
// decisions, the quad keeps the best under the search's tie rule (a total order, so every
// lane ends with the same code), and each lane writes the nibbles and errors of four of the
// group's elements.
__global__ void __launch_bounds__(128) block_kernel(const float* __restrict__ W, int64_t m, int64_t n, int64_t col0,
                                                    int B, const float* __restrict__ h, const float* __restrict__ U,
                                                    const float* __restrict__ global_scale, int down, int up,
                                                    uint8_t* __restrict__ codes, uint2* __restrict__ packed,
                                                    float* __restrict__ E) {
  const int gpb = B / 16;
  const int64_t total = m * gpb * 4;  // lanes
  const int q = threadIdx.x & 3;
  const ScaleDomain d = make_scale_domain(*global_scale);
  const float inv6 = rtn_inv6_raw(d.sgk);
  // block-uniform trip count: every lane of a warp reaches the shuffles together
  for (int64_t base = (int64_t)blockIdx.x * blockDim.x; base < total; base += (int64_t)gridDim.x * blockDim.x) {
    const int64_t lane_id = base + threadIdx.x;
    const bool active = lane_id < total;
    const int64_t g = active ? lane_id >> 2 : 0;
    const int64_t r = g / gpb;
    const int i = (int)(g - r * gpb);
    const int64_t col = col0 + 16 * i;
    float w[16], a[16], hj[16];
    float amax = 0.0f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float4 v = reinterpret_cast<const float4*>(W + r * n + col)[k];
      const float4 hv = reinterpret_cast<const float4*>(h + col)[k];
      w[4 * k] = v.x; w[4 * k + 1] = v.y; w[4 * k + 2] = v.z; w[4 * k + 3] = v.w;
      hj[4 * k] = hv.x; hj[4 * k + 1] = hv.y; hj[4 * k + 2] = hv.z; hj[4 * k + 3] = hv.w;
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      a[j] = __fmul_rn(fabsf(w[j]), d.pw);
      amax = fmaxf(amax, a[j]);
    }
    const int c0 = (int)rtn_code(amax, d.sgk, inv6);
    const int lo = max(1, c0 - down), hi = min((int)kE4M3MaxCode, c0 + up);
    float be = 0.0f;
    int bc = -1;
    for (int c = lo + q; c <= hi; c += 4) {
      const float e = exact_group_score(a, hj, (uint32_t)c, d.sgk);
      if (bc < 0 || better_code(e, c, be, bc, c0)) {
        be = e;
        bc = c;
      }
    }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      const float oe = __shfl_xor_sync(0xFFFFFFFFu, be, off);
      const int oc = __shfl_xor_sync(0xFFFFFFFFu, bc, off);
      if (oc >= 0 && (bc < 0 || better_code(oe, oc, be, bc, c0))) {
        be = oe;
        bc = oc;
      }
    }
    const float l = e4m3_mag((uint32_t)bc);
    const float inv = inv_raw_of(__fmul_rn(l, d.sgk));
    // this lane's elements 4q..4q+3 (read again as one vector: no dynamic register index)
    const float4 wq = reinterpret_cast<const float4*>(W + r * n + col)[q];
    const float wv[4] = {wq.x, wq.y, wq.z, wq.w};
    uint32_t part = 0u;  // this lane's four nibbles in their place in the group's 32-bit word
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = 4 * q + t;
      const float av = __fmul_rn(fabsf(wv[t]), d.pw);
      const uint32_t k = e2m1_code(av, inv, l, d.sgk);
      const uint32_t neg = signbit(wv[t]) ? 1u : 0u;
      part |= ((neg << 3) | k) << (4 * (j & 7));
      float what = __fmul_rn(d.sg, __fmul_rn(e2m1_from_raw(k << 22), l));  // s_g (l q), l q exact
      if (neg) what = -what;
      if (active) E[r * B + 16 * i + j] = __fdiv_rn(__fsub_rn(wv[t], what), U[(col + j) * n + col + j]);
    }
    const uint32_t word = part | __shfl_xor_sync(0xFFFFFFFFu, part, 1);  // lanes 0-1: word 0, 2-3: word 1
    const uint32_t other = __shfl_xor_sync(0xFFFFFFFFu, word, 2);
    if (active && q == 0) {
      codes[r * (n / 16) + col / 16] = (uint8_t)bc;
      packed[r * (n / 16) + col / 16] = make_uint2(word, other);
    }
  }
}

// The update W[:, c1:] -= E U[col0:c1, c1:] (c1 = col0 + B) runs on the tensor cores with
// fp32-level accuracy: every fp32 value x is split into three bf16 parts x1 + x2 + x3 (each
// difference exact in fp32, so the parts carry x to about 2^-24 relative), and the six
// products E1 U1, E1 U2, E2 U1, E1 U3, E2 U2, E3 U1 (every pair whose weight is above
// 2^-24) are one bf16 GEMM over K = 6B with fp32 accumulation: A' = [-E1 | -E1 | -E2 | -E1
// | -E2 | -E3] against B' = [U1 | U2 | U1 | U3 | U2 | U1] (the negation makes the GEMM's
// accumulate a subtract).
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

// A' [m, 6B] from E [m, B] (segments -E1, -E1, -E2, -E1, -E2, -E3)
__global__ void __launch_bounds__(256) split_e_kernel(const float* __restrict__ E, int64_t m, int B,
                                                      uint16_t* __restrict__ A) {
  const int64_t total = m * B;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / B;
    const int k = (int)(e - r * B);
    uint16_t p[3];
    split3(-E[e], p);
    uint16_t* row = A + r * 6 * B + k;
    row[0] = p[0];
    row[B] = p[0];
    row[2 * B] = p[1];
    row[3 * B] = p[0];
    row[4 * B] = p[1];
    row[5 * B] = p[2];
  }
}

// B' [nn, 6B] from U[col0 + k, c1 + j] (segments U1, U2, U1, U3, U2, U1), transposed through
// 32 x 32 shared-memory tiles so that the reads of U and the writes of B' are coalesced
__global__ void __launch_bounds__(256) split_u_kernel(const float* __restrict__ U, int64_t n, int64_t col0, int B,
                                                      int64_t c1, uint16_t* __restrict__ Bt) {
  __shared__ float t[32][33];
  const int64_t j0 = (int64_t)blockIdx.x * 32;
  const int k0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int kk = ty; kk < 32; kk += 8) {
    const int64_t col = c1 + j0 + tx;
    t[kk][tx] = (k0 + kk < B && col < n) ? U[(col0 + k0 + kk) * n + col] : 0.0f;
  }
  __syncthreads();
  for (int jj = ty; jj < 32; jj += 8) {
    const int64_t j = j0 + jj;
    const int k = k0 + tx;
    if (c1 + j < n && k < B) {
      uint16_t p[3];
      split3(t[tx][jj], p);
      uint16_t* row = Bt + j * 6 * B + k;
      row[0] = p[0];
      row[B] = p[1];
      row[2 * B] = p[0];
      row[3 * B] = p[2];
      row[4 * B] = p[1];
      row[5 * B] = p[0];
    }
  }
}

__global__ void __launch_bounds__(256) to_fp32_kernel(const uint16_t* __restrict__ w, int64_t m, int64_t n,
                                                      const uint8_t* __restrict__ dead, float* __restrict__ W) {
  const int64_t total = m * n;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t c = e % n;
    W[e] = (dead && dead[c]) ? 0.0f : __uint_as_float((uint32_t)w[e] << 16);
  }
}

}  // namespace

// ---------------------------------------------------------------- host side
bool gptq_solver_available() { return solver().ok && solver_handle() != nullptr && blas_handle() != nullptr; }

// The factor's workspace in floats: J A J and its Cholesky factor (n*n, rounded up to 64
// floats), then cuSOLVER's.
size_t gptq_factor_solver_floats(int64_t n) {
  if (!gptq_solver_available()) return 0;
  int a = 0;
  if (solver().potrf_size(solver_handle(), CUBLAS_FILL_MODE_LOWER, (int)n, nullptr, (int)n, &a) !=
      CUSOLVER_STATUS_SUCCESS)
    return 0;
  return ((size_t)n * (size_t)n + 63) / 64 * 64 + std::max(a, 1);
}

cudaError_t launch_gptq_factor(const float* H, int64_t n, int64_t ld_h, float damp, float* Uo, uint8_t* dead,
                               int32_t* info, float* work, size_t work_floats, cudaStream_t stream) {
  if (!gptq_solver_available()) return cudaErrorNotSupported;
  const Solver& sv = solver();
  cusolverDnHandle_t hd = solver_handle();
  cublasHandle_t hb = blas_handle();
  if (sv.set_stream(hd, stream) != CUSOLVER_STATUS_SUCCESS || sv.blas_set_stream(hb, stream) != CUBLAS_STATUS_SUCCESS)
    return cudaErrorUnknown;
  const size_t x_floats = ((size_t)n * (size_t)n + 63) / 64 * 64;
  if (work_floats <= x_floats) return cudaErrorInvalidValue;
  float* X = work;
  float* solver_work = work + x_floats;
  cudaError_t err = cudaMemcpy2DAsync(Uo, (size_t)n * 4, H, (size_t)ld_h * 4, (size_t)n * 4, (size_t)n,
                                      cudaMemcpyDeviceToDevice, stream);
  if (err != cudaSuccess) return err;
  damp_diagonal_kernel<<<1, 1024, 0, stream>>>(Uo, n, damp, dead);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  DeviceInfo dinfo;
  if ((err = current_device_info(&dinfo)) != cudaSuccess) return err;
  const unsigned blocks = (unsigned)std::max<int64_t>(1, std::min<int64_t>((n * n + 255) / 256,
                                                                          (int64_t)dinfo.sm_count * 16));
  // X = J A J, symmetric, from the upper triangle of the damped copy
  reverse_symmetric_kernel<<<blocks, 256, 0, stream>>>(Uo, n, X);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  if ((err = cudaMemsetAsync(info, 0, 3 * sizeof(int32_t), stream)) != cudaSuccess) return err;
  const int ni = (int)n, lw = (int)std::min<size_t>(work_floats - x_floats, (size_t)INT32_MAX);
  if (sv.potrf(hd, CUBLAS_FILL_MODE_LOWER, ni, X, ni, solver_work, lw, info) != CUSOLVER_STATUS_SUCCESS)
    return cudaErrorUnknown;
  // L^T Y = I: Y = L^-T (upper, column-major) in U's buffer
  identity_kernel<<<blocks, 256, 0, stream>>>(Uo, n);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  const float one = 1.0f;
  if (sv.trsm(hb, CUBLAS_SIDE_LEFT, CUBLAS_FILL_MODE_LOWER, CUBLAS_OP_T, CUBLAS_DIAG_NON_UNIT, ni, ni, &one, X, ni,
              Uo, ni) != CUBLAS_STATUS_SUCCESS)
    return cudaErrorUnknown;
  // reversed, column-major Y is row-major U; the other triangle is cleared
  reverse_upper_kernel<<<blocks, 256, 0, stream>>>(Uo, n);
  return cudaGetLastError();
}

cudaError_t launch_gptq_hscale(const void* w, int64_t m, int64_t n, const float* U, const float* h,
                               const float* global_scale, const uint8_t* dead, int block, int down, int up,
                               uint8_t* codes, uint8_t* packed, float* Wf, float* E, uint16_t* A6, uint16_t* B6,
                               cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const unsigned cvt_blocks = (unsigned)std::min<int64_t>((m * n + 255) / 256, (int64_t)info.sm_count * 16);
  to_fp32_kernel<<<cvt_blocks, 256, 0, stream>>>(static_cast<const uint16_t*>(w), m, n, dead, Wf);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  for (int64_t col0 = 0; col0 < n; col0 += block) {
    const int64_t groups = m * (block / 16);
    const unsigned qb = (unsigned)std::min<int64_t>((groups * 4 + 127) / 128, (int64_t)info.sm_count * 16);
    block_kernel<<<qb, 128, 0, stream>>>(Wf, m, n, col0, block, h, U, global_scale, down, up, codes,
                                         reinterpret_cast<uint2*>(packed), E);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    if (col0 + block < n) {
      const int64_t c1 = col0 + block, nn = n - c1;
      const unsigned eb = (unsigned)std::min<int64_t>((m * block + 255) / 256, (int64_t)info.sm_count * 16);
      split_e_kernel<<<eb, 256, 0, stream>>>(E, m, block, A6);
      if ((err = cudaGetLastError()) != cudaSuccess) return err;
      split_u_kernel<<<dim3((unsigned)((nn + 31) / 32), (unsigned)((block + 31) / 32)), 256, 0, stream>>>(
          U, n, col0, block, c1, B6);
      if ((err = cudaGetLastError()) != cudaSuccess) return err;
      if ((err = launch_gemm_accumulate(A6, B6, m, nn, 6 * (int64_t)block, Wf + c1, n, stream)) != cudaSuccess)
        return err;
    }
  }
  return cudaSuccess;
}

}  // namespace hscale
