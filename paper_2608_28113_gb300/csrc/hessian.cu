// hessian.cu -- diagonal-Hessian proxy h_j += sum_t x_tj^2 (Sec. 3.2, Eq. 4) on sm_103a.
//
// HBM-bound column sum of squares over a bf16 token chunk X[tokens, ld].
//
// Layout of the work
//   * A CTA owns a 64-channel column tile (eight 16-byte vectors per row) and a
//     contiguous run of tokens.  Its 256 threads are 32 row phases x 8 vectors: a warp
//     reads 4 rows x 128 contiguous bytes per load instruction, and each thread keeps
//     8 loads of 16 bytes in flight (rows r, r+32, ..., r+224).
//   * The token range of a tile is split over the CTAs of one thread-block cluster
//     (1, 2, 4 or 8 CTAs, picked so the grid is about one wave of resident CTAs).  The
//     CTAs of a cluster reduce their partial sums through distributed shared memory, so
//     the kernel needs no global scratch, no atomics and no second launch.
// Determinism and accuracy
//   x^2 of a bf16 value is exact in fp32.  Each thread adds at most 1024 squares in
//   token order; partials then meet in fixed-order pairwise trees (4 phases in a warp,
//   8 warps in the CTA, the cluster's CTAs), and the total is added to h once.  Every
//   run gives the same bits, and a call adds a relative error of at most
//   (1024 + 2 + 3 + 3 + 1) * 2^-24 to h.
#include <cooperative_groups.h>

#include "hscale_device.cuh"
#include "hscale_internal.h"

namespace cg = cooperative_groups;

namespace hscale {
namespace {

constexpr int kVecPerRow = 8;                      // 16-byte vectors per tile row
constexpr int kTileCols = kVecPerRow * 8;          // 64 channels
constexpr int kThreads = 256;
constexpr int kPhases = kThreads / kVecPerRow;     // 32 rows read side by side
constexpr int kUnroll = 8;                         // rows in flight per thread
constexpr int kWarps = kThreads / 32;
constexpr int64_t kMaxRunPerThread = 1024;         // longest sequential fp32 run
constexpr int kMaxCluster = 8;

__device__ __forceinline__ void accum_sq8(float (&acc)[8], const uint4& v) {
  const float f0 = bf16_lo(v.x), f1 = bf16_hi(v.x), f2 = bf16_lo(v.y), f3 = bf16_hi(v.y);
  const float f4 = bf16_lo(v.z), f5 = bf16_hi(v.z), f6 = bf16_lo(v.w), f7 = bf16_hi(v.w);
  acc[0] = __fmaf_rn(f0, f0, acc[0]);
  acc[1] = __fmaf_rn(f1, f1, acc[1]);
  acc[2] = __fmaf_rn(f2, f2, acc[2]);
  acc[3] = __fmaf_rn(f3, f3, acc[3]);
  acc[4] = __fmaf_rn(f4, f4, acc[4]);
  acc[5] = __fmaf_rn(f5, f5, acc[5]);
  acc[6] = __fmaf_rn(f6, f6, acc[6]);
  acc[7] = __fmaf_rn(f7, f7, acc[7]);
}

template <int CS>
__global__ void __launch_bounds__(kThreads)
hessian_colsumsq_kernel(const uint4* __restrict__ x, int64_t tokens, int64_t ld_vec, int nvec,
                        int n, float* __restrict__ h, int64_t rows_per_cta) {
  __shared__ float warp_part[kWarps][kTileCols];
  __shared__ float cta_part[kTileCols];

  cg::cluster_group cluster = cg::this_cluster();
  const unsigned crank = cluster.block_rank();
  const int tid = threadIdx.x;
  const int v = tid & (kVecPerRow - 1);
  const int phase = tid / kVecPerRow;
  const int vec = blockIdx.y * kVecPerRow + v;
  const int64_t r0 = (int64_t)crank * rows_per_cta;
  const int64_t r1 = min(tokens, r0 + rows_per_cta);

  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (vec < nvec) {
    const uint4* p = x + vec;
    int64_t r = r0 + phase;
    for (; r + (int64_t)(kUnroll - 1) * kPhases < r1; r += (int64_t)kUnroll * kPhases) {
      uint4 q[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) q[u] = ld_stream_v4(p + (r + (int64_t)u * kPhases) * ld_vec);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) accum_sq8(acc, q[u]);
    }
    for (; r < r1; r += kPhases) accum_sq8(acc, ld_stream_v4(p + r * ld_vec));
  }

  // phases 4w..4w+3 of a warp: lane bit 3 is phase bit 0, lane bit 4 is phase bit 1
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    float t = acc[k];
    t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, 8));
    t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, 16));
    acc[k] = t;
  }
  const int lane = tid & 31, warp = tid >> 5;
  if (lane < kVecPerRow) {
#pragma unroll
    for (int k = 0; k < 8; ++k) warp_part[warp][lane * 8 + k] = acc[k];
  }
  __syncthreads();
  if (tid < kTileCols) {
    float s[kWarps];
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s[w] = warp_part[w][tid];
#pragma unroll
    for (int step = 1; step < kWarps; step <<= 1)
#pragma unroll
      for (int w = 0; w + step < kWarps; w += 2 * step) s[w] = __fadd_rn(s[w], s[w + step]);
    cta_part[tid] = s[0];
  }

  if constexpr (CS == 1) {
    __syncthreads();
    if (tid < kTileCols) {
      const int col = blockIdx.y * kTileCols + tid;
      if (col < n) h[col] = __fadd_rn(h[col], cta_part[tid]);
    }
  } else {
    cluster.sync();
    if (crank == 0 && tid < kTileCols) {
      float s[CS];
#pragma unroll
      for (int r = 0; r < CS; ++r) s[r] = *cluster.map_shared_rank(&cta_part[tid], r);
#pragma unroll
      for (int step = 1; step < CS; step <<= 1)
#pragma unroll
        for (int r = 0; r + step < CS; r += 2 * step) s[r] = __fadd_rn(s[r], s[r + step]);
      const int col = blockIdx.y * kTileCols + tid;
      if (col < n) h[col] = __fadd_rn(h[col], s[0]);
    }
    cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
  }
}

template <int CS>
cudaError_t launch_cs(const uint4* x, int64_t tokens, int64_t ld_vec, int nvec, int n, float* h,
                      int tiles, cudaStream_t stream) {
  const int64_t max_rows_per_cta = kMaxRunPerThread * kPhases;
  const int64_t rows_per_launch = max_rows_per_cta * CS;
  for (int64_t t0 = 0; t0 < tokens; t0 += rows_per_launch) {
    const int64_t t = min(tokens - t0, rows_per_launch);
    int64_t rows_per_cta = (t + CS - 1) / CS;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CS, tiles, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t err = cudaLaunchKernelEx(&cfg, hessian_colsumsq_kernel<CS>, x + t0 * ld_vec, t,
                                         ld_vec, nvec, n, h, rows_per_cta);
    if (err != cudaSuccess) return err;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_hessian(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* h,
                           cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int nvec = (int)(n / 8);
  const int tiles = (nvec + kVecPerRow - 1) / kVecPerRow;
  // about one wave: 256-thread CTAs, 4 resident per SM
  const int64_t target = (int64_t)info.sm_count * 4;
  int cs = 1;
  while (cs < kMaxCluster && (int64_t)tiles * cs * 2 <= target && (int64_t)cs * 2 * kPhases * 4 <= tokens)
    cs *= 2;
  const uint4* xv = static_cast<const uint4*>(x);
  const int64_t ld_vec = ld_x / 8;
  switch (cs) {
    case 1: return launch_cs<1>(xv, tokens, ld_vec, nvec, (int)n, h, tiles, stream);
    case 2: return launch_cs<2>(xv, tokens, ld_vec, nvec, (int)n, h, tiles, stream);
    case 4: return launch_cs<4>(xv, tokens, ld_vec, nvec, (int)n, h, tiles, stream);
    default: return launch_cs<8>(xv, tokens, ld_vec, nvec, (int)n, h, tiles, stream);
  }
}

}  // namespace hscale
