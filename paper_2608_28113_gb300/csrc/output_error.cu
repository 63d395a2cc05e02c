// output_error.cu -- the layer-output error ||X dW^T||_F^2 of an NVFP4 quantization (Eq. 3)
// on the tcgen05 tensor cores of sm_103a.
//
//   residual_kernel       dW = W - W_hat with W_hat = s_g * E4M3(code) * E2M1(nibble), as a
//                         bf16 pair hi = bf16(dW), lo = bf16(dW - hi), written as one matrix
//                         [hi | lo] per row (each half zero-padded to n_pad = 64 * ceil(n/64))
//   output_error_kernel   C = [X | X] [hi | lo]^T = X (hi + lo)^T on the tensor cores (bf16
//                         operands, fp32 accumulation in tensor memory), fused with the sum of
//                         squares of C: one fp64 partial per 128 x 256 tile of C
//   reduce_kernel         the partials summed in tile order, added to the caller's scalar
//   gemm_kernel<3>        H += X^T X, the full Hessian of Algorithm 3, with the same tensor-
//                         core pipeline over K = tokens, reading X as it is (both operands
//                         MN-major), and an epilogue that adds each 128 x 256 tile of the
//                         product into H; tiles wholly below the diagonal are skipped (the
//                         factor reads the upper triangle only).  K runs in segments of 2048
//                         tokens, each accumulated from zero and folded into a running sum
//                         in tensor memory
//   transpose_kernel,     the same for X whose rows are not 16-byte aligned (no TMA): X is
//   gemm_kernel<1>        transposed into the workspace (tokens contiguous per channel)
//                         and both operands are K-major
//
// The residual is rounded once (one FMA of the exact w - s_g * (l q)), and hi + lo carries
// it to a relative 2^-17, so the GEMM sees dW, not a difference of two large products.
//
// GEMM tile: 128 tokens x 256 outputs, K in steps of 64 bf16 (one 128-byte swizzle atom
// per row), a 4-stage ring of TMA loads (48 KB per stage).  Warp 0 issues the loads, warp 1
// owns the tensor memory and issues the MMAs (M = 128, N = 256, K = 16 each), warps 2-9
// read the 128 x 256 fp32 accumulator back (each warp half the columns of its 32-lane
// quarter) and square and sum it.  Every wait is bounded; one that runs out sets the error flag and the tile's
// partial becomes NaN.
#include <algorithm>
#include <cuda_bf16.h>

#include "hscale_device.cuh"
#include "hscale_internal.h"
#include "tcgen05.cuh"
#include "tma.cuh"

namespace hscale {
namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kGemmThreads = 320;  // TMA warp, MMA warp, 8 epilogue warps
constexpr uint32_t kTileABytes = kBM * kBK * 2;  // 16 KB
constexpr uint32_t kTileBBytes = kBN * kBK * 2;  // 32 KB
constexpr uint32_t kStageBytes = kTileABytes + kTileBBytes;
constexpr uint32_t kTmemCols = kBN;  // fp32 accumulator: 128 lanes x 256 columns
// Full Hessian (modes 1, 3) and output error (mode 0): the tensor cores accumulate in fp32
// with an error that grows with the accumulation length (the Hessian's diagonal comes out
// low by about 0.9 u per K = 16 step, measured), so each tile's K loop is cut into
// segments of kSegBlocks K blocks (2048 tokens, or 2048 of the 2 n channels of [X | X]).
// Each segment accumulates from zero in TMEM columns [0, 256); the epilogue warps add it in
// fp32 round-to-nearest into a running sum kept in TMEM columns [256, 512) and, after the
// last segment, add the running sum into H (or square and sum it).  With H = 0 before the
// call the Hessian is bit for bit that of successive calls of 2048 tokens, whatever the
// call size.
constexpr int kSegBlocks = 32;
constexpr uint32_t kTmemColsSeg = 2 * kBN;
constexpr uint32_t kGemmSmemBytes = kStages * kStageBytes + 1024 /* alignment */ + 256 /* barriers */;
// the GPTQ update also stages its epilogue: barriers in a 1 KB block (keeping the staging
// buffers 1 KB aligned for the 128-byte swizzle), then 4 KB per epilogue warp
constexpr uint32_t kUpdateSmemBytes = kStages * kStageBytes + 1024 /* alignment */ + 1024 + 8 * 4096;
constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, kBN);
constexpr uint32_t kIdescMN = idesc_bf16_f32_mn(kBM, kBN);
constexpr uint32_t kBoxBytes = 64 * kBK * 2;  // mode 3: one 64-channel x 64-token TMA box

__device__ uint32_t g_output_error_flags = 0;

// ---------------------------------------------------------------- TMA reduce-add
// The GPTQ update's epilogue adds each tile into the running weights with TMA: a warp
// stages 32 rows x 32 fp32 columns (4 KB, 128-byte swizzled, as the tensor map says) and
// one lane issues a bulk reduce-add, which the L2 applies in fp32 round-to-nearest without
// the SM reading the weights.  The coordinates are (column, row), column a multiple of 4.
constexpr uint32_t kStageRows = 32, kStageCols = 32;
constexpr uint32_t kStageBufBytes = kStageRows * kStageCols * 4;  // per epilogue warp

__device__ __forceinline__ void tma_reduce_add_2d(const CUtensorMap* map, const void* src, int32_t c0, int32_t c1) {
  asm volatile("cp.reduce.async.bulk.tensor.2d.global.shared::cta.add.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(c0), "r"(c1), "r"(smem_addr(src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// every committed bulk operation has finished reading shared memory
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// every committed bulk operation has completed
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------- residual
__device__ __forceinline__ uint32_t bf16x2_pack(__nv_bfloat16 lo, __nv_bfloat16 hi) {
  return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}

// One thread per 16-element slot of a [hi | lo] row: slots below ng hold a group, the rest
// of the padded half is written with zeros.
__global__ void __launch_bounds__(256) residual_kernel(const uint4* __restrict__ w, int64_t m, int ng,
                                                       int ng_pad, const float* __restrict__ global_scale,
                                                       const uint8_t* __restrict__ codes,
                                                       const uint2* __restrict__ packed,
                                                       uint4* __restrict__ dw2, int64_t ld_dw2) {
  const float sg = *global_scale;
  const int64_t slots = m * ng_pad;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < slots;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = t / ng_pad;
    const int i = (int)(t - r * ng_pad);
    uint4* hi_dst = dw2 + (r * ld_dw2 + (int64_t)i * 16) / 8;
    uint4* lo_dst = dw2 + (r * ld_dw2 + (int64_t)(ng_pad + i) * 16) / 8;
    if (i >= ng) {
      const uint4 z = make_uint4(0u, 0u, 0u, 0u);
      hi_dst[0] = z; hi_dst[1] = z; lo_dst[0] = z; lo_dst[1] = z;
      continue;
    }
    const int64_t g = r * ng + i;
    const uint4 p0 = ld_stream_v4(w + 2 * g), p1 = ld_stream_v4(w + 2 * g + 1);
    const uint32_t wb[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
    uint32_t c = codes[g] & 0x7Fu;
    c = c < 1u ? 1u : (c > kE4M3MaxCode ? kE4M3MaxCode : c);
    const float l = e4m3_mag(c);
    const uint2 nib = packed[g];
    uint32_t hw[8], lw[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      __nv_bfloat16 h2[2], l2[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = 2 * k + e;
        const uint32_t nb = ((j < 8 ? nib.x : nib.y) >> (4 * (j & 7))) & 0xFu;
        float lq = __fmul_rn(l, e2m1_from_raw((nb & 7u) << 22));  // exact: <= 6 significant bits
        if (nb & 8u) lq = -lq;
        const float wv = e ? bf16_hi(wb[k]) : bf16_lo(wb[k]);
        const float d = __fmaf_rn(-sg, lq, wv);  // w - s_g * l * q, rounded once
        h2[e] = __float2bfloat16_rn(d);
        l2[e] = __float2bfloat16_rn(__fsub_rn(d, __bfloat162float(h2[e])));
      }
      hw[k] = bf16x2_pack(h2[0], h2[1]);
      lw[k] = bf16x2_pack(l2[0], l2[1]);
    }
    hi_dst[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    hi_dst[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
    lo_dst[0] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
    lo_dst[1] = make_uint4(lw[4], lw[5], lw[6], lw[7]);
  }
}

// ---------------------------------------------------------------- GEMM + sum of squares
__device__ __forceinline__ float sum_squares32(const uint32_t (&r)[32]) {
  float t[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float a = __uint_as_float(r[2 * j]), b = __uint_as_float(r[2 * j + 1]);
    t[j] = __fmaf_rn(a, a, __fmul_rn(b, b));
  }
#pragma unroll
  for (int step = 1; step < 16; step <<= 1)
#pragma unroll
    for (int j = 0; j + step < 16; j += 2 * step) t[j] = __fadd_rn(t[j], t[j + step]);
  return t[0];
}

// kMode 0: the sum-of-squares GEMM of the output error (K runs over [X | X], kb_half
// blocks per half).  kMode 1: H[rows, cols] += A B^T over kb_half K blocks, both operands
// rows of X^T, tiles wholly below the diagonal skipped.  kMode 2: C[rows, cols] += A B^T
// over kb_half K blocks, every tile (the GPTQ update).  kMode 3: kMode 1 read from X itself
// ([tokens, n], channels contiguous): each stage loads 64-channel x 64-token boxes and
// the MMAs take both operands MN-major, so no transpose is needed.
// Tile t of a persistent GEMM's sequence (tiles_n column tiles per row of tiles) in groups of
// kRasterRows rows of tiles, column-major within a group: the tiles in flight at once (about
// one per SM) then cover a few row strips of A and a part of B's column strips, rather than
// every column strip of B for one or two row strips, so their operands stay in L2.
constexpr int kRasterRows = 8;
__device__ __forceinline__ void raster_tile(int t, int tiles_n, int tiles_total, int& tm, int& tn) {
  const int tiles_m = tiles_total / tiles_n;
  const int first = t / (kRasterRows * tiles_n) * kRasterRows;
  const int rows = min(kRasterRows, tiles_m - first);
  const int within = t - first * tiles_n;
  tm = first + within % rows;
  tn = within / rows;
}

template <int kMode>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap wmap,
            const __grid_constant__ CUtensorMap cmap, int kb_half, int tiles_n, int tiles_total,
            double* __restrict__ partials, float* __restrict__ H, int64_t h_rows, int64_t h_cols, int64_t ld_h) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* tile_a = smem;
  uint8_t* tile_b = smem + kStages * kTileABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* acc_ready = empty + kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_ready + 1);
  uint32_t* failed = tmem_slot + 1;
  uint64_t* seg_full = acc_ready + 2;  // segmented modes: a segment's partial is complete
  uint64_t* seg_empty = seg_full + 1;  // segmented modes: the partial has been read out
  uint64_t* tacc_full = seg_empty + 1;  // mode 2: accumulator a holds a finished tile
  uint64_t* tacc_empty = tacc_full + 2;  // mode 2: accumulator a has been read out
  double* warp_sum = reinterpret_cast<double*>(smem + kStages * kStageBytes + 128);
  constexpr bool kHessian = kMode == 1 || kMode == 3;
  // K loops cut into accumulation segments folded in TMEM: the Hessian (K = tokens) and the
  // output error (K = 2 n); the GPTQ update's K = 6 B is a single segment anyway
  constexpr bool kSegmented = kMode != 2;
  // The GPTQ update and the output error are persistent: a CTA takes tiles blockIdx.x,
  // + gridDim.x, ...  The update alternates two 256-column accumulators, so a tile's
  // epilogue (the TMA reduce-add into the running weights) runs alongside the next tile's
  // loads and MMAs.  The output error's segments run on across its tiles (one segment
  // counter), so the MMAs of a tile's first segment start as soon as the previous tile's
  // last partial has been read out, alongside that tile's sum of squares.  The Hessian modes
  // take one tile per CTA.
  constexpr bool kPersistent = kMode == 2 || kMode == 0;
  constexpr bool kTwoAcc = kMode == 2;
  constexpr uint32_t kCols = (kSegmented || kPersistent) ? kTmemColsSeg : kTmemCols;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ntiles = kPersistent ? (tiles_total - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x : 1;
  const int tile_m = blockIdx.x / tiles_n, tile_n = blockIdx.x - tile_m * tiles_n;
  constexpr bool kAccum = kMode != 0;
  const int kb_total = kAccum ? kb_half : 2 * kb_half;
  // H is symmetric and only its upper triangle is used: a tile wholly below the diagonal
  // (every column index below every row index) is skipped, uniformly for the whole CTA
  if (kHessian && (int64_t)(tile_n + 1) * kBN <= (int64_t)tile_m * kBM) return;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_ready, 1);
    mbar_init(seg_full, 1);
    mbar_init(seg_empty, 256);  // every epilogue thread arrives
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tacc_full[a], 1);
      mbar_init(&tacc_empty[a], 256);
    }
    *failed = 0u;
    mbar_fence_init();
    prefetch_tensormap(&xmap);
    prefetch_tensormap(&wmap);
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(tmem_slot), kCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_d = *tmem_slot;
  if (kMode == 2) {
    // launched with programmatic dependent launch by the factor's sweep: let the next kernel
    // be scheduled (after the TMEM allocation), then wait for the previous one's writes
    // before the first load; without the launch attribute both are no-ops
    pdl_launch_dependents();
    pdl_wait_primary();
  }

  if (warp == 0) {
    if (lane == 0) {
      uint64_t policy;
      asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(policy));
      bool go = true;
      for (int i = 0; i < ntiles && go; ++i) {
        const int t = (int)blockIdx.x + i * (int)gridDim.x;
        int tm = t / tiles_n, tn = t - tm * tiles_n;
        if (kMode == 0) raster_tile(t, tiles_n, tiles_total, tm, tn);
        for (int kb = 0; kb < kb_total; ++kb) {
          // the ring's position counts K blocks over all of the CTA's tiles
          const int g = i * kb_total + kb;
          const int s = g % kStages;
          const uint32_t round = (uint32_t)(g / kStages);
          if (!mbar_wait(&empty[s], (round & 1u) ^ 1u)) {
            atomicOr(failed, 1u);
            go = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], kStageBytes);
          if (kMode == 3) {
#pragma unroll
            for (int j = 0; j < kBM / 64; ++j)
              tma_load_2d(tile_a + s * kTileABytes + j * kBoxBytes, &xmap, tm * kBM + 64 * j, kb * kBK, &full[s],
                          policy);
#pragma unroll
            for (int j = 0; j < kBN / 64; ++j)
              tma_load_2d(tile_b + s * kTileBBytes + j * kBoxBytes, &wmap, tn * kBN + 64 * j, kb * kBK, &full[s],
                          policy);
          } else {
            const int xk = (kAccum || kb < kb_half ? kb : kb - kb_half) * kBK;
            tma_load_2d(tile_a + s * kTileABytes, &xmap, xk, tm * kBM, &full[s], policy);
            tma_load_2d(tile_b + s * kTileBBytes, &wmap, kb * kBK, tn * kBN, &full[s], policy);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // the segmented modes: segments of kSegBlocks K blocks, each accumulated from zero;
      // the GPTQ update: one segment over its short K loop, per tile
      const int seg_blocks = kSegmented ? kSegBlocks : (kb_total > 0 ? kb_total : 1);
      const int nseg = (kb_total + seg_blocks - 1) / seg_blocks;
      bool ok = true;
      for (int i = 0; i < ntiles && ok; ++i) {
        const uint32_t acc = kTwoAcc ? (uint32_t)(i & 1) : 0u;
        // the accumulator's previous tile (two back) must have been read out of TMEM
        if (kTwoAcc && i >= 2 && !mbar_wait(&tacc_empty[acc], (uint32_t)((i >> 1) - 1) & 1u)) {
          atomicOr(failed, 1u);
          break;
        }
        for (int seg = 0; seg < nseg && ok; ++seg) {
          // the previous segment's partial (of this tile or the one before) must have been
          // read out of TMEM
          const int gs = i * nseg + seg;
          if (kSegmented && gs >= 1 && !mbar_wait(seg_empty, (uint32_t)(gs - 1) & 1u)) {
            atomicOr(failed, 1u);
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d = tmem_d + acc * kBN;
          const int kb0 = seg * seg_blocks, kb1 = min(kb_total, kb0 + seg_blocks);
          for (int kb = kb0; kb < kb1; ++kb) {
            const int g = i * kb_total + kb;
            const int s = g % kStages;
            const uint32_t round = (uint32_t)(g / kStages);
            if (!mbar_wait(&full[s], round & 1u)) {
              atomicOr(failed, 1u);
              ok = false;
              break;
            }
            tc_fence_after_sync();
            if (kMode == 3) {
              // MN-major: 16 K rows are two 1024-byte swizzle atoms further
              const uint64_t ad = smem_desc_mn_sw128(smem_addr(tile_a + s * kTileABytes), kBoxBytes);
              const uint64_t bd = smem_desc_mn_sw128(smem_addr(tile_b + s * kTileBBytes), kBoxBytes);
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk)
                umma_bf16(d, ad + 128 * kk, bd + 128 * kk, kIdescMN, (uint32_t)(kb > kb0 || kk > 0));
            } else {
              const uint64_t ad = smem_desc_k_sw128(smem_addr(tile_a + s * kTileABytes));
              const uint64_t bd = smem_desc_k_sw128(smem_addr(tile_b + s * kTileBBytes));
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk)
                umma_bf16(d, ad + 2 * kk, bd + 2 * kk, kIdesc, (uint32_t)(kb > kb0 || kk > 0));
            }
            umma_commit(smem_addr(&empty[s]));
          }
          // fires once every MMA issued above has completed
          if (ok) umma_commit(smem_addr(kSegmented ? seg_full : (kTwoAcc ? &tacc_full[acc] : acc_ready)));
        }
      }
    }
    __syncwarp();
  } else {
    // epilogue warps 2-9: TMEM lane quarter warp % 4 (a warp may only touch that quarter),
    // column half (warp - 2) / 4; each thread holds one tile row's half of the partial
    constexpr int kHalf = kBN / 2;
    const uint32_t quarter = (uint32_t)(warp & 3);
    const uint32_t cbase = (uint32_t)((warp - 2) >> 2) * kHalf;
    const uint32_t lane_base = (quarter * 32u) << 16;
    const int nseg = kSegmented ? (kb_total + kSegBlocks - 1) / kSegBlocks : 1;
    double acc = 0.0;
    bool alive = true;
    for (int i = 0; i < ntiles && alive; ++i) {
      const int t = (int)blockIdx.x + i * (int)gridDim.x;
      const int tm = t / tiles_n, tn = t - tm * tiles_n;
      const int64_t row = (int64_t)tm * kBM + quarter * 32 + lane;
      const int64_t col0 = (int64_t)tn * kBN + cbase;
      const uint32_t tacc = kTwoAcc ? (uint32_t)(i & 1) : 0u;
      for (int seg = 0; seg < nseg; ++seg) {
        uint64_t* ready = kSegmented ? seg_full : (kTwoAcc ? &tacc_full[tacc] : acc_ready);
        const uint32_t parity =
            kSegmented ? (uint32_t)(i * nseg + seg) & 1u : (kTwoAcc ? (uint32_t)(i >> 1) & 1u : 0u);
        if (!mbar_wait(ready, parity)) {
          atomicOr(failed, 1u);
          alive = false;
          break;
        }
        tc_fence_after_sync();
        const bool last = seg + 1 == nseg;
        uint32_t p[kHalf];
#pragma unroll
        for (int c = 0; c < kHalf; c += 32)
          tmem_ld_32x32b_x32(tmem_d + tacc * kBN + lane_base + cbase + (uint32_t)c,
                             *reinterpret_cast<uint32_t(*)[32]>(p + c));
        tmem_ld_wait();
        if ((kSegmented && (!last || kPersistent)) || kTwoAcc) {
          // the partial is in registers: the MMAs may go on with the next segment (of this
          // tile or the next), or the tile after next may use this accumulator
          tc_fence_before_sync();
          mbar_arrive(kTwoAcc ? &tacc_empty[tacc] : seg_empty);
        }
        if (kSegmented && seg > 0) {
          // fold into the running sum (TMEM columns [256, 512)), fp32 round-to-nearest
#pragma unroll
          for (int c = 0; c < kHalf; c += 32) {
            uint32_t q[32];
            tmem_ld_32x32b_x32(tmem_d + lane_base + kBN + cbase + (uint32_t)c, q);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 32; ++j)
              p[c + j] = __float_as_uint(__fadd_rn(__uint_as_float(q[j]), __uint_as_float(p[c + j])));
          }
        }
        if (kSegmented && !last) {
#pragma unroll
          for (int c = 0; c < kHalf; c += 32)
            tmem_st_32x32b_x32(tmem_d + lane_base + kBN + cbase + (uint32_t)c, *reinterpret_cast<uint32_t(*)[32]>(p + c));
          tmem_st_wait();
          continue;
        }
        if (!kAccum) {
          // the output error: the sum of squares of the complete tile
#pragma unroll
          for (int c = 0; c < kHalf; c += 32) acc += (double)sum_squares32(*reinterpret_cast<uint32_t(*)[32]>(p + c));
          continue;
        }
        if (kTwoAcc) {
          // the GPTQ update: staged 32 x 32 boxes reduce-added into C by TMA.  Row `lane`
          // of a box holds 128 bytes; the 128-byte swizzle puts its 16-byte chunk k at
          // k ^ (lane & 7), so a warp's stores hit every bank once.
          uint8_t* stage = smem + kStages * kStageBytes + 1024 + (uint32_t)(warp - 2) * kStageBufBytes;
          const int64_t row0 = (int64_t)tm * kBM + quarter * 32;
#pragma unroll
          for (int c = 0; c < kHalf; c += 32) {
            // the previous box must have been read out of the buffer
            if (lane == 0) bulk_wait_read();
            __syncwarp();
            float4* rowp = reinterpret_cast<float4*>(stage + lane * 128);
#pragma unroll
            for (int k = 0; k < 8; ++k)
              rowp[k ^ (lane & 7)] = make_float4(__uint_as_float(p[c + 4 * k]), __uint_as_float(p[c + 4 * k + 1]),
                                                 __uint_as_float(p[c + 4 * k + 2]), __uint_as_float(p[c + 4 * k + 3]));
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0 && row0 < h_rows && col0 + c < h_cols) {
              tma_reduce_add_2d(&cmap, stage, (int32_t)(col0 + c), (int32_t)row0);
              bulk_commit();
            }
          }
          continue;
        }
        // the Hessian: the tile row added into H
        if (row < h_rows) {
          float* dst = H + row * ld_h + col0;
          if (col0 + kHalf <= h_cols && ((ld_h | col0) & 3) == 0 && (reinterpret_cast<uintptr_t>(H) & 15) == 0) {
#pragma unroll
            for (int q = 0; q < kHalf / 4; ++q) {
              float4 v = reinterpret_cast<float4*>(dst)[q];
              v.x += __uint_as_float(p[4 * q]);
              v.y += __uint_as_float(p[4 * q + 1]);
              v.z += __uint_as_float(p[4 * q + 2]);
              v.w += __uint_as_float(p[4 * q + 3]);
              reinterpret_cast<float4*>(dst)[q] = v;
            }
          } else {
#pragma unroll
            for (int q = 0; q < kHalf; ++q)
              if (col0 + q < h_cols) dst[q] += __uint_as_float(p[q]);
          }
        }
      }
    }
    // the update's reduce-adds complete before the CTA ends
    if (kTwoAcc && lane == 0) bulk_wait_all();
    if (!kAccum) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, off);
      if (lane == 0) warp_sum[warp - 2] = acc;
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (kAccum) {
    // a wait that ran out makes the whole tile NaN (written after the partial sums above)
    if (*failed && warp >= 2) {
      const uint32_t quarter = (uint32_t)(warp & 3);
      for (int i = 0; i < ntiles; ++i) {
        const int t = (int)blockIdx.x + i * (int)gridDim.x;
        const int tm = t / tiles_n, tn = t - tm * tiles_n;
        const int64_t row = (int64_t)tm * kBM + quarter * 32 + lane;
        const int64_t c0 = (int64_t)tn * kBN + ((warp - 2) >> 2) * (kBN / 2);
        if (row < h_rows)
          for (int64_t c = c0; c < c0 + kBN / 2 && c < h_cols; ++c) H[row * ld_h + c] = __int_as_float(0x7FC00000);
      }
      if (threadIdx.x == 64) atomicOr(&g_output_error_flags, kErrMbarTimeout);
    }
  } else if (threadIdx.x == 0) {
    double total = ((warp_sum[0] + warp_sum[1]) + (warp_sum[2] + warp_sum[3])) +
                   ((warp_sum[4] + warp_sum[5]) + (warp_sum[6] + warp_sum[7]));
    if (*failed) {
      atomicOr(&g_output_error_flags, kErrMbarTimeout);
      total = __longlong_as_double(0x7FF8000000000000ll);
    }
    partials[blockIdx.x] = total;
  }
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_d, kCols);
  }
}

// X [tokens, n] (row stride ld_x) -> Xt [n, tokens] (row stride ld_t), 32 x 32 tiles
// through shared memory so both the reads and the writes are coalesced.
__global__ void __launch_bounds__(256) transpose_kernel(const uint16_t* __restrict__ x, int64_t tokens, int64_t n,
                                                        int64_t ld_x, uint16_t* __restrict__ xt, int64_t ld_t) {
  __shared__ uint16_t tile[32][33];
  const int64_t t0 = (int64_t)blockIdx.x * 32, c0 = (int64_t)blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 8 rows of 32 per pass
  for (int k = ty; k < 32; k += 8) {
    const int64_t t = t0 + k, c = c0 + tx;
    tile[k][tx] = (t < tokens && c < n) ? x[t * ld_x + c] : (uint16_t)0;
  }
  __syncthreads();
  for (int k = ty; k < 32; k += 8) {
    const int64_t c = c0 + k, t = t0 + tx;
    if (c < n && t < tokens) xt[c * ld_t + t] = tile[tx][k];
  }
}

// The partials summed in index order by one block (fixed tree), added to *out.
__global__ void __launch_bounds__(256) reduce_kernel(const double* __restrict__ partials, int64_t count,
                                                     double* __restrict__ out) {
  __shared__ double part[256];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < count; i += blockDim.x) s += partials[i];
  part[threadIdx.x] = s;
  __syncthreads();
  for (int step = 128; step > 0; step >>= 1) {
    if ((int)threadIdx.x < step) part[threadIdx.x] += part[threadIdx.x + step];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out += part[0];
}

}  // namespace

cudaError_t launch_residual(const void* w, int64_t m, int64_t n, const float* global_scale,
                            const uint8_t* codes, const uint8_t* packed, void* dw2, int64_t ld_dw2,
                            cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int ng = (int)(n / 16);
  const int ng_pad = (int)((n + 63) / 64 * 4);
  const int64_t slots = m * ng_pad;
  const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((slots + 255) / 256, (int64_t)info.sm_count * 8));
  residual_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4*>(w), m, ng, ng_pad, global_scale,
                                                        codes, reinterpret_cast<const uint2*>(packed),
                                                        static_cast<uint4*>(dw2), ld_dw2);
  return cudaGetLastError();
}

int64_t output_error_tiles(int64_t tokens, int64_t m) {
  return ((tokens + kBM - 1) / kBM) * ((m + kBN - 1) / kBN);
}

cudaError_t launch_output_error(const void* x, int64_t tokens, int64_t n, int64_t ld_x, const void* dw2,
                                int64_t ld_dw2, int64_t m, double* out, double* partials,
                                cudaStream_t stream) {
  EncodeTiledFn encode = nullptr;
  cudaError_t err = encode_tiled_fn(&encode);
  if (err != cudaSuccess) return err;
  const int64_t n_pad = (n + kBK - 1) / kBK * kBK;
  CUtensorMap xmap, wmap;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)n, (cuuint64_t)tokens};
    const cuuint64_t strides[1] = {(cuuint64_t)ld_x * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)(2 * n_pad), (cuuint64_t)m};
    const cuuint64_t strides[1] = {(cuuint64_t)ld_dw2 * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)kBN};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(dw2), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const cudaError_t attr_status =
      ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_kernel<0>), (int)kGemmSmemBytes);
  if (attr_status != cudaSuccess) return attr_status;
  const int64_t tiles_n = (m + kBN - 1) / kBN;
  const int64_t tiles = output_error_tiles(tokens, m);
  // persistent: one CTA per SM (the shared-memory ring and the 512 TMEM columns allow no
  // more), tiles strided; one partial per CTA
  DeviceInfo info;
  if ((err = current_device_info(&info)) != cudaSuccess) return err;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(tiles, info.sm_count));
  gemm_kernel<0><<<(unsigned)grid, kGemmThreads, kGemmSmemBytes, stream>>>(
      xmap, wmap, wmap, (int)(n_pad / kBK), (int)tiles_n, (int)tiles, partials, nullptr, 0, 0, 0);
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  reduce_kernel<<<1, 256, 0, stream>>>(partials, grid, out);
  return cudaGetLastError();
}

int64_t hessian_full_ld(int64_t tokens) { return (tokens + 7) / 8 * 8; }

cudaError_t launch_hessian_full(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* H, int64_t ld_h,
                                void* xt, cudaStream_t stream) {
  EncodeTiledFn encode = nullptr;
  cudaError_t err = encode_tiled_fn(&encode);
  if (err != cudaSuccess) return err;
  const int64_t tiles_n = (n + kBN - 1) / kBN;
  const int64_t tiles = ((n + kBM - 1) / kBM) * tiles_n;
  if ((reinterpret_cast<uintptr_t>(x) & 15) == 0 && ld_x % 8 == 0) {
    // X read as it is: 64-channel x 64-token boxes, MN-major operands (kMode 3)
    CUtensorMap map;
    const cuuint64_t dims[2] = {(cuuint64_t)n, (cuuint64_t)tokens};
    const cuuint64_t strides[1] = {(cuuint64_t)ld_x * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)kBK};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    err = ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_kernel<3>), (int)kGemmSmemBytes);
    if (err != cudaSuccess) return err;
    gemm_kernel<3><<<(unsigned)tiles, kGemmThreads, kGemmSmemBytes, stream>>>(
        map, map, map, (int)((tokens + kBK - 1) / kBK), (int)tiles_n, (int)tiles, nullptr, H, n, n, ld_h);
    return cudaGetLastError();
  }
  // X with rows that are not 16-byte aligned: transposed first (tokens contiguous per
  // channel), then both operands K-major (kMode 1)
  const int64_t ld_t = hessian_full_ld(tokens);
  const dim3 tgrid((unsigned)((tokens + 31) / 32), (unsigned)((n + 31) / 32));
  transpose_kernel<<<tgrid, 256, 0, stream>>>(static_cast<const uint16_t*>(x), tokens, n, ld_x,
                                              static_cast<uint16_t*>(xt), ld_t);
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  CUtensorMap amap, bmap;
  const cuuint64_t dims[2] = {(cuuint64_t)tokens, (cuuint64_t)n};
  const cuuint64_t strides[1] = {(cuuint64_t)ld_t * 2};
  const cuuint32_t estr[2] = {1, 1};
  const cuuint32_t abox[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
  const cuuint32_t bbox[2] = {(cuuint32_t)kBK, (cuuint32_t)kBN};
  if (encode(&amap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, xt, dims, strides, abox, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
      encode(&bmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, xt, dims, strides, bbox, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const cudaError_t attr_status =
      ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_kernel<1>), (int)kGemmSmemBytes);
  if (attr_status != cudaSuccess) return attr_status;
  gemm_kernel<1><<<(unsigned)tiles, kGemmThreads, kGemmSmemBytes, stream>>>(
      amap, bmap, bmap, (int)((tokens + kBK - 1) / kBK), (int)tiles_n, (int)tiles, nullptr, H, n, n, ld_h);
  return cudaGetLastError();
}

cudaError_t launch_gemm_accumulate(const void* a, const void* b, int64_t m, int64_t nn, int64_t k, float* C,
                                   int64_t ld_c, cudaStream_t stream, bool programmatic) {
  EncodeTiledFn encode = nullptr;
  cudaError_t err = encode_tiled_fn(&encode);
  if (err != cudaSuccess) return err;
  CUtensorMap amap, bmap, cmap;
  const cuuint64_t adims[2] = {(cuuint64_t)k, (cuuint64_t)m};
  const cuuint64_t bdims[2] = {(cuuint64_t)k, (cuuint64_t)nn};
  const cuuint64_t strides[1] = {(cuuint64_t)k * 2};
  const cuuint32_t estr[2] = {1, 1};
  const cuuint32_t abox[2] = {(cuuint32_t)kBK, (cuuint32_t)kBM};
  const cuuint32_t bbox[2] = {(cuuint32_t)kBK, (cuuint32_t)kBN};
  if (encode(&amap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a), adims, strides, abox, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
      encode(&bmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(b), bdims, strides, bbox, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  // C [m, nn] fp32 (row stride ld_c), reduce-added in 32 x 32 boxes
  const cuuint64_t cdims[2] = {(cuuint64_t)nn, (cuuint64_t)m};
  const cuuint64_t cstrides[1] = {(cuuint64_t)ld_c * 4};
  const cuuint32_t cbox[2] = {kStageCols, kStageRows};
  if ((reinterpret_cast<uintptr_t>(C) & 15) != 0 || (ld_c * 4) % 16 != 0) return cudaErrorInvalidValue;
  if (encode(&cmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, C, cdims, cstrides, cbox, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
      CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  err = ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_kernel<2>), (int)kUpdateSmemBytes);
  if (err != cudaSuccess) return err;
  const int64_t tiles_n = (nn + kBN - 1) / kBN;
  const int64_t tiles = ((m + kBM - 1) / kBM) * tiles_n;
  // persistent: one CTA per SM (the shared-memory ring allows no more), tiles strided
  DeviceInfo info;
  if ((err = current_device_info(&info)) != cudaSuccess) return err;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(tiles, info.sm_count));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kGemmThreads, 1, 1);
  cfg.dynamicSmemBytes = kUpdateSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = programmatic ? 1 : 0;
  err = cudaLaunchKernelEx(&cfg, gemm_kernel<2>, amap, bmap, cmap, (int)((k + kBK - 1) / kBK), (int)tiles_n,
                           (int)tiles, (double*)nullptr, C, m, nn, ld_c);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t read_output_error_device_error(uint32_t* flags) {
  uint32_t v = 0;
  cudaError_t err = cudaMemcpyFromSymbol(&v, g_output_error_flags, sizeof v);
  if (err != cudaSuccess) return err;
  *flags = v;
  if (v) {
    const uint32_t zero = 0;
    err = cudaMemcpyToSymbol(g_output_error_flags, &zero, sizeof zero);
  }
  return err;
}

}  // namespace hscale
