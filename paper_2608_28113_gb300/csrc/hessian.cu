// hessian.cu -- diagonal-Hessian proxy h_j += sum_t x_tj^2 (Sec. 3.2, Eq. 4) on sm_103a.
//
// HBM-bound column sum of squares over a bf16 token chunk X[tokens, ld].
//
// Layout of the work
//   * A CTA owns a 64-channel column tile (128 bytes of every row) and a contiguous
//     run of tokens.  A producer warp (one thread) streams the run into a ring of
//     shared-memory stages with 2-D TMA tensor loads (64 channels x 128 rows = 16 KB per
//     stage, 4 stages in flight per CTA, L2 evict-first), refilling each stage as soon as
//     the consumers release it; the CTA's 256 consumer threads (32 row phases x 8
//     16-byte vectors) read each stage back with conflict-free 128-bit shared loads
//     and accumulate in fp32.  mbarriers order the ring; every wait is bounded.
//   * The token range of a tile is split over the CTAs of one thread-block cluster
//     (1, 2, 4 or 8 CTAs, so a launch holds about one CTA per SM).  The CTAs
//     of a cluster reduce their partial sums through distributed shared memory: the
//     kernel needs no global scratch, no atomics and no second launch.
//   * Launches use programmatic dependent launch.  By default a call's kernel waits
//     (griddepcontrol.wait) for the kernel before it on the stream before it reads X, so
//     X may come from a kernel that lets its dependents start early; it then lets its
//     own dependents start.  When the caller declares X complete (nothing still running
//     writes it), and for the second and later launches of one call (whose predecessor
//     is this call's own launch), the kernel streams X at once, while the previous
//     kernel finishes, and waits only before it reads and writes h.
//   * Rows past the end of the chunk read as zero (TMA out-of-bounds fill), so ragged
//     chunks and ragged column tiles need no special cases.
// Determinism and accuracy
//   x^2 of a bf16 value is exact in fp32.  Each thread adds at most 1024 squares in
//   token order; partials then meet in fixed-order pairwise trees (4 phases in a warp,
//   8 warps in the CTA, the cluster's CTAs), and the total is added to h once.  Every
//   run gives the same bits, and a call adds a relative error of at most
//   (1024 + 2 + 3 + 3 + 1) * 2^-24 to h.
// Failure reporting
//   A wait that runs out of polls (it cannot on a healthy GPU) sets the library's
//   device error flag and turns the affected h entries into NaN instead of hanging.
#include <cooperative_groups.h>
#include <cuda.h>

#include <algorithm>
#include <mutex>

#include "hscale_device.cuh"
#include "hscale_internal.h"
#include "tma.cuh"

namespace cg = cooperative_groups;

namespace hscale {

__device__ uint32_t g_device_error = 0;

namespace {

constexpr int kTileCols = 64;                       // channels per CTA tile (128 bytes)
constexpr int kWarps = 8;                           // consumer warps
constexpr int kThreads = (kWarps + 1) * 32;         // and one producer warp
constexpr int kPhases = 32;                         // rows read side by side
constexpr int kStageRows = 128;
constexpr int kStages = 4;
constexpr uint32_t kStageBytes = kStageRows * kTileCols * 2;
constexpr size_t kRingBytes = (size_t)kStages * kStageBytes;
constexpr int64_t kMaxRowsPerCta = 1024 * kPhases;  // <= 1024 sequential adds per thread
constexpr int kMaxCluster = 8;

// acc += x^2 for the two bf16 values of a 32-bit word, taken straight from its halves by
// the mixed-precision FMA (a bf16 x bf16 product is exact in fp32; the add rounds once, as
// an fp32 FMA of the widened values would): one instruction per element, no unpacking.
__device__ __forceinline__ void accum_sq2(float& lo_acc, float& hi_acc, uint32_t pair) {
  asm("{\n\t.reg .b16 l, h;\n\tmov.b32 {l, h}, %2;\n\t"
      "fma.rn.f32.bf16 %0, l, l, %0;\n\t"
      "fma.rn.f32.bf16 %1, h, h, %1;\n\t}"
      : "+f"(lo_acc), "+f"(hi_acc)
      : "r"(pair));
}

__device__ __forceinline__ void accum_sq8(float (&acc)[8], const uint4& v) {
  accum_sq2(acc[0], acc[1], v.x);
  accum_sq2(acc[2], acc[3], v.y);
  accum_sq2(acc[4], acc[5], v.z);
  accum_sq2(acc[6], acc[7], v.w);
}

template <int CS>
__global__ void __launch_bounds__(kThreads, 4)
hessian_colsumsq_kernel(const __grid_constant__ CUtensorMap xmap, int64_t row0, int64_t rows,
                        int n, float* __restrict__ h, int64_t rows_per_cta, int x_ready) {
  extern __shared__ __align__(1024) uint8_t ring[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ float warp_part[kWarps][kTileCols];
  __shared__ float cta_part[kTileCols];
  __shared__ int s_bad;

  cg::cluster_group cluster = cg::this_cluster();
  const unsigned crank = cluster.block_rank();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int v = tid & 7, p = tid >> 3;
  const int64_t r0 = row0 + (int64_t)crank * rows_per_cta;
  const int64_t r1 = min(row0 + rows, r0 + rows_per_cta);
  const int nst = r1 > r0 ? (int)((r1 - r0 + kStageRows - 1) / kStageRows) : 0;
  const int x0 = blockIdx.y * kTileCols;

  if (tid == 0) {
    prefetch_tensormap(&xmap);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kWarps);
    }
    mbar_fence_init();
    s_bad = 0;
  }
  __syncthreads();
  // X may still be being written by the previous kernel on the stream: read it only once
  // that kernel has finished and its writes are visible
  if (!x_ready) pdl_wait_primary();
  pdl_launch_dependents();

  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (warp == kWarps) {
    // producer: one thread refills each stage as soon as the consumers have released it, so
    // a consumer warp that is slow to be scheduled delays no other stage's load
    if (lane == 0) {
      const uint64_t policy = l2_evict_first_policy();
      int issued = 0;
      for (; issued < nst; ++issued) {
        const int s = issued % kStages;
        if (issued >= kStages &&
            (*(volatile int*)&s_bad || !mbar_wait(&empty_bar[s], (uint32_t)(issued / kStages - 1) & 1u))) {
          s_bad = 1;
          break;
        }
        mbar_arrive_expect_tx(&full_bar[s], kStageBytes);
        tma_load_2d(ring + (size_t)s * kStageBytes, &xmap, x0, (int32_t)(r0 + issued * kStageRows), &full_bar[s],
                    policy);
      }
      if (*(volatile int*)&s_bad) {
        // let the copies still in flight land before the CTA's shared memory goes away (the
        // loads of earlier uses of a stage completed before the stage was refilled)
        for (int j = issued > kStages ? issued - kStages : 0; j < issued; ++j)
          mbar_wait(&full_bar[j % kStages], (uint32_t)(j / kStages) & 1u);
        atomicOr(&g_device_error, kErrMbarTimeout);
      }
    }
  } else {
    for (int i = 0; i < nst; ++i) {
      const int s = i % kStages;
      const uint32_t par = (uint32_t)(i / kStages) & 1u;
      bool ok = !*(volatile int*)&s_bad;
      if (ok && !mbar_wait(&full_bar[s], par)) {
        ok = false;
        s_bad = 1;
      }
      if (ok) {
        const uint8_t* st = ring + (size_t)s * kStageBytes + p * 128 + v * 16;
#pragma unroll
        for (int rr = 0; rr < kStageRows / kPhases; ++rr)
          accum_sq8(acc, *reinterpret_cast<const uint4*>(st + rr * kPhases * 128));
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);
    }
  }

  // phases 4w..4w+3 of a warp: lane bit 3 is phase bit 0, lane bit 4 is phase bit 1
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    float t = acc[k];
    t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, 8));
    t = __fadd_rn(t, __shfl_xor_sync(0xFFFFFFFFu, t, 16));
    acc[k] = t;
  }
  if (lane < 8 && warp < kWarps) {
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
    cta_part[tid] = s_bad ? __int_as_float(0x7FC00000) : s[0];
  }

  pdl_wait_primary();  // the previous chunk's kernel has finished writing h
  if constexpr (CS == 1) {
    __syncthreads();
    if (tid < kTileCols) {
      const int col = x0 + tid;
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
      const int col = x0 + tid;
      if (col < n) h[col] = __fadd_rn(h[col], s[0]);
    }
    cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
  }
}

// ---------------------------------------------------------------- host side
template <int CS>
cudaError_t launch_cs(const CUtensorMap& map, int64_t tokens, int n, float* h, int tiles, bool x_ready,
                      cudaStream_t stream) {
  const cudaError_t attr_status =
      ensure_dynamic_smem(reinterpret_cast<const void*>(hessian_colsumsq_kernel<CS>), (int)kRingBytes);
  if (attr_status != cudaSuccess) return attr_status;
  const int64_t rows_per_launch = kMaxRowsPerCta * CS;
  for (int64_t t0 = 0; t0 < tokens; t0 += rows_per_launch) {
    const int64_t t = std::min(tokens - t0, rows_per_launch);
    int64_t rows_per_cta = (t + CS - 1) / CS;
    rows_per_cta = (rows_per_cta + kStageRows - 1) / kStageRows * kStageRows;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CS, tiles, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kRingBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    // a later launch of this call follows this call's own launch, which reads X only
    const int ready = (x_ready || t0 > 0) ? 1 : 0;
    cudaError_t err = cudaLaunchKernelEx(&cfg, hessian_colsumsq_kernel<CS>, map, t0, t, n, h,
                                         rows_per_cta, ready);
    if (err != cudaSuccess) return err;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_hessian(const void* x, int64_t tokens, int64_t n, int64_t ld_x, float* h, bool x_ready,
                           cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  EncodeTiledFn encode = nullptr;
  err = encode_tiled_fn(&encode);
  if (err != cudaSuccess) return err;

  CUtensorMap map;
  const cuuint64_t dims[2] = {(cuuint64_t)n, (cuuint64_t)tokens};
  const cuuint64_t strides[1] = {(cuuint64_t)ld_x * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kTileCols, (cuuint32_t)kStageRows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides,
                      box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;

  const int tiles = (int)((n + kTileCols - 1) / kTileCols);
  // at most about one CTA per SM per launch: with programmatic dependent launch,
  // consecutive chunk launches share the GPU, so the next chunk streams while this one
  // drains (q_proj, 8192-token chunks, 64 tiles: cluster size 1 gives 10.2 us per chunk,
  // 2 (this rule) 9.8, 4 9.9, 8 11.2)
  const int64_t target = (int64_t)info.sm_count;
  int cs = 1;
  while (cs < kMaxCluster && (int64_t)tiles * cs * 2 <= target && (int64_t)cs * 2 * kStageRows * 4 <= tokens)
    cs *= 2;
  switch (cs) {
    case 1: return launch_cs<1>(map, tokens, (int)n, h, tiles, x_ready, stream);
    case 2: return launch_cs<2>(map, tokens, (int)n, h, tiles, x_ready, stream);
    case 4: return launch_cs<4>(map, tokens, (int)n, h, tiles, x_ready, stream);
    default: return launch_cs<8>(map, tokens, (int)n, h, tiles, x_ready, stream);
  }
}

// h[j] = (((p_0[j] + p_1[j]) + p_2[j]) + ...) + p_{parts-1}[j]: the partial sums of the ranks
// that each took a share of the calibration tokens, added in rank order with fp32 round-to-
// nearest adds, so every rank that runs this on the gathered partials gets the same bits.
__global__ void __launch_bounds__(256) sum_partials_kernel(const float* __restrict__ partials, int64_t parts,
                                                           int64_t n, int64_t ld, float* __restrict__ h) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < n; j += stride) {
    float s = partials[j];
    for (int64_t r = 1; r < parts; ++r) s = __fadd_rn(s, partials[r * ld + j]);
    h[j] = s;
  }
}

cudaError_t launch_sum_partials(const float* partials, int64_t parts, int64_t n, int64_t ld, float* h,
                                cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((n + 255) / 256, (int64_t)info.sm_count * 8));
  sum_partials_kernel<<<(unsigned)blocks, 256, 0, stream>>>(partials, parts, n, ld, h);
  return cudaGetLastError();
}

cudaError_t ensure_dynamic_smem(const void* func, int bytes) {
  static std::mutex mu;
  static const void* done_func[256];
  static int done_dev[256];
  static int done_count = 0;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < done_count; ++i)
    if (done_func[i] == func && done_dev[i] == dev) return cudaSuccess;
  err = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (err == cudaSuccess && done_count < 256) {
    done_func[done_count] = func;
    done_dev[done_count] = dev;
    ++done_count;
  }
  return err;
}

cudaError_t encode_tiled_fn(EncodeTiledFn* out) {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  static cudaError_t status = cudaSuccess;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    status = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q);
    if (status == cudaSuccess && q != cudaDriverEntryPointSuccess) status = cudaErrorNotSupported;
    fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  *out = fn;
  return status;
}

cudaError_t read_hessian_device_error(uint32_t* flags) {
  uint32_t v = 0;
  cudaError_t err = cudaMemcpyFromSymbol(&v, g_device_error, sizeof v);
  if (err != cudaSuccess) return err;
  *flags = v;
  if (v) {
    const uint32_t zero = 0;
    err = cudaMemcpyToSymbol(g_device_error, &zero, sizeof zero);
  }
  return err;
}

}  // namespace hscale
