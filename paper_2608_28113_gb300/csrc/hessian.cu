// hessian.cu -- diagonal-Hessian proxy h_j += sum_t x_tj^2 (Sec. 3.2, Eq. 4) on sm_103a.
//
// HBM-bound column sum of squares over a bf16 token chunk X[tokens, ld], with the squares
// taken on the tensor cores.
//
// Why the tensor cores: the pass streams X at the HBM rate and needs only one multiply-add
// per element, but it is meant to run alongside the ALU-bound scale search, whose warps
// keep the FMA pipe busy.  Measured on a GB300, an FMA-based version of this kernel made
// almost no progress while such warps were resident (its own FMAs waited behind theirs).
// Here the arithmetic goes to the otherwise idle tensor cores: a CTA's SIMT work is one
// thread issuing TMA loads, one issuing MMAs, and a short epilogue every 1024 tokens.
//
// Layout of the work
//   * A CTA owns a 128-channel column tile and a contiguous run of tokens.  A producer
//     thread streams the run into a ring of shared-memory stages with 2-D TMA tensor loads
//     (64 tokens x 128 channels = 16 KB per stage, two 64-channel boxes with 128-byte
//     swizzling, 4 stages in flight, L2 evict-first).
//   * One thread issues, per stage, four tcgen05 MMAs D += A^T A (M = N = 128, K = 16
//     tokens each) with A the stage itself taken as an MN-major operand (channels
//     contiguous), so D = X_tile^T X_tile accumulates in fp32 in tensor memory and its
//     diagonal D[j][j] is the column sum of squares.  The other 127 / 128 of D is not
//     used; the tensor cores have the throughput to spare (about 40 % of their peak at
//     the HBM rate).
//   * The token run is cut into accumulation segments of 1024 tokens: each accumulates
//     from zero in tensor memory; four epilogue warps read the diagonal (thread t of the
//     warp of lane quarter q takes lane 32 q + t, column 32 q + t) and add it to a running
//     fp32 sum in registers, then release the accumulator for the next segment.
//   * The token range of a tile is split over the CTAs of one thread-block cluster
//     (1, 2, 4 or 8 CTAs, so a launch holds about one CTA per SM).  The CTAs of a cluster
//     reduce their sums through distributed shared memory: the kernel needs no global
//     scratch, no atomics and no second launch.
//   * Launches use programmatic dependent launch.  By default a call's kernel waits
//     (griddepcontrol.wait) for the kernel before it on the stream before it reads X, so
//     X may come from a kernel that lets its dependents start early.  When the caller
//     declares X complete (nothing still running writes it), the kernel streams X at once,
//     while the previous kernel finishes, and waits only before it reads and writes h.  A
//     CTA lets the next kernel start only once it holds its tensor memory, so a CTA of the
//     next grid that waits for this grid never holds columns that a CTA of this grid still
//     needs.
//   * Rows past the end of the chunk read as zero (TMA out-of-bounds fill), so ragged
//     chunks and ragged column tiles need no special cases.
// Determinism and accuracy
//   x^2 of a bf16 value is exact in fp32.  The tensor cores accumulate in fp32 with a
//   small error that grows with the accumulation length (measured: low by about 0.9 units
//   in the last place per 16-token step), which the 1024-token segments bound to about
//   2^-18 relative; segments, the cluster's CTAs and the call's total then meet in fp32
//   round-to-nearest adds in a fixed order.  Every run gives the same bits.
// Failure reporting
//   A wait that runs out of polls (it cannot on a healthy GPU) sets the library's device
//   error flag and turns the affected h entries into NaN instead of hanging; the CTA lets
//   its copies and MMAs in flight finish and frees its tensor memory before it returns.
#include <cooperative_groups.h>
#include <cuda.h>

#include <algorithm>
#include <mutex>

#include "hscale_device.cuh"
#include "hscale_internal.h"
#include "tcgen05.cuh"
#include "tma.cuh"

namespace cg = cooperative_groups;

namespace hscale {

__device__ uint32_t g_device_error = 0;

namespace {

constexpr int kTileCols = 128;                            // channels per CTA tile: M = N = 128
constexpr int kBoxCols = 64;                              // channels per TMA box (128 bytes)
constexpr int kStageRows = 64;                            // tokens per stage: four K = 16 MMAs
constexpr int kStages = 4;
constexpr uint32_t kBoxBytes = kBoxCols * kStageRows * 2;  // 8 KB
constexpr uint32_t kStageBytes = 2 * kBoxBytes;            // 16 KB
constexpr int kSegStages = 16;                            // 1024 tokens per accumulation segment
constexpr int kEpiWarps = 4;                              // one per TMEM lane quarter
constexpr int kThreads = (2 + kEpiWarps) * 32;            // TMA warp, MMA warp, epilogue warps
constexpr uint32_t kTmemCols = 128;
constexpr uint32_t kIdesc = idesc_bf16_f32_mn(kTileCols, kTileCols);
constexpr int kSmemBytes = kStages * (int)kStageBytes + 1024;  // the ring, 1 KB aligned
constexpr int kMaxCluster = 8;
constexpr uint32_t kPollSlice = 256;  // polls between checks of the CTA's failure flag

// Bounded wait that gives up early once another thread of the CTA has reported a failure
// (try_wait: the waiting warp is suspended between polls).  The epilogue warps wait this way.
__device__ __forceinline__ bool wait_or_fail(uint64_t* bar, uint32_t parity, const int* bad) {
  for (uint32_t i = 0; i < kMbarPollLimit / kPollSlice; ++i) {
    if (mbar_wait_bounded(bar, parity, kPollSlice)) return true;
    if (*(const volatile int*)bad) return false;
  }
  return false;
}

// The same as a spin on test_wait, which never suspends the thread: the TMA and MMA threads
// wait this way, so that they issue again as soon as their barrier completes even while the
// search's warps keep the SM busy (measured: decoder step 1.187 against 1.197 ms, the search
// beside it unchanged).  At most 2^26 polls, well over a tenth of a second.
__device__ __forceinline__ bool spin_or_fail(uint64_t* bar, uint32_t parity, const int* bad) {
  const uint32_t a = smem_addr(bar);
  for (uint32_t i = 0; i < kMbarPollLimit * 4u; ++i) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(a), "r"(parity)
        : "memory");
    if (done) return true;
    if ((i & 255u) == 255u && *(const volatile int*)bad) return false;
  }
  return false;
}

template <int CS>
__global__ void __launch_bounds__(kThreads, 3)
hessian_colsumsq_kernel(const __grid_constant__ CUtensorMap xmap, int64_t row0, int64_t rows,
                        int n, float* __restrict__ h, int64_t rows_per_cta, int x_ready) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t seg_full, seg_empty, mma_done;
  __shared__ uint32_t tmem_slot;
  __shared__ float cta_part[kTileCols];
  __shared__ int s_bad;

  cg::cluster_group cluster = cg::this_cluster();
  const unsigned crank = cluster.block_rank();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r0 = row0 + (int64_t)crank * rows_per_cta;
  const int64_t r1 = min(row0 + rows, r0 + rows_per_cta);
  const int nst = r1 > r0 ? (int)((r1 - r0 + kStageRows - 1) / kStageRows) : 0;
  const int nseg = (nst + kSegStages - 1) / kSegStages;
  const int x0 = blockIdx.y * kTileCols;
  // a box wholly right of column n is not loaded: it only feeds entries of D off the
  // diagonal of valid channels
  const int boxes = x0 + kBoxCols < n ? 2 : 1;

  if (tid == 0) {
    prefetch_tensormap(&xmap);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&seg_full, 1);
    mbar_init(&seg_empty, kEpiWarps * 32);
    mbar_init(&mma_done, 1);
    mbar_fence_init();
    s_bad = 0;
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(&tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_d = tmem_slot;
  // X may still be being written by the previous kernel on the stream: read it only once
  // that kernel has finished and its writes are visible
  if (!x_ready) pdl_wait_primary();
  // every CTA of this grid holds its tensor memory by now (see the header)
  pdl_launch_dependents();

  float acc = 0.0f;
  if (warp == 0) {
    // producer: refills each stage as soon as the MMAs reading it have completed
    if (lane == 0) {
      const uint64_t policy = l2_evict_first_policy();
      const uint32_t bytes = (uint32_t)boxes * kBoxBytes;
      int issued = 0;
      for (; issued < nst; ++issued) {
        const int s = issued % kStages;
        if (issued >= kStages && !spin_or_fail(&empty_bar[s], (uint32_t)(issued / kStages - 1) & 1u, &s_bad)) {
          s_bad = 1;
          break;
        }
        mbar_arrive_expect_tx(&full_bar[s], bytes);
        const int32_t y = (int32_t)(r0 + (int64_t)issued * kStageRows);
        for (int j = 0; j < boxes; ++j)
          tma_load_2d(ring + (size_t)s * kStageBytes + j * kBoxBytes, &xmap, x0 + j * kBoxCols, y, &full_bar[s],
                      policy);
      }
      if (*(volatile int*)&s_bad) {
        // let the copies still in flight land before the CTA's shared memory goes away (the
        // loads of earlier uses of a stage completed before the stage was refilled)
        for (int j = issued > kStages ? issued - kStages : 0; j < issued; ++j)
          mbar_wait(&full_bar[j % kStages], (uint32_t)(j / kStages) & 1u);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      for (int seg = 0; seg < nseg && ok; ++seg) {
        // the previous segment's diagonal has been read out of tensor memory
        if (seg >= 1 && !spin_or_fail(&seg_empty, (uint32_t)(seg - 1) & 1u, &s_bad)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const int i0 = seg * kSegStages, i1 = min(nst, i0 + kSegStages);
        for (int i = i0; i < i1; ++i) {
          const int s = i % kStages;
          if (!spin_or_fail(&full_bar[s], (uint32_t)(i / kStages) & 1u, &s_bad)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          // A = B = the stage, MN-major; 16 tokens further is two 1024-byte swizzle atoms
          const uint64_t desc = smem_desc_mn_sw128(smem_addr(ring + (size_t)s * kStageBytes), kBoxBytes);
#pragma unroll
          for (int kk = 0; kk < kStageRows / 16; ++kk)
            umma_bf16(tmem_d, desc + 128 * kk, desc + 128 * kk, kIdesc, (uint32_t)(i > i0 || kk > 0));
          umma_commit(smem_addr(&empty_bar[s]));
        }
        if (ok) umma_commit(smem_addr(&seg_full));
      }
      if (!ok) s_bad = 1;
      // every MMA issued above has completed before the tensor memory is freed
      umma_commit(smem_addr(&mma_done));
      mbar_wait(&mma_done, 0u);
    }
    __syncwarp();
  } else {
    // epilogue: warp w reads TMEM lane quarter q = w % 4; its thread t owns channel 32 q + t,
    // whose square sum is the diagonal entry at lane 32 q + t, column 32 q + t
    const int q = warp & 3;
    const uint32_t taddr = tmem_d + ((uint32_t)(32 * q) << 16) + (uint32_t)(32 * q);
    for (int seg = 0; seg < nseg; ++seg) {
      if (!wait_or_fail(&seg_full, (uint32_t)seg & 1u, &s_bad)) {
        s_bad = 1;
        break;
      }
      tc_fence_after_sync();
      uint32_t r[32];
      tmem_ld_32x32b_x32(taddr, r);
      tmem_ld_wait();
      float v = 0.0f;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (lane == j) v = __uint_as_float(r[j]);
      acc = __fadd_rn(acc, v);
      tc_fence_before_sync();
      mbar_arrive(&seg_empty);
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_d, kTmemCols);
  }
  const bool bad = *(volatile int*)&s_bad != 0;
  if (bad && tid == 0) atomicOr(&g_device_error, kErrMbarTimeout);
  if (warp >= 2) cta_part[32 * (warp & 3) + lane] = bad ? __int_as_float(0x7FC00000) : acc;

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
      ensure_dynamic_smem(reinterpret_cast<const void*>(hessian_colsumsq_kernel<CS>), kSmemBytes);
  if (attr_status != cudaSuccess) return attr_status;
  int64_t rows_per_cta = (tokens + CS - 1) / CS;
  rows_per_cta = (rows_per_cta + kStageRows - 1) / kStageRows * kStageRows;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(CS, tiles, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
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
  cudaError_t err = cudaLaunchKernelEx(&cfg, hessian_colsumsq_kernel<CS>, map, (int64_t)0, tokens, n, h,
                                       rows_per_cta, x_ready ? 1 : 0);
  if (err != cudaSuccess) return err;
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
  const cuuint32_t box[2] = {(cuuint32_t)kBoxCols, (cuuint32_t)kStageRows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides,
                      box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;

  const int tiles = (int)((n + kTileCols - 1) / kTileCols);
  // at most about one CTA per SM per launch: with programmatic dependent launch,
  // consecutive chunk launches share the GPU, so the next chunk streams while this one
  // drains; the token split keeps at least four stages per CTA
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
  // every kernel with large dynamic shared memory also asks for the whole carveout, so an
  // SM it lands on first is not split in favour of L1
  if (err == cudaSuccess)
    err = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared);
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
