// gptq.cu -- GPTQ with H-Scale as the local quantizer (Algorithm 3) on sm_103a.
//
//   (the damped inverse-Cholesky factor U is formed in factor.cu)
//   block_kernel      four lanes per 16-element group of a block of B columns of the running
//                     fp32 weights: the RTN code (Eq. 7) of the current weights, the exact
//                     H-Scale search over the window (Algorithm 1, exact E2M1 decisions, the
//                     tie rule of the search), the codes and packed nibbles, and the
//                     propagated errors E = (W - W_hat) / U_jj
//   update            W[:, i+B:] -= E U[i:i+B, i+B:] with fp32-level accuracy on the tensor
//                     cores (three-way bf16 splits, six products, one GEMM)
#include <algorithm>
#include <cstdio>
#include <mutex>
#include <vector>

#include <cuda_bf16.h>

#include "hscale_device.cuh"
#include "hscale_internal.h"

namespace hscale {
namespace {

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

// Four lanes (a quad) per group: each scores every fourth candidate of the window with exact
// decisions, the quad keeps the best under the search's tie rule (a total order, so every
// lane ends with the same code), and each lane writes the nibbles of four of the group's
// elements and their scaled errors E = (w - w_hat) / U_jj, split, into the update's A
// operand [m, 6B]: A' = [-E1 | -E1 | -E2 | -E1 | -E2 | -E3], four bf16 (8 bytes) per segment.
__global__ void __launch_bounds__(128) block_kernel(const float* __restrict__ W, int64_t m, int64_t n, int64_t col0,
                                                    int B, const float* __restrict__ h, const float* __restrict__ U,
                                                    const float* __restrict__ global_scale, int down, int up,
                                                    uint8_t* __restrict__ codes, uint2* __restrict__ packed,
                                                    uint16_t* __restrict__ A) {
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
    uint16_t ep[3][4];   // the three bf16 parts of -E for this lane's four elements
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = 4 * q + t;
      const float av = __fmul_rn(fabsf(wv[t]), d.pw);
      const uint32_t k = e2m1_code(av, inv, l, d.sgk);
      const uint32_t neg = signbit(wv[t]) ? 1u : 0u;
      part |= ((neg << 3) | k) << (4 * (j & 7));
      float what = __fmul_rn(d.sg, __fmul_rn(e2m1_from_raw(k << 22), l));  // s_g (l q), l q exact
      if (neg) what = -what;
      const float e = __fdiv_rn(__fsub_rn(wv[t], what), U[(col + j) * n + col + j]);
      uint16_t pp[3];
      split3(-e, pp);
      ep[0][t] = pp[0];
      ep[1][t] = pp[1];
      ep[2][t] = pp[2];
    }
    if (active) {
      uint2 v[3];
#pragma unroll
      for (int p3 = 0; p3 < 3; ++p3)
        v[p3] = make_uint2((uint32_t)ep[p3][0] | ((uint32_t)ep[p3][1] << 16),
                           (uint32_t)ep[p3][2] | ((uint32_t)ep[p3][3] << 16));
      uint2* row = reinterpret_cast<uint2*>(A + r * 6 * (int64_t)B + 16 * i + 4 * q);
      const int seg = B / 4;  // one segment, in 8-byte words
      row[0] = v[0];
      row[seg] = v[0];
      row[2 * seg] = v[1];
      row[3 * seg] = v[0];
      row[4 * seg] = v[1];
      row[5 * seg] = v[2];
    }
    const uint32_t word = part | __shfl_xor_sync(0xFFFFFFFFu, part, 1);  // lanes 0-1: word 0, 2-3: word 1
    const uint32_t other = __shfl_xor_sync(0xFFFFFFFFu, word, 2);
    if (active && q == 0) {
      codes[r * (n / 16) + col / 16] = (uint8_t)bc;
      packed[r * (n / 16) + col / 16] = make_uint2(word, other);
    }
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
namespace {

// ---------------------------------------------------------------- the look-ahead stream
// Calls that work ahead (the block loop, the factor) run part of their work on a second
// stream.  The stream and its events are created once per device context and reused; a
// mutex keeps calls from enqueuing at the same time, so one call's events are never
// re-recorded while another call still has waits to enqueue on them.
struct LookAhead {
  cudaStream_t side = nullptr;
  cudaEvent_t ev[kLookAheadEvents] = {};
  unsigned long long ctx = 0;
};
constexpr int kMaxLookDevices = 64;
std::mutex g_look_mu;
LookAhead g_look[kMaxLookDevices];

}  // namespace

cudaError_t acquire_look_ahead(cudaStream_t stream, LookAheadLease* lease) {
  lease->lock = std::unique_lock<std::mutex>(g_look_mu);
  lease->side = nullptr;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (dev < 0 || dev >= kMaxLookDevices) return cudaSuccess;
  unsigned long long id = 0;
  if ((err = current_context_id(&id)) != cudaSuccess) return err;
  LookAhead& L = g_look[dev];
  if (L.side == nullptr || L.ctx != id) {
    // creating them is not allowed while the stream is being captured
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if ((err = cudaStreamIsCapturing(stream, &cap)) != cudaSuccess) return err;
    if (cap != cudaStreamCaptureStatusNone) return cudaSuccess;
    L = LookAhead{};  // the handles of an earlier context went with it
    if ((err = cudaStreamCreateWithFlags(&L.side, cudaStreamNonBlocking)) != cudaSuccess) return err;
    for (cudaEvent_t& e : L.ev)
      if ((err = cudaEventCreateWithFlags(&e, cudaEventDisableTiming)) != cudaSuccess) return err;
    L.ctx = id;
  }
  lease->side = L.side;
  for (int i = 0; i < kLookAheadEvents; ++i) lease->ev[i] = L.ev[i];
  return cudaSuccess;
}

// Algorithm 3's block loop.  Per block of B columns: the quantizer (block_kernel) writes
// the block's codes and nibbles and its scaled errors E, split into the update's A operand
// A'; then the running weights right of the block take the update W[:, c1:] += (-E)
// U[block, c1:] as one tcgen05 GEMM over the three-way bf16 splits of E and U
// (split_u_kernel writes U's, B'; K = 6 B).
//
// Look-ahead: the update is split into the next block's B columns (on the caller's
// stream, right after the block) and the rest (on a second stream).  The next block's
// quantization needs only the former, so it runs alongside the latter; U's split for a
// block is made one block ahead on the second stream.  Events order the two streams:
//   - block b reads its columns after the second stream's update of block b - 2;
//   - the next-columns update of block b follows the second stream's update of block
//     b - 1, which adds into the same columns, so every weight receives its updates in
//     block order, as in a one-stream loop, and every run gives the same bits;
//   - the split operands are double-buffered (A' and B' of block b in buffer b % 2) and
//     each buffer is rewritten only after both updates that read it.
// A6 and B6 hold two buffers each: A' [m, 6 B] and B' [n, 6 B] bf16.
cudaError_t launch_gptq_hscale(const void* w, int64_t m, int64_t n, const float* U, const float* h,
                               const float* global_scale, const uint8_t* dead, int block, int down, int up,
                               uint8_t* codes, uint8_t* packed, float* Wf, uint16_t* A6, uint16_t* B6,
                               cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = current_device_info(&info);
  if (err != cudaSuccess) return err;
  const int64_t B = block, nb = n / block;
  const unsigned cvt_blocks = (unsigned)std::min<int64_t>((m * n + 255) / 256, (int64_t)info.sm_count * 16);
  to_fp32_kernel<<<cvt_blocks, 256, 0, stream>>>(static_cast<const uint16_t*>(w), m, n, dead, Wf);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  const int64_t groups = m * (B / 16);
  const unsigned qb = (unsigned)std::min<int64_t>((groups * 4 + 127) / 128, (int64_t)info.sm_count * 16);
  uint16_t* Abuf[2] = {A6, A6 + m * 6 * B};
  uint16_t* Bbuf[2] = {B6, B6 + n * 6 * B};
  auto quantize = [&](int64_t b, cudaStream_t s) {
    block_kernel<<<qb, 128, 0, s>>>(Wf, m, n, b * B, block, h, U, global_scale, down, up, codes,
                                    reinterpret_cast<uint2*>(packed), Abuf[b & 1]);
    return cudaGetLastError();
  };
  auto split_u = [&](int64_t b, cudaStream_t s) {
    const int64_t c1 = (b + 1) * B, nn = n - c1;
    split_u_kernel<<<dim3((unsigned)((nn + 31) / 32), (unsigned)((B + 31) / 32)), 256, 0, s>>>(U, n, b * B, block, c1,
                                                                                                Bbuf[b & 1]);
    return cudaGetLastError();
  };

  LookAheadLease L;
  if (nb > 1 && (err = acquire_look_ahead(stream, &L)) != cudaSuccess) return err;
  if (L.side == nullptr) {
    // one stream: quantize, split, update, block after block
    if (L.lock.owns_lock()) L.lock.unlock();
    for (int64_t b = 0; b < nb; ++b) {
      if ((err = quantize(b, stream)) != cudaSuccess) return err;
      if (b + 1 == nb) break;
      const int64_t c1 = (b + 1) * B, nn = n - c1;
      if ((err = split_u(b, stream)) != cudaSuccess) return err;
      if ((err = launch_gemm_accumulate(Abuf[b & 1], Bbuf[b & 1], m, nn, 6 * B, Wf + c1, n, stream)) != cudaSuccess)
        return err;
    }
    return cudaSuccess;
  }

  cudaStream_t side = L.side;
  cudaEvent_t fork = L.ev[0], join = L.ev[1];
  cudaEvent_t ev_q[2] = {L.ev[2], L.ev[3]}, ev_su[2] = {L.ev[4], L.ev[5]};
  cudaEvent_t ev_ga[2] = {L.ev[6], L.ev[7]}, ev_gb[2] = {L.ev[8], L.ev[9]};
  if ((err = cudaEventRecord(fork, stream)) != cudaSuccess) return err;
  if ((err = cudaStreamWaitEvent(side, fork, 0)) != cudaSuccess) return err;
  if ((err = split_u(0, side)) != cudaSuccess) return err;
  if ((err = cudaEventRecord(ev_su[0], side)) != cudaSuccess) return err;
  for (int64_t b = 0; b < nb; ++b) {
    const int x = (int)(b & 1);
    const int64_t c1 = (b + 1) * B, nn = n - c1;
    // ---- the caller's stream
    // block b reads its columns, and its A' buffer was last read, by block b - 2's update
    if (b >= 2 && (err = cudaStreamWaitEvent(stream, ev_gb[x], 0)) != cudaSuccess) return err;
    if ((err = quantize(b, stream)) != cudaSuccess) return err;
    if (b + 1 == nb) break;
    if ((err = cudaEventRecord(ev_q[x], stream)) != cudaSuccess) return err;
    if ((err = cudaStreamWaitEvent(stream, ev_su[x], 0)) != cudaSuccess) return err;
    if (b >= 1 && (err = cudaStreamWaitEvent(stream, ev_gb[x ^ 1], 0)) != cudaSuccess) return err;
    if ((err = launch_gemm_accumulate(Abuf[x], Bbuf[x], m, std::min<int64_t>(B, nn), 6 * B, Wf + c1, n, stream)) !=
        cudaSuccess)
      return err;
    if ((err = cudaEventRecord(ev_ga[x], stream)) != cudaSuccess) return err;
    // ---- the second stream
    if ((err = cudaStreamWaitEvent(side, ev_q[x], 0)) != cudaSuccess) return err;
    if (nn > B && (err = launch_gemm_accumulate(Abuf[x], Bbuf[x] + B * 6 * B, m, nn - B, 6 * B, Wf + c1 + B, n,
                                                side)) != cudaSuccess)
      return err;
    if ((err = cudaEventRecord(ev_gb[x], side)) != cudaSuccess) return err;
    if (b + 2 < nb) {  // U's split for the next block, once both updates of block b - 1 have read its buffer
      if (b >= 1 && (err = cudaStreamWaitEvent(side, ev_ga[x ^ 1], 0)) != cudaSuccess) return err;
      if ((err = split_u(b + 1, side)) != cudaSuccess) return err;
      if ((err = cudaEventRecord(ev_su[x ^ 1], side)) != cudaSuccess) return err;
    }
  }
  if ((err = cudaEventRecord(join, side)) != cudaSuccess) return err;
  return cudaStreamWaitEvent(stream, join, 0);
}

}  // namespace hscale
