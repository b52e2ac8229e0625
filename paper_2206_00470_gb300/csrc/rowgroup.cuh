// Device helpers shared by the kernel files of the parameter manager.
//
// Rows are moved as float4 (128-bit) by "row groups" of G lanes, each lane
// owning columns lane, lane+G, ..., lane+(C-1)G of a row (D4 = D/4 <= G*C).
// Kernels are persistent grids (a multiple of the SM count) with several
// independent rows in flight per group (R-way unrolled address chains:
// key -> slot -> row, software-pipelined where registers allow), which is
// what an HBM-bound gather needs.
#pragma once

#include <type_traits>

#include "internal.cuh"

namespace adapm {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 f4zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }

// Block-wide sums of two per-thread counts, returned to thread 0 (every
// thread of the block calls it), so that a kernel adds its statistics to
// DevState with one atomic per block instead of one per thread: thousands of
// atomics on the one line of DevState would queue up in its L2 slice, in
// front of the row traffic that the slice also serves.
__device__ __forceinline__ void block_sum2(uint32_t& a, uint32_t& b) {
  __shared__ uint32_t wa[32], wb[32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a += __shfl_xor_sync(0xFFFFFFFFu, a, o);
    b += __shfl_xor_sync(0xFFFFFFFFu, b, o);
  }
  const int warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  if ((threadIdx.x & 31) == 0) {
    wa[warp] = a;
    wb[warp] = b;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    a = 0;
    b = 0;
    for (int w = 0; w < nw; ++w) {
      a += wa[w];
      b += wb[w];
    }
  }
}

// Exclusive block-wide scans of two per-thread counts (every thread of the
// block calls it); ta / tb receive the block totals.
__device__ __forceinline__ void block_exclusive_scan2(uint32_t& a, uint32_t& b, uint32_t& ta, uint32_t& tb) {
  __shared__ uint32_t sa[32], sb[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  uint32_t xa = a, xb = b;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t ya = __shfl_up_sync(0xFFFFFFFFu, xa, o);
    const uint32_t yb = __shfl_up_sync(0xFFFFFFFFu, xb, o);
    if (lane >= o) {
      xa += ya;
      xb += yb;
    }
  }
  if (lane == 31) {
    sa[warp] = xa;
    sb[warp] = xb;
  }
  __syncthreads();
  if (warp == 0) {
    uint32_t va = lane < nw ? sa[lane] : 0u, vb = lane < nw ? sb[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t ya = __shfl_up_sync(0xFFFFFFFFu, va, o);
      const uint32_t yb = __shfl_up_sync(0xFFFFFFFFu, vb, o);
      if (lane >= o) {
        va += ya;
        vb += yb;
      }
    }
    if (lane < nw) {
      sa[lane] = va;
      sb[lane] = vb;
    }
  }
  __syncthreads();
  a = (warp > 0 ? sa[warp - 1] : 0u) + xa - a;
  b = (warp > 0 ? sb[warp - 1] : 0u) + xb - b;
  ta = sa[nw - 1];
  tb = sb[nw - 1];
  __syncthreads();
}

template <int G>
__device__ __forceinline__ uint64_t group_id() {
  return ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) / G;
}
template <int G>
__device__ __forceinline__ uint64_t group_count() {
  return ((uint64_t)gridDim.x * blockDim.x) / G;
}

template <typename F>
void dispatch_gc(uint32_t D4, F&& f) {
  if (D4 <= 4) f(std::integral_constant<int, 4>{}, std::integral_constant<int, 1>{});
  else if (D4 <= 8) f(std::integral_constant<int, 8>{}, std::integral_constant<int, 1>{});
  else if (D4 <= 16) f(std::integral_constant<int, 16>{}, std::integral_constant<int, 1>{});
  else if (D4 <= 32) f(std::integral_constant<int, 32>{}, std::integral_constant<int, 1>{});
  else if (D4 <= 64) f(std::integral_constant<int, 32>{}, std::integral_constant<int, 2>{});
  else if (D4 <= 128) f(std::integral_constant<int, 32>{}, std::integral_constant<int, 4>{});
  else f(std::integral_constant<int, 32>{}, std::integral_constant<int, 8>{});
}

// The push kernels give each lane two float4 of a row where the row allows
// it, so every row's control work (flags, slots, addresses) is shared by
// half as many lanes.
template <class F>
void dispatch_push_gc(uint32_t D4, F&& f) {
  if (D4 <= 8) f(std::integral_constant<int, 4>{}, std::integral_constant<int, 2>{});
  else if (D4 <= 16) f(std::integral_constant<int, 8>{}, std::integral_constant<int, 2>{});
  else if (D4 <= 32) f(std::integral_constant<int, 16>{}, std::integral_constant<int, 2>{});
  else dispatch_gc(D4, f);
}

unsigned grid_for(uint64_t groups, int G, int sms) {
  const uint64_t per_block = kThreads / G;
  uint64_t b = (groups + per_block - 1) / per_block;
  const uint64_t cap = (uint64_t)sms * 8;
  if (b > cap) b = cap;
  if (b < 1) b = 1;
  return (unsigned)b;
}

}  // namespace
}  // namespace adapm
