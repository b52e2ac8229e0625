// Fused training steps of the three sparse workloads (App. C): each reads the
// rows a sample needs straight through the worker's slot map (replica, else
// main copy), computes loss and gradients in fp32 from those values, and
// writes one delta row per row occurrence for the push that follows:
//   AdaGrad rows [theta | a]:  delta = [-lr*g/sqrt(a + g*g + eps) | g*g]
//   (1/sqrt evaluated with the correctly rounded __frsqrt_rn)
//   plain SGD:                 delta = -lr*g
// Losses: MF 1/2 (v - u.w)^2; ComplEx softplus(-y phi), phi = Re(sum h r
// conj(t)) with rows [re | im]; SGNS softplus(-u_o.v_c) + sum softplus(u_n.v_c).
// Every sample's loss is added by one lane into a per-block fp64 partial in
// a fixed order, so the batch loss is deterministic.
#include "internal.cuh"
#include "store_launch.cuh"

namespace adapm {

namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float4 f4zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }
__device__ __forceinline__ float dot4(float4 a, float4 b) {
  return a.x * b.x + a.y * b.y + a.z * b.z + a.w * b.w;
}
__device__ __forceinline__ float4 f4scale(float4 a, float s) {
  return make_float4(a.x * s, a.y * s, a.z * s, a.w * s);
}
__device__ __forceinline__ float4 f4fma(float4 a, float s, float4 acc) {
  return make_float4(fmaf(a.x, s, acc.x), fmaf(a.y, s, acc.y), fmaf(a.z, s, acc.z), fmaf(a.w, s, acc.w));
}

__device__ __forceinline__ float softplus_f(float x) { return log1pf(expf(-fabsf(x))) + fmaxf(x, 0.f); }
__device__ __forceinline__ float sigmoid_f(float x) {
  if (x >= 0.f) return 1.f / (1.f + expf(-x));
  const float e = expf(x);
  return e / (1.f + e);
}

// AdaGrad delta of one float of gradient g with accumulator a
__device__ __forceinline__ float ada_theta(float g, float a, float lr, float eps) {
  return -lr * g * __frsqrt_rn(a + g * g + eps);   // correctly rounded 1/sqrt
}
__device__ __forceinline__ float4 ada_theta4(float4 g, float4 a, float lr, float eps) {
  return make_float4(ada_theta(g.x, a.x, lr, eps), ada_theta(g.y, a.y, lr, eps),
                     ada_theta(g.z, a.z, lr, eps), ada_theta(g.w, a.w, lr, eps));
}
__device__ __forceinline__ float4 sq4(float4 g) { return make_float4(g.x * g.x, g.y * g.y, g.z * g.z, g.w * g.w); }

template <int G>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

__device__ __forceinline__ const float4* row_ptr(const Store& s, const int32_t* mapw, uint32_t k) {
  const uint32_t D4 = s.D >> 2;
  const int32_t sl = mapw[k];
  return sl >= 0 ? reinterpret_cast<const float4*>(s.val) + (uint64_t)sl * D4
                 : reinterpret_cast<const float4*>(s.main) + (uint64_t)k * D4;
}

// Fixed-order block reduction of one double per thread into
// o.loss_part[blockIdx.x]; with o.loss_out the last block to finish then
// sums the partials (thread t the partials t, t + 256, ... in order, then a
// fixed tree) into *o.loss_out and clears the block counter.
__device__ void block_loss(double v, const StepOut& o) {
  __shared__ double sm[kThreads / 32];
  __shared__ double tree[kThreads];
  __shared__ int last;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, off);
  if ((threadIdx.x & 31) == 0) sm[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0;
    for (int i = 0; i < kThreads / 32; ++i) t += sm[i];
    o.loss_part[blockIdx.x] = t;
    last = 0;
    if (o.loss_out) {
      __threadfence();
      last = atomicAdd(o.loss_done, 1u) == gridDim.x - 1;
    }
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  double t = 0.0;
  for (unsigned i = threadIdx.x; i < gridDim.x; i += kThreads) t += __ldcg(o.loss_part + i);
  tree[threadIdx.x] = t;
  __syncthreads();
  for (int w = kThreads / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) tree[threadIdx.x] += tree[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    *o.loss_out = tree[0];
    *o.loss_done = 0u;
  }
}

// ---------------------------------------------------------------------------
// matrix factorisation: one cell per group of G lanes
// ---------------------------------------------------------------------------
template <int G, int C>
__global__ void __launch_bounds__(kThreads)
mf_step_kernel(Store s, uint32_t w, const uint32_t* __restrict__ rows, const uint32_t* __restrict__ cols,
               const float* __restrict__ vals, uint64_t n, uint32_t dim, int adagrad, float lr, float eps,
               StepOut o) {
  const int lane = threadIdx.x & (G - 1);
  constexpr int GPW = 32 / G;
  const int gi = (threadIdx.x & 31) / G;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t nwarps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t dim4 = dim >> 2, D4 = s.D >> 2;
  const int32_t* mapw = s.map + (uint64_t)w * s.K;
  float4* d4 = reinterpret_cast<float4*>(o.drows);
  double lsum = 0.0;
  // software-pipelined: a round loads the rows of its cell, the slots of the
  // next round's cell and the keys of the cell after
  const uint64_t step = nwarps * GPW;
  auto cell_keys = [&](uint64_t i, uint32_t& ku, uint32_t& kw) -> bool {   // both in range
    ku = 0;
    kw = 0;
    if (i >= n) return false;
    ku = rows[i];
    kw = cols[i];
    return ku < s.K && kw < s.K;
  };
  uint32_t ku0, kw0, ku1, kw1;
  bool ok0 = cell_keys(warp * GPW + gi, ku0, kw0);
  bool ok1 = cell_keys(warp * GPW + gi + step, ku1, kw1);
  int32_t su0 = ok0 ? mapw[ku0] : -1, sw0 = ok0 ? mapw[kw0] : -1;
  for (uint64_t b = warp * GPW; b < n; b += step) {
    const uint64_t i = b + gi;
    const bool in = i < n;
    const uint32_t ku = ku0, kw = kw0;
    const bool ok = ok0;
    if (in && !ok && lane == 0) set_error(s.st, ERR_KEY_RANGE);
    float4 tu[C], tw[C], au[C], aw[C];
    {
      const float4* pu = su0 >= 0 ? reinterpret_cast<const float4*>(s.val) + (uint64_t)su0 * D4
                                  : reinterpret_cast<const float4*>(s.main) + (uint64_t)ku * D4;
      const float4* pw = sw0 >= 0 ? reinterpret_cast<const float4*>(s.val) + (uint64_t)sw0 * D4
                                  : reinterpret_cast<const float4*>(s.main) + (uint64_t)kw * D4;
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        const bool cv = ok && col < dim4;
        tu[c] = cv ? pu[col] : f4zero();
        tw[c] = cv ? pw[col] : f4zero();
        au[c] = (cv && adagrad) ? pu[dim4 + col] : f4zero();
        aw[c] = (cv && adagrad) ? pw[dim4 + col] : f4zero();
      }
    }
    // the next cell's slots and the keys of the cell after, issued before
    // this cell's rows are used
    su0 = ok1 ? mapw[ku1] : -1;
    sw0 = ok1 ? mapw[kw1] : -1;
    ku0 = ku1;
    kw0 = kw1;
    ok0 = ok1;
    ok1 = cell_keys(i + 2 * step, ku1, kw1);
    float part = 0.f;
#pragma unroll
    for (int c = 0; c < C; ++c) part += dot4(tu[c], tw[c]);
    const float dot = group_sum<G>(part);
    if (!in) continue;
    if (!ok) {
      if (lane == 0) {
        o.dkeys[i] = kNoKey;
        o.dkeys[n + i] = kNoKey;
      }
      continue;
    }
    const float e = vals[i] - dot;
    if (lane == 0) lsum += 0.5 * (double)e * (double)e;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + c * G;
      if (col < dim4) {
        const float4 gu = f4scale(tw[c], -e);
        const float4 gw = f4scale(tu[c], -e);
        if (adagrad) {
          d4[i * D4 + col] = ada_theta4(gu, au[c], lr, eps);
          d4[i * D4 + dim4 + col] = sq4(gu);
          d4[(n + i) * D4 + col] = ada_theta4(gw, aw[c], lr, eps);
          d4[(n + i) * D4 + dim4 + col] = sq4(gw);
        } else {
          d4[i * D4 + col] = f4scale(gu, -lr);
          d4[(n + i) * D4 + col] = f4scale(gw, -lr);
        }
      }
    }
    if (lane == 0) {
      o.dkeys[i] = ku;
      o.dkeys[n + i] = kw;
    }
  }
  block_loss(lsum, o);
}

// ---------------------------------------------------------------------------
// ComplEx: one triple per warp; lane q holds float4 q of the re and im halves
// ---------------------------------------------------------------------------
template <int CC, int U>
__global__ void __launch_bounds__(kThreads)
complex_step_kernel(Store s, uint32_t w, const uint32_t* __restrict__ heads, const uint32_t* __restrict__ rels,
                    const uint32_t* __restrict__ tails, const uint32_t* __restrict__ negs, uint64_t n,
                    uint32_t n_neg, uint32_t dim, float lr, float eps, StepOut o) {
  const int lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t nwarps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t h4 = dim >> 3;          // float4 per half (re or im) of theta
  const uint32_t D4 = s.D >> 2;          // = 4 * h4: [theta re | theta im | a re | a im]
  const int32_t* mapw = s.map + (uint64_t)w * s.K;
  float4* d4 = reinterpret_cast<float4*>(o.drows);
  // delta rows in the order the keys of a batch are listed: all heads, all
  // relations, all true tails, then the negatives triple by triple
  const uint64_t rh = 0, rrel = n, rt = 2 * n, rneg = 3 * n;
  double lsum = 0.0;
  for (uint64_t i = warp; i < n; i += nwarps) {
    const uint32_t kh = heads[i], kr = rels[i], kt = tails[i];
    if (kh >= s.K || kr >= s.K || kt >= s.K) {
      if (lane == 0) set_error(s.st, ERR_KEY_RANGE);
      if (lane < 3) o.dkeys[(uint64_t)lane * n + i] = kNoKey;
      for (uint64_t q = lane; q < n_neg; q += 32) o.dkeys[rneg + i * n_neg + q] = kNoKey;
      continue;
    }
    const float4* ph = row_ptr(s, mapw, kh);
    const float4* pr = row_ptr(s, mapw, kr);
    float4 hre[CC], him[CC], rre[CC], rim[CC], xre[CC], xim[CC], Tre[CC], Tim[CC];
#pragma unroll
    for (int c = 0; c < CC; ++c) {
      const uint32_t q = lane + 32 * c;
      const bool cv = q < h4;
      hre[c] = cv ? ph[q] : f4zero();
      him[c] = cv ? ph[h4 + q] : f4zero();
      rre[c] = cv ? pr[q] : f4zero();
      rim[c] = cv ? pr[h4 + q] : f4zero();
      // complex product h*r: d phi / d t
      xre[c] = make_float4(hre[c].x * rre[c].x - him[c].x * rim[c].x, hre[c].y * rre[c].y - him[c].y * rim[c].y,
                           hre[c].z * rre[c].z - him[c].z * rim[c].z, hre[c].w * rre[c].w - him[c].w * rim[c].w);
      xim[c] = make_float4(hre[c].x * rim[c].x + him[c].x * rre[c].x, hre[c].y * rim[c].y + him[c].y * rre[c].y,
                           hre[c].z * rim[c].z + him[c].z * rre[c].z, hre[c].w * rim[c].w + him[c].w * rre[c].w);
      Tre[c] = f4zero();
      Tim[c] = f4zero();
    }
    // tails: j = 0 is the true tail (label +1), j >= 1 the negatives (label
    // -1); software-pipelined: a round loads the tail rows of U indices, the
    // slots of the next U and the keys of the U after
    const uint32_t J = 1 + n_neg;
    auto tail_key = [&](uint32_t j) -> uint32_t {   // kNoKey: skipped
      if (j >= J) return kNoKey;
      const uint32_t k = j == 0 ? kt : negs[i * n_neg + (j - 1)];
      if (k >= s.K) {
        if (lane == 0) set_error(s.st, ERR_KEY_RANGE);
        return kNoKey;
      }
      return k;
    };
    uint32_t k0[U], k1[U];
    int32_t s0[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      k0[u] = tail_key(u);
      k1[u] = tail_key(U + u);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) s0[u] = k0[u] != kNoKey ? mapw[k0[u]] : -1;
    for (uint32_t j0 = 0; j0 < J; j0 += U) {
      float4 tre[U][CC], tim[U][CC], are[U][CC], aim[U][CC];
      float part[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const bool vx = k0[u] != kNoKey;
        const float4* pt = s0[u] >= 0 ? reinterpret_cast<const float4*>(s.val) + (uint64_t)s0[u] * D4
                                      : reinterpret_cast<const float4*>(s.main) + (uint64_t)k0[u] * D4;
        part[u] = 0.f;
#pragma unroll
        for (int c = 0; c < CC; ++c) {
          const uint32_t q = lane + 32 * c;
          const bool cv = vx && q < h4;
          tre[u][c] = cv ? pt[q] : f4zero();
          tim[u][c] = cv ? pt[h4 + q] : f4zero();
          are[u][c] = cv ? pt[2 * h4 + q] : f4zero();
          aim[u][c] = cv ? pt[3 * h4 + q] : f4zero();
          part[u] += dot4(xre[c], tre[u][c]) + dot4(xim[c], tim[u][c]);
        }
      }
      int32_t s1[U];
      uint32_t k2[U];
#pragma unroll
      for (int u = 0; u < U; ++u) s1[u] = k1[u] != kNoKey ? mapw[k1[u]] : -1;
#pragma unroll
      for (int u = 0; u < U; ++u) k2[u] = tail_key(j0 + 2 * U + u);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t j = j0 + u;
        const float phi = group_sum<32>(part[u]);
        if (j >= J) continue;
        const uint64_t row = j == 0 ? rt + i : rneg + i * n_neg + (j - 1);
        if (k0[u] == kNoKey) {
          if (lane == 0) o.dkeys[row] = kNoKey;
          continue;
        }
        const float coef = j == 0 ? -sigmoid_f(-phi) : sigmoid_f(phi);
        if (lane == 0) lsum += (double)(j == 0 ? softplus_f(-phi) : softplus_f(phi));
#pragma unroll
        for (int c = 0; c < CC; ++c) {
          const uint32_t q = lane + 32 * c;
          Tre[c] = f4fma(tre[u][c], coef, Tre[c]);
          Tim[c] = f4fma(tim[u][c], coef, Tim[c]);
          if (q < h4) {
            const float4 gre = f4scale(xre[c], coef), gim = f4scale(xim[c], coef);
            d4[row * D4 + q] = ada_theta4(gre, are[u][c], lr, eps);
            d4[row * D4 + h4 + q] = ada_theta4(gim, aim[u][c], lr, eps);
            d4[row * D4 + 2 * h4 + q] = sq4(gre);
            d4[row * D4 + 3 * h4 + q] = sq4(gim);
          }
        }
        if (lane == 0) o.dkeys[row] = k0[u];
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        k0[u] = k1[u];
        s0[u] = s1[u];
        k1[u] = k2[u];
      }
    }
    // head and relation: gradients are linear in T = sum_j coef_j t_j
#pragma unroll
    for (int c = 0; c < CC; ++c) {
      const uint32_t q = lane + 32 * c;
      if (q >= h4) continue;
      const float4 gh_re = make_float4(rre[c].x * Tre[c].x + rim[c].x * Tim[c].x, rre[c].y * Tre[c].y + rim[c].y * Tim[c].y,
                                       rre[c].z * Tre[c].z + rim[c].z * Tim[c].z, rre[c].w * Tre[c].w + rim[c].w * Tim[c].w);
      const float4 gh_im = make_float4(rre[c].x * Tim[c].x - rim[c].x * Tre[c].x, rre[c].y * Tim[c].y - rim[c].y * Tre[c].y,
                                       rre[c].z * Tim[c].z - rim[c].z * Tre[c].z, rre[c].w * Tim[c].w - rim[c].w * Tre[c].w);
      const float4 gr_re = make_float4(hre[c].x * Tre[c].x + him[c].x * Tim[c].x, hre[c].y * Tre[c].y + him[c].y * Tim[c].y,
                                       hre[c].z * Tre[c].z + him[c].z * Tim[c].z, hre[c].w * Tre[c].w + him[c].w * Tim[c].w);
      const float4 gr_im = make_float4(hre[c].x * Tim[c].x - him[c].x * Tre[c].x, hre[c].y * Tim[c].y - him[c].y * Tre[c].y,
                                       hre[c].z * Tim[c].z - him[c].z * Tre[c].z, hre[c].w * Tim[c].w - him[c].w * Tre[c].w);
      const float4 ah_re = ph[2 * h4 + q], ah_im = ph[3 * h4 + q];
      const float4 ar_re = pr[2 * h4 + q], ar_im = pr[3 * h4 + q];
      d4[(rh + i) * D4 + q] = ada_theta4(gh_re, ah_re, lr, eps);
      d4[(rh + i) * D4 + h4 + q] = ada_theta4(gh_im, ah_im, lr, eps);
      d4[(rh + i) * D4 + 2 * h4 + q] = sq4(gh_re);
      d4[(rh + i) * D4 + 3 * h4 + q] = sq4(gh_im);
      d4[(rrel + i) * D4 + q] = ada_theta4(gr_re, ar_re, lr, eps);
      d4[(rrel + i) * D4 + h4 + q] = ada_theta4(gr_im, ar_im, lr, eps);
      d4[(rrel + i) * D4 + 2 * h4 + q] = sq4(gr_re);
      d4[(rrel + i) * D4 + 3 * h4 + q] = sq4(gr_im);
    }
    if (lane == 0) {
      o.dkeys[rh + i] = kh;
      o.dkeys[rrel + i] = kr;
    }
  }
  block_loss(lsum, o);
}

// ---------------------------------------------------------------------------
// skip-gram with negative sampling: one centre per warp
// rows per centre: [centre | for each context slot: positive, negatives...]
// ---------------------------------------------------------------------------
template <int C, int U>
__global__ void __launch_bounds__(kThreads)
sgns_step_kernel(Store s, uint32_t w, const uint32_t* __restrict__ centres, const uint32_t* __restrict__ contexts,
                 const uint32_t* __restrict__ negs, uint64_t n, uint32_t n_ctx, uint32_t n_neg, uint32_t vocab,
                 float lr, StepOut o) {
  const int lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t nwarps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t D4 = s.D >> 2;
  const int32_t* mapw = s.map + (uint64_t)w * s.K;
  float4* d4 = reinterpret_cast<float4*>(o.drows);
  const uint64_t per = 1 + (uint64_t)n_ctx * (1 + n_neg);
  double lsum = 0.0;
  for (uint64_t i = warp; i < n; i += nwarps) {
    const uint64_t base = i * per;
    const uint32_t kc = centres[i];
    if (kc >= vocab) {
      if (lane == 0) set_error(s.st, ERR_KEY_RANGE);
      for (uint64_t q = lane; q < per; q += 32) o.dkeys[base + q] = kNoKey;
      continue;
    }
    const float4* pv = row_ptr(s, mapw, kc);
    float4 v[C], gv[C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + 32 * c;
      v[c] = col < D4 ? pv[col] : f4zero();
      gv[c] = f4zero();
    }
    // the centre's rows in one index space t = j * (1 + n_neg) + q (q = 0:
    // the context word, q >= 1: its negatives), software-pipelined: a round
    // loads the rows of U indices, the slots of the next U and the tokens of
    // the U after, so one memory latency per round
    const uint32_t per_ctx = 1 + n_neg;
    const uint32_t T = n_ctx * per_ctx;
    auto token = [&](uint32_t t) -> uint32_t {   // the row's key, kNoKey when it is skipped
      if (t >= T) return kNoKey;
      const uint32_t j = t / per_ctx, q = t - j * per_ctx;
      const uint32_t oc = contexts[i * n_ctx + j];
      if (oc == kNoKey) return kNoKey;
      if (oc >= vocab) {
        if (q == 0 && lane == 0) set_error(s.st, ERR_KEY_RANGE);
        return kNoKey;
      }
      const uint32_t tok = q == 0 ? oc : negs[(i * n_ctx + j) * n_neg + (q - 1)];
      if (tok >= vocab) {
        if (lane == 0) set_error(s.st, ERR_KEY_RANGE);
        return kNoKey;
      }
      return vocab + tok;
    };
    uint32_t k0[U], k1[U];
    int32_t s0[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      k0[u] = token(u);
      k1[u] = token(U + u);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) s0[u] = k0[u] != kNoKey ? mapw[k0[u]] : -1;
    for (uint32_t t0 = 0; t0 < T; t0 += U) {
      float4 x[U][C];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const bool vx = k0[u] != kNoKey;
        const float4* px = s0[u] >= 0 ? reinterpret_cast<const float4*>(s.val) + (uint64_t)s0[u] * D4
                                      : reinterpret_cast<const float4*>(s.main) + (uint64_t)k0[u] * D4;
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + 32 * c;
          x[u][c] = (vx && col < D4) ? px[col] : f4zero();
        }
      }
      // the next round's slots and the tokens of the round after, issued
      // before this round's rows are used
      int32_t s1[U];
      uint32_t k2[U];
#pragma unroll
      for (int u = 0; u < U; ++u) s1[u] = k1[u] != kNoKey ? mapw[k1[u]] : -1;
#pragma unroll
      for (int u = 0; u < U; ++u) k2[u] = token(t0 + 2 * U + u);
      float part[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        part[u] = 0.f;
#pragma unroll
        for (int c = 0; c < C; ++c) part[u] += dot4(x[u][c], v[c]);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t t = t0 + u;
        const float sc = group_sum<32>(part[u]);
        if (t >= T) continue;
        const uint64_t row = base + 1 + t;
        if (k0[u] == kNoKey) {
          if (lane == 0) o.dkeys[row] = kNoKey;
          continue;
        }
        const bool positive = t % per_ctx == 0;
        const float coef = positive ? -sigmoid_f(-sc) : sigmoid_f(sc);
        if (lane == 0) lsum += (double)(positive ? softplus_f(-sc) : softplus_f(sc));
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + 32 * c;
          gv[c] = f4fma(x[u][c], coef, gv[c]);
          if (col < D4) d4[row * D4 + col] = f4scale(v[c], -lr * coef);
        }
        if (lane == 0) o.dkeys[row] = k0[u];
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        k0[u] = k1[u];
        s0[u] = s1[u];
        k1[u] = k2[u];
      }
    }
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + 32 * c;
      if (col < D4) d4[base * D4 + col] = f4scale(gv[c], -lr);
    }
    if (lane == 0) o.dkeys[base] = kc;
  }
  block_loss(lsum, o);
}

}  // namespace

unsigned step_loss_blocks(int sms) { return (unsigned)sms * 4; }

void launch_mf_step(const Store& s, uint32_t w, const uint32_t* rows, const uint32_t* cols,
                    const float* vals, uint64_t n, uint32_t dim, bool adagrad, float lr, float eps,
                    const StepOut& o, int sms, cudaStream_t stream) {
  const unsigned grid = o.loss_blocks;
  note_launches(1);
  const uint32_t dim4 = dim / 4;
  const int a = adagrad ? 1 : 0;
  if (dim4 <= 4) mf_step_kernel<4, 1><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
  else if (dim4 <= 8) mf_step_kernel<8, 1><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
  else if (dim4 <= 16) mf_step_kernel<16, 1><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
  else if (dim4 <= 32) mf_step_kernel<32, 1><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
  else if (dim4 <= 64) mf_step_kernel<32, 2><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
  else mf_step_kernel<32, 4><<<grid, kThreads, 0, stream>>>(s, w, rows, cols, vals, n, dim, a, lr, eps, o);
}

void launch_complex_step(const Store& s, uint32_t w, const uint32_t* heads, const uint32_t* rels,
                         const uint32_t* tails, const uint32_t* negs, uint64_t n, uint32_t n_neg,
                         uint32_t dim, float lr, float eps, const StepOut& o, int sms,
                         cudaStream_t stream) {
  const unsigned grid = o.loss_blocks;
  note_launches(1);
  const uint32_t h4 = dim / 8;
  if (h4 <= 32) complex_step_kernel<1, 4><<<grid, kThreads, 0, stream>>>(s, w, heads, rels, tails, negs, n, n_neg, dim, lr, eps, o);
  else complex_step_kernel<2, 2><<<grid, kThreads, 0, stream>>>(s, w, heads, rels, tails, negs, n, n_neg, dim, lr, eps, o);
}

void launch_sgns_step(const Store& s, uint32_t w, const uint32_t* centres, const uint32_t* contexts,
                      const uint32_t* negs, uint64_t n, uint32_t n_ctx, uint32_t n_neg,
                      uint32_t vocab, uint32_t dim, float lr, const StepOut& o, int sms,
                      cudaStream_t stream) {
  const unsigned grid = o.loss_blocks;
  note_launches(1);
  const uint32_t D4 = dim / 4;
  if (D4 <= 32) sgns_step_kernel<1, 8><<<grid, kThreads, 0, stream>>>(s, w, centres, contexts, negs, n, n_ctx, n_neg, vocab, lr, o);
  else if (D4 <= 64) sgns_step_kernel<2, 4><<<grid, kThreads, 0, stream>>>(s, w, centres, contexts, negs, n, n_ctx, n_neg, vocab, lr, o);
  else if (D4 <= 96) sgns_step_kernel<3, 2><<<grid, kThreads, 0, stream>>>(s, w, centres, contexts, negs, n, n_ctx, n_neg, vocab, lr, o);
  else sgns_step_kernel<8, 1><<<grid, kThreads, 0, stream>>>(s, w, centres, contexts, negs, n, n_ctx, n_neg, vocab, lr, o);
}

}  // namespace adapm
