// Kernels of the parameter manager's hot path.
//
// Rows are moved as float4 (128-bit) by "row groups" of G lanes, each lane
// owning columns lane, lane+G, ..., lane+(C-1)G of a row (D4 = D/4 <= G*C).
// Kernels are persistent grids (a multiple of the SM count) with several
// independent rows in flight per group (R-way unrolled address chains:
// key -> slot -> row, software-pipelined where registers allow), which is
// what an HBM-bound gather needs.
//
//   intent      the distinct keys of one call (hash set + stamps)       (Sec. 3)
//   pull        out[i] = replica of keys[i] at worker w, else main       (Sec. 5.1)
//   push        sorted (key, position) pairs are split into fixed chunks;
//               each group sums the delta rows of every key segment of its
//               chunk in position order and adds the sum to the worker's
//               replica (value and pending updates) or to main (Sec. 4,
//               App. B.1.2); segments cut by a chunk boundary leave partial
//               sums that one owner combines in chunk order (fix-up)
//   events      refcount +1 for every key of the opening intent lists,
//               then -1 for the closing ones; transitions 0 -> 1 (create)
//               and 1 -> 0 (evict)                                      (Sec. 3)
//   evict       main += pending updates; free the slot                 (Sec. 4.1)
//   create      val = main, pending = 0; take a slot                   (Sec. 4.1)
//   sync        main += sum of all holders' pending updates (ascending
//               worker), holders := main, pending := 0                 (App. B.1.2)
#include "internal.cuh"
#include "store_launch.cuh"

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

// ---------------------------------------------------------------------------
// pull (and main-only gather for inspection when w < 0)
// ---------------------------------------------------------------------------
// R rows per group and round, software-pipelined so that one round issues
// the row loads of round i, the slot lookups of round i+1 and the key loads
// of round i+2 together: one memory latency per round instead of three.
template <int G, int C, int R>
__global__ void __launch_bounds__(kThreads)
pull_kernel(Store s, int w, const uint32_t* __restrict__ keys, uint64_t n, float* __restrict__ out) {
  const int lane = threadIdx.x & (G - 1);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  const uint32_t D4 = s.D >> 2;
  const float4* main4 = reinterpret_cast<const float4*>(s.main);
  const float4* val4 = reinterpret_cast<const float4*>(s.val);
  float4* out4 = reinterpret_cast<float4*>(out);
  const int32_t* mapw = w >= 0 ? s.map + (uint64_t)w * s.K : nullptr;
  const uint64_t step = ng * R;
  bool bad = false;
  auto load_keys = [&](uint64_t b, uint32_t (&k)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) k[r] = b + r < n ? __ldg(keys + b + r) : kNoKey;
  };
  auto load_slots = [&](const uint32_t (&k)[R], int32_t (&sl)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) sl[r] = (mapw != nullptr && k[r] < s.K) ? __ldg(mapw + k[r]) : -1;
  };
  uint64_t base = g * R;
  uint32_t k0[R], k1[R];
  int32_t sl0[R];
  load_keys(base, k0);
  load_keys(base + step, k1);
  load_slots(k0, sl0);
  for (; base < n; base += step) {
    // this round's rows
    const float4* src[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      src[r] = nullptr;
      if (k0[r] < s.K) src[r] = sl0[r] >= 0 ? val4 + (uint64_t)sl0[r] * D4 : main4 + (uint64_t)k0[r] * D4;
      else if (base + r < n) bad = true;
    }
    float4 v[R][C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + c * G;
#pragma unroll
      for (int r = 0; r < R; ++r) v[r][c] = (src[r] != nullptr && col < D4) ? __ldg(src[r] + col) : f4zero();
    }
    // next round's slots and the keys of the round after
    int32_t sl1[R];
    uint32_t k2[R];
    load_slots(k1, sl1);
    load_keys(base + 2 * step, k2);
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + c * G;
      if (col < D4)
#pragma unroll
        for (int r = 0; r < R; ++r)
          if (base + r < n) __stcs(out4 + (base + r) * D4 + col, v[r][c]);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      k0[r] = k1[r];
      sl0[r] = sl1[r];
      k1[r] = k2[r];
    }
  }
  if (bad && lane == 0) set_error(s.st, ERR_KEY_RANGE);
}

// ---------------------------------------------------------------------------
// push: chunked segmented reduction over key-sorted (key, position) pairs
// ---------------------------------------------------------------------------
template <int C>
__device__ __forceinline__ void apply_sum(const Store& s, const int32_t* mapw, uint32_t k,
                                          const float4 (&sum)[C], int lane, int G) {
  const uint32_t D4 = s.D >> 2;
  const int32_t sl = mapw[k];
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  float4* main4 = reinterpret_cast<float4*>(s.main);
  float4* t1 = sl >= 0 ? val4 + (uint64_t)sl * D4 : main4 + (uint64_t)k * D4;
  // the segment is the only writer of its targets: vector atomic adds give
  // the plain fp32 sums without a round trip of the target rows
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const uint32_t col = lane + c * G;
    if (col < D4) atomicAdd(t1 + col, sum[c]);
  }
  if (sl >= 0) {
    float4* t2 = acc4 + (uint64_t)sl * D4;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + c * G;
      if (col < D4) atomicAdd(t2 + col, sum[c]);
    }
  }
}

// Each block stages a span of up to kPushSpan consecutive sorted positions
// (keys and source positions) in shared memory; its groups own consecutive
// chunks of it.  A segment cut by chunk boundaries leaves a partial sum per
// chunk (a tail piece in the chunk it starts in, head pieces in the chunks
// it continues into); push_fixup / push_long add the pieces up.
constexpr int kPushSpan = 3072;
// resident push_chunks blocks per SM (its launch bounds)
constexpr int push_blocks_per_sm(int C) { return C >= 4 ? 2 : 3; }
// a segment cut by chunk boundaries and spanning at most this many further
// chunks is combined by one group; longer ones (hot keys) by a whole block
constexpr int kShortSpan = 8;

template <int G, int C, int R>
__global__ void __launch_bounds__(kThreads, push_blocks_per_sm(C)) push_chunks_kernel(Store s, PushArgs a) {
  if (sort_failed(s.st)) return;
  constexpr int NG = kThreads / G;
  const uint32_t CH = (uint32_t)a.chunk;            // rows per group, NG * CH <= kPushSpan
  const uint32_t span = NG * CH;
  __shared__ uint32_t sk[kPushSpan + 2];   // sk[0]: key before the span; sk[1+len]: key after it
  __shared__ uint32_t sp[kPushSpan];       // source row of each sorted position
  __shared__ int32_t ss[kPushSpan];        // target slot of rows that end a whole segment
  __shared__ uint8_t sf[kPushSpan];        // row flags (below)
  // flags: bit0 a piece ends at this row, bit1 that piece began inside the
  // row's chunk, bit2 the key's segment ends here, bit3 a piece begins here,
  // bit4 the row holds a key (not a skipped one); a row with bits 0-2 all set
  // ends a segment that lies inside one chunk
  const int lane = threadIdx.x & (G - 1);
  const int gi = threadIdx.x / G;
  const uint32_t D4 = s.D >> 2;
  const float4* d4 = reinterpret_cast<const float4*>(a.deltas);
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  float4* main4 = reinterpret_cast<float4*>(s.main);
  float4* ph4 = reinterpret_cast<float4*>(a.part_head);
  float4* pt4 = reinterpret_cast<float4*>(a.part_tail);
  const int32_t* mapw = s.map + (uint64_t)a.worker * s.K;
  uint32_t heads = 0;
  for (uint64_t P0 = (uint64_t)blockIdx.x * span; P0 < a.n; P0 += (uint64_t)gridDim.x * span) {
    const uint32_t len = (uint32_t)(a.n - P0 < (uint64_t)span ? a.n - P0 : span);
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < len; i += kThreads) {
      sk[1 + i] = a.skeys[P0 + i];
      sp[i] = a.spos[P0 + i];
    }
    if (threadIdx.x == 0) {
      sk[0] = P0 > 0 ? a.skeys[P0 - 1] : kNoKey;
      sk[1 + len] = P0 + len < a.n ? a.skeys[P0 + len] : kNoKey;
    }
    __syncthreads();
    // per-row control, one thread per row, and the slot of every whole segment
    for (uint32_t i = threadIdx.x; i < len; i += kThreads) {
      const uint32_t k = sk[1 + i];
      uint8_t f = 0;
      int32_t slot = -2;
      if (k != kNoKey) {
        const uint32_t cs = i - i % CH;                          // first row of the chunk
        const uint32_t ce = cs + CH < len ? cs + CH : len;        // end of the chunk
        const bool seg_begin = (P0 + i == 0) || sk[i] != k;       // sk[i] is the key of row i-1
        const bool seg_end = (P0 + i + 1 >= a.n) || sk[1 + i + 1] != k;
        const bool started = (P0 + cs == 0) || sk[cs] != k;       // piece began inside the chunk
        const bool piece_end = seg_end || i + 1 == ce;
        f = (piece_end ? 1 : 0) | (started ? 2 : 0) | (seg_end ? 4 : 0) |
            ((seg_begin || i == cs) ? 8 : 0) | 16;
        if (seg_begin) ++heads;
        if ((f & 7) == 7) slot = mapw[k];
      }
      sf[i] = f;
      ss[i] = slot;
    }
    __syncthreads();
    const uint32_t p0 = gi * CH;
    const uint32_t p1 = p0 + CH < len ? p0 + CH : len;
    const uint64_t j = P0 / CH + gi;                 // global chunk index
    float4 run[C];
#pragma unroll
    for (int c = 0; c < C; ++c) run[c] = f4zero();
    for (uint32_t p = p0; p < p1; p += R) {
      // one round of loads: the delta rows
      uint8_t f[R];
      int32_t sl[R];
      uint32_t k[R];
      float4 d[R][C];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const bool v = p + r < p1;
        f[r] = v ? sf[p + r] : 0;
        sl[r] = (f[r] & 7) == 7 ? ss[p + r] : -2;
        k[r] = v ? sk[1 + p + r] : kNoKey;
        const uint32_t src = v ? sp[p + r] : 0u;
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          d[r][c] = ((f[r] & 16) && col < D4) ? __ldg(d4 + (uint64_t)src * D4 + col) : f4zero();
        }
      }
      // running sums in position order
#pragma unroll
      for (int r = 0; r < R; ++r) {
#pragma unroll
        for (int c = 0; c < C; ++c) {
          run[c] = (f[r] & 8) ? d[r][c] : f4add(run[c], d[r][c]);
          d[r][c] = run[c];
        }
      }
      // a whole segment's sum goes to its targets by vector atomic adds: the
      // segment is the only writer of those rows in this kernel, so the
      // result is the plain fp32 sum target + s, and no target row has to
      // travel to the SM and back
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (sl[r] != -2) {
          float4* dst = sl[r] >= 0 ? val4 + (uint64_t)sl[r] * D4 : main4 + (uint64_t)k[r] * D4;
#pragma unroll
          for (int c = 0; c < C; ++c) {
            const uint32_t col = lane + c * G;
            if (col < D4) atomicAdd(dst + col, d[r][c]);
          }
          if (sl[r] >= 0) {
#pragma unroll
            for (int c = 0; c < C; ++c) {
              const uint32_t col = lane + c * G;
              if (col < D4) atomicAdd(acc4 + (uint64_t)sl[r] * D4 + col, d[r][c]);
            }
          }
        } else if (f[r] & 1) {
          // a piece of a segment cut by a chunk boundary: partial sum
          float4* dst = (f[r] & 2) ? pt4 : ph4;
#pragma unroll
          for (int c = 0; c < C; ++c) {
            const uint32_t col = lane + c * G;
            if (col < D4) dst[j * D4 + col] = d[r][c];
          }
        }
      }
    }
  }
  uint32_t unused = 0;
  block_sum2(heads, unused);
  if (threadIdx.x == 0 && heads) {
    atomicAdd(&s.st->last_unique, heads);
    atomicAdd(&s.st->push_unique, (unsigned long long)heads);
  }
}

// A segment that starts in chunk j and continues past it is owned by j: its
// sum is j's tail piece plus the head pieces of chunks j+1 .. m_end.  Spans
// of at most kShortSpan further chunks are combined here (loads issued
// together); longer ones are listed for push_long_kernel.
template <int G, int C>
__global__ void __launch_bounds__(kThreads) push_fixup_kernel(Store s, PushArgs a, uint32_t* long_list,
                                                              uint32_t* long_count) {
  if (sort_failed(s.st)) return;
  const uint64_t CH = a.chunk;
  const int lane = threadIdx.x & (G - 1);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  const uint32_t D4 = s.D >> 2;
  const float4* ph4 = reinterpret_cast<const float4*>(a.part_head);
  const float4* pt4 = reinterpret_cast<const float4*>(a.part_tail);
  const int32_t* mapw = s.map + (uint64_t)a.worker * s.K;
  for (uint64_t j = g; j < a.nchunks; j += ng) {
    const uint64_t p0 = j * CH;
    const uint64_t p1 = p0 + CH;
    if (p1 >= a.n) continue;
    const uint32_t kl = a.skeys[p1 - 1];
    if (kl == kNoKey || a.skeys[p1] != kl) continue;
    if (p0 > 0 && a.skeys[p0 - 1] == kl) continue;           // started in an earlier chunk
    bool cont[kShortSpan];   // cont[t]: the segment continues past chunk j+1+t
#pragma unroll
    for (int t = 0; t < kShortSpan; ++t) {
      const uint64_t e = (j + 2 + t) * CH;
      cont[t] = e < a.n && a.skeys[e] == kl;
    }
    int span = 0;            // further chunks after j+1 that the segment reaches
#pragma unroll
    for (int t = 0; t < kShortSpan; ++t)
      if (span == t && cont[t]) ++span;
    if (span == kShortSpan) {
      if (lane == 0) {
        // last piece m whose first position still holds kl (a monotone predicate)
        uint64_t lo = j + 1 + kShortSpan, hi = a.nchunks - 1;
        while (lo < hi) {
          const uint64_t mid = (lo + hi + 1) / 2;
          if (a.skeys[mid * CH] == kl) lo = mid; else hi = mid - 1;
        }
        const uint32_t e = atomicAdd(long_count, 1u);
        long_list[4 * e] = (uint32_t)j;
        long_list[4 * e + 1] = (uint32_t)lo;
        long_list[4 * e + 2] = 0;             // finished work items of this entry
      }
      continue;
    }
    float4 tot[C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t col = lane + c * G;
      tot[c] = col < D4 ? pt4[j * D4 + col] : f4zero();
    }
    constexpr int UB = 8 / C > 0 ? 8 / C : 1;    // head pieces loaded together
    for (int u0 = 0; u0 <= span; u0 += UB) {
      float4 t[UB][C];
#pragma unroll
      for (int u = 0; u < UB; ++u)
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          t[u][c] = (u0 + u <= span && col < D4) ? ph4[(j + 1 + u0 + u) * D4 + col] : f4zero();
        }
#pragma unroll
      for (int u = 0; u < UB; ++u)
        if (u0 + u <= span)
#pragma unroll
          for (int c = 0; c < C; ++c) tot[c] = f4add(tot[c], t[u][c]);
    }
    apply_sum<C>(s, mapw, kl, tot, lane, G);
  }
}

// Hot keys: a segment whose pieces run over more than kShortSpan further
// chunks.  Its head pieces j+1 .. m_end are cut into work items of kLongSub
// pieces, spread over all blocks; a block sums its item (groups take strided
// pieces in increasing order, then the group sums in group order) into
// long_parts.  The block that finishes an entry's last item sums the item
// sums the same way (groups take strided items, then group order), adds the
// tail piece and applies the total.  Every sum has a fixed order, so the
// result does not depend on which block finishes last.
constexpr uint32_t kLongSub = 32;
constexpr uint32_t kLongSmem = 1024;   // long-list entries whose item bases sit in shared memory

template <int G, int C>
__global__ void __launch_bounds__(kThreads) push_long_kernel(Store s, PushArgs a, uint32_t* long_list,
                                                             const uint32_t* long_count) {
  if (sort_failed(s.st)) return;
  constexpr int NG = kThreads / G;
  const uint64_t CH = a.chunk;
  __shared__ float4 part[NG][G * C];
  __shared__ int s_last;
  const int lane = threadIdx.x & (G - 1);
  const int gi = threadIdx.x / G;
  const uint32_t D4 = s.D >> 2;
  const float4* ph4 = reinterpret_cast<const float4*>(a.part_head);
  const float4* pt4 = reinterpret_cast<const float4*>(a.part_tail);
  float4* lp4 = reinterpret_cast<float4*>(a.long_parts);
  const int32_t* mapw = s.map + (uint64_t)a.worker * s.K;
  const uint32_t nl = *long_count;
  // item bases of the first kLongSmem entries (block scan of their item
  // counts), so that locating an item is a binary search in shared memory
  __shared__ uint32_t s_base[kLongSmem + 1];
  __shared__ uint32_t s_scan[kThreads / 32];
  const uint32_t ns_tab = nl < kLongSmem ? nl : kLongSmem;
  {
    uint32_t carry = 0;
    for (uint32_t e0 = 0; e0 < ns_tab; e0 += kThreads) {   // block-uniform trip count
      const uint32_t e = e0 + threadIdx.x;
      const uint32_t cnt = e < ns_tab ? (long_list[4 * e + 1] - long_list[4 * e] + kLongSub - 1) / kLongSub : 0u;
      uint32_t x = cnt;
      const int ln = threadIdx.x & 31, wp = threadIdx.x >> 5;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (ln >= o) x += y;
      }
      if (ln == 31) s_scan[wp] = x;
      __syncthreads();
      uint32_t before = 0, total = 0;
      for (int w2 = 0; w2 < kThreads / 32; ++w2) {
        if (w2 < wp) before += s_scan[w2];
        total += s_scan[w2];
      }
      if (e < ns_tab) s_base[e] = carry + before + x - cnt;
      carry += total;
      __syncthreads();
    }
    if (threadIdx.x == 0) s_base[ns_tab] = carry;
    __syncthreads();
  }
  for (uint64_t q = blockIdx.x;; q += gridDim.x) {
    // locate work item q: entry e, item it, first item of the entry `base`
    uint64_t base = 0, it = 0, ns = 0, j = 0, m_end = 0;
    uint32_t e = 0;
    if (q < s_base[ns_tab]) {
      uint32_t lo = 0, hi = ns_tab - 1;   // last entry whose base <= q
      while (lo < hi) {
        const uint32_t mid = (lo + hi + 1) / 2;
        if (s_base[mid] <= q) lo = mid; else hi = mid - 1;
      }
      e = lo;
      base = s_base[e];
      j = long_list[4 * e];
      m_end = long_list[4 * e + 1];
      ns = (m_end - j + kLongSub - 1) / kLongSub;
      it = q - base;
    } else {
      // entries past the table: walk them
      base = s_base[ns_tab];
      for (e = ns_tab; e < nl; ++e) {
        j = long_list[4 * e];
        m_end = long_list[4 * e + 1];
        ns = (m_end - j + kLongSub - 1) / kLongSub;
        if (q < base + ns) {
          it = q - base;
          break;
        }
        base += ns;
      }
      if (e == nl) break;
    }
    const uint64_t lo = j + 1 + it * kLongSub;
    const uint64_t hi = lo + kLongSub - 1 < m_end ? lo + kLongSub - 1 : m_end;
    float4 acc[C];
#pragma unroll
    for (int c = 0; c < C; ++c) acc[c] = f4zero();
    constexpr int U = (kLongSub + NG - 1) / NG;
    float4 t[U][C];
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        const uint64_t m = lo + gi + (uint64_t)u * NG;
        t[u][c] = (m <= hi && col < D4) ? ph4[m * D4 + col] : f4zero();
      }
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int c = 0; c < C; ++c) acc[c] = f4add(acc[c], t[u][c]);
#pragma unroll
    for (int c = 0; c < C; ++c) part[gi][lane + c * G] = acc[c];
    __syncthreads();
    if (gi == 0) {
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        float4 tot = f4zero();
        for (int g2 = 0; g2 < NG; ++g2) tot = f4add(tot, part[g2][lane + c * G]);
        if (col < D4) lp4[q * D4 + col] = tot;
      }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(long_list + 4 * e + 2, 1u) == (uint32_t)(ns - 1);
    __syncthreads();
    if (s_last) {   // block-uniform
      // the entry's item sums: group g adds items g, g + NG, ... in order,
      // then group 0 adds the tail piece and the group sums in group order
      __threadfence();
      float4 acc2[C];
#pragma unroll
      for (int c = 0; c < C; ++c) acc2[c] = f4zero();
      constexpr int UB = 4 / C > 0 ? 4 / C : 1;
      for (uint64_t i0 = gi; i0 < ns; i0 += (uint64_t)NG * UB) {
        float4 t[UB][C];
#pragma unroll
        for (int u = 0; u < UB; ++u)
#pragma unroll
          for (int c = 0; c < C; ++c) {
            const uint32_t col = lane + c * G;
            const uint64_t it2 = i0 + (uint64_t)u * NG;
            t[u][c] = (it2 < ns && col < D4) ? __ldcg(lp4 + (base + it2) * D4 + col) : f4zero();
          }
#pragma unroll
        for (int u = 0; u < UB; ++u)
#pragma unroll
          for (int c = 0; c < C; ++c) acc2[c] = f4add(acc2[c], t[u][c]);
      }
#pragma unroll
      for (int c = 0; c < C; ++c) part[gi][lane + c * G] = acc2[c];
      __syncthreads();
      if (gi == 0) {
        const uint32_t kl = a.skeys[(j + 1) * CH - 1];
        float4 tot[C];
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          tot[c] = col < D4 ? pt4[j * D4 + col] : f4zero();
          for (int g2 = 0; g2 < NG; ++g2) tot[c] = f4add(tot[c], part[g2][lane + c * G]);
        }
        apply_sum<C>(s, mapw, kl, tot, lane, G);
      }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// intent: the distinct keys of one call (Sec. 3: an intent names a set of
// parameters, so a key listed twice in one call counts once)
// ---------------------------------------------------------------------------
constexpr int kDedupItems = 8;
constexpr int kDedupTile = kThreads * kDedupItems;   // keys per block and round
constexpr int kDedupTab = 2 * kDedupTile;            // shared hash table, half full at most

// Each block takes tiles of 2048 keys: a shared-memory hash set (open
// addressing) keeps the first copy of every key of the tile, and an exchange
// on the key's stamp keeps the first copy over all tiles (stamp == tag once
// some copy has been listed).  One atomic per block and round appends.
__global__ void __launch_bounds__(kThreads) intent_dedup_kernel(Store s, const uint32_t* __restrict__ keys,
                                                                uint64_t n, uint32_t tag,
                                                                uint32_t* __restrict__ out, uint32_t* count) {
  __shared__ uint32_t tab[kDedupTab];
  __shared__ uint32_t base_s;
  bool bad = false;
  for (uint64_t t0 = (uint64_t)blockIdx.x * kDedupTile; t0 < n;
       t0 += (uint64_t)gridDim.x * kDedupTile) {   // block-uniform trip count
    for (int i = threadIdx.x; i < kDedupTab; i += kThreads) tab[i] = kNoKey;
    __syncthreads();
    uint32_t k[kDedupItems];
    bool first[kDedupItems];
#pragma unroll
    for (int it = 0; it < kDedupItems; ++it) {
      const uint64_t i = t0 + (uint64_t)it * kThreads + threadIdx.x;
      k[it] = i < n ? __ldg(keys + i) : kNoKey;
      if (i < n && k[it] >= s.K) {
        bad = true;
        k[it] = kNoKey;
      }
    }
#pragma unroll
    for (int it = 0; it < kDedupItems; ++it) {
      first[it] = false;
      if (k[it] == kNoKey) continue;
      uint32_t h = (k[it] * 0x9E3779B1u) >> (32 - 12);   // 12 bits: kDedupTab = 4096
      for (int probe = 0; probe < kDedupTab; ++probe) {
        const uint32_t old = atomicCAS(&tab[h], kNoKey, k[it]);
        if (old == kNoKey) {
          first[it] = true;
          break;
        }
        if (old == k[it]) break;
        h = (h + 1) & (kDedupTab - 1);
      }
    }
#pragma unroll
    for (int it = 0; it < kDedupItems; ++it)
      if (first[it]) first[it] = atomicExch(s.stamp + k[it], tag) != tag;
    uint32_t c = 0, unused = 0, total, t2;
#pragma unroll
    for (int it = 0; it < kDedupItems; ++it) c += first[it] ? 1u : 0u;
    block_exclusive_scan2(c, unused, total, t2);
    if (threadIdx.x == 0) base_s = total ? atomicAdd(count, total) : 0u;
    __syncthreads();
    c += base_s;
#pragma unroll
    for (int it = 0; it < kDedupItems; ++it)
      if (first[it]) out[c++] = k[it];
    __syncthreads();
  }
  if (__any_sync(0xFFFFFFFFu, bad) && (threadIdx.x & 31) == 0) set_error(s.st, ERR_KEY_RANGE);
}

// ---------------------------------------------------------------------------
// advance: intent lists -> refcounts -> create / evict lists
// ---------------------------------------------------------------------------
// Up to kEventLists intent lists handled by one launch.
constexpr int kEventLists = 8;
struct EventBatch {
  const uint32_t* keys[kEventLists];
  const uint32_t* count[kEventLists];
  int n;
};

// The lists of a batch as one index space: pre[l] = keys before list l.
__device__ __forceinline__ uint32_t batch_prefix(const EventBatch& eb, uint32_t (&pre)[kEventLists + 1]) {
  pre[0] = 0;
#pragma unroll
  for (int l = 0; l < kEventLists; ++l) pre[l + 1] = pre[l] + (l < eb.n ? *eb.count[l] : 0u);
  return pre[kEventLists];
}

// Key at flat index i (< total) of the batch.
__device__ __forceinline__ uint32_t batch_key(const EventBatch& eb, const uint32_t (&pre)[kEventLists + 1],
                                              uint32_t i) {
  int l = 0;
#pragma unroll
  for (int m = 1; m < kEventLists; ++m)
    if (i >= pre[m]) l = m;
  return eb.keys[l][i - pre[l]];
}

// Refcount transitions of one advance.  All lists whose window opens are
// applied first (START, rc += 1; a key whose count was 0 is listed for
// creation), then all lists whose window closes (rc -= 1; a key whose count
// reaches 0 and that holds a replica is listed for eviction).  Every key of a
// closing list had a positive count before the advance (its intent was
// active), so with the openings first a key in both kinds of list never
// crosses 0, and one atomic per listed key gives exactly the transitions of
// the net change.  Four keys per thread and round; one list append per block
// and round.  The order of a list is not specified.
template <bool START>
__global__ void events_kernel(Store s, uint32_t w, EventBatch eb, uint32_t* out_list) {
  if (sort_failed(s.st)) return;
  constexpr int Q = 4;
  __shared__ uint32_t base_s;
  uint32_t* rcw = s.rc + (uint64_t)w * s.K;
  const int32_t* mapw = s.map + (uint64_t)w * s.K;
  uint32_t* counter = START ? &s.st->n_create : &s.st->n_evict;
  uint32_t pre[kEventLists + 1];
  const uint32_t n = batch_prefix(eb, pre);
  const uint32_t stride = gridDim.x * blockDim.x * Q;
  for (uint32_t b = blockIdx.x * blockDim.x * Q; b < n; b += stride) {   // block-uniform trip count
    uint32_t k[Q], old[Q];
    bool hit[Q];
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      const uint32_t i = b + q * blockDim.x + threadIdx.x;
      k[q] = i < n ? batch_key(eb, pre, i) : 0u;
    }
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      const uint32_t i = b + q * blockDim.x + threadIdx.x;
      old[q] = 1u;   // neither transition
      if (i < n) old[q] = START ? atomicAdd(rcw + k[q], 1u) : atomicSub(rcw + k[q], 1u);
    }
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      const uint32_t i = b + q * blockDim.x + threadIdx.x;
      if (START) {
        hit[q] = i < n && old[q] == 0u;
        if (i < n && old[q] >= 65535u) set_error(s.st, ERR_REFCOUNT);
      } else {
        hit[q] = i < n && old[q] == 1u;
        if (i < n && old[q] == 0u) {   // more closings than openings: undo, report
          atomicAdd(rcw + k[q], 1u);
          set_error(s.st, ERR_REFCOUNT);
        }
      }
    }
    // a key whose replica was never created (capacity exhausted) has nothing to destroy
    if (!START) {
#pragma unroll
      for (int q = 0; q < Q; ++q)
        if (hit[q]) hit[q] = mapw[k[q]] >= 0;
    }
    uint32_t c = 0, unused = 0, total, t2;
#pragma unroll
    for (int q = 0; q < Q; ++q) c += hit[q] ? 1u : 0u;
    block_exclusive_scan2(c, unused, total, t2);
    if (threadIdx.x == 0) base_s = total ? atomicAdd(counter, total) : 0u;
    __syncthreads();
    c += base_s;
#pragma unroll
    for (int q = 0; q < Q; ++q)
      if (hit[q]) out_list[c++] = k[q];
    __syncthreads();
  }
}

// evict: main[k] += acc[slot]; the freed slot goes on the stack at
// free_top + i (every listed key holds a replica), so no list atomics are
// needed.  R keys per row group at a time: list entries, slots, then the
// pending rows, each as one round of independent loads.
template <int G, int C>
__global__ void __launch_bounds__(kThreads, C >= 8 ? 2 : 4) evict_kernel(Store s, uint32_t w,
                                                                       const uint32_t* __restrict__ list) {
  constexpr int R = 4 / C > 0 ? 4 / C : 1;
  const int lane = threadIdx.x & (G - 1);
  const uint32_t D4 = s.D >> 2;
  const uint32_t n = s.st->n_evict;
  const int32_t top = s.st->free_top;
  int32_t* mapw = s.map + (uint64_t)w * s.K;
  float4* main4 = reinterpret_cast<float4*>(s.main);
  const float4* acc4 = reinterpret_cast<const float4*>(s.acc);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  const uint64_t step = ng * R;
  // software-pipelined: a round loads the pending rows of its keys, the
  // slots of the next round's keys and the list entries of the round after
  auto load_keys = [&](uint64_t i0, uint32_t (&k)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) k[r] = i0 + r < n ? list[i0 + r] : 0u;
  };
  auto load_slots = [&](uint64_t i0, const uint32_t (&k)[R], int32_t (&sl)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) sl[r] = i0 + r < n ? mapw[k[r]] : 0;
  };
  uint32_t k[R], k1[R];
  int32_t sl[R];
  load_keys(g * R, k);
  load_keys(g * R + step, k1);
  load_slots(g * R, k, sl);
  for (uint64_t i0 = g * R; i0 < n; i0 += step) {
    float4 ac[R][C];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        ac[r][c] = (i0 + r < n && col < D4) ? acc4[(uint64_t)sl[r] * D4 + col] : f4zero();
      }
    int32_t sl1[R];
    uint32_t k2[R];
    load_slots(i0 + step, k1, sl1);
    load_keys(i0 + 2 * step, k2);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (i0 + r >= n) break;
      // each listed key is evicted once, so main[k] has no other writer
      // here: a vector atomic add gives main + acc without loading main
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) atomicAdd(main4 + (uint64_t)k[r] * D4 + col, ac[r][c]);
      }
      if (lane == 0) {
        mapw[k[r]] = -1;
        atomicAnd(s.holders + k[r], ~(1u << w));
        s.slot_owner[sl[r]] = kEmptySlot;
        s.free_stack[top + (int32_t)(i0 + r)] = sl[r];
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      k[r] = k1[r];
      sl[r] = sl1[r];
      k1[r] = k2[r];
    }
  }
}

// Single thread: account the evictions, then reserve the creations.  The
// stack initially holds slots S-1 .. 0 (slot 0 on top) and positions below
// S - high_water are never written, so popping down to alloc_base has used
// every slot below S - alloc_base.
__global__ void alloc_kernel(DevState* st, int32_t S) {
  const uint32_t ne = st->n_evict;
  st->free_top += (int32_t)ne;
  st->live -= (int32_t)ne;
  st->destroyed += ne;
  const uint32_t n = st->n_create;
  if ((int64_t)n > (int64_t)st->free_top) {
    st->errors |= ERR_NO_SLOTS;
    st->n_create_ok = 0;
    st->alloc_base = st->free_top;
    return;
  }
  st->alloc_base = st->free_top - (int32_t)n;
  st->free_top = st->alloc_base;
  st->n_create_ok = n;
  st->live += (int32_t)n;
  st->created += n;
  if (S - st->alloc_base > st->high_water) st->high_water = S - st->alloc_base;
}

// create: val = main[k], acc = 0, take a slot from the stack (R keys per
// row group at a time, as in evict_kernel)
template <int G, int C>
__global__ void __launch_bounds__(kThreads, C >= 8 ? 2 : 4) create_kernel(Store s, uint32_t w,
                                                                        const uint32_t* __restrict__ list) {
  constexpr int R = 4 / C > 0 ? 4 / C : 1;
  const int lane = threadIdx.x & (G - 1);
  const uint32_t D4 = s.D >> 2;
  const uint32_t n = s.st->n_create_ok;
  const int32_t base = s.st->alloc_base;
  int32_t* mapw = s.map + (uint64_t)w * s.K;
  const float4* main4 = reinterpret_cast<const float4*>(s.main);
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  const uint64_t step = ng * R;
  // software-pipelined: a round loads the main rows of its keys and the list
  // entries and slots of the next round together
  auto load_entries = [&](uint64_t i0, uint32_t (&k)[R], int32_t (&sl)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const bool v = i0 + r < n;
      k[r] = v ? list[i0 + r] : 0u;
      // slots popped from the top of the stack: lowest free slots come first
      sl[r] = v ? s.free_stack[base + (int32_t)(n - 1 - (i0 + r))] : 0;
    }
  };
  uint32_t k[R];
  int32_t sl[R];
  load_entries(g * R, k, sl);
  for (uint64_t i0 = g * R; i0 < n; i0 += step) {
    float4 m[R][C];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        m[r][c] = (i0 + r < n && col < D4) ? main4[(uint64_t)k[r] * D4 + col] : f4zero();
      }
    uint32_t k1[R];
    int32_t sl1[R];
    load_entries(i0 + step, k1, sl1);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (i0 + r >= n) break;
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) {
          val4[(uint64_t)sl[r] * D4 + col] = m[r][c];
          acc4[(uint64_t)sl[r] * D4 + col] = f4zero();
        }
      }
      if (lane == 0) {
        mapw[k[r]] = sl[r];
        atomicOr(s.holders + k[r], 1u << w);
        s.slot_owner[sl[r]] = ((unsigned long long)w << 32) | k[r];
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      k[r] = k1[r];
      sl[r] = sl1[r];
    }
  }
}

// ---------------------------------------------------------------------------
// sync
// ---------------------------------------------------------------------------
template <int G, int C>
__global__ void __launch_bounds__(kThreads, C >= 8 ? 2 : 4) sync_kernel(Store s) {
  const int lane = threadIdx.x & (G - 1);
  const uint32_t D4 = s.D >> 2;
  const uint64_t hw = (uint64_t)s.st->high_water;
  float4* main4 = reinterpret_cast<float4*>(s.main);
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  uint32_t nkeys = 0, nreps = 0;
  // R slots per group at a time: owners, holder masks, then (for keys held
  // by one worker only, the common case) main and pending rows, each as one
  // round of independent loads
  constexpr int R = 4 / C > 0 ? 4 / C : 1;
  for (uint64_t b = g * R; b < hw; b += ng * R) {
    unsigned long long own[R];
    uint32_t mk[R];
#pragma unroll
    for (int r = 0; r < R; ++r) own[r] = b + r < hw ? s.slot_owner[b + r] : kEmptySlot;
#pragma unroll
    for (int r = 0; r < R; ++r) mk[r] = own[r] != kEmptySlot ? s.holders[(uint32_t)own[r]] : 0u;
    bool single[R];
    float4 mv[R][C], av[R][C];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const uint32_t w = (uint32_t)(own[r] >> 32);
      single[r] = own[r] != kEmptySlot && mk[r] == (1u << w);
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        const bool cv = single[r] && col < D4;
        mv[r][c] = cv ? main4[(uint64_t)(uint32_t)own[r] * D4 + col] : f4zero();
        av[r][c] = cv ? acc4[(b + r) * D4 + col] : f4zero();
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (!single[r]) continue;
      if (lane == 0) {
        nkeys += 1;
        nreps += 1;
      }
      const uint32_t k = (uint32_t)own[r];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) {
          const float4 m = f4add(mv[r][c], av[r][c]);
          main4[(uint64_t)k * D4 + col] = m;
          val4[(b + r) * D4 + col] = m;
          acc4[(b + r) * D4 + col] = f4zero();
        }
      }
    }
    // keys with several holders: the lowest holder merges all of them
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (own[r] == kEmptySlot || single[r]) continue;
      const uint32_t w = (uint32_t)(own[r] >> 32);
      const uint32_t k = (uint32_t)own[r];
      const uint32_t mask = mk[r];
      if ((uint32_t)(__ffs(mask) - 1) != w) continue;   // the lowest holder merges
      if (lane == 0) {
        nkeys += 1;
        nreps += (uint32_t)__popc(mask);
      }
      float4 m[C];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        m[c] = col < D4 ? main4[(uint64_t)k * D4 + col] : f4zero();
      }
      constexpr int Q = 4 / C > 0 ? 4 / C : 1;
      uint32_t mm = mask;
      while (mm) {
        int32_t hs[Q];
#pragma unroll
        for (int q = 0; q < Q; ++q) {
          hs[q] = -1;
          if (mm) {
            const uint32_t wb = __ffs(mm) - 1;
            mm &= mm - 1;
            hs[q] = s.map[(uint64_t)wb * s.K + k];
          }
        }
        float4 t[Q][C];
#pragma unroll
        for (int q = 0; q < Q; ++q)
#pragma unroll
          for (int c = 0; c < C; ++c) {
            const uint32_t col = lane + c * G;
            t[q][c] = (hs[q] >= 0 && col < D4) ? acc4[(uint64_t)hs[q] * D4 + col] : f4zero();
          }
#pragma unroll
        for (int q = 0; q < Q; ++q)
          if (hs[q] >= 0)
#pragma unroll
            for (int c = 0; c < C; ++c) m[c] = f4add(m[c], t[q][c]);
      }
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) main4[(uint64_t)k * D4 + col] = m[c];
      }
      mm = mask;
      while (mm) {
        const uint32_t wb = __ffs(mm) - 1;
        mm &= mm - 1;
        const int32_t h = s.map[(uint64_t)wb * s.K + k];
        if (h < 0) continue;
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          if (col < D4) {
            val4[(uint64_t)h * D4 + col] = m[c];
            acc4[(uint64_t)h * D4 + col] = f4zero();
          }
        }
      }
    }
  }
  block_sum2(nkeys, nreps);
  if (threadIdx.x == 0 && nkeys) {
    atomicAdd(&s.st->sync_keys, (unsigned long long)nkeys);
    atomicAdd(&s.st->sync_replicas, (unsigned long long)nreps);
  }
}

// ---------------------------------------------------------------------------
// inspection
// ---------------------------------------------------------------------------
__global__ void refcounts_kernel(Store s, uint32_t w, const uint32_t* __restrict__ keys, uint64_t n,
                                 uint32_t* __restrict__ out) {
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (uint64_t)gridDim.x * blockDim.x) {
    const uint32_t k = keys[i];
    if (k < s.K) out[i] = s.rc[(uint64_t)w * s.K + k];
    else {
      out[i] = 0;
      set_error(s.st, ERR_KEY_RANGE);
    }
  }
}

__global__ void replica_rows_kernel(Store s, uint32_t w, const uint32_t* __restrict__ keys, uint64_t n,
                                    float* __restrict__ val_out, float* __restrict__ acc_out,
                                    uint8_t* __restrict__ has_out) {
  const uint32_t D = s.D;
  for (uint64_t i = blockIdx.x; i < n; i += gridDim.x) {
    const uint32_t k = keys[i];
    const int32_t sl = k < s.K ? s.map[(uint64_t)w * s.K + k] : -1;
    if (threadIdx.x == 0) {
      has_out[i] = sl >= 0 ? 1 : 0;
      if (k >= s.K) set_error(s.st, ERR_KEY_RANGE);
    }
    for (uint32_t c = threadIdx.x; c < D; c += blockDim.x) {
      val_out[i * D + c] = sl >= 0 ? s.val[(uint64_t)sl * D + c] : 0.f;
      acc_out[i * D + c] = sl >= 0 ? s.acc[(uint64_t)sl * D + c] : 0.f;
    }
  }
}

__global__ void init_pool_kernel(int32_t* free_stack, uint64_t S, unsigned long long* owner) {
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < S;
       i += (uint64_t)gridDim.x * blockDim.x) {
    free_stack[i] = (int32_t)(S - 1 - i);   // top of the stack holds slot 0
    owner[i] = kEmptySlot;
  }
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

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
void launch_intent_dedup(const Store& s, const uint32_t* keys, uint64_t n, uint32_t tag, uint32_t* out,
                         uint32_t* count, int sms, cudaStream_t stream) {
  if (n == 0) return;
  uint64_t b = (n + kDedupTile - 1) / kDedupTile;
  if (b > (uint64_t)sms * 8) b = (uint64_t)sms * 8;
  note_launches(1);
  intent_dedup_kernel<<<(unsigned)b, kThreads, 0, stream>>>(s, keys, n, tag, out, count);
}

void launch_pull(const Store& s, int w, const uint32_t* keys, uint64_t n, float* out, int sms,
                 cudaStream_t stream) {
  if (n == 0) return;
  dispatch_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr int R = 8 / C > 0 ? 8 / C : 1;
    note_launches(1);
    pull_kernel<G, C, R><<<grid_for((n + R - 1) / R, G, sms), kThreads, 0, stream>>>(s, w, keys, n, out);
  });
}

uint64_t push_chunk_rows(uint32_t D, uint64_t n, int sms) {
  // one span per resident block where the span fits in shared memory: rows
  // per group = n / (groups per block x resident blocks), in [8, kPushSpan / groups]
  uint64_t ch = 0;
  dispatch_push_gc(D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr uint64_t NG = kThreads / G;
    const uint64_t groups = NG * (uint64_t)sms * push_blocks_per_sm(C);
    ch = (n + groups - 1) / groups;
    if (ch < 8) ch = 8;
    if (ch > kPushSpan / NG) ch = kPushSpan / NG;
  });
  return ch;
}

uint64_t push_long_list_words(uint64_t nchunks) { return 4 * (nchunks / 8 + 2) + 1; }
uint64_t push_long_part_rows(uint64_t nchunks) { return nchunks / kLongSub + nchunks / 8 + 2; }

void launch_push(const Store& s, const PushArgs& a, int sms, cudaStream_t stream) {
  if (a.n == 0) return;
  dispatch_push_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr int R = 4 / C > 0 ? 4 / C : 1;
    // one block per span: the block scheduler balances spans over the SMs
    const uint64_t spans = (a.n + a.chunk * (kThreads / G) - 1) / (a.chunk * (kThreads / G));
    note_launches(3);
    push_chunks_kernel<G, C, R><<<(unsigned)spans, kThreads, 0, stream>>>(s, a);
    push_fixup_kernel<G, C><<<grid_for(a.nchunks, G, sms), kThreads, 0, stream>>>(s, a, a.long_list,
                                                                                 a.long_count);
    push_long_kernel<G, C><<<(unsigned)sms * 2, kThreads, 0, stream>>>(s, a, a.long_list, a.long_count);
  });
}

void launch_events(const Store& s, uint32_t w, const EventList* lists, int nlists,
                   uint32_t* create_list, uint32_t* evict_list, int sms, cudaStream_t stream) {
  // all opening lists first, then all closing lists, in batches of kEventLists
  const uint64_t cap_blocks = (uint64_t)sms * 8;
  for (int pass = 0; pass < 2; ++pass) {
    const int sign = pass == 0 ? +1 : -1;
    EventBatch eb{};
    uint64_t cap = 0;
    auto flush = [&]() {
      if (eb.n == 0) return;
      uint64_t b = (cap + 4 * kThreads - 1) / (4 * kThreads);   // 4 keys per thread
      if (b > cap_blocks) b = cap_blocks;
      if (b == 0) b = 1;
      note_launches(1);
      if (pass == 0)
        events_kernel<true><<<(unsigned)b, kThreads, 0, stream>>>(s, w, eb, create_list);
      else
        events_kernel<false><<<(unsigned)b, kThreads, 0, stream>>>(s, w, eb, evict_list);
      eb = EventBatch{};
      cap = 0;
    };
    for (int i = 0; i < nlists; ++i) {
      if (lists[i].sign != sign) continue;
      eb.keys[eb.n] = lists[i].keys;
      eb.count[eb.n] = lists[i].count;
      eb.n += 1;
      cap += lists[i].cap;   // the kernel covers the batch's lists as one index space
      if (eb.n == kEventLists) flush();
    }
    flush();
  }
}

void launch_evict_create(const Store& s, uint32_t w, const uint32_t* create_list,
                         const uint32_t* evict_list, uint64_t max_events, int sms,
                         cudaStream_t stream) {
  dispatch_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr uint64_t R = 4 / C > 0 ? 4 / C : 1;   // keys per group, as in the kernels
    const unsigned grid = grid_for((max_events + R - 1) / R, G, sms);
    note_launches(3);
    evict_kernel<G, C><<<grid, kThreads, 0, stream>>>(s, w, evict_list);
    alloc_kernel<<<1, 1, 0, stream>>>(s.st, (int32_t)s.S);
    create_kernel<G, C><<<grid, kThreads, 0, stream>>>(s, w, create_list);
  });
}

void launch_sync(const Store& s, uint64_t slot_bound, int sms, cudaStream_t stream) {
  if (slot_bound == 0) return;
  dispatch_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    note_launches(1);
    constexpr uint64_t R = 4 / C > 0 ? 4 / C : 1;   // slots per group, as in sync_kernel
    sync_kernel<G, C><<<grid_for((slot_bound + R - 1) / R, G, sms), kThreads, 0, stream>>>(s);
  });
}

void launch_refcounts(const Store& s, uint32_t w, const uint32_t* keys, uint64_t n, uint32_t* out,
                      cudaStream_t stream) {
  if (n == 0) return;
  note_launches(1);
  refcounts_kernel<<<(unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096), 256, 0, stream>>>(
      s, w, keys, n, out);
}

void launch_replica_rows(const Store& s, uint32_t w, const uint32_t* keys, uint64_t n, float* val,
                         float* acc, uint8_t* has, cudaStream_t stream) {
  if (n == 0) return;
  note_launches(1);
  replica_rows_kernel<<<(unsigned)(n < 4096 ? n : 4096), 128, 0, stream>>>(s, w, keys, n, val, acc, has);
}

void launch_init_pool(int32_t* free_stack, uint64_t S, unsigned long long* owner, cudaStream_t stream) {
  uint64_t b = (S + 255) / 256;
  if (b > 65535) b = 65535;
  if (b == 0) return;
  note_launches(1);
  init_pool_kernel<<<(unsigned)b, 256, 0, stream>>>(free_stack, S, owner);
}

}  // namespace adapm
