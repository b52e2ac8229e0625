// push: the rows of each distinct key of one call are summed and added to the
// worker's replica (value and pending updates) or to main (Sec. 4,
// App. B.1.2).  Sorted (key, position) pairs are split into fixed chunks;
// each group sums the delta rows of every key segment of its chunk in
// position order and adds the sum to its target; segments cut by a chunk
// boundary leave partial sums that one owner combines in chunk order
// (fix-up), and segments spanning many chunks (hot keys) are combined by
// several blocks (push_long).
#include "internal.cuh"
#include "rowgroup.cuh"
#include "store_launch.cuh"

namespace adapm {

namespace {

// The sorted keys and positions a push kernel reads: the plan's, unless its
// check stored a mismatch for this push (then the sort made instead).
__device__ __forceinline__ PushArgs resolve(const PushArgs& a0) {
  PushArgs a = a0;
  if (a.plan_seq != 0u && *reinterpret_cast<const volatile uint32_t*>(a.plan_word) == a.plan_seq) {
    a.skeys = a.alt_keys;
    a.spos = a.alt_pos;
  }
  return a;
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
  } else if (s.dirty != nullptr && lane == 0) {
    s.dirty[k] = 1;   // versioned refresh: main written by a worker without a replica
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
__global__ void __launch_bounds__(kThreads, push_blocks_per_sm(C)) push_chunks_kernel(Store s, PushArgs a0) {
  if (sort_failed(s.st)) return;
  const PushArgs a = resolve(a0);
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
        if ((f & 7) == 7) {
          slot = mapw[k];
          // versioned refresh: main written by a worker without a replica
          if (slot < 0 && s.dirty != nullptr) s.dirty[k] = 1;
        }
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
__global__ void __launch_bounds__(kThreads) push_fixup_kernel(Store s, PushArgs a0, uint32_t* long_list,
                                                              uint32_t* long_count) {
  if (sort_failed(s.st)) return;
  const PushArgs a = resolve(a0);
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
__global__ void __launch_bounds__(kThreads) push_long_kernel(Store s, PushArgs a0, uint32_t* long_list,
                                                             const uint32_t* long_count) {
  if (sort_failed(s.st)) return;
  const PushArgs a = resolve(a0);
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

}  // namespace

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

}  // namespace adapm
