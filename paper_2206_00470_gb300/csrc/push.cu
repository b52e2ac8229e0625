// push: the rows of each distinct key of one call are summed and added to the
// worker's replica (value and pending updates) or to main (Sec. 4,
// App. B.1.2).  Sorted (key, position) pairs are split into fixed chunks,
// a block's groups taking consecutive chunks of one span; each group sums
// the delta rows of every key segment of its chunk in position order and
// adds the sum to its target.  A segment cut by chunk boundaries leaves a
// partial sum per chunk; the block adds those of segments inside its span
// in chunk order and applies them, and the partial sums of segments that run
// past a span are added in span order by push_combine.
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
// it continues into).
constexpr int kPushSpan = 3072;
// resident push_chunks blocks per SM (its launch bounds)
constexpr int push_blocks_per_sm(int C) { return C >= 4 ? 2 : 3; }

// Dynamic shared memory of push_chunks: the head and tail piece of every
// chunk (a row of G * C float4 per group each), then the staged span.
template <int C>
constexpr size_t push_chunks_smem() {
  return 2 * (size_t)kThreads * C * sizeof(float4) + (kPushSpan + 2) * sizeof(uint32_t) +
         kPushSpan * sizeof(uint32_t) + kPushSpan * sizeof(int32_t) + kPushSpan;
}

template <int G, int C, int R>
__global__ void __launch_bounds__(kThreads, push_blocks_per_sm(C)) push_chunks_kernel(Store s, PushArgs a0) {
  if (sort_failed(s.st)) return;
  const PushArgs a = resolve(a0);
  constexpr int NG = kThreads / G;
  const uint32_t CH = (uint32_t)a.chunk;            // rows per group, NG * CH <= kPushSpan
  const uint32_t span = NG * CH;
  extern __shared__ __align__(16) unsigned char dsm[];
  float4* ph = reinterpret_cast<float4*>(dsm);                    // head piece of each chunk
  float4* pt = ph + kThreads * C;                                 // tail piece of each chunk
  uint32_t* sk = reinterpret_cast<uint32_t*>(pt + kThreads * C);  // sk[0]: key before the span; sk[1+len]: after it
  uint32_t* sp = sk + kPushSpan + 2;                              // source row of each sorted position
  int32_t* ss = reinterpret_cast<int32_t*>(sp + kPushSpan);       // target slot of rows that end a whole segment
  uint8_t* sf = reinterpret_cast<uint8_t*>(ss + kPushSpan);       // row flags (below)
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
  float4* sp4 = reinterpret_cast<float4*>(a.span_parts);
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
      // (sorted keys are valid or the skip sentinel; anything else out of
      // range, like a position outside the batch, is an internal error)
      if (k < s.K && sp[i] < a.n) {
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
      else if (k != kNoKey || sp[i] >= a.n) set_error(s.st, ERR_INTERNAL);
      sf[i] = f;
      ss[i] = slot;
    }
    __syncthreads();
    const uint32_t p0 = gi * CH;
    const uint32_t p1 = p0 + CH < len ? p0 + CH : len;
    float4 run[C];
#pragma unroll
    for (int c = 0; c < C; ++c) run[c] = f4zero();
    // software-pipelined: the delta rows of the next round are in flight
    // while this round's are summed and applied
    auto fetch = [&](uint32_t p, uint8_t (&f)[R], float4 (&d)[R][C]) {
#pragma unroll
      for (int r = 0; r < R; ++r) {
        const bool v = p + r < p1;
        f[r] = v ? sf[p + r] : 0;
        const uint32_t src = v ? sp[p + r] : 0u;
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          d[r][c] = ((f[r] & 16) && col < D4) ? __ldg(d4 + (uint64_t)src * D4 + col) : f4zero();
        }
      }
    };
    uint8_t f[R];
    float4 d[R][C];
    fetch(p0, f, d);
    for (uint32_t p = p0; p < p1; p += R) {
      uint8_t fn[R];
      float4 dn[R][C];
      fetch(p + R, fn, dn);
      int32_t sl[R];
      uint32_t k[R];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        sl[r] = (f[r] & 7) == 7 ? ss[p + r] : -2;
        k[r] = p + r < p1 ? sk[1 + p + r] : kNoKey;
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
          // a piece of a segment cut by a chunk boundary: partial sum, kept
          // in shared memory (a chunk has at most one head and one tail piece)
          float4* dst = (f[r] & 2) ? pt : ph;
#pragma unroll
          for (int c = 0; c < C; ++c) dst[gi * G * C + lane + c * G] = d[r][c];
        }
      }
#pragma unroll
      for (int r = 0; r < R; ++r) {
        f[r] = fn[r];
#pragma unroll
        for (int c = 0; c < C; ++c) d[r][c] = dn[r][c];
      }
    }
    // Pieces of the span's cut segments are in shared memory, visible to the
    // whole block after the barrier.  A segment that begins in chunk
    // gi and continues is combined here by group gi (its tail piece, then the
    // head pieces of the chunks it covers, in chunk order) and applied when it
    // ends inside the span; one that runs past the span leaves that sum as
    // the span's tail piece, and the rows the span's first segment holds when
    // it continues from the previous span are its head piece (group 0);
    // push_combine adds span pieces up.
    __syncthreads();
    const uint32_t nch = (len + CH - 1) / CH;          // chunks of this span that hold rows
    const uint64_t sidx = P0 / span;
    auto chunk_end = [&](uint32_t m) { return (m + 1) * CH < len ? (m + 1) * CH : len; };
    // last chunk m >= g the segment of key kk covers, given it reaches chunk g;
    // out: it continues past the span
    auto walk = [&](uint32_t g, uint32_t kk, bool& out) {
      while (true) {
        const uint32_t e = chunk_end(g);
        const bool through = sk[e] == kk && sk[1 + e] == kk;   // last row kk, next row kk
        if (!through || g + 1 >= nch) {
          out = through;
          return g;
        }
        ++g;
      }
    };
    if (gi < (int)nch) {
      const uint32_t kl = sk[p1];        // the chunk's last row
      if (kl < s.K && sk[1 + p1] == kl) {
        const bool whole = sk[1 + p0] == kl;
        const bool began = !whole || P0 + p0 == 0 || sk[p0] != kl;
        if (began) {
          bool out = true;
          const uint32_t g1 = (uint32_t)gi + 1 < nch ? walk(gi + 1, kl, out) : (uint32_t)gi;
          float4 tot[C];
#pragma unroll
          for (int c = 0; c < C; ++c) tot[c] = pt[gi * G * C + lane + c * G];
          for (uint32_t m = gi + 1; m <= g1; ++m)
#pragma unroll
            for (int c = 0; c < C; ++c) tot[c] = f4add(tot[c], ph[m * G * C + lane + c * G]);
          if (out) {
#pragma unroll
            for (int c = 0; c < C; ++c) {
              const uint32_t col = lane + c * G;
              if (col < D4) sp4[(2 * sidx + 1) * D4 + col] = tot[c];
            }
          } else {
            apply_sum<C>(s, mapw, kl, tot, lane, G);
          }
        }
      }
    }
    if (gi == 0 && P0 > 0 && sk[1] < s.K && sk[0] == sk[1]) {
      bool out = false;
      const uint32_t g1 = walk(0, sk[1], out);
      float4 tot[C];
#pragma unroll
      for (int c = 0; c < C; ++c) tot[c] = ph[lane + c * G];
      for (uint32_t m = 1; m <= g1; ++m)
#pragma unroll
        for (int c = 0; c < C; ++c) tot[c] = f4add(tot[c], ph[m * G * C + lane + c * G]);
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) sp4[2 * sidx * D4 + col] = tot[c];
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

// Segments that run past a span: the span where one begins owns it; its sum
// is that span's tail piece plus the head pieces of the spans it continues
// into (the spans whose first row holds the key, counted by the block).  The groups of the block take those head pieces in strides, in
// increasing order, then group 0 adds the tail piece and the group sums in
// group order: a fixed order, whatever the number of spans.
template <int G, int C>
__global__ void __launch_bounds__(kThreads) push_combine_kernel(Store s, PushArgs a0, uint64_t span,
                                                                uint64_t nspans) {
  if (sort_failed(s.st)) return;
  const PushArgs a = resolve(a0);
  constexpr int NG = kThreads / G;
  __shared__ float4 part[NG][G * C];
  const int lane = threadIdx.x & (G - 1);
  const int gi = threadIdx.x / G;
  const uint32_t D4 = s.D >> 2;
  const float4* sp4 = reinterpret_cast<const float4*>(a.span_parts);
  const int32_t* mapw = s.map + (uint64_t)a.worker * s.K;
  for (uint64_t b = blockIdx.x; b < nspans; b += gridDim.x) {   // block-uniform
    const uint64_t st = b * span;
    const uint64_t en = st + span < a.n ? st + span : a.n;
    const uint32_t kl = a.skeys[en - 1];
    if (en >= a.n || kl >= s.K || a.skeys[en] != kl) continue;
    if (st > 0 && a.skeys[st - 1] == kl) continue;             // it began in an earlier span
    // the last span whose first row holds kl: the spans after b that do form
    // a prefix (the keys are sorted), so the block tests kThreads of them at
    // once and counts
    uint64_t lo = b;
    for (uint64_t m0 = b + 1; m0 < nspans; m0 += kThreads) {   // block-uniform
      const uint64_t m = m0 + threadIdx.x;
      const int cnt = __syncthreads_count(m < nspans && a.skeys[m * span] == kl);
      lo += (uint64_t)cnt;
      if (cnt < kThreads) break;
    }
    float4 acc[C];
#pragma unroll
    for (int c = 0; c < C; ++c) acc[c] = f4zero();
    constexpr int UB = 8 / C > 0 ? 8 / C : 1;   // span pieces per group in flight
    for (uint64_t m0 = b + 1 + gi; m0 <= lo; m0 += (uint64_t)NG * UB) {
      float4 t[UB][C];
#pragma unroll
      for (int u = 0; u < UB; ++u)
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          const uint64_t m = m0 + (uint64_t)u * NG;
          t[u][c] = (m <= lo && col < D4) ? __ldcg(sp4 + 2 * m * D4 + col) : f4zero();
        }
#pragma unroll
      for (int u = 0; u < UB; ++u)
#pragma unroll
        for (int c = 0; c < C; ++c) acc[c] = f4add(acc[c], t[u][c]);
    }
#pragma unroll
    for (int c = 0; c < C; ++c) part[gi][lane + c * G] = acc[c];
    __syncthreads();
    if (gi == 0) {
      float4 tot[C];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        tot[c] = col < D4 ? __ldcg(sp4 + (2 * b + 1) * D4 + col) : f4zero();
        for (int g2 = 0; g2 < NG; ++g2) tot[c] = f4add(tot[c], part[g2][lane + c * G]);
      }
      apply_sum<C>(s, mapw, kl, tot, lane, G);
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

uint64_t push_span_part_rows(uint64_t nchunks) { return 2 * (nchunks / 8 + 2); }

void launch_push(const Store& s, const PushArgs& a, int sms, cudaStream_t stream) {
  if (a.n == 0) return;
  dispatch_push_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr int R = 4 / C > 0 ? 4 / C : 1;
    // one block per span: the block scheduler balances spans over the SMs
    const uint64_t span = a.chunk * (kThreads / G);
    const uint64_t spans = (a.n + span - 1) / span;
    note_launches(spans > 1 ? 2 : 1);
    constexpr size_t smem = push_chunks_smem<C>();
    // the kernel's dynamic shared-memory limit is a per-device attribute
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64 || !attr_set[dev]) {
      cudaFuncSetAttribute(push_chunks_kernel<G, C, R>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (dev >= 0 && dev < 64) attr_set[dev] = true;
    }
    push_chunks_kernel<G, C, R><<<(unsigned)spans, kThreads, smem, stream>>>(s, a);
    if (spans > 1) {
      const unsigned grid = (unsigned)(spans < (uint64_t)sms * 8 ? spans : (uint64_t)sms * 8);
      push_combine_kernel<G, C><<<grid, kThreads, 0, stream>>>(s, a, span, spans);
    }
  });
}

}  // namespace adapm
