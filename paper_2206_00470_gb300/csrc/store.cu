// Kernels of the parameter manager's hot path that read and write rows
// through the slot maps: pull, sync and the inspection gathers.  The push is
// in push.cu, the intent and advance kernels in advance.cu.
//
//   pull        out[i] = replica of keys[i] at worker w, else main       (Sec. 5.1)
//   sync        main += sum of all holders' pending updates (ascending
//               worker), holders := main, pending := 0                 (App. B.1.2)
#include "internal.cuh"
#include "rowgroup.cuh"
#include "store_launch.cuh"

namespace adapm {

namespace {

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
// sync
// ---------------------------------------------------------------------------
// VER: versioned refresh (s.dirty is set)
template <int G, int C, bool VER>
__global__ void __launch_bounds__(kThreads, C >= 8 ? 2 : (VER && C == 1 ? 3 : 4)) sync_kernel(Store s) {
  const int lane = threadIdx.x & (G - 1);
  const uint32_t D4 = s.D >> 2;
  const uint64_t hw = (uint64_t)s.st->high_water;
  float4* main4 = reinterpret_cast<float4*>(s.main);
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  uint32_t nkeys = 0, nreps = 0, nref = 0;   // nref: VER only
  __shared__ int32_t hslots[kThreads / G][32];   // holders' slots of the key a group merges (W <= 32)
  const unsigned gmask = G == 32 ? 0xFFFFFFFFu : (((1u << G) - 1u) << ((threadIdx.x & 31) & ~(G - 1)));
  // R slots per group at a time: owners, holder masks, then (for keys held
  // by one worker only, the common case) main and pending rows, each as one
  // round of independent loads.  Versioned refresh (App. B.1.2: a holder
  // receives only updates it has not seen): a sole holder's value is left
  // alone unless main[k] was written other than by a sync since the last
  // sync of k (dirty[k]); keys with several holders are always refreshed.
  constexpr int R = 4 / C > 0 ? 4 / C : 1;
  for (uint64_t b = g * R; b < hw; b += ng * R) {
    unsigned long long own[R];
    uint32_t mk[R];
#pragma unroll
    for (int r = 0; r < R; ++r) own[r] = b + r < hw ? s.slot_owner[b + r] : kEmptySlot;
#pragma unroll
    for (int r = 0; r < R; ++r) mk[r] = own[r] != kEmptySlot ? s.holders[(uint32_t)own[r]] : 0u;
    // a live slot's key is held by this worker alone iff its mask has one bit
    // (its own); such a mask is known, so it is replaced by the refresh flag
    // (1: write the value, 0: leave it), which keeps at most one bit set
    auto is_single = [&](int r) { return own[r] != kEmptySlot && __popc(mk[r]) <= 1; };
    float4 mv[R][C], av[R][C];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const bool single = is_single(r);
      if (VER && single) mk[r] = (uint32_t)s.dirty[(uint32_t)own[r]];
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        const bool cv = single && col < D4;
        mv[r][c] = cv ? main4[(uint64_t)(uint32_t)own[r] * D4 + col] : f4zero();
        av[r][c] = cv ? acc4[(b + r) * D4 + col] : f4zero();
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (!is_single(r)) continue;
      const uint32_t k = (uint32_t)own[r];
      if (lane == 0) {
        nkeys += 1;
        nreps += 1;
        if (VER && mk[r]) {
          nref += 1;
          s.dirty[k] = 0;
        }
      }
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        if (col < D4) {
          const float4 m = f4add(mv[r][c], av[r][c]);
          main4[(uint64_t)k * D4 + col] = m;
          if (!VER || mk[r]) val4[(b + r) * D4 + col] = m;
          acc4[(b + r) * D4 + col] = f4zero();
        }
      }
    }
    // keys with several holders: the lowest holder merges all of them
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (own[r] == kEmptySlot || is_single(r)) continue;
      const uint32_t w = (uint32_t)(own[r] >> 32);
      const uint32_t k = (uint32_t)own[r];
      const uint32_t mask = mk[r];
      if ((uint32_t)(__ffs(mask) - 1) != w) continue;   // the lowest holder merges
      if (lane == 0) {
        nkeys += 1;
        nreps += (uint32_t)__popc(mask);
        if (VER) {
          nref += (uint32_t)__popc(mask);
          s.dirty[k] = 0;
        }
      }
      // Holders that fit in one round of Q rows: their slots are looked up with
      // the sum and again for the writes.  More: each lane looks up one
      // holder's slot (G at a time) into shared memory, so the sum and the
      // writes need no second lookup.  Both add the pending rows to main in
      // ascending worker order.
      if (__popc(mask) <= (4 / C > 0 ? 4 / C : 1)) {
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
      } else {
        float4 m[C];   // (loaded with the holders' slots)
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          m[c] = col < D4 ? main4[(uint64_t)k * D4 + col] : f4zero();
        }
        // the holders' slots: one slot-map lookup per lane (holder j by lane j,
        // G at a time), kept in shared memory for the sum and the writes
        const int nh = __popc(mask);
        int32_t* hsl = hslots[threadIdx.x / G];
        for (int j = lane; j < nh; j += G) {
          uint32_t mm = mask;   // the j-th set bit (j < nh, so mm stays nonzero)
          for (int t = 0; t < j; ++t) mm &= mm - 1;
          const uint32_t wb = (uint32_t)(__ffs(mm) - 1);
          hsl[j] = s.map[(uint64_t)wb * s.K + k];
        }
        __syncwarp(gmask);
        constexpr int Q = 4 / C > 0 ? 4 / C : 1;
        // pending rows added in ascending worker order, Q rows in flight
        for (int j0 = 0; j0 < nh; j0 += Q) {
          int32_t hs[Q];
#pragma unroll
          for (int q = 0; q < Q; ++q) hs[q] = j0 + q < nh ? hsl[j0 + q] : -1;
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
        for (int j = 0; j < nh; ++j) {
          const int32_t h = hsl[j];
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
        __syncwarp(gmask);   // hsl is reused by the group's next key
      }
    }
  }
  block_sum2(nkeys, nreps);
  if (VER) {
    __syncthreads();   // block_sum2's shared words are reused below
    uint32_t unused = 0;
    block_sum2(nref, unused);
  }
  if (threadIdx.x == 0 && nkeys) {
    atomicAdd(&s.st->sync_keys, (unsigned long long)nkeys);
    atomicAdd(&s.st->sync_replicas, (unsigned long long)nreps);
    atomicAdd(&s.st->sync_refreshed, (unsigned long long)(VER ? nref : nreps));
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

// owner of each key: -1 at its home (and always without relocation)
__global__ void owners_kernel(Store s, const uint32_t* __restrict__ keys, uint64_t n, int32_t* __restrict__ out) {
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (uint64_t)gridDim.x * blockDim.x) {
    const uint32_t k = keys[i];
    if (k < s.K) out[i] = s.own ? own_owner(s.own[k]) : -1;
    else {
      out[i] = -1;
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

}  // namespace

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
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

void launch_sync(const Store& s, uint64_t slot_bound, int sms, cudaStream_t stream) {
  if (slot_bound == 0) return;
  dispatch_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    note_launches(1);
    constexpr uint64_t R = 4 / C > 0 ? 4 / C : 1;   // slots per group, as in sync_kernel
    const unsigned grid = grid_for((slot_bound + R - 1) / R, G, sms);
    if (s.dirty != nullptr)
      sync_kernel<G, C, true><<<grid, kThreads, 0, stream>>>(s);
    else
      sync_kernel<G, C, false><<<grid, kThreads, 0, stream>>>(s);
  });
}

void launch_refcounts(const Store& s, uint32_t w, const uint32_t* keys, uint64_t n, uint32_t* out,
                      cudaStream_t stream) {
  if (n == 0) return;
  note_launches(1);
  refcounts_kernel<<<(unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096), 256, 0, stream>>>(
      s, w, keys, n, out);
}

void launch_owners(const Store& s, const uint32_t* keys, uint64_t n, int32_t* out, cudaStream_t stream) {
  if (n == 0) return;
  note_launches(1);
  owners_kernel<<<(unsigned)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096), 256, 0, stream>>>(s, keys, n,
                                                                                                 out);
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
