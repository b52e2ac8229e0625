// Stable LSD radix sort of uint32 keys (optionally with uint32 values) and
// stream compaction, for the intent table (sort + unique of the keys of one
// Intent call, Sec. 3) and for push (grouping a batch's delta rows by key).
//
// Only ceil(log2(K + 1)) key bits are sorted, in ceil(bits / 9) passes of at
// most 9 bits (512 buckets): 27-bit keys (100M) take 3 passes.  One pass =
//   hist    per tile of 1024 keys, digit counts (shared-memory atomics)
//   scan    one block per digit: exclusive prefix of that digit's counts over
//           the tiles (digit-major table), digit total
//   scatter per tile: stable rank of each key among equal digits of the tile
//           (a warp-level multi-split: one ballot per digit bit gives the
//           lanes with the same digit; per-warp digit counters in shared
//           memory order the warps), then position = digit base + earlier
//           tiles' count + rank
// No block waits on another, so the passes have no serial dependency chain.
#include "internal.cuh"

namespace adapm {

namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 8;                      // compaction: keys per thread
constexpr int kTile = kSortThreads * kSortItems;
constexpr int kRankItems = 4;                      // sort passes: keys per thread
constexpr int kRankTile = kSortThreads * kRankItems;
constexpr int kWarps = kSortThreads / 32;

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Lanes of the warp whose `valid` flag and low `nbits` digit bits equal this
// lane's (one ballot per bit: a warp-level multi-split).
__device__ __forceinline__ uint32_t digit_peers(uint32_t d, bool valid, int nbits) {
  const uint32_t v = __ballot_sync(0xFFFFFFFFu, valid);
  uint32_t peers = valid ? v : ~v;
  for (int b = 0; b < nbits; ++b) {
    const bool bit = (d >> b) & 1u;
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, bit);
    peers &= bit ? bal : ~bal;
  }
  return peers;
}

// Exclusive scan of one value per thread over a block of NT threads.
template <int NT>
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* total,
                                                         uint32_t* sm /* NT/32 words */) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sm[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t s = lane < NT / 32 ? sm[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < NT / 32) sm[lane] = s;
  }
  __syncthreads();
  const uint32_t before = warp > 0 ? sm[warp - 1] : 0u;
  *total = sm[NT / 32 - 1];
  __syncthreads();
  return before + x - v;
}

constexpr int kRadixBits = 9;
constexpr int kDigits = 1 << kRadixBits;          // 512

struct PassPlan {
  int passes;
  int per;
};

PassPlan plan_for(int bits) {
  PassPlan p;
  p.passes = (bits + kRadixBits - 1) / kRadixBits;
  if (p.passes < 1) p.passes = 1;
  p.per = (bits + p.passes - 1) / p.passes;
  return p;
}

// hist[d * nt + tile] = number of keys of the tile with digit d
__global__ void __launch_bounds__(kSortThreads)
tile_hist_kernel(const uint32_t* __restrict__ keys, uint64_t n, int shift, uint32_t mask,
                 uint32_t* __restrict__ hist, uint32_t nt) {
  __shared__ uint32_t h[kDigits];
  for (int i = threadIdx.x; i < kDigits; i += kSortThreads) h[i] = 0;
  __syncthreads();
  const uint64_t t0 = (uint64_t)blockIdx.x * kRankTile;
  uint32_t k[kRankItems];
#pragma unroll
  for (int it = 0; it < kRankItems; ++it) {
    const uint64_t i = t0 + (uint64_t)it * kSortThreads + threadIdx.x;
    k[it] = i < n ? keys[i] : 0u;
  }
#pragma unroll
  for (int it = 0; it < kRankItems; ++it) {
    const uint64_t i = t0 + (uint64_t)it * kSortThreads + threadIdx.x;
    if (i < n) atomicAdd(&h[(k[it] >> shift) & mask], 1u);
  }
  __syncthreads();
  for (uint32_t d = threadIdx.x; d <= mask; d += kSortThreads) hist[(uint64_t)d * nt + blockIdx.x] = h[d];
}

// one block per digit: exclusive prefix over tiles in place, digit total
__global__ void __launch_bounds__(kSortThreads)
digit_scan_kernel(uint32_t* __restrict__ hist, uint32_t nt, uint32_t* __restrict__ totals) {
  __shared__ uint32_t sm[kWarps];
  uint32_t* row = hist + (uint64_t)blockIdx.x * nt;
  uint32_t carry = 0;
  for (uint32_t b0 = 0; b0 < nt; b0 += kSortThreads) {
    const uint32_t idx = b0 + threadIdx.x;
    const uint32_t v = idx < nt ? row[idx] : 0u;
    uint32_t tot;
    const uint32_t ex = block_exclusive_scan<kSortThreads>(v, &tot, sm);
    if (idx < nt) row[idx] = carry + ex;
    carry += tot;
  }
  if (threadIdx.x == 0) totals[blockIdx.x] = carry;
}

// stable scatter of one tile: position = digit base + earlier tiles' count + rank
template <bool VALS, bool IOTA>
__global__ void __launch_bounds__(kSortThreads)
tile_scatter_kernel(const uint32_t* __restrict__ kin, const uint32_t* __restrict__ vin,
                    uint32_t* __restrict__ kout, uint32_t* __restrict__ vout, uint64_t n, int shift,
                    int nbits, const uint32_t* __restrict__ hist, uint32_t nt,
                    const uint32_t* __restrict__ totals) {
  __shared__ uint32_t wcnt[kWarps][kDigits];
  __shared__ uint32_t base_s[kDigits];
  __shared__ uint32_t sm[kWarps];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t mask = (1u << nbits) - 1u;
  const uint32_t nd = mask + 1;
  constexpr int DPT = kDigits / kSortThreads;
  for (int i = threadIdx.x; i < kWarps * kDigits; i += kSortThreads) (&wcnt[0][0])[i] = 0;
  {
    // digit bases: exclusive scan of the digit totals (blocked, DPT per thread)
    uint32_t v[DPT], local = 0;
#pragma unroll
    for (int q = 0; q < DPT; ++q) {
      const uint32_t d = threadIdx.x * DPT + q;
      v[q] = d < nd ? totals[d] : 0u;
      local += v[q];
    }
    uint32_t total;
    uint32_t run = block_exclusive_scan<kSortThreads>(local, &total, sm);
#pragma unroll
    for (int q = 0; q < DPT; ++q) {
      const uint32_t d = threadIdx.x * DPT + q;
      if (d < nd) base_s[d] = run + hist[(uint64_t)d * nt + blockIdx.x];
      run += v[q];
    }
  }
  const uint64_t t0 = (uint64_t)blockIdx.x * kRankTile;
  uint32_t key[kRankItems], val[kRankItems], rank[kRankItems];
#pragma unroll
  for (int it = 0; it < kRankItems; ++it) {
    // warp w owns tile positions [w*128, (w+1)*128), item-major then lane
    const uint64_t i = t0 + ((uint64_t)(warp * kRankItems + it) << 5) + lane;
    const bool valid = i < n;
    key[it] = valid ? kin[i] : 0u;
    if (VALS) val[it] = IOTA ? (uint32_t)i : (valid ? vin[i] : 0u);
  }
  __syncthreads();
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int it = 0; it < kRankItems; ++it) {
    const uint64_t i = t0 + ((uint64_t)(warp * kRankItems + it) << 5) + lane;
    const bool valid = i < n;
    const uint32_t d = (key[it] >> shift) & mask;
    const uint32_t peers = digit_peers(d, valid, nbits);
    const uint32_t prior = valid ? wcnt[warp][d] : 0u;
    rank[it] = prior + __popc(peers & lt);
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) wcnt[warp][d] = prior + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
#pragma unroll
  for (int q = 0; q < DPT; ++q) {
    const uint32_t d = threadIdx.x + q * kSortThreads;
    if (d < nd) {
      uint32_t run = 0;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t c = wcnt[w][d];
        wcnt[w][d] = run;
        run += c;
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int it = 0; it < kRankItems; ++it) {
    const uint64_t i = t0 + ((uint64_t)(warp * kRankItems + it) << 5) + lane;
    if (i < n) {
      const uint32_t d = (key[it] >> shift) & mask;
      const uint32_t pos = base_s[d] + wcnt[warp][d] + rank[it];
      kout[pos] = key[it];
      if (VALS) vout[pos] = val[it];
    }
  }
}

// ---- compaction ------------------------------------------------------------

struct UniqueSel {
  const uint32_t* s;
  uint64_t n;
  __device__ bool flag(uint64_t i) const {
    const uint32_t k = s[i];
    return k != kNoKey && (i == 0 || s[i - 1] != k);
  }
  __device__ uint32_t value(uint64_t i) const { return s[i]; }
};

struct MapSel {
  const int32_t* m;
  uint64_t n;
  __device__ bool flag(uint64_t i) const { return m[i] >= 0; }
  __device__ uint32_t value(uint64_t i) const { return (uint32_t)i; }
};

template <class Sel>
__global__ void __launch_bounds__(kSortThreads) compact_count_kernel(Sel sel, uint32_t* tile_cnt) {
  __shared__ uint32_t sm[kWarps];
  const uint64_t start = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kSortItems;
  uint32_t c = 0;
#pragma unroll
  for (int j = 0; j < kSortItems; ++j) {
    const uint64_t i = start + j;
    if (i < sel.n && sel.flag(i)) ++c;
  }
  uint32_t tot;
  block_exclusive_scan<kSortThreads>(c, &tot, sm);
  if (threadIdx.x == 0) tile_cnt[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(1024) scan_tiles_kernel(uint32_t* tile_cnt, uint32_t nb,
                                                          uint32_t* total) {
  __shared__ uint32_t sm[32];
  uint32_t carry = 0;
  for (uint32_t b0 = 0; b0 < nb; b0 += 1024) {
    const uint32_t idx = b0 + threadIdx.x;
    const uint32_t v = idx < nb ? tile_cnt[idx] : 0u;
    uint32_t tot;
    const uint32_t ex = block_exclusive_scan<1024>(v, &tot, sm);
    if (idx < nb) tile_cnt[idx] = carry + ex;
    carry += tot;
  }
  if (threadIdx.x == 0) *total = carry;
}

template <class Sel>
__global__ void __launch_bounds__(kSortThreads)
compact_write_kernel(Sel sel, const uint32_t* __restrict__ tile_off, uint32_t* __restrict__ out) {
  __shared__ uint32_t sm[kWarps];
  const uint64_t start = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kSortItems;
  bool f[kSortItems];
  uint32_t c = 0;
#pragma unroll
  for (int j = 0; j < kSortItems; ++j) {
    const uint64_t i = start + j;
    f[j] = i < sel.n && sel.flag(i);
    c += f[j] ? 1u : 0u;
  }
  uint32_t tot;
  uint32_t pos = tile_off[blockIdx.x] + block_exclusive_scan<kSortThreads>(c, &tot, sm);
#pragma unroll
  for (int j = 0; j < kSortItems; ++j) {
    if (f[j]) out[pos++] = sel.value(start + j);
  }
}

template <class Sel>
void compact(Sel sel, uint32_t* out, uint32_t* count, uint32_t* tmp, cudaStream_t stream) {
  const uint32_t nb = (uint32_t)((sel.n + kTile - 1) / kTile);
  if (nb == 0) {
    cudaMemsetAsync(count, 0, sizeof(uint32_t), stream);
    return;
  }
  note_launches(3);
  compact_count_kernel<Sel><<<nb, kSortThreads, 0, stream>>>(sel, tmp);
  scan_tiles_kernel<<<1, 1024, 0, stream>>>(tmp, nb, count);
  compact_write_kernel<Sel><<<nb, kSortThreads, 0, stream>>>(sel, tmp, out);
}

}  // namespace

int bits_for(uint64_t num_keys) {
  int b = 1;
  while (b < 32 && ((1ull << b) - 1) < num_keys) ++b;   // 2^b - 1 >= K: room for the sentinel
  return b;
}

size_t sort_hist_words(uint64_t n, int bits) {
  (void)bits;
  const uint64_t nt = (n + kRankTile - 1) / kRankTile;
  return (size_t)(kDigits * nt + kDigits);
}

void radix_sort(uint32_t* ka, uint32_t* kb, uint32_t* va, uint32_t* vb, bool with_vals,
                bool iota_vals, uint64_t n, int bits, uint32_t* hist, DevState* st,
                cudaStream_t stream, uint32_t** keys_out, uint32_t** vals_out) {
  (void)st;
  uint32_t *kin = ka, *kout = kb, *vin = va, *vout = vb;
  if (n == 0) {
    *keys_out = kin;
    *vals_out = vin;
    return;
  }
  const uint32_t nt = (uint32_t)((n + kRankTile - 1) / kRankTile);
  uint32_t* totals = hist + (uint64_t)kDigits * nt;
  const PassPlan pl = plan_for(bits);
  int shift = 0;
  for (int p = 0; p < pl.passes; ++p) {
    const int b = pl.per < bits - shift ? pl.per : bits - shift;
    const uint32_t mask = (1u << b) - 1u;
    note_launches(3);
    tile_hist_kernel<<<nt, kSortThreads, 0, stream>>>(kin, n, shift, mask, hist, nt);
    digit_scan_kernel<<<mask + 1, kSortThreads, 0, stream>>>(hist, nt, totals);
    if (!with_vals) {
      tile_scatter_kernel<false, false><<<nt, kSortThreads, 0, stream>>>(
          kin, nullptr, kout, nullptr, n, shift, b, hist, nt, totals);
    } else if (p == 0 && iota_vals) {
      tile_scatter_kernel<true, true><<<nt, kSortThreads, 0, stream>>>(
          kin, nullptr, kout, vout, n, shift, b, hist, nt, totals);
    } else {
      tile_scatter_kernel<true, false><<<nt, kSortThreads, 0, stream>>>(
          kin, vin, kout, vout, n, shift, b, hist, nt, totals);
    }
    uint32_t* t = kin; kin = kout; kout = t;
    t = vin; vin = vout; vout = t;
    shift += b;
  }
  *keys_out = kin;
  *vals_out = vin;
}

size_t compact_tmp_words(uint64_t n) { return (size_t)((n + kTile - 1) / kTile + 1); }

void unique_sorted(const uint32_t* sorted, uint64_t n, uint32_t* out, uint32_t* count,
                   uint32_t* tmp, cudaStream_t stream) {
  compact(UniqueSel{sorted, n}, out, count, tmp, stream);
}

void compact_replica_keys(const int32_t* map_w, uint64_t K, uint32_t* out, uint32_t* count,
                          uint32_t* tmp, cudaStream_t stream) {
  compact(MapSel{map_w, K}, out, count, tmp, stream);
}

}  // namespace adapm
