// Stable LSD radix sort of uint32 keys (optionally with uint32 values) and
// stream compaction, for the intent table (sort + unique of the keys of one
// Intent call, Sec. 3) and for push (grouping a batch's delta rows by key).
//
// One pass over `b` <= 8 key bits = three kernels:
//   hist    per tile of 2048 keys, digit counts (warp-aggregated with
//           __match_any_sync, so a skewed digit costs one shared atomic per
//           warp and item)
//   scan    one block per digit: exclusive prefix of that digit's counts
//           over tiles (digit-major table), digit total
//   scatter per tile: stable rank of each key among equal digits of the
//           tile (warp-ordered match_any ranks + per-warp digit counters),
//           global position = digit base + tile prefix + rank
// Only ceil(log2(K + 1)) bits are sorted, split evenly over
// ceil(bits / 8) passes.
#include "internal.cuh"

namespace adapm {

namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 8;
constexpr int kTile = kSortThreads * kSortItems;
constexpr int kBuckets = 256;
constexpr int kWarps = kSortThreads / 32;

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
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

__global__ void __launch_bounds__(kSortThreads)
radix_hist_kernel(const uint32_t* __restrict__ keys, uint64_t n, int shift, uint32_t mask,
                  uint32_t* __restrict__ hist, uint32_t nb) {
  __shared__ uint32_t cnt[kBuckets];
  for (int i = threadIdx.x; i < kBuckets; i += kSortThreads) cnt[i] = 0;
  __syncthreads();
  const uint64_t tile = (uint64_t)blockIdx.x * kTile;
  const int lane = threadIdx.x & 31;
  uint32_t k[kSortItems];
#pragma unroll
  for (int it = 0; it < kSortItems; ++it) {
    const uint64_t i = tile + (uint64_t)it * kSortThreads + threadIdx.x;
    k[it] = i < n ? keys[i] : 0u;
  }
#pragma unroll
  for (int it = 0; it < kSortItems; ++it) {
    const uint64_t i = tile + (uint64_t)it * kSortThreads + threadIdx.x;
    const bool valid = i < n;
    const uint32_t d = valid ? ((k[it] >> shift) & mask) : 0xFFFFFFFFu;
    const uint32_t peers = __match_any_sync(0xFFFFFFFFu, d);
    if (valid && lane == __ffs(peers) - 1) atomicAdd(&cnt[d], (uint32_t)__popc(peers));
  }
  __syncthreads();
  for (uint32_t d = threadIdx.x; d <= mask; d += kSortThreads)
    hist[(uint64_t)d * nb + blockIdx.x] = cnt[d];
}

__global__ void __launch_bounds__(kSortThreads)
radix_scan_kernel(uint32_t* __restrict__ hist, uint32_t nb, uint32_t* __restrict__ totals) {
  __shared__ uint32_t sm[kWarps];
  uint32_t* row = hist + (uint64_t)blockIdx.x * nb;
  uint32_t carry = 0;
  for (uint32_t b0 = 0; b0 < nb; b0 += kSortThreads) {
    const uint32_t idx = b0 + threadIdx.x;
    const uint32_t v = idx < nb ? row[idx] : 0u;
    uint32_t tot;
    const uint32_t ex = block_exclusive_scan<kSortThreads>(v, &tot, sm);
    if (idx < nb) row[idx] = carry + ex;
    carry += tot;
  }
  if (threadIdx.x == 0) totals[blockIdx.x] = carry;
}

template <bool VALS, bool IOTA>
__global__ void __launch_bounds__(kSortThreads)
radix_scatter_kernel(const uint32_t* __restrict__ kin, const uint32_t* __restrict__ vin,
                     uint32_t* __restrict__ kout, uint32_t* __restrict__ vout, uint64_t n,
                     int shift, uint32_t mask, const uint32_t* __restrict__ hist, uint32_t nb,
                     const uint32_t* __restrict__ totals) {
  __shared__ uint32_t wcnt[kWarps][kBuckets];
  __shared__ uint32_t base_s[kBuckets];
  __shared__ uint32_t sm[kWarps];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t nd = mask + 1;
  for (int i = threadIdx.x; i < kWarps * kBuckets; i += kSortThreads) (&wcnt[0][0])[i] = 0;
  {
    // kSortThreads == kBuckets: thread d owns digit d
    const uint32_t t = threadIdx.x < nd ? totals[threadIdx.x] : 0u;
    uint32_t tot;
    const uint32_t ex = block_exclusive_scan<kSortThreads>(t, &tot, sm);
    if (threadIdx.x < nd) base_s[threadIdx.x] = ex + hist[(uint64_t)threadIdx.x * nb + blockIdx.x];
  }
  const uint64_t tile = (uint64_t)blockIdx.x * kTile;
  uint32_t key[kSortItems], val[kSortItems], rank[kSortItems];
#pragma unroll
  for (int it = 0; it < kSortItems; ++it) {
    // warp w owns tile positions [w*256, (w+1)*256), item-major then lane
    const uint64_t i = tile + ((uint64_t)(warp * kSortItems + it) << 5) + lane;
    const bool valid = i < n;
    key[it] = valid ? kin[i] : 0u;
    if (VALS) val[it] = IOTA ? (uint32_t)i : (valid ? vin[i] : 0u);
  }
  __syncthreads();
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int it = 0; it < kSortItems; ++it) {
    const uint64_t i = tile + ((uint64_t)(warp * kSortItems + it) << 5) + lane;
    const bool valid = i < n;
    const uint32_t d = valid ? ((key[it] >> shift) & mask) : 0xFFFFFFFFu;
    const uint32_t peers = __match_any_sync(0xFFFFFFFFu, d);
    const uint32_t prior = valid ? wcnt[warp][d] : 0u;
    rank[it] = prior + __popc(peers & lt);
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) wcnt[warp][d] = prior + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  if (threadIdx.x < nd) {
    uint32_t run = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const uint32_t c = wcnt[w][threadIdx.x];
      wcnt[w][threadIdx.x] = run;
      run += c;
    }
  }
  __syncthreads();
#pragma unroll
  for (int it = 0; it < kSortItems; ++it) {
    const uint64_t i = tile + ((uint64_t)(warp * kSortItems + it) << 5) + lane;
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

size_t sort_hist_words(uint64_t n) {
  const uint64_t nb = (n + kTile - 1) / kTile;
  return (size_t)(kBuckets * nb + kBuckets);
}

void radix_sort(uint32_t* ka, uint32_t* kb, uint32_t* va, uint32_t* vb, bool with_vals,
                bool iota_vals, uint64_t n, int bits, uint32_t* hist, cudaStream_t stream,
                uint32_t** keys_out, uint32_t** vals_out) {
  uint32_t *kin = ka, *kout = kb, *vin = va, *vout = vb;
  if (n == 0) {
    *keys_out = kin;
    *vals_out = vin;
    return;
  }
  const uint32_t nb = (uint32_t)((n + kTile - 1) / kTile);
  uint32_t* totals = hist + (uint64_t)kBuckets * nb;
  const int passes = (bits + 7) / 8;
  const int per = (bits + passes - 1) / passes;
  int shift = 0;
  for (int p = 0; p < passes; ++p) {
    const int b = per < bits - shift ? per : bits - shift;
    const uint32_t mask = (1u << b) - 1u;
    note_launches(3);
    radix_hist_kernel<<<nb, kSortThreads, 0, stream>>>(kin, n, shift, mask, hist, nb);
    radix_scan_kernel<<<mask + 1, kSortThreads, 0, stream>>>(hist, nb, totals);
    if (!with_vals) {
      radix_scatter_kernel<false, false><<<nb, kSortThreads, 0, stream>>>(
          kin, nullptr, kout, nullptr, n, shift, mask, hist, nb, totals);
    } else if (p == 0 && iota_vals) {
      radix_scatter_kernel<true, true><<<nb, kSortThreads, 0, stream>>>(
          kin, nullptr, kout, vout, n, shift, mask, hist, nb, totals);
    } else {
      radix_scatter_kernel<true, false><<<nb, kSortThreads, 0, stream>>>(
          kin, vin, kout, vout, n, shift, mask, hist, nb, totals);
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
