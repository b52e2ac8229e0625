// Stable LSD radix sort of uint32 keys carrying their positions, for push
// (grouping a batch's delta rows by key, App. B.1.2), and stream compaction.
//
// Only ceil(log2(K + 1)) key bits are sorted, in ceil(bits / 9) passes of at
// most 9 bits (512 buckets): 27-bit keys (100M) take 3 passes.  The whole
// sort is ONE cooperative launch of B blocks (all resident at once), block b
// owning the contiguous chunk [b*n/B, (b+1)*n/B) of every pass.  The first
// pass's digit counts of each chunk go to column b of a 512 x B table, then
// every pass is
//   1. scan    grid barrier; warp j scans row d = j of the table (the
//              exclusive prefix of digit d over the chunks) and its total
//   2. scatter grid barrier; digit bases = exclusive scan of the totals;
//              the chunk is ranked in sub-tiles of 2048 keys (a warp-level
//              multi-split: one ballot per digit bit gives the lanes with
//              equal digits), reordered by digit in shared memory and
//              written out in runs of equal digit (coalesced stores); each
//              written key adds to the next pass's table, in the column of
//              the chunk its position falls in (one atomic per distinct
//              digit and chunk of a warp)
// so a pass costs two grid barriers.  With one sub-tile per chunk
// (n <= 2048 B) the first pass's ranks are kept in registers from the
// count.
//
// The grid barrier is a monotonic arrival counter in DevState: the host
// knows how many barriers each launch passes and hands the next launch its
// starting value.  Its wait is bounded; a wait that gives up sets
// ERR_TIMEOUT and the kernel returns, and since all later barriers need
// every block, the whole launch stops within one bounded wait.
#include "internal.cuh"

namespace adapm {

namespace {

constexpr int kSortThreads = 256;
constexpr int kWarps = kSortThreads / 32;
constexpr int kItems = 8;                          // keys per thread per sub-tile (largest)
constexpr int kSub = kSortThreads * kItems;        // 2048 keys per sub-tile (largest)
constexpr int kSubMin = kSortThreads * 4;          // sub-tile of small batches (4 keys per thread)
constexpr int kRadixBits = 9;
constexpr int kDigits = 1 << kRadixBits;           // 512
constexpr int kDPT = kDigits / kSortThreads;       // digits per thread (2)
constexpr uint32_t kMaxSortBlocks = 4096;
constexpr uint32_t kSpinLimit = 1u << 21;          // polls of one barrier wait
constexpr int kScratchHead = 32;                   // words before the totals
constexpr int kScanQ = 5;                          // digit-row entries per lane, four warps a row

constexpr int kCompactItems = 8;                   // compaction: keys per thread
constexpr int kTile = kSortThreads * kCompactItems;

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
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

struct SortArgs {
  const uint32_t* raw;
  uint64_t n;
  uint64_t K;
  uint32_t* ka;
  uint32_t* kb;
  uint32_t* va;
  uint32_t* vb;
  uint32_t* table;        // kDigits x gridDim.x (digit-major)
  uint32_t* totals;       // kDigits
  DevState* st;
  uint32_t* clear0;              // words set to zero by the launch (nullptr: none)
  uint32_t* clear1;
  unsigned long long bar_base;   // st->bar_arrivals when the launch starts
  // Plan check (cooperative launch): with plan_keys, the blocks first compare
  // raw with plan_keys position by position; a mismatch stores plan_seq in
  // *plan_word, and after a grid barrier the sort runs only if it did.
  const uint32_t* plan_keys;
  uint32_t* plan_word;
  uint32_t plan_seq;
  int phase;                     // -1: every phase, grid barriers between (cooperative launch);
                                 // k >= 0: phase k alone (0 count, 1 + 2p scan, 2 + 2p scatter of pass p)
  int allow_nokey;
  int passes;
  int per;
  int bits;
};

struct SortSmem {
  uint32_t wcnt[kWarps][kDigits];   // per-warp digit counts, then warp offsets
  uint32_t sk[kSub];                // sub-tile keys in digit order
  uint32_t sv[kSub];                // their positions
  uint32_t base[kDigits];           // output position of the chunk's next key per digit
  uint32_t lofs[kDigits];           // first index of each digit in the reordered sub-tile
  uint32_t cnt[kDigits];            // digit counts (chunk in step 1, sub-tile in step 3)
  uint32_t scan[kWarps];
  int abort;
};

__device__ __forceinline__ unsigned long long ld_acquire64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Grid barrier on a monotonic arrival counter: the k-th barrier of a launch
// waits, bounded, until the counter reaches base + k * gridDim.x.  Arrival
// is a release add, the wait an acquire load.  Block-wide: every thread
// calls it.
__device__ bool grid_barrier(const SortArgs& a, uint32_t& nbar, SortSmem& sm) {
  __syncthreads();
  ++nbar;
  if (threadIdx.x == 0) {
    const unsigned long long target = a.bar_base + (unsigned long long)nbar * gridDim.x;
    asm volatile("red.release.gpu.global.add.u64 [%0], 1;" ::"l"(&a.st->bar_arrivals) : "memory");
    uint32_t it = 0;
    while (ld_acquire64(&a.st->bar_arrivals) < target) {
      if (++it > kSpinLimit) {
        set_error(a.st, ERR_TIMEOUT);
        sm.abort = 1;
        break;
      }
    }
  }
  __syncthreads();
  return sm.abort == 0;
}

// Load a sub-tile [s0, s1) (warp w owns positions s0 + [256w, 256w + 256),
// item-major then lane) and rank every key among the equal digits before it:
// afterwards sm.wcnt[w][d] = keys of digit d in warps < w, sm.cnt[d] = keys
// of digit d in the sub-tile, rank[it] = earlier keys of the same digit in
// the same warp.  `first`: keys come from the caller's array (mapped to
// kNoKey when out of range, positions are the indices).
template <bool POS, int ITEMS>
__device__ __forceinline__ void load_rank(const SortArgs& a, const uint32_t* kin, const uint32_t* vin,
                                          bool first, uint64_t s0, uint64_t s1, int shift, int nbits,
                                          uint32_t (&key)[ITEMS], uint32_t (&val)[ITEMS],
                                          uint32_t (&rank)[ITEMS], bool& bad, SortSmem& sm) {
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < kWarps * kDigits; i += kSortThreads) (&sm.wcnt[0][0])[i] = 0;
#pragma unroll
  for (int it = 0; it < ITEMS; ++it) {
    const uint64_t i = s0 + ((uint64_t)(warp * ITEMS + it) << 5) + lane;
    const bool valid = i < s1;
    uint32_t k = 0;
    if (valid) {
      if (first) {
        k = __ldg(kin + i);
        if (k >= a.K) {
          if (!(a.allow_nokey && k == kNoKey)) bad = true;
          k = kNoKey;
        }
      } else {
        k = __ldcg(kin + i);
      }
    }
    key[it] = k;
    if (POS) val[it] = first ? (uint32_t)i : (valid ? __ldcg(vin + i) : 0u);
  }
  __syncthreads();
  const uint32_t mask = (1u << nbits) - 1u;
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int it = 0; it < ITEMS; ++it) {
    const uint64_t i = s0 + ((uint64_t)(warp * ITEMS + it) << 5) + lane;
    const bool valid = i < s1;
    const uint32_t d = (key[it] >> shift) & mask;
    const uint32_t peers = digit_peers(d, valid, nbits);
    const uint32_t prior = valid ? sm.wcnt[warp][d] : 0u;
    rank[it] = prior + __popc(peers & lt);
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) sm.wcnt[warp][d] = prior + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
#pragma unroll
  for (int q = 0; q < kDPT; ++q) {
    const int d = threadIdx.x * kDPT + q;
    uint32_t run = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const uint32_t c = sm.wcnt[w][d];
      sm.wcnt[w][d] = run;
      run += c;
    }
    sm.cnt[d] = run;
  }
  __syncthreads();
}

// Number of grid barriers one sort_kernel launch passes.
__host__ __device__ constexpr uint32_t sort_barriers(int passes) { return 2u * (uint32_t)passes; }

// What one sort launch runs: every phase with grid barriers between
// (cooperative), or one phase of a phased sort.  A phased launch is compiled
// with its own phase's code alone (registers, occupancy).
enum SortKind { kSortAll = 0, kSortCount = 1, kSortScan = 2, kSortScatter = 3 };

template <bool POS, int ITEMS, int KIND>
__global__ void __launch_bounds__(kSortThreads, 4) sort_kernel(SortArgs a) {
  constexpr int SUB = kSortThreads * ITEMS;   // keys per sub-tile
  __shared__ SortSmem sm;
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const uint32_t B = gridDim.x;
  const uint32_t b = blockIdx.x;
  constexpr bool coop = KIND == kSortAll;
  if (b == 0 && threadIdx.x == 0 && (coop || a.phase == 0)) {
    if (a.clear0) *a.clear0 = 0u;
    if (a.clear1) *a.clear1 = 0u;
  }
  // an earlier sort gave up (the barrier state is unknown): do nothing
  if (threadIdx.x == 0) sm.abort = (ld_acquire(&a.st->errors) & ERR_TIMEOUT) ? 1 : 0;
  __syncthreads();
  if (sm.abort) return;
  uint32_t nbar = 0;
  if (coop && a.plan_keys) {
    // the plan holds this sort's result iff the push's keys equal the keys it
    // was made from at every position (out-of-range keys all counting as the
    // sentinel); every key is read once, so out-of-range keys are reported
    // here as the sort's first pass would
    constexpr int U = 4;
    bool miss = false, bad = false;
    const uint64_t stride = (uint64_t)gridDim.x * kSortThreads;
    for (uint64_t i0 = (uint64_t)b * kSortThreads + threadIdx.x; i0 < a.n; i0 += U * stride) {
      uint32_t kv[U], xv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint64_t i = i0 + u * stride;
        kv[u] = i < a.n ? __ldg(a.raw + i) : 0u;
        xv[u] = i < a.n ? __ldg(a.plan_keys + i) : 0u;
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (i0 + u * stride >= a.n) continue;
        const uint32_t k = kv[u], x = xv[u];
        if (k >= a.K && !(a.allow_nokey && k == kNoKey)) bad = true;
        miss |= (k < a.K ? k : kNoKey) != (x < a.K ? x : kNoKey);
      }
    }
    if (__any_sync(0xFFFFFFFFu, miss) && lane == 0 && atomicExch(a.plan_word, a.plan_seq) != a.plan_seq)
      atomicAdd(&a.st->plan_misses, 1ull);
    if (__any_sync(0xFFFFFFFFu, bad) && lane == 0) set_error(a.st, ERR_KEY_RANGE);
    if (!grid_barrier(a, nbar, sm)) return;
    // the plan matched: arrive at every later barrier of the launch at once
    // (the host counts them) and stop
    if (threadIdx.x == 0) {
      sm.abort = ld_acquire(a.plan_word) != a.plan_seq ? 2 : 0;
      if (sm.abort == 2) {
        const unsigned long long nb = sort_barriers(a.passes);
        asm volatile("red.release.gpu.global.add.u64 [%0], %1;" ::"l"(&a.st->bar_arrivals), "l"(nb) : "memory");
      }
    }
    __syncthreads();
    if (sm.abort) return;
  }
  auto run = [&](int ph) { return coop || a.phase == ph; };
  constexpr bool has_count = KIND == kSortAll || KIND == kSortCount;
  constexpr bool has_scan = KIND == kSortAll || KIND == kSortScan;
  constexpr bool has_scatter = KIND == kSortAll || KIND == kSortScatter;
    const uint64_t chunk = (a.n + B - 1) / B;
  const uint64_t c0 = a.n < b * chunk ? a.n : b * chunk;
  const uint64_t c1 = a.n < c0 + chunk ? a.n : c0 + chunk;
  const bool single = c1 - c0 <= (uint64_t)SUB;
  uint32_t* const table0 = a.table;                       // passes 0, 2, ...
  uint32_t* const table1 = a.table + (uint64_t)kDigits * B;   // passes 1, 3, ...
  const uint32_t* kin = a.raw;
  const uint32_t* vin = nullptr;
  uint32_t* kout = a.ka;
  uint32_t* vout = a.va;
  uint32_t key[ITEMS], val[ITEMS], rank[ITEMS];
  bool bad = false;
  // 0. first pass digit counts of the chunk (ranks kept when one sub-tile
  // and the scatter follows in this launch)
  if (has_count && run(0)) {
    const int nbits = a.per < a.bits ? a.per : a.bits;
    const uint32_t mask = (1u << nbits) - 1u;
    if (single && coop) {
      load_rank<POS, ITEMS>(a, kin, vin, true, c0, c1, 0, nbits, key, val, rank, bad, sm);
    } else {
      for (int d = threadIdx.x; d < kDigits; d += kSortThreads) sm.cnt[d] = 0;
      __syncthreads();
      // ITEMS keys per thread and round, their loads issued together
      for (uint64_t i0 = c0 + threadIdx.x; i0 < c1; i0 += (uint64_t)kSortThreads * ITEMS) {
        uint32_t kk[ITEMS];
#pragma unroll
        for (int it = 0; it < ITEMS; ++it) {
          const uint64_t i = i0 + (uint64_t)it * kSortThreads;
          kk[it] = i < c1 ? __ldg(kin + i) : 0u;
        }
#pragma unroll
        for (int it = 0; it < ITEMS; ++it) {
          if (i0 + (uint64_t)it * kSortThreads >= c1) continue;
          uint32_t k = kk[it];
          if (k >= a.K) {
            if (!(a.allow_nokey && k == kNoKey)) bad = true;
            k = kNoKey;
          }
          atomicAdd(&sm.cnt[k & mask], 1u);
        }
      }
      __syncthreads();
    }
    for (uint32_t d = threadIdx.x; d <= mask; d += kSortThreads) table0[(uint64_t)d * B + b] = sm.cnt[d];
    if (__any_sync(0xFFFFFFFFu, bad) && lane == 0) set_error(a.st, ERR_KEY_RANGE);
  }
  if (coop && !grid_barrier(a, nbar, sm)) return;
  int shift = 0;
  for (int p = 0; p < a.passes; ++p) {
    const bool first = p == 0;
    const bool more = p + 1 < a.passes;
    const int nbits = a.per < a.bits - shift ? a.per : a.bits - shift;
    const uint32_t mask = (1u << nbits) - 1u;
    const int nshift = shift + nbits;   // next pass
    const int nnbits = more ? (a.per < a.bits - nshift ? a.per : a.bits - nshift) : 0;
    const uint32_t nmask = (1u << nnbits) - 1u;
    uint32_t* tcur = (p & 1) ? table1 : table0;
    uint32_t* tnext = (p & 1) ? table0 : table1;
    // 1. exclusive prefix of each digit over the chunks and digit totals.
    // Up to 16 chunks: one thread per digit (its row in one round of
    // loads); 129 to 640: four warps per digit row, a quarter each in one
    // round of coalesced loads, combined through shared memory; otherwise
    // one warp per digit row, read in batches.  Every block
    // also clears its own column of the next pass's table.
    if (has_scan && run(1 + 2 * p)) {
    if (more)
      for (uint32_t d = threadIdx.x; d <= nmask; d += kSortThreads) tnext[(uint64_t)d * B + b] = 0u;
    if (B <= 16) {
      for (uint32_t d = b * kSortThreads + threadIdx.x; d <= mask; d += B * kSortThreads) {
        uint32_t* row = tcur + (uint64_t)d * B;
        uint32_t v[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = (uint32_t)j < B ? __ldcg(row + j) : 0u;
        uint32_t run = 0;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          if ((uint32_t)j < B) row[j] = run;
          run += v[j];
        }
        a.totals[d] = run;
      }
    } else if (B > 128 && B <= 4 * 32 * kScanQ) {
      // four warps per digit row (a quarter each, kept in registers), two
      // rows per block at a time
      const uint32_t half = warp >> 2, quarter = warp & 3;
      const uint32_t seg = (B + 3) / 4;
      const uint32_t jb = quarter * seg;
      const uint32_t je = jb + seg < B ? jb + seg : B;
      for (uint32_t dp = b; dp * 2 <= mask; dp += B) {   // block-uniform trip count
        const uint32_t d = dp * 2 + half;
        const bool act = d <= mask;
        uint32_t* row = tcur + (uint64_t)d * B;
        uint32_t v[kScanQ], x[kScanQ];
#pragma unroll
        for (int q = 0; q < kScanQ; ++q) {
          const uint32_t j = jb + q * 32 + lane;
          v[q] = act && j < je ? __ldcg(row + j) : 0u;
        }
        uint32_t carry = 0;
#pragma unroll
        for (int q = 0; q < kScanQ; ++q) {
          uint32_t y = v[q];
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, y, o);
            if (lane >= o) y += t;
          }
          x[q] = carry + y - v[q];   // exclusive within the quarter
          carry += __shfl_sync(0xFFFFFFFFu, y, 31);
        }
        if (lane == 0) sm.scan[warp] = carry;
        __syncthreads();
        uint32_t before = 0;
        for (uint32_t w2 = 0; w2 < quarter; ++w2) before += sm.scan[half * 4 + w2];
#pragma unroll
        for (int q = 0; q < kScanQ; ++q) {
          const uint32_t j = jb + q * 32 + lane;
          if (act && j < je) row[j] = before + x[q];
        }
        if (act && quarter == 3 && lane == 0) a.totals[d] = before + carry;
        __syncthreads();
      }
    } else {
      // (the first pass's ranks stay in registers with positions: a smaller batch)
      constexpr int QB = POS ? 8 : 16;
      for (uint32_t d = b * kWarps + warp; d <= mask; d += B * kWarps) {
        uint32_t* row = tcur + (uint64_t)d * B;
        uint32_t carry = 0;
        for (uint32_t j0 = 0; j0 < B; j0 += 32 * QB) {
          uint32_t v[QB];
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            const uint32_t j = j0 + q * 32 + lane;
            v[q] = j < B ? __ldcg(row + j) : 0u;
          }
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            uint32_t x = v[q];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
              const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
              if (lane >= o) x += y;
            }
            const uint32_t j = j0 + q * 32 + lane;
            if (j < B) row[j] = carry + x - v[q];
            carry += __shfl_sync(0xFFFFFFFFu, x, 31);
          }
        }
        if (lane == 0) a.totals[d] = carry;
      }
    }
    }   // scan phase
    if (coop && !grid_barrier(a, nbar, sm)) return;
    // 2. scatter: digit bases, then the chunk's sub-tiles in order; each
    // written key is counted for the next pass in the chunk it lands in
    if (has_scatter && run(2 + 2 * p)) {
    {
      uint32_t v[kDPT], local = 0;
#pragma unroll
      for (int q = 0; q < kDPT; ++q) {
        const uint32_t d = threadIdx.x * kDPT + q;
        v[q] = d <= mask ? __ldcg(a.totals + d) : 0u;
        local += v[q];
      }
      uint32_t total;
      uint32_t run = block_exclusive_scan<kSortThreads>(local, &total, sm.scan);
#pragma unroll
      for (int q = 0; q < kDPT; ++q) {
        const uint32_t d = threadIdx.x * kDPT + q;
        sm.base[d] = run + (d <= mask ? __ldcg(tcur + (uint64_t)d * B + b) : 0u);
        run += v[q];
      }
    }
    for (uint64_t s0 = c0; s0 < c1; s0 += SUB) {
      const uint64_t s1 = s0 + SUB < c1 ? s0 + SUB : c1;
      // (the first pass's ranks survive from the count only within one launch)
      if (!(single && first && coop))
        load_rank<POS, ITEMS>(a, kin, vin, first, s0, s1, shift, nbits, key, val, rank, bad, sm);
      {
        uint32_t local = 0;
#pragma unroll
        for (int q = 0; q < kDPT; ++q) local += sm.cnt[threadIdx.x * kDPT + q];
        uint32_t total;
        uint32_t run = block_exclusive_scan<kSortThreads>(local, &total, sm.scan);
#pragma unroll
        for (int q = 0; q < kDPT; ++q) {
          const int d = threadIdx.x * kDPT + q;
          sm.lofs[d] = run;
          run += sm.cnt[d];
        }
      }
      __syncthreads();
#pragma unroll
      for (int it = 0; it < ITEMS; ++it) {
        const uint64_t i = s0 + ((uint64_t)(warp * ITEMS + it) << 5) + lane;
        if (i < s1) {
          const uint32_t d = (key[it] >> shift) & mask;
          const uint32_t lp = sm.lofs[d] + sm.wcnt[warp][d] + rank[it];
          sm.sk[lp] = key[it];
          if (POS) sm.sv[lp] = val[it];
        }
      }
      __syncthreads();
      const uint32_t m = (uint32_t)(s1 - s0);
      for (uint32_t i0 = 0; i0 < m; i0 += kSortThreads) {   // block-uniform trip count
        const uint32_t i = i0 + threadIdx.x;
        uint32_t tag = 0xFFFFFFFFu;
        if (i < m) {
          const uint32_t k = sm.sk[i];
          const uint32_t d = (k >> shift) & mask;
          const uint32_t pos = sm.base[d] + (i - sm.lofs[d]);
          // (positions come from the digit tables in scratch memory; one out of
          // range is skipped and reported, never written)
          if (pos < a.n) {
            kout[pos] = k;
            if (POS) vout[pos] = sm.sv[i];
            if (more) tag = (((k >> nshift) & nmask) << 12) | (uint32_t)(pos / chunk);
          } else {
            set_error(a.st, ERR_INTERNAL);
          }
        }
        if (more) {
          // one atomic per distinct (digit, chunk) of the warp
          const uint32_t peers = __match_any_sync(0xFFFFFFFFu, tag);
          if (tag != 0xFFFFFFFFu && lane == __ffs(peers) - 1)
            atomicAdd(tnext + (uint64_t)(tag >> 12) * B + (tag & 0xFFFu), (uint32_t)__popc(peers));
        }
      }
      __syncthreads();
#pragma unroll
      for (int q = 0; q < kDPT; ++q) {
        const int d = threadIdx.x * kDPT + q;
        sm.base[d] += sm.cnt[d];
      }
      __syncthreads();
    }
    }   // scatter phase
    if (coop && more) {
      if (!grid_barrier(a, nbar, sm)) return;
    }
    kin = kout;
    vin = vout;
    kout = kout == a.ka ? a.kb : a.ka;
    vout = vout == a.va ? a.vb : a.va;
    shift = nshift;
  }
}

// ---- compaction ------------------------------------------------------------

struct MapSel {
  const int32_t* m;
  uint64_t n;
  __device__ bool flag(uint64_t i) const { return m[i] >= 0; }
  __device__ uint32_t value(uint64_t i) const { return (uint32_t)i; }
};

// the first copy of every valid key of a sorted array (the distinct keys, ascending)
struct HeadSel {
  const uint32_t* sk;
  uint64_t n;
  __device__ bool flag(uint64_t i) const {
    const uint32_t k = sk[i];
    return k != kNoKey && (i == 0 || sk[i - 1] != k);
  }
  __device__ uint32_t value(uint64_t i) const { return sk[i]; }
};

template <class Sel>
__global__ void __launch_bounds__(kSortThreads) compact_count_kernel(Sel sel, uint32_t* tile_cnt) {
  __shared__ uint32_t sm[kWarps];
  const uint64_t start = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kCompactItems;
  uint32_t c = 0;
#pragma unroll
  for (int j = 0; j < kCompactItems; ++j) {
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
  const uint64_t start = (uint64_t)blockIdx.x * kTile + (uint64_t)threadIdx.x * kCompactItems;
  bool f[kCompactItems];
  uint32_t c = 0;
#pragma unroll
  for (int j = 0; j < kCompactItems; ++j) {
    const uint64_t i = start + j;
    f[j] = i < sel.n && sel.flag(i);
    c += f[j] ? 1u : 0u;
  }
  uint32_t tot;
  uint32_t pos = tile_off[blockIdx.x] + block_exclusive_scan<kSortThreads>(c, &tot, sm);
#pragma unroll
  for (int j = 0; j < kCompactItems; ++j) {
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

// Resident blocks per SM of one sort_kernel instance (its shared memory and
// registers), looked up once.
template <bool POS, int ITEMS>
int sort_blocks_per_sm() {
  static const int occ = [] {
    int o = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, sort_kernel<POS, ITEMS, kSortAll>, kSortThreads, 0) !=
        cudaSuccess) {
      cudaGetLastError();
      o = 1;
    }
    return o < 1 ? 1 : o;
  }();
  return occ;
}

template <bool POS, int ITEMS>
cudaError_t launch_sort(SortArgs& a, unsigned long long* bar_base, int sms, cudaStream_t stream) {
  constexpr uint64_t SUB = (uint64_t)kSortThreads * ITEMS;
  const int occ = sort_blocks_per_sm<POS, ITEMS>();
  uint64_t B = (a.n + SUB - 1) / SUB;
  // A launch that checks a plan expects it to match and only to check: one
  // block per SM needs room for one block on each SM, not four, before it can
  // start beside other streams' kernels (a miss then sorts with that grid).
  const uint64_t resident = (uint64_t)sms * (a.plan_keys ? 1 : (occ < 4 ? occ : 4));
  if (B > resident) B = resident;
  if (B > kMaxSortBlocks) B = kMaxSortBlocks;
  if (B < 1) B = 1;
  a.bar_base = *bar_base;
  a.phase = -1;
  void* params[] = {&a};
  note_launches(1);
  const cudaError_t e = cudaLaunchCooperativeKernel((const void*)sort_kernel<POS, ITEMS, kSortAll>, dim3((unsigned)B),
                                                    dim3(kSortThreads), params, 0, stream);
  if (e == cudaSuccess) *bar_base += (unsigned long long)(sort_barriers(a.passes) + (a.plan_keys ? 1u : 0u)) * B;
  return e;
}

// The same sort as 1 + 2 * passes ordinary launches, one phase each: the
// kernel boundaries are its barriers, so nothing waits on another block and
// the blocks need not be resident together (for a stream that runs beside
// other work).  B = one block per sub-tile of keys.
template <bool POS, int ITEMS>
cudaError_t launch_sort_phased(SortArgs& a, cudaStream_t stream) {
  constexpr uint64_t SUB = (uint64_t)kSortThreads * ITEMS;
  uint64_t B = (a.n + SUB - 1) / SUB;
  if (B > kMaxSortBlocks) B = kMaxSortBlocks;
  if (B < 1) B = 1;
  a.bar_base = 0;
  const int phases = 1 + 2 * a.passes;
  note_launches((uint64_t)phases);
  for (int ph = 0; ph < phases; ++ph) {
    a.phase = ph;
    if (ph == 0)
      sort_kernel<POS, ITEMS, kSortCount><<<(unsigned)B, kSortThreads, 0, stream>>>(a);
    else if (ph & 1)
      sort_kernel<POS, ITEMS, kSortScan><<<(unsigned)B, kSortThreads, 0, stream>>>(a);
    else
      sort_kernel<POS, ITEMS, kSortScatter><<<(unsigned)B, kSortThreads, 0, stream>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace

int bits_for(uint64_t num_keys) {
  int b = 1;
  while (b < 32 && ((1ull << b) - 1) < num_keys) ++b;   // 2^b - 1 >= K: room for the sentinel
  return b;
}

size_t sort_scratch_words(uint64_t n) {
  uint64_t rows = (n + kSubMin - 1) / kSubMin;
  if (rows > kMaxSortBlocks) rows = kMaxSortBlocks;
  if (rows < 1) rows = 1;
  return (size_t)(kScratchHead + kDigits + 2 * rows * kDigits);   // totals, two tables
}

int sort_passes(int bits) { return plan_for(bits).passes; }

cudaError_t sort_keys(const uint32_t* raw, uint64_t n, uint64_t K, bool allow_nokey, int bits,
                      uint32_t* ka, uint32_t* kb, uint32_t* va, uint32_t* vb, uint32_t* scratch, int sms,
                      DevState* st, unsigned long long* bar_base, uint32_t* clear0, uint32_t* clear1,
                      cudaStream_t stream, uint32_t** keys_out, uint32_t** pos_out, const uint32_t* plan_keys,
                      uint32_t* plan_word, uint32_t plan_seq, bool phased) {
  const PassPlan pl = plan_for(bits);
  if (keys_out) *keys_out = pl.passes % 2 ? ka : kb;
  if (pos_out) *pos_out = va ? (pl.passes % 2 ? va : vb) : nullptr;
  if (n == 0) return cudaSuccess;
  SortArgs a;
  a.plan_keys = (plan_keys && plan_word && !phased) ? plan_keys : nullptr;
  a.plan_word = plan_word;
  a.plan_seq = plan_seq;
  a.phase = -1;
  a.raw = raw;
  a.n = n;
  a.K = K;
  a.ka = ka;
  a.kb = kb;
  a.va = va;
  a.vb = vb;
  a.totals = scratch + kScratchHead;
  a.table = scratch + kScratchHead + kDigits;
  a.st = st;
  a.clear0 = clear0;
  a.clear1 = clear1;
  a.allow_nokey = allow_nokey ? 1 : 0;
  a.passes = pl.passes;
  a.per = pl.per;
  a.bits = bits;
  // batches that would give fewer blocks than SMs take sub-tiles of half the
  // size: twice the blocks, half the ranking work per block
  const bool small = (n + kSub - 1) / kSub < (uint64_t)sms;
  if (phased) {
    if (small) return va ? launch_sort_phased<true, 4>(a, stream) : launch_sort_phased<false, 4>(a, stream);
    return va ? launch_sort_phased<true, kItems>(a, stream) : launch_sort_phased<false, kItems>(a, stream);
  }
  if (small)
    return va ? launch_sort<true, 4>(a, bar_base, sms, stream) : launch_sort<false, 4>(a, bar_base, sms, stream);
  return va ? launch_sort<true, kItems>(a, bar_base, sms, stream) : launch_sort<false, kItems>(a, bar_base, sms, stream);
}

size_t compact_tmp_words(uint64_t n) { return (size_t)((n + kTile - 1) / kTile + 1); }

void compact_replica_keys(const int32_t* map_w, uint64_t K, uint32_t* out, uint32_t* count,
                          uint32_t* tmp, cudaStream_t stream) {
  compact(MapSel{map_w, K}, out, count, tmp, stream);
}

void compact_sorted_heads(const uint32_t* sk, uint64_t n, uint32_t* out, uint32_t* count, uint32_t* tmp,
                          cudaStream_t stream) {
  compact(HeadSel{sk, n}, out, count, tmp, stream);
}

}  // namespace adapm
