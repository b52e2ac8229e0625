// Intent bookkeeping on the device: the distinct keys of an Intent call, and
// the refcount events of advanceClock with the replicas they create and
// destroy (Sec. 3, Sec. 4.1).
//
//   intent        the distinct keys of one call (hash set + stamps)     (Sec. 3)
//   events        refcount +1 for every key of the opening intent lists,
//                 then -1 for the closing ones; transitions 0 -> 1
//                 (create) and 1 -> 0 (evict); the last block of the
//                 closing launch settles the advance's slot counts        (Sec. 3)
//   evict_create  main += pending updates of every evicted replica, and
//                 val = main, pending = 0 for every created one, the i-th
//                 evicted slot going to the i-th created key             (Sec. 4.1)
#include <utility>
#include <vector>

#include "internal.cuh"
#include "rowgroup.cuh"
#include "store_launch.cuh"

namespace adapm {

namespace {

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

// Single thread, after every list append of the advance: the slot counts.
// Evicted slots are handed to created keys pair by pair; only the surplus
// of either list touches the free stack (pushes above the old top, or pops
// from it).  The stack initially holds slots S-1 .. 0 (slot 0 on top) and
// positions below S - high_water are never written, so popping down to
// position p has used every slot below S - p.  Creations that need more
// free slots than there are fail all together (ERR_NO_SLOTS).
__device__ __forceinline__ uint32_t creations_ok(uint32_t ne, uint32_t nc, int32_t top) {
  return (nc > ne && (int64_t)(nc - ne) > (int64_t)top) ? 0u : nc;
}

// The free stack and the store's counters after an advance of ne evictions
// and nc listed creations from stack top `top`; returns the creations made.
__device__ uint32_t settle_counts(DevState* st, int32_t S, uint32_t ne, uint32_t nc, int32_t top) {
  const uint32_t nc_ok = creations_ok(ne, nc, top);
  if (nc_ok != nc) atomicOr(&st->errors, (uint32_t)ERR_NO_SLOTS);
  const int32_t ntop = top + (int32_t)ne - (int32_t)nc_ok;
  st->free_top = ntop;
  st->live += (int32_t)nc_ok - (int32_t)ne;
  st->destroyed += ne;
  st->created += nc_ok;
  const int32_t lowest = ntop < top ? ntop : top;
  if (S - lowest > st->high_water) st->high_water = S - lowest;
  return nc_ok;
}

__device__ void settle_advance(DevState* st, int32_t S) {
  const uint32_t ne = st->n_evict, nc = st->n_create;
  const int32_t top = st->free_top;
  st->adv_ne = ne;
  st->adv_nc = settle_counts(st, S, ne, nc, top);
  st->adv_top = top;
  st->n_create = 0;   // ready for the next advance
  st->n_evict = 0;
  st->ev_done = 0;
}

// Refcount transitions of one advance of worker w.  All lists whose window
// opens are applied first (START, rc += 1), then all lists whose window
// closes (rc -= 1).  Every key of a closing list had a positive count before
// the advance (its intent was active), so with the openings first a key in
// both kinds of list never crosses 0, and one atomic per listed key gives
// exactly the transitions of the net change: 0 -> 1 (w's intent for k became
// active, a "join") and 1 -> 0 (a "leave").  Only the thread that sees a
// key's transition handles it, so the per-key state below has one writer.
//
// Always replicate: a join lists k for creation; a leave lists w's replica
// slot (if it got one) for eviction.
// Relocation (Sec. 4.1, App. B.2.4): own[k] counts the workers with active
// intent and names the owner, which holds no replica.  A join with no other
// worker active makes w the owner; otherwise w gets a replica unless it
// owns k already.  A leave destroys w's replica (if any); when exactly one
// worker stays active and it holds a replica (so it is not the owner), that
// replica is destroyed too and the worker becomes the owner.  The holders
// other than w come from holders[k], which only w's own advance changes.
//
// The create list takes keys (of worker w), the evict list slots (of any
// worker).  Four keys per thread and round; one list append per block and
// round.  The order of a list is not specified.
//
// Early events (AdvCounts given): the lists are computed ahead of the
// advance, beside the worker's push, with their own counters; the map
// entries stay until evict_create clears them, and evict_create settles.
template <bool START>
__global__ void events_kernel(Store s, uint32_t w, EventBatch eb, uint32_t* out_list, int settle,
                              AdvCounts* early) {
  if (sort_failed(s.st)) return;
  constexpr int Q = 4;
  __shared__ uint32_t base_s;
  uint32_t* rcw = s.rc + (uint64_t)w * s.K;
  int32_t* mapw_mut = s.map + (uint64_t)w * s.K;
  const int32_t* mapw = mapw_mut;
  uint32_t* counter = early ? (START ? &early->nc : &early->ne) : (START ? &s.st->n_create : &s.st->n_evict);
  const bool reloc = s.own != nullptr;
  uint32_t pre[kEventLists + 1];
  const uint32_t n = batch_prefix(eb, pre);
  const uint32_t stride = gridDim.x * blockDim.x * Q;
  for (uint32_t b = blockIdx.x * blockDim.x * Q; b < n; b += stride) {   // block-uniform trip count
    uint32_t k[Q], old[Q], e0[Q], e1[Q];
    bool hit[Q], hit1[Q];
    bool in[Q];   // a listed key in range (list entries are keys < K; anything else is skipped)
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      const uint32_t i = b + q * blockDim.x + threadIdx.x;
      k[q] = i < n ? batch_key(eb, pre, i) : 0u;
      in[q] = i < n && k[q] < s.K;
      if (i < n && !in[q]) set_error(s.st, ERR_INTERNAL);
    }
    // closing lists: the slot-map entry of every listed key is read with its
    // atomic, not after it (only this thread touches it in this launch), so
    // a transition costs one memory latency instead of two
    int32_t msl[Q];
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      old[q] = 1u;   // neither transition
      msl[q] = -1;
      if (!START && in[q]) msl[q] = mapw[k[q]];
      if (in[q]) old[q] = START ? atomicAdd(rcw + k[q], 1u) : atomicSub(rcw + k[q], 1u);
    }
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      hit1[q] = false;
      if (START) {
        hit[q] = in[q] && old[q] == 0u;
        if (in[q] && old[q] >= 65535u) set_error(s.st, ERR_REFCOUNT);
      } else {
        hit[q] = in[q] && old[q] == 1u;
        if (in[q] && old[q] == 0u) {   // more closings than openings: undo, report
          atomicAdd(rcw + k[q], 1u);
          set_error(s.st, ERR_REFCOUNT);
        }
      }
    }
    uint32_t moved = 0;   // owner changes in this round
    if (START) {
      // keys with a transition are distinct, so all their loads go first
      uint32_t o[Q] = {};
#pragma unroll
      for (int q = 0; q < Q; ++q)
        if (reloc && hit[q]) o[q] = s.own[k[q]];
#pragma unroll
      for (int q = 0; q < Q; ++q) {
        e0[q] = k[q];
        if (reloc && hit[q]) {
          const uint32_t m = own_count(o[q]);
          const int owner = own_owner(o[q]);
          if (m == 0u) {   // the only worker with active intent: relocate to w
            s.own[k[q]] = own_pack((int)w, 1u);
            moved += owner != (int)w ? 1u : 0u;
            hit[q] = false;
          } else {
            s.own[k[q]] = own_pack(owner, m + 1u);
            hit[q] = owner != (int)w;
          }
        }
      }
    } else {
      int32_t sl[Q];
      uint32_t o[Q] = {}, hm[Q] = {};
#pragma unroll
      for (int q = 0; q < Q; ++q) {
        sl[q] = hit[q] ? msl[q] : -1;
        if (reloc && hit[q]) {
          o[q] = s.own[k[q]];
          hm[q] = s.holders[k[q]];
        }
      }
#pragma unroll
      for (int q = 0; q < Q; ++q) {
        if (reloc && hit[q]) {
          const uint32_t m = own_count(o[q]) - 1u;
          int owner = own_owner(o[q]);
          const uint32_t rem = hm[q] & ~(1u << w);
          if (m == 1u && rem != 0u) {   // one worker left, holding a replica: relocate to it
            const uint32_t a = (uint32_t)(__ffs(rem) - 1);
            e1[q] = (uint32_t)s.map[(uint64_t)a * s.K + k[q]];
            hit1[q] = true;
            owner = (int)a;
            moved += 1u;
          }
          s.own[k[q]] = own_pack(owner, m);
        }
        // a key whose replica was never created (capacity exhausted) has nothing to destroy
        hit[q] = sl[q] >= 0;
        e0[q] = (uint32_t)sl[q];
        // always replicating, the slot map entry is cleared here, where its line was just read
        // (nothing reads the map between this kernel and the eviction of the listed slot); with
        // relocation the eviction clears it, off this kernel's longer chain of dependent accesses
        if (hit[q] && !reloc && !early) mapw_mut[k[q]] = -1;
      }
    }
    uint32_t c = 0, total, mtotal;
#pragma unroll
    for (int q = 0; q < Q; ++q) c += (hit[q] ? 1u : 0u) + (hit1[q] ? 1u : 0u);
    block_exclusive_scan2(c, moved, total, mtotal);
    if (threadIdx.x == 0) {
      base_s = total ? atomicAdd(counter, total) : 0u;
      if (mtotal) atomicAdd(&s.st->relocations, (unsigned long long)mtotal);
    }
    __syncthreads();
    c += base_s;
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      if (hit[q]) out_list[c++] = e0[q];
      if (hit1[q]) out_list[c++] = e1[q];
    }
    __syncthreads();
  }
  if (!START && settle) {
    // the last block to finish settles the advance's slot counts
    __shared__ int last;
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      last = atomicAdd(&s.st->ev_done, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (last && threadIdx.x == 0) {
      __threadfence();
      settle_advance(s.st, (int32_t)s.S);
    }
  }
}

// evict_create: entry i of the advance evicts the i-th listed slot (any
// worker's: a relocation destroys another worker's replica) -- main[k] +=
// its pending row, by vector atomic adds since main[k] may receive two
// pending rows in one advance (the leaving worker's and a relocated
// holder's) -- and creates the i-th listed key of worker w, val = main,
// pending = 0, in that same slot when there is one (the thread reads the
// pending row before it overwrites it), else in a slot popped from the
// stack; an evicted slot with no creation to take it is pushed.  A created
// key is never one whose replica this advance destroys (a worker joins or
// leaves a key, not both), so its main row is final.  R entries per row
// group at a time; a round's loads (owner records, pending rows, main rows)
// go out together with the next round's list entries.
//
// After early events (AdvCounts given) every block takes the list lengths
// from the counters and the stack top from the store (the same values in
// every block: the store changes only after all blocks have finished),
// evicted slots also clear their map entries, and the last block to finish
// settles the advance.
template <int G, int C>
__global__ void __launch_bounds__(kThreads, C >= 8 ? 2 : 3) evict_create_kernel(Store s, uint32_t w,
                                                                              const uint32_t* __restrict__ evict_list,
                                                                              const uint32_t* __restrict__ create_list,
                                                                              AdvCounts* early) {
  constexpr int R = 4 / C > 0 ? 4 / C : 1;
  const int lane = threadIdx.x & (G - 1);
  const uint32_t D4 = s.D >> 2;
  uint32_t ne, nc;
  int32_t top;
  if (early) {
    ne = early->ne;
    top = s.st->free_top;
    nc = creations_ok(ne, early->nc, top);
  } else {
    ne = s.st->adv_ne;
    nc = s.st->adv_nc;
    top = s.st->adv_top;
  }
  const uint64_t n = ne > nc ? ne : nc;
  float4* main4 = reinterpret_cast<float4*>(s.main);
  float4* val4 = reinterpret_cast<float4*>(s.val);
  float4* acc4 = reinterpret_cast<float4*>(s.acc);
  int32_t* mapw = s.map + (uint64_t)w * s.K;
  const uint64_t g = group_id<G>(), ng = group_count<G>();
  const uint64_t step = ng * R;
  // list entries out of range (slots >= S, keys >= K) are skipped and reported
  auto load_entries = [&](uint64_t i0, int32_t (&es)[R], uint32_t (&ck)[R]) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const uint64_t i = i0 + r;
      const uint32_t e = i < ne ? evict_list[i] : 0xFFFFFFFFu;
      es[r] = e < s.S ? (int32_t)e : -1;
      ck[r] = i < nc ? create_list[i] : kNoKey;
      if ((i < ne && e >= s.S) || (i < nc && ck[r] >= s.K)) {
        set_error(s.st, ERR_INTERNAL);
        if (ck[r] >= s.K) ck[r] = kNoKey;
      }
    }
  };
  int32_t es[R];
  uint32_t ck[R];
  load_entries(g * R, es, ck);
  for (uint64_t i0 = g * R; i0 < n; i0 += step) {
    int32_t cs[R];
    unsigned long long ow[R];
    float4 ac[R][C], mv[R][C];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const uint64_t i = i0 + r;
      // slot of the creation: the paired evicted slot, else popped (top first)
      cs[r] = ck[r] == kNoKey ? -1 : (es[r] >= 0 ? es[r] : s.free_stack[top - 1 - (int32_t)(i - ne)]);
      ow[r] = es[r] >= 0 ? s.slot_owner[es[r]] : 0ull;
      const bool bad_slot = ck[r] != kNoKey && (cs[r] < 0 || (uint64_t)cs[r] >= s.S);
      const bool bad_owner = es[r] >= 0 && ((uint32_t)ow[r] >= s.K || (ow[r] >> 32) >= s.W);
      if (bad_slot || bad_owner) {
        set_error(s.st, ERR_INTERNAL);   // a free-stack entry or owner record out of range: skipped
        if (bad_slot) {
          cs[r] = -1;
          ck[r] = kNoKey;
        }
        if (bad_owner) es[r] = -1;
      }
#pragma unroll
      for (int c = 0; c < C; ++c) {
        const uint32_t col = lane + c * G;
        ac[r][c] = (es[r] >= 0 && col < D4) ? acc4[(uint64_t)es[r] * D4 + col] : f4zero();
        mv[r][c] = (ck[r] != kNoKey && col < D4) ? main4[(uint64_t)ck[r] * D4 + col] : f4zero();
      }
    }
    int32_t es1[R];
    uint32_t ck1[R];
    load_entries(i0 + step, es1, ck1);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const uint64_t i = i0 + r;
      if (es[r] >= 0) {
        const uint32_t k = (uint32_t)ow[r], a = (uint32_t)(ow[r] >> 32);
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          if (col < D4) atomicAdd(main4 + (uint64_t)k * D4 + col, ac[r][c]);
        }
        if (lane == 0) {
          if (s.dirty != nullptr) s.dirty[k] = 1;   // versioned refresh: main changed
          // (always replicating, the events kernel that listed the slot has
          // cleared its map entry, unless it ran early)
          if (s.own != nullptr || early) s.map[(uint64_t)a * s.K + k] = -1;
          atomicAnd(s.holders + k, ~(1u << a));
          if (ck[r] == kNoKey) {
            s.slot_owner[es[r]] = kEmptySlot;
            s.free_stack[top + (int32_t)(i - nc)] = es[r];
          }
        }
      }
      if (ck[r] != kNoKey) {
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const uint32_t col = lane + c * G;
          if (col < D4) {
            val4[(uint64_t)cs[r] * D4 + col] = mv[r][c];
            acc4[(uint64_t)cs[r] * D4 + col] = f4zero();
          }
        }
        if (lane == 0) {
          // versioned refresh: the new replica has seen every update (a stale
          // replica of another worker is refreshed anyway: the key has two holders)
          if (s.dirty != nullptr) s.dirty[ck[r]] = 0;
          mapw[ck[r]] = cs[r];
          atomicOr(s.holders + ck[r], 1u << w);
          s.slot_owner[cs[r]] = ((unsigned long long)w << 32) | ck[r];
        }
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      es[r] = es1[r];
      ck[r] = ck1[r];
    }
  }
  if (early) {
    // the last block to finish settles the advance (all blocks have read
    // the stack top by then) and clears the counters for the next one
    __shared__ int last;
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      last = atomicAdd(&early->done, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (last && threadIdx.x == 0) {
      __threadfence();
      // (the counters and the stack top are unchanged since every block read them)
      settle_counts(s.st, (int32_t)s.S, early->ne, early->nc, s.st->free_top);
      early->nc = 0;
      early->ne = 0;
      early->done = 0;
    }
  }
}

// Undo early events whose advance did not happen as computed (a list was
// added or applied after them): refcount -= 1 for every key of the opening
// lists and += 1 for the closing ones, with no transitions (nothing else
// touched the worker's counts or lists since).
__global__ void events_undo_kernel(Store s, uint32_t w, EventBatch eb, int sign) {
  uint32_t* rcw = s.rc + (uint64_t)w * s.K;
  uint32_t pre[kEventLists + 1];
  const uint32_t n = batch_prefix(eb, pre);
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const uint32_t k = batch_key(eb, pre, i);
    if (k < s.K) atomicAdd(rcw + k, sign > 0 ? 0xFFFFFFFFu : 1u);
  }
}

}  // namespace

void launch_intent_dedup(const Store& s, const uint32_t* keys, uint64_t n, uint32_t tag, uint32_t* out,
                         uint32_t* count, int sms, cudaStream_t stream) {
  if (n == 0) return;
  uint64_t b = (n + kDedupTile - 1) / kDedupTile;
  if (b > (uint64_t)sms * 8) b = (uint64_t)sms * 8;
  note_launches(1);
  intent_dedup_kernel<<<(unsigned)b, kThreads, 0, stream>>>(s, keys, n, tag, out, count);
}

namespace {

// The opening (pass 0) and closing (pass 1) lists in batches of kEventLists,
// each with its summed capacity; with `end` an empty closing batch stands in
// when no list closes.
void event_batches(const EventList* lists, int nlists, bool end,
                   std::vector<std::pair<EventBatch, uint64_t>> (&batches)[2]) {
  for (int pass = 0; pass < 2; ++pass) {
    const int sign = pass == 0 ? +1 : -1;
    EventBatch eb{};
    uint64_t cap = 0;
    for (int i = 0; i < nlists; ++i) {
      if (lists[i].sign != sign) continue;
      eb.keys[eb.n] = lists[i].keys;
      eb.count[eb.n] = lists[i].count;
      eb.n += 1;
      cap += lists[i].cap;   // the kernel covers the batch's lists as one index space
      if (eb.n == kEventLists) {
        batches[pass].emplace_back(eb, cap);
        eb = EventBatch{};
        cap = 0;
      }
    }
    if (eb.n > 0 || (end && pass == 1 && batches[1].empty())) batches[pass].emplace_back(eb, cap);
  }
}

}  // namespace

void launch_events(const Store& s, uint32_t w, const EventList* lists, int nlists,
                   uint32_t* create_list, uint32_t* evict_list, int sms, cudaStream_t stream,
                   AdvCounts* early) {
  // all opening lists first, then all closing lists; without `early` the
  // last closing launch (an empty one if no list closes) settles the slot counts
  const uint64_t cap_blocks = (uint64_t)sms * 8;
  std::vector<std::pair<EventBatch, uint64_t>> batches[2];
  event_batches(lists, nlists, early == nullptr, batches);
  for (int pass = 0; pass < 2; ++pass) {
    for (size_t i = 0; i < batches[pass].size(); ++i) {
      const EventBatch& eb = batches[pass][i].first;
      uint64_t b = (batches[pass][i].second + 4 * kThreads - 1) / (4 * kThreads);   // 4 keys per thread
      if (b > cap_blocks) b = cap_blocks;
      if (b == 0) b = 1;
      note_launches(1);
      if (pass == 0)
        events_kernel<true><<<(unsigned)b, kThreads, 0, stream>>>(s, w, eb, create_list, 0, early);
      else
        events_kernel<false><<<(unsigned)b, kThreads, 0, stream>>>(
            s, w, eb, evict_list, (!early && i + 1 == batches[1].size()) ? 1 : 0, early);
    }
  }
}

void launch_events_undo(const Store& s, uint32_t w, const EventList* lists, int nlists, int sms,
                        cudaStream_t stream) {
  std::vector<std::pair<EventBatch, uint64_t>> batches[2];
  event_batches(lists, nlists, false, batches);
  for (int pass = 0; pass < 2; ++pass) {
    for (const auto& bc : batches[pass]) {
      uint64_t b = (bc.second + kThreads - 1) / kThreads;
      if (b > (uint64_t)sms * 8) b = (uint64_t)sms * 8;
      if (b == 0) b = 1;
      note_launches(1);
      events_undo_kernel<<<(unsigned)b, kThreads, 0, stream>>>(s, w, bc.first, pass == 0 ? +1 : -1);
    }
  }
}

void launch_evict_create(const Store& s, uint32_t w, const uint32_t* create_list,
                         const uint32_t* evict_list, uint64_t max_events, int sms,
                         cudaStream_t stream, AdvCounts* early) {
  dispatch_gc(s.D / 4, [&](auto Gc, auto Cc) {
    constexpr int G = decltype(Gc)::value, C = decltype(Cc)::value;
    constexpr uint64_t R = 4 / C > 0 ? 4 / C : 1;   // list entries per group, as in the kernel
    const unsigned grid = grid_for((max_events + R - 1) / R, G, sms);
    note_launches(1);
    evict_create_kernel<G, C><<<grid, kThreads, 0, stream>>>(s, w, evict_list, create_list, early);
  });
}

}  // namespace adapm
