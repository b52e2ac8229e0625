// Internal declarations of the GB300 parameter manager (not part of the ABI).
//
// Device data layout (all in HBM, owned by the context):
//   main        [K][D] fp32     main copy of every parameter
//   val, acc    [S][D] fp32     replica pool: local value and pending updates
//   map         [W][K] int32    slot of worker w's replica of key k, or -1
//   rc          [W][K] uint32   number of w's active intents containing k
//   holders     [K]    uint32   bit w set iff worker w holds a replica of k
//   slot_owner  [S]    uint64   (w << 32) | k of a live slot, kEmptySlot if free
//   free_stack  [S]    int32    free slots, top at free_stack[free_top - 1]
//   stamp       [K]    uint32   tag of the last Intent call that listed k
//   dirty       [K]    uint8    versioned refresh only: main[k] written other
//                               than by a sync merge since the last sync of k
//   own         [K]    uint16   relocation mode only: ((owner + 1) << 8) |
//                               number of workers with active intent; owner
//                               -1 is the key's home (no worker held it yet)
//   DevState                    counters and the sticky error bits
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

struct adapm_ctx;

namespace adapm {

constexpr uint32_t kNoKey = 0xFFFFFFFFu;          // sentinel: skipped element
constexpr uint64_t kEmptySlot = ~0ull;
constexpr int kMaxWorkers = 32;
constexpr int kNumSms = 152;                      // GB300; refreshed at create

enum ErrBits : uint32_t {
  ERR_KEY_RANGE = 1u,   // a key >= K was passed
  ERR_NO_SLOTS = 2u,    // replica capacity exhausted
  ERR_REFCOUNT = 4u,    // refcount over/underflow
  ERR_TIMEOUT = 8u,     // a bounded wait on another block gave up
  ERR_INTERNAL = 16u,   // an index read from the library's own scratch or lists was out of
                        // range: the element was skipped instead of accessed
};

struct DevState {
  int32_t free_top;       // free slots on the stack
  int32_t high_water;     // slots [0, high_water) have been used
  uint32_t n_create;      // keys appended to the create list of this advance (0 between advances)
  uint32_t n_evict;       // slots appended to the evict list of this advance (0 between advances)
  int32_t adv_top;        // free_top before this advance's slots moved
  uint32_t adv_nc;        // creations of this advance (0 if the slots ran out)
  uint32_t errors;        // ErrBits, sticky until read by adapm_wait
  uint32_t last_unique;   // distinct keys of the last push
  uint32_t plan_miss;     // sequence number of the last push whose plan did not match its keys
  uint32_t adv_ne;        // evictions of this advance
  unsigned long long created;
  unsigned long long destroyed;
  int32_t live;
  uint32_t ev_done;       // blocks of the closing events launch that finished (0 between advances)
  uint32_t loss_done;     // blocks of a training step that finished (0 between steps)
  unsigned long long push_rows;       // rows pushed (cumulative)
  unsigned long long push_unique;     // distinct keys over all pushes (cumulative)
  unsigned long long sync_keys;       // keys merged by sync (cumulative)
  unsigned long long sync_replicas;   // replicas refreshed by sync (cumulative)
  unsigned long long relocations;     // owner changes (relocation mode, cumulative)
  unsigned long long sync_refreshed;  // replica values written by sync (cumulative)
  unsigned long long plan_misses;     // pushes whose plan did not match their keys (cumulative)
  // grid barriers of the sort: blocks arrived, over the context's lifetime
  // (a line of its own, away from the counters above)
  alignas(128) unsigned long long bar_arrivals;
};

// Counters of one worker's early advance events (computed ahead of the
// advance, on a stream of their own): list lengths, and the blocks of the
// evict_create launch that have finished.  Zero between advances.
struct AdvCounts {
  uint32_t nc;     // keys on the create list
  uint32_t ne;     // slots on the evict list
  uint32_t done;   // evict_create blocks finished
  uint32_t pad;
};

// Plain view of the device state passed to kernels by value.
struct Store {
  float* main;
  float* val;
  float* acc;
  int32_t* map;
  uint32_t* rc;
  uint32_t* holders;
  unsigned long long* slot_owner;
  int32_t* free_stack;
  uint32_t* stamp;
  uint16_t* own;    // null unless relocation mode
  uint8_t* dirty;   // null unless versioned refresh
  DevState* st;
  uint64_t K;
  uint64_t S;
  uint32_t D;
  uint32_t W;
};

// Fields of own[k] (relocation mode).
__device__ __forceinline__ uint32_t own_count(uint32_t o) { return o & 0xFFu; }
__device__ __forceinline__ int own_owner(uint32_t o) { return (int)(o >> 8) - 1; }
__device__ __forceinline__ uint16_t own_pack(int owner, uint32_t count) {
  return (uint16_t)(((uint32_t)(owner + 1) << 8) | count);
}

__device__ __forceinline__ void set_error(DevState* st, uint32_t bits) {
  atomicOr(&st->errors, bits);
}

// True once a sort has given up (ERR_TIMEOUT): its output is incomplete and
// the kernels that consume sorted keys return without touching the store.
__device__ __forceinline__ bool sort_failed(const DevState* st) {
  return (*reinterpret_cast<const volatile uint32_t*>(&st->errors) & ERR_TIMEOUT) != 0u;
}

// ---- radix sort / compaction (sort.cu) --------------------------------------
// Stable sort of n uint32 keys by their low `bits` bits in one cooperative
// launch on `stream`.  `raw` (n keys, not modified) is the first pass's
// input; a key >= K is sorted as kNoKey (after every valid key) and sets
// ERR_KEY_RANGE unless allow_nokey and it equals kNoKey.  ka/kb are
// ping-pong space of n keys; with va/vb non-null the positions 0..n-1
// travel with the keys.  The sorted keys (and positions) end in the buffers
// returned through *keys_out / *pos_out.  `scratch` holds
// sort_scratch_words(n) uint32 words.  *bar_base is the host's copy of
// st->bar_arrivals, advanced by the launch.  clear0 / clear1 (may be null)
// are device words the launch sets to zero before any later kernel on the
// stream runs (counters of the consumer).  If a grid-barrier wait gives
// up, the kernel sets ERR_TIMEOUT and returns; every kernel that consumes a
// sort checks that bit first and does nothing while it is set.
//
// Plans (cooperative launch only): with plan_keys and plan_word, the blocks
// first compare raw with plan_keys, the keys a plan was sorted from,
// position by position (out-of-range keys all counting as the sentinel); a
// mismatch stores plan_seq in *plan_word and counts a plan miss.  After one
// more grid barrier the launch sorts only if *plan_word == plan_seq;
// otherwise its blocks account their remaining barriers and return, leaving
// ka/kb/va/vb as they are (the plan holds the result).  Out-of-range keys
// are reported by the check as the sort would.
// phased = true runs the sort as 1 + 2 * passes ordinary launches (kernel
// boundaries instead of grid barriers, *bar_base untouched): for a stream
// that runs beside other work, where a cooperative launch would wait for
// the whole GPU.
size_t sort_scratch_words(uint64_t n);
int sort_passes(int bits);
cudaError_t sort_keys(const uint32_t* raw, uint64_t n, uint64_t K, bool allow_nokey, int bits,
                      uint32_t* ka, uint32_t* kb, uint32_t* va, uint32_t* vb, uint32_t* scratch, int sms,
                      DevState* st, unsigned long long* bar_base, uint32_t* clear0, uint32_t* clear1,
                      cudaStream_t stream, uint32_t** keys_out, uint32_t** pos_out,
                      const uint32_t* plan_keys = nullptr, uint32_t* plan_word = nullptr, uint32_t plan_seq = 0,
                      bool phased = false);

// The distinct valid keys of a sorted array, ascending, into out; count to *count.
void compact_sorted_heads(const uint32_t* sk, uint64_t n, uint32_t* out, uint32_t* count, uint32_t* tmp,
                          cudaStream_t stream);

// Stream compaction (a count / scan / write pass), tmp of compact_tmp_words(n).
size_t compact_tmp_words(uint64_t n);

// Keys k < K with map_w[k] >= 0, ascending, into out; count to *count.
void compact_replica_keys(const int32_t* map_w, uint64_t K, uint32_t* out, uint32_t* count,
                          uint32_t* tmp, cudaStream_t stream);

int bits_for(uint64_t num_keys);   // bits covering [0, K] (K itself is the sentinel range)

// Process-wide count of kernels launched by the library (capi.cu).
void note_launches(uint64_t n);

// What an entry point outside capi.cu needs of a context (capi.cu).
struct CtxView {
  Store s;
  DevState* dstate;
  cudaStream_t stream;
  int device;
  int sms;
  int bits;
  bool broken;
  unsigned long long* bar_base;   // the context's copy of dstate->bar_arrivals
};
bool ctx_view(struct ::adapm_ctx* ctx, CtxView* out);
void ctx_set_error(struct ::adapm_ctx* ctx, const char* msg);
void ctx_add_push_rows(struct ::adapm_ctx* ctx, uint64_t n);
// The checks every entry point starts with: a live context (ADAPM_EINVAL for
// null, ADAPM_ECUDA once it is unusable), its last error cleared, its device
// current.  Returns an adapm_status value (0 = ADAPM_OK).
int ctx_begin(struct ::adapm_ctx* ctx);
// A CUDA runtime error: records "where: message", marks the context unusable
// (as every entry point does) and returns ADAPM_ECUDA.
int ctx_fail_cuda(struct ::adapm_ctx* ctx, cudaError_t e, const char* where);
// cudaGetLastError() after a call's launches, or the launch failure that
// adapm_debug_fail_next_launch asked for (taken once).
cudaError_t ctx_launch_error(struct ::adapm_ctx* ctx);
// Per-operation timing (adapm_profile_enable): events recorded around an
// operation's work on the context's stream; a no-op while profiling is off.
struct ProfToken {
  int op = -1;
  cudaEvent_t a = nullptr, b = nullptr;
};
ProfToken ctx_prof_start(struct ::adapm_ctx* ctx, int op);
void ctx_prof_stop(struct ::adapm_ctx* ctx, ProfToken& t);

}  // namespace adapm
