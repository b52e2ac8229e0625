// Internal declarations of the GB300 parameter manager (not part of the ABI).
//
// Device data layout (all in HBM, owned by the context):
//   main        [K][D] fp32     main copy of every parameter
//   val, acc    [S][D] fp32     replica pool: local value and pending updates
//   map         [W][K] int32    slot of worker w's replica of key k, or -1
//   rc          [W][K] uint16   number of w's active intents containing k
//   holders     [K]    uint32   bit w set iff worker w holds a replica of k
//   slot_owner  [S]    uint64   (w << 32) | k of a live slot, kEmptySlot if free
//   free_stack  [S]    int32    free slots, top at free_stack[free_top - 1]
//   ev_delta    [K]    int32    scratch for net refcount changes, kept zero
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
};

struct DevState {
  int32_t free_top;       // free slots on the stack
  int32_t high_water;     // slots [0, high_water) have been used
  uint32_t n_create;      // keys appended to the create list of this advance
  uint32_t n_evict;       // keys appended to the evict list of this advance
  int32_t alloc_base;     // first stack index popped by this advance
  uint32_t n_create_ok;   // creates that got a slot
  uint32_t errors;        // ErrBits, sticky until read by adapm_wait
  uint32_t last_unique;   // distinct keys of the last push
  unsigned long long created;
  unsigned long long destroyed;
  int32_t live;
  int32_t pad;
  unsigned long long push_rows;       // rows pushed (cumulative)
  unsigned long long push_unique;     // distinct keys over all pushes (cumulative)
  unsigned long long sync_keys;       // keys merged by sync (cumulative)
  unsigned long long sync_replicas;   // replicas refreshed by sync (cumulative)
};

// Plain view of the device state passed to kernels by value.
struct Store {
  float* main;
  float* val;
  float* acc;
  int32_t* map;
  uint16_t* rc;
  uint32_t* holders;
  unsigned long long* slot_owner;
  int32_t* free_stack;
  int32_t* ev_delta;
  DevState* st;
  uint64_t K;
  uint64_t S;
  uint32_t D;
  uint32_t W;
};

__device__ __forceinline__ void set_error(DevState* st, uint32_t bits) {
  atomicOr(&st->errors, bits);
}

// ---- radix sort / compaction (sort.cu) --------------------------------------
// Sort n uint32 keys (with uint32 values if with_vals; iota_vals = the
// values are the positions 0..n-1) by their low `bits` bits, stable, on
// `stream`.  Buffers a/b (keys) and va/vb (values) are ping-pong space of n
// elements each; the result ends in the buffer returned through *keys_out /
// *vals_out.  `hist` is scratch of sort_hist_words(n, bits) uint32 words
// (8-byte aligned); `st` receives ERR_TIMEOUT if a look-back wait gives up.
size_t sort_hist_words(uint64_t n, int bits);
void radix_sort(uint32_t* ka, uint32_t* kb, uint32_t* va, uint32_t* vb, bool with_vals,
                bool iota_vals, uint64_t n, int bits, uint32_t* hist, DevState* st,
                cudaStream_t stream, uint32_t** keys_out, uint32_t** vals_out);

// Compact the distinct keys of a sorted array (dropping kNoKey) into out;
// the count goes to *count (device).  tmp needs compact_tmp_words(n) words.
size_t compact_tmp_words(uint64_t n);
void unique_sorted(const uint32_t* sorted, uint64_t n, uint32_t* out, uint32_t* count,
                   uint32_t* tmp, cudaStream_t stream);

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
};
bool ctx_view(struct ::adapm_ctx* ctx, CtxView* out);
void ctx_set_error(struct ::adapm_ctx* ctx, const char* msg);
void ctx_add_push_rows(struct ::adapm_ctx* ctx, uint64_t n);

}  // namespace adapm
