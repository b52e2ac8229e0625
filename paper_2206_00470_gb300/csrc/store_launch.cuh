// Host-side launchers of the kernels in store.cu, push.cu and advance.cu, and of the step kernels (steps.cu).
#pragma once

#include "internal.cuh"

namespace adapm {

// Arguments of the chunked push reduction.  skeys/spos: key-sorted keys and
// their positions in `deltas` (n rows of D floats).  span_parts:
// push_span_part_rows(nchunks) x D floats of scratch for the partial sums
// of segments cut by span boundaries (a head and a tail row per span).
struct PushArgs {
  const uint32_t* skeys;
  const uint32_t* spos;
  uint64_t n;
  const float* deltas;
  uint64_t chunk;
  uint64_t nchunks;
  uint32_t worker;
  float* span_parts;
  // With plan_seq != 0, skeys / spos are a push plan and alt_keys / alt_pos
  // the sort made in its place; the kernels take the latter when
  // *plan_word == plan_seq (the plan did not match this push's keys).
  const uint32_t* alt_keys = nullptr;
  const uint32_t* alt_pos = nullptr;
  const uint32_t* plan_word = nullptr;
  uint32_t plan_seq = 0;
};

// Rows of span_parts scratch for nchunks chunks (2 per span, spans of >= 8 chunks).
uint64_t push_span_part_rows(uint64_t nchunks);

// Rows per push chunk for value length D and a batch of n rows.
uint64_t push_chunk_rows(uint32_t D, uint64_t n, int sms);

// One stored intent list (distinct keys, device count) and the sign of
// its refcount event: +1 when its window opens, -1 when it closes.
struct EventList {
  const uint32_t* keys;
  const uint32_t* count;
  uint64_t cap;
  int sign;
};

// The distinct keys of one Intent call (keys >= K set ERR_KEY_RANGE and are
// dropped), in no particular order, appended to out; *count (zeroed by the
// caller) receives their number.  `tag` must differ from every stamp left
// by earlier calls.
void launch_intent_dedup(const Store& s, const uint32_t* keys, uint64_t n, uint32_t tag, uint32_t* out,
                         uint32_t* count, int sms, cudaStream_t stream);
void launch_pull(const Store& s, int w, const uint32_t* keys, uint64_t n, float* out, int sms,
                 cudaStream_t stream);
// The same pull with rows staged in shared memory by the bulk-copy engine
// (pull_bulk.cu); usable when pull_bulk_fits(D, out): out 16-byte aligned.
bool pull_bulk_fits(uint32_t D, const void* out);
void launch_pull_bulk(const Store& s, int w, const uint32_t* keys, uint64_t n, float* out, int sms,
                      cudaStream_t stream);
void launch_push(const Store& s, const PushArgs& a, int sms, cudaStream_t stream);
// Refcount events of one advance of worker w: keys to create a replica of
// for w go to create_list, replica slots to destroy (of w, and in relocation
// mode of a worker the key is relocated to) to evict_list; the counters
// n_create / n_evict in DevState are zero between advances (the last events
// launch settles the advance's slot counts and clears them).  With cap =
// the summed caps of the lists, create_list needs cap entries and
// evict_list cap (always replicate) or 2 * cap (relocation).
// launch_evict_create applies both lists in one launch; max_events bounds
// either list's length.
// With `early` (always replicating only) the events run ahead of the
// advance: the list lengths go to *early (zero before), the map entries of
// the listed slots stay, nothing is settled; launch_evict_create with the
// same `early` then clears those map entries and settles.  Early events
// that are not followed by their advance are taken back by
// launch_events_undo (refcounts only) on the same lists.
void launch_events(const Store& s, uint32_t w, const EventList* lists, int nlists,
                   uint32_t* create_list, uint32_t* evict_list, int sms, cudaStream_t stream,
                   AdvCounts* early = nullptr);
void launch_events_undo(const Store& s, uint32_t w, const EventList* lists, int nlists, int sms,
                        cudaStream_t stream);
void launch_evict_create(const Store& s, uint32_t w, const uint32_t* create_list,
                         const uint32_t* evict_list, uint64_t max_events, int sms,
                         cudaStream_t stream, AdvCounts* early = nullptr);
void launch_sync(const Store& s, uint64_t slot_bound, int sms, cudaStream_t stream);
void launch_refcounts(const Store& s, uint32_t w, const uint32_t* keys, uint64_t n, uint32_t* out,
                      cudaStream_t stream);
void launch_owners(const Store& s, const uint32_t* keys, uint64_t n, int32_t* out, cudaStream_t stream);
void launch_replica_rows(const Store& s, uint32_t w, const uint32_t* keys, uint64_t n, float* val,
                         float* acc, uint8_t* has, cudaStream_t stream);
void launch_init_pool(int32_t* free_stack, uint64_t S, unsigned long long* owner, cudaStream_t stream);

// Fused training steps (steps.cu): read rows through the worker's slot map,
// write one delta row per row occurrence (keys to dkeys, rows to drows) and
// the per-block loss partials to loss_part; then the caller pushes.
struct StepOut {
  uint32_t* dkeys;
  float* drows;
  double* loss_part;     // grid-sized partial sums
  unsigned loss_blocks;  // number of partials written
  double* loss_out;      // the batch loss (summed by the last block), or nullptr
  uint32_t* loss_done;   // blocks finished (zero between launches)
};

void launch_mf_step(const Store& s, uint32_t w, const uint32_t* rows, const uint32_t* cols,
                    const float* vals, uint64_t n, uint32_t dim, bool adagrad, float lr, float eps,
                    const StepOut& o, int sms, cudaStream_t stream);
void launch_complex_step(const Store& s, uint32_t w, const uint32_t* heads, const uint32_t* rels,
                         const uint32_t* tails, const uint32_t* negs, uint64_t n, uint32_t n_neg,
                         uint32_t dim, float lr, float eps, const StepOut& o, int sms,
                         cudaStream_t stream);
void launch_sgns_step(const Store& s, uint32_t w, const uint32_t* centres, const uint32_t* contexts,
                      const uint32_t* negs, uint64_t n, uint32_t n_ctx, uint32_t n_neg,
                      uint32_t vocab, uint32_t dim, float lr, const StepOut& o, int sms,
                      cudaStream_t stream);
unsigned step_loss_blocks(int sms);

}  // namespace adapm
