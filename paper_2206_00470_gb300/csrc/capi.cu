// extern "C" entry points of libadapm (include/adapm.h) and the host-side
// state of a context: worker clocks and the per-clock buckets of stored
// intent lists (Sec. 3: an intent is inactive before C_start, active in
// [C_start, C_end), expired after).  All device work is enqueued on one
// stream; scratch comes from a context-owned stream-ordered memory pool.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <deque>
#include <map>
#include <new>
#include <string>
#include <tuple>
#include <vector>

#include "adapm.h"
#include "internal.cuh"
#include "store_launch.cuh"

using namespace adapm;

namespace {
std::atomic<unsigned long long> g_launches{0};
}  // namespace

void adapm::note_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

namespace {

struct IntentList {
  uint32_t* keys = nullptr;   // device: cap distinct keys (no particular order), then the count word
  uint32_t* count = nullptr;
  uint64_t cap = 0;
  // Push plan: the stable sort of the call's n keys with their positions
  // (psk, psp), made on the plan stream; `ready` is recorded there after it
  // (and after the distinct keys, when they come from the plan: from_plan).
  uint32_t* psk = nullptr;
  uint32_t* psp = nullptr;
  uint32_t* px = nullptr;     // the call's keys as given (what a matching push's keys equal)
  uint64_t n = 0;
  bool from_plan = false;
  bool plan_used = false;      // a push took this plan
  cudaEvent_t ready = nullptr;
  void* in_owned = nullptr;   // the call's staged copy of host keys, read by the plan stream
  int64_t start = 0, end = 0; // the window as signalled
};

struct WorkerState {
  int64_t clock = 0;
  double est = 0.0;          // Algorithm 1: clocks per round, smoothed
  int64_t round_clock = 0;   // clock at the previous round
  std::map<int64_t, std::vector<int64_t>> starts;   // clock -> lists whose window opens
  std::map<int64_t, std::vector<int64_t>> ends;     // clock -> lists whose window closes
  std::vector<int64_t> order;                       // recorded lists, oldest first
  // Lists closed in a row whose plan no push took, and intents recorded: a
  // worker whose pushes never match its intents (the SGNS step) stops
  // getting plans, except every kPlanProbe-th intent.
  int unused_plans = 0;
  uint64_t intents = 0;
  // Early events of the next advance (made at the worker's first push after
  // its last advance): the lists they cover, the create and evict lists
  // they fill, and the event after them on the early stream.
  struct Early {
    bool active = false;
    int64_t clock = 0;                 // the clock the advance reaches
    std::vector<int64_t> open, close;  // list ids, in advance order
    uint32_t* create_list = nullptr;
    uint32_t* evict_list = nullptr;
    uint64_t cap = 0;
    cudaEvent_t done = nullptr;
  } early;
};

}  // namespace

struct adapm_ctx {
  adapm_config cfg{};
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  int device = 0;
  int sms = kNumSms;
  int bits = 32;
  cudaMemPool_t pool = nullptr;
  Store s{};
  DevState* dstate = nullptr;
  std::vector<WorkerState> workers;
  std::map<int64_t, IntentList> lists;
  int64_t next_list = 0;
  std::string err;
  bool broken = false;
  unsigned long long bar_base = 0;   // dstate->bar_arrivals once the queued sorts have run
  uint32_t intent_tag = 0;           // tag of the last Intent call (stamp array)
  uint64_t push_rows_host = 0;
  bool prof = false;
  std::vector<std::tuple<int, cudaEvent_t, cudaEvent_t>> pending;
  std::vector<cudaEvent_t> spare_events;
  double prof_ms[ADAPM_NUM_OPS] = {0};
  uint64_t prof_calls[ADAPM_NUM_OPS] = {0};
  // Pinned host inputs are copied on a stream of their own from a pool of
  // their own, so that a call's copies overlap the kernels of the calls
  // enqueued before it.  `stream` waits for each copy (event `staged`).  A
  // mark (an event on `stream` with the bytes staged before it) is taken at
  // each staging call; while more than kStageAhead bytes are staged beyond
  // the oldest mark, copy_in waits for that mark, which bounds the staging
  // memory in flight.
  cudaStream_t copy_in = nullptr;
  cudaMemPool_t stage_pool = nullptr;
  cudaEvent_t staged = nullptr;
  std::deque<std::pair<cudaEvent_t, uint64_t>> stage_marks;
  std::vector<cudaEvent_t> spare_marks;
  uint64_t stage_unmarked = 0;   // bytes staged since the last mark
  uint64_t stage_live = 0;       // bytes staged since the oldest mark
  // Push plans are sorted on plan_stream (lowest priority, so its blocks
  // take what the library stream leaves), with scratch from plan_pool, which
  // never makes one stream wait for the other on its own.
  cudaStream_t plan_stream = nullptr;
  cudaMemPool_t plan_pool = nullptr;
  std::vector<cudaEvent_t> spare_ready;
  uint32_t plan_seq = 0;
  uint64_t planned_pushes = 0;
  // Early advance events run on early_stream, beside the library stream's
  // push, with per-worker counters early_counts[w] (device, zero between
  // advances).
  cudaStream_t early_stream = nullptr;
  AdvCounts* early_counts = nullptr;
  uint64_t early_advances = 0;   // advances that used their early events
  uint64_t early_undone = 0;     // early events taken back
  bool fake_launch_error = false;   // adapm_debug_fail_next_launch
};

namespace {

adapm_status fail(adapm_ctx* c, adapm_status st, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return st;
}

adapm_status cuda_fail(adapm_ctx* c, cudaError_t e, const char* where) {
  if (c) c->broken = true;
  return fail(c, ADAPM_ECUDA, "%s: %s", where, cudaGetErrorString(e));
}

#define CK(call)                                             \
  do {                                                       \
    cudaError_t e_ = (call);                                 \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, #call); \
  } while (0)

enum class MemKind { Device, PinnedHost, PageableHost };

MemKind mem_kind(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return MemKind::PageableHost;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return MemKind::Device;
  return a.type == cudaMemoryTypeHost ? MemKind::PinnedHost : MemKind::PageableHost;
}

bool is_device_ptr(const void* p) { return mem_kind(p) == MemKind::Device; }

constexpr uint64_t kStageAhead = 8ull << 30;   // staged input bytes ahead of the kernels, at most

// The staging stream and pool, made on the first pinned host input: their own
// stream, and a pool that reuses a block only once its free is known to be
// done, never by making copy_in wait for `stream` on its own.
cudaError_t ensure_copy_in(adapm_ctx* ctx) {
  if (ctx->copy_in) return cudaSuccess;
  cudaMemPoolProps props{};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = ctx->device;
  cudaMemPool_t pool = nullptr;
  cudaEvent_t ev = nullptr;
  cudaStream_t st = nullptr;
  uint64_t keep = ~0ull;
  int no = 0;
  cudaError_t e = cudaMemPoolCreate(&pool, &props);
  if (e == cudaSuccess) e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
  if (e == cudaSuccess) e = cudaMemPoolSetAttribute(pool, cudaMemPoolReuseAllowInternalDependencies, &no);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
  if (e != cudaSuccess) {   // nothing half-made is kept
    if (st) cudaStreamDestroy(st);
    if (ev) cudaEventDestroy(ev);
    if (pool) cudaMemPoolDestroy(pool);
    return e;
  }
  ctx->stage_pool = pool;
  ctx->staged = ev;
  ctx->copy_in = st;
  return cudaSuccess;
}

// The plan stream and its pool, made on the first intent that gets a plan.
cudaError_t ensure_plan_stream(adapm_ctx* ctx) {
  if (ctx->plan_stream) return cudaSuccess;
  cudaMemPoolProps props{};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = ctx->device;
  cudaMemPool_t pool = nullptr;
  cudaStream_t st = nullptr;
  uint64_t keep = ~0ull;
  int no = 0, least = 0, greatest = 0;
  cudaError_t e = cudaDeviceGetStreamPriorityRange(&least, &greatest);
  if (e == cudaSuccess) e = cudaMemPoolCreate(&pool, &props);
  if (e == cudaSuccess) e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
  if (e == cudaSuccess) e = cudaMemPoolSetAttribute(pool, cudaMemPoolReuseAllowInternalDependencies, &no);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&st, cudaStreamNonBlocking, least);
  if (e != cudaSuccess) {
    if (st) cudaStreamDestroy(st);
    if (pool) cudaMemPoolDestroy(pool);
    return e;
  }
  ctx->plan_pool = pool;
  ctx->plan_stream = st;
  return cudaSuccess;
}

cudaError_t take_ready_event(adapm_ctx* ctx, cudaEvent_t* ev) {
  if (!ctx->spare_ready.empty()) {
    *ev = ctx->spare_ready.back();
    ctx->spare_ready.pop_back();
    return cudaSuccess;
  }
  return cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
}

// Take a mark on `stream` for the bytes staged since the last one, then let
// copy_in wait for the oldest marks while too much is staged beyond them.
cudaError_t stage_mark(adapm_ctx* ctx, uint64_t next_bytes) {
  cudaError_t e = cudaSuccess;
  // marks already passed release their bytes without a wait
  while (!ctx->stage_marks.empty()) {
    const cudaError_t q = cudaEventQuery(ctx->stage_marks.front().first);
    if (q == cudaErrorNotReady) {
      if (cudaPeekAtLastError() == cudaErrorNotReady) cudaGetLastError();
      break;
    }
    if (q != cudaSuccess) return q;
    ctx->spare_marks.push_back(ctx->stage_marks.front().first);
    ctx->stage_live -= ctx->stage_marks.front().second;
    ctx->stage_marks.pop_front();
  }
  if (ctx->stage_unmarked) {
    cudaEvent_t ev = nullptr;
    if (!ctx->spare_marks.empty()) {
      ev = ctx->spare_marks.back();
      ctx->spare_marks.pop_back();
    } else if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming)) != cudaSuccess) {
      return e;
    }
    if ((e = cudaEventRecord(ev, ctx->stream)) != cudaSuccess) return e;
    ctx->stage_marks.emplace_back(ev, ctx->stage_unmarked);
    ctx->stage_unmarked = 0;
  }
  while (!ctx->stage_marks.empty() && ctx->stage_live + next_bytes > kStageAhead) {
    auto m = ctx->stage_marks.front();
    ctx->stage_marks.pop_front();
    if ((e = cudaStreamWaitEvent(ctx->copy_in, m.first, 0)) != cudaSuccess) return e;
    ctx->spare_marks.push_back(m.first);   // the wait has captured it; it can be recorded again
    ctx->stage_live -= m.second;
  }
  return cudaSuccess;
}

template <class T>
cudaError_t pool_alloc(adapm_ctx* ctx, T** p, size_t count) {
  if (count == 0) count = 1;
  return cudaMallocFromPoolAsync(reinterpret_cast<void**>(p), count * sizeof(T), ctx->pool,
                                 ctx->stream);
}

void pool_free(adapm_ctx* ctx, void* p) {
  if (p) cudaFreeAsync(p, ctx->stream);
}

// Device view of an input array; copies host arrays in.
template <class T>
struct Input {
  const T* dev = nullptr;
  T* owned = nullptr;
};

template <class T>
cudaError_t stage_in(adapm_ctx* ctx, const T* p, size_t count, Input<T>* in) {
  if (count == 0 || p == nullptr) {
    in->dev = p;
    return cudaSuccess;
  }
  const MemKind kind = mem_kind(p);
  if (kind == MemKind::Device) {
    in->dev = p;
    return cudaSuccess;
  }
  const uint64_t bytes = count * sizeof(T);
  if (kind == MemKind::PinnedHost) {
    cudaError_t e = ensure_copy_in(ctx);
    if (e == cudaSuccess) e = stage_mark(ctx, bytes);
    if (e != cudaSuccess) return e;
    e = cudaMallocFromPoolAsync(reinterpret_cast<void**>(&in->owned), bytes, ctx->stage_pool, ctx->copy_in);
    if (e != cudaSuccess) return e;
    in->dev = in->owned;
    e = cudaMemcpyAsync(in->owned, p, bytes, cudaMemcpyHostToDevice, ctx->copy_in);
    if (e == cudaSuccess) e = cudaEventRecord(ctx->staged, ctx->copy_in);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->stream, ctx->staged, 0);
    ctx->stage_unmarked += bytes;
    ctx->stage_live += bytes;
    return e;   // the buffer is freed on `stream` after its consumer, like any pool buffer
  }
  cudaError_t e = pool_alloc(ctx, &in->owned, count);
  if (e != cudaSuccess) return e;
  in->dev = in->owned;
  return cudaMemcpyAsync(in->owned, p, bytes, cudaMemcpyHostToDevice, ctx->stream);
}

// Device buffer for an output array; copied out to host arrays at finish.
template <class T>
struct Output {
  T* dev = nullptr;
  T* host = nullptr;
  size_t count = 0;
};

template <class T>
cudaError_t stage_out(adapm_ctx* ctx, T* p, size_t count, Output<T>* o) {
  o->count = count;
  if (count == 0 || is_device_ptr(p)) {
    o->dev = p;
    return cudaSuccess;
  }
  o->host = p;
  return pool_alloc(ctx, &o->dev, count);
}

template <class T>
cudaError_t finish_out(adapm_ctx* ctx, Output<T>* o) {
  if (!o->host) return cudaSuccess;
  cudaError_t e = cudaMemcpyAsync(o->host, o->dev, o->count * sizeof(T), cudaMemcpyDeviceToHost,
                                  ctx->stream);
  pool_free(ctx, o->dev);
  return e;
}

cudaEvent_t take_prof_event(adapm_ctx* ctx) {
  if (!ctx->spare_events.empty()) {
    cudaEvent_t e = ctx->spare_events.back();
    ctx->spare_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

struct ProfScope {
  adapm_ctx* ctx;
  ProfToken t;
  ProfScope(adapm_ctx* c, int o) : ctx(c) { t = ctx_prof_start(ctx, o); }
  ~ProfScope() { ctx_prof_stop(ctx, t); }
};

adapm_status check_launch(adapm_ctx* ctx, const char* where) {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && ctx->fake_launch_error) e = cudaErrorLaunchFailure;   // adapm_debug_fail_next_launch
  ctx->fake_launch_error = false;
  if (e != cudaSuccess) return cuda_fail(ctx, e, where);
  return ADAPM_OK;
}

adapm_status check_ctx(adapm_ctx* ctx) {
  if (!ctx) return ADAPM_EINVAL;
  if (ctx->broken) return fail(ctx, ADAPM_ECUDA, "context unusable after an earlier CUDA error");
  ctx->err.clear();
  if (cudaSetDevice(ctx->device) != cudaSuccess) return fail(ctx, ADAPM_ECUDA, "cudaSetDevice");
  return ADAPM_OK;
}

constexpr uint64_t kMaxN = 1ull << 31;
constexpr int kPlanPatience = 4;       // unused plans in a row after which a worker gets none ...
constexpr uint64_t kPlanProbe = 16;    // ... but for one intent in this many

// Refcount events of one worker -> destroy, then create replicas.
// ---------------------------------------------------------------------------
// Early advance events.  The refcount events of a worker's next advance
// read and write only that worker's refcounts and read its slot map, which
// nothing but its own advances changes (always replicating), so they can run
// before the advance, beside the worker's pull and push: at the worker's
// first pull, push or step after an advance, the lists whose window opens
// or closes at its next clock are applied on early_stream, into lists and
// counters of the worker's own.  The advance then waits for them and runs
// evict_create alone, which clears the evicted map entries and settles.  If
// the advance's lists are not the ones used (an intent recorded or applied
// in between), the early events are undone and the advance runs in full.
// Not with relocation (its events read other workers' state) or adaptive
// timing (its openings happen at syncs).
// ---------------------------------------------------------------------------
bool early_enabled(const adapm_ctx* ctx) {
  return !ctx->cfg.no_early_events && ctx->s.own == nullptr && ctx->cfg.action_timing != ADAPM_ACT_ADAPTIVE;
}

// The lists of worker w's advance to clock c: opening ones, closing ones.
void advance_lists(const WorkerState& ws, int64_t c, std::vector<int64_t>& open, std::vector<int64_t>& close) {
  open.clear();
  close.clear();
  auto it = ws.starts.find(c);
  if (it != ws.starts.end()) open = it->second;
  it = ws.ends.find(c);
  if (it != ws.ends.end()) close = it->second;
}

std::vector<EventList> event_lists(adapm_ctx* ctx, const std::vector<int64_t>& open,
                                   const std::vector<int64_t>& close) {
  std::vector<EventList> ev;
  for (int64_t id : open) {
    const IntentList& L = ctx->lists[id];
    ev.push_back(EventList{L.keys, L.count, L.cap, +1});
  }
  for (int64_t id : close) {
    const IntentList& L = ctx->lists[id];
    ev.push_back(EventList{L.keys, L.count, L.cap, -1});
  }
  return ev;
}

adapm_status early_make(adapm_ctx* ctx, uint32_t w) {
  WorkerState& ws = ctx->workers[w];
  if (!early_enabled(ctx) || ws.early.active) return ADAPM_OK;
  WorkerState::Early E;
  E.clock = ws.clock + 1;
  advance_lists(ws, E.clock, E.open, E.close);
  if (E.open.empty() && E.close.empty()) return ADAPM_OK;
  if (!ctx->early_stream) CK(cudaStreamCreateWithFlags(&ctx->early_stream, cudaStreamNonBlocking));
  const std::vector<EventList> ev = event_lists(ctx, E.open, E.close);
  for (const auto& e : ev) E.cap += e.cap;
  CK(pool_alloc(ctx, &E.create_list, E.cap));
  CK(pool_alloc(ctx, &E.evict_list, E.cap));
  cudaEvent_t after = nullptr;
  CK(take_ready_event(ctx, &after));
  CK(cudaEventRecord(after, ctx->stream));
  CK(cudaStreamWaitEvent(ctx->early_stream, after, 0));
  ctx->spare_ready.push_back(after);   // the wait has captured it
  for (int64_t id : E.open)
    if (ctx->lists[id].from_plan) CK(cudaStreamWaitEvent(ctx->early_stream, ctx->lists[id].ready, 0));
  launch_events(ctx->s, w, ev.data(), (int)ev.size(), E.create_list, E.evict_list, ctx->sms, ctx->early_stream,
                ctx->early_counts + w);
  CK(take_ready_event(ctx, &E.done));
  CK(cudaEventRecord(E.done, ctx->early_stream));
  E.active = true;
  ws.early = std::move(E);
  return ADAPM_OK;
}

// The library stream waits for w's early events; their lists are freed
// after what the stream does with them.
adapm_status early_release(adapm_ctx* ctx, WorkerState::Early& E) {
  CK(cudaStreamWaitEvent(ctx->stream, E.done, 0));
  return ADAPM_OK;
}

void early_clear(adapm_ctx* ctx, WorkerState::Early& E) {
  pool_free(ctx, E.create_list);
  pool_free(ctx, E.evict_list);
  ctx->spare_ready.push_back(E.done);
  E = WorkerState::Early{};
}

adapm_status early_undo(adapm_ctx* ctx, uint32_t w) {
  WorkerState::Early& E = ctx->workers[w].early;
  if (!E.active) return ADAPM_OK;
  adapm_status st = early_release(ctx, E);
  if (st != ADAPM_OK) return st;
  const std::vector<EventList> ev = event_lists(ctx, E.open, E.close);
  launch_events_undo(ctx->s, w, ev.data(), (int)ev.size(), ctx->sms, ctx->stream);
  CK(cudaMemsetAsync(ctx->early_counts + w, 0, sizeof(AdvCounts), ctx->stream));
  early_clear(ctx, E);
  ctx->early_undone += 1;
  return check_launch(ctx, "early events (undo)");
}

adapm_status early_apply(adapm_ctx* ctx, uint32_t w) {
  WorkerState::Early& E = ctx->workers[w].early;
  adapm_status st = early_release(ctx, E);
  if (st != ADAPM_OK) return st;
  launch_evict_create(ctx->s, w, E.create_list, E.evict_list, E.cap, ctx->sms, ctx->stream,
                      ctx->early_counts + w);
  early_clear(ctx, E);
  ctx->early_advances += 1;
  return check_launch(ctx, "advance");
}

adapm_status apply_events(adapm_ctx* ctx, uint32_t w, const std::vector<EventList>& ev,
                          const std::vector<cudaEvent_t>& waits = {}) {
  {
    const adapm_status st = early_undo(ctx, w);   // the lists change: early events no longer hold
    if (st != ADAPM_OK) return st;
  }
  for (cudaEvent_t r : waits) CK(cudaStreamWaitEvent(ctx->stream, r, 0));
  uint64_t total = 0;
  for (const auto& e : ev) total += e.cap;
  if (total == 0) return ADAPM_OK;
  uint32_t *create_list = nullptr, *evict_list = nullptr;
  // with relocation a leaving key can also destroy another worker's replica
  const uint64_t max_events = ctx->s.own ? 2 * total : total;
  CK(pool_alloc(ctx, &create_list, total));
  CK(pool_alloc(ctx, &evict_list, max_events));
  // (the list counters are zero between advances: the last events launch clears them)
  launch_events(ctx->s, w, ev.data(), (int)ev.size(), create_list, evict_list, ctx->sms, ctx->stream);
  launch_evict_create(ctx->s, w, create_list, evict_list, max_events, ctx->sms, ctx->stream);
  pool_free(ctx, create_list);
  pool_free(ctx, evict_list);
  return check_launch(ctx, "apply_events");
}

// Group, sum and apply n delta rows (device keys/rows); keys may hold kNoKey
// when allow_nokey (rows the caller wants skipped).
// The plan a push of n keys by worker w may use: the newest recorded intent
// of w with n keys whose window (as signalled) holds the worker's clock.
IntentList* find_plan(adapm_ctx* ctx, uint32_t w, uint64_t n) {
  WorkerState& ws = ctx->workers[w];
  for (auto it = ws.order.rbegin(); it != ws.order.rend(); ++it) {
    IntentList& L = ctx->lists[*it];
    if (L.psk && L.n == n && L.start <= ws.clock && ws.clock < L.end) return &L;
  }
  return nullptr;
}

// plans = false: the caller knows its keys never follow an intent's order
// (the SGNS step), so no plan is looked up.
adapm_status push_device(adapm_ctx* ctx, uint32_t w, const uint32_t* dkeys, uint64_t n,
                         const float* drows, bool allow_nokey, bool plans = true) {
  if (n == 0) return ADAPM_OK;
  {
    const adapm_status st = early_make(ctx, w);
    if (st != ADAPM_OK) return st;
  }
  uint32_t *ka = nullptr, *kb = nullptr, *va = nullptr, *vb = nullptr, *hist = nullptr;
  // with a plan, the sort launch first checks on the device that the push's
  // keys are the ones the plan was made from, and sorts (into this push's
  // own arrays) only if they are not; the scatter kernels read the plan's
  // arrays or the sort's by the same check
  IntentList* plan = plans ? find_plan(ctx, w, n) : nullptr;
  uint32_t seq = 0;
  if (plan) {
    plan->plan_used = true;
    CK(cudaStreamWaitEvent(ctx->stream, plan->ready, 0));
    if (++ctx->plan_seq == 0) ctx->plan_seq = 1;
    seq = ctx->plan_seq;
    ctx->planned_pushes += 1;
  }
  CK(pool_alloc(ctx, &ka, n));
  CK(pool_alloc(ctx, &kb, n));
  CK(pool_alloc(ctx, &va, n));
  CK(pool_alloc(ctx, &vb, n));
  CK(pool_alloc(ctx, &hist, sort_scratch_words(n)));
  const uint64_t chunk = push_chunk_rows(ctx->s.D, n, ctx->sms);
  const uint64_t nchunks = (n + chunk - 1) / chunk;
  float* sparts = nullptr;
  CK(pool_alloc(ctx, &sparts, push_span_part_rows(nchunks) * ctx->s.D));
  // the sort also clears the distinct-key counter
  uint32_t *sk = nullptr, *sp = nullptr;
  CK(sort_keys(dkeys, n, ctx->s.K, allow_nokey, ctx->bits, ka, kb, va, vb, hist, ctx->sms, ctx->dstate,
               &ctx->bar_base, &ctx->dstate->last_unique, nullptr, ctx->stream, &sk, &sp,
               plan ? plan->px : nullptr, plan ? &ctx->dstate->plan_miss : nullptr, seq));
  ctx->push_rows_host += n;
  PushArgs a{sk, sp, n, drows, chunk, nchunks, w, sparts};
  if (plan) {
    a.skeys = plan->psk;
    a.spos = plan->psp;
    a.alt_keys = sk;
    a.alt_pos = sp;
    a.plan_word = &ctx->dstate->plan_miss;
    a.plan_seq = seq;
  }
  {
    ProfScope ps(ctx, 6);
    launch_push(ctx->s, a, ctx->sms, ctx->stream);
  }
  for (uint32_t* p : {ka, kb, va, vb}) pool_free(ctx, p);
  pool_free(ctx, hist);
  pool_free(ctx, sparts);
  return check_launch(ctx, "push");
}

// The p quantile of Poisson(lam): P(X = j) added for j = 0, 1, ... in order
// until the sum reaches p.  The loop ends: the sum tends to 1 > p (a bound on
// the index guards against rounding for huge lam).
int64_t poisson_quantile(double lam, double p) {
  const double ln_lam = std::log(lam);
  const double qmax = lam + 64.0 * std::sqrt(lam) + 64.0;
  double cdf = 0.0;
  int64_t q = 0;
  for (;; ++q) {
    const double j = (double)q;
    cdf += std::exp(-lam + j * ln_lam - std::lgamma(j + 1.0));
    if (cdf >= p || j >= qmax) return q;
  }
}

// One communication round of adaptive action timing (Sec. 4.2, Algorithm 1),
// after the sync's merge: each worker in ascending order updates its rate
// estimate and activates the recorded intents that start before its clock
// plus the Poisson bound.
adapm_status act_in_round(adapm_ctx* ctx) {
  const double alpha = ctx->cfg.timing_alpha, p = ctx->cfg.timing_p;
  for (uint32_t w = 0; w < ctx->s.W; ++w) {
    WorkerState& ws = ctx->workers[w];
    const int64_t delta = ws.clock - ws.round_clock;
    if (delta > 0) ws.est = (1.0 - alpha) * ws.est + alpha * (double)delta;
    ws.round_clock = ws.clock;
    const int64_t bound = poisson_quantile(2.0 * std::max(ws.est, (double)delta), p);
    std::vector<EventList> ev;
    std::vector<cudaEvent_t> waits;
    auto it = ws.starts.begin();
    while (it != ws.starts.end() && it->first < ws.clock + bound) {
      for (int64_t id : it->second) {
        const IntentList& L = ctx->lists[id];
        ev.push_back(EventList{L.keys, L.count, L.cap, +1});
        if (L.from_plan) waits.push_back(L.ready);
      }
      it = ws.starts.erase(it);
    }
    if (!ev.empty()) {
      const adapm_status st = apply_events(ctx, w, ev, waits);
      if (st != ADAPM_OK) return st;
    }
  }
  return ADAPM_OK;
}

// Sort an intent's keys with their positions on the plan stream (a phased
// sort: no block waits for another, so it runs in whatever the library
// stream leaves of the GPU), into L.psk / L.psp; with from_plan the distinct
// keys follow from the sorted ones (ascending) into L.keys / L.count.
// L.ready is recorded on the plan stream after all of it.  The library
// stream must have enqueued the keys (and L's arrays) before `after`.
cudaError_t make_plan(adapm_ctx* ctx, IntentList& L, const uint32_t* keys, cudaEvent_t after) {
  cudaError_t e = ensure_plan_stream(ctx);
  if (e != cudaSuccess) return e;
  cudaStream_t ps = ctx->plan_stream;
  const uint64_t n = L.n;
  if ((e = cudaStreamWaitEvent(ps, after, 0)) != cudaSuccess) return e;
  if ((e = cudaMemcpyAsync(L.px, keys, n * sizeof(uint32_t), cudaMemcpyDeviceToDevice, ps)) != cudaSuccess) return e;
  uint32_t *tk = nullptr, *tv = nullptr, *hist = nullptr, *tmp = nullptr;
  auto palloc = [&](uint32_t** p, size_t words) {
    return cudaMallocFromPoolAsync(reinterpret_cast<void**>(p), (words ? words : 1) * sizeof(uint32_t),
                                   ctx->plan_pool, ps);
  };
  if ((e = palloc(&tk, n)) != cudaSuccess || (e = palloc(&tv, n)) != cudaSuccess ||
      (e = palloc(&hist, sort_scratch_words(n))) != cudaSuccess ||
      (e = palloc(&tmp, compact_tmp_words(n))) != cudaSuccess)
    return e;
  const bool odd = sort_passes(ctx->bits) % 2 == 1;   // the sort ends in ka / va after odd passes
  unsigned long long no_barriers = 0;
  uint32_t *sk = nullptr, *sp = nullptr;
  e = sort_keys(keys, n, ctx->s.K, false, ctx->bits, odd ? L.psk : tk, odd ? tk : L.psk, odd ? L.psp : tv,
                odd ? tv : L.psp, hist, ctx->sms, ctx->dstate, &no_barriers, nullptr, nullptr, ps, &sk, &sp,
                nullptr, nullptr, 0, /*phased=*/true);
  if (e != cudaSuccess) return e;
  if (L.from_plan) compact_sorted_heads(L.psk, n, L.keys, L.count, tmp, ps);
  for (uint32_t* p : {tk, tv, hist, tmp}) cudaFreeAsync(p, ps);
  if ((e = take_ready_event(ctx, &L.ready)) != cudaSuccess) return e;
  if ((e = cudaEventRecord(L.ready, ps)) != cudaSuccess) return e;
  return cudaGetLastError();
}

// Free an intent list whose window closed (on the library stream, after
// its plan is complete).
cudaError_t close_list(adapm_ctx* ctx, uint32_t w, int64_t id) {
  IntentList& L = ctx->lists[id];
  cudaError_t e = cudaSuccess;
  if (L.psk) {
    int& unused = ctx->workers[w].unused_plans;
    unused = L.plan_used ? 0 : unused + 1;
  }
  if (L.ready) {
    e = cudaStreamWaitEvent(ctx->stream, L.ready, 0);
    ctx->spare_ready.push_back(L.ready);   // the wait has captured it; it can be recorded again
  }
  for (void* p : {(void*)L.keys, (void*)L.psk, (void*)L.psp, (void*)L.px, L.in_owned}) pool_free(ctx, p);
  auto& order = ctx->workers[w].order;
  order.erase(std::remove(order.begin(), order.end(), id), order.end());
  ctx->lists.erase(id);
  return e;
}

}  // namespace

bool adapm::ctx_view(adapm_ctx* ctx, CtxView* out) {
  if (!ctx || !out) return false;
  out->s = ctx->s;
  out->dstate = ctx->dstate;
  out->stream = ctx->stream;
  out->device = ctx->device;
  out->sms = ctx->sms;
  out->bits = ctx->bits;
  out->broken = ctx->broken;
  out->bar_base = &ctx->bar_base;
  return true;
}

void adapm::ctx_set_error(adapm_ctx* ctx, const char* msg) {
  if (ctx) ctx->err = msg;
}

void adapm::ctx_add_push_rows(adapm_ctx* ctx, uint64_t n) {
  if (ctx) ctx->push_rows_host += n;
}

int adapm::ctx_begin(adapm_ctx* ctx) { return check_ctx(ctx); }

int adapm::ctx_fail_cuda(adapm_ctx* ctx, cudaError_t e, const char* where) { return cuda_fail(ctx, e, where); }

cudaError_t adapm::ctx_launch_error(adapm_ctx* ctx) {
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess && ctx->fake_launch_error) e = cudaErrorLaunchFailure;   // adapm_debug_fail_next_launch
  ctx->fake_launch_error = false;
  return e;
}

ProfToken adapm::ctx_prof_start(adapm_ctx* ctx, int op) {
  ProfToken t;
  if (!ctx || !ctx->prof) return t;
  t.op = op;
  t.a = take_prof_event(ctx);
  t.b = take_prof_event(ctx);
  if (t.a) cudaEventRecord(t.a, ctx->stream);
  return t;
}

void adapm::ctx_prof_stop(adapm_ctx* ctx, ProfToken& t) {
  if (!ctx || t.op < 0) return;
  if (t.a && t.b) {
    cudaEventRecord(t.b, ctx->stream);
    ctx->pending.emplace_back(t.op, t.a, t.b);
  } else {   // an event could not be made: give back the one that was
    if (t.a) ctx->spare_events.push_back(t.a);
    if (t.b) ctx->spare_events.push_back(t.b);
  }
  t = ProfToken{};
}

extern "C" {

adapm_status adapm_create(const adapm_config* cfg, adapm_ctx** out) {
  if (!cfg || !out) return ADAPM_EINVAL;
  *out = nullptr;
  if (cfg->num_keys < 1 || cfg->num_keys >= 0xFFFFFFFFull || cfg->value_len == 0 ||
      cfg->value_len % 4 != 0 || cfg->value_len > 1024 || cfg->num_workers < 1 ||
      cfg->num_workers > (uint32_t)kMaxWorkers || (cfg->relocate != 0 && cfg->relocate != 1) ||
      cfg->action_timing < ADAPM_ACT_AT_START || cfg->action_timing > ADAPM_ACT_ON_SIGNAL ||
      !(cfg->timing_alpha >= 0.0 && cfg->timing_alpha <= 1.0) ||
      !(cfg->timing_p >= 0.0 && cfg->timing_p < 1.0) || !(cfg->timing_lambda0 >= 0.0) ||
      (cfg->delta_refresh != 0 && cfg->delta_refresh != 1) || (cfg->no_push_plans != 0 && cfg->no_push_plans != 1) ||
      (cfg->pull_staging != 0 && cfg->pull_staging != 1) ||
      (cfg->no_early_events != 0 && cfg->no_early_events != 1))
    return ADAPM_EINVAL;
  adapm_ctx* ctx = new (std::nothrow) adapm_ctx();
  if (!ctx) return ADAPM_ENOMEM;
  ctx->cfg = *cfg;
  if (ctx->cfg.timing_alpha == 0.0) ctx->cfg.timing_alpha = 0.1;
  if (ctx->cfg.timing_p == 0.0) ctx->cfg.timing_p = 0.9999;
  if (ctx->cfg.timing_lambda0 == 0.0) ctx->cfg.timing_lambda0 = 10.0;
  const uint64_t K = cfg->num_keys, D = cfg->value_len, W = cfg->num_workers;
  uint64_t S = cfg->replica_capacity;
  if (S == 0) S = W * K < (1ull << 24) ? W * K : (1ull << 24);
  if (S >= (1ull << 31)) S = (1ull << 31) - 1;
  auto bail = [&](adapm_status st) {
    adapm_destroy(ctx);
    return st;
  };
  if (cudaGetDevice(&ctx->device) != cudaSuccess) return bail(ADAPM_ECUDA);
  cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, ctx->device);
  if (cfg->stream) {
    ctx->stream = (cudaStream_t)cfg->stream;
  } else {
    if (cudaStreamCreateWithFlags(&ctx->stream, cudaStreamNonBlocking) != cudaSuccess)
      return bail(ADAPM_ECUDA);
    ctx->own_stream = true;
  }
  cudaMemPoolProps props{};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = ctx->device;
  if (cudaMemPoolCreate(&ctx->pool, &props) != cudaSuccess) return bail(ADAPM_ECUDA);
  uint64_t keep = ~0ull;
  cudaMemPoolSetAttribute(ctx->pool, cudaMemPoolAttrReleaseThreshold, &keep);

  ctx->bits = bits_for(K);
  Store& s = ctx->s;
  s.K = K;
  s.S = S;
  s.D = (uint32_t)D;
  s.W = (uint32_t)W;
  auto dmalloc = [&](void** p, size_t bytes) { return cudaMalloc(p, bytes) == cudaSuccess; };
  if (!dmalloc((void**)&s.main, K * D * 4) || !dmalloc((void**)&s.val, S * D * 4) ||
      !dmalloc((void**)&s.acc, S * D * 4) || !dmalloc((void**)&s.map, W * K * 4) ||
      !dmalloc((void**)&s.rc, W * K * 4) || !dmalloc((void**)&s.holders, K * 4) ||
      !dmalloc((void**)&s.slot_owner, S * 8) || !dmalloc((void**)&s.free_stack, S * 4) ||
      !dmalloc((void**)&s.stamp, K * 4) || (cfg->relocate && !dmalloc((void**)&s.own, K * 2)) ||
      (cfg->delta_refresh && !dmalloc((void**)&s.dirty, K)) ||
      !dmalloc((void**)&ctx->dstate, sizeof(DevState)) ||
      !dmalloc((void**)&ctx->early_counts, W * sizeof(AdvCounts))) {
    cudaGetLastError();
    return bail(ADAPM_ENOMEM);
  }
  s.st = ctx->dstate;
  cudaStream_t st = ctx->stream;
  bool ok = true;
  if (cfg->init_values) {
    ok &= cudaMemcpyAsync(s.main, cfg->init_values, K * D * 4, cudaMemcpyDefault, st) == cudaSuccess;
  } else {
    ok &= cudaMemsetAsync(s.main, 0, K * D * 4, st) == cudaSuccess;
  }
  ok &= cudaMemsetAsync(s.map, 0xFF, W * K * 4, st) == cudaSuccess;   // -1: no replica
  ok &= cudaMemsetAsync(s.rc, 0, W * K * 4, st) == cudaSuccess;
  ok &= cudaMemsetAsync(s.holders, 0, K * 4, st) == cudaSuccess;
  ok &= cudaMemsetAsync(s.stamp, 0, K * 4, st) == cudaSuccess;   // intent tags start at 1
  if (s.own) ok &= cudaMemsetAsync(s.own, 0, K * 2, st) == cudaSuccess;   // home, no active worker
  if (s.dirty) ok &= cudaMemsetAsync(s.dirty, 0, K, st) == cudaSuccess;
  ok &= cudaMemsetAsync(ctx->early_counts, 0, W * sizeof(AdvCounts), st) == cudaSuccess;
  DevState h{};
  h.free_top = (int32_t)S;
  ok &= cudaMemcpyAsync(ctx->dstate, &h, sizeof h, cudaMemcpyHostToDevice, st) == cudaSuccess;
  launch_init_pool(s.free_stack, S, s.slot_owner, st);
  ok &= cudaStreamSynchronize(st) == cudaSuccess;
  if (!ok || cudaGetLastError() != cudaSuccess) return bail(ADAPM_ECUDA);
  ctx->workers.resize(W);
  for (auto& ws : ctx->workers) ws.est = ctx->cfg.timing_lambda0;
  *out = ctx;
  return ADAPM_OK;
}

adapm_status adapm_destroy(adapm_ctx* ctx) {
  if (!ctx) return ADAPM_EINVAL;
  cudaSetDevice(ctx->device);
  if (ctx->stream) cudaStreamSynchronize(ctx->stream);
  if (ctx->plan_stream) cudaStreamSynchronize(ctx->plan_stream);
  if (ctx->early_stream) cudaStreamSynchronize(ctx->early_stream);
  for (auto& ws : ctx->workers) {
    if (!ws.early.active) continue;
    for (void* p : {(void*)ws.early.create_list, (void*)ws.early.evict_list})
      if (p) cudaFree(p);
    if (ws.early.done) cudaEventDestroy(ws.early.done);
  }
  for (auto& kv : ctx->lists) {
    for (void* p : {(void*)kv.second.keys, (void*)kv.second.psk, (void*)kv.second.psp, (void*)kv.second.px,
                    kv.second.in_owned})
      if (p) cudaFree(p);
    if (kv.second.ready) cudaEventDestroy(kv.second.ready);
  }
  for (auto e : ctx->spare_ready) cudaEventDestroy(e);
  Store& s = ctx->s;
  void* ptrs[] = {s.main, s.val, s.acc, s.map, s.rc, s.holders, s.slot_owner, s.free_stack,
                  s.stamp, s.own, s.dirty, ctx->dstate, ctx->early_counts};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  for (auto& t : ctx->pending) {
    cudaEventDestroy(std::get<1>(t));
    cudaEventDestroy(std::get<2>(t));
  }
  for (auto e : ctx->spare_events) cudaEventDestroy(e);
  if (ctx->copy_in) cudaStreamSynchronize(ctx->copy_in);
  for (auto& m : ctx->stage_marks) cudaEventDestroy(m.first);
  for (auto e : ctx->spare_marks) cudaEventDestroy(e);
  if (ctx->staged) cudaEventDestroy(ctx->staged);
  if (ctx->copy_in) cudaStreamDestroy(ctx->copy_in);
  if (ctx->stage_pool) cudaMemPoolDestroy(ctx->stage_pool);
  if (ctx->plan_stream) cudaStreamDestroy(ctx->plan_stream);
  if (ctx->early_stream) cudaStreamDestroy(ctx->early_stream);
  if (ctx->plan_pool) cudaMemPoolDestroy(ctx->plan_pool);
  if (ctx->pool) cudaMemPoolDestroy(ctx->pool);
  if (ctx->own_stream && ctx->stream) cudaStreamDestroy(ctx->stream);
  cudaGetLastError();
  delete ctx;
  return ADAPM_OK;
}

adapm_status adapm_intent(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                          int64_t clock_start, int64_t clock_end) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  if (n > kMaxN || (n > 0 && !keys)) return fail(ctx, ADAPM_EINVAL, "bad keys/n");
  WorkerState& ws = ctx->workers[worker];
  if (clock_end <= clock_start || clock_end <= ws.clock) return ADAPM_OK;   // never active
  const int64_t signalled_start = clock_start;
  // acting on signal: the window starts now
  if (ctx->cfg.action_timing == ADAPM_ACT_ON_SIGNAL && clock_start > ws.clock) clock_start = ws.clock;
  ProfScope ps(ctx, 0);
  IntentList L;
  L.cap = n;
  L.n = n;
  L.start = signalled_start;
  L.end = clock_end;
  const bool now = clock_start <= ws.clock;   // the window contains the current clock: active at once
  // a plan unless the worker's recent ones all went unused (then one probe in kPlanProbe)
  const bool plan = n > 0 && !ctx->cfg.no_push_plans &&
                    (ws.unused_plans < kPlanPatience || ws.intents % kPlanProbe == 0);
  ws.intents += 1;
  CK(cudaMallocFromPoolAsync((void**)&L.keys, (n + 1) * sizeof(uint32_t), ctx->pool, ctx->stream));
  L.count = L.keys + n;
  if (n == 0) {
    CK(cudaMemsetAsync(L.count, 0, sizeof(uint32_t), ctx->stream));
  } else {
    Input<uint32_t> in;
    CK(stage_in(ctx, keys, n, &in));
    if (plan) {
      CK(pool_alloc(ctx, &L.psk, n));
      CK(pool_alloc(ctx, &L.psp, n));
      CK(pool_alloc(ctx, &L.px, n));
    }
    // a window that opens two or more clocks ahead takes its distinct keys
    // from the plan; one that opens at the next advance (or is active now)
    // would wait there for the plan, so its keys come from the hash-set pass
    // here, and the plan only serves the push a clock later
    L.from_plan = plan && clock_start > ws.clock + 1;
    if (!L.from_plan) {
      if (++ctx->intent_tag == 0) {   // tags wrapped: clear the stamps
        CK(cudaMemsetAsync(ctx->s.stamp, 0, ctx->s.K * 4, ctx->stream));
        ctx->intent_tag = 1;
      }
      CK(cudaMemsetAsync(L.count, 0, sizeof(uint32_t), ctx->stream));
      launch_intent_dedup(ctx->s, in.dev, n, ctx->intent_tag, L.keys, L.count, ctx->sms, ctx->stream);
    }
    if (plan) {
      cudaEvent_t after = nullptr;
      CK(take_ready_event(ctx, &after));
      CK(cudaEventRecord(after, ctx->stream));
      CK(make_plan(ctx, L, in.dev, after));
      ctx->spare_ready.push_back(after);   // the plan stream's wait has captured it
      L.in_owned = in.owned;               // freed when the list closes, after the plan
    } else {
      pool_free(ctx, in.owned);
    }
  }
  const int64_t id = ctx->next_list++;
  ctx->lists[id] = L;
  ws.order.push_back(id);
  if (now) {
    st = apply_events(ctx, worker, {EventList{L.keys, L.count, L.cap, +1}});
    if (st != ADAPM_OK) return st;
  } else {
    ws.starts[clock_start].push_back(id);
  }
  ws.ends[clock_end].push_back(id);
  return check_launch(ctx, "intent");
}

adapm_status adapm_advance_clock(adapm_ctx* ctx, uint32_t worker) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  WorkerState& ws = ctx->workers[worker];
  ws.clock += 1;
  const int64_t c = ws.clock;
  if (ws.early.active) {
    std::vector<int64_t> open, close;
    advance_lists(ws, c, open, close);
    if (ws.early.clock == c && open == ws.early.open && close == ws.early.close) {
      // the events ran ahead: evict and create only
      {
        ProfScope ps(ctx, 1);
        st = early_apply(ctx, worker);
      }
      ws.starts.erase(c);
      ws.ends.erase(c);
      for (int64_t id : close) CK(close_list(ctx, worker, id));
      return st;
    }
    st = early_undo(ctx, worker);
    if (st != ADAPM_OK) return st;
  }
  std::vector<EventList> ev;
  std::vector<int64_t> closing;
  std::vector<cudaEvent_t> waits;   // plans that the opening lists' distinct keys come from
  auto it = ws.starts.find(c);
  if (it != ws.starts.end()) {
    for (int64_t id : it->second) {
      const IntentList& L = ctx->lists[id];
      ev.push_back(EventList{L.keys, L.count, L.cap, +1});
      if (L.from_plan) waits.push_back(L.ready);
    }
    ws.starts.erase(it);
  }
  it = ws.ends.find(c);
  if (it != ws.ends.end()) {
    for (int64_t id : it->second) {
      const IntentList& L = ctx->lists[id];
      ev.push_back(EventList{L.keys, L.count, L.cap, -1});
      closing.push_back(id);
    }
    ws.ends.erase(it);
  }
  if (ev.empty()) return ADAPM_OK;
  ProfScope ps(ctx, 1);
  st = apply_events(ctx, worker, ev, waits);
  for (int64_t id : closing) CK(close_list(ctx, worker, id));
  return st;
}

adapm_status adapm_pull(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                        float* out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  if (n > kMaxN || (n > 0 && (!keys || !out))) return fail(ctx, ADAPM_EINVAL, "bad pointers/n");
  if (n == 0) return ADAPM_OK;
  st = early_make(ctx, worker);
  if (st != ADAPM_OK) return st;
  ProfScope ps(ctx, 2);
  Input<uint32_t> in;
  CK(stage_in(ctx, keys, n, &in));
  Output<float> o;
  CK(stage_out(ctx, out, n * ctx->s.D, &o));
  {
    ProfScope pk(ctx, 7);
    if (ctx->cfg.pull_staging && pull_bulk_fits(ctx->s.D, o.dev))
      launch_pull_bulk(ctx->s, (int)worker, in.dev, n, o.dev, ctx->sms, ctx->stream);
    else
      launch_pull(ctx->s, (int)worker, in.dev, n, o.dev, ctx->sms, ctx->stream);
  }
  CK(finish_out(ctx, &o));
  pool_free(ctx, in.owned);
  return check_launch(ctx, "pull");
}

adapm_status adapm_push(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                        const float* deltas) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  if (n > kMaxN || (n > 0 && (!keys || !deltas))) return fail(ctx, ADAPM_EINVAL, "bad pointers/n");
  if (n == 0) return ADAPM_OK;
  ProfScope ps(ctx, 3);
  Input<uint32_t> ik;
  Input<float> id;
  CK(stage_in(ctx, keys, n, &ik));
  CK(stage_in(ctx, deltas, n * ctx->s.D, &id));
  if (reinterpret_cast<uintptr_t>(id.dev) % 16 != 0) {
    // the push copies whole rows with the bulk-copy engine: 16-byte aligned rows
    float* aligned = nullptr;
    CK(pool_alloc(ctx, &aligned, n * ctx->s.D));
    CK(cudaMemcpyAsync(aligned, id.dev, n * ctx->s.D * sizeof(float), cudaMemcpyDeviceToDevice,
                       ctx->stream));
    pool_free(ctx, id.owned);
    id.owned = aligned;
    id.dev = aligned;
  }
  st = push_device(ctx, worker, ik.dev, n, id.dev, false);
  pool_free(ctx, ik.owned);
  pool_free(ctx, id.owned);
  return st;
}

adapm_status adapm_sync(adapm_ctx* ctx) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  {
    ProfScope ps(ctx, 4);
    launch_sync(ctx->s, ctx->s.S, ctx->sms, ctx->stream);
    st = check_launch(ctx, "sync");
    if (st != ADAPM_OK) return st;
  }
  if (ctx->cfg.action_timing == ADAPM_ACT_ADAPTIVE) return act_in_round(ctx);
  return ADAPM_OK;
}

adapm_status adapm_poisson_quantile(double lambda, double p, int64_t* out) {
  if (!out || !(lambda > 0.0) || !(p > 0.0 && p < 1.0)) return ADAPM_EINVAL;
  *out = poisson_quantile(lambda, p);
  return ADAPM_OK;
}

adapm_status adapm_debug_fail_next_launch(adapm_ctx* ctx) {
  if (!ctx) return ADAPM_EINVAL;
  ctx->fake_launch_error = true;
  return ADAPM_OK;
}

adapm_status adapm_debug_fail_next_barrier(adapm_ctx* ctx) {
  if (!ctx) return ADAPM_EINVAL;
  // the next sort expects arrivals far beyond those that can happen
  ctx->bar_base += 1ull << 40;
  return ADAPM_OK;
}

adapm_status adapm_wait(adapm_ctx* ctx) {
  if (!ctx) return ADAPM_EINVAL;
  if (ctx->broken) return fail(ctx, ADAPM_ECUDA, "context unusable after an earlier CUDA error");
  cudaSetDevice(ctx->device);
  CK(cudaStreamSynchronize(ctx->stream));
  if (ctx->plan_stream) CK(cudaStreamSynchronize(ctx->plan_stream));   // plans read the callers' keys
  if (ctx->early_stream) CK(cudaStreamSynchronize(ctx->early_stream));
  uint32_t errors = 0;
  CK(cudaMemcpy(&errors, &ctx->dstate->errors, sizeof errors, cudaMemcpyDeviceToHost));
  if (errors) CK(cudaMemset(&ctx->dstate->errors, 0, sizeof errors));
  if (errors & ERR_TIMEOUT) {
    ctx->broken = true;   // the grid-barrier state of the sort is unknown
    return fail(ctx, ADAPM_ETIMEOUT, "a bounded device wait gave up");
  }
  if (errors & ERR_KEY_RANGE) return fail(ctx, ADAPM_ERANGE, "a key >= num_keys was passed");
  if (errors & ERR_NO_SLOTS) return fail(ctx, ADAPM_ENOMEM, "replica capacity exhausted");
  if (errors & ERR_REFCOUNT) return fail(ctx, ADAPM_ESTATE, "intent refcount overflow");
  if (errors & ERR_INTERNAL)
    return fail(ctx, ADAPM_ESTATE, "an index in the library's own state was out of range (element skipped)");
  return ADAPM_OK;
}

adapm_status adapm_mf_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* row_keys,
                           const uint32_t* col_keys, const float* vals, uint64_t n, uint32_t dim,
                           int adagrad, float lr, float eps, double* loss_out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  if (n > kMaxN / 2 || (n > 0 && (!row_keys || !col_keys || !vals)))
    return fail(ctx, ADAPM_EINVAL, "bad pointers/n");
  if (dim == 0 || (adagrad ? 2 * dim : dim) != ctx->s.D)
    return fail(ctx, ADAPM_EINVAL, "dim %u does not match value_len %u", dim, ctx->s.D);
  Output<double> lo;
  if (loss_out) CK(stage_out(ctx, loss_out, 1, &lo));
  if (n == 0) {
    if (loss_out) {
      CK(cudaMemsetAsync(lo.dev, 0, sizeof(double), ctx->stream));
      CK(finish_out(ctx, &lo));
    }
    return ADAPM_OK;
  }
  Input<uint32_t> ir, ic;
  Input<float> iv;
  CK(stage_in(ctx, row_keys, n, &ir));
  CK(stage_in(ctx, col_keys, n, &ic));
  CK(stage_in(ctx, vals, n, &iv));
  const uint64_t m = 2 * n;
  StepOut o{};
  o.loss_blocks = step_loss_blocks(ctx->sms);
  o.loss_out = loss_out ? lo.dev : nullptr;   // summed by the step kernel's last block
  o.loss_done = &ctx->dstate->loss_done;
  CK(pool_alloc(ctx, &o.dkeys, m));
  CK(pool_alloc(ctx, &o.drows, m * ctx->s.D));
  CK(pool_alloc(ctx, &o.loss_part, o.loss_blocks));
  st = early_make(ctx, worker);
  if (st != ADAPM_OK) return st;
  {
    ProfScope ps(ctx, 5);
    launch_mf_step(ctx->s, worker, ir.dev, ic.dev, iv.dev, n, dim, adagrad != 0, lr, eps, o,
                   ctx->sms, ctx->stream);
  }
  {
    ProfScope ps(ctx, 3);
    st = push_device(ctx, worker, o.dkeys, m, o.drows, true);
  }
  if (loss_out) CK(finish_out(ctx, &lo));
  pool_free(ctx, ir.owned);
  pool_free(ctx, ic.owned);
  pool_free(ctx, iv.owned);
  pool_free(ctx, o.dkeys);
  pool_free(ctx, o.drows);
  pool_free(ctx, o.loss_part);
  if (st != ADAPM_OK) return st;
  return check_launch(ctx, "mf_step");
}

adapm_status adapm_complex_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* heads,
                                const uint32_t* rels, const uint32_t* tails,
                                const uint32_t* neg_tails, uint64_t n, uint32_t n_neg,
                                uint32_t dim, float lr, float eps, double* loss_out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  if (n > kMaxN / (3 + (uint64_t)n_neg) ||
      (n > 0 && (!heads || !rels || !tails || (n_neg > 0 && !neg_tails))))
    return fail(ctx, ADAPM_EINVAL, "bad pointers/n");
  if (dim == 0 || dim % 2 != 0 || 2 * dim != ctx->s.D)
    return fail(ctx, ADAPM_EINVAL, "dim %u: need even dim with value_len = 2*dim", dim);
  Output<double> lo;
  if (loss_out) CK(stage_out(ctx, loss_out, 1, &lo));
  if (n == 0) {
    if (loss_out) {
      CK(cudaMemsetAsync(lo.dev, 0, sizeof(double), ctx->stream));
      CK(finish_out(ctx, &lo));
    }
    return ADAPM_OK;
  }
  Input<uint32_t> ih, ir, it, ineg;
  CK(stage_in(ctx, heads, n, &ih));
  CK(stage_in(ctx, rels, n, &ir));
  CK(stage_in(ctx, tails, n, &it));
  CK(stage_in(ctx, neg_tails, n * n_neg, &ineg));
  const uint64_t m = n * (3 + (uint64_t)n_neg);
  StepOut o{};
  o.loss_blocks = step_loss_blocks(ctx->sms);
  o.loss_out = loss_out ? lo.dev : nullptr;   // summed by the step kernel's last block
  o.loss_done = &ctx->dstate->loss_done;
  CK(pool_alloc(ctx, &o.dkeys, m));
  CK(pool_alloc(ctx, &o.drows, m * ctx->s.D));
  CK(pool_alloc(ctx, &o.loss_part, o.loss_blocks));
  st = early_make(ctx, worker);
  if (st != ADAPM_OK) return st;
  {
    ProfScope ps(ctx, 5);
    launch_complex_step(ctx->s, worker, ih.dev, ir.dev, it.dev, ineg.dev, n, n_neg, dim, lr, eps,
                        o, ctx->sms, ctx->stream);
  }
  {
    ProfScope ps(ctx, 3);
    st = push_device(ctx, worker, o.dkeys, m, o.drows, true);
  }
  if (loss_out) CK(finish_out(ctx, &lo));
  for (void* p : {(void*)ih.owned, (void*)ir.owned, (void*)it.owned, (void*)ineg.owned,
                  (void*)o.dkeys, (void*)o.drows, (void*)o.loss_part})
    pool_free(ctx, p);
  if (st != ADAPM_OK) return st;
  return check_launch(ctx, "complex_step");
}

adapm_status adapm_sgns_step(adapm_ctx* ctx, uint32_t worker, const uint32_t* centres,
                             const uint32_t* contexts, const uint32_t* negatives, uint64_t n,
                             uint32_t n_ctx, uint32_t n_neg, uint32_t vocab, uint32_t dim,
                             float lr, double* loss_out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  const uint64_t per = 1 + (uint64_t)n_ctx * (1 + (uint64_t)n_neg);
  if (n > kMaxN / per || (n > 0 && (!centres || (n_ctx > 0 && !contexts) ||
                                    (n_ctx > 0 && n_neg > 0 && !negatives))))
    return fail(ctx, ADAPM_EINVAL, "bad pointers/n");
  if (dim != ctx->s.D) return fail(ctx, ADAPM_EINVAL, "dim %u != value_len %u", dim, ctx->s.D);
  if (2ull * vocab > ctx->s.K) return fail(ctx, ADAPM_EINVAL, "2*vocab exceeds num_keys");
  Output<double> lo;
  if (loss_out) CK(stage_out(ctx, loss_out, 1, &lo));
  if (n == 0) {
    if (loss_out) {
      CK(cudaMemsetAsync(lo.dev, 0, sizeof(double), ctx->stream));
      CK(finish_out(ctx, &lo));
    }
    return ADAPM_OK;
  }
  Input<uint32_t> ic, ix, ineg;
  CK(stage_in(ctx, centres, n, &ic));
  CK(stage_in(ctx, contexts, n * n_ctx, &ix));
  CK(stage_in(ctx, negatives, n * n_ctx * n_neg, &ineg));
  const uint64_t m = n * per;
  StepOut o{};
  o.loss_blocks = step_loss_blocks(ctx->sms);
  o.loss_out = loss_out ? lo.dev : nullptr;   // summed by the step kernel's last block
  o.loss_done = &ctx->dstate->loss_done;
  CK(pool_alloc(ctx, &o.dkeys, m));
  CK(pool_alloc(ctx, &o.drows, m * ctx->s.D));
  CK(pool_alloc(ctx, &o.loss_part, o.loss_blocks));
  st = early_make(ctx, worker);
  if (st != ADAPM_OK) return st;
  {
    ProfScope ps(ctx, 5);
    launch_sgns_step(ctx->s, worker, ic.dev, ix.dev, ineg.dev, n, n_ctx, n_neg, vocab, dim, lr, o,
                     ctx->sms, ctx->stream);
  }
  {
    ProfScope ps(ctx, 3);
    // its rows follow the centres (each with its context and negative slots),
    // never an intent's key order: no plan
    st = push_device(ctx, worker, o.dkeys, m, o.drows, true, /*plans=*/false);
  }
  if (loss_out) CK(finish_out(ctx, &lo));
  for (void* p : {(void*)ic.owned, (void*)ix.owned, (void*)ineg.owned, (void*)o.dkeys,
                  (void*)o.drows, (void*)o.loss_part})
    pool_free(ctx, p);
  if (st != ADAPM_OK) return st;
  return check_launch(ctx, "sgns_step");
}

adapm_status adapm_clock(adapm_ctx* ctx, uint32_t worker, int64_t* out) {
  if (!ctx || !out) return ADAPM_EINVAL;
  if (worker >= ctx->s.W) return fail(ctx, ADAPM_EINVAL, "worker %u >= %u", worker, ctx->s.W);
  *out = ctx->workers[worker].clock;
  return ADAPM_OK;
}

adapm_status adapm_replica_keys(adapm_ctx* ctx, uint32_t worker, uint32_t* out, uint64_t cap,
                                uint64_t* n) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W || !n || (cap > 0 && !out)) return fail(ctx, ADAPM_EINVAL, "bad arguments");
  uint32_t *buf = nullptr, *tmp = nullptr, *cnt = nullptr;
  CK(pool_alloc(ctx, &buf, ctx->s.K));
  CK(pool_alloc(ctx, &tmp, compact_tmp_words(ctx->s.K)));
  CK(pool_alloc(ctx, &cnt, 1));
  compact_replica_keys(ctx->s.map + (uint64_t)worker * ctx->s.K, ctx->s.K, buf, cnt, tmp, ctx->stream);
  uint32_t hcnt = 0;
  CK(cudaMemcpyAsync(&hcnt, cnt, sizeof hcnt, cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  *n = hcnt;
  const uint64_t m = hcnt < cap ? hcnt : cap;
  if (m > 0) CK(cudaMemcpyAsync(out, buf, m * 4, cudaMemcpyDefault, ctx->stream));
  pool_free(ctx, buf);
  pool_free(ctx, tmp);
  pool_free(ctx, cnt);
  CK(cudaStreamSynchronize(ctx->stream));
  return check_launch(ctx, "replica_keys");
}

adapm_status adapm_replica_rows(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                                float* val_out, float* acc_out, uint8_t* has_out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W || n > kMaxN || (n > 0 && (!keys || !val_out || !acc_out || !has_out)))
    return fail(ctx, ADAPM_EINVAL, "bad arguments");
  if (n == 0) return ADAPM_OK;
  Input<uint32_t> in;
  CK(stage_in(ctx, keys, n, &in));
  Output<float> ov, oa;
  Output<uint8_t> oh;
  CK(stage_out(ctx, val_out, n * ctx->s.D, &ov));
  CK(stage_out(ctx, acc_out, n * ctx->s.D, &oa));
  CK(stage_out(ctx, has_out, n, &oh));
  launch_replica_rows(ctx->s, worker, in.dev, n, ov.dev, oa.dev, oh.dev, ctx->stream);
  CK(finish_out(ctx, &ov));
  CK(finish_out(ctx, &oa));
  CK(finish_out(ctx, &oh));
  pool_free(ctx, in.owned);
  CK(cudaStreamSynchronize(ctx->stream));
  return check_launch(ctx, "replica_rows");
}

adapm_status adapm_refcounts(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys, uint64_t n,
                             uint32_t* out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (worker >= ctx->s.W || n > kMaxN || (n > 0 && (!keys || !out)))
    return fail(ctx, ADAPM_EINVAL, "bad arguments");
  if (n == 0) return ADAPM_OK;
  st = early_undo(ctx, worker);   // the counts as of the worker's clock
  if (st != ADAPM_OK) return st;
  Input<uint32_t> in;
  CK(stage_in(ctx, keys, n, &in));
  Output<uint32_t> o;
  CK(stage_out(ctx, out, n, &o));
  launch_refcounts(ctx->s, worker, in.dev, n, o.dev, ctx->stream);
  CK(finish_out(ctx, &o));
  pool_free(ctx, in.owned);
  CK(cudaStreamSynchronize(ctx->stream));
  return check_launch(ctx, "refcounts");
}

adapm_status adapm_owners(adapm_ctx* ctx, const uint32_t* keys, uint64_t n, int32_t* out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (n > kMaxN || (n > 0 && (!keys || !out))) return fail(ctx, ADAPM_EINVAL, "bad arguments");
  if (n == 0) return ADAPM_OK;
  Input<uint32_t> in;
  CK(stage_in(ctx, keys, n, &in));
  Output<int32_t> o;
  CK(stage_out(ctx, out, n, &o));
  launch_owners(ctx->s, in.dev, n, o.dev, ctx->stream);
  CK(finish_out(ctx, &o));
  pool_free(ctx, in.owned);
  CK(cudaStreamSynchronize(ctx->stream));
  return check_launch(ctx, "owners");
}

adapm_status adapm_read_main(adapm_ctx* ctx, const uint32_t* keys, uint64_t n, float* out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (n > kMaxN || (n > 0 && (!keys || !out))) return fail(ctx, ADAPM_EINVAL, "bad arguments");
  if (n == 0) return ADAPM_OK;
  Input<uint32_t> in;
  CK(stage_in(ctx, keys, n, &in));
  Output<float> o;
  CK(stage_out(ctx, out, n * ctx->s.D, &o));
  launch_pull(ctx->s, -1, in.dev, n, o.dev, ctx->sms, ctx->stream);
  CK(finish_out(ctx, &o));
  pool_free(ctx, in.owned);
  CK(cudaStreamSynchronize(ctx->stream));
  return check_launch(ctx, "read_main");
}

adapm_status adapm_get_stats(adapm_ctx* ctx, adapm_stats* out) {
  adapm_status st = check_ctx(ctx);
  if (st != ADAPM_OK) return st;
  if (!out) return fail(ctx, ADAPM_EINVAL, "null output");
  DevState h{};
  CK(cudaMemcpyAsync(&h, ctx->dstate, sizeof h, cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  out->live_replicas = (uint64_t)(h.live > 0 ? h.live : 0);
  out->high_water = (uint64_t)h.high_water;
  out->capacity = ctx->s.S;
  out->created = h.created;
  out->destroyed = h.destroyed;
  out->last_push_unique = h.last_unique;
  out->push_rows = ctx->push_rows_host;
  out->push_unique = h.push_unique;
  out->sync_keys = h.sync_keys;
  out->sync_replicas = h.sync_replicas;
  out->relocations = h.relocations;
  out->sync_refreshed = h.sync_refreshed;
  out->planned_pushes = ctx->planned_pushes;
  out->plan_misses = h.plan_misses;
  out->early_advances = ctx->early_advances;
  out->early_undone = ctx->early_undone;
  return ADAPM_OK;
}

adapm_status adapm_profile_enable(adapm_ctx* ctx, int enable) {
  if (!ctx) return ADAPM_EINVAL;
  ctx->prof = enable != 0;
  return ADAPM_OK;
}

adapm_status adapm_profile_read(adapm_ctx* ctx, double* ms_out, uint64_t* calls_out) {
  if (!ctx) return ADAPM_EINVAL;
  cudaSetDevice(ctx->device);
  CK(cudaStreamSynchronize(ctx->stream));
  for (auto& t : ctx->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, std::get<1>(t), std::get<2>(t)) == cudaSuccess) {
      ctx->prof_ms[std::get<0>(t)] += ms;
      ctx->prof_calls[std::get<0>(t)] += 1;
    }
    ctx->spare_events.push_back(std::get<1>(t));
    ctx->spare_events.push_back(std::get<2>(t));
  }
  ctx->pending.clear();
  cudaGetLastError();
  for (int i = 0; i < ADAPM_NUM_OPS; ++i) {
    if (ms_out) ms_out[i] = ctx->prof_ms[i];
    if (calls_out) calls_out[i] = ctx->prof_calls[i];
    ctx->prof_ms[i] = 0;
    ctx->prof_calls[i] = 0;
  }
  return ADAPM_OK;
}

adapm_status adapm_kernel_launches(uint64_t* out) {
  if (!out) return ADAPM_EINVAL;
  *out = g_launches.load(std::memory_order_relaxed);
  return ADAPM_OK;
}

const char* adapm_last_error(adapm_ctx* ctx) {
  if (!ctx) return "null context";
  return ctx->err.c_str();
}

}  // extern "C"
