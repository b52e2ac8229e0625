// adapm_push_noalloc: the push of adapm_push for callers that cannot let the
// library allocate device memory during a call.
//
// adapm_push takes its sort buffers and partial-sum buffers from a
// stream-ordered memory pool on every call.  Some callers cannot allow that:
// a framework whose own allocator owns the device memory budget (an
// allocation behind its back can fail or fragment it), or a latency-critical
// serving loop in which cudaMalloc / cudaFree may synchronise the device.
// This variant allocates nothing: its scratch is one file-scope device array
// of kScratchBytes, which every GPU that loads this library holds until the
// process exits.  The caller passes device arrays only; host arrays would
// need staging buffers and are rejected.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "adapm.h"
#include "internal.cuh"
#include "store_launch.cuh"

namespace {

constexpr size_t kScratchBytes = 16u << 20;    // 16 MiB per GPU
constexpr size_t kAlign = 256;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_push_scratch[kScratchBytes];

// Device address of g_push_scratch per device.  In host code the symbol is
// only a host-side stand-in, so the address is looked up once per device,
// with that device current, on the first call made on it.
std::mutex g_mu;
unsigned char* g_scratch_addr[kMaxDevices] = {nullptr};

cudaError_t scratch_for(int device, unsigned char** out) {
  if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_push_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[device] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_addr[device];
  return cudaSuccess;
}

size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// Byte offsets of the scratch regions of one push of n rows.
struct Layout {
  size_t ka, kb, va, vb, hist, sparts, total;
  uint64_t chunk, nchunks;
};

Layout layout(uint32_t D, uint64_t n, int sms) {
  Layout L{};
  L.chunk = adapm::push_chunk_rows(D, n, sms);
  L.nchunks = (n + L.chunk - 1) / L.chunk;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off += round_up(bytes);
    return at;
  };
  L.ka = take(n * 4);
  L.kb = take(n * 4);
  L.va = take(n * 4);
  L.vb = take(n * 4);
  L.hist = take(adapm::sort_scratch_words(n) * 4);
  L.sparts = take(adapm::push_span_part_rows(L.nchunks) * D * 4);
  L.total = off;
  return L;
}

// Profiling of one noalloc push: the same operations as adapm_push (3: the
// whole push, 6: the scatter kernels), stopped on every path out.
struct ProfGuard {
  adapm_ctx* ctx;
  adapm::ProfToken t;
  ProfGuard(adapm_ctx* c, int op) : ctx(c) { t = adapm::ctx_prof_start(ctx, op); }
  ~ProfGuard() { adapm::ctx_prof_stop(ctx, t); }
};

}  // namespace

extern "C" adapm_status adapm_push_noalloc(adapm_ctx* ctx, uint32_t worker, const uint32_t* keys,
                                           uint64_t n, const float* deltas) {
  using namespace adapm;
  // a live context, its last error cleared, its device current
  const adapm_status st = static_cast<adapm_status>(ctx_begin(ctx));
  if (st != ADAPM_OK) return st;
  CtxView v;
  if (!ctx_view(ctx, &v)) return ADAPM_EINVAL;
  if (worker >= v.s.W) {
    ctx_set_error(ctx, "worker out of range");
    return ADAPM_EINVAL;
  }
  if (n == 0) return ADAPM_OK;
  if (!keys || !deltas || n > (1ull << 31)) {
    ctx_set_error(ctx, "bad pointers/n");
    return ADAPM_EINVAL;
  }
  if (!is_device_ptr(keys) || !is_device_ptr(deltas)) {
    ctx_set_error(ctx, "adapm_push_noalloc takes device arrays only");
    return ADAPM_EINVAL;
  }
  if (reinterpret_cast<uintptr_t>(deltas) % 16 != 0) {
    ctx_set_error(ctx, "adapm_push_noalloc needs 16-byte aligned delta rows");
    return ADAPM_EINVAL;
  }
  const Layout L = layout(v.s.D, n, v.sms);
  if (L.total > kScratchBytes) {
    char msg[160];
    snprintf(msg, sizeof msg,
             "push of %llu rows x %u floats needs %zu bytes of scratch; adapm_push_noalloc has %zu",
             (unsigned long long)n, v.s.D, L.total, kScratchBytes);
    ctx_set_error(ctx, msg);
    return ADAPM_EINVAL;
  }
  unsigned char* base = nullptr;
  cudaError_t e = scratch_for(v.device, &base);
  if (e != cudaSuccess) return static_cast<adapm_status>(ctx_fail_cuda(ctx, e, "cudaGetSymbolAddress"));
  auto at = [&](size_t off) { return reinterpret_cast<uint32_t*>(base + off); };
  ProfGuard whole(ctx, 3);
  uint32_t *sk = nullptr, *sp = nullptr;
  // the array keeps the previous call's contents: every scratch word is
  // written before it is read, except the distinct-key counter, which the
  // sort clears
  e = sort_keys(keys, n, v.s.K, false, v.bits, at(L.ka), at(L.kb), at(L.va), at(L.vb), at(L.hist), v.sms,
                v.dstate, v.bar_base, &v.dstate->last_unique, nullptr, v.stream, &sk, &sp);
  if (e != cudaSuccess) return static_cast<adapm_status>(ctx_fail_cuda(ctx, e, "push_noalloc sort"));
  ctx_add_push_rows(ctx, n);
  PushArgs a{sk,
             sp,
             n,
             deltas,
             L.chunk,
             L.nchunks,
             worker,
             reinterpret_cast<float*>(base + L.sparts)};
  {
    ProfGuard scatter(ctx, 6);
    launch_push(v.s, a, v.sms, v.stream);
  }
  e = ctx_launch_error(ctx);
  if (e != cudaSuccess) return static_cast<adapm_status>(ctx_fail_cuda(ctx, e, "push_noalloc scatter"));
  return ADAPM_OK;
}
