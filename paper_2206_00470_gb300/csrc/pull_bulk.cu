// pull with shared-memory staging by the bulk-copy engine (Sec. 5.1 reads:
// out[i] = worker w's replica of keys[i], else the main copy).
//
// A block takes tiles of T consecutive output rows.  For each row one thread
// resolves key -> slot -> source row and starts a 1-D cp.async.bulk of the
// row (D * 4 bytes, 16-byte aligned) from global into the tile's shared
// memory, completing on the stage's mbarrier (transaction bytes); when the
// tile has landed, one thread writes it to out with a single bulk copy of
// T * D * 4 contiguous bytes.  Two stages: the loads of tile t+1 are in
// flight while tile t is stored.  Rows move without passing through
// registers, and the output leaves as one large bulk store per tile.
//
// Every wait is bounded: an mbarrier wait that gives up sets ERR_TIMEOUT
// (the context is then retired by adapm_wait), waits (bounded) for the
// block's own copies and returns.  A key >= K sets ERR_KEY_RANGE and its row
// is zero, as in the register gather.
#include "internal.cuh"
#include "rowgroup.cuh"
#include "store_launch.cuh"

namespace adapm {

namespace {

constexpr int kBulkThreads = 128;
constexpr uint32_t kStageBytes = 32768;      // bytes of rows per stage
constexpr uint32_t kWaitLimit = 1u << 22;    // polls of one mbarrier wait

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

// true once the phase with the given parity has completed; bounded
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    uint32_t done;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

__device__ __forceinline__ void bulk_load(void* dst_smem, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst_smem)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void bulk_store(void* dst, const void* src_smem, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src_smem)),
               "r"(bytes)
               : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// the block's bulk stores have finished reading shared memory
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and have completed
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__global__ void __launch_bounds__(kBulkThreads) pull_bulk_kernel(Store s, int w, const uint32_t* __restrict__ keys,
                                                                uint64_t n, float* __restrict__ out, uint32_t T) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t bar[2];
  __shared__ int s_abort;
  const uint32_t rowb = s.D * 4u;
  const size_t stage_bytes = (size_t)T * rowb;
  const int32_t* mapw = w >= 0 ? s.map + (uint64_t)w * s.K : nullptr;
  const uint64_t ntiles = (n + T - 1) / T;
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    s_abort = 0;
    // the initialised barriers visible to the bulk-copy engine before any copy names them
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  fence_proxy_async();
  __syncthreads();
  bool bad = false;
  // the rows of tile t go to stage b: thread i < T starts row i's copy, or
  // zero-fills it for a key out of range; thread 0 arrives with the bytes
  // that will land
  auto issue = [&](uint64_t t, int b) {
    const uint64_t r0 = t * T;
    const uint32_t rows = (uint32_t)(n - r0 < T ? n - r0 : T);
    const uint32_t i = threadIdx.x;
    unsigned char* dst = smem + (size_t)b * stage_bytes + (size_t)i * rowb;
    uint32_t nbad = 0;
    if (i < rows) {
      const uint32_t k = __ldg(keys + r0 + i);
      if (k < s.K) {
        const int32_t sl = mapw != nullptr ? __ldg(mapw + k) : -1;
        const float* src = sl >= 0 ? s.val + (uint64_t)sl * s.D : s.main + (uint64_t)k * s.D;
        bulk_load(dst, src, rowb, &bar[b]);
      } else {
        bad = true;
        nbad = 1;
        for (uint32_t c = 0; c < rowb; c += 16) *reinterpret_cast<float4*>(dst + c) = f4zero();
      }
    }
    // rows whose copy started: all but the zero-filled ones
    const uint32_t landed = rows - __syncthreads_count(nbad);
    if (threadIdx.x == 0) mbar_arrive_expect_tx(&bar[b], landed * rowb);
  };
  uint32_t use[2] = {0, 0};   // completed phases per stage
  uint64_t t = blockIdx.x;
  if (t < ntiles) issue(t, 0);
  int b = 0;
  for (; t < ntiles; t += gridDim.x) {
    const uint64_t tn = t + gridDim.x;
    if (tn < ntiles) {
      // stage b^1 is free once the store of the tile before has read it
      if (threadIdx.x == 0) bulk_wait_read();
      __syncthreads();
      issue(tn, b ^ 1);
    }
    if (threadIdx.x == 0 && !mbar_wait(&bar[b], use[b] & 1u)) s_abort = 1;
    use[b] += 1;
    fence_proxy_async();   // zero-filled rows (generic writes) before the bulk store reads them
    __syncthreads();
    if (s_abort) break;
    if (threadIdx.x == 0) {
      const uint64_t r0 = t * T;
      const uint32_t rows = (uint32_t)(n - r0 < T ? n - r0 : T);
      bulk_store(out + r0 * s.D, smem + (size_t)b * stage_bytes, rows * rowb);
    }
    b ^= 1;
  }
  if (s_abort) {
    // a copy that never landed: report, and give the others a bounded wait
    if (threadIdx.x == 0) {
      set_error(s.st, ERR_TIMEOUT);
      mbar_wait(&bar[b ^ 1], use[b ^ 1] & 1u);
    }
  }
  if (threadIdx.x == 0) bulk_wait_all();
  if (__any_sync(0xFFFFFFFFu, bad) && (threadIdx.x & 31) == 0) set_error(s.st, ERR_KEY_RANGE);
}

}  // namespace

bool pull_bulk_fits(uint32_t D, const void* out) {
  return (reinterpret_cast<uintptr_t>(out) & 15u) == 0 && D * 4u <= kStageBytes;
}

void launch_pull_bulk(const Store& s, int w, const uint32_t* keys, uint64_t n, float* out, int sms,
                      cudaStream_t stream) {
  if (n == 0) return;
  const uint32_t rowb = s.D * 4u;
  uint32_t T = kStageBytes / rowb;
  if (T > kBulkThreads) T = kBulkThreads;
  const size_t smem = 2 * (size_t)T * rowb;
  // the shared-memory limit of the kernel is a per-device attribute
  static bool attr_set[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64 || !attr_set[dev]) {
    cudaFuncSetAttribute(pull_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 2 * (int)kStageBytes);
    if (dev >= 0 && dev < 64) attr_set[dev] = true;
  }
  const uint64_t ntiles = (n + T - 1) / T;
  uint64_t grid = (uint64_t)sms * 3;   // three 64 KB blocks per SM
  if (grid > ntiles) grid = ntiles;
  note_launches(1);
  pull_bulk_kernel<<<(unsigned)grid, kBulkThreads, smem, stream>>>(s, w, keys, n, out, T);
}

}  // namespace adapm
