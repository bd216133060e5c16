// Internal helpers shared by the PACE CUDA translation units (sm_103a only).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "pace.h"

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ < 1000)
#error "PACE kernels target sm_103a (Blackwell datacenter) only"
#endif

namespace pace {

// ---------------------------------------------------------------- host side

#define PACE_TRY_CUDA(expr)                         \
  do {                                              \
    cudaError_t pace_e_ = (expr);                   \
    if (pace_e_ != cudaSuccess) return PACE_ERR_CUDA; \
  } while (0)

#define PACE_TRY(expr)                \
  do {                                \
    pace_status pace_s_ = (expr);     \
    if (pace_s_ != PACE_OK) return pace_s_; \
  } while (0)

// Kernels launched by this library from the calling thread.
uint64_t& launch_counter();

// Vocabulary splits the LM head should use on large batches (0 = automatic),
// set by pace_set_lmhead_splits for the whole process.
std::atomic<int>& lmhead_split_pref();

// Called right after every kernel launch: counts it and checks it started.
inline pace_status last_launch_status() {
  ++launch_counter();
  return cudaGetLastError() == cudaSuccess ? PACE_OK : PACE_ERR_CUDA;
}

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

// Carves 256-byte-aligned sub-buffers out of the caller's workspace.  The
// same sequence of take() calls with size-only bookkeeping gives the size
// query, so the two can never disagree.
struct Carver {
  char* base;
  size_t cap;
  size_t used;
  explicit Carver(void* b = nullptr, size_t c = 0) : base(static_cast<char*>(b)), cap(c), used(0) {}
  template <typename T>
  T* take(size_t count) {
    size_t off = align_up(used, 256);
    used = off + count * sizeof(T);
    return base ? reinterpret_cast<T*>(base + off) : nullptr;
  }
  bool fits() const { return used <= cap; }
};

inline bool aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

// Number of SMs of the current device (cached per device).
int sm_count();

// Events set by pace_set_profile_events for this host thread (null = off).
struct ProfileEvents {
  cudaEvent_t begin = nullptr;
  cudaEvent_t end = nullptr;
};
ProfileEvents& profile_events(int kernel);

// -------------------------------------------------------------- device side

// First device-side error wins; later ones are dropped.
__device__ __forceinline__ void report(int32_t* status, int32_t code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded waits give up after this long and report PACE_ERR_TIMEOUT.
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---- mbarrier

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with the given parity to complete, for at most
// kWaitLimitNs.  Returns false on timeout (the caller reports and unwinds),
// and also when *abort is set by another thread of the block.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort,
                                                  uint64_t limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (abort && *abort) return false;
      if (global_timer_ns() - t0 > limit_ns) return false;
    }
  }
}

// ---- thread-block clusters

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Full cluster barrier (every thread of every CTA of the cluster).
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

// Shared::cluster address of the same shared-memory offset in CTA `rank` of
// this cluster (rank = this CTA's own rank gives its own window address).
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}

// Arrive once on an mbarrier of any CTA of the cluster (release at cluster scope).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_caddr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_caddr)
               : "memory");
}

// Arrive on the mbarrier at cluster address bar_caddr (this CTA's or a peer's)
// and raise its expected transaction bytes by `bytes`, in one step.
__device__ __forceinline__ void mbar_arrive_expect_tx_cluster(uint32_t bar_caddr, uint32_t bytes) {
  asm volatile(
      "mbarrier.arrive.expect_tx.shared::cluster.b64 _, [%0], %1;" ::"r"(bar_caddr),
      "r"(bytes)
      : "memory");
}

__device__ __forceinline__ void st_cluster_u32(uint32_t caddr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(caddr), "r"(v) : "memory");
}

// Phase test with acquire at cluster scope, for barriers that threads of the
// other CTA arrive on.
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_bounded_cluster(uint64_t* bar, uint32_t parity,
                                                          volatile int* abort) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (abort && *abort) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) return false;
    }
  }
}

// ---- pacing of persistent clusters

// Longest a cluster waits at a round boundary for the others (a soft barrier:
// it proceeds after this even if some cluster is late, so it can never hang).
constexpr uint64_t kRoundWaitNs = 250000;  // 250 us

// Persistent clusters that take items c, c + n_clusters, ... share the operand
// tiles of a round through L2 only while they stay in step.  Before its k-th
// item a cluster waits until the counter (items whose loads were issued,
// zeroed before the launch, incremented once per item by each cluster) reaches
// k * n_clusters, for at most kRoundWaitNs.  A timing signal only: no data is
// passed through the counter.
__device__ __forceinline__ void wait_round(const unsigned* ctr, unsigned target) {
  const uint64_t t0 = global_timer_ns();
  for (;;) {
    if (*reinterpret_cast<const volatile unsigned*>(ctr) >= target) return;
    if (global_timer_ns() - t0 > kRoundWaitNs) return;
    __nanosleep(128);
  }
}

// ---- TMA (bulk tensor copies, global -> shared)

__device__ __forceinline__ void tma_prefetch_desc(const void* desc) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(desc)) : "memory");
}

// One box into this CTA's shared memory; its transaction bytes complete on the
// mbarrier at shared::cluster address bar_caddr, which may belong to either CTA
// of this CTA's pair (both CTAs of a pair feed the even CTA's barrier).
__device__ __forceinline__ void tma_load_2d_pair(void* smem_dst, const void* desc,
                                                 uint32_t bar_caddr, int32_t x, int32_t y,
                                                 uint64_t cache_hint) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(desc)), "r"(bar_caddr), "r"(x), "r"(y), "l"(cache_hint)
      : "memory");
}

// Four whole rows (r0..r3) of a 2-D tensor map whose box is one row high,
// starting at column x, into this CTA's shared memory at smem_dst, one row
// after the other; the transaction bytes (4 box rows) complete on the mbarrier
// at cluster address bar_caddr, as tma_load_2d_pair's do.  With the 128-byte
// swizzle, each row's 16-byte chunks land at the positions their shared-memory
// address selects, so four gathers into consecutive 512-byte slices build the
// same tile as one box of 4 n rows.
__device__ __forceinline__ void tma_gather4_pair(void* smem_dst, const void* desc,
                                                 uint32_t bar_caddr, int32_t x, int32_t r0,
                                                 int32_t r1, int32_t r2, int32_t r3,
                                                 uint64_t cache_hint) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      ".cta_group::2.L2::cache_hint [%0], [%1, {%3, %4, %5, %6, %7}], [%2], %8;" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(desc)), "r"(bar_caddr), "r"(x), "r"(r0), "r"(r1), "r"(r2),
      "r"(r3), "l"(cache_hint)
      : "memory");
}

// ---- tcgen05 on CTA pairs (5th-generation tensor cores, accumulators in
// tensor memory).  Every tcgen05 instruction of a kernel names the same CTA
// group; the kernels here all run on pairs (cta_group::2): one MMA of
// M = 256 takes A rows 0-127 and the first half of the B tile from the even
// CTA's shared memory, A rows 128-255 and the second half of B from the odd
// CTA's, at the same offsets, and writes each CTA's 128 rows of D into that
// CTA's tensor memory.

// Allocation and release are collective: one warp of each CTA of the pair.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* smem_dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(smem_dst)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs here), issued by one
// thread of the even CTA for the pair.
__device__ __forceinline__ void tc_mma_f16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier at shared::cluster address bar_caddr (in either
// CTA of the pair) when every tcgen05 op this thread issued so far is done.
__device__ __forceinline__ void tc_commit_pair(uint32_t bar_caddr) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          bar_caddr)
      : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp gets lane
// (base lane + i), columns [col, col + 32).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major bf16 tile whose rows are 128
// bytes (64 elements) with the 128-byte swizzle: 8-row core groups 1024 bytes
// apart (stride byte offset), leading byte offset unused for this layout,
// descriptor version 1, swizzle mode 2 (128B).  `saddr` is the shared-space
// address of the first element of the K slice (must lie in a 1024-aligned
// tile; advancing K by 16 elements adds 32 bytes).
__device__ __forceinline__ uint64_t smem_desc_k128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);   // start address
  d |= static_cast<uint64_t>(1u) << 16;                   // leading byte offset (unused)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;           // stride byte offset
  d |= static_cast<uint64_t>(1u) << 46;                   // descriptor version
  d |= static_cast<uint64_t>(2u) << 61;                   // 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: bf16 A and B, fp32 D, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(uint32_t m, uint32_t n) {
  return (1u << 4)            // D format: f32
         | (1u << 7)          // A format: bf16
         | (1u << 10)         // B format: bf16
         | ((n >> 3) << 17)   // N / 8
         | ((m >> 4) << 24);  // M / 16
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

}  // namespace pace
