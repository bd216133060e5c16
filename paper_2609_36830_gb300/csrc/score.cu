// Pool scoring: Lemma 1 / Eq. 2 staleness decomposition, Eqs. 7-10 scores and
// the per-group mean, on sm_103a.
//
//   tag_reduce_kernel   one streaming pass over the int32 version tags (HBM
//                       bound): per trajectory the count T of policy tokens,
//                       the exact integer sum of their tags and the largest
//                       tag (+1, for the Lemma 1 premise check).
//                       On pools of 8k trajectories and more the same launch
//                       also prepares the prefix-score window (extra blocks
//                       after the streaming ones, run in its tail): one sorts W,
//                       the others tabulate F = phi(count / |W|) (Eqs. 9-10)
//                       for every possible count 0..|W| (F depends on s only
//                       through the count).
//   score_finalize_kernel  one thread per trajectory: K_gen, K_wait, the ECDF
//                       count of s against the window (binary search in the
//                       sorted window, or a direct count on small pools), F
//                       (from the table, or computed), the mode's score
//                       (Eqs. 7-8), and the mean of each group of G in fixed
//                       left-to-right order.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "pace_internal.cuh"

namespace pace {
namespace {

constexpr int kReduceThreads = 256;  // 8 warps
constexpr int kTileTokens = 128;     // one int4 per lane
// Tiles per warp batch (128 tokens each) and resident blocks per SM, by pool
// size.  Large pools: 8 tiles (1024 tokens, 4 KB in flight per register set),
// 126 registers, 2 blocks per SM.  Pools of up to kSmallPoolTokens tags: 4
// tiles, 79 registers, 3 blocks per SM; more warps with half the work each
// shorten the ramp and the tail where those dominate (16k sweep pool, 55 M
// tags: 62 -> 52 us), and cost ~0.5 % on long streams (128k and 1M pools).
constexpr int kTilesLarge = 8, kBlocksLarge = 2;
constexpr int kTilesSmall = 4, kBlocksSmall = 3;
constexpr int64_t kSmallPoolTokens = int64_t(1) << 27;
// Short streams get fewer warps rather than fewer batches a warp: below this
// many batches a warp, trajectories spread over several warps' ranges and their
// totals need more head slots.  On the 1k sweep pool (3.6 M tags, ~3,500 a
// trajectory) whole calls took 30.3 / 29.0 / 27.2 / 28.6 / 31.3 us with at
// least 1 / 2 / 4 / 8 / 16 batches a warp (the stream itself 12.3 -> 18.3 us);
// pools from ~15 M tags keep one full wave and are not affected.
constexpr int64_t kMinBatchesPerWarp = 4;
constexpr int kMaxWindow = 4096;
// Pools of at least this many trajectories finalise inside the tag reduction's
// launch (pace_set_score_fused_min_traj); smaller ones use a launch of their own.
constexpr int64_t kFusedMinTrajDefault = int64_t(1) << 18;

std::atomic<int64_t>& fused_min_traj() {
  static std::atomic<int64_t> v{kFusedMinTrajDefault};
  return v;
}

// Whether the current device takes cooperative launches (cached per device);
// where it does not, every pool finalises in a launch of its own.
bool cooperative_launch_ok() {
  constexpr int kMaxDevices = 64;
  static std::atomic<int> cache[kMaxDevices];  // 0 unknown, 1 yes, 2 no
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  int c = cache[dev].load();
  if (c == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess) {
      (void)cudaGetLastError();
      v = 0;
    }
    c = v ? 1 : 2;
    cache[dev].store(c);
  }
  return c == 1;
}
constexpr int64_t kTableMinTraj = 8192;  // pools from this size sort W and tabulate F

__device__ __forceinline__ int4 ld_stream_v4(const int32_t* p) {
  int4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.s32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

constexpr int64_t kPrefetchAhead = 4;

// Bulk prefetch of a 16-byte-aligned range into L2 (no data returned).
__device__ __forceinline__ void l2_prefetch_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(p)),
               "r"(bytes)
               : "memory");
}

// ---- exact integer quotients without the fp64 pipe
//
// GB300's fp64 pipe is narrow, and the finalisation is bound by it (one int64
// to double conversion and one correctly rounded division per trajectory).  The
// functions below build the same doubles from integer arithmetic: the result
// of __ddiv_rn(__ll2double_rn(S), T) for 64-bit S and 32-bit T > 0, and of
// __ll2double_rn(x), bit for bit.

// (double)x rounded to nearest even, from its bits (every int64 is in range).
__device__ __forceinline__ double i64_to_double_rn(long long x) {
  if (x == 0) return 0.0;
  const unsigned long long sign = x < 0 ? (1ull << 63) : 0ull;
  unsigned long long a = x < 0 ? 0ull - static_cast<unsigned long long>(x)
                               : static_cast<unsigned long long>(x);
  int top = 63 - __clzll(static_cast<long long>(a));  // leading bit position
  unsigned long long mant;
  if (top <= 52) {
    mant = a << (52 - top);
  } else {
    const int sh = top - 52;  // bits dropped, 1..11
    mant = a >> sh;
    const unsigned long long rem = a & ((1ull << sh) - 1);
    const unsigned long long half = 1ull << (sh - 1);
    if (rem > half || (rem == half && (mant & 1ull))) ++mant;
    if (mant >> 53) {  // carried into a new bit: 2^53 -> 2^52 one binade up
      mant >>= 1;
      ++top;
    }
  }
  const unsigned long long bits = sign | (static_cast<unsigned long long>(top + 1023) << 52) |
                                  (mant & ((1ull << 52) - 1));
  return __longlong_as_double(static_cast<long long>(bits));
}

// RN(RN53(S) / T): exactly __ddiv_rn(__ll2double_rn(S), (double)T), T >= 1.
// |S| is first rounded to 53 significant bits (a * 2^e, a < 2^53) as the
// conversion does; then q = a / T, r = a % T and the fraction r / T is
// developed in 32-bit digits by integer division, giving a 64-bit quotient
// with its leading bit set plus a sticky bit, which is rounded to 53 bits
// (nearest, ties to even).  The quotient lies in [2^-32, 2^63], always normal.
__device__ __forceinline__ double i64_div_u32_rn(long long S, unsigned T) {
  if (S == 0) return 0.0;
  const unsigned long long sign = S < 0 ? (1ull << 63) : 0ull;
  unsigned long long a = S < 0 ? 0ull - static_cast<unsigned long long>(S)
                               : static_cast<unsigned long long>(S);
  int e = 0;  // the dividend is a * 2^e
  {
    const int top = 63 - __clzll(static_cast<long long>(a));
    if (top > 52) {
      const int sh = top - 52;
      unsigned long long m = a >> sh;
      const unsigned long long rem = a & ((1ull << sh) - 1);
      const unsigned long long half = 1ull << (sh - 1);
      if (rem > half || (rem == half && (m & 1ull))) ++m;
      e = sh;
      if (m >> 53) {  // 2^53 = 2^52 * 2: keep a below 2^53
        m >>= 1;
        ++e;
      }
      a = m;
    }
  }
  const unsigned long long t = T;
  const unsigned long long q = a / t;
  const unsigned long long r = a - q * t;
  // fraction digits of r / T (r < T < 2^32, so each digit fits 32 bits)
  const unsigned long long n1 = r << 32;
  const unsigned long long d1 = n1 / t;
  const unsigned long long r1 = n1 - d1 * t;
  const unsigned long long n2 = r1 << 32;
  const unsigned long long d2 = n2 / t;
  const unsigned long long r2 = n2 - d2 * t;
  const unsigned long long frac = (d1 << 32) | d2;  // r / T = frac * 2^-64 + ...
  unsigned long long x;  // 64 significant bits, leading bit at 63
  bool sticky;
  int exp2;              // exponent of the leading bit
  if (q != 0) {
    const int lq = 64 - __clzll(static_cast<long long>(q));  // bits of q, 1..53
    const int f = 64 - lq;                                   // fraction bits kept, 11..63
    x = (q << f) | (frac >> lq);
    sticky = r2 != 0 || (frac & ((1ull << lq) - 1)) != 0;
    exp2 = lq - 1 + e;
  } else {
    // r / T >= 2^-32: frac has at most 31 leading zeros; a third digit refills them
    const unsigned long long n3 = r2 << 32;
    const unsigned long long d3 = n3 / t;
    const unsigned long long r3 = n3 - d3 * t;
    const int lz = __clzll(static_cast<long long>(frac));  // 0..31
    x = lz ? (frac << lz) | (d3 >> (32 - lz)) : frac;
    sticky = r3 != 0 || (lz ? ((d3 << (32 + lz)) != 0) : (d3 != 0));
    exp2 = -1 - lz + e;
  }
  unsigned long long mant = x >> 11;  // 53 bits
  const bool round_bit = (x >> 10) & 1ull;
  const bool rest = sticky || (x & 0x3FFull) != 0;
  if (round_bit && (rest || (mant & 1ull))) ++mant;
  if (mant >> 53) {
    mant >>= 1;
    ++exp2;
  }
  const unsigned long long bits = sign | (static_cast<unsigned long long>(exp2 + 1023) << 52) |
                                  (mant & ((1ull << 52) - 1));
  return __longlong_as_double(static_cast<long long>(bits));
}

struct LaneAcc {
  long long sum;   // sum of policy tags seen by this lane for the current trajectory
  unsigned cnt;    // number of policy tokens
  unsigned maxp1;  // max over policy tokens of (unsigned)v + 1 (0 if none)
};

__device__ __forceinline__ void acc_elem(LaneAcc& a, int32_t v, bool in_range) {
  const bool in = in_range && (v != -1);
  a.sum += in ? static_cast<long long>(v) : 0ll;
  a.cnt += in ? 1u : 0u;
  const unsigned vp1 = static_cast<unsigned>(v) + 1u;
  a.maxp1 = (in && vp1 > a.maxp1) ? vp1 : a.maxp1;
}

// The stream's per-trajectory totals, written without atomics (so nothing has
// to be zeroed before a call).  The warp holding a trajectory's first token
// writes its slot with one 16-byte store: x = the sum of its part's policy tags
// with bit 63 set when the trajectory continues past that warp's range (the sum
// of valid tags is below 2^63), y = count | (max tag + 1) << 32.  Every warp
// writes one head slot: its part of the trajectory that began before its range
// (traj = -1 if none).  A continuing trajectory's totals are its slot plus the
// head slots of the following warps up to the one holding its last token.
constexpr unsigned long long kContinues = 1ull << 63;

struct HeadSlot {
  long long traj;
  unsigned long long sum;
  unsigned cnt, maxp1;
  long long pad;
};

struct TagTotals {
  ulonglong2* slot;  // [n_traj]
  HeadSlot* head;    // [stream warps]
};

// Geometry of one tag-reduction launch: warp w streams batches
// [n_batches w / n_warps, n_batches (w + 1) / n_warps).
struct StreamGeom {
  int64_t batch_tokens;
  int64_t n_batches;
  int64_t n_warps;
};

// The last warp whose range starts at or before batch b (the one that streams it).
__host__ __device__ __forceinline__ int64_t warp_of_batch(const StreamGeom& g, int64_t b) {
  return ((b + 1) * g.n_warps - 1) / g.n_batches;
}

// Warp-reduce the lane partials and write them: the head slot of this warp, or
// trajectory traj's slot.  Integer adds and max are order-independent, so the
// totals are exact and deterministic however trajectories are split.
__device__ __forceinline__ void emit(LaneAcc& a, int64_t traj, bool continues, bool head,
                                     int64_t warp, const TagTotals& tt) {
  const unsigned full = 0xffffffffu;
  long long s = a.sum;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(full, s, o);
  const unsigned c = __reduce_add_sync(full, a.cnt);
  const unsigned m = __reduce_max_sync(full, a.maxp1);
  if ((threadIdx.x & 31) == 0) {
    if (head) {
      HeadSlot h;
      h.traj = traj;
      h.sum = static_cast<unsigned long long>(s);
      h.cnt = c;
      h.maxp1 = m;
      h.pad = 0;
      tt.head[warp] = h;
    } else {
      ulonglong2 v;
      v.x = static_cast<unsigned long long>(s) | (continues ? kContinues : 0ull);
      v.y = static_cast<unsigned long long>(c) | (static_cast<unsigned long long>(m) << 32);
      tt.slot[traj] = v;
    }
  }
  a.sum = 0;
  a.cnt = 0;
  a.maxp1 = 0;
}

// Trajectory i's totals (T, the exact sum of its policy tags, the largest tag
// + 1) from its slot v and the head slots, given its offsets o0, o1.  Empty (or
// inconsistent) ranges have zero totals (their slot, loaded regardless so that
// the load need not wait for the offsets, is not used).  The head slots of a continuing
// trajectory are loaded two at a time before either is used.  L2 loads: other
// blocks of the same launch may have written the slots.
__device__ __forceinline__ void traj_totals(const TagTotals& tt, const StreamGeom& g,
                                            int64_t n_tokens, int64_t i, int64_t o0, int64_t o1,
                                            const ulonglong2& v, long long& sum, unsigned& cnt,
                                            unsigned& maxp1) {
  sum = 0;
  cnt = 0u;
  maxp1 = 0u;
  if (o0 < 0 || o1 <= o0 || o0 >= n_tokens) return;
  sum = static_cast<long long>(v.x & ~kContinues);
  cnt = static_cast<unsigned>(v.y);
  maxp1 = static_cast<unsigned>(v.y >> 32);
  if (v.x & kContinues) {
    const int64_t last = (o1 < n_tokens ? o1 : n_tokens) - 1;
    const int64_t w0 = warp_of_batch(g, o0 / g.batch_tokens);
    const int64_t w1 = warp_of_batch(g, last / g.batch_tokens);
    for (int64_t w = w0 + 1; w <= w1; w += 2) {
      longlong2 h0[2], h1[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (w + u <= w1) {
          const longlong2* hp = reinterpret_cast<const longlong2*>(tt.head + w + u);
          h0[u] = __ldcg(hp);
          h1[u] = __ldcg(hp + 1);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (w + u <= w1 && h0[u].x == i) {
          sum += h0[u].y;
          cnt += static_cast<unsigned>(h1[u].x);
          const unsigned m = static_cast<unsigned>(static_cast<unsigned long long>(h1[u].x) >> 32);
          maxp1 = m > maxp1 ? m : maxp1;
        }
      }
    }
  }
}

// The stream is integer-ALU heavy (a few operations per 4-byte tag), so the
// common cases avoid per-element work: a tag is a policy tag below 2^26 exactly
// when none of its bits 26..31 is set, so one OR over a group of tags decides
// whether the whole group is (no tool tag -1, nothing negative or huge), and
// then up to 32 of them fit a 32-bit sum; 3-input max (DPX) halves the max tree.
__device__ __forceinline__ bool small_policy(int bits_or) {
  return (static_cast<unsigned>(bits_or) >> 26) == 0u;
}

// Sum, count and max of a batch that lies inside one trajectory and holds only
// policy tags below 2^26.  Returns false (and leaves acc untouched) when the
// batch needs the per-group path.
template <int kTilesPerBatch>
__device__ __forceinline__ bool acc_batch_fast(LaneAcc& a, const int4 (&v)[kTilesPerBatch]) {
  int o = 0, mx = 0, s = 0;
#pragma unroll
  for (int u = 0; u < kTilesPerBatch; ++u) {
    o |= (v[u].x | v[u].y) | (v[u].z | v[u].w);
    mx = __vimax3_s32(__vimax3_s32(mx, v[u].x, v[u].y), v[u].z, v[u].w);
    s += (v[u].x + v[u].y) + (v[u].z + v[u].w);
  }
  if (!small_policy(o)) return false;
  a.sum += s;
  a.cnt += 4 * kTilesPerBatch;
  const unsigned mp1 = static_cast<unsigned>(mx) + 1u;
  a.maxp1 = mp1 > a.maxp1 ? mp1 : a.maxp1;
  return true;
}

// The four tags of one lane's int4, all inside the current trajectory.
__device__ __forceinline__ void acc_group(LaneAcc& a, const int4& q) {
  if (small_policy((q.x | q.y) | (q.z | q.w))) {
    a.sum += (q.x + q.y) + (q.z + q.w);
    a.cnt += 4u;
    const unsigned mp1 = static_cast<unsigned>(__vimax3_s32(q.x, q.y, max(q.z, q.w))) + 1u;
    a.maxp1 = mp1 > a.maxp1 ? mp1 : a.maxp1;
  } else {
    acc_elem(a, q.x, true);
    acc_elem(a, q.y, true);
    acc_elem(a, q.z, true);
    acc_elem(a, q.w, true);
  }
}

// Each warp owns a contiguous range of batches (kTilesPerBatch x 128 tokens) of
// the flattened tag stream and walks the CSR offsets forward through it, so trajectories of
// any length mix are balanced across warps.  The walk never leaves
// [0, n_traj) and loads only tags[0, n_tokens), whatever the offsets hold;
// inconsistent offsets are reported by the finalize kernel.
// phi_gamma(q) of Eq. 10 with integer gamma, powers by repeated
// multiplication, every operation rounded once (no FMA).
__device__ __forceinline__ double sharpen(double q, int gamma) {
  const double omq = __dsub_rn(1.0, q);
  double a = q, b = omq;
  for (int g = 1; g < gamma; ++g) {
    a = __dmul_rn(a, q);
    b = __dmul_rn(b, omq);
  }
  return __ddiv_rn(a, __dadd_rn(a, b));
}

// The prefix-score window's preparation, done by extra blocks of the tag
// reduction's launch (the blocks after its streaming blocks): they are
// scheduled as the streaming blocks retire, so the preparation runs in the
// reduction's ragged tail instead of as a launch of its own.  Prep block 0
// sorts the window ascending (bitonic, in dynamic shared memory, padded to a
// power of two with +inf, which sorts last and is never read back); the other
// prep blocks tabulate F[c] = phi_gamma(c / n) for c = 0..n, kFPerBlock entries
// each, so the table's fp64 divisions and products run on many SMs instead of
// queueing on one SM's fp64 units.  NaN in the window is a data error.
constexpr int kFPerBlock = 32;

struct WindowPrep {
  const float* window;  // null: no preparation blocks
  int n;
  int gamma;
  float* sorted;        // [n]
  double* f_table;      // [n + 1]
  int32_t* status;
};

inline unsigned window_prep_blocks(int64_t n) {
  return 1u + static_cast<unsigned>((n + 1 + kFPerBlock - 1) / kFPerBlock);
}

inline size_t window_prep_smem(int64_t n) {
  size_t np2 = 1;
  while (np2 < static_cast<size_t>(n)) np2 <<= 1;
  return np2 * sizeof(float);
}

__device__ void window_prep_block(int b, const WindowPrep& w) {
  const int n = w.n;
  if (b > 0) {
    const int c = (b - 1) * kFPerBlock + static_cast<int>(threadIdx.x);
    if (threadIdx.x < kFPerBlock && c <= n)
      w.f_table[c] = sharpen(__ddiv_rn(static_cast<double>(c), static_cast<double>(n)), w.gamma);
    return;
  }
  extern __shared__ float sw[];
  int np2 = 1;
  while (np2 < n) np2 <<= 1;
  for (int k = threadIdx.x; k < np2; k += blockDim.x) {
    float v = k < n ? w.window[k] : __int_as_float(0x7f800000);
    if (isnan(v)) {
      report(w.status, PACE_ERR_NAN_INPUT);
      v = __int_as_float(0x7f800000);
    }
    sw[k] = v;
  }
  // Each step compares the pairs (lo, lo + stride): pair i puts a zero bit at
  // the stride's position of i, so every thread has work on every step.
  for (int size = 2; size <= np2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      __syncthreads();
      for (int i = threadIdx.x; i < (np2 >> 1); i += blockDim.x) {
        const int lo = ((i & ~(stride - 1)) << 1) | (i & (stride - 1));
        const int hi = lo | stride;
        const float a = sw[lo], c = sw[hi];
        if ((a > c) == ((lo & size) == 0)) {
          sw[lo] = c;
          sw[hi] = a;
        }
      }
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < n; k += blockDim.x) w.sorted[k] = sw[k];
}

// One warp's share of the stream (every warp of the first n_stream_blocks
// blocks calls it; it returns early when the range is empty or the offsets end
// before the tokens do).
template <int kTilesPerBatch>
__device__ __forceinline__ void stream_warp_range(const int32_t* __restrict__ tags,
                                                  const int64_t* __restrict__ offsets,
                                                  int64_t n_traj, int64_t n_tokens,
                                                  const TagTotals& tt, int n_stream_blocks) {
  constexpr int64_t kBatchTokens = kTileTokens * kTilesPerBatch;
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t n_warps = (static_cast<int64_t>(n_stream_blocks) * blockDim.x) >> 5;
  const int64_t n_batches = (n_tokens + kBatchTokens - 1) / kBatchTokens;
  const int64_t b_begin = n_batches * warp / n_warps;
  const int64_t b_end = n_batches * (warp + 1) / n_warps;
  if (b_begin >= b_end) {  // no tokens: no head part either
    if (lane == 0) tt.head[warp].traj = -1;
    return;
  }
  const int64_t t_begin = b_begin * kBatchTokens;
  const int64_t t_end = b_end * kBatchTokens < n_tokens ? b_end * kBatchTokens : n_tokens;

  // Start the stream before the search below: the warp's first batches are
  // requested into L2 while the offsets are searched (lanes 0..kPrefetchAhead-1,
  // one batch each; the pipeline then keeps kPrefetchAhead batches ahead).
  if (lane < kPrefetchAhead) {
    const int64_t pf = b_begin + lane;
    if (pf < b_end && (pf + 1) * kBatchTokens <= n_tokens)
      l2_prefetch_bulk(tags + pf * kBatchTokens, static_cast<uint32_t>(kBatchTokens * 4));
  }

  // trajectory holding token t_begin: the largest i in [1, n_traj) with
  // offsets[i] <= t_begin, else 0.  A 32-way search: the lanes probe 32 points of
  // [lo, hi) at once and a ballot keeps the sub-range after the last probe that
  // is <= t_begin (4 rounds for a million trajectories instead of 20 dependent
  // loads).  Whatever the offsets hold, lo stays in [0, n_traj).
  int64_t lo = 0, hi = n_traj;
  while (hi - lo > 1) {
    const int64_t span = hi - lo;
    const int64_t q = lo + 1 + ((span - 1) * lane) / 32;  // in [lo + 1, hi - 1], nondecreasing
    const unsigned bal = __ballot_sync(0xffffffffu, offsets[q] <= t_begin);
    if (bal == 0u) {
      hi = lo + 1;
    } else {
      const int j = 31 - __clz(bal);
      const int64_t qj = lo + 1 + ((span - 1) * j) / 32;
      hi = j < 31 ? lo + 1 + ((span - 1) * (j + 1)) / 32 : hi;
      lo = qj;
    }
  }
  int64_t cur = lo;
  int64_t cur_begin = offsets[cur];
  int64_t cur_end = offsets[cur + 1];
  // the first trajectory began before this range: this warp's part of it is its
  // head slot; otherwise the head slot says there is none
  const bool head_open = cur_begin < t_begin;
  if (!head_open && lane == 0) tt.head[warp].traj = -1;
  LaneAcc acc{0, 0u, 0u};

  auto load_batch = [&](int4 (&v)[kTilesPerBatch], int64_t b) {
    const int64_t bt0 = b * kBatchTokens;
    // ask L2 for a batch further ahead (no registers held while it is in flight)
    const int64_t pf = b + kPrefetchAhead;
    if (lane == 0 && pf < b_end && (pf + 1) * kBatchTokens <= n_tokens)
      l2_prefetch_bulk(tags + pf * kBatchTokens, static_cast<uint32_t>(kBatchTokens * 4));
    if (bt0 + kBatchTokens <= n_tokens) {
#pragma unroll
      for (int u = 0; u < kTilesPerBatch; ++u)
        v[u] = ld_stream_v4(tags + bt0 + u * kTileTokens + lane * 4);
    } else {
#pragma unroll
      for (int u = 0; u < kTilesPerBatch; ++u) {
        const int64_t t = bt0 + u * kTileTokens + lane * 4;
        v[u].x = (t + 0 < n_tokens) ? tags[t + 0] : -1;
        v[u].y = (t + 1 < n_tokens) ? tags[t + 1] : -1;
        v[u].z = (t + 2 < n_tokens) ? tags[t + 2] : -1;
        v[u].w = (t + 3 < n_tokens) ? tags[t + 3] : -1;
      }
    }
  };

  // Adds batch b to the running trajectory sums; false when the offsets end
  // before the tokens do (inconsistent offsets: stop).
  auto process = [&](const int4 (&v)[kTilesPerBatch], int64_t b) -> bool {
    const int64_t bt0 = b * kBatchTokens;
    const int64_t bt1 = (bt0 + kBatchTokens < n_tokens) ? bt0 + kBatchTokens : n_tokens;
    int64_t pos = bt0;
    while (true) {
      const int64_t seg_hi = cur_end < bt1 ? cur_end : bt1;
      if (pos == bt0 && seg_hi == bt0 + kBatchTokens) {
        // whole batch inside one trajectory: no position tests
        if (!acc_batch_fast<kTilesPerBatch>(acc, v)) {
#pragma unroll
          for (int u = 0; u < kTilesPerBatch; ++u) acc_group(acc, v[u]);
        }
      } else if (seg_hi > pos) {
        // batch-relative bounds fit 32 bits; they are the same in every lane, so
        // whole 128-token tiles outside [lo_r, hi_r) are skipped and tiles inside
        // it need no position tests
        const int lo_r = static_cast<int>(pos - bt0), hi_r = static_cast<int>(seg_hi - bt0);
#pragma unroll
        for (int u = 0; u < kTilesPerBatch; ++u) {
          const int t0 = u * kTileTokens;
          if (t0 + kTileTokens <= lo_r || t0 >= hi_r) continue;
          if (t0 >= lo_r && t0 + kTileTokens <= hi_r) {
            acc_group(acc, v[u]);
          } else {
            const int t = t0 + lane * 4;
            acc_elem(acc, v[u].x, t + 0 >= lo_r && t + 0 < hi_r);
            acc_elem(acc, v[u].y, t + 1 >= lo_r && t + 1 < hi_r);
            acc_elem(acc, v[u].z, t + 2 >= lo_r && t + 2 < hi_r);
            acc_elem(acc, v[u].w, t + 3 >= lo_r && t + 3 < hi_r);
          }
        }
      }
      if (cur_end > bt1) return true;  // trajectory continues into the next batch
      emit(acc, cur, false, head_open && cur == lo, warp, tt);
      if (seg_hi > pos) pos = seg_hi;
      ++cur;
      if (cur >= n_traj) return false;  // tokens past the last trajectory: offsets are bad
      cur_begin = cur_end;
      cur_end = offsets[cur + 1];
      // the next trajectory starts at the batch edge: continue in the next batch;
      // otherwise loop (more of this batch, or empty trajectories to step over)
      if (pos >= bt1 && cur_end > bt1) return true;
    }
  };

  // two register sets: the next batch's loads are in flight while one is added up
  int4 va[kTilesPerBatch], vb[kTilesPerBatch];
  int64_t b = b_begin;
  load_batch(va, b);
  while (true) {
    if (b + 1 < b_end) load_batch(vb, b + 1);
    if (!process(va, b)) return;
    if (++b >= b_end) break;
    if (b + 1 < b_end) load_batch(va, b + 1);
    if (!process(vb, b)) return;
    if (++b >= b_end) break;
  }
  // the trajectory still open continues past this range (one that begins at
  // t_end belongs to the next warp)
  if (cur < n_traj && cur_begin < t_end) emit(acc, cur, true, head_open && cur == lo, warp, tt);
}

struct FinalizeArgs {
  const int64_t* offsets;
  const int32_t* c_version;
  const float* s_pre;
  const float* window;           // W as given (used when window_sorted is null)
  const float* window_sorted;   // ascending, window_len values, or null
  const double* f_table;        // F for counts 0..window_len (with window_sorted)
  TagTotals tt;
  StreamGeom geom;
  int64_t n_traj;
  int64_t n_tokens;
  int32_t j;
  int32_t window_len;
  int32_t window_ready;
  int32_t mode;
  int32_t gamma;
  int32_t group_size;
  int32_t lanes;                // threads per trajectory for the direct count
  double f_missing;
  double* kgen;
  double* kwait;
  double* weight;
  double* score;
  double* unit_score;
  int32_t* status;
};

// Shared memory of one finalisation pass: the window (padded to a multiple of
// 4 floats), optionally the F table, the scores of the pass's trajectories and
// the partial counts.
struct FinalizeSmem {
  float* swin;
  double* ftab;    // [window_len + 1] or null (then F is read from global memory)
  double* sscore;  // [tpb]
  int* pcount;     // [lanes][tpb]
};

__host__ __device__ inline size_t finalize_smem_bytes(int64_t window_len, int tpb, int threads,
                                                      bool table_in_smem) {
  return align_up(static_cast<size_t>((window_len + 3) & ~3) * sizeof(float), 16) +
         (table_in_smem ? static_cast<size_t>(window_len + 1) * sizeof(double) : 0) +
         static_cast<size_t>(tpb) * sizeof(double) + static_cast<size_t>(threads) * sizeof(int);
}

__device__ __forceinline__ FinalizeSmem finalize_smem(unsigned char* raw, int window_len, int tpb,
                                                      bool table_in_smem) {
  FinalizeSmem m;
  const int wpad = (window_len + 3) & ~3;
  m.swin = reinterpret_cast<float*>(raw);
  double* d = reinterpret_cast<double*>(raw + align_up(wpad * sizeof(float), 16));
  m.ftab = table_in_smem ? d : nullptr;
  m.sscore = table_in_smem ? d + window_len + 1 : d;
  m.pcount = reinterpret_cast<int*>(m.sscore + tpb);
  return m;
}

// The window into shared memory: the sorted window, or the raw one NaN-padded
// to a multiple of 4 (NaN never counts as <= s); four loads per thread in
// flight at a time; with m.ftab set, the F table too.  L2 loads: the sorted
// window and the table may have been written by another block of the same
// launch.  Every thread of the block calls it.
__device__ void finalize_load_window(const FinalizeArgs& p, const FinalizeSmem& m) {
  if (p.window_ready) {
    const bool sorted = p.window_sorted != nullptr;
    const bool table = m.ftab && sorted;
    const int wpad = (p.window_len + 3) & ~3;
    const int tlen = table ? p.window_len + 1 : 0;
    const int span = wpad > tlen ? wpad : tlen;
    const float* src = sorted ? p.window_sorted : p.window;
    const int nb = static_cast<int>(blockDim.x);
    // four window values and four table entries per thread in flight at once
    for (int k0 = threadIdx.x; k0 < span; k0 += 4 * nb) {
      float w[4];
      double f[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k = k0 + j * nb;
        w[j] = k < p.window_len ? __ldcg(src + k) : __int_as_float(0x7fc00000);
        f[j] = k < tlen ? __ldcg(p.f_table + k) : 0.0;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k = k0 + j * nb;
        if (k < wpad) m.swin[k] = w[j];
        if (k < tlen) m.ftab[k] = f[j];
        if (!sorted && k < p.window_len && isnan(w[j])) report(p.status, PACE_ERR_NAN_INPUT);
      }
    }
  }
  __syncthreads();
}

// What one thread of a pass reads for its trajectory: the inputs (loadable any
// time) and the stream's totals from the slots (only once the stream blocks that
// hold its tokens are done).
struct TrajIn {
  float s;
  int32_t c;
  int64_t o0, o1;
  ulonglong2 slot;
  unsigned long long sum;
  unsigned cnt, maxp1;
};

__device__ __forceinline__ void load_traj_inputs(const FinalizeArgs& p, int64_t i0, int64_t i_end,
                                                 int tpb, int lanes, TrajIn& in) {
  const int tid = static_cast<int>(threadIdx.x);
  const int64_t i = i0 + tid % tpb;
  const bool valid = tid < tpb * lanes && i < i_end;
  in.s = (valid && p.s_pre) ? p.s_pre[i] : __int_as_float(0x7fc00000);
  if (tid < tpb && i < i_end) {
    in.c = p.c_version[i];
    in.o0 = p.offsets[i];
    in.o1 = p.offsets[i + 1];
  }
}

// The stream's slot of this thread's trajectory (issue it early: its load need
// not wait for anything), then the totals (which may load head slots).
__device__ __forceinline__ void load_traj_slot(const FinalizeArgs& p, int64_t i0, int64_t i_end,
                                               int tpb, TrajIn& in) {
  const int tid = static_cast<int>(threadIdx.x);
  const int64_t i = i0 + tid;
  if (tid < tpb && i < i_end) in.slot = __ldcg(p.tt.slot + i);
}

__device__ __forceinline__ void load_traj_acc(const FinalizeArgs& p, int64_t i0, int64_t i_end,
                                              int tpb, TrajIn& in) {
  const int tid = static_cast<int>(threadIdx.x);
  const int64_t i = i0 + tid;
  if (tid < tpb && i < i_end) {
    long long sum;
    traj_totals(p.tt, p.geom, p.n_tokens, i, in.o0, in.o1, in.slot, sum, in.cnt, in.maxp1);
    in.sum = static_cast<unsigned long long>(sum);
  }
}

// One pass over trajectories [i0, i0 + tpb) clipped to i_end (i0 and tpb whole
// groups), from what load_traj_inputs and load_traj_acc read: thread t <
// tpb * lanes counts for trajectory slot t % tpb (on the direct-count path
// `lanes` threads per trajectory each count one strided share of the window;
// lanes = 1 with the sorted window); threads t < tpb then do that trajectory's
// fp64 work, and the first thread of each group its mean in fixed left-to-right
// order.  Every thread of the block calls it.
__device__ void finalize_pass(const FinalizeArgs& p, int64_t i0, int64_t i_end, int tpb,
                              int lanes, const FinalizeSmem& m, const TrajIn& in) {
  const bool sorted = p.window_sorted != nullptr;
  const int wpad = (p.window_len + 3) & ~3;
  const int tid = static_cast<int>(threadIdx.x);
  const bool active = tid < tpb * lanes;
  const int slot = tid % tpb;
  const int64_t i = i0 + slot;
  const bool lead = tid < tpb;  // owns trajectory i's results
  const float s = in.s;
  if (p.window_ready && !sorted) {
    // direct count of window values <= s, one strided share of the window per lane
    int count = 0;
    if (active && !isnan(s)) {
      const float4* w4 = reinterpret_cast<const float4*>(m.swin);
      for (int k = tid / tpb; k < wpad / 4; k += lanes) {
        const float4 w = w4[k];
        count += (w.x <= s) + (w.y <= s) + (w.z <= s) + (w.w <= s);
      }
    }
    if (active) m.pcount[tid] = count;
    __syncthreads();
  }

  if (lead && i < i_end) {
    const int64_t o0 = in.o0, o1 = in.o1;
    if (o1 < o0 || (i == 0 && o0 != 0) || (i == p.n_traj - 1 && o1 != p.n_tokens))
      report(p.status, PACE_ERR_INVALID_ARG);
    const int64_t c = in.c;
    const unsigned t_count = in.cnt;
    const unsigned mp1 = in.maxp1;
    const long long tag_sum = static_cast<long long>(in.sum);
    if (c < 0 || mp1 >= 0x80000000u) report(p.status, PACE_ERR_INVALID_ARG);
    if (c > p.j || (mp1 != 0u && static_cast<int64_t>(mp1) - 1 > c))
      report(p.status, PACE_ERR_VERSION_ORDER);
    // Lemma 1: K_gen = (1/T) sum (c - v_t) = (c T - sum v_t) / T, exact integers
    const long long gen_sum = static_cast<long long>(c) * static_cast<long long>(t_count) - tag_sum;
    // the correctly rounded K_gen and K_wait, built on the integer pipe
    const double kgen = t_count > 0u ? i64_div_u32_rn(gen_sum, t_count) : 0.0;
    const double kwait = i64_to_double_rn(static_cast<long long>(p.j) - c);
    double f;
    if (!p.window_ready) {
      f = 1.0;
    } else if (isnan(s)) {
      f = p.f_missing;
    } else if (sorted) {
      // count of window values <= s: the first index of the sorted window
      // holding a value > s
      int lo = 0, hi = p.window_len;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (m.swin[mid] <= s) lo = mid + 1;
        else hi = mid;
      }
      f = m.ftab ? m.ftab[lo] : __ldcg(p.f_table + lo);
    } else {  // small pools: F from the summed partial counts
      int count = 0;
      for (int l = 0; l < lanes; ++l) count += m.pcount[l * tpb + slot];
      f = sharpen(__ddiv_rn(static_cast<double>(count), static_cast<double>(p.window_len)),
                  p.gamma);
    }
    double sc;
    if (p.mode == PACE_SCORE_EFF) sc = __dadd_rn(kwait, __dmul_rn(f, kgen));
    else if (p.mode == PACE_SCORE_RAW) sc = __dadd_rn(kwait, kgen);
    else sc = __dmul_rn(f, kgen);
    if (p.kgen) p.kgen[i] = kgen;
    if (p.kwait) p.kwait[i] = kwait;
    if (p.weight) p.weight[i] = f;
    p.score[i] = sc;
    m.sscore[slot] = sc;
  }
  __syncthreads();
  const int G = p.group_size;
  if (p.unit_score && lead && i < i_end && (slot % G) == 0) {
    double acc = 0.0;
    for (int g = 0; g < G; ++g) acc = __dadd_rn(acc, m.sscore[slot + g]);
    // for G = 2^m, acc * 2^-m is the same correctly rounded value as acc / G
    // (2^-m is exact), one multiplication instead of a division
    p.unit_score[i / G] = (G & (G - 1)) == 0 ? __dmul_rn(acc, 1.0 / static_cast<double>(G))
                                             : __ddiv_rn(acc, static_cast<double>(G));
  }
}

// The finalisation as a launch of its own (groups of more than 256): blockDim.x
// = tpb * lanes, tpb trajectories (whole groups) per block.
__global__ void score_finalize_kernel(FinalizeArgs p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int tpb = static_cast<int>(blockDim.x) / p.lanes;
  const FinalizeSmem m = finalize_smem(smem_raw, p.window_len, tpb, p.window_sorted != nullptr);
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * tpb;
  // the inputs, the slot and the window are in flight together; the head slots
  // of continuing trajectories are loaded once the window is in place
  TrajIn in;
  load_traj_inputs(p, i0, p.n_traj, tpb, p.lanes, in);
  load_traj_slot(p, i0, p.n_traj, tpb, in);
  finalize_load_window(p, m);
  load_traj_acc(p, i0, p.n_traj, tpb, in);
  finalize_pass(p, i0, p.n_traj, tpb, p.lanes, m, in);
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// The finalisation inside the tag reduction's launch (groups of at most 256).
// The launch is cooperative, so all its blocks are resident at once and every
// wait below ends as soon as the blocks it waits for have streamed their share.
struct FusedFinalize {
  unsigned* done;       // [stream blocks] set once a block's warps have all streamed; null: off
  unsigned* ticket;     // counts the blocks that have finished streaming
  unsigned* prep_done;  // counts the finished preparation tasks
  int prep_tasks;       // window sort + F-table slices (0: no table)
  int tpb, lanes;       // trajectories per finalisation pass, threads per trajectory
  WindowPrep prep;
  FinalizeArgs fin;
};

// Run by every block once its own warps have streamed: publish that, take a
// finishing ticket (the first finishers, idle in the reduction's ragged tail,
// run the window's preparation tasks: task 0 sorts W, task 1 + k tabulates F
// for 32 counts), then finalise this block's slice of the groups,
// [U b / S, U (b + 1) / S), once the stream blocks covering those groups'
// tokens and the preparation are done.  Each block thus finalises in the tail
// as soon as its neighbourhood of the stream is complete, and no launch of its
// own is needed.
__device__ __forceinline__ void fused_finalize(const int64_t* __restrict__ offsets,
                                               int64_t n_tokens, int n_stream_blocks,
                                               const FusedFinalize& fz) {
  __shared__ unsigned s_ticket;
  const int tid = static_cast<int>(threadIdx.x);
  const int S = n_stream_blocks;
  const int64_t blk = blockIdx.x;
  __threadfence();  // this thread's slot stores before the block's flag
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    atomicAdd(fz.done + blk, 1u);
    s_ticket = atomicAdd(fz.ticket, 1u);
  }
  __syncthreads();
  for (unsigned task = s_ticket; task < static_cast<unsigned>(fz.prep_tasks);
       task += static_cast<unsigned>(S)) {
    window_prep_block(static_cast<int>(task), fz.prep);
    __threadfence();
    __syncthreads();
    if (tid == 0) atomicAdd(fz.prep_done, 1u);
  }

  const FinalizeArgs& p = fz.fin;
  const int G = p.group_size;
  const int64_t U = p.n_traj / G;
  const int64_t u_lo = U * blk / S, u_hi = U * (blk + 1) / S;
  if (u_lo >= u_hi) return;
  const int64_t i_lo = u_lo * G, i_hi = u_hi * G;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const bool sorted = p.window_sorted != nullptr;
  const FinalizeSmem m = finalize_smem(smem_raw, p.window_len, fz.tpb, sorted);
  // the first pass's inputs are in flight while the waits below run
  TrajIn cur;
  load_traj_inputs(p, i_lo, i_hi, fz.tpb, fz.lanes, cur);
  if (tid < 32) {
    const int lane = tid;
    // stream blocks holding the tokens of trajectories [i_lo, i_hi): the warp of
    // batch b is the last w with n_batches * w / n_warps <= b
    int64_t b_lo = 0, b_hi = -1;
    int64_t t0 = offsets[i_lo], t1 = offsets[i_hi];
    t0 = t0 < 0 ? 0 : (t0 > n_tokens ? n_tokens : t0);
    t1 = t1 < 0 ? 0 : (t1 > n_tokens ? n_tokens : t1);
    if (t1 < t0) {  // inconsistent offsets (reported by the pass): wait for every block
      b_hi = S - 1;
    } else if (t1 > t0) {
      const StreamGeom& g = p.geom;
      b_lo = warp_of_batch(g, t0 / g.batch_tokens) / (kReduceThreads / 32);
      b_hi = warp_of_batch(g, (t1 - 1) / g.batch_tokens) / (kReduceThreads / 32);
    }
    bool ok = true;
    const uint64_t start = global_timer_ns();
    for (int64_t b = b_lo + lane; ok && b <= b_hi; b += 32) {
      while (ld_acquire_u32(fz.done + b) == 0u) {
        if (global_timer_ns() - start > kWaitLimitNs) {
          ok = false;
          break;
        }
        __nanosleep(64);
      }
    }
    if (lane == 0 && fz.prep_tasks > 0) {
      while (ok && ld_acquire_u32(fz.prep_done) < static_cast<unsigned>(fz.prep_tasks)) {
        if (global_timer_ns() - start > kWaitLimitNs) ok = false;
        else __nanosleep(64);
      }
    }
    if (!__all_sync(0xffffffffu, ok) && lane == 0) report(p.status, PACE_ERR_TIMEOUT);
  }
  __syncthreads();
  load_traj_slot(p, i_lo, i_hi, fz.tpb, cur);
  finalize_load_window(p, m);
  load_traj_acc(p, i_lo, i_hi, fz.tpb, cur);
  for (int64_t i0 = i_lo; i0 < i_hi; i0 += fz.tpb) {
    // the next pass's reads are in flight while this pass computes
    TrajIn nxt;
    const int64_t i1 = i0 + fz.tpb;
    if (i1 < i_hi) {
      load_traj_inputs(p, i1, i_hi, fz.tpb, fz.lanes, nxt);
      load_traj_slot(p, i1, i_hi, fz.tpb, nxt);
      load_traj_acc(p, i1, i_hi, fz.tpb, nxt);
    }
    finalize_pass(p, i0, i_hi, fz.tpb, fz.lanes, m, cur);
    __syncthreads();  // the pass's shared scores and counts are reused
    cur = nxt;
  }
}

template <int kTilesPerBatch, int kMinBlocks>
__global__ void __launch_bounds__(kReduceThreads, kMinBlocks)
    tag_reduce_kernel(const int32_t* __restrict__ tags, const int64_t* __restrict__ offsets,
                      int64_t n_traj, int64_t n_tokens, TagTotals tt, int n_stream_blocks,
                      WindowPrep prep, FusedFinalize fz) {
  if (static_cast<int>(blockIdx.x) >= n_stream_blocks) {  // the window's preparation
    window_prep_block(static_cast<int>(blockIdx.x) - n_stream_blocks, prep);
    return;
  }
  stream_warp_range<kTilesPerBatch>(tags, offsets, n_traj, n_tokens, tt, n_stream_blocks);
  if (fz.done) fused_finalize(offsets, n_tokens, n_stream_blocks, fz);
}

// Stale-k admission (Sec. 2): kbar = sum (j - v_t) / T = (j T - sum v_t) / T in
// exact integers, one rounding; admitted when kbar <= k_max.
__global__ void stale_k_kernel(const int64_t* __restrict__ offsets, TagTotals tt, StreamGeom geom,
                               int64_t n_traj, int64_t n_tokens, int32_t j, double k_max,
                               double* __restrict__ kbar, uint8_t* __restrict__ admitted,
                               int32_t* status) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n_traj) return;
  const int64_t o0 = offsets[i], o1 = offsets[i + 1];
  if (o1 < o0 || (i == 0 && o0 != 0) || (i == n_traj - 1 && o1 != n_tokens))
    report(status, PACE_ERR_INVALID_ARG);
  long long tag_sum;
  unsigned t_count, mp1;
  traj_totals(tt, geom, n_tokens, i, o0, o1, __ldcg(tt.slot + i), tag_sum, t_count, mp1);
  if (mp1 >= 0x80000000u) report(status, PACE_ERR_INVALID_ARG);
  if (mp1 != 0u && static_cast<int64_t>(mp1) - 1 > j) report(status, PACE_ERR_VERSION_ORDER);
  const long long lag_sum = static_cast<long long>(j) * static_cast<long long>(t_count) - tag_sum;
  const double kb = t_count > 0u ? i64_div_u32_rn(lag_sum, t_count) : 0.0;
  if (kbar) kbar[i] = kb;
  admitted[i] = kb <= k_max ? 1 : 0;
}

// Stream blocks of one launch at most (one wave: SMs x resident blocks per SM).
constexpr int kMaxStreamBlocks = 2048;

struct ScoreWs {
  TagTotals tt;     // slots [n_traj], head slots [kMaxStreamBlocks x 8 warps]
  unsigned* flags;  // [2 + kMaxStreamBlocks]: ticket, preparation count, stream blocks done
};

struct WindowWs {
  float* sorted;    // [window_len]
  double* f_table;  // [window_len + 1]
};

WindowWs carve_window_ws(Carver& cv, int64_t window_len) {
  WindowWs w;
  w.sorted = cv.take<float>(static_cast<size_t>(window_len > 0 ? window_len : 1));
  w.f_table = cv.take<double>(static_cast<size_t>(window_len + 1));
  return w;
}

ScoreWs carve_score_ws(Carver& cv, int64_t n_traj) {
  ScoreWs w;
  w.tt.slot = cv.take<ulonglong2>(static_cast<size_t>(n_traj));
  w.tt.head = cv.take<HeadSlot>(static_cast<size_t>(kMaxStreamBlocks) * (kReduceThreads / 32));
  w.flags = cv.take<unsigned>(2 + kMaxStreamBlocks);
  return w;
}

// Resident blocks per SM of a tag-reduction instance with the given dynamic
// shared memory (cached per device, instance and size).
template <int kTiles, int kBlocks>
pace_status reduce_blocks_per_sm(size_t smem, int* out) {
  constexpr int kMaxDevices = 64;
  static int cache[kMaxDevices][2] = {};
  static size_t cache_smem[kMaxDevices][2] = {};
  static std::mutex mu;
  int dev = 0;
  PACE_TRY_CUDA(cudaGetDevice(&dev));
  const int which = kTiles == kTilesSmall ? 0 : 1;
  std::lock_guard<std::mutex> g(mu);
  if (dev >= 0 && dev < kMaxDevices && cache[dev][which] > 0 && cache_smem[dev][which] == smem) {
    *out = cache[dev][which];
    return PACE_OK;
  }
  int nb = 0;
  // above the default 48 KB (windows of more than ~2,000 values with their F
  // table) the kernel must be allowed the larger dynamic shared memory first
  if (smem > 48 * 1024)
    PACE_TRY_CUDA(cudaFuncSetAttribute(tag_reduce_kernel<kTiles, kBlocks>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem)));
  PACE_TRY_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(
      &nb, tag_reduce_kernel<kTiles, kBlocks>, kReduceThreads, smem));
  if (dev >= 0 && dev < kMaxDevices) {
    cache[dev][which] = nb;
    cache_smem[dev][which] = smem;
  }
  *out = nb;
  return PACE_OK;
}

template <int kTiles, int kBlocks>
pace_status launch_tag_reduce(unsigned grid, size_t smem, bool cooperative, cudaStream_t st,
                              const int32_t* tags, const int64_t* offsets, int64_t n_traj,
                              int64_t n_tokens, const ScoreWs& ws, int stream_blocks,
                              const WindowPrep& prep, const FusedFinalize& fz) {
  if (!cooperative) {
    tag_reduce_kernel<kTiles, kBlocks><<<grid, kReduceThreads, smem, st>>>(
        tags, offsets, n_traj, n_tokens, ws.tt, stream_blocks, prep, fz);
    return last_launch_status();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kReduceThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  PACE_TRY_CUDA(cudaLaunchKernelEx(&cfg, tag_reduce_kernel<kTiles, kBlocks>, tags, offsets,
                                   n_traj, n_tokens, ws.tt, stream_blocks, prep, fz));
  return last_launch_status();
}

// Stream the tags once into the slots (nothing to zero first).  With
// prep.window set, the same launch also sorts the window and tabulates F
// (extra blocks, run in the stream's tail).  With `fused` (fz.done is filled in
// here, its flags zeroed), the launch is cooperative and also finalises every
// trajectory and group (fused_finalize): one wave of stream blocks, at least
// one block even for an empty stream.  *geom receives the launch's geometry.
pace_status run_tag_reduce(const int32_t* tags, const int64_t* offsets, int64_t n_traj,
                           int64_t n_tokens, const ScoreWs& ws, const WindowPrep& prep,
                           FusedFinalize fz, bool fused, size_t fused_smem, StreamGeom* geom,
                           cudaStream_t st) {
  const unsigned prep_blocks = (prep.window && !fused) ? window_prep_blocks(prep.n) : 0u;
  size_t smem = prep_blocks ? window_prep_smem(prep.n) : 0;
  if (fused) smem = fused_smem;
  const bool small = n_tokens <= kSmallPoolTokens;
  const int tiles = small ? kTilesSmall : kTilesLarge;
  int per_sm = small ? kBlocksSmall : kBlocksLarge;
  if (fused) {
    int nb = 0;
    const pace_status occ = small ? reduce_blocks_per_sm<kTilesSmall, kBlocksSmall>(smem, &nb)
                                  : reduce_blocks_per_sm<kTilesLarge, kBlocksLarge>(smem, &nb);
    if (occ != PACE_OK) return occ;
    if (nb < 1) return PACE_ERR_UNSUPPORTED_SHAPE;
    per_sm = nb < per_sm ? nb : per_sm;
  }
  const int64_t batch_tokens = static_cast<int64_t>(kTileTokens) * tiles;
  const int64_t n_batches = (n_tokens + batch_tokens - 1) / batch_tokens;
  const int warps_per_block = kReduceThreads / 32;
  const int64_t per_block = warps_per_block * kMinBatchesPerWarp;
  int64_t blocks = (n_batches + per_block - 1) / per_block;
  int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;  // one wave
  if (cap > kMaxStreamBlocks) cap = kMaxStreamBlocks;
  if (blocks > cap) blocks = cap;
  if (fused && blocks < 1) blocks = 1;
  geom->batch_tokens = batch_tokens;
  geom->n_batches = n_batches;
  geom->n_warps = blocks * warps_per_block;
  if (blocks == 0 && prep_blocks == 0) return PACE_OK;
  if (fused) {
    PACE_TRY_CUDA(cudaMemsetAsync(ws.flags, 0, static_cast<size_t>(2 + blocks) * sizeof(unsigned),
                                  st));
    fz.ticket = ws.flags;
    fz.prep_done = ws.flags + 1;
    fz.done = ws.flags + 2;
    fz.fin.geom = *geom;
  } else {
    fz = FusedFinalize{};
  }
  const unsigned grid = static_cast<unsigned>(blocks) + prep_blocks;
  const int stream_blocks = static_cast<int>(blocks);
  const ProfileEvents& pe = profile_events(PACE_PROFILE_TAG_REDUCE);
  if (pe.begin) PACE_TRY_CUDA(cudaEventRecord(pe.begin, st));
  if (small)
    PACE_TRY((launch_tag_reduce<kTilesSmall, kBlocksSmall>(grid, smem, fused, st, tags, offsets,
                                                            n_traj, n_tokens, ws, stream_blocks,
                                                            prep, fz)));
  else
    PACE_TRY((launch_tag_reduce<kTilesLarge, kBlocksLarge>(grid, smem, fused, st, tags, offsets,
                                                            n_traj, n_tokens, ws, stream_blocks,
                                                            prep, fz)));
  if (pe.end) PACE_TRY_CUDA(cudaEventRecord(pe.end, st));
  return PACE_OK;
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_stale_k_workspace_size(int64_t n_traj) {
  return pace_score_pool_workspace_size(n_traj, 0);
}

extern "C" pace_status pace_stale_k(const int32_t* tags, const int64_t* offsets, int64_t n_traj,
                                    int64_t n_tokens, int32_t trainer_version, double k_max,
                                    double* kbar, uint8_t* admitted, void* workspace,
                                    size_t workspace_bytes, int32_t* status_dev, void* stream) {
  if (n_traj < 0 || n_tokens < 0 || n_traj > (int64_t(1) << 31)) return PACE_ERR_INVALID_ARG;
  if (n_traj > 0 && (!offsets || !admitted)) return PACE_ERR_INVALID_ARG;
  if (n_tokens > 0 && !tags) return PACE_ERR_INVALID_ARG;
  if (isnan(k_max)) return PACE_ERR_INVALID_ARG;
  if (tags && !aligned(tags, 16)) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (n_traj == 0) return n_tokens == 0 ? PACE_OK : PACE_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  ScoreWs ws = carve_score_ws(cv, n_traj);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  cudaStream_t st = as_stream(stream);
  StreamGeom geom{};
  PACE_TRY(run_tag_reduce(tags, offsets, n_traj, n_tokens, ws, WindowPrep{}, FusedFinalize{},
                          false, 0, &geom, st));
  const int threads = 256;
  stale_k_kernel<<<static_cast<unsigned>((n_traj + threads - 1) / threads), threads, 0, st>>>(
      offsets, ws.tt, geom, n_traj, n_tokens, trainer_version, k_max, kbar,
      admitted, status_dev);
  return last_launch_status();
}

extern "C" pace_status pace_set_score_fused_min_traj(int64_t min_traj) {
  if (min_traj < 0) return PACE_ERR_INVALID_ARG;
  fused_min_traj().store(min_traj == 0 ? 0 : min_traj);
  return PACE_OK;
}

extern "C" int64_t pace_score_fused_min_traj_default(void) { return kFusedMinTrajDefault; }

extern "C" void pace_score_params_default(PaceScoreParams* p) {
  if (!p) return;
  p->mode = PACE_SCORE_EFF;
  p->gamma = 4;
  p->min_obs = 32;
  p->group_size = 8;
  p->f_missing = 1.0;
}

extern "C" size_t pace_score_pool_workspace_size(int64_t n_traj, int64_t window_len) {
  if (n_traj < 0 || window_len < 0) return 0;
  Carver cv;
  carve_score_ws(cv, n_traj);
  carve_window_ws(cv, window_len);
  return cv.used;
}

extern "C" pace_status pace_score_pool(const int32_t* tags, const int64_t* offsets,
                                       const int32_t* c_version, const float* s_pre,
                                       int64_t n_traj, int64_t n_tokens, int32_t trainer_version,
                                       const float* window, int64_t window_len,
                                       const PaceScoreParams* params, double* kgen,
                                       double* kwait, double* weight, double* score,
                                       double* unit_score, void* workspace,
                                       size_t workspace_bytes, int32_t* status_dev,
                                       void* stream) {
  if (!params) return PACE_ERR_INVALID_ARG;
  if (n_traj < 0 || n_tokens < 0 || n_traj > (int64_t(1) << 31)) return PACE_ERR_INVALID_ARG;
  if (n_traj > 0 && (!offsets || !c_version || !score)) return PACE_ERR_INVALID_ARG;
  if (n_tokens > 0 && !tags) return PACE_ERR_INVALID_ARG;
  const int G = params->group_size;
  if (G < 1 || G > 1024 || n_traj % G != 0) return PACE_ERR_INVALID_ARG;
  if (params->gamma < 1 || params->gamma > 64) return PACE_ERR_INVALID_ARG;
  if (params->mode != PACE_SCORE_EFF && params->mode != PACE_SCORE_RAW &&
      params->mode != PACE_SCORE_GEN)
    return PACE_ERR_INVALID_ARG;
  if (window_len < 0 || window_len > kMaxWindow) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (window_len > 0 && !window) return PACE_ERR_INVALID_ARG;
  if (tags && !aligned(tags, 16)) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (n_traj == 0) return n_tokens == 0 ? PACE_OK : PACE_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  ScoreWs ws = carve_score_ws(cv, n_traj);
  WindowWs wws = carve_window_ws(cv, window_len);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;

  cudaStream_t st = as_stream(stream);
  const bool window_ready = window_len > 0 && window_len >= params->min_obs;
  // With the sorted window and the F table the finalisation takes one binary
  // search and one table read per trajectory; their preparation runs inside the
  // tag reduction's launch.  Small pools count against the raw window instead
  // (the same bits either way).
  const bool use_table = window_ready && n_traj >= kTableMinTraj;
  WindowPrep prep{};
  if (use_table) {
    prep.window = window;
    prep.n = static_cast<int>(window_len);
    prep.gamma = params->gamma;
    prep.sorted = wws.sorted;
    prep.f_table = wws.f_table;
    prep.status = status_dev;
  }
  FinalizeArgs a;
  a.offsets = offsets;
  a.c_version = c_version;
  a.s_pre = s_pre;
  a.window = window;
  a.window_sorted = use_table ? wws.sorted : nullptr;
  a.f_table = use_table ? wws.f_table : nullptr;
  a.tt = ws.tt;
  a.geom = StreamGeom{};
  a.n_traj = n_traj;
  a.n_tokens = n_tokens;
  a.j = trainer_version;
  a.window_len = static_cast<int32_t>(window_len);
  a.window_ready = window_ready ? 1 : 0;
  a.mode = params->mode;
  a.gamma = params->gamma;
  a.group_size = G;
  a.f_missing = params->f_missing;
  a.kgen = kgen;
  a.kwait = kwait;
  a.weight = weight;
  a.score = score;
  a.unit_score = unit_score;
  a.status = status_dev;

  if (G <= kReduceThreads && n_traj >= fused_min_traj().load() && cooperative_launch_ok()) {
    // Large pools whose groups fit one block: the finalisation runs inside the
    // tag reduction's launch, each stream block finalising its slice of the
    // groups in the stream's ragged tail, where most of the per-trajectory work
    // hides (1M sweep pool: 2.31 -> 2.28 ms per call).  On small pools the chain
    // after the last stream block (flags, waits, one pass) costs more than a
    // launch of its own (16k: 65.6 -> 71 us), so they keep that launch.  Passes
    // of whole groups over the block's 256 threads; on the direct-count path
    // up to 8 threads per trajectory share the count.
    int lanes = 1;
    if (!use_table && window_ready) {
      lanes = 8;
      while (lanes > 1 && G * lanes > kReduceThreads) lanes /= 2;
    }
    FusedFinalize fz{};
    fz.lanes = lanes;
    fz.tpb = (kReduceThreads / lanes / G) * G;
    a.lanes = lanes;
    fz.fin = a;
    if (use_table) {
      fz.prep = prep;
      fz.prep_tasks = static_cast<int>(window_prep_blocks(prep.n));
    }
    size_t smem = finalize_smem_bytes(window_len, fz.tpb, kReduceThreads, use_table);
    if (use_table && window_prep_smem(prep.n) > smem) smem = window_prep_smem(prep.n);
    StreamGeom geom{};
    return run_tag_reduce(tags, offsets, n_traj, n_tokens, ws, WindowPrep{}, fz, true, smem, &geom,
                          st);
  }

  PACE_TRY(run_tag_reduce(tags, offsets, n_traj, n_tokens, ws, prep, FusedFinalize{}, false, 0,
                          &a.geom, st));
  // A launch of its own: whole groups per block.  With the sorted window: one
  // thread per trajectory, 256 threads (whole groups) per block, so that one
  // round of loads brings the window and the F table into shared memory.
  // Otherwise small pools take fewer groups per block so that the
  // per-trajectory fp64 work of F (GB300's fp64 rate is low) is spread over
  // about two blocks per SM instead of queueing on a few SMs; with the direct
  // count, up to 8 threads per trajectory share the count so its chain is 8
  // times shorter.
  const int max_units = G >= 256 ? 1 : 256 / G;
  const int64_t n_units = n_traj / G;
  const int64_t spread = 2 * static_cast<int64_t>(sm_count());
  int64_t want = (n_units + spread - 1) / spread;
  int min_units = 1;
  int lanes = 1;
  if (use_table) {
    min_units = max_units;
  } else if (window_ready) {
    lanes = 8;
  } else {
    min_units = G >= 64 ? 1 : (64 + G - 1) / G;
  }
  want = want < min_units ? min_units : want;
  const int units_per_block = want > max_units ? max_units : static_cast<int>(want);
  const int tpb = units_per_block * G;
  while (lanes > 1 && tpb * lanes > 1024) lanes /= 2;
  a.lanes = lanes;
  const int threads = tpb * lanes;
  const int64_t blocks = (n_traj + tpb - 1) / tpb;
  const size_t smem = finalize_smem_bytes(window_len, tpb, threads, use_table);
  if (smem > 48 * 1024)
    PACE_TRY_CUDA(cudaFuncSetAttribute(score_finalize_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem)));
  score_finalize_kernel<<<static_cast<unsigned>(blocks), threads, smem, st>>>(a);
  return last_launch_status();
}

namespace pace {
namespace {

// Both constructions of the same doubles, side by side (the self-test below).
__global__ void div_selftest_kernel(const long long* __restrict__ S,
                                    const unsigned* __restrict__ T, int64_t n,
                                    double* __restrict__ q_int, double* __restrict__ q_fp64,
                                    double* __restrict__ c_int, double* __restrict__ c_fp64) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    q_int[i] = i64_div_u32_rn(S[i], T[i]);
    q_fp64[i] = __ddiv_rn(__ll2double_rn(S[i]), __ull2double_rn(T[i]));
    c_int[i] = i64_to_double_rn(S[i]);
    c_fp64[i] = __ll2double_rn(S[i]);
  }
}

}  // namespace
}  // namespace pace

extern "C" pace_status pace_div_selftest(const int64_t* S, const uint32_t* T, int64_t n,
                                         double* q_int, double* q_fp64, double* c_int,
                                         double* c_fp64, void* stream) {
  if (n < 0 || (n > 0 && (!S || !T || !q_int || !q_fp64 || !c_int || !c_fp64)))
    return PACE_ERR_INVALID_ARG;
  if (n == 0) return PACE_OK;
  pace::div_selftest_kernel<<<static_cast<unsigned>(n < 4096 ? (n + 255) / 256 : 16 * pace::sm_count()),
                              256, 0, pace::as_stream(stream)>>>(
      reinterpret_cast<const long long*>(S), reinterpret_cast<const unsigned*>(T), n, q_int,
      q_fp64, c_int, c_fp64);
  return pace::last_launch_status();
}
