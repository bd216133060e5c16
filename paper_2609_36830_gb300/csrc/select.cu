// Rejection budget (Eqs. 3-4, host) and deterministic top-k rejection of
// units (Sec. 3.1 quantile rule read as "reject the r-hat fraction of the
// current pool with the largest scores"; Algorithm 1, trainer side).
//
// Order: score descending, then unit id ascending.  The k first units in that
// order are rejected; outputs list trajectory ids ascending.
//
//   small pools (U <= 512): one block ranks every unit against every other
//     unit in shared memory and compacts the ids (one launch).
//   mid-size pools (U <= 131,072): one cluster of up to 8 CTAs holds every key
//     in shared memory (16,384 per CTA), finds the pivot by a radix select that
//     skips the bits all remaining candidates share (histograms combined
//     through distributed shared memory), and each CTA writes the ids and flags
//     of its own units (one launch).
//   large pools: MSB-first radix select over order-preserving 64-bit keys
//     (six 11/10-bit digit passes; each pass's blocks derive the previous
//     pass's digit from its histogram themselves), then a three-phase scan
//     compaction over 256-unit tiles that rejects the units above the pivot
//     and the lowest-id units equal to it.
//
// Also here: the retained-vs-rejected staleness histograms (f4), the literal
// sliding-window quantile admission (Sec. 3.1, Algorithm 1), and the
// selection entry point that needs no caller workspace.
#include <cooperative_groups.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "pace_block.cuh"
#include "pace_internal.cuh"

namespace pace {
namespace {

namespace cg = cooperative_groups;

constexpr int kSmallMax = 512;
constexpr int kSmallThreads = 512;
constexpr int kHistBins = 2048;
constexpr int kTile = 256;  // units per compaction block of the radix path
constexpr int kTileThreads = 256;
constexpr int kPerThread = kTile / kTileThreads;
constexpr int kPasses = 6;
__constant__ int c_shift[kPasses] = {53, 42, 31, 20, 10, 0};
__constant__ int c_width[kPasses] = {11, 11, 11, 11, 10, 10};

// Order-preserving map of a double to uint64 (after folding -0.0 into +0.0),
// so unsigned key order equals numeric order for every non-NaN value.
__device__ __forceinline__ uint64_t order_key(double x) {
  uint64_t b = static_cast<uint64_t>(__double_as_longlong(x));
  if (b == 0x8000000000000000ull) b = 0;
  return (b & 0x8000000000000000ull) ? ~b : (b | 0x8000000000000000ull);
}

struct SelectState {
  unsigned long long prefix;
  unsigned long long mask;
  long long k_rem;
  int done;
  int pad;
};

// Start state of the radix select (nothing fixed yet, k units left to reject) in
// state slot 0 and a cleared first histogram.  A kernel rather than a host copy,
// so the call stays valid inside a captured CUDA graph (a captured copy would
// re-read host memory that no longer holds the values at replay).
__global__ void select_init_kernel(SelectState* states, long long k, unsigned* hist0) {
  if (threadIdx.x == 0) {
    states[0].prefix = 0ull;
    states[0].mask = 0ull;
    states[0].k_rem = k;
    states[0].done = 0;
    states[0].pad = 0;
  }
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) hist0[b] = 0u;
}

// The radix step of one pass, computed identically by every block that needs
// it: in the histogram of the keys matching st's prefix, find the digit holding
// the k_rem-th largest of them, and narrow st to it.  Thread t (of 256) owns the
// eight digits below nbins - 8t, so an exclusive scan in thread order counts the
// keys with larger digits.  Every thread of the block must call it; st is the
// same in every thread before and after.
__device__ void block_pick(const unsigned* __restrict__ hist, int pass, SelectState& st) {
  __shared__ int s_digit;
  __shared__ long long s_left;
  const int shift = c_shift[pass];
  const int nbins = 1 << c_width[pass];
  const int top = nbins - 1 - 8 * static_cast<int>(threadIdx.x);
  long long h[8];
  long long mine = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    h[i] = top - i >= 0 ? hist[top - i] : 0;
    mine += h[i];
  }
  if (threadIdx.x == 0) s_digit = -1;
  long long run = block_exclusive_scan<long long>(mine, nullptr);  // has a barrier after s_digit
  const long long k_rem = st.k_rem;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (top - i >= 0 && run < k_rem && k_rem <= run + h[i]) {  // exactly one thread and digit
      s_digit = top - i;
      s_left = k_rem - run;
    }
    run += h[i];
  }
  __syncthreads();
  const int digit = s_digit;
  if (digit >= 0) {
    st.prefix |= static_cast<unsigned long long>(digit) << shift;
    st.mask |= static_cast<unsigned long long>(nbins - 1) << shift;
    st.k_rem = s_left;
  }
  __syncthreads();  // s_digit and s_left may be rewritten by the next call
}

// Unit u's G trajectories: ids id_base + u * G + g in the lists, flags at u * G + g.
__device__ __forceinline__ void write_unit(int64_t u, bool rejected, int64_t rej_pos,
                                           int64_t acc_pos, int G, int64_t id_base,
                                           int32_t* accepted_ids, int32_t* rejected_ids,
                                           uint8_t* flags) {
  for (int g = 0; g < G; ++g) {
    const int64_t id = u * G + g;
    if (rejected) {
      if (rejected_ids) rejected_ids[rej_pos * G + g] = static_cast<int32_t>(id_base + id);
    } else {
      accepted_ids[acc_pos * G + g] = static_cast<int32_t>(id_base + id);
    }
    if (flags) flags[id] = rejected ? 0 : 1;
  }
}

// U <= 512: rank of u = number of units ordered before it.  The ranks compare
// order keys, not doubles: the same order (-0.0 equals +0.0), on the integer
// pipe instead of GB300's narrow fp64 pipe.
__global__ void __launch_bounds__(kSmallThreads)
    select_small_kernel(const double* __restrict__ score, int n_units, int G, int64_t k,
                        int32_t* accepted_ids, int32_t* rejected_ids, uint8_t* flags,
                        int32_t* status) {
  __shared__ uint64_t s[kSmallMax];
  for (int u = threadIdx.x; u < n_units; u += blockDim.x) {
    const double x = score[u];
    if (isnan(x)) report(status, PACE_ERR_NAN_INPUT);
    s[u] = order_key(x);
  }
  __syncthreads();
  const int u = threadIdx.x;
  int rejected = 0;
  if (u < n_units) {
    const uint64_t x = s[u];
    int rank = 0;
    for (int w = 0; w < n_units; ++w) {
      const uint64_t y = s[w];
      rank += (y > x) || (y == x && w < u);
    }
    rejected = rank < k;
  }
  int n_rej = 0;
  const int rej_before = block_exclusive_scan<int>(rejected, &n_rej);
  if (u < n_units)
    write_unit(u, rejected, rej_before, u - rej_before, G, 0, accepted_ids, rejected_ids, flags);
}

// 512 < U <= 131,072: one launch of one thread-block cluster of C CTAs (1, 2,
// 4 or 8; 1024 threads each).  CTA r owns the contiguous units
// [r * B, r * B + B) with B = ceil(U / C) <= 16,384; its thread t owns the
// contiguous units t * per .. t * per + per - 1 of that range (per, a power of
// two, <= 16), whose order keys sit in shared memory at [i * (1024 + 1) + t], so
// a warp's accesses are conflict-free.
//
// The k-th largest key (the pivot) is found by a radix select that adapts to
// the keys.  Each round takes the minimum and maximum of the remaining
// candidates over the whole cluster, stops when they are equal, and otherwise
// histograms the (up to 11) bits just below the highest bit where they differ;
// each CTA counts its own keys and sums the C histograms through distributed
// shared memory.  Candidates in one round share every bit above that one, so a
// round fixes at least one bit and there are at most 64 rounds (two to four for
// spread-out scores).  Every CTA computes the same values from the same shared
// data, so all of them take the same branches and pass the same sequence of
// cluster barriers.
//
// Then each CTA counts its keys above and equal to the pivot, learns the
// counts of the lower-ranked CTAs (ties are rejected lowest id first), lists
// its accepted units and then its rejected units in shared memory, and writes
// its own contiguous runs of the id lists and flags, consecutive threads at
// consecutive positions (whole 32-byte sectors per warp store), four ids and
// four flags per store when G is a multiple of 4 and the buffers are aligned.
// C is the smallest power of two that keeps each CTA at 16,384 units and
// 32,768 outputs or fewer; a cluster of one uses block barriers and plain
// shared memory instead (the kMulti = false instance).
constexpr int kSelCtaUnits = 16384;  // units per CTA at most
constexpr int kSelThreads = 1024;
constexpr int kSelPer = kSelCtaUnits / kSelThreads;  // units per thread at most
constexpr int kSelMaxCluster = 8;
constexpr int64_t kSelMaxUnits = int64_t(kSelCtaUnits) * kSelMaxCluster;
constexpr int kSelRow = kSelThreads + 1;  // keys per slot row (one pad key)
static_assert(kSelPer * kSelThreads == kSelCtaUnits, "whole units per thread");
static_assert(kSelCtaUnits <= 65536, "a CTA's unit numbers are stored in 16 bits");

// log2 of the units per thread: the smallest power of two that covers b units.
__host__ __device__ inline int sel_per_log2(int b) {
  int lg = 0;
  while ((kSelThreads << lg) < b) ++lg;
  return lg;
}

// Dynamic shared memory of a CTA holding b units: keys, unit order, rejected bytes.
__host__ __device__ inline size_t sel_smem_bytes(int b) {
  return static_cast<size_t>(1 << sel_per_log2(b)) * kSelRow * sizeof(uint64_t) +
         static_cast<size_t>(b) * (sizeof(uint16_t) + 1);
}

// This CTA's minimum and maximum of (lo, hi) over its threads, written to its
// slot s_mm (read by the other CTAs).  Every thread of the block must call it;
// the caller's next block or cluster barrier publishes the slot.
__device__ __forceinline__ void cta_min_max_to_slot(uint64_t lo, uint64_t hi, uint64_t* s_wlo,
                                                    uint64_t* s_whi, uint64_t* s_mm) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t a = __shfl_xor_sync(0xffffffffu, lo, o);
    const uint64_t b = __shfl_xor_sync(0xffffffffu, hi, o);
    lo = a < lo ? a : lo;
    hi = b > hi ? b : hi;
  }
  if (lane == 0) {
    s_wlo[wid] = lo;
    s_whi[wid] = hi;
  }
  __syncthreads();
  if (wid == 0) {  // one warp folds the 32 warp results into this CTA's slot
    lo = s_wlo[lane];
    hi = s_whi[lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t a = __shfl_xor_sync(0xffffffffu, lo, o);
      const uint64_t b = __shfl_xor_sync(0xffffffffu, hi, o);
      lo = a < lo ? a : lo;
      hi = b > hi ? b : hi;
    }
    if (lane == 0) {
      s_mm[0] = lo;
      s_mm[1] = hi;
    }
  }
}

// The cluster's minimum and maximum from the CTAs' published slots, in every
// thread.  Every thread of the block must call it, after the barrier that
// published the slots.
template <bool kMulti>
__device__ __forceinline__ void cluster_fold_slots(cg::cluster_group& cluster, uint64_t& lo,
                                                   uint64_t& hi, uint64_t* s_mm, uint64_t* s_g) {
  if (!kMulti) {  // one CTA: its slot is the result
    lo = s_mm[0];
    hi = s_mm[1];
    return;
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (wid == 0) {  // lanes < C read the peers' slots; one warp folds them
    const int nc = static_cast<int>(cluster.num_blocks());
    lo = ~0ull;
    hi = 0ull;
    if (lane < nc) {
      const uint64_t* peer = cluster.map_shared_rank(s_mm, static_cast<unsigned>(lane));
      lo = peer[0];
      hi = peer[1];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t a = __shfl_xor_sync(0xffffffffu, lo, o);
      const uint64_t b = __shfl_xor_sync(0xffffffffu, hi, o);
      lo = a < lo ? a : lo;
      hi = b > hi ? b : hi;
    }
    if (lane == 0) {
      s_g[0] = lo;
      s_g[1] = hi;
    }
  }
  __syncthreads();
  lo = s_g[0];
  hi = s_g[1];
}

// kMulti = false: a cluster of one CTA, with block barriers and plain shared
// memory in place of cluster barriers and distributed shared memory.
template <bool kMulti>
__global__ void __launch_bounds__(kSelThreads, 1)
    select_cluster_kernel(const double* __restrict__ score, int n_units, int G, long long k,
                          int32_t* accepted_ids, int32_t* rejected_ids, uint8_t* flags,
                          int32_t* status, int vec4) {
  extern __shared__ __align__(16) unsigned char sel_smem[];
  __shared__ unsigned hist[kHistBins];
  __shared__ uint64_t s_wlo[kSelThreads / 32], s_whi[kSelThreads / 32];
  __shared__ uint64_t s_mm[2], s_g[2];
  __shared__ long long s_cnt[2];  // this CTA's keys equal to / above the pivot (peers read)
  __shared__ long long s_off[2];  // ties and rejections in lower-ranked CTAs
  __shared__ int s_digit;
  __shared__ long long s_left;
  cg::cluster_group cluster = cg::this_cluster();
  const int nc = static_cast<int>(cluster.num_blocks());
  const int rank = static_cast<int>(cluster.block_rank());
  const int t = threadIdx.x;
  const int B = (n_units + nc - 1) / nc;
  const int base = rank * B;                        // first unit of this CTA
  const int nb = max(0, min(B, n_units - base));    // units of this CTA
  const int lg = sel_per_log2(B);
  const int per = 1 << lg;
  uint64_t* keys = reinterpret_cast<uint64_t*>(sel_smem);
  uint16_t* order = reinterpret_cast<uint16_t*>(sel_smem + static_cast<size_t>(per) * kSelRow *
                                                               sizeof(uint64_t));
  uint8_t* rej_u = reinterpret_cast<uint8_t*>(order + B);
  const int u0 = t * per;
  const int n_mine = max(0, min(per, nb - u0));

  // coalesced loads: unit v (read by thread v % 1024) belongs to thread v / per,
  // slot v % per; the padded rows make this scatter at most two-way conflicted
  for (int v = t; v < nb; v += kSelThreads) {
    const double x = score[base + v];
    if (isnan(x)) report(status, PACE_ERR_NAN_INPUT);
    keys[(v & (per - 1)) * kSelRow + (v >> lg)] = order_key(x);
  }
  __syncthreads();
  uint64_t lo = ~0ull, hi = 0ull;
  for (int i = 0; i < n_mine; ++i) {
    const uint64_t key = keys[i * kSelRow + t];
    lo = key < lo ? key : lo;
    hi = key > hi ? key : hi;
  }
  uint64_t prefix = 0ull, mask = 0ull;
  long long k_rem = k;
  bool ok = true;
  // Each round fixes at least one more bit, so 64 rounds always suffice; the
  // bound and the digit check only guard against a broken invariant.  Every
  // branch below depends only on cluster-wide values, so it is uniform.
  // Two cluster barriers per round: one after the histograms, and one that
  // both ends the reading of the histograms and publishes the next round's
  // minimum / maximum slots (written only after every CTA has passed the
  // histogram barrier, so after every CTA has read the previous values).
  cta_min_max_to_slot(lo, hi, s_wlo, s_whi, s_mm);
  if (kMulti) cluster.sync();
  else __syncthreads();
  for (int round = 0;; ++round) {
    cluster_fold_slots<kMulti>(cluster, lo, hi, s_mm, s_g);
    if (lo == hi) break;
    if (round >= 64) {
      ok = false;
      break;
    }
    const int d = 63 - __clzll(static_cast<long long>(lo ^ hi));
    const int shift = d >= 10 ? d - 10 : 0;
    const int nbins = 1 << (d - shift + 1);
    mask = d == 63 ? 0ull : (~0ull << (d + 1));
    prefix = lo & mask;
    for (int b = t; b < nbins; b += kSelThreads) hist[b] = 0u;
    if (t == 0) s_digit = -1;
    __syncthreads();
    for (int i = 0; i < n_mine; ++i) {
      const uint64_t key = keys[i * kSelRow + t];
      if ((key & mask) == prefix)
        atomicAdd(&hist[static_cast<unsigned>(key >> shift) & (nbins - 1)], 1u);
    }
    if (kMulti) cluster.sync();  // every CTA's histogram is complete
    else __syncthreads();
    // thread t owns digits nbins-1-2t and nbins-2-2t, summed over the cluster: an
    // exclusive scan in thread order counts the candidates with larger digits
    // (the loads of all peers are issued together: a fixed-bound loop the
    // compiler unrolls, one distributed-shared-memory round trip per round)
    const int top = nbins - 1 - 2 * t;
    long long h0 = 0, h1 = 0;
    if (kMulti) {
      unsigned c0[kSelMaxCluster], c1[kSelMaxCluster];
#pragma unroll
      for (int r = 0; r < kSelMaxCluster; ++r) {
        c0[r] = 0u;
        c1[r] = 0u;
        if (r < nc) {
          const unsigned* ph = cluster.map_shared_rank(hist, static_cast<unsigned>(r));
          if (top >= 0) c0[r] = ph[top];
          if (top >= 1) c1[r] = ph[top - 1];
        }
      }
#pragma unroll
      for (int r = 0; r < kSelMaxCluster; ++r) {
        h0 += c0[r];
        h1 += c1[r];
      }
    } else {
      if (top >= 0) h0 = hist[top];
      if (top >= 1) h1 = hist[top - 1];
    }
    // every count fits 32 bits (at most kSelMaxUnits keys in the cluster)
    long long run = block_exclusive_scan<unsigned>(static_cast<unsigned>(h0 + h1), nullptr);
    if (top >= 0 && run < k_rem && k_rem <= run + h0) {
      s_digit = top;
      s_left = k_rem - run;
    }
    run += h0;
    if (top >= 1 && run < k_rem && k_rem <= run + h1) {
      s_digit = top - 1;
      s_left = k_rem - run;
    }
    __syncthreads();  // s_digit and s_left are set
    if (s_digit < 0) {  // the same in every CTA: the histograms summed are the same
      ok = false;
      break;
    }
    prefix |= static_cast<uint64_t>(s_digit) << shift;
    mask |= static_cast<uint64_t>(nbins - 1) << shift;
    k_rem = s_left;
    lo = ~0ull;
    hi = 0ull;
    for (int i = 0; i < n_mine; ++i) {
      const uint64_t key = keys[i * kSelRow + t];
      if ((key & mask) == prefix) {
        lo = key < lo ? key : lo;
        hi = key > hi ? key : hi;
      }
    }
    cta_min_max_to_slot(lo, hi, s_wlo, s_whi, s_mm);
    if (kMulti) cluster.sync();  // histograms read everywhere; the new slots published
    else __syncthreads();
  }
  if (!ok && t == 0 && rank == 0) report(status, PACE_ERR_INVALID_ARG);
  const uint64_t pivot = lo;  // k_rem of the keys equal to it are rejected, lowest ids first

  // keys equal to the pivot (high 16 bits) and above it (low 16 bits) of this
  // thread, scanned together: a CTA holds at most 16,384 keys, so neither field
  // carries into the other
  unsigned eqgt = 0u;
  for (int i = 0; i < n_mine; ++i) {
    const uint64_t key = keys[i * kSelRow + t];
    eqgt += (key == pivot ? 0x10000u : 0u) + (key > pivot ? 1u : 0u);
  }
  unsigned cta_eqgt = 0u;
  const long long tie_local = block_exclusive_scan<unsigned>(eqgt, &cta_eqgt) >> 16;
  if (t == 0) {
    s_cnt[0] = cta_eqgt >> 16;
    s_cnt[1] = cta_eqgt & 0xffffu;
  }
  if (kMulti) cluster.sync();  // every CTA's counts are written
  else __syncthreads();
  if (t < 32) {
    // lanes r < rank read CTA r's counts at once; lane 0 folds them in rank order
    long long e = 0, g = 0;
    if (kMulti && t < rank) {
      const long long* pc = cluster.map_shared_rank(s_cnt, static_cast<unsigned>(t));
      e = pc[0];
      g = pc[1];
    }
    long long ties_before = 0, rej_before = 0;
    for (int r = 0; r < kSelMaxCluster; ++r) {
      const long long er = __shfl_sync(0xffffffffu, e, r);
      const long long gr = __shfl_sync(0xffffffffu, g, r);
      if (r < (kMulti ? rank : 0)) {
        long long take = k_rem - ties_before;  // ties of CTA r that are rejected
        take = take < 0 ? 0 : (take > er ? er : take);
        rej_before += gr + take;
        ties_before += er;
      }
    }
    if (t == 0) {
      s_off[0] = ties_before;
      s_off[1] = rej_before;
    }
  }
  if (kMulti) cluster.sync();  // peers' counts are read: no CTA touches another's memory after this
  else __syncthreads();
  if (!ok) return;

  const long long tie0 = s_off[0] + tie_local;
  const long long rej_off = s_off[1];
  int nrej = 0;
  long long tie = tie0;
  for (int i = 0; i < n_mine; ++i) {
    const uint64_t key = keys[i * kSelRow + t];
    nrej += key > pivot || (key == pivot && (tie++) < k_rem);
  }
  unsigned cta_rej32 = 0u;
  long long lrpos = block_exclusive_scan<unsigned>(static_cast<unsigned>(nrej), &cta_rej32);
  const long long cta_rej = cta_rej32;
  const long long n_acc_cta = nb - cta_rej;
  tie = tie0;
  for (int i = 0; i < n_mine; ++i) {
    const uint64_t key = keys[i * kSelRow + t];
    const bool r = key > pivot || (key == pivot && (tie++) < k_rem);
    const int u = u0 + i;
    order[r ? n_acc_cta + lrpos : u - lrpos] = static_cast<uint16_t>(u);
    rej_u[u] = r ? 1 : 0;
    lrpos += r;
  }
  __syncthreads();

  // this CTA's runs: accepted ids from position (base - rej_off) * G, rejected
  // ids from rej_off * G, flags from base * G.  Local position p of the CTA's
  // [accepted | rejected] list holds trajectory (base + order[p / G]) * G + p % G;
  // (q, r) = (p / G, p % G) is advanced by 1024 per step without dividing.
  const int64_t n_out = static_cast<int64_t>(nb) * G;
  const int64_t acc_end = n_acc_cta * G;
  int32_t* acc_run = accepted_ids + (static_cast<int64_t>(base) - rej_off) * G;
  int32_t* rej_run = rejected_ids ? rejected_ids + rej_off * G : nullptr;
  if (vec4) {
    // G % 4 == 0, id lists 16-byte and flags 4-byte aligned (checked on the
    // host): four consecutive ids (one int4) and four flags (one 32-bit word)
    // per store, an eighth of the scalar writer's instructions at G = 8.  Every
    // run starts at a multiple of 4 entries.
    const int G4 = G / 4;
    const int64_t n_out4 = static_cast<int64_t>(nb) * G4;
    const int64_t acc_end4 = n_acc_cta * G4;
    int4* acc4 = reinterpret_cast<int4*>(acc_run);
    int4* rej4 = reinterpret_cast<int4*>(rej_run);
    const int sq4 = kSelThreads / G4, sr4 = kSelThreads % G4;
    int q = t / G4, r = t % G4;
    for (int64_t p = t; p < n_out4; p += kSelThreads) {
      const int32_t id = (base + static_cast<int32_t>(order[q])) * G + 4 * r;
      const int4 v = make_int4(id, id + 1, id + 2, id + 3);
      if (p < acc_end4) acc4[p] = v;
      else if (rej4) rej4[p - acc_end4] = v;
      q += sq4;
      r += sr4;
      if (r >= G4) {
        r -= G4;
        ++q;
      }
    }
    if (flags) {
      uint32_t* f4 = reinterpret_cast<uint32_t*>(flags + static_cast<int64_t>(base) * G);
      q = t / G4;
      r = t % G4;
      for (int64_t p = t; p < n_out4; p += kSelThreads) {
        f4[p] = rej_u[q] ? 0u : 0x01010101u;
        q += sq4;
        r += sr4;
        if (r >= G4) {
          r -= G4;
          ++q;
        }
      }
    }
    return;
  }
  const int sq = kSelThreads / G, sr = kSelThreads % G;
  int q = t / G, r = t % G;
  for (int64_t p = t; p < n_out; p += kSelThreads) {
    const int32_t id = (base + static_cast<int32_t>(order[q])) * G + r;
    if (p < acc_end) acc_run[p] = id;
    else if (rej_run) rej_run[p - acc_end] = id;
    q += sq;
    r += sr;
    if (r >= G) {
      r -= G;
      ++q;
    }
  }
  if (flags) {
    uint8_t* f_run = flags + static_cast<int64_t>(base) * G;
    q = t / G;
    r = t % G;
    for (int64_t p = t; p < n_out; p += kSelThreads) {
      f_run[p] = rej_u[q] ? 0 : 1;
      q += sq;
      r += sr;
      if (r >= G) {
        r -= G;
        ++q;
      }
    }
  }
}

// Pass `pass` of the MSB-first radix select (256 threads per block).  The state
// it filters with is the previous pass's result, which every block derives
// from the previous histogram (block 0 stores it for the next pass), so the
// passes need no separate pick launches.  Histograms rotate through three
// buffers: pass p adds into hist[p % 3], reads hist[(p - 1) % 3] and clears
// hist[(p + 1) % 3] (last read by pass p - 1) for pass p + 1.  State slots
// alternate: pass p reads slot (p - 1) & 1 and writes slot p & 1.
//
// hist_prev is the previous pass's histogram (unused at pass 0), hist_out the
// cleared histogram this pass adds into, hist_clear (or null) a histogram to
// clear for the next pass.  The sharded entry points pass the caller's
// histograms, summed over the ranks between passes.
__global__ void __launch_bounds__(256)
    radix_pass_kernel(const double* __restrict__ score, int64_t n_units, int pass,
                      SelectState* states, const unsigned* hist_prev, unsigned* hist_out,
                      unsigned* hist_clear, int32_t* status) {
  __shared__ unsigned h[kHistBins];
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x) h[b] = 0;
  SelectState st = states[pass == 0 ? 0 : (pass - 1) & 1];
  if (pass > 0) {
    block_pick(hist_prev, pass - 1, st);
    if (blockIdx.x == 0 && threadIdx.x == 0) states[pass & 1] = st;
  }
  if (hist_clear)
    for (int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; b < kHistBins;
         b += static_cast<int64_t>(gridDim.x) * blockDim.x)
      hist_clear[b] = 0u;
  __syncthreads();
  const unsigned long long prefix = st.prefix, mask = st.mask;
  const int shift = c_shift[pass];
  const unsigned dmask = (1u << c_width[pass]) - 1u;
  for (int64_t u = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; u < n_units;
       u += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const double x = score[u];
    if (pass == 0 && isnan(x)) report(status, PACE_ERR_NAN_INPUT);
    const uint64_t key = order_key(x);
    if ((key & mask) == prefix) atomicAdd(&h[(key >> shift) & dmask], 1u);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < kHistBins; b += blockDim.x)
    if (h[b]) atomicAdd(&hist_out[b], h[b]);
}

// Phase 1: per tile, units equal to the pivot and above it.  The pivot is the
// last pass's result, derived here from its histogram (block 0 stores it in
// state slot kPasses & 1 for the later phases).
__global__ void __launch_bounds__(kTileThreads)
    count_tile_kernel(const double* __restrict__ score, int64_t n_units, SelectState* states,
                      const unsigned* hist_last, int* eq_cnt, int* gt_cnt) {
  SelectState st = states[(kPasses - 1) & 1];
  block_pick(hist_last, kPasses - 1, st);
  if (blockIdx.x == 0 && threadIdx.x == 0) states[kPasses & 1] = st;
  const unsigned long long pivot = st.prefix;
  int eq = 0, gt = 0;
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kTile + threadIdx.x * kPerThread;
  for (int i = 0; i < kPerThread; ++i) {
    const int64_t u = base + i;
    if (u < n_units) {
      const uint64_t key = order_key(score[u]);
      eq += key == pivot;
      gt += key > pivot;
    }
  }
  int te = 0, tg = 0;
  block_exclusive_scan<int>(eq, &te);
  block_exclusive_scan<int>(gt, &tg);
  if (threadIdx.x == 0) {
    eq_cnt[blockIdx.x] = te;
    gt_cnt[blockIdx.x] = tg;
  }
}

// Phase 2 (one block): per tile, ties before it and rejections before it.
// eq_start (or null = 0) counts the ties at the pivot held before this pool's
// first unit (on lower ranks of a sharded pool); rej_total (or null) receives
// the number of units rejected here.
__global__ void __launch_bounds__(1024)
    scan_tiles_kernel(int n_tiles, const SelectState* __restrict__ state, const int* eq_cnt,
                      const int* gt_cnt, long long* eq_before, long long* rej_before,
                      const long long* eq_start, long long* rej_total) {
  __shared__ long long carry_eq, carry_rej;
  if (threadIdx.x == 0) {
    carry_eq = eq_start ? *eq_start : 0;
    carry_rej = 0;
  }
  __syncthreads();
  const long long k_rem = state->k_rem;
  for (int t0 = 0; t0 < n_tiles; t0 += blockDim.x) {
    const int t = t0 + threadIdx.x;
    const int e = t < n_tiles ? eq_cnt[t] : 0;
    int te = 0;
    const int eb = block_exclusive_scan<int>(e, &te);
    const long long eq_b = carry_eq + eb;
    long long take = k_rem - eq_b;
    take = take < 0 ? 0 : (take > e ? e : take);
    const int r = t < n_tiles ? gt_cnt[t] + static_cast<int>(take) : 0;
    int tr = 0;
    const int rb = block_exclusive_scan<int>(r, &tr);
    if (t < n_tiles) {
      eq_before[t] = eq_b;
      rej_before[t] = carry_rej + rb;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      carry_eq += te;
      carry_rej += tr;
    }
    __syncthreads();
  }
  if (rej_total && threadIdx.x == 0) *rej_total = carry_rej;
}

// Phase 3: flags and output positions inside each tile.
__global__ void __launch_bounds__(kTileThreads)
    write_tile_kernel(const double* __restrict__ score, int64_t n_units, int G, int64_t id_base,
                      const SelectState* __restrict__ state, const long long* eq_before,
                      const long long* rej_before, int32_t* accepted_ids,
                      int32_t* rejected_ids, uint8_t* flags) {
  const unsigned long long pivot = state->prefix;
  const long long k_rem = state->k_rem;
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kTile + threadIdx.x * kPerThread;
  uint64_t keys[kPerThread];
  int eq = 0;
  for (int i = 0; i < kPerThread; ++i) {
    const int64_t u = base + i;
    keys[i] = u < n_units ? order_key(score[u]) : 0;
    eq += (u < n_units) && keys[i] == pivot;
  }
  const long long tie0 = eq_before[blockIdx.x] + block_exclusive_scan<int>(eq, nullptr);
  bool rej[kPerThread];
  int nrej = 0;
  long long tie = tie0;
  for (int i = 0; i < kPerThread; ++i) {
    const int64_t u = base + i;
    bool r = false;
    if (u < n_units) {
      if (keys[i] > pivot) r = true;
      else if (keys[i] == pivot) r = (tie++) < k_rem;
    }
    rej[i] = r;
    nrej += r;
  }
  long long rpos = rej_before[blockIdx.x] + block_exclusive_scan<int>(nrej, nullptr);
  for (int i = 0; i < kPerThread; ++i) {
    const int64_t u = base + i;
    if (u >= n_units) break;
    const long long apos = u - rpos;
    write_unit(u, rej[i], rpos, apos, G, id_base, accepted_ids, rejected_ids, flags);
    rpos += rej[i];
  }
}

__global__ void fill_identity_kernel(int64_t n_units, int G, bool accept, int64_t id_base,
                                     int32_t* accepted_ids, int32_t* rejected_ids,
                                     uint8_t* flags) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_units * G;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (accept) accepted_ids[i] = static_cast<int32_t>(id_base + i);
    else if (rejected_ids) rejected_ids[i] = static_cast<int32_t>(id_base + i);
    if (flags) flags[i] = accept ? 1 : 0;
  }
}

__global__ void nan_check_kernel(const double* __restrict__ score, int64_t n, int32_t* status) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    if (isnan(score[i])) report(status, PACE_ERR_NAN_INPUT);
}

struct SelectWs {
  SelectState* states;  // two slots, alternating between passes
  unsigned* hist;       // three rotating histograms of kHistBins
  int* eq_cnt;
  int* gt_cnt;
  long long* eq_before;
  long long* rej_before;
};

SelectWs carve_select_ws(Carver& cv, int64_t n_units) {
  const int64_t n_tiles = (n_units + kTile - 1) / kTile;
  SelectWs w;
  w.states = cv.take<SelectState>(2);
  w.hist = cv.take<unsigned>(3 * kHistBins);
  w.eq_cnt = cv.take<int>(n_tiles);
  w.gt_cnt = cv.take<int>(n_tiles);
  w.eq_before = cv.take<long long>(n_tiles);
  w.rej_before = cv.take<long long>(n_tiles);
  return w;
}

// Opts select_cluster_kernel into its largest dynamic shared memory and finds
// the largest cluster (8, 4, 2 or 1 CTAs) of such blocks the current device can
// hold, once per device.
pace_status sel_cluster_limit(int* out) {
  constexpr int kMaxDevices = 64;
  static int limit[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  PACE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_CUDA;
  std::lock_guard<std::mutex> g(mu);
  if (limit[dev] == 0) {
    const size_t smem = sel_smem_bytes(kSelCtaUnits);
    PACE_TRY_CUDA(cudaFuncSetAttribute(select_cluster_kernel<true>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem)));
    PACE_TRY_CUDA(cudaFuncSetAttribute(select_cluster_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem)));
    int c = kSelMaxCluster;
    for (; c > 1; c /= 2) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(static_cast<unsigned>(c), 1, 1);
      cfg.blockDim = dim3(kSelThreads, 1, 1);
      cfg.dynamicSmemBytes = smem;
      cudaLaunchAttribute attr;
      attr.id = cudaLaunchAttributeClusterDimension;
      attr.val.clusterDim.x = static_cast<unsigned>(c);
      attr.val.clusterDim.y = 1;
      attr.val.clusterDim.z = 1;
      cfg.attrs = &attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, select_cluster_kernel<true>, &cfg) == cudaSuccess &&
          n >= 1)
        break;
      (void)cudaGetLastError();  // a refused size is not an error of this call
    }
    limit[dev] = c;
  }
  *out = limit[dev];
  return PACE_OK;
}

// Cluster size for U units of G trajectories: enough CTAs to hold the keys
// (16,384 each) and one more SM per doubling of the outputs above 32,768, up to
// the device's limit; 0 when the keys do not fit the largest cluster.  Fewer
// CTAs mean cheaper cluster barriers and fewer distributed-shared-memory reads
// per round; more spread the writing of the id lists.  On the 16,384 groups of
// the 128k sweep pool (131,072 outputs) 4 CTAs took 331.5 us per scoring +
// selection call against 336 with 8 and 336 with 2 (CUDA-graph replays).
int sel_cluster_size(int64_t n_units, int G, int limit) {
  const int64_t total = n_units * G;
  int c = 1;
  while (c < limit && (n_units > static_cast<int64_t>(c) * kSelCtaUnits ||
                       total > static_cast<int64_t>(c) * 32768))
    c *= 2;
  return n_units <= static_cast<int64_t>(c) * kSelCtaUnits ? c : 0;
}

pace_status launch_select_cluster(const double* unit_score, int n_units, int G, long long k,
                                  int c, int32_t* accepted_ids, int32_t* rejected_ids,
                                  uint8_t* flags, int32_t* status, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(c), 1, 1);
  cfg.blockDim = dim3(kSelThreads, 1, 1);
  cfg.dynamicSmemBytes = sel_smem_bytes((n_units + c - 1) / c);
  cfg.stream = st;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = static_cast<unsigned>(c);
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  const int vec4 = G % 4 == 0 && aligned(accepted_ids, 16) &&
                   (!rejected_ids || aligned(rejected_ids, 16)) && (!flags || aligned(flags, 4));
  if (c > 1) {
    PACE_TRY_CUDA(cudaLaunchKernelEx(&cfg, select_cluster_kernel<true>, unit_score, n_units, G,
                                     k, accepted_ids, rejected_ids, flags, status, vec4));
  } else {
    PACE_TRY_CUDA(cudaLaunchKernelEx(&cfg, select_cluster_kernel<false>, unit_score, n_units, G,
                                     k, accepted_ids, rejected_ids, flags, status, vec4));
  }
  return last_launch_status();
}

int grid_for(int64_t n, int threads, int per_sm) {
  int64_t b = (n + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;
  if (b > cap) b = cap;
  if (b < 1) b = 1;
  return static_cast<int>(b);
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" void pace_budget_params_default(PaceBudgetParams* p) {
  if (!p) return;
  p->n_target = 0;
  p->beta = 0.0;
  p->r_max = 0.9;
  p->r_hat_prev = 0.0;
}

extern "C" pace_status pace_budget(int64_t n_traj, int64_t n_units, const PaceBudgetParams* p,
                                   double* r_out, double* r_hat_out, int64_t* k_units_out) {
  if (!p || !r_hat_out || !k_units_out) return PACE_ERR_INVALID_ARG;
  if (n_traj < 0 || n_units < 0 || p->n_target < 0) return PACE_ERR_INVALID_ARG;
  if (!(p->beta >= 0.0 && p->beta < 1.0)) return PACE_ERR_INVALID_ARG;
  if (!(p->r_max >= 0.0 && p->r_max <= 1.0)) return PACE_ERR_INVALID_ARG;
  if (!(p->r_hat_prev >= 0.0 && p->r_hat_prev <= 1.0)) return PACE_ERR_INVALID_ARG;
  // Eq. 3: surplus fraction of the pool above its target occupancy
  const int64_t denom = n_traj > 1 ? n_traj : 1;
  volatile double r = static_cast<double>(n_traj - p->n_target) / static_cast<double>(denom);
  double rr = r;
  if (rr < 0.0) rr = 0.0;
  if (rr > 1.0) rr = 1.0;
  // Eq. 4: EMA smoothing; each product rounded on its own (no contraction)
  volatile double t1 = p->beta * p->r_hat_prev;
  volatile double one_minus_beta = 1.0 - p->beta;
  volatile double t2 = one_minus_beta * rr;
  const double r_hat = t1 + t2;
  const double r_eff = r_hat < p->r_max ? r_hat : p->r_max;
  volatile double prod = r_eff * static_cast<double>(n_units);
  int64_t k = static_cast<int64_t>(floor(prod + 1e-9));
  if (k > n_units) k = n_units;
  if (k < 0) k = 0;
  if (r_out) *r_out = rr;
  *r_hat_out = r_hat;
  *k_units_out = k;
  return PACE_OK;
}

extern "C" size_t pace_select_workspace_size(int64_t n_units) {
  if (n_units < 0) return 0;
  Carver cv;
  carve_select_ws(cv, n_units);
  return cv.used;
}

extern "C" pace_status pace_select_k(const double* unit_score, int64_t n_units, int32_t group_size,
                                     int64_t k, int32_t* accepted_ids, int32_t* rejected_ids,
                                     uint8_t* traj_accepted, void* workspace,
                                     size_t workspace_bytes, int32_t* status_dev, void* stream) {
  if (n_units < 0 || group_size < 1 || k < 0 || k > n_units) return PACE_ERR_INVALID_ARG;
  if (n_units > (int64_t(1) << 30) ||
      n_units * static_cast<int64_t>(group_size) > (int64_t(1) << 31) - 1)
    return PACE_ERR_INVALID_ARG;
  if (n_units == 0) return PACE_OK;
  if (!unit_score || (!accepted_ids && k < n_units)) return PACE_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const int G = group_size;
  if (k == 0 || k == n_units) {
    nan_check_kernel<<<grid_for(n_units, 256, 4), 256, 0, st>>>(unit_score, n_units, status_dev);
    PACE_TRY(last_launch_status());
    fill_identity_kernel<<<grid_for(n_units * G, 256, 8), 256, 0, st>>>(
        n_units, G, k == 0, 0, accepted_ids, rejected_ids, traj_accepted);
    return last_launch_status();
  }
  if (n_units <= kSmallMax) {
    select_small_kernel<<<1, kSmallThreads, 0, st>>>(unit_score, static_cast<int>(n_units), G, k,
                                                     accepted_ids, rejected_ids, traj_accepted,
                                                     status_dev);
    return last_launch_status();
  }
  if (n_units <= kSelMaxUnits) {
    int limit = 1;
    PACE_TRY(sel_cluster_limit(&limit));
    const int c = sel_cluster_size(n_units, G, limit);
    if (c > 0)
      return launch_select_cluster(unit_score, static_cast<int>(n_units), G,
                                   static_cast<long long>(k), c, accepted_ids, rejected_ids,
                                   traj_accepted, status_dev, st);
  }
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  SelectWs ws = carve_select_ws(cv, n_units);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  select_init_kernel<<<1, 256, 0, st>>>(ws.states, static_cast<long long>(k), ws.hist);
  PACE_TRY(last_launch_status());
  const int hist_grid = grid_for(n_units, 256, 2);
  // histograms rotate through three buffers: pass p adds into hist[p % 3],
  // reads hist[(p - 1) % 3] and clears hist[(p + 1) % 3] (last read by pass p - 1)
  for (int pass = 0; pass < kPasses; ++pass) {
    radix_pass_kernel<<<hist_grid, 256, 0, st>>>(
        unit_score, n_units, pass, ws.states, ws.hist + ((pass + 2) % 3) * kHistBins,
        ws.hist + (pass % 3) * kHistBins, ws.hist + ((pass + 1) % 3) * kHistBins, status_dev);
    PACE_TRY(last_launch_status());
  }
  const int64_t n_tiles = (n_units + kTile - 1) / kTile;
  const SelectState* final_state = ws.states + (kPasses & 1);
  count_tile_kernel<<<static_cast<unsigned>(n_tiles), kTileThreads, 0, st>>>(
      unit_score, n_units, ws.states, ws.hist + ((kPasses - 1) % 3) * kHistBins, ws.eq_cnt,
      ws.gt_cnt);
  PACE_TRY(last_launch_status());
  scan_tiles_kernel<<<1, 1024, 0, st>>>(static_cast<int>(n_tiles), final_state, ws.eq_cnt,
                                        ws.gt_cnt, ws.eq_before, ws.rej_before, nullptr, nullptr);
  PACE_TRY(last_launch_status());
  write_tile_kernel<<<static_cast<unsigned>(n_tiles), kTileThreads, 0, st>>>(
      unit_score, n_units, G, 0, final_state, ws.eq_before, ws.rej_before, accepted_ids,
      rejected_ids, traj_accepted);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// Sharded rejection (the pool's units partitioned across ranks in contiguous
// id ranges).  The rule is unchanged: the k top-scored units of the WHOLE pool
// are rejected, ties lowest id first (Sec. 3.1, Algorithm 1).  The radix
// select above runs on each shard with the histogram of every pass summed over
// the ranks by the caller between the calls; then each shard counts its units
// tied at the pivot, the caller turns those counts into the ties held by lower
// ranks, and each shard writes its own id lists.
// ---------------------------------------------------------------------------

namespace pace {
namespace {

struct ShardWs {
  SelectState* states;  // two slots, alternating between passes
  int* eq_cnt;
  int* gt_cnt;
  long long* eq_before;
  long long* rej_before;
};

ShardWs carve_shard_ws(Carver& cv, int64_t n_units) {
  const int64_t n_tiles = (n_units + kTile - 1) / kTile;
  const int64_t t = n_tiles > 0 ? n_tiles : 1;
  ShardWs w;
  w.states = cv.take<SelectState>(2);
  w.eq_cnt = cv.take<int>(t);
  w.gt_cnt = cv.take<int>(t);
  w.eq_before = cv.take<long long>(t);
  w.rej_before = cv.take<long long>(t);
  return w;
}

pace_status shard_ws(void* workspace, size_t bytes, int64_t n_units, ShardWs* out) {
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, bytes);
  *out = carve_shard_ws(cv, n_units);
  return cv.fits() ? PACE_OK : PACE_ERR_WORKSPACE;
}

// A shard's number of units tied at the pivot: the sum of the per-tile counts.
__global__ void tile_total_kernel(int n_tiles, const int* __restrict__ cnt,
                                  long long* __restrict__ total) {
  __shared__ long long sh[1024];
  long long a = 0;
  for (int t = threadIdx.x; t < n_tiles; t += blockDim.x) a += cnt[t];
  sh[threadIdx.x] = a;
  __syncthreads();
  for (int o = 512; o > 0; o >>= 1) {
    if (static_cast<int>(threadIdx.x) < o) sh[threadIdx.x] += sh[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) *total = sh[0];
}

bool shard_shape_ok(int64_t n_units) { return n_units >= 0 && n_units <= (int64_t(1) << 30); }

}  // namespace
}  // namespace pace

extern "C" size_t pace_select_shard_workspace_size(int64_t n_units) {
  if (!shard_shape_ok(n_units)) return 0;
  Carver cv;
  carve_shard_ws(cv, n_units);
  return cv.used;
}

extern "C" pace_status pace_select_shard_pass(const double* unit_score, int64_t n_units,
                                              int32_t pass, int64_t k_units,
                                              const uint32_t* hist_prev, uint32_t* hist_out,
                                              void* workspace, size_t workspace_bytes,
                                              int32_t* status_dev, void* stream) {
  if (!shard_shape_ok(n_units) || pass < 0 || pass >= kPasses || k_units < 0 || !hist_out ||
      (pass > 0 && !hist_prev) || (n_units > 0 && !unit_score))
    return PACE_ERR_INVALID_ARG;
  ShardWs ws;
  PACE_TRY(shard_ws(workspace, workspace_bytes, n_units, &ws));
  cudaStream_t st = as_stream(stream);
  unsigned* out = reinterpret_cast<unsigned*>(hist_out);
  if (pass == 0) {
    select_init_kernel<<<1, 256, 0, st>>>(ws.states, static_cast<long long>(k_units), out);
    PACE_TRY(last_launch_status());
  } else {
    PACE_TRY_CUDA(cudaMemsetAsync(out, 0, kHistBins * sizeof(unsigned), st));
  }
  radix_pass_kernel<<<grid_for(n_units, 256, 2), 256, 0, st>>>(
      unit_score, n_units, pass, ws.states, reinterpret_cast<const unsigned*>(hist_prev), out,
      nullptr, status_dev);
  return last_launch_status();
}

extern "C" pace_status pace_select_shard_ties(const double* unit_score, int64_t n_units,
                                              const uint32_t* hist_last, int64_t* n_tied_out,
                                              void* workspace, size_t workspace_bytes,
                                              int32_t* status_dev, void* stream) {
  (void)status_dev;
  if (!shard_shape_ok(n_units) || !hist_last || !n_tied_out || (n_units > 0 && !unit_score))
    return PACE_ERR_INVALID_ARG;
  ShardWs ws;
  PACE_TRY(shard_ws(workspace, workspace_bytes, n_units, &ws));
  cudaStream_t st = as_stream(stream);
  long long* tied = reinterpret_cast<long long*>(n_tied_out);
  if (n_units == 0) {
    PACE_TRY_CUDA(cudaMemsetAsync(tied, 0, sizeof(long long), st));
    return PACE_OK;
  }
  const int64_t n_tiles = (n_units + kTile - 1) / kTile;
  count_tile_kernel<<<static_cast<unsigned>(n_tiles), kTileThreads, 0, st>>>(
      unit_score, n_units, ws.states, reinterpret_cast<const unsigned*>(hist_last), ws.eq_cnt,
      ws.gt_cnt);
  PACE_TRY(last_launch_status());
  tile_total_kernel<<<1, 1024, 0, st>>>(static_cast<int>(n_tiles), ws.eq_cnt, tied);
  return last_launch_status();
}

extern "C" pace_status pace_select_shard_write(const double* unit_score, int64_t n_units,
                                               int32_t group_size, int64_t k_units,
                                               const int64_t* tied_before, int64_t id_base,
                                               int32_t* accepted_ids, int32_t* rejected_ids,
                                               uint8_t* traj_accepted, int64_t* n_rejected_out,
                                               void* workspace, size_t workspace_bytes,
                                               int32_t* status_dev, void* stream) {
  (void)status_dev;
  if (!shard_shape_ok(n_units) || group_size < 1 || k_units < 0 || id_base < 0 || !tied_before)
    return PACE_ERR_INVALID_ARG;
  if (id_base + n_units * static_cast<int64_t>(group_size) > (int64_t(1) << 31) - 1)
    return PACE_ERR_INVALID_ARG;
  if (n_units > 0 && (!unit_score || !accepted_ids)) return PACE_ERR_INVALID_ARG;
  ShardWs ws;
  PACE_TRY(shard_ws(workspace, workspace_bytes, n_units, &ws));
  cudaStream_t st = as_stream(stream);
  long long* n_rej = reinterpret_cast<long long*>(n_rejected_out);
  if (n_units == 0 || k_units == 0) {
    if (n_rej) PACE_TRY_CUDA(cudaMemsetAsync(n_rej, 0, sizeof(long long), st));
    if (n_units == 0) return PACE_OK;
    fill_identity_kernel<<<grid_for(n_units * group_size, 256, 8), 256, 0, st>>>(
        n_units, group_size, true, id_base, accepted_ids, rejected_ids, traj_accepted);
    return last_launch_status();
  }
  const int64_t n_tiles = (n_units + kTile - 1) / kTile;
  const SelectState* final_state = ws.states + (kPasses & 1);
  scan_tiles_kernel<<<1, 1024, 0, st>>>(static_cast<int>(n_tiles), final_state, ws.eq_cnt,
                                        ws.gt_cnt, ws.eq_before, ws.rej_before,
                                        reinterpret_cast<const long long*>(tied_before), n_rej);
  PACE_TRY(last_launch_status());
  write_tile_kernel<<<static_cast<unsigned>(n_tiles), kTileThreads, 0, st>>>(
      unit_score, n_units, group_size, id_base, final_state, ws.eq_before, ws.rej_before,
      accepted_ids, rejected_ids, traj_accepted);
  return last_launch_status();
}

extern "C" pace_status pace_select(const double* unit_score, int64_t n_units, int32_t group_size,
                                   const PaceBudgetParams* budget, double* r_hat_out,
                                   int64_t* k_units_out, int32_t* accepted_ids,
                                   int32_t* rejected_ids, uint8_t* traj_accepted,
                                   void* workspace, size_t workspace_bytes, int32_t* status_dev,
                                   void* stream) {
  if (!budget || !r_hat_out || !k_units_out || group_size < 1 || n_units < 0)
    return PACE_ERR_INVALID_ARG;
  double r_hat = 0.0;
  int64_t k = 0;
  PACE_TRY(pace_budget(n_units * static_cast<int64_t>(group_size), n_units, budget, nullptr,
                       &r_hat, &k));
  PACE_TRY(pace_select_k(unit_score, n_units, group_size, k, accepted_ids, rejected_ids,
                         traj_accepted, workspace, workspace_bytes, status_dev, stream));
  *r_hat_out = r_hat;
  *k_units_out = k;
  return PACE_OK;
}

// ---------------------------------------------------------------------------
// Staleness diagnostics: histograms of a per-unit value for rejected and
// accepted units (the paper's retained-vs-rejected admission analysis).
// ---------------------------------------------------------------------------

namespace pace {
namespace {

constexpr int kMaxHistBins = 4096;

__global__ void staleness_hist_kernel(const double* __restrict__ values,
                                      const uint8_t* __restrict__ flags, int64_t n, double lo,
                                      double hi, int n_bins, unsigned* __restrict__ hist,
                                      int32_t* status) {
  extern __shared__ unsigned h[];  // [2 * n_bins]
  for (int b = threadIdx.x; b < 2 * n_bins; b += blockDim.x) h[b] = 0;
  __syncthreads();
  const double width = __dsub_rn(hi, lo);
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const double x = values[i];
    if (isnan(x)) {
      report(status, PACE_ERR_NAN_INPUT);
      continue;
    }
    int b;
    if (x < lo) b = 0;
    else if (x >= hi) b = n_bins - 1;
    else {
      const double f = floor(__dmul_rn(__ddiv_rn(__dsub_rn(x, lo), width), (double)n_bins));
      b = f > (double)(n_bins - 1) ? n_bins - 1 : static_cast<int>(f);
    }
    atomicAdd(&h[(flags && flags[i] ? n_bins : 0) + b], 1u);
  }
  __syncthreads();
  for (int b = threadIdx.x; b < 2 * n_bins; b += blockDim.x)
    if (h[b]) atomicAdd(&hist[b], h[b]);
}

}  // namespace
}  // namespace pace

extern "C" pace_status pace_staleness_histogram(const double* values, const uint8_t* flags,
                                                int64_t n, double lo, double hi, int32_t n_bins,
                                                uint32_t* hist, int32_t* status_dev,
                                                void* stream) {
  if (n < 0 || n_bins < 1 || n_bins > kMaxHistBins || !(hi > lo) || !isfinite(lo) ||
      !isfinite(hi) || !hist || (n > 0 && !values))
    return PACE_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  PACE_TRY_CUDA(cudaMemsetAsync(hist, 0, sizeof(uint32_t) * 2 * n_bins, st));
  if (n == 0) return PACE_OK;
  staleness_hist_kernel<<<grid_for(n, 256, 4), 256, sizeof(unsigned) * 2 * n_bins, st>>>(
      values, flags, n, lo, hi, n_bins, hist, status_dev);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// The literal sliding-window quantile rule (Sec. 3.1, Algorithm 1).
// ---------------------------------------------------------------------------

namespace pace {
namespace {

constexpr int kMaxWindowSlots = 4096;
constexpr int kAdmitThreads = 1024;

// One block: sort the window's recent scores in shared memory (bitonic, +inf
// padding), take the inverted-CDF (1 - r) quantile, decide the candidates in
// draw order with block scans, then append the drawn scores to the ring.
__global__ void __launch_bounds__(kAdmitThreads)
    quantile_admit_kernel(const double* __restrict__ score, int64_t n_cand, double r,
                          int64_t batch_units, int32_t min_obs, double* __restrict__ window,
                          int64_t capacity, long long* __restrict__ state,
                          uint8_t* __restrict__ decision, double* __restrict__ kappa_out,
                          int32_t* status) {
  __shared__ double sw[kMaxWindowSlots];
  __shared__ long long s_retained, s_drawn;
  const long long n = state[0], head = state[1];
  if (n < 0 || n > capacity || head < 0 || head >= capacity) {
    if (threadIdx.x == 0) report(status, PACE_ERR_INVALID_ARG);
    return;
  }
  double kappa = __longlong_as_double(0x7ff0000000000000ll);  // +inf: no threshold
  if (n > 0 && n >= min_obs) {
    int pw = 1;
    while (pw < n) pw <<= 1;
    for (int t = threadIdx.x; t < pw; t += blockDim.x)
      sw[t] = t < n ? window[(head - n + t + capacity) % capacity]
                    : __longlong_as_double(0x7ff0000000000000ll);
    __syncthreads();
    for (int size = 2; size <= pw; size <<= 1) {
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int t = threadIdx.x; t < pw; t += blockDim.x) {
          const int u = t ^ stride;
          if (u > t) {
            const bool up = (t & size) == 0;
            const double a = sw[t], b = sw[u];
            if ((a > b) == up) {
              sw[t] = b;
              sw[u] = a;
            }
          }
        }
        __syncthreads();
      }
    }
    long long k = static_cast<long long>(
        ceil(__dsub_rn(__dmul_rn(__dsub_rn(1.0, r), static_cast<double>(n)), 1e-9)));
    if (k < 1) k = 1;
    if (k > n) k = n;
    kappa = sw[k - 1];
  }
  if (threadIdx.x == 0) {
    s_retained = 0;
    s_drawn = 0;
    *kappa_out = kappa;
  }
  __syncthreads();
  for (int64_t c0 = 0; c0 < n_cand; c0 += blockDim.x) {
    const int64_t i = c0 + threadIdx.x;
    const double x = i < n_cand ? score[i] : 0.0;
    if (i < n_cand && isnan(x)) report(status, PACE_ERR_NAN_INPUT);
    const int keep = (i < n_cand && !(x > kappa)) ? 1 : 0;
    int tot = 0;
    const int before = block_exclusive_scan<int>(keep, &tot);
    const long long ret0 = s_retained;
    if (i < n_cand) {
      const bool drawn = batch_units <= 0 || ret0 + before < batch_units;
      decision[i] = drawn ? (keep ? 1 : 0) : 2;
    }
    int last_drawn = -1;  // last candidate of this chunk that was drawn
    if (i < n_cand && (batch_units <= 0 || ret0 + before < batch_units))
      last_drawn = threadIdx.x;
    int chunk_drawn = 0;
    block_exclusive_scan<int>(last_drawn >= 0 ? 1 : 0, &chunk_drawn);
    __syncthreads();
    if (threadIdx.x == 0) {
      s_retained = ret0 + tot;
      s_drawn += chunk_drawn;
    }
    __syncthreads();
  }
  // append the drawn scores (in draw order) to the ring; when more were drawn
  // than the ring holds, only the newest `capacity` of them survive
  const long long drawn = s_drawn;
  const long long keep_n = drawn < capacity ? drawn : capacity;
  for (long long t = drawn - keep_n + threadIdx.x; t < drawn; t += blockDim.x)
    window[(head + t) % capacity] = score[t];
  __syncthreads();
  if (threadIdx.x == 0) {
    state[1] = (head + drawn) % capacity;
    state[0] = n + drawn < capacity ? n + drawn : capacity;
  }
}

}  // namespace
}  // namespace pace

extern "C" pace_status pace_quantile_admit(const double* unit_score, int64_t n_cand,
                                           double r_hat, int64_t batch_units, int32_t min_obs,
                                           double* window, int64_t capacity,
                                           int64_t* window_state, uint8_t* decision,
                                           double* kappa, int32_t* status_dev, void* stream) {
  if (n_cand < 0 || capacity < 1 || capacity > pace::kMaxWindowSlots || !window ||
      !window_state || !kappa || (n_cand > 0 && (!unit_score || !decision)))
    return PACE_ERR_INVALID_ARG;
  if (!(r_hat >= 0.0 && r_hat <= 1.0)) return PACE_ERR_INVALID_ARG;
  pace::quantile_admit_kernel<<<1, pace::kAdmitThreads, 0, pace::as_stream(stream)>>>(
      unit_score, n_cand, r_hat, batch_units, min_obs, window, capacity,
      reinterpret_cast<long long*>(window_state), decision, kappa, status_dev);
  return pace::last_launch_status();
}

// ---------------------------------------------------------------------------
// Selection without a caller-provided workspace.
//
// For callers that may not allocate device memory themselves, the radix path's
// scratch lives in this file-scope array instead of a workspace.  Every GPU
// that loads the library holds it (128 KB) until the process exits; every call
// on a device shares it, so calls that overlap on that device race.
// ---------------------------------------------------------------------------

namespace {

constexpr int64_t kNoAllocMaxUnits = int64_t(1) << 20;
constexpr size_t kNoAllocScratchBytes = 131072;

}  // namespace

static __device__ __align__(256) unsigned char g_select_scratch[kNoAllocScratchBytes];

namespace {

// Device address of g_select_scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is asked from the
// runtime once per device (with that device current) and cached.  The cached
// address belongs to the device's context at that time; after cudaDeviceReset
// the entry point is not to be used again in the process (stated in pace.h).
pace_status select_scratch_address(void** out) {
  constexpr int kMaxDevices = 64;
  static void* addr[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  PACE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_CUDA;
  std::lock_guard<std::mutex> g(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_scratch) != cudaSuccess || !p) return PACE_ERR_CUDA;
    addr[dev] = p;
  }
  *out = addr[dev];
  return PACE_OK;
}

}  // namespace

extern "C" pace_status pace_select_k_noalloc(const double* unit_score, int64_t n_units,
                                             int32_t group_size, int64_t k_units,
                                             int32_t* accepted_ids, int32_t* rejected_ids,
                                             uint8_t* traj_accepted, int32_t* status_dev,
                                             void* stream) {
  if (n_units > kNoAllocMaxUnits) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (pace_select_workspace_size(n_units) > kNoAllocScratchBytes) return PACE_ERR_UNSUPPORTED_SHAPE;
  void* scratch = nullptr;
  PACE_TRY(select_scratch_address(&scratch));
  return pace_select_k(unit_score, n_units, group_size, k_units, accepted_ids, rejected_ids,
                       traj_accepted, scratch, kNoAllocScratchBytes, status_dev, stream);
}
