// Fused LM head: per-token log-probabilities under the current policy
// (Sec. 2: the policy factorises over tokens, log pi_theta(y_t | x, y_<t);
// training temperature from the shared settings), without writing logits.
//
// lmhead_lse_kernel (sm_103a, persistent CTA pairs, one CTA per SM, 192
// threads, warp-specialised, tcgen05 on the pair):
//   warp 0            TMA producer, in both CTAs: per K step the CTA's own
//                     128x64 hidden tile and its own half (128x64) of the pair's
//                     256x64 vocabulary tile, into its own 4-stage shared-memory
//                     ring (128-byte swizzle), as one TMA instruction of lanes
//                     0..n (lane 0 the vocabulary half-tile, lanes 1..n the n
//                     boxes of the hidden tile); each CTA arrives on the even
//                     CTA's full barrier with its own bytes.  Contiguous rows:
//                     one 128-row box.  Rows in the loss a subset (mask,
//                     rejected groups, fewer than 128 rows): the hidden tile is
//                     read straight from the caller's hidden-state tensor
//                     through the compact-row index.  Per work item the warp
//                     splits the block's 128 rows into runs of consecutive
//                     source rows (plan_block_loads) and the runs into boxes of
//                     2^j rows (one box for a block inside a response; the
//                     first and last of several runs spill into 16 KB regions
//                     around the tile).  A block of more than 31 boxes is
//                     fetched by four-row TMA gathers (tile::gather4), one per
//                     lane.  No copy of the rows is made.
//   warp 1 / lane 0   MMA issuer, even CTA only: tcgen05.mma.cta_group::2
//                     kind::f16 (bf16 x bf16 -> fp32), M=256 (128 rows from each
//                     CTA), N=256 (128 vocabulary rows from each CTA), K=16 per
//                     instruction; each CTA's tensor memory receives its own
//                     128x256 logit tile; two accumulators (512 TMEM columns)
//                     so the epilogue of tile n overlaps the MMAs of tile n+1.
//   warps 2..5        epilogue, in both CTAs: each thread owns one row (one
//                     TMEM lane), reads its 256 logits 32 columns at a time
//                     with tcgen05.ld, keeps a running base-2 max and sum of
//                     exponentials (online log-sum-exp) and picks out the
//                     target's logit.
// No operand is multicast: every CTA reads only its own tiles; the pair shares
// the vocabulary tile through the 2-CTA MMA itself.
// A work item is a pair of 128-row blocks (one per CTA of the cluster) and one
// of S contiguous vocabulary splits; each CTA writes one (max, sum) pair per row
// and split.  Consecutive items share a row pair, so the hidden tiles re-read
// for every vocabulary tile stay in L2 while the vocabulary streams.  S is
// chosen on the device from the rows actually present (pick_splits).  A soft
// barrier at item boundaries (wait_round) keeps the clusters of a split
// together, so each vocabulary tile is fetched from DRAM about once per round:
// left alone, the clusters' small speed differences add up over the hundreds
// of rounds of a long launch, the leaders fetch tiles from DRAM that the
// laggards fetch again later, and the extra DRAM traffic costs the
// power-capped SMs their clock (a 1.01M-row launch of the 7B head read the
// vocabulary 8.7 times per round; paced, 1.02 times).
//
// lse_merge_kernel: per row, merges the S partial pairs into the log-sum-exp
//   and writes lp = z_y / tau - lse.
//
// Every mbarrier wait is bounded (2 s); on timeout the CTA reports
// PACE_ERR_TIMEOUT, tells its peer to stop, waits (bounded) for its in-flight
// copies and MMAs, frees its tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "pace_internal.cuh"
#include "pace_loss.cuh"
#include "pace_tma.cuh"

namespace pace {
namespace {

constexpr int BM = 128;                         // rows per CTA; the pair's MMA covers 256
constexpr int BN = 256;                         // vocabulary rows per MMA tile (both CTAs)
constexpr int BK = 64;
constexpr int STAGES = 4;
constexpr int CLUSTER = 2;                      // the CTA pair of one 2-CTA MMA
constexpr int kThreads = 192;
constexpr uint32_t kStageA = BM * BK * 2;       // 16 KB: this CTA's 128 hidden rows
constexpr uint32_t kStageB = BN / CLUSTER * BK * 2;  // 16 KB: this CTA's half of the vocabulary tile
constexpr uint32_t kTmemCols = 2 * BN;          // two fp32 accumulators of 256 columns
constexpr uint32_t kIdesc = idesc_bf16_f32(CLUSTER * BM, BN);
// Shared memory: the hidden tiles, each with a 16 KB spill region before and
// after it (shared by neighbours: spill | A0 | spill | A1 | ... | A3 | spill),
// so a 128-row box may start up to 127 rows before or after its tile's first
// row; then the vocabulary tiles; then barriers and flags (256 bytes) and, for
// rows read by index, the block's source rows (int32 [128]) and its planned
// loads (int2 [128]).
constexpr uint32_t kSpill = kStageA;
constexpr uint32_t kARegion = kSpill + STAGES * (kStageA + kSpill);
constexpr uint32_t kMiscBytes = 256 + BM * 4 + BM * 8;
constexpr size_t kSmemBytes =
    1024 /* alignment slack */ + kARegion + STAGES * kStageB + kMiscBytes;
__host__ __device__ constexpr uint32_t a_tile_off(uint32_t s) {
  return kSpill + s * (kStageA + kSpill);
}
__host__ __device__ constexpr uint32_t b_tile_off(uint32_t s) { return kARegion + s * kStageB; }
// Tensor maps of the hidden states with boxes of 1, 2, 4, ..., 128 rows (64
// columns, 128-byte swizzle).
constexpr int kBoxLevels = 8;
constexpr int kMaxBoxes = 31;  // more boxes in a block: four-row gathers instead
struct AMaps {
  CUtensorMap box[kBoxLevels];  // box[j]: 2^j rows
};
constexpr int kMaxSplits = 8;

// Number of vocabulary splits S for row_pairs row pairs on n_clusters persistent
// clusters.  With S = 4 the 19 clusters sweeping one split stay close enough
// for L2 to serve each vocabulary tile to all of them: the vocabulary is read
// from HBM about once per round of items.  With S = 2 the 38 clusters of a
// split drift apart over its 545 MB and it is read ~4 times per round (18.9 GB
// of DRAM reads for four 9,728-row rounds of the 7B head), yet on some GPUs the
// power-capped clock still comes out 2-10 % higher, on others as much lower;
// S = 1 is far slower.  Small batches need more splits to give
// every cluster an item.  So: the first of 4, 2, 3, 6, 8 whose rounds of items
// are at least 90 % full, else whichever fills its rounds best (the earlier on
// ties); a preferred count (pace_set_lmhead_splits, from a measurement on this
// GPU) replaces the choice when it still gives every cluster at least four
// items.  Evaluated identically on the device by the LM head and the merge,
// from the device-side row count.
__host__ __device__ inline int pick_splits(int64_t row_pairs, int64_t n_clusters, int n_vtiles,
                                           int pref) {
  if (pref > 0) {
    const int sp = pref < n_vtiles ? pref : (n_vtiles > 0 ? n_vtiles : 1);
    if (row_pairs * sp >= 4 * n_clusters) return sp;
  }
  const int cand[5] = {4, 2, 3, 6, kMaxSplits};
  int best = 1;
  int64_t best_items = 0, best_rounds = 1;
  for (int i = 0; i < 5; ++i) {
    const int sp = cand[i] < n_vtiles ? cand[i] : (n_vtiles > 0 ? n_vtiles : 1);
    const int64_t items = row_pairs * sp;
    const int64_t rounds = (items + n_clusters - 1) / n_clusters;
    if (items * 10 >= 9 * rounds * n_clusters) return sp;
    if (best_items == 0 || items * best_rounds > best_items * rounds) {
      best = sp;
      best_items = items;
      best_rounds = rounds;
    }
  }
  return best;
}

struct LmArgs {
  int64_t rows_cap;             // rows of the A tensor map
  const long long* n_valid_dev; // rows actually present (device), or null = rows_cap
  int32_t H, V;
  int32_t n_vtiles;
  int32_t split_pref;           // preferred vocabulary splits, 0 = automatic
  float scale_log2;             // log2(e) / temperature
  const int32_t* targets;
  const int32_t* rowidx;        // compact row -> original row, or null (identity)
  int32_t gather;               // 1: rows read by index (rowidx), in planned boxes
  int32_t max_level;            // largest box level no taller than the hidden-state tensor
  float* part_m;                // [rows_cap * kMaxSplits], row r's splits at r * S
  float* part_s;
  float* tgt_logit;             // [rows_cap]
  unsigned* round_ctr;          // pacing counter, zero at launch (or null: no pacing)
  int32_t* status;
};

__device__ __forceinline__ uint64_t make_policy_evict_normal() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// A work item is (row pair, vocabulary split): the two CTAs of a cluster take
// the two 128-row blocks of the pair and sweep the same vocabulary tiles, each
// loading its half of every 256-row vocabulary tile.  Clusters are persistent
// and take items round-robin, so all clusters sweep their splits in step and
// each vocabulary tile is read from HBM about once per round of items.
struct ItemCursor {
  int64_t item, n_items;
  int n_clusters;
  __device__ ItemCursor(int cid, int nc, int64_t ni) : item(cid), n_items(ni), n_clusters(nc) {}
  __device__ bool valid() const { return item < n_items; }
  __device__ void next() { item += n_clusters; }
};

// The loads of one 128-row block whose rows are read by index.  Block row r is
// compact row row0 + r; its source row is rowidx[row0 + r] while that is below
// n_valid.  A run is a maximal stretch of block rows with consecutive source
// rows; the rows past n_valid (loaded, never written back) belong to the last
// run.  A block of one run is loaded as one box per set bit of its length (one
// 128-row box when the tensor has 128 rows or more).  Of several runs, the
// first is one box of the smallest power of two rows that covers it, ending at
// the run's end (its earlier rows land in the spill region before the tile),
// the last one such box starting at the run's start (its later rows land in the
// spill region after the tile), and a run in between one box per set bit of
// its length, largest first.  Boxes never overlap inside the tile, and no box
// is taller than 2^max_level rows (the tallest map the hidden-state tensor
// allows).  Writes the source rows to row_src[BM], the boxes to piece[] as
// (first source row, (first block row + 128) | level << 9), their number to
// plan[0] and their bytes per K step to plan[1].  All 32 lanes call it.
__device__ void plan_block_loads(const int32_t* __restrict__ rowidx, int64_t row0,
                                 int64_t n_valid, int max_level, int lane, int32_t* row_src,
                                 int2* piece, volatile int* plan) {
  const int64_t left = n_valid - row0;
  const int r_inv = left <= 0 ? 0 : (left >= BM ? BM : static_cast<int>(left));
  int32_t v[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int r = 32 * j + lane;
    v[j] = r < r_inv ? rowidx[row0 + r] : 0;
  }
  uint32_t starts[4];
  uint32_t carry = 0;  // source row of the previous word's last row
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int r = 32 * j + lane;
    uint32_t prev = __shfl_up_sync(0xffffffffu, static_cast<uint32_t>(v[j]), 1);
    if (lane == 0) prev = carry;
    const bool st = r == 0 || (r < r_inv && static_cast<uint32_t>(v[j]) != prev + 1u);
    starts[j] = __ballot_sync(0xffffffffu, st);
    carry = __shfl_sync(0xffffffffu, static_cast<uint32_t>(v[j]), 31);
    row_src[r] = v[j];
  }
  __syncwarp();
  if (lane == 0) {
    const uint64_t lo = starts[0] | (static_cast<uint64_t>(starts[1]) << 32);
    const uint64_t hi = starts[2] | (static_cast<uint64_t>(starts[3]) << 32);
    const int m = __popcll(lo) + __popcll(hi);  // runs in the block
    int n = 0, k = 0, r = 0;
    uint32_t rows = 0;
    while (r < BM) {
      const int q = r + 1;  // the run ends at the next start at or after q (BM: none)
      const uint64_t mlo = q < 64 ? (lo & (~0ull << q)) : 0ull;
      int e;
      if (mlo) {
        e = __ffsll(static_cast<long long>(mlo)) - 1;
      } else {
        const uint64_t mhi = q < 64 ? hi : (q < BM ? (hi & (~0ull << (q - 64))) : 0ull);
        e = mhi ? 64 + __ffsll(static_cast<long long>(mhi)) - 1 : BM;
      }
      const int32_t s0 = row_src[r];
      const int len = e - r;
      const int cl = len <= 1 ? 0 : 32 - __clz(len - 1);  // smallest level that covers the run
      if (m > 1 && (k == 0 || k == m - 1) && cl <= max_level) {
        // first or last of several runs: one box of 2^cl rows, ending at the
        // first run's end (spilling before the tile) or starting at the last
        // run's start (spilling after it)
        const int at = k == 0 ? len - (1 << cl) : r;
        piece[n++] = make_int2(s0 + (at - r), (at + BM) | (cl << 9));
        rows += 1u << cl;
      } else {  // the only run, or one in between: one box per set bit of its length
        int at = r, left_rows = len;
        int32_t src = s0;
        while (left_rows > 0) {
          int lev = 31 - __clz(left_rows);
          if (lev > max_level) lev = max_level;
          piece[n++] = make_int2(src, (at + BM) | (lev << 9));
          rows += 1u << lev;
          at += 1 << lev;
          src += 1 << lev;
          left_rows -= 1 << lev;
        }
      }
      r = e;
      ++k;
    }
    plan[0] = n;
    plan[1] = static_cast<int>(rows * (BK * 2));
  }
  __syncwarp();
}

__global__ void __cluster_dims__(CLUSTER, 1, 1) __launch_bounds__(kThreads, 1)
    lmhead_lse_kernel(const __grid_constant__ AMaps am, const __grid_constant__ CUtensorMap tm_b,
                      LmArgs p) {
  extern __shared__ unsigned char smem_raw[];
  // the same offsets in both CTAs: the pair's MMA reads each CTA's operand
  // tiles at the addresses the even CTA's descriptors name
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kARegion + STAGES * kStageB);
  uint64_t* full = bars;                     // [STAGES] even CTA: both CTAs' tiles landed
  uint64_t* empty = bars + STAGES;           // [STAGES] the pair's MMAs are done with the stage
  uint64_t* tmem_full = bars + 2 * STAGES;   // [2] this CTA's accumulator is ready
  uint64_t* tmem_empty = tmem_full + 2;      // [2] even CTA: both CTAs' epilogues drained it
  uint64_t* mma_done = tmem_empty + 2;       // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* plan = reinterpret_cast<volatile int*>(tmem_slot + 2);  // [2] boxes, A bytes
  int32_t* row_src = reinterpret_cast<int32_t*>(reinterpret_cast<unsigned char*>(bars) + 256);
  int2* piece = reinterpret_cast<int2*>(row_src + BM);                            // [BM]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();
  const bool leader = crank == 0;
  const int n_clusters = static_cast<int>(gridDim.x) / CLUSTER;
  const int cid = static_cast<int>(blockIdx.x) / CLUSTER;
  const int64_t n_valid = p.n_valid_dev ? static_cast<int64_t>(*p.n_valid_dev) : p.rows_cap;
  const int64_t row_pairs = (n_valid + 2 * BM - 1) / (2 * BM);
  const int n_splits = pick_splits(row_pairs, n_clusters, p.n_vtiles, p.split_pref);
  const int tiles_per_split = (p.n_vtiles + n_splits - 1) / n_splits;
  const int64_t n_items = row_pairs * n_splits;
  // both CTAs of a cluster read the same n_valid and cid: the exit is uniform,
  // and comes before the pair's collective tensor-memory allocation
  if (cid >= n_items) return;
  const int nkb = p.H / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], CLUSTER);  // each CTA's producer arrives with its bytes
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tmem_full[b], 1);
      mbar_init(&tmem_empty[b], CLUSTER * 4);  // one arrival per epilogue warp of the pair
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  cluster_sync();  // both CTAs run and their barriers exist
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' tensor memory is allocated before any MMA writes it
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t peer_abort = cluster_addr(const_cast<int*>(abort_flag), crank ^ 1u);
  // first timeout: report it, and make both CTAs of the pair stop issuing
  auto give_up = [&]() {
    if (!*abort_flag) report(p.status, PACE_ERR_TIMEOUT);
    *abort_flag = 1;
    st_cluster_u32(peer_abort, 1u);
  };

  if (warp == 0) {
    // ------------------------------------------------ TMA producer (both CTAs)
    // The whole warp produces.  Per K step one TMA instruction, issued by
    // lanes 0..n: lane 0 loads the CTA's half of the vocabulary tile, lanes
    // 1..n the n boxes of its hidden tile (one 128-row box for contiguous rows;
    // for rows read by index, the boxes plan_block_loads gives).  A block of
    // more than kMaxBoxes boxes is gathered four rows a lane instead.
    const bool gather = p.gather != 0;
    if (lane == 0) tma_prefetch_desc(&tm_b);
    if (lane < kBoxLevels) tma_prefetch_desc(&am.box[lane]);
    const uint64_t pol = make_policy_evict_normal();
    uint32_t it = 0;
    bool ok = true;
    unsigned round = 0;  // this cluster's items so far (the round of the current one)
    for (ItemCursor c(cid, n_clusters, n_items); c.valid() && ok; c.next(), ++round) {
      const int64_t rp = c.item / n_splits;
      const int split = static_cast<int>(c.item % n_splits);
      const int64_t row0 = (rp * CLUSTER + crank) * BM;
      // this lane's load: lane 0 the vocabulary half-tile (its coordinates are
      // set per tile below), lane 1 + q the hidden tile's box q
      int n = 1;
      uint32_t a_bytes = kStageA;  // this CTA's hidden-tile bytes per K step
      int32_t psrc = static_cast<int32_t>(row0);
      int pdst = 0, plev = kBoxLevels - 1;
      int32_t g4[4] = {0, 0, 0, 0};
      bool scattered = false;
      if (gather) {
        plan_block_loads(p.rowidx, row0, n_valid, p.max_level, lane, row_src, piece, plan);
        n = plan[0];
        scattered = n > kMaxBoxes;
        if (!scattered) {
          a_bytes = static_cast<uint32_t>(plan[1]);
          if (lane >= 1 && lane <= n) {
            const int2 pc = piece[lane - 1];
            psrc = pc.x;
            pdst = (pc.y & 0x1ff) - BM;  // first block row, -127..127
            plev = pc.y >> 9;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) g4[j] = row_src[4 * lane + j];  // row 0 past the end
        }
      }
      // every round before the last is full, so round k starts once all
      // clusters issued their round k-1 loads (the even CTA paces the pair)
      if (leader && lane == 0 && round > 0 && p.round_ctr)
        wait_round(p.round_ctr, round * static_cast<unsigned>(n_clusters));
      __syncwarp();
      const int tile0 = split * tiles_per_split;
      const int tile1 = min(tile0 + tiles_per_split, p.n_vtiles);
      const int issuers = scattered ? 1 : n + 1;
      for (int t = tile0; t < tile1 && ok; ++t) {
        const int32_t nb = t * BN + static_cast<int32_t>(crank) * (BN / CLUSTER);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1u;
          // one outcome for the warp
          if (!__all_sync(0xffffffffu, mbar_wait_bounded(&empty[s], ph ^ 1u, abort_flag))) {
            ok = false;
            break;
          }
          unsigned char* sa = smem + a_tile_off(s);
          unsigned char* sb = smem + b_tile_off(s);
          const uint32_t bar = cluster_addr(&full[s], 0);
          if (lane == 0) {
            // this CTA's bytes of the stage, announced with its arrival on the
            // even CTA's barrier (which completes once both CTAs' bytes land)
            if (leader)
              mbar_arrive_expect_tx(&full[s], a_bytes + kStageB);
            else
              mbar_arrive_expect_tx_cluster(bar, a_bytes + kStageB);
          }
          if (lane < issuers) {
            const void* desc = lane == 0 ? static_cast<const void*>(&tm_b)
                                         : static_cast<const void*>(&am.box[plev]);
            unsigned char* dst = lane == 0 ? sb : sa + pdst * (BK * 2);
            tma_load_2d_pair(dst, desc, bar, kb * BK, lane == 0 ? nb : psrc, pol);
          }
          if (scattered)
            tma_gather4_pair(sa + lane * 4 * (BK * 2), &am.box[0], bar, kb * BK, g4[0], g4[1],
                             g4[2], g4[3], pol);
        }
      }
      if (leader && lane == 0 && ok && p.round_ctr) atomicAdd(p.round_ctr, 1u);
      __syncwarp();  // row_src and piece are rewritten for the next item
    }
    if (lane == 0) {
      if (!ok) give_up();
      // Drain: every copy issued must have landed before the CTA exits.  The
      // even CTA sees both CTAs' bytes (every lane's loads included) on its
      // full barriers; the odd CTA sees its stages consumed on its empty
      // barriers.  After a timeout anywhere the waits are short: copies land
      // in microseconds.
      const uint64_t lim = *abort_flag ? 1000000ull : kWaitLimitNs;
      for (uint32_t s = 0; s < STAGES && s < it; ++s) {
        const uint32_t last = it - 1 - ((it - 1 - s) % STAGES);  // last index with stage s
        if (leader)
          mbar_wait_bounded(&full[s], (last / STAGES) & 1u, nullptr, lim);
        else
          mbar_wait_bounded(&empty[s], (last / STAGES) & 1u, nullptr, lim);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------ MMA issuer (even CTA)
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (ItemCursor c(cid, n_clusters, n_items); c.valid() && ok; c.next()) {
        const int split = static_cast<int>(c.item % n_splits);
        const int tile0 = split * tiles_per_split;
        const int tile1 = min(tile0 + tiles_per_split, p.n_vtiles);
        for (int t = tile0; t < tile1 && ok; ++t, ++tcount) {
          const uint32_t acc = tcount & 1u;
          const uint32_t acc_ph = (tcount >> 1) & 1u;
          if (!mbar_wait_bounded_cluster(&tmem_empty[acc], acc_ph ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * BN;
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const uint32_t s = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1u;
            if (!mbar_wait_bounded(&full[s], ph, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + a_tile_off(s));
            const uint32_t sb = smem_u32(smem + b_tile_off(s));
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              tc_mma_f16_pair(d_tmem, smem_desc_k128(sa + k * 32), smem_desc_k128(sb + k * 32),
                              kIdesc, (kb > 0 || k > 0) ? 1u : 0u);
            }
            // the stage is free in both CTAs once these MMAs have read it
            tc_commit_pair(cluster_addr(&empty[s], 0));
            tc_commit_pair(cluster_addr(&empty[s], 1));
          }
          if (!ok) break;
          tc_commit_pair(cluster_addr(&tmem_full[acc], 0));
          tc_commit_pair(cluster_addr(&tmem_full[acc], 1));
        }
      }
      if (!ok) give_up();
      // all MMAs issued by this thread complete before tensor memory is freed
      tc_commit_pair(cluster_addr(mma_done, 0));
      mbar_wait_bounded(mma_done, 0, nullptr);
    }
  } else {
    // ------------------------------------------------ epilogue (4 warps, both CTAs)
    const int quad = warp & 3;  // TMEM lanes this warp may access
    const int r_local = quad * 32 + lane;
    const float scale = p.scale_log2;
    const uint32_t empty0 = cluster_addr(&tmem_empty[0], 0);
    const uint32_t empty1 = cluster_addr(&tmem_empty[1], 0);
    uint32_t tcount = 0;
    bool ok = true;
    for (ItemCursor c(cid, n_clusters, n_items); c.valid() && ok; c.next()) {
      const int64_t rp = c.item / n_splits;
      const int split = static_cast<int>(c.item % n_splits);
      const int tile0 = split * tiles_per_split;
      const int tile1 = min(tile0 + tiles_per_split, p.n_vtiles);
      const int64_t row = (rp * CLUSTER + crank) * BM + r_local;
      const bool row_ok = row < n_valid;
      int32_t y = -1;
      if (row_ok) {
        const int64_t orig = p.rowidx ? static_cast<int64_t>(p.rowidx[row]) : row;
        y = p.targets[orig];
      }
      float m = -INFINITY, s = 0.0f, tgt = 0.0f;
      bool have_tgt = false;
      for (int t = tile0; t < tile1; ++t, ++tcount) {
        const uint32_t acc = tcount & 1u;
        const uint32_t acc_ph = (tcount >> 1) & 1u;
        // one outcome for the whole warp: tcgen05.ld below is warp-collective,
        // and a lane that saw the peer's abort must not leave its warp behind
        const bool got = __all_sync(0xffffffffu,
                                    mbar_wait_bounded(&tmem_full[acc], acc_ph, abort_flag));
        if (!got) {
          give_up();
          ok = false;
          break;
        }
        tc_fence_after();
        const int32_t n0 = t * BN;
        const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + acc * BN;
#pragma unroll 1
        for (int cc = 0; cc < BN; cc += 32) {
          float v[32];
          tmem_ld_32x32b_x32(tbase + cc, v);
          tmem_wait_ld();
          const int32_t col0 = n0 + cc;
          if (col0 + 32 > p.V) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (col0 + i >= p.V) v[i] = -INFINITY;
          }
          float cm = v[0];
#pragma unroll
          for (int i = 1; i < 32; ++i) cm = fmaxf(cm, v[i]);
          const float m_new = fmaxf(m, cm * scale);
          float acc_s = 0.0f;
#pragma unroll
          for (int i = 0; i < 32; ++i) acc_s += ex2_approx(fmaf(v[i], scale, -m_new));
          s = s * ex2_approx(m - m_new) + acc_s;
          m = m_new;
          const uint32_t off = static_cast<uint32_t>(y - col0);
          if (off < 32u) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (off == static_cast<uint32_t>(i)) tgt = v[i];
            have_tgt = true;
          }
        }
        // this warp is done reading the accumulator: one arrival per warp on the
        // even CTA's barrier, after every lane's loads have completed
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(acc ? empty1 : empty0);
      }
      if (row_ok && ok) {
        const int64_t o = row * n_splits + split;
        p.part_m[o] = m;
        p.part_s[o] = s;
        if (have_tgt) p.tgt_logit[row] = tgt;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA frees its tensor memory or leaves while the pair's MMAs, copies
  // or arrivals may still reach it
  cluster_sync();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, kTmemCols);
  cluster_sync();  // the collective release is complete in both CTAs
}

// Per row in the loss: log-sum-exp from the split partials, then
// lp = z_y / tau - lse, scattered back to the original row.
__global__ void lse_merge_kernel(int64_t rows_cap, const long long* __restrict__ n_valid_dev,
                                 int lm_clusters, int n_vtiles, int split_pref, int32_t V,
                                 float inv_temp,
                                 const float* __restrict__ part_m, const float* __restrict__ part_s,
                                 const float* __restrict__ tgt_logit,
                                 const int32_t* __restrict__ targets,
                                 const int32_t* __restrict__ rowidx, float* __restrict__ logprob,
                                 float* __restrict__ lse_out, int32_t* status) {
  const int64_t n_valid = n_valid_dev ? static_cast<int64_t>(*n_valid_dev) : rows_cap;
  // the split count the LM head used for these rows
  const int splits =
      pick_splits((n_valid + 2 * BM - 1) / (2 * BM), lm_clusters, n_vtiles, split_pref);
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; r < n_valid;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t orig = rowidx ? static_cast<int64_t>(rowidx[r]) : r;
    float mm = -INFINITY;
    for (int s = 0; s < splits; ++s) mm = fmaxf(mm, part_m[r * splits + s]);
    float ss = 0.0f;
    for (int s = 0; s < splits; ++s) ss += part_s[r * splits + s] * ex2_approx(part_m[r * splits + s] - mm);
    const float lse = (mm + lg2_approx(ss)) * 0.69314718055994531f;
    const int32_t y = targets[orig];
    float lp;
    if (y < 0 || y >= V) {
      report(status, PACE_ERR_INVALID_ARG);
      lp = __int_as_float(0x7fc00000);
    } else {
      lp = tgt_logit[r] * inv_temp - lse;
    }
    logprob[orig] = lp;
    if (lse_out) lse_out[orig] = lse;
  }
}

// ---------------------------------------------------------------- host side

struct LmLaunchInfo {
  int max_clusters = 0;
};

// Dynamic shared memory opt-in and the number of 2-CTA clusters that can be
// resident at once on the current device (cached per device).
pace_status lm_launch_info(LmLaunchInfo* out) {
  constexpr int kMaxDevices = 64;
  static LmLaunchInfo info[kMaxDevices];
  static std::mutex mu;
  int dev = 0;
  PACE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_CUDA;
  std::lock_guard<std::mutex> g(mu);
  if (info[dev].max_clusters == 0) {
    PACE_TRY_CUDA(cudaFuncSetAttribute(lmhead_lse_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kSmemBytes)));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(sm_count()), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmemBytes;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = CLUSTER;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, lmhead_lse_kernel, &cfg) != cudaSuccess || n < 1)
      n = sm_count() / CLUSTER;
    info[dev].max_clusters = n;
  }
  *out = info[dev];
  return PACE_OK;
}

}  // namespace

void carve_lm_ws(Carver& cv, int64_t n_rows, int64_t n_seq, int H, bool dense_rows,
                 LmWs* w) {
  const int64_t rows_cap = n_rows > BM ? n_rows : BM;
  carve_compact_ws(cv, n_seq, n_rows, &w->cw);
  carve_surrogate_ws(cv, n_seq, &w->sw);
  w->hidden_c =
      dense_rows ? static_cast<void*>(cv.take<uint16_t>(static_cast<size_t>(rows_cap) * H))
                 : nullptr;
  w->part_m = cv.take<float>(static_cast<size_t>(rows_cap) * kMaxSplits);
  w->part_s = cv.take<float>(static_cast<size_t>(rows_cap) * kMaxSplits);
  w->tgt = cv.take<float>(static_cast<size_t>(rows_cap));
  w->round_ctr = cv.take<unsigned>(1);
}

bool lm_needs_compaction(const PaceBatch* b) {
  return b->mask || b->seq_accepted || b->n_rows < BM;
}

pace_status check_lm_args(const PaceBatch* batch, const void* hidden, const void* w_vocab,
                          const int32_t* targets, int H, int V, float temperature,
                          const float* logprob) {
  PACE_TRY(check_batch(batch));
  if (H < 64 || H > 16384 || H % 64 != 0) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (V < 1 || V > (1 << 24)) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (!(temperature > 0.0f) || !isfinite(temperature)) return PACE_ERR_INVALID_ARG;
  if (batch->n_rows > 0 && (!hidden || !w_vocab || !targets || !logprob))
    return PACE_ERR_INVALID_ARG;
  if (!aligned(hidden, 16) || !aligned(w_vocab, 16)) return PACE_ERR_UNSUPPORTED_SHAPE;
  return PACE_OK;
}

// Compaction, fused LM head and merge: lp (and lse) for every row in
// the batch's loss, 0 elsewhere.
pace_status run_logprob(const PaceBatch* batch, const void* hidden, const void* w_vocab,
                        const int32_t* targets, int H, int V, float temperature, float* logprob,
                        float* lse, const LmWs& ws, int32_t* status_dev, cudaStream_t st) {
  const int64_t n_rows = batch->n_rows;
  const bool compact = lm_needs_compaction(batch);
  if (n_rows > 0) {
    PACE_TRY_CUDA(cudaMemsetAsync(logprob, 0, static_cast<size_t>(n_rows) * sizeof(float), st));
    if (lse) PACE_TRY_CUDA(cudaMemsetAsync(lse, 0, static_cast<size_t>(n_rows) * sizeof(float), st));
  }
  const long long* n_valid_dev = nullptr;
  const int32_t* rowidx = nullptr;
  int64_t rows_cap = n_rows;
  if (compact) {
    // the LM head reads the rows in the loss through rowidx (no dense copy)
    PACE_TRY(run_compaction(batch, ws.cw, status_dev, st));
    n_valid_dev = ws.cw.total;
    rowidx = ws.cw.rowidx;
    rows_cap = n_rows > BM ? n_rows : BM;
  }
  if (n_rows == 0) return PACE_OK;
  const int n_vtiles = (V + BN - 1) / BN;
  AMaps am;
  CUtensorMap tm_b;
  // boxes of 2^j hidden rows for j up to the tensor's height (at most 128);
  // taller levels repeat the tallest valid map and are never used
  int max_level = 0;
  while (max_level + 1 < kBoxLevels && (int64_t{1} << (max_level + 1)) <= n_rows) ++max_level;
  if (!compact && max_level != kBoxLevels - 1) return PACE_ERR_INVALID_ARG;  // n_rows >= 128
  for (int j = 0; j < kBoxLevels; ++j) {
    if (j <= max_level) PACE_TRY(encode_bf16_2d(&am.box[j], hidden, n_rows, H, H, BK, 1 << j));
    else am.box[j] = am.box[max_level];
  }
  PACE_TRY(encode_bf16_2d(&tm_b, w_vocab, V, H, H, BK, BN / CLUSTER));  // one CTA's half tile
  LmLaunchInfo li;
  PACE_TRY(lm_launch_info(&li));
  LmArgs a;
  a.rows_cap = rows_cap;
  a.n_valid_dev = n_valid_dev;
  a.H = H;
  a.V = V;
  a.n_vtiles = n_vtiles;
  a.split_pref = lmhead_split_pref().load();
  a.scale_log2 = 1.4426950408889634f / temperature;
  a.targets = targets;
  a.rowidx = rowidx;
  a.gather = compact ? 1 : 0;
  a.max_level = max_level;
  a.part_m = ws.part_m;
  a.part_s = ws.part_s;
  a.tgt_logit = ws.tgt;
  a.round_ctr = ws.round_ctr;
  a.status = status_dev;
  // persistent: at most one wave of 2-CTA clusters, never more clusters than the
  // most items the rows could make (the split count is chosen on the device)
  const int64_t items = (rows_cap + 2 * BM - 1) / (2 * BM) * kMaxSplits;
  const int64_t clusters = items < li.max_clusters ? items : li.max_clusters;
  const int64_t grid = clusters * CLUSTER;
  PACE_TRY_CUDA(cudaMemsetAsync(ws.round_ctr, 0, sizeof(unsigned), st));
  const ProfileEvents& pe = profile_events(PACE_PROFILE_LMHEAD);
  if (pe.begin) PACE_TRY_CUDA(cudaEventRecord(pe.begin, st));
  lmhead_lse_kernel<<<static_cast<unsigned>(grid), kThreads, kSmemBytes, st>>>(am, tm_b, a);
  PACE_TRY(last_launch_status());
  if (pe.end) PACE_TRY_CUDA(cudaEventRecord(pe.end, st));
  int64_t mblocks = (rows_cap + 255) / 256;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  if (mblocks > cap) mblocks = cap;
  lse_merge_kernel<<<static_cast<unsigned>(mblocks), 256, 0, st>>>(
      rows_cap, n_valid_dev, static_cast<int>(clusters), n_vtiles, a.split_pref, V,
      1.0f / temperature,
      ws.part_m, ws.part_s, ws.tgt, targets,
      rowidx, logprob, lse, status_dev);
  return last_launch_status();
}

}  // namespace pace

using namespace pace;

extern "C" size_t pace_token_logprob_workspace_size(int64_t n_rows, int64_t n_seq,
                                                    int32_t hidden_size, int32_t vocab_size) {
  if (n_rows < 0 || n_seq < 0 || hidden_size <= 0 || vocab_size <= 0) return 0;
  Carver cv;
  LmWs w;
  carve_lm_ws(cv, n_rows, n_seq, hidden_size, false, &w);
  return cv.used;
}

extern "C" pace_status pace_token_logprob(const PaceBatch* batch, const void* hidden,
                                          const void* w_vocab, const int32_t* targets,
                                          int32_t hidden_size, int32_t vocab_size,
                                          float temperature, float* logprob, float* lse,
                                          const PaceLossArgs* loss, void* workspace,
                                          size_t workspace_bytes, int32_t* status_dev,
                                          void* stream) {
  PACE_TRY(check_lm_args(batch, hidden, w_vocab, targets, hidden_size, vocab_size, temperature,
                         logprob));
  if (loss) PACE_TRY(check_loss_args(batch, loss));
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  LmWs ws;
  carve_lm_ws(cv, batch->n_rows, batch->n_seq, hidden_size, false, &ws);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  cudaStream_t st = as_stream(stream);
  PACE_TRY(run_logprob(batch, hidden, w_vocab, targets, hidden_size, vocab_size, temperature,
                       logprob, lse, ws, status_dev, st));
  if (loss) PACE_TRY(run_surrogate(batch, logprob, loss, ws.sw, status_dev, st));
  return PACE_OK;
}
