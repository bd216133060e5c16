// Backward of the fused LM head and of the clipped surrogate (what the unchanged
// policy update needs after the log-probs: gradients with respect to the hidden
// states and the vocabulary matrix), without ever holding the logits of more
// than one chunk of rows.
//
// For the rows in the loss, in chunks of up to kChunkRows compacted rows:
//   1. gemm_kernel<EPI_G>:    z = H_c W^T recomputed on the tensor cores; the
//                             epilogue writes G = (g / tau) (onehot(y) - softmax(z / tau))
//                             in bf16, using the forward's log-sum-exp, in 64-column
//                             blocks: G[v / 64][row][v % 64], so that both later
//                             GEMMs read it in long contiguous runs (a K step of
//                             dH is one 16 KB run, a K step of dW 8 KB);
//   2. gemm_kernel<EPI_ROWS>: dH_c = G W (A = G K-major, B = W read MN-major),
//                             fp32 rows scattered back to their original row;
//   3. gemm_kernel<EPI_ACC>:  dW += G^T H_c (A = G and B = H_c, both read
//                             MN-major), fp32 accumulation in place.
// The GEMM is one warp-specialised tcgen05 kernel on CTA pairs: in each CTA
// warp 0 issues TMA for the CTA's own A tile and its own half of the B tile
// into a 4-stage ring (128-byte swizzle), both CTAs' bytes completing on the
// even CTA's barrier; warp 1 of the even CTA issues tcgen05.mma.cta_group::2
// (M 256 = 128 rows per CTA, N 256 = 128 columns from each CTA, K 16; the
// instruction descriptor's major bits select K- or MN-major operand layouts);
// warps 2-5 of each CTA drain its two TMEM accumulators.  Every CTA loads only
// its own tiles.  Every wait is bounded.
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

constexpr int GBM = 128;
constexpr int GBN = 256;
constexpr int GBK = 64;
constexpr int GSTAGES = 4;
constexpr int kGemmThreads = 192;
constexpr uint32_t kGStageA = GBM * GBK * 2;  // 16 KB
constexpr uint32_t kGStageB = GBN / 2 * GBK * 2;  // 16 KB: this CTA's half of the B tile
constexpr uint32_t kGStageBytes = kGStageA + kGStageB;
constexpr uint32_t kGTmemCols = 2 * GBN;
constexpr size_t kGSmemBytes = 1024 + GSTAGES * kGStageBytes + 256;
constexpr int64_t kChunkRows = 32768;         // rows of G held at once (bf16 M x V)
constexpr int kGroupM = 38;                   // M tiles per raster group

enum { EPI_G = 0, EPI_ROWS = 1, EPI_ACC = 2 };
enum { TRIM_NONE = 0, TRIM_M = 1, TRIM_K = 2 };

struct GemmArgs {
  int64_t M, N, K;
  int64_t m_tiles, n_tiles;
  int raster_n_fast;            // 1: N tile fastest; 0: groups of kGroupM M tiles, M fastest
  int trim;                     // TRIM_M / TRIM_K: that extent is cut, on the device, to the
                                // chunk's rows in the loss rounded up to GBM (TRIM_NONE: as given)
  // EPI_G
  int64_t chunk_row0;           // compact row of the chunk's first row
  const long long* n_valid;     // rows in the loss (device)
  const int32_t* rowidx;        // compact -> original row
  const int32_t* targets;
  const float* lse;             // forward log-sum-exp per original row
  const float* dlp;             // dLoss/dlp per original row
  float scale_log2;             // log2(e) / tau
  float inv_tau;
  uint16_t* g_out;              // bf16 G in 64-column blocks: [g_cols / 64][g_pitch][64]
  int64_t g_cols;               // V rounded up to 64 (columns >= V hold zeros)
  int64_t g_pitch;              // rows per 64-column block
  // A operand from the blocked G (a_pitch > 0: rows per 64-column block); 0: plain matrix
  int64_t a_pitch;
  int32_t V;
  // EPI_ROWS
  float* rows_out;              // fp32 [orig rows][ldo]
  int64_t ldo;
  // EPI_ACC
  float* acc_out;               // fp32 [M][ldo]
  unsigned* round_ctr;          // pacing counter, zeroed before the launch (or null)
  int32_t* status;
};

// Work items are (pair of M tiles, N tile); the two CTAs of a cluster take the
// two M tiles of a pair and share every B tile through the 2-CTA MMA, each
// loading its own half of it.
__device__ __forceinline__ void item_of(const GemmArgs& p, int64_t m_tiles, int64_t item,
                                        int64_t* mp, int64_t* n) {
  const int64_t pairs = (m_tiles + 1) / 2;
  if (p.raster_n_fast) {
    *mp = item / p.n_tiles;
    *n = item % p.n_tiles;
    return;
  }
  const int64_t gp = kGroupM / 2;  // pairs per raster group
  const int64_t per_group = gp * p.n_tiles;
  const int64_t g = item / per_group;
  const int64_t r = item % per_group;
  const int64_t g0 = g * gp;
  const int64_t gm = (pairs - g0) < gp ? (pairs - g0) : gp;
  *mp = g0 + r % gm;
  *n = r / gm;
}

// 128-byte-swizzled operand tiles.  K-major: rows of 64 K elements (128 B),
// 8-row groups 1024 B apart; a 16-deep K step is +32 B.  MN-major: 64 MN
// elements per 128-byte row, one row per k; boxes of 64 (MN) x 64 (K) stacked
// along MN 8 KB apart (leading byte offset), 8-k groups 1024 B apart (stride
// byte offset); a 16-deep K step is +2048 B.
__device__ __forceinline__ uint64_t operand_desc(uint32_t saddr, bool mn_major) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(mn_major ? (8192u >> 4) : 1u) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// M = 256: the pair's two 128-row tiles.
__host__ __device__ constexpr uint32_t idesc_bf16(bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) |
         ((b_mn ? 1u : 0u) << 16) | ((static_cast<uint32_t>(GBN) >> 3) << 17) |
         ((static_cast<uint32_t>(2 * GBM) >> 4) << 24);
}

__device__ __forceinline__ uint16_t f32_to_bf16_rn(float x) {
  uint32_t u = __float_as_uint(x);
  if ((u & 0x7fffffffu) > 0x7f800000u) return static_cast<uint16_t>((u >> 16) | 0x40u);  // NaN
  u += 0x7fffu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

template <bool A_MN, bool B_MN, int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                GemmArgs p) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + GSTAGES * kGStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + GSTAGES;
  uint64_t* tmem_full = bars + 2 * GSTAGES;
  uint64_t* tmem_empty = tmem_full + 2;
  uint64_t* mma_done = tmem_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();
  const bool leader = crank == 0;
  // The host sizes a chunk by its row capacity; the rows of it that are in the
  // loss are known only on the device (the compaction's count).  Tiles past
  // them hold zero rows: M (G, dH) or K (dW) is cut to the count rounded up to
  // GBM, the same value in every CTA, so every early exit below is uniform.
  int64_t M = p.M, K = p.K, m_tiles = p.m_tiles;
  if (p.trim != TRIM_NONE) {
    int64_t v = static_cast<int64_t>(*p.n_valid) - p.chunk_row0;
    const int64_t cap = p.trim == TRIM_M ? p.M : p.K;
    v = v < 0 ? 0 : (v > cap ? cap : v);
    v = (v + GBM - 1) / GBM * GBM;
    if (v > cap) v = cap;
    if (p.trim == TRIM_M) {
      M = v;
      m_tiles = (v + GBM - 1) / GBM;
    } else {
      K = v;
    }
  }
  const int64_t n_items = (m_tiles + 1) / 2 * p.n_tiles;
  const int64_t cid = blockIdx.x / 2, n_clusters = gridDim.x / 2;
  const int nkb = static_cast<int>((K + GBK - 1) / GBK);
  // uniform over the grid, and before the pair's collective TMEM allocation
  if (nkb == 0 || n_items == 0) return;

  if (threadIdx.x == 0) {
    for (int s = 0; s < GSTAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tmem_full[b], 1);
      mbar_init(&tmem_empty[b], 2 * 4);  // one arrival per epilogue warp of the pair
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  cluster_sync();  // both CTAs run and their barriers exist
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kGTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' tensor memory is allocated before any MMA writes it
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  constexpr uint32_t kIdesc = idesc_bf16(A_MN, B_MN);
  const uint32_t peer_abort = cluster_addr(const_cast<int*>(abort_flag), crank ^ 1u);
  auto give_up = [&]() {
    if (!*abort_flag) report(p.status, PACE_ERR_TIMEOUT);
    *abort_flag = 1;
    st_cluster_u32(peer_abort, 1u);
  };

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_a);
      tma_prefetch_desc(&tm_b);
      uint64_t pol;
      asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
      uint32_t it = 0;
      bool ok = true;
      unsigned round = 0;  // this cluster's items so far
      for (int64_t t = cid; t < n_items && ok; t += n_clusters, ++round) {
        int64_t mp, nt;
        item_of(p, m_tiles, t, &mp, &nt);
        const int32_t m0 = static_cast<int32_t>((2 * mp + crank) * GBM);
        const int32_t n0 = static_cast<int32_t>(nt * GBN);
        // the clusters start each round together (every round but the last is full)
        if (leader && round > 0 && p.round_ctr)
          wait_round(p.round_ctr, round * static_cast<unsigned>(n_clusters));
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % GSTAGES, ph = (it / GSTAGES) & 1u;
          if (!mbar_wait_bounded(&empty[s], ph ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          unsigned char* sa = smem + s * kGStageBytes;
          unsigned char* sb = sa + kGStageA;
          const uint32_t bar = cluster_addr(&full[s], 0);
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * kGStageBytes);
          const int32_t k0 = kb * GBK;
          if (p.a_pitch > 0) {  // blocked G: one 64-wide block is the inner dimension
            const int64_t ap = p.a_pitch;
            if (A_MN) {  // M = vocabulary: blocks m0 / 64 and m0 / 64 + 1, rows k0..k0+63
              const int64_t b0 = m0 / 64;
              tma_load_2d_pair(sa, &tm_a, bar, 0, static_cast<int32_t>(b0 * ap + k0), pol);
              tma_load_2d_pair(sa + 8192, &tm_a, bar, 0,
                               static_cast<int32_t>((b0 + 1) * ap + k0), pol);
            } else {     // K = vocabulary: block kb, rows m0..m0+127
              tma_load_2d_pair(sa, &tm_a, bar, 0, static_cast<int32_t>(kb * ap + m0), pol);
            }
          } else if (A_MN) {  // box {64 MN, 64 K}: two along M
            tma_load_2d_pair(sa, &tm_a, bar, m0, k0, pol);
            tma_load_2d_pair(sa + 8192, &tm_a, bar, m0 + 64, k0, pol);
          } else {     // box {64 K, 128 rows}
            tma_load_2d_pair(sa, &tm_a, bar, k0, m0, pol);
          }
          // this CTA's half of B: columns n0 + 128 * crank .. + 127
          const int32_t nh = n0 + static_cast<int32_t>(crank) * (GBN / 2);
          if (B_MN) {  // two {64 N, 64 K} boxes along N
            tma_load_2d_pair(sb, &tm_b, bar, nh, k0, pol);
            tma_load_2d_pair(sb + 8192, &tm_b, bar, nh + 64, k0, pol);
          } else {     // {64 K, 128 rows}
            tma_load_2d_pair(sb, &tm_b, bar, k0, nh, pol);
          }
        }
        if (leader && ok && p.round_ctr) atomicAdd(p.round_ctr, 1u);
      }
      if (!ok) give_up();
      // every copy issued has landed before the CTA exits: the even CTA sees
      // both CTAs' bytes on its full barriers, the odd CTA its stages consumed
      const uint64_t lim = *abort_flag ? 1000000ull : kWaitLimitNs;
      for (uint32_t s = 0; s < GSTAGES && s < it; ++s) {
        const uint32_t last = it - 1 - ((it - 1 - s) % GSTAGES);
        if (leader)
          mbar_wait_bounded(&full[s], (last / GSTAGES) & 1u, nullptr, lim);
        else
          mbar_wait_bounded(&empty[s], (last / GSTAGES) & 1u, nullptr, lim);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      uint32_t it = 0, tc = 0;
      bool ok = true;
      for (int64_t t = cid; t < n_items && ok; t += n_clusters, ++tc) {
        const uint32_t acc = tc & 1u, acc_ph = (tc >> 1) & 1u;
        if (!mbar_wait_bounded_cluster(&tmem_empty[acc], acc_ph ^ 1u, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * GBN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % GSTAGES, ph = (it / GSTAGES) & 1u;
          if (!mbar_wait_bounded(&full[s], ph, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * kGStageBytes);
          const uint32_t sb = sa + kGStageA;
#pragma unroll
          for (int k = 0; k < GBK / 16; ++k) {
            const uint32_t ka = A_MN ? sa + k * 2048 : sa + k * 32;
            const uint32_t kbb = B_MN ? sb + k * 2048 : sb + k * 32;
            tc_mma_f16_pair(d_tmem, operand_desc(ka, A_MN), operand_desc(kbb, B_MN), kIdesc,
                            (kb > 0 || k > 0) ? 1u : 0u);
          }
          tc_commit_pair(cluster_addr(&empty[s], 0));
          tc_commit_pair(cluster_addr(&empty[s], 1));
        }
        if (!ok) break;
        tc_commit_pair(cluster_addr(&tmem_full[acc], 0));
        tc_commit_pair(cluster_addr(&tmem_full[acc], 1));
      }
      if (!ok) give_up();
      tc_commit_pair(cluster_addr(mma_done, 0));
      mbar_wait_bounded(mma_done, 0, nullptr);
    }
  } else {
    const int quad = warp & 3;
    const int r_local = quad * 32 + lane;
    const uint32_t empty0 = cluster_addr(&tmem_empty[0], 0);
    const uint32_t empty1 = cluster_addr(&tmem_empty[1], 0);
    uint32_t tc = 0;
    for (int64_t t = cid; t < n_items; t += n_clusters, ++tc) {
      int64_t mp, nt;
      item_of(p, m_tiles, t, &mp, &nt);
      const int64_t mt = 2 * mp + crank;
      const uint32_t acc = tc & 1u, acc_ph = (tc >> 1) & 1u;
      // one outcome for the whole warp (tcgen05.ld below is warp-collective)
      const bool got = __all_sync(0xffffffffu,
                                  mbar_wait_bounded(&tmem_full[acc], acc_ph, abort_flag));
      if (!got) {
        give_up();
        break;
      }
      tc_fence_after();
      const int64_t row = mt * GBM + r_local;  // row of C
      const int64_t n0 = nt * GBN;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + acc * GBN;
      // per-row context
      bool row_ok = row < M;
      int32_t y = -1;
      float gscale = 0.0f, lse2 = 0.0f;
      int64_t orig = -1;
      if (EPI == EPI_G || EPI == EPI_ROWS) {
        const int64_t crow = p.chunk_row0 + row;
        const bool in_loss = row_ok && crow < static_cast<int64_t>(*p.n_valid);
        if (in_loss) orig = p.rowidx[crow];
        if (EPI == EPI_G && in_loss) {
          y = p.targets[orig];
          gscale = p.dlp[orig] * p.inv_tau;
          lse2 = p.lse[orig] * 1.4426950408889634f;
        }
        if (EPI == EPI_ROWS) row_ok = in_loss;
      }
#pragma unroll 1
      for (int c = 0; c < GBN; c += 32) {
        float v[32];
        tmem_ld_32x32b_x32(tbase + c, v);
        tmem_wait_ld();
        const int64_t col0 = n0 + c;
        if (EPI == EPI_G) {
          if (row_ok && col0 < p.g_cols) {
            // G = (g / tau) (onehot - p), zero for rows outside the loss
            uint32_t packed[16];
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              float g0 = 0.0f, g1 = 0.0f;
              if (gscale != 0.0f) {
                const float p0 = ex2_approx(fmaf(v[i], p.scale_log2, -lse2));
                const float p1 = ex2_approx(fmaf(v[i + 1], p.scale_log2, -lse2));
                g0 = col0 + i < p.V ? gscale * ((col0 + i == y ? 1.0f : 0.0f) - p0) : 0.0f;
                g1 = col0 + i + 1 < p.V ? gscale * ((col0 + i + 1 == y ? 1.0f : 0.0f) - p1) : 0.0f;
              }
              packed[i / 2] = static_cast<uint32_t>(f32_to_bf16_rn(g0)) |
                              (static_cast<uint32_t>(f32_to_bf16_rn(g1)) << 16);
            }
            // col0 is a multiple of 32, so the 32 columns lie in one 64-column block
            uint4* d4 = reinterpret_cast<uint4*>(
                p.g_out + ((col0 >> 6) * p.g_pitch + row) * 64 + (col0 & 63));
#pragma unroll
            for (int q = 0; q < 4; ++q)
              d4[q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2],
                                 packed[4 * q + 3]);
          }
        } else if (EPI == EPI_ROWS) {
          if (row_ok) {
            float* dst = p.rows_out + orig * p.ldo + col0;
            if (col0 + 32 <= p.N) {
              float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
              for (int q = 0; q < 8; ++q)
                d4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            } else {
              for (int i = 0; i < 32 && col0 + i < p.N; ++i) dst[i] = v[i];
            }
          }
        } else {
          if (row_ok) {
            float* dst = p.acc_out + row * p.ldo + col0;
            if (col0 + 32 <= p.N) {
              float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                float4 o = d4[q];
                o.x += v[4 * q];
                o.y += v[4 * q + 1];
                o.z += v[4 * q + 2];
                o.w += v[4 * q + 3];
                d4[q] = o;
              }
            } else {
              for (int i = 0; i < 32 && col0 + i < p.N; ++i) dst[i] += v[i];
            }
          }
        }
      }
      // one arrival per warp on the even CTA's barrier, after every lane's loads
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc ? empty1 : empty0);
    }
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA frees its tensor memory or leaves while the pair's MMAs, copies
  // or arrivals may still reach it
  cluster_sync();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, kGTmemCols);
  cluster_sync();  // the collective release is complete in both CTAs
}

// Zero the gathered rows from n_valid up to the next multiple of GBM (at most
// rows_end) of the compact buffer: dW reads whole GBM-row tiles of them, and the
// rows outside the loss must contribute exactly 0 (0 x garbage could be NaN).
__global__ void zero_tail_rows_kernel(uint4* __restrict__ buf, int64_t row_vecs,
                                      const long long* __restrict__ n_valid, int64_t rows_end) {
  const int64_t start = *n_valid;
  int64_t end = (start + GBM - 1) / GBM * GBM;
  if (end > rows_end) end = rows_end;
  const int64_t total = (end - start) * row_vecs;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    buf[start * row_vecs + i] = make_uint4(0, 0, 0, 0);
}

// dLoss/dlp per row of the clipped surrogate (oracle: oracle_surrogate_grad).
__global__ void surrogate_grad_kernel(const int64_t* __restrict__ seq_offsets,
                                      const uint8_t* __restrict__ seq_accepted,
                                      const uint8_t* __restrict__ mask,
                                      const float* __restrict__ logprob,
                                      const float* __restrict__ behav,
                                      const float* __restrict__ adv,
                                      const long long* __restrict__ seq_in,
                                      const long long* __restrict__ total, int64_t n_seq,
                                      int64_t n_rows, float eps_low, float eps_high, float dual,
                                      int agg, const int* __restrict__ n_seq_used,
                                      float* __restrict__ dlp) {
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    const int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows) continue;
    const bool acc = seq_accepted ? seq_accepted[i] != 0 : true;
    const float a = adv[i];
    const double scale = agg == PACE_AGG_TOKEN_MEAN
                             ? 1.0 / static_cast<double>(*total)
                             : 1.0 / (static_cast<double>(*n_seq_used) *
                                      static_cast<double>(seq_in[i]));
    for (int64_t r = r0 + threadIdx.x; r < r1; r += blockDim.x) {
      const bool in = acc && (mask ? mask[r] != 0 : true);
      float g = 0.0f;
      if (in) {
        const float d = logprob[r] - behav[r];
        const float dc = fminf(fmaxf(d, -20.0f), 20.0f);
        const float rho = expf(dc);
        const float rc = fminf(fmaxf(rho, 1.0f - eps_low), 1.0f + eps_high);
        const float p1 = -a * rho, p2 = -a * rc;
        const float l = fmaxf(p1, p2);
        if (d > -20.0f && d < 20.0f && p1 >= p2) g = -a * rho;
        if (a < 0.0f && -dual * a < l) g = 0.0f;
        g = static_cast<float>(static_cast<double>(g) * scale);
      }
      dlp[r] = g;
    }
  }
}

__global__ void count_used_seqs_kernel(const long long* __restrict__ seq_in, int64_t n_seq,
                                       int* __restrict__ out) {
  __shared__ int sh[256];
  int c = 0;
  for (int64_t i = threadIdx.x; i < n_seq; i += blockDim.x) c += seq_in[i] > 0;
  sh[threadIdx.x] = c;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) sh[threadIdx.x] += sh[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = sh[0];
}

// ---------------------------------------------------------------- host side

template <bool A_MN, bool B_MN, int EPI>
pace_status launch_gemm(const CUtensorMap& ta, const CUtensorMap& tb, GemmArgs a,
                        unsigned* round_ctr, cudaStream_t st) {
  constexpr int kMaxDevices = 64;
  static bool done[kMaxDevices] = {};  // shared-memory opt-in made on that device
  static std::mutex mu;
  int dev = 0;
  PACE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_CUDA;
  {
    std::lock_guard<std::mutex> g(mu);
    if (!done[dev]) {
      PACE_TRY_CUDA(cudaFuncSetAttribute(gemm_kernel<A_MN, B_MN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kGSmemBytes)));
      done[dev] = true;
    }
  }
  a.m_tiles = (a.M + GBM - 1) / GBM;
  a.n_tiles = (a.N + GBN - 1) / GBN;
  const int64_t items = (a.m_tiles + 1) / 2 * a.n_tiles;
  if (items == 0) return PACE_OK;
  const int64_t max_clusters = sm_count() / 2;
  const int64_t grid = 2 * (items < max_clusters ? items : max_clusters);
  PACE_TRY_CUDA(cudaMemsetAsync(round_ctr, 0, sizeof(unsigned), st));
  a.round_ctr = round_ctr;
  gemm_kernel<A_MN, B_MN, EPI><<<static_cast<unsigned>(grid), kGemmThreads, kGSmemBytes, st>>>(
      ta, tb, a);
  return last_launch_status();
}

struct BwWs {
  LmWs lm;            // compaction + gathered rows (hidden_c)
  uint16_t* g;        // bf16 G of one chunk, 64-column blocks [ceil(V / 64)][chunk][64]
  int* n_seq_used;
  unsigned* round_ctr;  // the GEMMs' pacing counter
};

int64_t chunk_rows(int64_t n_rows) {
  int64_t c = n_rows < kChunkRows ? n_rows : kChunkRows;
  return (c + GBM - 1) / GBM * GBM;
}

void carve_bw_ws(Carver& cv, int64_t n_rows, int64_t n_seq, int H, int V, BwWs* w) {
  carve_lm_ws(cv, n_rows, n_seq, H, true, &w->lm);
  const int64_t g_cols = (static_cast<int64_t>(V) + 63) / 64 * 64;
  w->g = cv.take<uint16_t>(static_cast<size_t>(chunk_rows(n_rows > 0 ? n_rows : 1)) * g_cols);
  w->n_seq_used = cv.take<int>(1);
  w->round_ctr = cv.take<unsigned>(1);
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_surrogate_backward_workspace_size(int64_t n_rows, int64_t n_seq) {
  Carver cv;
  CompactWs cw;
  SurrogateWs sw;
  carve_compact_ws(cv, n_seq, n_rows, &cw);
  carve_surrogate_ws(cv, n_seq, &sw);
  cv.take<int>(1);
  return cv.used;
}

extern "C" pace_status pace_surrogate_backward(const PaceBatch* batch, const float* logprob,
                                               const PaceLossArgs* loss, float* dlp,
                                               void* workspace, size_t workspace_bytes,
                                               int32_t* status_dev, void* stream) {
  PACE_TRY(check_batch(batch));
  PACE_TRY(check_loss_args(batch, loss));
  if (batch->n_rows > 0 && (!logprob || !dlp)) return PACE_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  CompactWs cw;
  SurrogateWs sw;
  carve_compact_ws(cv, batch->n_seq, batch->n_rows, &cw);
  carve_surrogate_ws(cv, batch->n_seq, &sw);
  int* n_used = cv.take<int>(1);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  cudaStream_t st = as_stream(stream);
  if (batch->n_rows > 0)
    PACE_TRY_CUDA(cudaMemsetAsync(dlp, 0, static_cast<size_t>(batch->n_rows) * 4, st));
  if (batch->n_seq == 0) return PACE_OK;
  float* adv = loss->adv ? loss->adv : sw.adv;
  PACE_TRY(launch_group_adv(loss->reward, batch->seq_accepted, batch->n_seq,
                                   loss->group_size, loss->params.adv_eps,
                                   loss->params.std_unbiased, adv, st));
  PACE_TRY(run_compaction(batch, cw, status_dev, st));  // rows in the loss per sequence
  count_used_seqs_kernel<<<1, 256, 0, st>>>(cw.seq_in, batch->n_seq, n_used);
  PACE_TRY(last_launch_status());
  int64_t grid = batch->n_seq;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  surrogate_grad_kernel<<<static_cast<unsigned>(grid), 256, 0, st>>>(
      batch->seq_offsets, batch->seq_accepted, batch->mask, logprob, loss->behav_lp, adv,
      cw.seq_in, cw.total, batch->n_seq, batch->n_rows, loss->params.eps_low,
      loss->params.eps_high, loss->params.dual_clip, loss->params.agg, n_used, dlp);
  return last_launch_status();
}

extern "C" size_t pace_token_logprob_backward_workspace_size(int64_t n_rows, int64_t n_seq,
                                                             int32_t hidden_size,
                                                             int32_t vocab_size) {
  if (n_rows < 0 || n_seq < 0 || hidden_size <= 0 || vocab_size <= 0) return 0;
  Carver cv;
  BwWs w;
  carve_bw_ws(cv, n_rows, n_seq, hidden_size, vocab_size, &w);
  return cv.used;
}

extern "C" pace_status pace_token_logprob_backward(
    const PaceBatch* batch, const void* hidden, const void* w_vocab, const int32_t* targets,
    int32_t hidden_size, int32_t vocab_size, float temperature, const float* lse,
    const float* dlp, float* grad_hidden, float* grad_w, void* workspace,
    size_t workspace_bytes, int32_t* status_dev, void* stream) {
  const int H = hidden_size, V = vocab_size;
  PACE_TRY(check_lm_args(batch, hidden, w_vocab, targets, H, V, temperature, dlp));
  if (batch->n_rows > 0 && (!lse || !grad_hidden || !grad_w)) return PACE_ERR_INVALID_ARG;
  if (!aligned(grad_hidden, 16) || !aligned(grad_w, 16)) return PACE_ERR_UNSUPPORTED_SHAPE;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  BwWs ws;
  carve_bw_ws(cv, batch->n_rows, batch->n_seq, H, V, &ws);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  cudaStream_t st = as_stream(stream);
  const int64_t n_rows = batch->n_rows;
  PACE_TRY_CUDA(cudaMemsetAsync(grad_w, 0, static_cast<size_t>(V) * H * 4, st));
  if (n_rows == 0) return PACE_OK;
  PACE_TRY_CUDA(cudaMemsetAsync(grad_hidden, 0, static_cast<size_t>(n_rows) * H * 4, st));
  // the rows in the loss, gathered densely (always compacted here)
  PACE_TRY(run_compaction(batch, ws.lm.cw, status_dev, st));
  PACE_TRY(run_gather(hidden, H, n_rows, ws.lm.cw, ws.lm.hidden_c, st));
  const int64_t rows_cap = n_rows > 128 ? n_rows : 128;
  const int64_t row_vecs = static_cast<int64_t>(H) * 2 / 16;
  zero_tail_rows_kernel<<<static_cast<unsigned>(sm_count() * 4), 256, 0, st>>>(
      static_cast<uint4*>(ws.lm.hidden_c), row_vecs, ws.lm.cw.total, rows_cap);
  PACE_TRY(last_launch_status());
  const int64_t chunk = chunk_rows(n_rows);
  const int64_t g_cols = (static_cast<int64_t>(V) + 63) / 64 * 64;
  const int64_t g_blocks = g_cols / 64;
  // TMA row coordinates of the blocked G are 32-bit
  if (g_blocks * chunk > static_cast<int64_t>(INT32_MAX)) return PACE_ERR_UNSUPPORTED_SHAPE;
  for (int64_t c0 = 0; c0 < n_rows; c0 += chunk) {
    const int64_t rows_c = (n_rows - c0) < chunk ? (n_rows - c0) : chunk;
    const int64_t rows_c_pad = (rows_c + GBM - 1) / GBM * GBM;
    const void* hc = static_cast<const uint16_t*>(ws.lm.hidden_c) + c0 * H;
    // rows of the gathered buffer from c0 on (the padded tail of a chunk past the
    // buffer is read as zeros by TMA)
    const int64_t hc_rows = (rows_cap - c0) < rows_c_pad ? (rows_cap - c0) : rows_c_pad;
    // 1. G = (g / tau) (onehot - softmax) for the chunk's rows (bf16)
    {
      CUtensorMap ta, tb;
      PACE_TRY(encode_bf16_2d(&ta, hc, hc_rows, H, H, 64, GBM));
      PACE_TRY(encode_bf16_2d(&tb, w_vocab, V, H, H, 64, GBN / 2));
      GemmArgs a = {};
      a.M = rows_c_pad;
      a.N = V;
      a.K = H;
      a.raster_n_fast = 0;
      a.trim = TRIM_M;
      a.chunk_row0 = c0;
      a.n_valid = ws.lm.cw.total;
      a.rowidx = ws.lm.cw.rowidx;
      a.targets = targets;
      a.lse = lse;
      a.dlp = dlp;
      a.scale_log2 = 1.4426950408889634f / temperature;
      a.inv_tau = 1.0f / temperature;
      a.g_out = ws.g;
      a.g_cols = g_cols;
      a.g_pitch = rows_c_pad;
      a.V = V;
      a.status = status_dev;
      PACE_TRY((launch_gemm<false, false, EPI_G>(ta, tb, a, ws.round_ctr, st)));
    }
    // 2. dH rows = G W   (W read MN-major: [K = V][N = H])
    {
      CUtensorMap ta, tb;
      PACE_TRY(encode_bf16_2d(&ta, ws.g, g_blocks * rows_c_pad, 64, 64, 64, GBM));
      PACE_TRY(encode_bf16_2d(&tb, w_vocab, V, H, H, 64, 64));
      GemmArgs a = {};
      a.M = rows_c_pad;
      a.N = H;
      a.K = V;
      a.a_pitch = rows_c_pad;
      a.raster_n_fast = 1;
      a.trim = TRIM_M;
      a.chunk_row0 = c0;
      a.n_valid = ws.lm.cw.total;
      a.rowidx = ws.lm.cw.rowidx;
      a.rows_out = grad_hidden;
      a.ldo = H;
      a.status = status_dev;
      PACE_TRY((launch_gemm<false, true, EPI_ROWS>(ta, tb, a, ws.round_ctr, st)));
    }
    // 3. dW += G^T H_c   (G read MN-major: [K = rows][M = V]; H_c MN-major: [K = rows][N = H])
    {
      CUtensorMap ta, tb;
      PACE_TRY(encode_bf16_2d(&ta, ws.g, g_blocks * rows_c_pad, 64, 64, 64, 64));
      PACE_TRY(encode_bf16_2d(&tb, hc, hc_rows, H, H, 64, 64));
      GemmArgs a = {};
      a.M = V;
      a.N = H;
      a.K = rows_c_pad;
      a.a_pitch = rows_c_pad;
      a.raster_n_fast = 1;
      a.trim = TRIM_K;
      a.chunk_row0 = c0;
      a.n_valid = ws.lm.cw.total;
      a.acc_out = grad_w;
      a.ldo = H;
      a.status = status_dev;
      PACE_TRY((launch_gemm<true, true, EPI_ACC>(ta, tb, a, ws.round_ctr, st)));
    }
  }
  return PACE_OK;
}
