// GRPO advantages, the asymmetric dual-clipped token-mean surrogate, and the
// row compaction that feeds the fused LM head (shared training settings of
// the paper's appendix: GRPO with within-group standardisation, clip widths
// 0.20 / 0.28, dual-clip coefficient 10, token-mean aggregation; tool output
// kept in context but masked from the loss).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "pace_block.cuh"
#include "pace_internal.cuh"
#include "pace_loss.cuh"

namespace pace {

// ------------------------------------------------------------ advantages

// One thread per prompt group: mean and standard deviation of the accepted
// members' rewards in fp64, summed from the lowest index up, then
// A_i = (R_i - mean) / (std + eps).
__global__ void group_adv_kernel(const float* __restrict__ reward,
                                 const uint8_t* __restrict__ accepted, int64_t n_groups, int G,
                                 double eps, int unbiased, float* __restrict__ adv) {
  const int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (g >= n_groups) return;
  const int64_t i0 = g * G;
  int64_t n = 0;
  double sum = 0.0;
  for (int k = 0; k < G; ++k) {
    if (accepted && !accepted[i0 + k]) continue;
    sum = __dadd_rn(sum, static_cast<double>(reward[i0 + k]));
    ++n;
  }
  const double mean = n > 0 ? __ddiv_rn(sum, static_cast<double>(n)) : 0.0;
  double ss = 0.0;
  for (int k = 0; k < G; ++k) {
    if (accepted && !accepted[i0 + k]) continue;
    const double d = __dsub_rn(static_cast<double>(reward[i0 + k]), mean);
    ss = __dadd_rn(ss, __dmul_rn(d, d));
  }
  const int64_t div = unbiased ? n - 1 : n;
  const double sd = div > 0 ? __dsqrt_rn(__ddiv_rn(ss, static_cast<double>(div))) : 0.0;
  const double den = __dadd_rn(sd, eps);
  for (int k = 0; k < G; ++k) {
    double a = 0.0;
    if (!accepted || accepted[i0 + k]) {
      const double d = __dsub_rn(static_cast<double>(reward[i0 + k]), mean);
      a = d == 0.0 ? 0.0 : __ddiv_rn(d, den);
    }
    adv[i0 + k] = static_cast<float>(a);
  }
}

pace_status launch_group_adv(const float* reward, const uint8_t* accepted, int64_t n_seq, int G,
                             float eps, int unbiased, float* adv, cudaStream_t st) {
  const int64_t n_groups = n_seq / G;
  if (n_groups == 0) return PACE_OK;
  const int threads = 128;
  group_adv_kernel<<<static_cast<unsigned>((n_groups + threads - 1) / threads), threads, 0, st>>>(
      reward, accepted, n_groups, G, static_cast<double>(eps), unbiased, adv);
  return last_launch_status();
}

// ------------------------------------------------------------ surrogate

constexpr int kSurThreads = 256;

__device__ __forceinline__ float clipped_term(float lp, float behav, float a, float eps_low,
                                              float eps_high, float dual, float* rho_out) {
  float d = lp - behav;
  d = fminf(fmaxf(d, -20.0f), 20.0f);
  const float rho = expf(d);
  const float rc = fminf(fmaxf(rho, 1.0f - eps_low), 1.0f + eps_high);
  const float p1 = -a * rho;
  const float p2 = -a * rc;
  float l = fmaxf(p1, p2);
  if (a < 0.0f) l = fminf(l, -dual * a);
  *rho_out = rho;
  return l;
}

// One block per sequence (grid-stride): per-token terms in fp32, the
// sequence's sum and count in fp64 with a fixed reduction shape.
__global__ void __launch_bounds__(kSurThreads)
    surrogate_seq_kernel(const int64_t* __restrict__ seq_offsets,
                         const uint8_t* __restrict__ seq_accepted,
                         const uint8_t* __restrict__ mask, const float* __restrict__ logprob,
                         const float* __restrict__ behav, const float* __restrict__ adv,
                         int64_t n_seq, float eps_low, float eps_high, float dual,
                         int64_t n_rows, float* __restrict__ ratio,
                         double* __restrict__ seq_sum, double* __restrict__ seq_cnt,
                         int32_t* status) {
  __shared__ double sh[kSurThreads];
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows || (i == 0 && r0 != 0)) {
      if (threadIdx.x == 0) report(status, PACE_ERR_INVALID_ARG);
      r0 = r1 = 0;
    }
    const bool acc = seq_accepted ? seq_accepted[i] != 0 : true;
    const float a = adv[i];
    double tot = 0.0, cnt = 0.0;
    for (int64_t r = r0 + threadIdx.x; r < r1; r += kSurThreads) {
      const bool in = acc && (mask ? mask[r] != 0 : true);
      float rho = 0.0f;
      if (in) {
        const float l = clipped_term(logprob[r], behav[r], a, eps_low, eps_high, dual, &rho);
        tot = __dadd_rn(tot, static_cast<double>(l));
        cnt = __dadd_rn(cnt, 1.0);
      }
      if (ratio) ratio[r] = in ? rho : 0.0f;
    }
    const double ts = block_sum_fixed<kSurThreads>(tot, sh);
    const double tc = block_sum_fixed<kSurThreads>(cnt, sh);
    if (threadIdx.x == 0) {
      seq_sum[i] = ts;
      seq_cnt[i] = tc;
    }
  }
}

// One block: the aggregate over sequences in a fixed order.
__global__ void __launch_bounds__(kSurThreads)
    surrogate_reduce_kernel(const double* __restrict__ seq_sum,
                            const double* __restrict__ seq_cnt, int64_t n_seq, int agg,
                            double* __restrict__ loss, double* __restrict__ partial) {
  __shared__ double sh[kSurThreads];
  double a = 0.0, b = 0.0;
  for (int64_t i = threadIdx.x; i < n_seq; i += kSurThreads) {
    if (agg == PACE_AGG_TOKEN_MEAN) {
      a = __dadd_rn(a, seq_sum[i]);
      b = __dadd_rn(b, seq_cnt[i]);
    } else if (seq_cnt[i] > 0.0) {
      a = __dadd_rn(a, __ddiv_rn(seq_sum[i], seq_cnt[i]));
      b = __dadd_rn(b, 1.0);
    }
  }
  const double ta = block_sum_fixed<kSurThreads>(a, sh);
  const double tb = block_sum_fixed<kSurThreads>(b, sh);
  if (threadIdx.x == 0) {
    *loss = tb > 0.0 ? __ddiv_rn(ta, tb) : 0.0;
    if (partial) {
      partial[0] = ta;
      partial[1] = tb;
    }
  }
}

// loss = numerator / denominator of partials summed over the parts of a batch
// (0 for an empty loss), the same correctly rounded division as above.
__global__ void loss_from_partial_kernel(const double* __restrict__ partial,
                                         double* __restrict__ loss) {
  if (threadIdx.x == 0 && blockIdx.x == 0)
    *loss = partial[1] > 0.0 ? __ddiv_rn(partial[0], partial[1]) : 0.0;
}

void carve_surrogate_ws(Carver& cv, int64_t n_seq, SurrogateWs* w) {
  w->seq_sum = cv.take<double>(n_seq > 0 ? n_seq : 1);
  w->seq_cnt = cv.take<double>(n_seq > 0 ? n_seq : 1);
  w->adv = cv.take<float>(n_seq > 0 ? n_seq : 1);
}

pace_status check_batch(const PaceBatch* b) {
  if (!b) return PACE_ERR_INVALID_ARG;
  if (b->n_seq < 0 || b->n_rows < 0) return PACE_ERR_INVALID_ARG;
  if (b->n_seq > 0 && !b->seq_offsets) return PACE_ERR_INVALID_ARG;
  if (b->n_rows >= (int64_t(1) << 31)) return PACE_ERR_UNSUPPORTED_SHAPE;
  return PACE_OK;
}

pace_status check_loss_args(const PaceBatch* b, const PaceLossArgs* l) {
  if (!l || !l->behav_lp || !l->reward || !l->loss) return PACE_ERR_INVALID_ARG;
  if (l->group_size < 1 || b->n_seq % l->group_size != 0) return PACE_ERR_INVALID_ARG;
  const PaceLossParams& p = l->params;
  if (!(p.eps_low >= 0.0f && p.eps_low < 1.0f) || !(p.eps_high >= 0.0f) ||
      !(p.dual_clip >= 1.0f) || !(p.adv_eps >= 0.0f))
    return PACE_ERR_INVALID_ARG;
  if (p.agg != PACE_AGG_TOKEN_MEAN && p.agg != PACE_AGG_SEQ_MEAN_TOKEN_MEAN)
    return PACE_ERR_INVALID_ARG;
  return PACE_OK;
}

// Advantages, per-token terms and the aggregate; logprob is [n_rows].
pace_status run_surrogate(const PaceBatch* b, const float* logprob, const PaceLossArgs* l,
                          const SurrogateWs& ws, int32_t* status, cudaStream_t st) {
  float* adv = l->adv ? l->adv : ws.adv;
  PACE_TRY(launch_group_adv(l->reward, b->seq_accepted, b->n_seq, l->group_size,
                            l->params.adv_eps, l->params.std_unbiased, adv, st));
  if (b->n_seq > 0) {
    int64_t grid = b->n_seq;
    const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
    if (grid > cap) grid = cap;
    surrogate_seq_kernel<<<static_cast<unsigned>(grid), kSurThreads, 0, st>>>(
        b->seq_offsets, b->seq_accepted, b->mask, logprob, l->behav_lp, adv, b->n_seq,
        l->params.eps_low, l->params.eps_high, l->params.dual_clip, b->n_rows, l->ratio,
        ws.seq_sum, ws.seq_cnt, status);
    PACE_TRY(last_launch_status());
  }
  surrogate_reduce_kernel<<<1, kSurThreads, 0, st>>>(ws.seq_sum, ws.seq_cnt, b->n_seq,
                                                     l->params.agg, l->loss, l->partial);
  return last_launch_status();
}

// ------------------------------------------------------------ compaction

constexpr int kCompThreads = 256;

// Per sequence: number of rows in the loss.
__global__ void __launch_bounds__(kCompThreads)
    count_rows_kernel(const int64_t* __restrict__ seq_offsets,
                      const uint8_t* __restrict__ seq_accepted, const uint8_t* __restrict__ mask,
                      int64_t n_seq, int64_t n_rows, long long* __restrict__ seq_in,
                      int32_t* status) {
  __shared__ long long sh[kCompThreads];
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    const int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows || (i == 0 && r0 != 0)) {
      if (threadIdx.x == 0) {
        report(status, PACE_ERR_INVALID_ARG);
        seq_in[i] = 0;
      }
      continue;
    }
    const bool acc = seq_accepted ? seq_accepted[i] != 0 : true;
    long long c = 0;
    if (acc)
      for (int64_t r = r0 + threadIdx.x; r < r1; r += kCompThreads) c += mask ? (mask[r] != 0) : 1;
    sh[threadIdx.x] = c;
    __syncthreads();
    for (int o = kCompThreads / 2; o > 0; o >>= 1) {
      if (threadIdx.x < o) sh[threadIdx.x] += sh[threadIdx.x + o];
      __syncthreads();
    }
    if (threadIdx.x == 0) seq_in[i] = sh[0];
    __syncthreads();
  }
}

// One block: exclusive scan of the per-sequence counts; total rows in M.
__global__ void __launch_bounds__(1024)
    scan_rows_kernel(const long long* __restrict__ seq_in, int64_t n_seq, int64_t n_rows,
                     long long* __restrict__ seq_base, long long* __restrict__ total) {
  __shared__ long long warp_sums[32];
  __shared__ long long carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int64_t i0 = 0; i0 < n_seq; i0 += blockDim.x) {
    const int64_t i = i0 + threadIdx.x;
    const long long v = i < n_seq ? seq_in[i] : 0;
    long long x = v;
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[wid] = x;
    __syncthreads();
    if (wid == 0) {
      long long w = warp_sums[lane];
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      warp_sums[lane] = w;
    }
    __syncthreads();
    const long long before = (wid > 0 ? warp_sums[wid - 1] : 0) + x - v;
    if (i < n_seq) seq_base[i] = carry + before;
    __syncthreads();
    if (threadIdx.x == 0) carry += warp_sums[31];
    __syncthreads();
  }
  // overlapping sequences (reported by count_rows_kernel) must not overflow rowidx
  if (threadIdx.x == 0) *total = carry < n_rows ? carry : n_rows;
}

// Per sequence: write the original row index of every row in the loss, in
// row order, at the sequence's base offset.
__global__ void __launch_bounds__(kCompThreads)
    write_rows_kernel(const int64_t* __restrict__ seq_offsets,
                      const uint8_t* __restrict__ seq_accepted, const uint8_t* __restrict__ mask,
                      int64_t n_seq, int64_t n_rows, const long long* __restrict__ seq_base,
                      int32_t* __restrict__ rowidx) {
  __shared__ int warp_sums[kCompThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    const int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows) continue;
    if (seq_accepted && !seq_accepted[i]) continue;
    long long base = seq_base[i];
    for (int64_t c0 = r0; c0 < r1; c0 += kCompThreads) {
      const int64_t r = c0 + threadIdx.x;
      const int in = (r < r1) && (mask ? mask[r] != 0 : 1);
      const unsigned bal = __ballot_sync(0xffffffffu, in);
      if (lane == 0) warp_sums[wid] = __popc(bal);
      __syncthreads();
      int before = 0, tot = 0;
      for (int w = 0; w < kCompThreads / 32; ++w) {
        before += w < wid ? warp_sums[w] : 0;
        tot += warp_sums[w];
      }
      before += __popc(bal & ((1u << lane) - 1u));
      if (in && base + before < n_rows) rowidx[base + before] = static_cast<int32_t>(r);
      base += tot;
      __syncthreads();
    }
  }
}

// Copy the hidden rows listed in rowidx into a dense buffer, one warp per row,
// 16 bytes per lane per step.
__global__ void gather_rows_kernel(const uint4* __restrict__ hidden, int64_t row_vecs,
                                   const int32_t* __restrict__ rowidx,
                                   const long long* __restrict__ n_in, uint4* __restrict__ out) {
  const long long m = *n_in;
  const int lane = threadIdx.x & 31;
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; r < m;
       r += warps) {
    const uint4* src = hidden + static_cast<int64_t>(rowidx[r]) * row_vecs;
    uint4* dst = out + r * row_vecs;
    for (int64_t v = lane; v < row_vecs; v += 32) dst[v] = __ldg(src + v);
  }
}

void carve_compact_ws(Carver& cv, int64_t n_seq, int64_t n_rows, CompactWs* w) {
  w->seq_in = cv.take<long long>(n_seq > 0 ? n_seq : 1);
  w->seq_base = cv.take<long long>(n_seq > 0 ? n_seq : 1);
  w->total = cv.take<long long>(1);
  w->rowidx = cv.take<int32_t>(n_rows > 0 ? n_rows : 1);
}

pace_status run_compaction(const PaceBatch* b, const CompactWs& ws, int32_t* status,
                           cudaStream_t st) {
  if (b->n_seq == 0) {
    PACE_TRY_CUDA(cudaMemsetAsync(ws.total, 0, sizeof(long long), st));
    return PACE_OK;
  }
  int64_t grid = b->n_seq;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  count_rows_kernel<<<static_cast<unsigned>(grid), kCompThreads, 0, st>>>(
      b->seq_offsets, b->seq_accepted, b->mask, b->n_seq, b->n_rows, ws.seq_in, status);
  PACE_TRY(last_launch_status());
  scan_rows_kernel<<<1, 1024, 0, st>>>(ws.seq_in, b->n_seq, b->n_rows, ws.seq_base, ws.total);
  PACE_TRY(last_launch_status());
  write_rows_kernel<<<static_cast<unsigned>(grid), kCompThreads, 0, st>>>(
      b->seq_offsets, b->seq_accepted, b->mask, b->n_seq, b->n_rows, ws.seq_base, ws.rowidx);
  return last_launch_status();
}

pace_status run_gather(const void* hidden, int H, int64_t n_rows, const CompactWs& ws,
                       void* out, cudaStream_t st) {
  if (n_rows == 0) return PACE_OK;
  const int64_t row_vecs = static_cast<int64_t>(H) * 2 / 16;
  int64_t blocks = (n_rows + 7) / 8;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  gather_rows_kernel<<<static_cast<unsigned>(blocks), 256, 0, st>>>(
      static_cast<const uint4*>(hidden), row_vecs, ws.rowidx, ws.total,
      static_cast<uint4*>(out));
  return last_launch_status();
}

}  // namespace pace

using namespace pace;

extern "C" void pace_loss_params_default(PaceLossParams* p) {
  if (!p) return;
  p->eps_low = 0.2f;
  p->eps_high = 0.28f;
  p->dual_clip = 10.0f;
  p->adv_eps = 1e-6f;
  p->agg = PACE_AGG_TOKEN_MEAN;
  p->std_unbiased = 1;
}

extern "C" pace_status pace_group_advantages(const float* reward, const uint8_t* seq_accepted,
                                             int64_t n_seq, int32_t group_size, float adv_eps,
                                             int32_t std_unbiased, float* adv, void* stream) {
  if (n_seq < 0 || group_size < 1 || n_seq % group_size != 0) return PACE_ERR_INVALID_ARG;
  if (n_seq > 0 && (!reward || !adv)) return PACE_ERR_INVALID_ARG;
  if (!(adv_eps >= 0.0f)) return PACE_ERR_INVALID_ARG;
  return launch_group_adv(reward, seq_accepted, n_seq, group_size, adv_eps, std_unbiased, adv,
                          as_stream(stream));
}

extern "C" size_t pace_surrogate_loss_workspace_size(int64_t n_rows, int64_t n_seq) {
  (void)n_rows;
  Carver cv;
  SurrogateWs w;
  carve_surrogate_ws(cv, n_seq, &w);
  return cv.used;
}

extern "C" pace_status pace_surrogate_loss(const PaceBatch* batch, const float* logprob,
                                           const PaceLossArgs* loss, void* workspace,
                                           size_t workspace_bytes, int32_t* status_dev,
                                           void* stream) {
  PACE_TRY(check_batch(batch));
  PACE_TRY(check_loss_args(batch, loss));
  if (batch->n_rows > 0 && !logprob) return PACE_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  SurrogateWs ws;
  carve_surrogate_ws(cv, batch->n_seq, &ws);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  return run_surrogate(batch, logprob, loss, ws, status_dev, as_stream(stream));
}

extern "C" pace_status pace_loss_from_partial(const double* partial, double* loss,
                                              void* stream) {
  if (!partial || !loss) return PACE_ERR_INVALID_ARG;
  pace::loss_from_partial_kernel<<<1, 32, 0, pace::as_stream(stream)>>>(partial, loss);
  return pace::last_launch_status();
}
