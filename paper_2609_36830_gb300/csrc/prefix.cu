// Prefix Forgetting Score on the GPU (Eq. 6, Sec. 3.2): the rows of each
// interrupted prefix are re-scored under the updated rollout policy with the
// fused LM head, and each prefix gets the mean absolute log-ratio against the
// recorded behaviour log-probs over its first cap_tokens eligible tokens
// (admission settings: at least 32 eligible tokens; caps of 1,024 / 2,048).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "pace_block.cuh"
#include "pace_internal.cuh"
#include "pace_loss.cuh"

namespace pace {
namespace {

constexpr int kThreads = 256;

// Per prefix: keep the first cap eligible rows (row order), count all eligible.
__global__ void __launch_bounds__(kThreads)
    cap_mask_kernel(const int64_t* __restrict__ seq_offsets,
                    const uint8_t* __restrict__ seq_accepted, const uint8_t* __restrict__ mask,
                    int64_t n_seq, int64_t n_rows, int32_t cap, uint8_t* __restrict__ mask_c,
                    long long* __restrict__ n_elig, int32_t* status) {
  __shared__ int warp_sums[kThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    const int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows || (i == 0 && r0 != 0)) {
      if (threadIdx.x == 0) {
        report(status, PACE_ERR_INVALID_ARG);
        n_elig[i] = 0;
      }
      continue;
    }
    const bool acc = seq_accepted ? seq_accepted[i] != 0 : true;
    long long base = 0;
    for (int64_t c0 = r0; c0 < r1; c0 += kThreads) {
      const int64_t r = c0 + threadIdx.x;
      const int in = (r < r1) && acc && (mask ? mask[r] != 0 : 1);
      const unsigned bal = __ballot_sync(0xffffffffu, in);
      if (lane == 0) warp_sums[wid] = __popc(bal);
      __syncthreads();
      int before = 0, tot = 0;
      for (int w = 0; w < kThreads / 32; ++w) {
        before += w < wid ? warp_sums[w] : 0;
        tot += warp_sums[w];
      }
      before += __popc(bal & ((1u << lane) - 1u));
      if (r < r1) mask_c[r] = (in && base + before < cap) ? 1 : 0;
      base += tot;
      __syncthreads();
    }
    if (threadIdx.x == 0) n_elig[i] = base;
  }
}

__global__ void __launch_bounds__(kThreads)
    prefix_reduce_kernel(const int64_t* __restrict__ seq_offsets,
                         const uint8_t* __restrict__ mask_c, const long long* __restrict__ n_elig,
                         const float* __restrict__ logprob, const float* __restrict__ behav,
                         int64_t n_seq, int64_t n_rows, int32_t min_tokens, int32_t cap,
                         float* __restrict__ s_pre) {
  __shared__ double sh[kThreads];
  for (int64_t i = blockIdx.x; i < n_seq; i += gridDim.x) {
    int64_t r0 = seq_offsets[i], r1 = seq_offsets[i + 1];
    if (r1 < r0 || r0 < 0 || r1 > n_rows) r0 = r1 = 0;
    const long long ne = n_elig[i];
    double acc = 0.0;
    if (ne >= min_tokens)
      for (int64_t r = r0 + threadIdx.x; r < r1; r += kThreads)
        if (mask_c[r])
          acc = __dadd_rn(acc, fabs(static_cast<double>(logprob[r]) - static_cast<double>(behav[r])));
    const double tot = block_sum_fixed<kThreads>(acc, sh);
    if (threadIdx.x == 0) {
      const long long m = ne < cap ? ne : cap;
      s_pre[i] = ne >= min_tokens ? static_cast<float>(__ddiv_rn(tot, static_cast<double>(m)))
                                  : __int_as_float(0x7fc00000);
    }
  }
}

struct PrefixWs {
  LmWs lm;
  uint8_t* mask_c;
  long long* n_elig;
  float* logprob;
};

void carve_prefix_ws(Carver& cv, int64_t n_rows, int64_t n_seq, int H, PrefixWs* w) {
  carve_lm_ws(cv, n_rows, n_seq, H, false, &w->lm);
  w->mask_c = cv.take<uint8_t>(n_rows > 0 ? n_rows : 1);
  w->n_elig = cv.take<long long>(n_seq > 0 ? n_seq : 1);
  w->logprob = cv.take<float>(n_rows > 0 ? n_rows : 1);
}

}  // namespace
}  // namespace pace

using namespace pace;

extern "C" size_t pace_prefix_score_workspace_size(int64_t n_rows, int64_t n_seq,
                                                   int32_t hidden_size, int32_t vocab_size) {
  if (n_rows < 0 || n_seq < 0 || hidden_size <= 0 || vocab_size <= 0) return 0;
  Carver cv;
  PrefixWs w;
  carve_prefix_ws(cv, n_rows, n_seq, hidden_size, &w);
  return cv.used;
}

extern "C" pace_status pace_prefix_score(const PaceBatch* batch, const void* hidden,
                                         const void* w_vocab, const int32_t* targets,
                                         const float* behav_lp, int32_t hidden_size,
                                         int32_t vocab_size, float temperature,
                                         int32_t min_tokens, int32_t cap_tokens, float* s_pre,
                                         float* logprob, void* workspace,
                                         size_t workspace_bytes, int32_t* status_dev,
                                         void* stream) {
  PACE_TRY(check_batch(batch));
  if (min_tokens < 1 || cap_tokens < 1) return PACE_ERR_INVALID_ARG;
  if (batch->n_seq > 0 && !s_pre) return PACE_ERR_INVALID_ARG;
  if (batch->n_rows > 0 && !behav_lp) return PACE_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return PACE_ERR_WORKSPACE;
  Carver cv(workspace, workspace_bytes);
  PrefixWs ws;
  carve_prefix_ws(cv, batch->n_rows, batch->n_seq, hidden_size, &ws);
  if (!cv.fits()) return PACE_ERR_WORKSPACE;
  float* lp = logprob ? logprob : ws.logprob;
  PACE_TRY(check_lm_args(batch, hidden, w_vocab, targets, hidden_size, vocab_size, temperature,
                         lp));
  if (batch->n_seq == 0) return PACE_OK;
  cudaStream_t st = as_stream(stream);
  int64_t grid = batch->n_seq;
  const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
  if (grid > cap) grid = cap;
  cap_mask_kernel<<<static_cast<unsigned>(grid), kThreads, 0, st>>>(
      batch->seq_offsets, batch->seq_accepted, batch->mask, batch->n_seq, batch->n_rows,
      cap_tokens, ws.mask_c, ws.n_elig, status_dev);
  PACE_TRY(last_launch_status());
  // the scored rows: the first cap_tokens eligible rows of every prefix
  PaceBatch scored = *batch;
  scored.seq_accepted = nullptr;
  scored.mask = ws.mask_c;
  PACE_TRY(run_logprob(&scored, hidden, w_vocab, targets, hidden_size, vocab_size, temperature,
                       lp, nullptr, ws.lm, status_dev, st));
  prefix_reduce_kernel<<<static_cast<unsigned>(grid), kThreads, 0, st>>>(
      batch->seq_offsets, ws.mask_c, ws.n_elig, lp, behav_lp, batch->n_seq, batch->n_rows,
      min_tokens, cap_tokens, s_pre);
  return last_launch_status();
}
