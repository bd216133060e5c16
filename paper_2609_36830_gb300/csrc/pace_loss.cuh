// Internal interface between the surrogate / compaction code and the fused
// LM-head entry point.
#pragma once

#include "pace_internal.cuh"

namespace pace {

struct SurrogateWs {
  double* seq_sum;
  double* seq_cnt;
  float* adv;
};

struct CompactWs {
  long long* seq_in;    // rows in the loss per sequence
  long long* seq_base;  // exclusive scan of seq_in
  long long* total;     // M, the number of rows in the loss (clamped to n_rows)
  int32_t* rowidx;      // [n_rows]: compact row -> original row
};

// Workspace of the log-prob pipeline (compaction, gathered rows, split partials).
struct LmWs {
  CompactWs cw;
  SurrogateWs sw;
  void* hidden_c;  // dense copy of the rows in the loss [max(n_rows, 128)][H] (backward
                   // only; null for the forward, whose LM head reads rows by index)
  float* part_m;
  float* part_s;
  float* tgt;
  unsigned* round_ctr;  // the LM head's pacing counter (items whose loads were issued)
};

void carve_surrogate_ws(Carver& cv, int64_t n_seq, SurrogateWs* w);
pace_status launch_group_adv(const float* reward, const uint8_t* accepted, int64_t n_seq, int G,
                             float eps, int unbiased, float* adv, cudaStream_t st);
void carve_lm_ws(Carver& cv, int64_t n_rows, int64_t n_seq, int H, bool dense_rows,
                 LmWs* w);
bool lm_needs_compaction(const PaceBatch* b);
pace_status check_lm_args(const PaceBatch* batch, const void* hidden, const void* w_vocab,
                          const int32_t* targets, int H, int V, float temperature,
                          const float* logprob);
pace_status run_logprob(const PaceBatch* batch, const void* hidden, const void* w_vocab,
                        const int32_t* targets, int H, int V, float temperature, float* logprob,
                        float* lse, const LmWs& ws, int32_t* status_dev, cudaStream_t st);
void carve_compact_ws(Carver& cv, int64_t n_seq, int64_t n_rows, CompactWs* w);
pace_status check_batch(const PaceBatch* b);
pace_status check_loss_args(const PaceBatch* b, const PaceLossArgs* l);
pace_status run_surrogate(const PaceBatch* b, const float* logprob, const PaceLossArgs* l,
                          const SurrogateWs& ws, int32_t* status, cudaStream_t st);
pace_status run_compaction(const PaceBatch* b, const CompactWs& ws, int32_t* status,
                           cudaStream_t st);
pace_status run_gather(const void* hidden, int H, int64_t n_rows, const CompactWs& ws,
                       void* out, cudaStream_t st);

}  // namespace pace
