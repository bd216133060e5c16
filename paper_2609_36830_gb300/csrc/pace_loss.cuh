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

void carve_surrogate_ws(Carver& cv, int64_t n_seq, SurrogateWs* w);
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
