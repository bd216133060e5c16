/* A plain C client of the PACE C ABI that runs the scoring, selection and
 * log-probability calls on the GPU with no Python or torch in the process:
 * device memory comes from cudaMalloc, every call takes the legacy default
 * stream.
 *
 *   pace_gpu_c <input file> <output file> <eps_low> <eps_high>
 *
 * Input (little-endian): int64 n_traj, n_tokens, n_rows, hidden, vocab,
 * window_len, group_size, n_target, trainer_version; then tags int32[n_tokens],
 * offsets int64[n_traj+1], c_version int32[n_traj], s_pre float32[n_traj],
 * window float32[window_len], row_offsets int64[n_traj+1], mask uint8[n_rows],
 * targets int32[n_rows], hidden bf16 bits uint16[n_rows*hidden], w_vocab bf16
 * bits uint16[vocab*hidden], behav_lp float32[n_rows], reward float32[n_traj].
 * A second log-prob call also computes the fused loss (GRPO advantages over the
 * accepted group members and the clipped surrogate, default loss parameters
 * with the given clip widths).
 * Output: int32 host status of the four calls and the device status word,
 * int64 k, float64 r_hat, float64 unit_score[n_traj/G], uint8 flags[n_traj],
 * float32 logprob[n_rows], float64 loss, float32 adv[n_traj].  Exit code 0
 * when every step ran. */
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime.h>

#include "pace.h"

#define CHECK_CUDA(x)                                                           \
  do {                                                                          \
    cudaError_t e_ = (x);                                                       \
    if (e_ != cudaSuccess) {                                                    \
      fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));                  \
      return 2;                                                                 \
    }                                                                           \
  } while (0)

static void* read_array(FILE* f, size_t bytes) {
  void* p = malloc(bytes > 0 ? bytes : 1);
  if (p && bytes > 0 && fread(p, 1, bytes, f) != bytes) {
    free(p);
    return NULL;
  }
  return p;
}

static void* to_device(const void* host, size_t bytes) {
  void* d = NULL;
  if (cudaMalloc(&d, bytes > 0 ? bytes : 1) != cudaSuccess) return NULL;
  if (bytes > 0 && cudaMemcpy(d, host, bytes, cudaMemcpyHostToDevice) != cudaSuccess) return NULL;
  return d;
}

int main(int argc, char** argv) {
  int64_t hdr[9];
  FILE* f;
  if (argc != 5) return 1;
  f = fopen(argv[1], "rb");
  if (!f || fread(hdr, sizeof(int64_t), 9, f) != 9) return 1;
  {
    const int64_t n_traj = hdr[0], n_tokens = hdr[1], n_rows = hdr[2];
    const int32_t H = (int32_t)hdr[3], V = (int32_t)hdr[4];
    const int64_t wlen = hdr[5];
    const int32_t G = (int32_t)hdr[6];
    const int64_t n_target = hdr[7];
    const int32_t j = (int32_t)hdr[8];
    const int64_t U = n_traj / G;
    void* h_tags = read_array(f, (size_t)n_tokens * 4);
    void* h_off = read_array(f, (size_t)(n_traj + 1) * 8);
    void* h_c = read_array(f, (size_t)n_traj * 4);
    void* h_spre = read_array(f, (size_t)n_traj * 4);
    void* h_win = read_array(f, (size_t)wlen * 4);
    void* h_roff = read_array(f, (size_t)(n_traj + 1) * 8);
    void* h_mask = read_array(f, (size_t)n_rows);
    void* h_tgt = read_array(f, (size_t)n_rows * 4);
    void* h_hid = read_array(f, (size_t)n_rows * H * 2);
    void* h_w = read_array(f, (size_t)V * H * 2);
    void* h_behav = read_array(f, (size_t)n_rows * 4);
    void* h_rew = read_array(f, (size_t)n_traj * 4);
    int32_t st[5] = {-1, -1, -1, -1, -1};
    PaceLossArgs la;
    double loss = 0.0;
    double* d_loss;
    float *d_lp2, *d_adv, *adv;
    void *d_behav, *d_rew;
    double r_hat = -1.0;
    int64_t k = -1;
    PaceScoreParams sp;
    PaceBudgetParams bp;
    PaceBatch batch;
    size_t ws_bytes;
    void *d_ws, *d_ws2, *d_ws3;
    double *d_kgen, *d_kwait, *d_weight, *d_score, *d_unit;
    int32_t *d_acc, *d_rej, *d_status;
    uint8_t* d_flags;
    float* d_lp;
    double* unit;
    uint8_t* flags;
    float* lp;
    FILE* o;
    void *d_tags, *d_off, *d_c, *d_spre, *d_win, *d_roff, *d_mask, *d_tgt, *d_hid, *d_w;
    fclose(f);
    if (!h_tags || !h_off || !h_c || !h_spre || !h_win || !h_roff || !h_mask || !h_tgt ||
        !h_hid || !h_w || !h_behav || !h_rew)
      return 1;
    d_tags = to_device(h_tags, (size_t)n_tokens * 4);
    d_off = to_device(h_off, (size_t)(n_traj + 1) * 8);
    d_c = to_device(h_c, (size_t)n_traj * 4);
    d_spre = to_device(h_spre, (size_t)n_traj * 4);
    d_win = to_device(h_win, (size_t)wlen * 4);
    d_roff = to_device(h_roff, (size_t)(n_traj + 1) * 8);
    d_mask = to_device(h_mask, (size_t)n_rows);
    d_tgt = to_device(h_tgt, (size_t)n_rows * 4);
    d_hid = to_device(h_hid, (size_t)n_rows * H * 2);
    d_w = to_device(h_w, (size_t)V * H * 2);
    d_behav = to_device(h_behav, (size_t)n_rows * 4);
    d_rew = to_device(h_rew, (size_t)n_traj * 4);
    if (!d_tags || !d_off || !d_c || !d_spre || !d_win || !d_roff || !d_mask || !d_tgt ||
        !d_hid || !d_w || !d_behav || !d_rew)
      return 2;
    CHECK_CUDA(cudaMalloc((void**)&d_kgen, (size_t)n_traj * 8));
    CHECK_CUDA(cudaMalloc((void**)&d_kwait, (size_t)n_traj * 8));
    CHECK_CUDA(cudaMalloc((void**)&d_weight, (size_t)n_traj * 8));
    CHECK_CUDA(cudaMalloc((void**)&d_score, (size_t)n_traj * 8));
    CHECK_CUDA(cudaMalloc((void**)&d_unit, (size_t)U * 8));
    CHECK_CUDA(cudaMalloc((void**)&d_acc, (size_t)n_traj * 4));
    CHECK_CUDA(cudaMalloc((void**)&d_rej, (size_t)n_traj * 4));
    CHECK_CUDA(cudaMalloc((void**)&d_flags, (size_t)n_traj));
    CHECK_CUDA(cudaMalloc((void**)&d_lp, (size_t)n_rows * 4));
    CHECK_CUDA(cudaMalloc((void**)&d_status, 4));
    CHECK_CUDA(cudaMemset(d_status, 0, 4));

    /* (a) staleness scores and group means, default EFF parameters */
    pace_score_params_default(&sp);
    sp.group_size = G;
    ws_bytes = pace_score_pool_workspace_size(n_traj, wlen);
    CHECK_CUDA(cudaMalloc(&d_ws, ws_bytes));
    st[0] = pace_score_pool((const int32_t*)d_tags, (const int64_t*)d_off, (const int32_t*)d_c,
                            (const float*)d_spre, n_traj, n_tokens, j, (const float*)d_win, wlen,
                            &sp, d_kgen, d_kwait, d_weight, d_score, d_unit, d_ws, ws_bytes,
                            d_status, NULL);
    /* (a) budget on the host, rejection of the top-scored groups on the device */
    pace_budget_params_default(&bp);
    bp.n_target = n_target;
    ws_bytes = pace_select_workspace_size(U);
    CHECK_CUDA(cudaMalloc(&d_ws2, ws_bytes));
    st[1] = pace_select(d_unit, U, G, &bp, &r_hat, &k, d_acc, d_rej, d_flags, d_ws2, ws_bytes,
                        d_status, NULL);
    /* (b) log-probs of the accepted trajectories' rows in the loss */
    batch.seq_offsets = (const int64_t*)d_roff;
    batch.seq_accepted = d_flags;
    batch.mask = (const uint8_t*)d_mask;
    batch.n_seq = n_traj;
    batch.n_rows = n_rows;
    ws_bytes = pace_token_logprob_workspace_size(n_rows, n_traj, H, V);
    CHECK_CUDA(cudaMalloc(&d_ws3, ws_bytes));
    st[2] = pace_token_logprob(&batch, d_hid, d_w, (const int32_t*)d_tgt, H, V, 1.0f, d_lp, NULL,
                               NULL, d_ws3, ws_bytes, d_status, NULL);
    /* (b) the same rows again with the fused advantages + clipped surrogate */
    CHECK_CUDA(cudaMalloc((void**)&d_lp2, (size_t)n_rows * 4));
    CHECK_CUDA(cudaMalloc((void**)&d_adv, (size_t)n_traj * 4));
    CHECK_CUDA(cudaMalloc((void**)&d_loss, 8));
    la.behav_lp = (const float*)d_behav;
    la.reward = (const float*)d_rew;
    la.group_size = G;
    pace_loss_params_default(&la.params);
    la.params.eps_low = (float)atof(argv[3]);
    la.params.eps_high = (float)atof(argv[4]);
    la.loss = d_loss;
    la.adv = d_adv;
    la.ratio = NULL;
    la.partial = NULL;
    st[3] = pace_token_logprob(&batch, d_hid, d_w, (const int32_t*)d_tgt, H, V, 1.0f, d_lp2, NULL,
                               &la, d_ws3, ws_bytes, d_status, NULL);
    CHECK_CUDA(cudaDeviceSynchronize());
    CHECK_CUDA(cudaMemcpy(&st[4], d_status, 4, cudaMemcpyDeviceToHost));
    CHECK_CUDA(cudaMemcpy(&loss, d_loss, 8, cudaMemcpyDeviceToHost));
    adv = (float*)malloc((size_t)n_traj * 4);
    if (!adv) return 1;
    CHECK_CUDA(cudaMemcpy(adv, d_adv, (size_t)n_traj * 4, cudaMemcpyDeviceToHost));
    unit = (double*)malloc((size_t)U * 8);
    flags = (uint8_t*)malloc((size_t)n_traj);
    lp = (float*)malloc((size_t)n_rows * 4);
    if (!unit || !flags || !lp) return 1;
    CHECK_CUDA(cudaMemcpy(unit, d_unit, (size_t)U * 8, cudaMemcpyDeviceToHost));
    CHECK_CUDA(cudaMemcpy(flags, d_flags, (size_t)n_traj, cudaMemcpyDeviceToHost));
    CHECK_CUDA(cudaMemcpy(lp, d_lp, (size_t)n_rows * 4, cudaMemcpyDeviceToHost));
    o = fopen(argv[2], "wb");
    if (!o) return 1;
    fwrite(st, 4, 5, o);
    fwrite(&k, 8, 1, o);
    fwrite(&r_hat, 8, 1, o);
    fwrite(unit, 8, (size_t)U, o);
    fwrite(flags, 1, (size_t)n_traj, o);
    fwrite(lp, 4, (size_t)n_rows, o);
    fwrite(&loss, 8, 1, o);
    fwrite(adv, 4, (size_t)n_traj, o);
    fclose(o);
  }
  return 0;
}
