/* A plain C99 client of the PACE C ABI (include/pace.h) that uses only the
 * host-side entry points, so it runs without a GPU: the library version,
 * status strings, parameter defaults and the rejection budget of Eqs. 3-4.
 *
 * stdin: one budget case per line, "n_traj n_target beta r_max r_hat_prev n_units".
 * stdout: header lines, then per case "status r r_hat k" with the doubles in
 * hexadecimal (%a) so the caller can compare them bit for bit. */
#include <stdio.h>

#include "pace.h"

int main(void) {
  PaceScoreParams sp;
  PaceBudgetParams bp;
  PaceLossParams lp;
  char line[512];
  printf("version %d\n", (int)pace_version());
  printf("status %s %s %s\n", pace_status_string(PACE_OK), pace_status_string(PACE_ERR_TIMEOUT),
         pace_status_string((pace_status)99));
  pace_score_params_default(&sp);
  printf("score_defaults %d %d %d %d %a\n", (int)sp.mode, (int)sp.gamma, (int)sp.min_obs,
         (int)sp.group_size, sp.f_missing);
  pace_budget_params_default(&bp);
  printf("budget_defaults %lld %a %a %a\n", (long long)bp.n_target, bp.beta, bp.r_max,
         bp.r_hat_prev);
  pace_loss_params_default(&lp);
  printf("loss_defaults %a %a %a %a %d %d\n", (double)lp.eps_low, (double)lp.eps_high,
         (double)lp.dual_clip, (double)lp.adv_eps, (int)lp.agg, (int)lp.std_unbiased);
  while (fgets(line, sizeof line, stdin)) {
    long long n_traj = 0, n_target = 0, n_units = 0;
    double beta = 0.0, r_max = 0.0, r_prev = 0.0, r = -1.0, r_hat = -1.0;
    int64_t k = -1;
    pace_status st;
    if (sscanf(line, "%lld %lld %lf %lf %lf %lld", &n_traj, &n_target, &beta, &r_max, &r_prev,
               &n_units) != 6)
      continue;
    bp.n_target = n_target;
    bp.beta = beta;
    bp.r_max = r_max;
    bp.r_hat_prev = r_prev;
    st = pace_budget(n_traj, n_units, &bp, &r, &r_hat, &k);
    printf("%d %a %a %lld\n", (int)st, r, r_hat, (long long)k);
  }
  return 0;
}
