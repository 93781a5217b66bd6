/* Host-only use of the C ABI from plain C (C99), for tests/test_c_abi.py: creates
 * plans, reads their shape, byte counts, schedule and cost model, exercises the error
 * path, and prints one line per plan that the test compares with the Python binding. */
#include <stdio.h>

#include "gar.h"

int main(void) {
  const int cases[][3] = {{5, 1024, 3}, {24, 16777216, GAR_STEPS_BO}, {127, 4194304, 7}, {24, 1000, 22},
                          {8, 100, GAR_STEPS_RING}};
  for (unsigned c = 0; c < sizeof cases / sizeof cases[0]; ++c) {
    gar_plan *plan = NULL;
    int rc = gar_plan_create(&plan, cases[c][0], (uint64_t)cases[c][1], GAR_F32, GAR_SUM, cases[c][2]);
    if (rc != GAR_OK) {
      printf("error %d %s\n", rc, gar_last_error());
      return 1;
    }
    gar_plan_info info;
    size_t ws = 0;
    uint64_t per_step[128];
    int S = 0, phase = -1, partner = 0, count = 0;
    if (gar_plan_get_info(plan, &info) != GAR_OK || gar_plan_bytes(plan, &ws, per_step, &S) != GAR_OK ||
        gar_plan_step(plan, 0, &phase, &partner, NULL, &count) != GAR_OK)
      return 2;
    unsigned long long total = 0;
    for (int t = 0; t < S; ++t) total += per_step[t];
    printf("P=%d S=%d K=%d ws=%zu bytes=%llu step0=%d,%d,%d\n", info.P, info.S, info.K, ws, total, phase,
           partner, count);
    gar_plan_destroy(plan);
  }
  gar_plan *bad = NULL;
  int rc = gar_plan_create(&bad, 5, 10, GAR_F32, GAR_SUM, 2); /* below ceil(log2 5) */
  printf("bad=%d %s null=%d\n", rc, gar_strerror(rc), bad == NULL);
  double tau = 0.0;
  int steps = 0;
  gar_cost_model(127, 7, 425.0, 1e-5, 1e-9, 1e-10, &tau);
  gar_optimal_steps(127, 425.0, 1e-5, 1e-9, 1e-10, &steps);
  printf("cost=%.6e best=%d\n", tau, steps);
  return 0;
}
