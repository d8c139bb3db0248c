/* A C program (not C++) against include/rf.h: builds the tiny workload's plan on the host and
 * checks the schedule's pattern and a bad-argument status.  No GPU is used. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "rf.h"

int main(void) {
  enum { F = 4, S = 4 };
  const uint8_t is_key[F] = {1, 0, 0, 1};
  const int32_t stride[S] = {2, 2, 2, 2};
  uint8_t mask[S * F], slot[S * F];
  float alpha[S * F], beta[S * F], dt[S * F];
  rf_status st = rf_plan_build(F, S, is_key, stride, 0, NULL, mask, alpha, beta, dt, slot);
  if (st != RF_OK) {
    printf("rf_plan_build: %s\n", rf_status_str(st));
    return 1;
  }
  /* keyframes every step; non-keyframes on steps 0 and 2 */
  static const uint8_t want[S * F] = {1, 1, 1, 1, 1, 0, 0, 1, 1, 1, 1, 1, 1, 0, 0, 1};
  if (memcmp(mask, want, sizeof want) != 0) {
    printf("mask mismatch\n");
    return 2;
  }
  if (dt[1] != -0.5f || dt[0] != -0.25f || alpha[F + 1] != 0.5f) {
    printf("weights mismatch: dt %g %g alpha %g\n", dt[1], dt[0], alpha[F + 1]);
    return 3;
  }
  st = rf_plan_build(0, S, is_key, stride, 0, NULL, mask, alpha, beta, dt, slot);
  if (st != RF_ERR_INVALID_ARG) {
    printf("expected RF_ERR_INVALID_ARG, got %d\n", (int)st);
    return 4;
  }
  printf("ok %d\n", rf_version());
  return 0;
}
