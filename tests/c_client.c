/* A plain C99 client of the library's boundary (test infrastructure).  The
 * CPU tests compile it with warnings as errors against include/ and link it
 * to liblstm_approx.so, which checks that the header is valid C; it then
 * calls the entry points that need no device and prints their answers. */
#include <stdio.h>

#include "lstm_approx.h"

int main(void) {
  int out[LSTM_APPROX_PLAN_ITEMS];
  char msg[256];
  const int cps[2] = {16, 64};
  int rc = lstm_approx_plan(LSTM_APPROX_FP32, 512, 20, 1, 256, cps, 2, 0, 0, 0, out, LSTM_APPROX_PLAN_ITEMS, msg,
                            (int)sizeof msg);
  printf("plan %d path %d variant %d cluster %d\n", rc, out[LSTM_APPROX_PLAN_PATH],
         out[LSTM_APPROX_PLAN_PERSISTENT_VARIANT], out[LSTM_APPROX_PLAN_CLUSTER]);
  rc = lstm_approx_plan(LSTM_APPROX_BF16, 64, 2, 1, 32, NULL, 0, LSTM_APPROX_PATH_PERSISTENT, 0, 0, out,
                        LSTM_APPROX_PLAN_ITEMS, msg, (int)sizeof msg);
  printf("forced %d %s\n", rc, msg);
  lstm_approx_t *h = NULL;
  const int dims[1] = {16};
  rc = lstm_approx_create(&h, 1, dims, 8, 4, 1, LSTM_APPROX_FP32, NULL);
  printf("create %d %s\n", rc, h == NULL ? "null" : "handle");
  printf("error %s\n", lstm_approx_last_error(NULL));
  lstm_approx_destroy(h);
  rc = lstm_approx_plan(LSTM_APPROX_BF16, 2048, 16, 64, 1024, NULL, 0, 0, 0, 0, out, LSTM_APPROX_PLAN_ITEMS, msg,
                        (int)sizeof msg);
  printf("tensor plan %d tau splits %d tau streams %d\n", rc, out[LSTM_APPROX_PLAN_TAU_SPLITS],
         out[LSTM_APPROX_PLAN_TAU_TILE_STREAMS]);
  printf("dense order %d %d\n", lstm_approx_dense_set_launch_order(1), lstm_approx_dense_set_launch_order(0));
  return 0;
}
