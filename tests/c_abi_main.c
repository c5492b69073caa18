/* A plain C99 caller of libcopes.so: include/copes.h must compile without CUDA or C++
 * headers, and the host helpers must link and run without a GPU.  Prints one line per
 * result for tests/test_c_abi.py to compare with the Python binding. */
#include <inttypes.h>
#include <stdio.h>

#include "copes.h"

int main(void) {
  printf("version %s\n", copes_version());
  const uint64_t numel[3] = {1000, 7, 130};
  copes_layout_desc layout = {3, numel, NULL};
  uint64_t offsets[4];
  if (copes_layout(&layout, offsets) != COPES_OK) return 1;
  printf("offsets %" PRIu64 " %" PRIu64 " %" PRIu64 " %" PRIu64 "\n", offsets[0], offsets[1], offsets[2],
         offsets[3]);
  int32_t noise_id[6];
  int8_t sign[6];
  const int P = copes_member_table(6, COPES_ANTITHETIC, noise_id, sign);
  printf("members %d", P);
  for (int i = 0; i < 6; ++i) printf(" %d:%d", noise_id[i], sign[i]);
  printf("\n");
  printf("seed %" PRIu64 "\n", copes_member_seed(33, 2, 1, 5));
  printf("sigma %.17g\n", copes_sigma_eff(1e-3, 4000.0, 1000.0, 1));
  printf("coef %.17g\n", copes_step_coef(5e-4, 32, 1e-3, COPES_COEF_OPENAI));
  /* an invalid call returns an error code and leaves a message */
  char msg[256];
  const int rc = copes_member_table(7, COPES_ANTITHETIC, noise_id, sign);
  copes_last_error(msg, sizeof msg);
  printf("error %d %s\n", rc, msg);
  return 0;
}
