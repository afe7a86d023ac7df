/* A plain C caller of the library's host-side entry points: the header
 * compiles as C, the shared library links without C++ or Python, and the
 * sizing and validation rules answer as include/taskpress.h states.  No
 * device work is requested. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "taskpress.h"

static int failures = 0;
#define CHECK(cond)                                              \
  do {                                                           \
    if (!(cond)) {                                               \
      fprintf(stderr, "check failed: %s (line %d)\n", #cond, __LINE__); \
      ++failures;                                                \
    }                                                            \
  } while (0)

int main(void) {
  /* Sec. 4 budget: ceil(ratio * n) with a small tolerance, clamped to [0, n] */
  CHECK(tp_budget(2000, 0.25) == 500);
  CHECK(tp_budget(10, 0.15) == 2);
  CHECK(tp_budget(0, 0.5) == 0);
  CHECK(tp_budget(100, 1.0) == 100);
  CHECK(tp_budget(100, 1.5) == -1);

  int64_t offs[3] = {0, 1500, 3000};
  tp_problem p;
  memset(&p, 0, sizeof(p));
  p.n_heads_q = 32;
  p.n_heads_kv = 8;
  p.head_dim = 128;
  p.guide_len = 64;
  p.batch = 2;
  p.pool_kernel = 5;
  p.quant_bits = 8;
  p.doc_offsets = offs;
  CHECK(tp_kept_capacity(&p, 0.1, -1) == 150);
  CHECK(tp_kept_capacity(&p, 0.0, 2048) == 1500);
  CHECK(tp_workspace_bytes(&p, 0.1, -1) > 0);

  /* the stack workspace: short documents get room for up to 7 more layers'
   * key scores, scales and selection scratch; one layer needs none */
  CHECK(tp_workspace_bytes_stack(&p, 0.1, -1, 1) == tp_workspace_bytes(&p, 0.1, -1));
  CHECK(tp_workspace_bytes_stack(&p, 0.1, -1, 4) > tp_workspace_bytes(&p, 0.1, -1));
  CHECK(tp_stack_layers_per_selection(&p, 0.1, -1, 4, tp_workspace_bytes(&p, 0.1, -1)) == 1);
  CHECK(tp_stack_layers_per_selection(&p, 0.1, -1, 0, 0) == -1);

  /* a 256-token guide at G = 4 (1024 stacked rows) is taken in blocks; one
   * above TP_MAX_GUIDE_ROWS is not */
  p.guide_len = 256;
  CHECK(tp_workspace_bytes(&p, 0.1, -1) > 0);
  p.guide_len = TP_MAX_GUIDE_ROWS / 4 + 1;
  CHECK(tp_workspace_bytes(&p, 0.1, -1) == 0);
  p.guide_len = 64;

  p.head_dim = 96; /* unsupported head size */
  CHECK(tp_kept_capacity(&p, 0.1, -1) == -1);
  p.head_dim = 128;
  p.flags = TP_SCORE_NORM_ADD | TP_SCORE_HARMONIC; /* at most one blend */
  CHECK(tp_kept_capacity(&p, 0.1, -1) == -1);
  p.flags = 0;

  /* null device pointers are refused before anything is enqueued */
  CHECK(tp_quantize_v(&p, NULL, NULL, NULL, NULL) == TP_ERR_INVALID_ARG);
  CHECK(tp_compress_layers(&p, -1, NULL, NULL, NULL, 0.1, -1, NULL, NULL, NULL, NULL, NULL, NULL,
                           0, NULL) == TP_ERR_INVALID_ARG);
  CHECK(strcmp(tp_status_string(TP_OK), "") != 0);
  if (failures == 0) printf("abi_host ok\n");
  return failures == 0 ? 0 : 1;
}
