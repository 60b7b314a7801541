/* A C11 program that uses the library only through include/asap_moe.h:
 * the header compiles as strict C, and the pure-host calls work without a
 * GPU.  Exit status 0 when every check holds. */
#include "asap_moe.h"

#include <stdio.h>
#include <string.h>

static int fails = 0;
#define CHECK(cond)                                             \
  do {                                                          \
    if (!(cond)) {                                              \
      fprintf(stderr, "check failed: %s (line %d)\n", #cond, __LINE__); \
      ++fails;                                                  \
    }                                                           \
  } while (0)

int main(void) {
  asap_moe_config c;
  memset(&c, 0, sizeof(c));
  c.hidden = 7168;
  c.n_experts = 256;
  c.top_k = 8;
  c.inter = 2048;
  c.n_shared = 1;
  c.shared_inter = 2048;
  c.gating = ASAP_GATE_SIGMOID_GROUPED;
  c.n_groups = 8;
  c.topk_groups = 4;
  c.route_scale = 2.5f;
  c.dtype = ASAP_BF16;
  c.max_tokens = 4096;

  CHECK(asap_moe_check_config(&c) == ASAP_OK);
  size_t bytes = 0, bytes_half = 0;
  CHECK(asap_moe_workspace_size(&c, 4096, &bytes) == ASAP_OK);
  CHECK(asap_moe_workspace_size(&c, 2048, &bytes_half) == ASAP_OK);
  CHECK(bytes > bytes_half && bytes_half > 0);

  /* invalid requests are refused before anything touches CUDA */
  asap_moe_config bad = c;
  bad.top_k = 0;
  CHECK(asap_moe_check_config(&bad) != ASAP_OK);
  CHECK(asap_moe_last_error() != NULL && asap_moe_last_error()[0] != '\0');
  CHECK(asap_moe_workspace_size(&c, 4096, NULL) != ASAP_OK);
  asap_moe_t h = NULL;
  CHECK(asap_moe_create(NULL, NULL, &h) != ASAP_OK && h == NULL);
  CHECK(asap_moe_layer(NULL, NULL, 0, NULL, NULL, 0, NULL) != ASAP_OK);

  printf("consumer: workspace for 4096 tokens %zu bytes, %d failed checks\n", bytes, fails);
  return fails == 0 ? 0 : 1;
}
