/* A plain C99 consumer of the C ABI (include/arckv.h): it includes the header,
 * links libarckv.so and calls the entry points that need no GPU (workspace
 * sizing, the realized anchor count, status strings and host-side argument
 * rejection).  tests/test_abi_host.py compiles and runs it and compares its
 * output with the Python binding's.  One "key value" pair per line. */
#include <stdio.h>
#include <string.h>

#include "arckv.h"

static arckv_config layer_config(int32_t T, int32_t t, int32_t chunk_len) {
  arckv_config c;
  memset(&c, 0, sizeof c);
  c.H_kv = 8; c.G = 4; c.T = T; c.d = 128; c.n_pos = 256; c.d_x = 4096;
  c.H_I = 8; c.d_I = 128; c.d_A = 128; c.t = t; c.chunk_len = chunk_len;
  c.lambda_m = 0.25f; c.logit_scale = 0.0f; c.ridge_w = 1e-4f; c.ridge_v = 1e-3f;
  c.eps_w = 2.0611536e-09f; c.b_min = -20.0f; c.b_max = 20.0f;
  c.flags = 0u; c.selector = ARCKV_SELECTOR_INDEXER;
  return c;
}

int main(void) {
  arckv_config c = layer_config(8192, 819, 0);
  arckv_config chunked = layer_config(32768, 1638, 8192);
  arckv_config bad = layer_config(8192, 9000, 0);   /* t > T */
  arckv_indexer idx;
  int s;
  memset(&idx, 0, sizeof idx);
  printf("workspace_bytes %zu\n", arckv_workspace_bytes(&c));
  printf("workspace_bytes_bad %zu\n", arckv_workspace_bytes(&bad));
  printf("anchor_count_chunked %d\n", (int)arckv_anchor_count(&chunked));
  printf("attend_workspace_bytes %zu\n", arckv_attend_workspace_bytes(2, 16, 8, 128));
  for (s = ARCKV_OK; s <= ARCKV_ERR_UNSUPPORTED; ++s) printf("status_%d %s\n", s, arckv_status_string((arckv_status)s));
  /* rejected on the host before anything is enqueued: no GPU is touched */
  printf("compact_null_config %d\n",
         (int)arckv_compact(NULL, NULL, NULL, NULL, NULL, &idx, NULL, NULL, NULL, NULL, NULL, 0, NULL));
  printf("compact_bad_shape %d\n",
         (int)arckv_compact(&bad, NULL, NULL, NULL, NULL, &idx, NULL, NULL, NULL, NULL, NULL, 0, NULL));
  return 0;
}
