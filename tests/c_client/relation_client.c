/*
 * A plain C client of librelation: includes only include/relation.h, links the shared
 * library, and exercises the calls that need no GPU (version, status strings, workspace
 * queries, synchronous argument checks).  Built and run by tests/test_c_client.py.
 * Exit status 0 when every check holds; otherwise the number of the failing check.
 */
#include <stdio.h>
#include <string.h>

#include "relation.h"

static relation_shape shape(int B, int T, int H, int d) {
  relation_shape s;
  s.B = B;
  s.T = T;
  s.H = H;
  s.d_h = d;
  s.sH = d;
  s.sT = (long long)H * d;
  s.sB = (long long)T * H * d;
  return s;
}

int main(void) {
  if (relation_version() <= 0) return 1;
  if (strcmp(relation_status_string(RELATION_OK), "") == 0) return 2;
  if (relation_status_string(RELATION_ERR_TIMEOUT) == NULL) return 3;

  const relation_shape s = shape(2, 100, 3, 64);
  const size_t ws = relation_bwd_workspace_size(s, RELATION_BF16);
  if (ws < (size_t)2 * 3 * 100 * 64 * 4) return 4; /* at least the fp32 dQ accumulator */
  if (relation_bwd_workspace_size(shape(2, 0, 3, 64), RELATION_BF16) != 0) return 5;

  /* synchronous argument checks: nothing is launched */
  void* p = (void*)0x10000; /* aligned, never dereferenced */
  if (relation_fwd(NULL, p, p, p, (float*)p, 0.5f, 2.0f, s, RELATION_BF16, NULL, NULL) !=
      RELATION_ERR_INVALID_ARG)
    return 6;
  if (relation_fwd(p, p, p, p, (float*)p, 0.5f, 0.0f, s, RELATION_BF16, NULL, NULL) !=
      RELATION_ERR_INVALID_ARG)
    return 7;
  if (relation_fwd(p, p, p, p, (float*)p, 0.5f, 2.0f, shape(1, 8, 2, 136), RELATION_BF16, NULL,
                   NULL) != RELATION_ERR_UNSUPPORTED)
    return 8;
  if (relation_bwd(p, p, p, p, p, (const float*)p, p, p, p, (float*)p, 0.5f, 2.0f, s,
                   RELATION_BF16, p, ws - 1, NULL, NULL) != RELATION_ERR_WORKSPACE)
    return 9;

  /* the widening entry points' size queries */
  if (relation_linear_bwd_workspace_size(shape(1, 16, 2, 64), RELATION_BF16) == 0) return 10;
  if (relation_decode_workspace_size(shape(1, 1024, 2, 128), RELATION_BF16) == 0) return 11;
  if (relation_layer_grad_workspace_size(shape(1, 32, 4, 64), RELATION_BF16) == 0) return 12;
  if (relation_layer_grad_workspace_size(shape(1, 32, 3, 64), RELATION_BF16) != 0) return 13;

  printf("relation C client: version %d, bwd workspace %zu bytes, all checks passed\n",
         relation_version(), ws);
  return 0;
}
