/* The WHTMix C ABI from plain C11: the header compiles as C, the library links, and every
 * argument check returns its documented status before any device work.  Each call below either
 * fails validation or needs no device (status strings, plans, workspace sizes, an empty batch), so
 * nothing is launched whether or not a GPU is present.  The pointers are aligned host integers
 * that are never dereferenced. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "whtmix.h"

static int failures = 0;

#define EXPECT(call, want)                                                              \
  do {                                                                                  \
    const int got_ = (call);                                                            \
    if (got_ != (int)(want)) {                                                          \
      fprintf(stderr, "%s: got %d, want %d\n", #call, got_, (int)(want));              \
      ++failures;                                                                       \
    }                                                                                   \
  } while (0)

#define P(a) ((void *)(uintptr_t)(a))

int main(void) {
  const uintptr_t base = (uintptr_t)1 << 20;
  void *x = P(base), *g = P(2 * base), *y = P(3 * base), *dy = P(4 * base), *dx = P(5 * base);
  void *dg = P(6 * base);
  size_t bytes = 0;

  /* forward: one status per rule, checked in the order the header lists them */
  EXPECT(whtmix_forward(NULL, g, y, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_INVALID_ARG);
  EXPECT(whtmix_forward(x, g, y, -1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_INVALID_ARG);
  EXPECT(whtmix_forward(x, g, y, 1, 6, 4, WHTMIX_F32, NULL), WHTMIX_ERR_BAD_SHAPE);
  EXPECT(whtmix_forward(x, g, y, 1, 1 << 24, 1 << 7, WHTMIX_F32, NULL), WHTMIX_ERR_BAD_SHAPE); /* 2^31 */
  EXPECT(whtmix_forward(x, g, y, ((int64_t)1 << 56) + 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_BAD_SHAPE);
  EXPECT(whtmix_forward(x, g, y, 1, 4, 4, 7, NULL), WHTMIX_ERR_BAD_DTYPE);
  EXPECT(whtmix_forward(P(base + 4), g, y, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_MISALIGNED);
  EXPECT(whtmix_forward(x, g, P(base + 16), 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_ALIAS);
  EXPECT(whtmix_forward(x, g, g, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_ALIAS);
  EXPECT(whtmix_forward(NULL, NULL, NULL, 0, 4, 4, WHTMIX_BF16, NULL), WHTMIX_OK); /* empty batch */
  EXPECT(whtmix_forward_x16(NULL, g, y, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_INVALID_ARG);
  EXPECT(whtmix_forward_x16(x, g, y, 1, 6, 4, WHTMIX_BF16, NULL), WHTMIX_ERR_BAD_SHAPE);
  EXPECT(whtmix_forward_x16(x, g, P(base + 16), 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_ALIAS);
  EXPECT(whtmix_forward_x16(NULL, NULL, NULL, 0, 4, 4, WHTMIX_BF16, NULL), WHTMIX_OK);

  /* backward */
  EXPECT(whtmix_backward(x, g, dy, dx, NULL, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_INVALID_ARG);
  EXPECT(whtmix_backward(x, g, dy, dx, P(6 * base + 2), 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_MISALIGNED);
  EXPECT(whtmix_backward(x, g, dy, dx, dx, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_ALIAS);
  EXPECT(whtmix_backward(x, g, dy, P(4 * base + 16), dg, 1, 4, 4, WHTMIX_F32, NULL), WHTMIX_ERR_ALIAS);

  /* the other entry points' host checks */
  EXPECT(whtmix_forward_padded(x, g, y, 1, 5, 6, 4, WHTMIX_F32, NULL), WHTMIX_ERR_BAD_SHAPE);
  EXPECT(whtmix_forward_separable(x, (const float *)g, (const float *)dg, y, 1, 4, 4, 4, WHTMIX_I32, NULL),
         WHTMIX_ERR_BAD_DTYPE);
  EXPECT(whtmix_project(x, g, y, 1, 96, WHTMIX_BF16, NULL), WHTMIX_ERR_BAD_SHAPE);
  EXPECT(whtmix_block_forward(x, g, dg, dy, y, 1, 4, 64, WHTMIX_F32, NULL), WHTMIX_ERR_BAD_DTYPE);
  EXPECT(whtmix_forward_ex(x, g, y, 1, 256, 64, WHTMIX_F32, NULL, 0, NULL), WHTMIX_ERR_WORKSPACE);

  /* plans, workspace sizes and status strings */
  EXPECT(whtmix_plan(256, 32), 1);
  EXPECT(whtmix_plan(256, 64), 2);
  EXPECT(whtmix_plan(65536, 2048), 3);
  EXPECT(whtmix_plan(3, 4), 0);
  EXPECT(whtmix_workspace_bytes(1, 256, 32, WHTMIX_F32, 0, &bytes), WHTMIX_OK);
  EXPECT((int)bytes, 256);
  EXPECT(whtmix_workspace_bytes(1, 256, 32, WHTMIX_F32, 0, NULL), WHTMIX_ERR_INVALID_ARG);
  EXPECT(strcmp(whtmix_status_string(WHTMIX_OK), "ok"), 0);
  EXPECT(strcmp(whtmix_status_string(12345), "unknown status"), 0);
  EXPECT(whtmix_last_cuda_error(), 0); /* no call above reached the CUDA runtime */

  if (failures == 0) printf("c abi ok\n");
  return failures != 0;
}
