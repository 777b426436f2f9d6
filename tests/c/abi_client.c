/* A plain C99 client of the library's C ABI: it includes every public
 * header, links against libshard.so, and calls entry points whose argument
 * checks fail on the host before any CUDA call, so it runs without a GPU.
 * Exit status 0 means every check held; a nonzero status names the check. */
#include <stdio.h>
#include <string.h>

#include "head.h"
#include "shard.h"
#include "shard_debug.h"

static int has(const char* msg, const char* word) { return msg != NULL && strstr(msg, word) != NULL; }

int main(void) {
  shard_t sh = NULL;
  kvstate_t st = NULL;
  head_t hd = NULL;
  shard_config cfg;
  memset(&cfg, 0, sizeof(cfg));

  if (strcmp(shard_last_error(), "") != 0) return 1;
  if (shard_create(NULL, NULL, &sh) != SHARD_EINVAL || sh != NULL) return 2;
  if (!has(shard_last_error(), "null")) return 3;
  if (shard_destroy(NULL) != SHARD_EINVAL) return 4;
  if (kv_state_alloc(NULL, 1, 16, &st) != SHARD_EINVAL || st != NULL) return 5;
  if (kv_state_free(NULL) != SHARD_EINVAL) return 6;
  if (kv_state_reset(NULL, -1) != SHARD_EINVAL) return 7;
  if (shard_step(NULL, NULL, NULL, NULL, NULL, 0, NULL, NULL, 0, NULL, NULL, NULL) != SHARD_EINVAL) return 8;
  if (shard_gemv_noalloc(NULL, 0, 0, NULL, 1, NULL, 0, NULL) != SHARD_EINVAL) return 9;
  if (head_create(NULL, NULL, &hd) != SHARD_EINVAL || hd != NULL) return 10;
  if (head_destroy(NULL) != SHARD_EINVAL) return 11;
  if (shard_debug_op_info(NULL, 0, 0, NULL, NULL, NULL) != SHARD_EINVAL) return 12;
  /* the error codes are distinct negative values */
  if (!(SHARD_OK == 0 && SHARD_EINVAL < 0 && SHARD_ECAPACITY < 0 && SHARD_ENOMEM < 0 && SHARD_ECUDA < 0 &&
        SHARD_EUNSUPPORTED < 0 && SHARD_EINVAL != SHARD_ECAPACITY))
    return 13;
  (void)cfg;
  printf("abi client ok\n");
  return 0;
}
