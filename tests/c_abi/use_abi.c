/* A plain C99 user of the library's C ABI: includes tv.h, takes the address
   of every entry point (so the link checks each one) and, on a machine
   without a GPU, checks the calls that need no device. */
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "tv.h"

typedef void (*any_fn)(void);

int main(int argc, char** argv) {
  const any_fn entry[] = {
      (any_fn)tv_create,         (any_fn)tv_verify_batch,        (any_fn)tv_verify_batch_debug,
      (any_fn)tv_verify_batch_host, (any_fn)tv_last_host_copy_bytes, (any_fn)tv_lm_head,
      (any_fn)tv_draft_children, (any_fn)tv_verify_batch_stats,  (any_fn)tv_get_status,
      (any_fn)tv_destroy,        (any_fn)tv_strerror,            (any_fn)tv_version};
  size_t k;
  tv_handle* h = NULL;
  int rc;
  (void)argv;
  for (k = 0; k < sizeof(entry) / sizeof(entry[0]); ++k)
    if (!entry[k]) return 2;
  if (tv_version() < 100) return 3;
  if (strcmp(tv_strerror(-99), "unknown error code") != 0) return 4;
  /* argument errors are found on the host, before any device work */
  if (tv_create(&h, 0, 0, 7, 1, TV_BF16, 0) >= 0) return 5;          /* V = 0 */
  if (tv_create(&h, 0, 32000, -1, 1, TV_BF16, 0) >= 0) return 6;     /* N < 0 */
  if (tv_verify_batch(NULL, 1, 1, NULL, NULL, NULL, NULL, 1.0f, NULL, NULL, NULL, NULL,
                      NULL) != TV_ERR_INVALID_ARG)
    return 7;
  if (tv_destroy(NULL) > 0) return 8;
  if (argc > 1) {   /* with a GPU: create, query, destroy */
    rc = tv_create(&h, 0, 32000, 7, 4, TV_BF16, 0);
    printf("tv_create: %d (%s)\n", rc, tv_strerror(rc));
    if (rc == 0) tv_destroy(h);
  }
  printf("ok\n");
  return 0;
}
