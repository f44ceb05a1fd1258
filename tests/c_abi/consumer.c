/* A plain C99 program using libvcs through include/vcs.h only: the header compiles as C
 * (no C++ or torch types in the interface) and the calls that need no GPU answer from C.
 * Prints one line per check; exits non-zero on the first wrong answer. */
#include <stdio.h>
#include <string.h>

#include "vcs.h"

#define CHECK(cond, what)                        \
  do {                                           \
    if (!(cond)) {                               \
      fprintf(stderr, "FAILED: %s\n", what);     \
      return 1;                                  \
    }                                            \
    printf("ok %s\n", what);                     \
  } while (0)

int main(void) {
  CHECK(strncmp(vcs_version(), "libvcs", 6) == 0, "version string");
  CHECK(strncmp(vcs_status_string(VCS_ERR_INVALID_ARG), "VCS_ERR_INVALID_ARG", 19) == 0, "status string");
  CHECK(strcmp(vcs_status_string((vcs_status)99), "VCS_ERR_UNKNOWN") == 0, "unknown status string");

  /* workspace sizes are host arithmetic: monotone in the problem, 256-byte granular */
  const size_t small = vcs_attn_bwd_workspace_size(2, 1000, 600, 28, 4, 128);
  const size_t large = vcs_attn_bwd_workspace_size(2, 2000, 1200, 28, 4, 128);
  CHECK(small > 0 && large > small && small % 256 == 0, "attention backward workspace size");
  CHECK(vcs_attn_fwd_workspace_size(2, 1000, 600, 28, 4, 128) >= 256, "attention forward workspace size");
  CHECK(vcs_segments_workspace_size(4, 100) > 0, "segment builder workspace size");

  /* host-detectable errors return before any launch */
  CHECK(vcs_gather(NULL, NULL, NULL, 10, NULL, 10, 28, 4, 128, NULL, NULL, NULL, NULL, NULL) == VCS_ERR_INVALID_ARG,
        "gather rejects null pointers");
  CHECK(vcs_plan_segments(NULL, 1, 4, NULL, NULL, 2, 0, NULL, NULL, 0, NULL) == VCS_ERR_INVALID_ARG,
        "plan rejects null pointers");
  return 0;
}
