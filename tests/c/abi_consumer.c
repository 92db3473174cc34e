/* A plain C11 program against include/mosa.h: the header compiles as C and
 * the library links and answers its host-only calls (no device needed).
 * Prints one line per check; exits non-zero on the first failure. */
#include <stdio.h>
#include <string.h>

#include "mosa.h"

#define CHECK(cond, what)                                     \
    do {                                                      \
        if (!(cond)) {                                        \
            printf("FAIL %s\n", what);                        \
            return 1;                                         \
        }                                                     \
        printf("ok %s\n", what);                              \
    } while (0)

int main(void) {
    mosa_shape s = {2, 64, 48, 3, 32, 8, MOSA_BF16, 0, 1};
    size_t n = mosa_workspace_bytes(&s);
    CHECK(n > 0 && n % 256 == 0, "workspace bytes of a valid shape");
    mosa_shape bad = s;
    bad.k = 65;
    CHECK(mosa_workspace_bytes(&bad) == 0, "k > T is refused");
    CHECK(strncmp(mosa_status_string(MOSA_ERR_WORKSPACE), "MOSA_ERR_WORKSPACE", 18) == 0,
          "status string");
    mosa_hybrid_shape h = {s, 2, 16};
    CHECK(mosa_hybrid_workspace_bytes(&h) > n, "hybrid workspace holds both head groups");
    h.window = 24;
    CHECK(mosa_hybrid_workspace_bytes(&h) == 0, "a window must tile the sequence");
    CHECK(mosa_adaptive_k(1024, 8) == 128 && mosa_adaptive_k(10, 64) == 2, "adaptive k");
    CHECK(mosa_forward(&bad, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0) == MOSA_ERR_INVALID_ARG,
          "forward refuses before launching");
    return 0;
}
