/* A plain C11 client of liblrar.so: the header must compile as C (no C++ or
 * torch types at the boundary) and the library must link into a C program.
 * It makes only calls that return before any device work: the version, an
 * argument the library rejects (NULL values with T > 0) and the error text. */
#include <stdio.h>
#include <string.h>

#include "lrar.h"

int main(void) {
    int rc = lrar_forward(LRAR_SLICED, LRAR_BF16, LRAR_BF16, NULL, NULL, NULL, 1, 16, 64, 8, 1e-6f, NULL, NULL, NULL);
    const char *msg = lrar_last_error();
    printf("version %d, status %d (%s): %s\n", lrar_version(), rc, lrar_strerror(rc), msg ? msg : "");
    if (rc != LRAR_ERR_INVALID_ARG) return 1;
    if (lrar_backward_workspace_size(LRAR_SLICED, 49, 16384, 1024, 16) == 0) return 2;
    return msg && strlen(msg) > 0 ? 0 : 3;
}
