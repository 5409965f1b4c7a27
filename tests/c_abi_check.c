/* A plain C99 program against the C ABI: the header compiles as C, and libmone.so links
 * and answers the calls that need no GPU (argument errors are reported before any device
 * work). */
#include <stdio.h>
#include <string.h>

#include "mone.h"

int main(void) {
    mone_mem* h = NULL;
    mone_config cfg;
    if (mone_abi_version() != MONE_ABI_VERSION) return 1;
    if (strcmp(mone_status_string(MONE_OK), "ok") != 0) return 2;
    if (mone_mem_init(NULL, NULL, NULL, NULL, NULL, &h) != MONE_ERR_INVALID_ARG || h != NULL) return 3;
    memset(&cfg, 0, sizeof cfg); /* zero widths: rejected by the configuration check */
    if (mone_mem_init(&cfg, NULL, NULL, NULL, NULL, &h) != MONE_ERR_INVALID_ARG || h != NULL) return 4;
    if (mone_mem_free(NULL) != MONE_ERR_INVALID_ARG) return 5;
    if (mone_mem_launch_count(NULL) != -1) return 6;
    printf("c abi ok\n");
    return 0;
}
