/*
 * lrar_testing.h -- test hooks of liblrar.so.  Not part of the library's
 * interface (lrar.h): they exist so that the test suite can reach code paths
 * that ordinary inputs do not choose, and they may change with any version.
 * The paper has no counterpart of either; each is a variant of a call in
 * lrar.h with one extra knob, and every other argument, rule and error is that
 * call's.
 */
#ifndef LRAR_TESTING_H
#define LRAR_TESTING_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * lrar_project with the tile form and width forced instead of chosen from the
 * shape: tile is one of the compiled widths 160, 176, 192, 224, 240, 256 for
 * the single-CTA form (128-row tiles), or 2000 plus one of them for the
 * CTA-pair form (256-row tiles over a cluster of two CTAs on two SMs,
 * tcgen05.mma.cta_group::2); anything else is LRAR_ERR_INVALID_ARG.  So a test
 * covers every width of both forms.
 */
int lrar_test_project_tile(int tile, int in_dtype, const void *a, const void *w, int64_t T, int m, int d, int r,
                           void *o, void *keys, int *status, void *stream);

/*
 * lrar_block_phase1 whose key-staging waits wait on a barrier that nothing
 * ever completes, with the bound on each wait set to wait_cycles SM clock
 * cycles (1 .. 2^32).  The bulk copies of the keys are still issued and land
 * normally; only the waits for them are diverted.  Every wait therefore runs
 * out: the launch must OR LRAR_STATUS_WAIT_TIMEOUT into *status (required
 * here), stop issuing copies, drain the ones in flight and return -- the
 * give-up path, exercised without a fault or a hang.  h_pre and lse_pre are
 * written with meaningless values.  Only launches that stage keys in shared
 * memory have such waits: low-rank keys whose key rows are whole 16-byte
 * vectors and whose n_completed keys of a token fit 4 KB; other shapes return
 * LRAR_ERR_UNSUPPORTED.
 */
int lrar_test_block_phase1_stalled(int variant, int in_dtype, int pre_dtype, const void *values, const void *keys,
                                   const float *queries, int n_completed, int n_sites, int64_t T, int d, int r,
                                   float eps, void *h_pre, float *lse_pre, int *status, long long wait_cycles,
                                   void *stream);

#ifdef __cplusplus
}
#endif

#endif /* LRAR_TESTING_H */
