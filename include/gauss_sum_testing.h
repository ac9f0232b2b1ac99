/*
 * gauss_sum_testing.h -- test hooks of libgauss_sum.so.  Not part of the
 * Gauss-sum computation (the paper has no counterpart); they exist so that
 * the library's failure paths can be exercised without faulting a GPU or
 * exhausting its memory.  Production code never needs them: with neither
 * hook called, the library behaves as documented in gauss_sum.h.
 */
#ifndef GAUSS_SUM_TESTING_H
#define GAUSS_SUM_TESTING_H

#include "gauss_sum.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * on != 0: every workspace allocation the library would make from now on
 * (the workspaces of gauss_sum_ex and friends, and of gauss_sum_mmd2)
 * fails with GS_ERR_OUT_OF_MEMORY before any GPU work; on = 0 restores
 * normal behaviour.  Process-wide.  Calls that allocate nothing (a caller
 * workspace, gauss_sum_noalloc) are unaffected.
 */
void gauss_sum_testing_fail_allocations(int on);

/*
 * Makes one bounded device-side wait of every launch of the fused FMA
 * kernel (C <= 4 forward) on the current device run out until the request
 * is cleared: control warp 0 of block 0 waits on a barrier that nothing
 * arrives on, gives up after the kernel's 2 s limit, raises the block's
 * abort flag and records GS_ERR_DEVICE_TIMEOUT, which
 * gauss_sum_device_status then reports.  The request is written on
 * `stream` (a cudaStream_t as void*; the call synchronises it) into the
 * device status words and cleared with them by gauss_sum_device_status.
 */
gs_status gauss_sum_testing_request_stall(void* stream);

/*
 * Bit flags describing the fused FMA kernel (C <= 4 forward) that the last
 * call of this process launched: bit 0 = overlapped segment transitions
 * (short runs of key tiles per pair of query tiles), bit 1 = banded key
 * order, bit 2 = q^ in TMEM, bit 3 = value magnitudes folded into the key
 * operands (two passes), bit 4 = exponent scale folded into the query
 * operands; -1 before the first such launch.  Lets the
 * parity tests check that each side of a planning switch is exercised.
 */
int gauss_sum_testing_last_fma_variant(void);

#ifdef __cplusplus
}
#endif

#endif /* GAUSS_SUM_TESTING_H */
