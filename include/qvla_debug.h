/*
 * libqvla test hooks.  They have no counterpart in the paper: they exist so that the tests can
 * make one of the kernels' bounded waits run out (the failure path of QVLA_ERR_TIMEOUT in
 * qvla.h) without a GPU fault, a trap or a hang.  Off by default; not for production use.
 */
#ifndef QVLA_DEBUG_H
#define QVLA_DEBUG_H

#include "qvla.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Set, for every GEMM kernel of the library, the time limit of a device-side wait and whether
 * the load warp holds back every copy.
 *   wait_limit_ns   limit of each bounded mbarrier wait in nanoseconds of the global timer;
 *                   0 restores the default of 2 s.
 *   hold_gemm_loads nonzero: a tensor-core GEMM launched afterwards issues no copy of weights or
 *                   activations, so every wait on them runs out after wait_limit_ns; the kernel
 *                   records QVLA_ERR_TIMEOUT (read by qvla_check_device), issues no MMA, leaves
 *                   y unwritten and returns.  The decode GEMV (one to four tokens, K split over a
 *                   cluster) then sends nothing between its CTAs (no row maximum, no partial
 *                   sum), and neither do the passes of a row in the few-row rotate-quantise
 *                   kernel (no row maximum, no code sum), so their receiving waits run out the
 *                   same way.  0 restores normal operation.
 * Synchronises the device first; affects every later launch on the current device until called
 * again. */
qvla_status qvla_debug_set_hooks(unsigned long long wait_limit_ns, int hold_gemm_loads);

#ifdef __cplusplus
}
#endif

#endif /* QVLA_DEBUG_H */
