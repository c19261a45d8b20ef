/*
 * libqvla test hooks.  They have no counterpart in the paper: they exist so that the tests can
 * make one of the kernels' bounded waits run out (the failure path of QVLA_ERR_TIMEOUT in
 * qvla.h) without a GPU fault, a trap or a hang, and read the GEMM's host-side launch plan on a
 * machine without a GPU.  Off by default; not for production use.
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

/* The launch plan that qvla_w4a4_linear's GEMM (Sec. 4.2, Eq. 7) takes for M > 128 tokens of an
 * M x K -> N layer on a device of num_sms SMs: the host-side choice of tile shape and split of K,
 * computed without touching a device.
 *   N          the layer's weight rows (2H for a gated layer)
 *   gated      nonzero: a gated gate/up layer (qvla_layer_create_gated)
 *   split_room nonzero: the workspace has the room qvla_linear_workspace_bytes counts for the
 *              split of K; 0: the linear runs in a workspace of the required parts only
 *   shape      out: 0 single CTAs with 128 x 128 tiles, 1 single CTAs with 128 x 256, 2 CTA pairs
 *              with 256 x 128, 3 CTA pairs with 256 x 256 (tokens x weight rows)
 *   parts      out: work units per tile; 1 = whole tiles
 * QVLA_ERR_INVALID_ARG for null outputs, M <= 128 (those batches run weight-major), K not a
 * positive multiple of 128, N not a positive multiple of 16 (256 when gated), num_sms < 2. */
qvla_status qvla_debug_gemm_plan(int M, int K, int N, int gated, int num_sms, int split_room, int* shape, int* parts);

#ifdef __cplusplus
}
#endif

#endif /* QVLA_DEBUG_H */
