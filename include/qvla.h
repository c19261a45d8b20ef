/*
 * libqvla -- the W4A4 quantized linear of Omega-QVLA (arxiv 2605.28803) on GB300 (sm_103a).
 *
 * The paper states the problem as Y ~= Delta_X' Delta_W' Q_X' Q_W' (Sec. 4.2, Eq. 7) after the
 * composite rotation X' = X P R_hat, W' = P^T R_hat^T W (Sec. 4.1, Eq. 3-5), with symmetric
 * int4 quantisation Delta = max|Z| / 7, Q = clamp(round(Z / Delta), -7, 7) (Sec. 4.2, Eq. 5-6),
 * weight scales per output channel, activation scales per token (backbone) or from a per-step
 * table indexed by the denoising step t (DiT head, Eq. 6 second display).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Matrices are row-major and dense.  Activations x are [M][K] (token-major), weights are
 *    stored [N][K] (output channel n in row n, y = x W^T), outputs y are [M][N].
 *  - Packed int4: byte j of a row holds code 2j in its low nibble and code 2j+1 in its high
 *    nibble, each a 4-bit two's-complement integer.  The quantiser only produces [-7, 7].
 *  - "device" pointers are CUDA global-memory addresses on the current device; "host"
 *    pointers are ordinary CPU memory.  The caller owns every buffer it passes in; the
 *    library owns what it allocates for a layer (packed weights, scales, bias, step table).
 *  - Calls taking a `stream` (a cudaStream_t passed as void*, NULL = legacy default stream)
 *    only enqueue work and return; they allocate nothing and never synchronise, so they can
 *    be captured in a CUDA graph.  All other calls are synchronous.
 *  - Every call returns a qvla_status.  On failure nothing was enqueued and
 *    qvla_last_error() returns a message for the calling thread.
 *  - Shapes: K % 128 == 0, the Hadamard block b is a power of two with 1 <= b <= 4096 and
 *    K % b == 0 (b == 1 disables the online rotation), N % 16 == 0, 0 <= M <= 1 << 20,
 *    K <= 16384 (so every integer accumulator is exact in float32).
 *  - Kernels wait on nothing without a time limit.  A wait that runs out records
 *    QVLA_ERR_TIMEOUT in a device-side word that qvla_check_device() reports.
 */
#ifndef QVLA_H
#define QVLA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  QVLA_OK = 0,
  QVLA_ERR_INVALID_ARG = 1,  /* a pointer, shape or dtype is not acceptable */
  QVLA_ERR_UNSUPPORTED = 2,  /* well-formed but outside what the kernels implement */
  QVLA_ERR_CUDA = 3,         /* a CUDA runtime call failed (message carries its text) */
  QVLA_ERR_OOM = 4,          /* device or host allocation failed */
  QVLA_ERR_STEP_RANGE = 5,   /* step t is outside [0, T) of the layer's table (or no table) */
  QVLA_ERR_TIMEOUT = 6       /* a device-side wait ran out of its time limit */
} qvla_status;

typedef enum { QVLA_F16 = 0, QVLA_BF16 = 1, QVLA_F32 = 2 } qvla_dtype;

/* Opaque device-resident layer: packed int4 weights, Delta_W, weight code sums, optional bias
 * and optional per-step table.  Created by qvla_pack_weights / qvla_layer_create. */
typedef struct qvla_layer qvla_layer;

/* Message describing the last failure on the calling thread ("" if none).  The pointer
 * stays valid until the next libqvla call on the same thread. */
const char* qvla_last_error(void);

/* Version of this interface; bumps on any incompatible change. */
int qvla_abi_version(void);

/* ------------------------------------------------------------------------------------------
 * Offline weight preparation (Sec. 4.1 Eq. 4-5; Sec. 4.2 Eq. 5-6 per output channel).  Host
 * only, touches no GPU.
 *
 * Folds the composite rotation into the weights, W'_n = W_n . P . BlockDiag(U_b) . BlockDiag(H_b)
 * (the [N][K] form of W' = P^T R_hat^T W), in float64; rounds W' once to float32; then per
 * output channel Delta_W[n] = max_k |W'[n,k]| / 7 (float32) and codes
 * clamp(round(W'/Delta_W), -7, 7), round half to even on the exact quotient.
 *
 *   W         host [N][K] of dtype wdt (F16, BF16 or F32).
 *   rot       host float64, NULL (U = I) or (K / rot_block) orthogonal blocks, each
 *             rot_block x rot_block row-major, block b acting on channels [b*rot_block, ...).
 *             A dense K x K factor is rot_block = K.  Orthogonality is the caller's promise.
 *   perm      host int32 [K] or NULL: column j of W.P is column perm[j] of W (a permutation).
 *   had_block Hadamard block b of the online rotation (the activations get the same block).
 *   wq        host out [N][K/2] packed codes.      wscale  host out [N] Delta_W (float32).
 *   wsum      host out [N] (may be NULL): sum over k of the weight codes of row n.
 * ------------------------------------------------------------------------------------------ */
qvla_status qvla_pack_weights_host(const void* W, qvla_dtype wdt, int N, int K,
                                   const double* rot, int rot_block, const int32_t* perm,
                                   int had_block, uint8_t* wq, float* wscale, int32_t* wsum);

/* The data-dependent factors of the composite rotation, chosen offline from the weights alone
 * (Sec. 4.1, Eq. 4 and the permutation P that follows it).  Host only.
 *   perm: input channels sorted by descending energy sum_n W[n,k]^2 (ties: lower channel
 *         first) and dealt across the K / block blocks in zigzag order -- forwards in even
 *         rounds, backwards in odd ones -- each block taking its channels in dealing order;
 *         column j of W.P is column perm[j] of W.
 *   rot:  for each block b of block channels of W.P, U_b = the block x block left singular
 *         vectors of the paper's row partition W_b = (W.P)[:, block b]^T, columns by
 *         descending singular value, each column's largest-magnitude entry positive; stored
 *         as qvla_pack_weights_host takes it (rot_block = block).
 * Pass both to qvla_pack_weights_host (with any Hadamard block that is a multiple of block) and
 * apply x . P . BlockDiag(U_b) to the activations upstream (reading: the library's online
 * rotation is the Hadamard factor).
 *   W     host [N][K] of dtype wdt.   block  divides K, 1 <= block <= 512.
 *   perm  host out int32 [K].          rot    host out float64 [K/block][block][block].
 * ------------------------------------------------------------------------------------------ */
qvla_status qvla_block_svd_rotation(const void* W, qvla_dtype wdt, int N, int K, int block, int32_t* perm,
                                    double* rot);

/* GPTQ-style weight codes (Sec. 5.1: the LLM side uses GPTQ with block size 128 and damping
 * ratio 0.01; the appendix on weight-quantisation solvers), written from the published GPTQ
 * algorithm.  Host only; a drop-in replacement of qvla_pack_weights_host's RTN codes with the
 * same fold, scales and packed layout.
 *   The weights are folded as in qvla_pack_weights_host and rounded to float32; Delta_W[n] is
 *   the RTN scale max |W'_n| / 7.  The n_cal calibration rows X (host [n_cal][K], dtype xdt,
 *   in the basis of W's input) are folded by the same P, U_b and Hadamard blocks, giving the
 *   Hessian H = 2/n_cal X'^T X'.  A column with H_kk = 0 is dead (its codes are 0); H gets
 *   damp * mean(diag H) on its diagonal.  With U the upper Cholesky factor of H^-1, the columns
 *   are quantised in order, q = clamp(round(w_i / Delta), +-7), and the error
 *   (w_i - Delta q) / U_ii is fed to every later column j times U_ij; updates beyond the current
 *   block of `block` columns are applied once per block (block = 128 in the paper).
 * Cost: O(K^3) for the factorisation and O(N K^2) for the codes (float64, all host cores);
 * memory 2 K^2 doubles.  Returns QVLA_ERR_INVALID_ARG if the damped Hessian is not positive
 * definite (e.g. damp = 0 with rank-deficient calibration data).
 *   block >= 1, damp >= 0, n_cal >= 1, K <= 16384; other arguments as qvla_pack_weights_host. */
qvla_status qvla_gptq_pack_host(const void* W, qvla_dtype wdt, int N, int K, const void* X, qvla_dtype xdt,
                                int n_cal, const double* rot, int rot_block, const int32_t* perm,
                                int had_block, int block, double damp, uint8_t* wq, float* wscale,
                                int32_t* wsum);

/* Upload already-packed weights as a layer (synchronous; allocates device memory the layer
 * owns).  wq host [N][K/2], wscale host [N], bias host [N] float32 or NULL.  xdt is the
 * activation dtype the layer accepts (F16, BF16 or F32); ydt the output dtype (F16 or BF16).
 * had_block as in qvla_pack_weights_host.  *out receives the layer. */
qvla_status qvla_layer_create(int N, int K, int had_block, qvla_dtype xdt, qvla_dtype ydt,
                              const uint8_t* wq, const float* wscale, const float* bias,
                              qvla_layer** out);

/* A gated-MLP layer: the gate and up projections of a backbone MLP (the Pi-0.5 / PaliGemma
 * backbone of Sec. 5.1), H output channels each, sharing one input.  They run as one GEMM whose
 * epilogue rounds gate and up to ydt like two stand-alone linears, then writes
 * h = ydt( gelu_tanh(gate) * up ), the input of the down projection.  The glue is the model's,
 * not the paper's method; it is fused here only to avoid storing gate and up.
 *   wq_gate, wq_up   host [H][K/2] packed codes (qvla_pack_weights_host of each projection)
 *   wscale_gate/_up  host [H];  bias_gate/_up host [H] float32 or NULL.
 * H % 128 == 0.  For this layer qvla_gemm_w4a4 and qvla_w4a4_linear write y as [M][H] (h),
 * and the optional acc output is [M][2H]: the H gate accumulators, then the H up ones. */
qvla_status qvla_layer_create_gated(int H, int K, int had_block, qvla_dtype xdt, qvla_dtype ydt,
                                    const uint8_t* wq_gate, const float* wscale_gate, const uint8_t* wq_up,
                                    const float* wscale_up, const float* bias_gate, const float* bias_up,
                                    qvla_layer** out);

/* qvla_pack_weights_host followed by qvla_layer_create (the spec entry point). */
qvla_status qvla_pack_weights(const void* W, qvla_dtype wdt, int N, int K,
                              const double* rot, int rot_block, const int32_t* perm,
                              int had_block, const float* bias, qvla_dtype xdt, qvla_dtype ydt,
                              qvla_layer** out);

/* Free a layer and everything it owns (synchronises the device first).  NULL is a no-op. */
qvla_status qvla_layer_destroy(qvla_layer* layer);

/* Per-step activation scale table of Eq. 6 (second display), read as one float32 per step
 * (per-tensor): scales host [T], each > 0 and finite, T >= 1.  Replaces any earlier table.
 * Synchronous. */
qvla_status qvla_set_step_scales(qvla_layer* layer, const float* scales, int T);

/* Per-step, per-group activation scales (Eq. 6 read per channel group; reading: one float32
 * per (step, group of max(128, had_block) channels) -- one k-block of the integer GEMM, or one
 * Hadamard block when that is larger).  scales host [T][G] with G = K / group (see
 * qvla_layer_scale_groups), each > 0 and finite.  Replaces any earlier table (per step or per
 * group).  With such a table, qvla_w4a4_linear at step t quantises channel k with
 * scales[t][k / group] and computes y = Delta_W[n] sum_g scales[t][g] acc_g[m,n] + bias[n],
 * acc_g the exact integer product over group g's channels: each group's accumulator is
 * corrected exactly and scaled before the float32 sum over the groups.  Not for gated layers
 * (QVLA_ERR_UNSUPPORTED); the other step-taking entry points refuse grouped tables with
 * QVLA_ERR_UNSUPPORTED (per-token calls, step == -1, are unaffected).  Synchronous. */
qvla_status qvla_set_step_group_scales(qvla_layer* layer, const float* scales, int T, int G);

/* Online data-dependent rotation for a layer whose activations cannot take x . P . BlockDiag(U_b)
 * upstream (Sec. 4.1, Eq. 4-5: layers that share one input but fold different P and U_b, such
 * as Q, K and V).  With it set, qvla_w4a4_linear, qvla_w4a4_linear_noalloc and
 * qvla_linear_quantize first form x' = x . P . BlockDiag(U_b) in the workspace -- float32
 * products summed in the order i = 0 .. rot_block - 1, one rounding to the activation dtype --
 * and run the Hadamard factor and the quantiser on x'; the workspace grows by M x K elements of
 * the activation dtype (qvla_linear_workspace_bytes accounts for it).  Pack the weights with the
 * same perm and rot (qvla_pack_weights_host).  qvla_rotate_quantize and qvla_w4a8_linear refuse
 * such a layer (QVLA_ERR_UNSUPPORTED).
 *   perm       host int32 [K] or NULL (identity): column j of x.P is column perm[j] of x.
 *   rot        host float64 [K/rot_block][rot_block][rot_block], row-major U_b (uploaded as
 *              float32), or NULL (U = I; perm alone).  Orthogonality is the caller's promise.
 *   rot_block  16, 32 or 64 (QVLA_ERR_UNSUPPORTED otherwise), dividing K.
 * perm == NULL and rot == NULL removes the online rotation.  Synchronous; the layer's device
 * must be current (QVLA_ERR_INVALID_ARG otherwise). */
qvla_status qvla_layer_set_online_rotation(qvla_layer* layer, const int32_t* perm, const double* rot, int rot_block);

/* The layer's online rotation alone: out = x . P . BlockDiag(U_b) as above (x, out device
 * [M][K] of the layer's activation dtype, distinct buffers), e.g. to calibrate step tables on the
 * values the quantiser sees.  QVLA_ERR_INVALID_ARG if the layer has no online rotation. */
qvla_status qvla_online_rotate(const qvla_layer* layer, const void* x, int M, void* out, void* stream);

/* The layer's scale groups: G groups of `group` channels (group = max(128, had_block)). */
qvla_status qvla_layer_scale_groups(const qvla_layer* layer, int* G, int* group);

/* Shape of a layer (N = output channels: H for a gated layer); any output pointer may be
 * NULL.  T is 0 when no table is set. */
qvla_status qvla_layer_info(const qvla_layer* layer, int* N, int* K, int* had_block, int* T);

/* ------------------------------------------------------------------------------------------
 * Online rotation + activation quantisation (Sec. 4.1 Eq. 5 online factor; Sec. 4.2 Eq. 5-6).
 *
 * For each row m of x (device [M][K], the layer's activation dtype, already in the P.U basis
 * applied upstream): y = x_m . BlockDiag(H_b/sqrt(b)) in float32, then
 *   step == -1 : per-token scale xscale[m] = max_k |y_k| / 7               (backbone)
 *   step >= 0  : xscale[m] = table[step] of the layer                        (DiT, Eq. 6)
 * and codes clamp(round(y / xscale[m]), -7, 7), round half to even on the exact quotient of
 * the float32 operands; xscale = 0 gives codes 0.
 *   xq      device out [M][K/2] packed codes.     xscale device out [M] float32.
 *   xsum    device out [M] int32 (may be NULL): sum over k of the codes of row m.  The GEMM
 *           needs it (its operand encoding is offset binary; the sum removes the offset).
 * Returns QVLA_ERR_STEP_RANGE for step outside [0, T) (or step >= 0 without a table).
 * ------------------------------------------------------------------------------------------ */
qvla_status qvla_rotate_quantize(const qvla_layer* layer, const void* x, int M, int step,
                                 uint8_t* xq, float* xscale, int32_t* xsum, void* stream);

/* The same operation without a layer, for any [M][K] input of dtype xdt and any block b
 * (b == 1: quantise x as given, no rotation).  step_scale is a DEVICE pointer to one float32
 * used as the per-step scale, or NULL for per-token scales. */
qvla_status qvla_rotate_quantize_rows(const void* x, qvla_dtype xdt, int M, int K, int had_block,
                                      const float* step_scale, uint8_t* xq, float* xscale,
                                      int32_t* xsum, void* stream);

/* Calibration helper for the per-step table (Eq. 6, sigma_hat = max abs): raises the device
 * float *absmax (which the caller initialises, e.g. to 0) to max |x . BlockDiag(H_b/sqrt(b))|
 * over all M x K entries.  The table entry is then absmax / 7. */
qvla_status qvla_rotated_absmax(const void* x, qvla_dtype xdt, int M, int K, int had_block,
                                float* absmax, void* stream);

/* The same calibration per scale group: absmax device [K / group] floats (group =
 * max(128, had_block), K a multiple of it), entry g raised to the max over the M rows and the
 * group's channels.  The per-group table entry is then absmax[g] / 7. */
qvla_status qvla_rotated_absmax_groups(const void* x, qvla_dtype xdt, int M, int K, int had_block,
                                       float* absmax, void* stream);

/* ------------------------------------------------------------------------------------------
 * Integer GEMM + dequantisation epilogue (Sec. 4.2 Eq. 7, scales "folded into
 * dequantization", Sec. 5.1):
 *   acc[m,n] = sum_k xq[m,k] * wq[n,k]                       (exact integer)
 *   y[m,n]   = ydt( fma( (float)acc[m,n], xscale[m] * Delta_W[n], bias[n] ) )
 * with xscale[m] * Delta_W[n] one float32 product, the fma in float32 and one
 * round-to-nearest-even conversion to the layer's output dtype.
 *   xq device [M][K/2], xscale device [M], xsum device [M] (from qvla_rotate_quantize),
 *   y device out [M][N] of the layer's output dtype,
 *   acc device out [M][N] int32, or NULL (debug/test hook: the exact integer accumulator);
 *       16-byte aligned like xq and y.
 * ------------------------------------------------------------------------------------------ */
qvla_status qvla_gemm_w4a4(const qvla_layer* layer, const uint8_t* xq, const float* xscale,
                           const int32_t* xsum, int M, void* y, int32_t* acc, void* stream);

/* Bytes of device workspace qvla_w4a4_linear takes for M rows (a multiple of 256): the codes
 * travel between its two kernels as one tensor-core operand byte each (M x K bytes), plus the
 * scales, the code sums and the per-group code sums (M x G x 4 bytes), and, for a layer with an
 * online rotation, x . P . BlockDiag(U_b) (M x K elements of the activation dtype).  Where the
 * GEMM's tiles could leave SMs idle (M > 128, not gated, fewer 128 x 256 tiles than SMs) it adds
 * room for splitting each tile's K into up to 4 work units: 4 FP32 partials per output (M and N
 * rounded up to 256) and 4 bytes of counter per 128 x 128 tile.  The linear also runs in a
 * workspace of the first parts only; its GEMM then does not split K. */
size_t qvla_linear_workspace_bytes(const qvla_layer* layer, int M);

/* The whole online linear (Sec. 4): rotate + quantise x (as qvla_rotate_quantize, step as
 * there), then the integer GEMM and epilogue (as qvla_gemm_w4a4).  x device [M][K], y device
 * out [M][N].  workspace: caller-owned device memory of at least
 * qvla_linear_workspace_bytes(layer, M) bytes, 256-byte aligned, used only during the call's
 * kernels on `stream` (calls that overlap on the GPU must not share it).
 * One token (M = 1, the decode step) runs as a single kernel where the layer allows it (f16 or
 * bf16 input of the output's dtype, Hadamard block <= 2048, no per-group step table, a split of
 * K whose CTAs each see at most two 2048-channel rotation passes): a GEMV whose CTAs rotate and
 * quantise their share of x themselves, with the same results bit for bit; the workspace is
 * then not touched unless the layer has an online rotation. */
qvla_status qvla_w4a4_linear(const qvla_layer* layer, const void* x, int M, int step, void* y,
                             void* workspace, size_t workspace_bytes, void* stream);

/* The one-launch linear for a small batch with a per-step scale: the rotation, the quantiser, the
 * integer GEMM and the epilogue of qvla_w4a4_linear (same arithmetic, same results) in a single
 * kernel -- the DiT head's case (Sec. 4.2, Eq. 6: the scale is the step's table entry, so no
 * reduction along a row precedes the quantiser).  The CTAs that split the reduction over K
 * rotate and quantise the token rows among themselves and exchange the codes in shared memory;
 * nothing goes through a workspace.  Every CTA of a cluster rotates whole token rows, so each
 * weight tile's cluster repeats the rotation of all M rows: on GB300 this takes longer than the
 * two launches of qvla_w4a4_linear at every DiT shape measured except K = 512 at M = 1, and
 * qvla_w4a4_linear does not use it.  x device [M][K] (f16 or bf16), y device out [M][N], step in
 * [0, T).
 * QVLA_ERR_UNSUPPORTED (nothing enqueued) where it does not apply: step == -1, M > 128, K outside
 * [512, 4096] or not a multiple of the task width (512 channels up to K = 512, 1024 up to 1024,
 * 2048 beyond), activation and output dtypes that differ or are f32, gated layers, per-group
 * tables, an online P.U, or no split of K whose tiles fit the kernel's shared memory. */
qvla_status qvla_w4a4_linear_fused(const qvla_layer* layer, const void* x, int M, int step, void* y, void* stream);

/* The two halves of qvla_w4a4_linear, for callers that schedule them separately (for example to
 * time them, or to overlap one layer's GEMM with the next layer's rotation on another stream).
 * qvla_linear_quantize rotates and quantises x into `workspace` (as qvla_rotate_quantize, step
 * as there); qvla_linear_gemm then runs the integer GEMM and epilogue on it (as qvla_gemm_w4a4).
 * The workspace contents in between are internal to the library: the codes as tensor-core
 * operand bytes, the scales and the code sums, which the GEMM only reads, and the counters of
 * the GEMM's split of K, which qvla_linear_quantize zeroes and the GEMM leaves zero (it uses the
 * split's room as scratch).  So qvla_linear_gemm must follow a qvla_linear_quantize of the same
 * layer, M and workspace; it may run again on the same codes.  Same workspace rules as
 * qvla_w4a4_linear. */
qvla_status qvla_linear_quantize(const qvla_layer* layer, const void* x, int M, int step, void* workspace,
                                 size_t workspace_bytes, void* stream);
qvla_status qvla_linear_gemm(const qvla_layer* layer, void* workspace, size_t workspace_bytes, int M, void* y,
                             void* stream);

/* Allocation-free variant of qvla_w4a4_linear.  The paper has no counterpart: this entry
 * point exists for callers that must not allocate device memory once they are running --
 * for example a robot controller's real-time loop, which reserves all of its memory at start-up
 * because an allocation inside the loop can stall for milliseconds or fail mid-episode, or a
 * plug-in whose host runtime hands out device memory only from its own pool.  Such a caller
 * cannot provide qvla_w4a4_linear's workspace on demand, so this call uses a fixed scratch area
 * that the library itself holds instead.
 *
 * The scratch is one file-scope device array of QVLA_NOALLOC_SCRATCH_BYTES (8 MiB).  Every GPU
 * that loads the library holds it until the process exits.  The call allocates nothing: it
 * makes no cudaMalloc/cudaFree and calls no allocating library routine.  Its first call on each
 * device looks up the array's device address with that device current; make that first call
 * before any stream capture.  The scratch must hold qvla_linear_workspace_bytes(layer, M)
 * bytes, each part rounded up to a multiple of 256: the codes as operand bytes (M x K), the
 * scales and the code sums (M x 4 each), the per-group code sums (M x G x 4, G = K / max(128,
 * had_block)) and, for a layer with an online rotation, x . P . BlockDiag(U_b) (M x K elements
 * of the activation dtype).  Larger requests fail with QVLA_ERR_UNSUPPORTED and enqueue
 * nothing.  The layer must live on the current device (QVLA_ERR_INVALID_ARG otherwise).  Every call shares the one array and leaves the
 * last call's contents in it; each call overwrites all it reads, so nothing needs clearing
 * in between.  Two calls whose kernels overlap on the GPU (different streams or threads, on
 * the same device) race on the array: issue them on one stream.
 * Arguments and results are those of qvla_w4a4_linear without the workspace. */
#define QVLA_NOALLOC_SCRATCH_BYTES ((size_t)8 << 20)
qvla_status qvla_w4a4_linear_noalloc(const qvla_layer* layer, const void* x, int M, int step, void* y,
                                     void* stream);

/* ------------------------------------------------------------------------------------------
 * W4A8 variant (the appendix on the real-quantization kernel, "Real-Quantization Kernel
 * Implementation", Table 5): the same int4 weights of the layer against 8-bit activation codes,
 * with the same scales and epilogue.  Per token (step == -1) the scale is max_k |y_k| / 127;
 * per step it is the table entry as given (a table calibrated for 8-bit codes holds
 * absmax / 127); codes are clamp(round(y / xscale[m]), -127, 127), round half to even on the
 * exact quotient of the float32 operands.  With had_block == 1 no rotation runs at all, the
 * appendix's configuration (rotations folded into the weights offline).
 *
 * The accumulator stays exact for K <= 4096 (255 x 15 x K < 2^24 units of the tensor cores'
 * float32 accumulator); layers with a longer K return QVLA_ERR_UNSUPPORTED.
 * ------------------------------------------------------------------------------------------ */

/* Rotate + quantise to 8-bit codes: as qvla_rotate_quantize_rows with q_max = 127.
 *   xq device out [M][K] int8 codes, natural k order, 16-byte aligned.
 *   xscale device out [M] float32; xsum device out [M] int32 or NULL (sum of row m's codes). */
qvla_status qvla_rotate_quantize_rows_a8(const void* x, qvla_dtype xdt, int M, int K, int had_block,
                                         const float* step_scale, int8_t* xq, float* xscale,
                                         int32_t* xsum, void* stream);

/* Bytes of device workspace qvla_w4a8_linear and qvla_gemm_w4a8 need for M rows (a multiple of
 * 256): the codes as two tensor-core operand planes (M x 2K bytes), the scales and the sums. */
size_t qvla_w4a8_workspace_bytes(const qvla_layer* layer, int M);

/* The whole W4A8 linear: rotate + quantise x to 8-bit codes (step as in qvla_rotate_quantize),
 * then the integer GEMM and the epilogue of qvla_gemm_w4a4 on them.  x device [M][K], y device
 * out [M][N] (H for a gated layer); workspace as for qvla_w4a4_linear but of
 * qvla_w4a8_workspace_bytes(layer, M) bytes. */
qvla_status qvla_w4a8_linear(const qvla_layer* layer, const void* x, int M, int step, void* y,
                             void* workspace, size_t workspace_bytes, void* stream);

/* Integer GEMM + epilogue on 8-bit codes quantised elsewhere (e.g. by
 * qvla_rotate_quantize_rows_a8):  acc[m,n] = sum_k xq[m,k] * wq[n,k] (exact),
 * y[m,n] = ydt(fma((float)acc[m,n], xscale[m] * Delta_W[n], bias[n])).
 *   xq device [M][K] int8 (16-byte aligned), xscale device [M];
 *   y device out, acc device out [M][N] int32 or NULL (test hook), as in qvla_gemm_w4a4;
 *   workspace of qvla_w4a8_workspace_bytes(layer, M) bytes, 256-byte aligned (the operand
 *   planes and the code sums are built there first). */
qvla_status qvla_gemm_w4a8(const qvla_layer* layer, const int8_t* xq, const float* xscale, int M, void* y,
                           int32_t* acc, void* workspace, size_t workspace_bytes, void* stream);

/* Synchronise `stream`, then report (and clear) the device-side error word: QVLA_OK, or
 * QVLA_ERR_TIMEOUT if a kernel gave up waiting since the last check. */
qvla_status qvla_check_device(void* stream);

#ifdef __cplusplus
}
#endif

#endif /* QVLA_H */
