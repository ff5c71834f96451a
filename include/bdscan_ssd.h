/*
 * bdscan_ssd.h -- C ABI of the Mamba-2 (SSD) form of the block-restricted
 * bidirectional scan in libbdscan (arXiv 2607.02805, sm_103a).
 *
 * The paper's trained BDLM Mamba-H layers are Mamba-2 mixers (Appendix C:
 * state 64 or 128, chunk 128, expansion 2; block 256 in the hyperparameter
 * table; the head dimension is not given for the Mamba mixers, 64 is the
 * Mamba-2 default). In that form the decay is one scalar per head and
 * B_t, C_t are shared by every channel (one group): for channel p of head h,
 *   h_t[p, :] = exp(dt_t[h] A[h]) h_{t-1}[p, :] + dt_t[h] x_t[h, p] B_t
 *   y_t[h, p] = C_t . h_t[p, :] + D[h] x_t[h, p]
 * (Sec. 3, eq. mamba-scan-background with tied parameters). The block
 * restriction is the one of bdscan.h (Sec. 4, eqs. boundary-state and
 * partial-reverse): a clean forward scan whose block-end states are the
 * prefix cache; every noisy block scanned forward from the clean state at its
 * start plus a reverse scan confined to the block and started from zero,
 * outputs summed, each direction with its own dt, B, C, A, D.
 *
 * Because the decay is scalar per head, one block's output is a product of
 * small matrices (the SSD form): y = (L_f o C_f B_f^T + U_r o C_r B_r^T) diag(dt) x
 * + diag(decay) C_f seed^T + D x, with lower/upper-triangular decay masks
 * L_f, U_r inside the block. The kernels evaluate these products on the
 * tcgen05 tensor cores (bf16 operands, fp32 accumulation in TMEM).
 *
 * Notation: Bt batch, L tokens per stream, Bs block size, nb = L / Bs,
 * H heads, P = 64 channels per head, N state size.
 *
 * Layouts (row-major, contiguous, no padding):
 *   x, y             [Bt][L][H][P] bf16
 *   dt               [Bt][L][H]    bf16 (after softplus)
 *   B, C             [Bt][L][N]    bf16
 *   A, D             [H] fp32 (A < 0)
 *   states           [Bt][nS][H][P][N] fp32; states[b][k] is the clean state
 *                    after token (k+1)*Bs-1; noisy block k is seeded with
 *                    states[b][k-1], block 0 with zero.
 *   seed, init state [Bt][H][P][N] fp32
 * The structs bdscan_clean, bdscan_noisy and bdscan_params of bdscan.h carry
 * the pointers, with these layouts.
 *
 * Supported shapes: dtype bf16 (inputs and outputs), P = 64, N = 64 or 128,
 * Bs = 128 or 256, L a multiple of Bs.
 *
 * Conventions are those of bdscan.h: device pointers, 16-byte aligned,
 * caller-owned memory, asynchronous on the given stream, return codes
 * BDSCAN_OK / BDSCAN_ERR_ARG / BDSCAN_ERR_UNSUPPORTED / BDSCAN_ERR_CUDA with
 * a thread-local message (bdscan_last_error). The kernels wait on their own
 * tensor-core work with a bounded number of polls; a wait that gives up sets
 * a device flag (bdscan_ssd_wait_flag) instead of hanging.
 */
#ifndef BDSCAN_SSD_H
#define BDSCAN_SSD_H

#include <stddef.h>
#include <stdint.h>

#include "bdscan.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int64_t batch;     /* Bt */
  int64_t len;       /* L, tokens per stream */
  int64_t block;     /* Bs: 128 or 256 */
  int64_t heads;     /* H */
  int64_t head_dim;  /* P: 64 */
  int64_t d_state;   /* N: 64 or 128 */
  int32_t dtype;     /* BDSCAN_BF16 */
} bdscan_ssd_dims;

/* Workspace bytes of bdscan_ssd_forward: the per-block sums of dt of the
 * clean stream, [Bt][nb][H] fp32. 0 for invalid dims. */
size_t bdscan_ssd_forward_workspace_size(const bdscan_ssd_dims* dims);

/* All-block forward (Sec. 4.1): clean output y_c, noisy output y_n and every
 * block-end state of the clean stream.
 *   clean  x [Bt][L][H][P], dt [Bt][L][H], B, C [Bt][L][N] (bf16);
 *   noisy  x, dt_f, B_f, C_f, dt_r, B_r, C_r, same layouts;
 *   params A_f, D_f, A_r, D_r [H] fp32;
 *   y_c, y_n [Bt][L][H][P] bf16 (written); states [Bt][nb][H][P][N] fp32
 *   (written); workspace of at least bdscan_ssd_forward_workspace_size. */
int bdscan_ssd_forward(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                       const bdscan_params* params, void* y_c, void* y_n, float* states, void* workspace,
                       size_t workspace_bytes, void* stream);

/* Workspace bytes of bdscan_ssd_boundary_states: the dt sums [Bt][nb][H]
 * fp32, plus the block-local states [Bt][nb][H][P][N] fp32 when only the
 * final state is emitted. 0 for invalid dims. */
size_t bdscan_ssd_boundary_states_workspace_size(const bdscan_ssd_dims* dims, int emit_all);

/* Cache build / append (Sec. 3 block-cached decoding; Sec. 4
 * eq. boundary-state): the clean forward scan from init_state (nullable,
 * [Bt][H][P][N] fp32; zero if NULL). emit_all != 0 writes every block-end
 * state, states [Bt][nb][H][P][N]; emit_all == 0 writes the final state only,
 * states [Bt][1][H][P][N]. y_c (nullable) receives the clean output. The same
 * kernels as bdscan_ssd_forward, so the states are the same bits. */
int bdscan_ssd_boundary_states(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const float* A_f,
                               const float* D_f, const float* init_state, void* y_c, float* states,
                               int emit_all, void* workspace, size_t workspace_bytes, void* stream);

/* Cached active-block step (Sec. 3: denoise the current block against the
 * cache; Sec. 4 eq. prefix-cache): one noisy block, len == block, seeded with
 * the read-only cached state seed [Bt][H][P][N] fp32 (NULL = zero). Writes
 * y_n [Bt][Bs][H][P] bf16. Same kernel as the noisy blocks of
 * bdscan_ssd_forward: the outputs equal that call's block bit for bit. */
int bdscan_ssd_active_block(const bdscan_ssd_dims* dims, const float* seed, const bdscan_noisy* noisy,
                            const bdscan_params* params, void* y_n, void* stream);

/* Workspace bytes of bdscan_ssd_full_bidir_forward: dt sums, one direction's
 * block states and one direction's fp32 output. 0 for invalid dims. */
size_t bdscan_ssd_full_bidir_workspace_size(const bdscan_ssd_dims* dims);

/* Full-sequence bidirectional layer (no block restriction): the fully
 * bidirectional Mamba of DiffuMamba that the block partial-reverse design
 * replaces (Sec. 4). y = F_fwd(x) + rev(F_rev(rev(x))) over the whole sequence
 * of the noisy tensors: the forward direction uses dt_f, B_f, C_f, A_f, D_f
 * from the start of the sequence, the reverse direction dt_r, B_r, C_r, A_r,
 * D_r from its end, both from zero states; y [Bt][L][H][P] bf16 (written).
 * A comparator for the cache: without one, a denoising step of such a layer
 * rescans the whole context. Same kernels as the clean scan (the reverse
 * direction reads tokens right to left); dims.block sets the internal blocking. */
int bdscan_ssd_full_bidir_forward(const bdscan_ssd_dims* dims, const bdscan_noisy* noisy, const bdscan_params* params,
                                  void* y, void* workspace, size_t workspace_bytes, void* stream);

/* All-block backward of the SSD form (Sec. 4.1, eq. prefix-cache-gradient):
 * gradients of <dy_c, y_c> + <dy_n, y_n> + <dstates, states> with respect to
 * every input of bdscan_ssd_forward. `states` must be the states that
 * bdscan_ssd_forward wrote for the same inputs; dy_c and dstates
 * ([Bt][nb][H][P][N] fp32) are nullable (zero). Per-token gradients are bf16
 * in the layouts of their inputs (gclean: dx [Bt][L][H][P], ddt [Bt][L][H],
 * dB, dC [Bt][L][N]; gnoisy likewise, dx summing both directions); dA, dD
 * [H] fp32. Gradients are overwritten.
 *
 * Per block, head and direction the products G = C B^T and Q = dy x^T and the
 * transposed mixing products (dx = (G o decay dt)^T dy, dC = (Q o decay dt) B,
 * dB = (Q o decay dt)^T C, and the seed term's) run on the tensor cores with
 * bf16 operands and fp32 accumulation; the decay, row and column sums that
 * give the dt and A gradients are fp32. A reverse pass carries the state
 * gradients over the clean stream's blocks, and the transpose of each block's
 * state product (the state gradient split into bf16 high and low parts)
 * finishes the clean stream. Partial sums are combined in a fixed order:
 * results are deterministic. */
size_t bdscan_ssd_backward_workspace_size(const bdscan_ssd_dims* dims);
int bdscan_ssd_backward(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                        const bdscan_params* params, const float* states, const void* dy_c, const void* dy_n,
                        const float* dstates, const bdscan_clean_grads* gclean, const bdscan_noisy_grads* gnoisy,
                        const bdscan_param_grads* gparams, void* workspace, size_t workspace_bytes, void* stream);

/* The device flag set by a kernel whose bounded wait on its tensor-core work
 * gave up (0 = never). Synchronises the current device; reset != 0 clears it.
 * Returns -1 if the flag cannot be read. */
int bdscan_ssd_wait_flag(int reset);

/* Failure-detection check of the bounded waits (no GPU fault, no hang): runs
 * one CTA that waits, through the kernels' own wait path, on an mbarrier that
 * nothing completes, giving up after `polls` polls (1..2^20). Synchronises
 * the current device. Returns the wait flag the probe left (1 = the wait gave
 * up and was reported) after clearing it, or a negative BDSCAN_ERR_* code. */
int bdscan_ssd_wait_selftest(uint32_t polls);

/* 1 if the kernels load their operand tiles with the tensor memory
 * accelerator (TMA: the driver provides the tensor-map encoder), 0 if they
 * fall back to cp.async. Left-to-right streams use TMA when available. */
int bdscan_ssd_tma_enabled(void);

/* Allows (enable != 0, the default) or forbids TMA operand loads for the
 * calls that follow, process-wide; forbidden, every kernel stages its tiles
 * with cp.async, the path taken where the driver has no tensor-map encoder.
 * The results are the same bits either way (the arithmetic does not depend
 * on how tiles arrive). Returns bdscan_ssd_tma_enabled() afterwards. Not to
 * be changed while calls are in flight on another thread. */
int bdscan_ssd_set_tma(int enable);

#ifdef __cplusplus
}
#endif

#endif /* BDSCAN_SSD_H */
