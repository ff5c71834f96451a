/*
 * bdscan_mixer.h -- the steps either side of the block-restricted
 * bidirectional scan in a Mamba mixer, on NVIDIA GB300 (sm_103a): the causal
 * depthwise convolution of width 4 with SiLU, whose last three inputs are
 * part of the cached boundary state (Sec. 4, eq. prefix-cache; Sec. 4.1,
 * eq. cache-c4: the cache holds the convolution and state-space states;
 * Appendix C: convolution width 4), the step size softplus(dt_raw + bias),
 * and the SiLU-gated output. The scan itself is the one of bdscan.h.
 *
 * The layer, per stream (clean c, noisy n) and channel d:
 *   pre_t = conv_b[d] + sum_{j=0..3} conv_w[d][j] xr_{t-3+j}   (tap 3: token t)
 *   x_t   = SiLU(pre_t) = pre_t / (1 + exp(-pre_t))
 *   dt    = softplus(dt_raw + bias): dt_bias_f for the clean stream and the
 *           noisy forward direction, dt_bias_r for the noisy reverse one
 *   y     = the scan of bdscan.h on x, dt, B, C (both directions and skip
 *           terms for the noisy stream)
 *   out   = y * SiLU(z)
 * A noisy block's convolution continues from the clean stream: its window
 * positions before the block's first token read the clean raw inputs there
 * (positions before token 0 read the initial convolution state, zero unless
 * given); both scan directions of the block read its convolved input.
 *
 * Layouts: raw inputs xr, dt_raw, gates z, outputs out and their gradients
 * [Bt][L][D]; B, C [Bt][L][N]; conv_w [D][4], conv_b, dt_bias_f, dt_bias_r
 * [D] fp32; convolution states [Bt][nS][3][D] fp32, oldest token first; SSM
 * states as in bdscan.h. Element types as in bdscan.h (bdscan_dims.dtype for
 * the inputs, out_dtype for out and the per-token gradients). The raw inputs
 * travel in the bdscan_clean / bdscan_noisy structs: x holds xr, dt (dt_f,
 * dt_r) holds dt_raw.
 *
 * Conventions of bdscan.h: device pointers, 16-byte aligned, caller-owned
 * memory with a caller workspace (sizes from the *_workspace_size queries),
 * asynchronous on `stream`, return codes and bdscan_last_error(). The
 * intermediate scan inputs are kept in fp32 in the workspace; the scan runs
 * in fp32.
 */
#ifndef BDSCAN_MIXER_H
#define BDSCAN_MIXER_H

#include "bdscan.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct bdscan_mixer_params {
  const float* conv_w;    /* [D][4] */
  const float* conv_b;    /* [D] */
  const float* dt_bias_f; /* [D] */
  const float* dt_bias_r; /* [D] */
} bdscan_mixer_params;

typedef struct bdscan_mixer_grads {
  float* dconv_w;    /* [D][4] */
  float* dconv_b;    /* [D] */
  float* ddt_bias_f; /* [D] */
  float* ddt_bias_r; /* [D] */
} bdscan_mixer_grads;

/* All-block forward of the mixer (Sec. 4.1): writes out_c, out_n [Bt][L][D]
 * and the SSM boundary states [Bt][L/Bs][D][N] (the backward's checkpoints;
 * the convolution part of each boundary state is the clean raw input and is
 * not copied). z_c and z_n are the gates of the two streams. */
size_t bdscan_mixer_forward_workspace_size(const bdscan_dims* dims);
int bdscan_mixer_forward(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                         const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                         const bdscan_mixer_params* mparams, void* out_c, void* out_n, float* states,
                         void* workspace, size_t workspace_bytes, void* stream);

/* Gradients of <dout_c, out_c> + <dout_n, out_n> + <dstates, states> with
 * respect to every input (eq. prefix-cache-gradient, through the
 * convolution as well: a noisy block's convolution sends gradient into the
 * clean raw inputs before it). The forward (its scan inputs, outputs and
 * boundary states) is recomputed from the inputs.
 * gclean / gnoisy receive dxr, ddt_raw, dB, dC (in the dx / ddt fields);
 * dz_c, dz_n the gates' gradients; gparams dA, dD; gmparams the convolution
 * taps, its bias and both step-size biases. dout_c and dstates are nullable
 * (zero). */
size_t bdscan_mixer_backward_workspace_size(const bdscan_dims* dims);
int bdscan_mixer_backward(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                          const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                          const bdscan_mixer_params* mparams, const void* dout_c,
                          const void* dout_n, const float* dstates, const bdscan_clean_grads* gclean, void* dz_c,
                          const bdscan_noisy_grads* gnoisy, void* dz_n, const bdscan_param_grads* gparams,
                          const bdscan_mixer_grads* gmparams, void* workspace, size_t workspace_bytes,
                          void* stream);

/* Cache build / append over a clean prefix (eq. cache-c4): the SSM states and
 * the convolution states ([Bt][L/Bs][3][D] with emit_all, else [Bt][1][3][D],
 * the raw inputs of the last three tokens), continued from init_state
 * [Bt][D][N] and conv_init [Bt][3][D] (both nullable: zero). With z_c and
 * out_c given (both or neither), also the clean outputs. */
size_t bdscan_mixer_boundary_states_workspace_size(const bdscan_dims* dims);
int bdscan_mixer_boundary_states(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                                 const float* A_f, const float* D_f, const bdscan_mixer_params* mparams,
                                 const float* init_state, const float* conv_init, void* out_c, float* states,
                                 float* conv_states, int emit_all, void* workspace, size_t workspace_bytes,
                                 void* stream);

/* One noisy block from the cached SSM state seed [Bt][D][N] and convolution
 * state conv_seed [Bt][3][D], both read only (dims.len == dims.block). */
size_t bdscan_mixer_active_block_workspace_size(const bdscan_dims* dims);
int bdscan_mixer_active_block(const bdscan_dims* dims, const float* seed, const float* conv_seed,
                              const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                              const bdscan_mixer_params* mparams, void* out_n, void* workspace,
                              size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* BDSCAN_MIXER_H */
