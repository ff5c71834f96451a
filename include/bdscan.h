/*
 * bdscan.h -- C ABI of libbdscan: the block-restricted bidirectional selective
 * state-space scan of BDLM Mamba-H (arXiv 2607.02805), on NVIDIA GB300
 * (sm_103a).
 *
 * The layer (Sec. 4 of the paper):
 *   - a causal forward selective scan over the clean token stream
 *     (Sec. 3, eq. mamba-scan-background, with A_t = exp(dt_t * A) for a
 *     diagonal A holding one decay per channel d and state index n), whose
 *     state at every block end is the exact prefix cache
 *     s_k = F_fwd(c^(k))                          (eq. boundary-state);
 *   - for every noisy block k, a forward scan seeded from the clean state at
 *     the block start, plus a reverse scan confined to block k and started
 *     from zero, with the two outputs summed    (eq. partial-reverse);
 *   - all blocks at once (the all-block objective, Sec. 4.1), and the
 *     backward pass through the cached seeds into the clean prefix scan
 *     (eq. prefix-cache-gradient).
 * Each direction has its own dt, B, C and its own A, D. The forward direction
 * of the noisy stream shares A_f and D_f with the clean scan (both are the
 * layer's forward scan). No argument carries a diffusion timestep: the cache
 * is a function of the clean prefix alone (eq. cacheable-layer).
 *
 * Notation: Bt batch, L tokens per stream (clean and noisy streams have the
 * same length), Bs block size, nb = L / Bs, D channels (d_inner), N state
 * size (d_state).
 *
 * Layouts (row-major, contiguous, no padding):
 *   token x channel  x, dt, y, dy, dx, ddt        [Bt][L][D]
 *   token x state    B, C, dB, dC                 [Bt][L][N]
 *   parameters       A, dA [D][N] fp32;  D, dD [D] fp32
 *   states           [Bt][nS][D][N] fp32; states[b][k] is the clean state
 *                    after token (k+1)*Bs-1 (the paper's s_{k+1}); noisy
 *                    block k is seeded with states[b][k-1], block 0 with 0.
 *   seed, init state [Bt][D][N] fp32
 * Element types: inputs x, dt, B, C and upstream gradients dy use
 * bdscan_dims.dtype; outputs y and per-token gradients use
 * bdscan_dims.out_dtype. States, parameters and parameter gradients are
 * always fp32. Arithmetic is fp32 throughout (state, accumulation).
 *
 * Conventions:
 *   - All pointers are DEVICE pointers (except the bdscan_dims and the
 *     pointer structs themselves, which are read on the host during the
 *     call) and must be 16-byte aligned.
 *   - The caller owns all memory. No call allocates device memory; scratch
 *     comes from a caller-provided workspace whose size the matching
 *     *_workspace_size function returns. The workspace contents need no
 *     initialisation and are meaningless after the call.
 *   - Calls enqueue work on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and return without synchronising. Argument errors are detected
 *     on the host before anything is enqueued.
 *   - Gradients are overwritten, not accumulated.
 *   - Return codes: BDSCAN_OK, or a negative code; bdscan_last_error()
 *     then returns a message for the calling thread. No C++ exception
 *     crosses this interface.
 *   - Supported: d_state N in {8, 16} for every entry point, and any
 *     multiple of 4 up to 64 for bdscan_forward, bdscan_backward,
 *     bdscan_boundary_states and bdscan_active_block: those run the scan
 *     once per group of 16 states (the last group 8 or 16, zero-padded; the
 *     state index is separable in the recurrence, only y, dx and dt sum over
 *     it) and add the groups' fp32 outputs in group order. Their workspaces
 *     grow accordingly; the grouped bdscan_active_block uses a static 16 MiB
 *     device scratch (calls that overlap in time on one device race on it).
 *     dtype/out_dtype pairs (f32,f32),
 *     (bf16,bf16), (bf16,f32); d_inner a multiple of 8 (bf16 inputs) or 4
 *     (f32 inputs); len a multiple of block; block <= 256 for forward-only
 *     calls (<= 128 with AdaLN) and block <= 16, or a multiple of 16 up to
 *     256, for the backward (above 128 tokens its segment checkpoints are
 *     kept in the workspace).
 *     Any batch and len >= 0 (zero-size problems are no-ops).
 */
#ifndef BDSCAN_H
#define BDSCAN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BDSCAN_OK 0
#define BDSCAN_ERR_ARG (-1)         /* null/misaligned pointer, bad size, len % block != 0, small workspace */
#define BDSCAN_ERR_UNSUPPORTED (-2) /* valid arguments outside the supported set above */
#define BDSCAN_ERR_CUDA (-3)        /* a CUDA launch or runtime call failed */
#define BDSCAN_ERR_DEVICE (-4)      /* debug build only: a device-side check failed (see bdscan_debug_build) */

#define BDSCAN_F32 0
#define BDSCAN_BF16 1

typedef struct bdscan_dims {
  int64_t batch;     /* Bt */
  int64_t len;       /* L, tokens per stream */
  int64_t block;     /* Bs, noisy block size */
  int64_t d_inner;   /* D, channels */
  int64_t d_state;   /* N, state size */
  int32_t dtype;     /* BDSCAN_F32 or BDSCAN_BF16: x, dt, B, C, dy */
  int32_t out_dtype; /* BDSCAN_F32 or BDSCAN_BF16: y and per-token gradients */
} bdscan_dims;

/* Clean token stream c (the prefix): x, dt [Bt][L][D]; B, C [Bt][L][N]. */
typedef struct bdscan_clean {
  const void* x;
  const void* dt; /* step size after its softplus */
  const void* B;
  const void* C;
} bdscan_clean;

/* Noisy stream: shared tokens x [Bt][L][D]; forward-direction dt_f, B_f, C_f;
 * reverse-direction dt_r, B_r, C_r. */
typedef struct bdscan_noisy {
  const void* x;
  const void* dt_f;
  const void* B_f;
  const void* C_f;
  const void* dt_r;
  const void* B_r;
  const void* C_r;
} bdscan_noisy;

/* Per-direction parameters: A_f, A_r [D][N] (negative decays), D_f, D_r [D]. */
typedef struct bdscan_params {
  const float* A_f;
  const float* D_f;
  const float* A_r;
  const float* D_r;
} bdscan_params;

typedef struct bdscan_clean_grads {
  void* dx;  /* [Bt][L][D] out_dtype */
  void* ddt; /* [Bt][L][D] out_dtype */
  void* dB;  /* [Bt][L][N] out_dtype */
  void* dC;  /* [Bt][L][N] out_dtype */
} bdscan_clean_grads;

typedef struct bdscan_noisy_grads {
  void* dx;    /* [Bt][L][D], both directions summed */
  void* ddt_f; /* [Bt][L][D] */
  void* dB_f;  /* [Bt][L][N] */
  void* dC_f;  /* [Bt][L][N] */
  void* ddt_r; /* [Bt][L][D] */
  void* dB_r;  /* [Bt][L][N] */
  void* dC_r;  /* [Bt][L][N] */
} bdscan_noisy_grads;

typedef struct bdscan_param_grads {
  float* dA_f; /* [D][N]: clean stream + noisy forward direction */
  float* dD_f; /* [D] */
  float* dA_r; /* [D][N] */
  float* dD_r; /* [D] */
} bdscan_param_grads;

/* Message describing the last error of the calling thread ("" if none). */
const char* bdscan_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int bdscan_version(void);

/* Tokens per time chunk of the chunked clean scan for a given block size.
 * The clean stream is split into chunks of this many tokens from position 0;
 * the value depends on `block` only, so boundary states of a prefix are
 * bit-identical to the states of any longer stream that extends it. */
int64_t bdscan_chunk_tokens(int64_t block);

/* Timing hook for benchmarks. After this call, every entry point called from
 * the same host thread records events[i] (cudaEvent_t handles owned by the
 * caller, passed as void*) on its stream right after its i-th kernel launch,
 * for i < n; events == NULL or n == 0 switches the hook off. The events are
 * only recorded, never waited on. Returns BDSCAN_OK. */
int bdscan_profile_events(void* const* events, int n);

/* Number of kernels the last successful call of this host thread launched. */
int bdscan_last_launch_count(void);

/* Debug build (lib/libbdscan_debug.so, the same sources compiled with
 * BDSCAN_DEBUG=1; same symbols). Each kernel first checks, from its block
 * index and the call's sizes alone, that the last element its CTA touches in
 * every buffer lies inside that buffer's extent; a failed check writes a
 * device status word and the CTA skips its work (no out-of-range access is
 * made, nothing traps). The cached boundary states and the parameter
 * gradients are also checked for NaN and infinity. Every entry point of the
 * debug build then synchronizes the device before it returns (so it cannot
 * be captured into a CUDA graph) and returns BDSCAN_ERR_DEVICE, with the
 * kernel and offset in bdscan_last_error(), if any check failed; the status
 * words are cleared for the next call.
 * bdscan_debug_build() returns 1 in the debug build and 0 otherwise.
 * bdscan_debug_set_slack(e): every extent is taken e >= 0 elements shorter
 * than the sizes give, so a test can make the checks fail on in-range
 * accesses (the flagged CTAs then skip their work and the outputs are
 * incomplete); 0 restores the exact extents. Needs a CUDA device; returns
 * BDSCAN_ERR_UNSUPPORTED in the release build, BDSCAN_ERR_ARG for e < 0. */
int bdscan_debug_build(void);
int bdscan_debug_set_slack(long long elements);

/* ---------------------------------------------------------------------- */
/* All-block forward (Sec. 4 eqs. boundary-state and partial-reverse, all  */
/* blocks evaluated in parallel as in Sec. 4.1).                           */
/* ---------------------------------------------------------------------- */
size_t bdscan_forward_workspace_size(const bdscan_dims* dims);

/* Writes y_c [Bt][L][D] (clean-stream outputs, forward scan only),
 * y_n [Bt][L][D] (noisy outputs: seeded forward + block-local reverse, both
 * D terms included) and states [Bt][L/Bs][D][N] (every block-end state; the
 * backward pass takes them as its recompute checkpoints). */
int bdscan_forward(const bdscan_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                   const bdscan_params* params, void* y_c, void* y_n, float* states,
                   void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* All-block backward (eq. prefix-cache-gradient): gradients of            */
/*   <dy_c, y_c> + <dy_n, y_n> + <dstates, states>                          */
/* with respect to every input of bdscan_forward.                          */
/* ---------------------------------------------------------------------- */
size_t bdscan_backward_workspace_size(const bdscan_dims* dims);

/* `states` must be the states written by bdscan_forward for the same
 * inputs. dy_c (nullable: zero) and dy_n use dims.dtype; dstates (nullable:
 * zero) is fp32 [Bt][L/Bs][D][N]. Every gradient pointer in the three grad
 * structs is required. */
int bdscan_backward(const bdscan_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                    const bdscan_params* params, const float* states, const void* dy_c,
                    const void* dy_n, const float* dstates, const bdscan_clean_grads* gclean,
                    const bdscan_noisy_grads* gnoisy, const bdscan_param_grads* gparams,
                    void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* Cache build / append (Sec. 3 cache interface: a clean forward pass over  */
/* finalised blocks; eq. boundary-state).                                  */
/* ---------------------------------------------------------------------- */
size_t bdscan_boundary_states_workspace_size(const bdscan_dims* dims, int emit_all);

/* Clean forward scan of x, dt, B, C over L tokens, continued from
 * init_state [Bt][D][N] (nullable: zero; pass the cached state to append).
 * emit_all != 0: states is [Bt][L/Bs][D][N], every block-end state.
 * emit_all == 0: states is [Bt][1][D][N], the state after the last token.
 * y_c (nullable) receives the clean outputs [Bt][L][D] (out_dtype). */
int bdscan_boundary_states(const bdscan_dims* dims, const bdscan_clean* clean, const float* A_f,
                           const float* D_f, const float* init_state, void* y_c, float* states,
                           int emit_all, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* Cached active-block denoising step (Sec. 3: denoise the current block    */
/* while reading the prefix cache; Sec. 4: the cache stays valid because the */
/* reverse scan is local). dims.len must equal dims.block.                  */
/* ---------------------------------------------------------------------- */
/* seed [Bt][D][N] fp32 is read only (reused across denoising steps). The
 * noisy tensors hold one block: x, dt_* [Bt][Bs][D], B_*, C_* [Bt][Bs][N].
 * Writes y_n [Bt][Bs][D]. Each channel goes through the same arithmetic, in
 * the same order, as the noisy blocks of bdscan_forward, so outputs are
 * bit-identical to the forward's outputs for the same block and seed. */
int bdscan_active_block(const bdscan_dims* dims, const float* seed, const bdscan_noisy* noisy,
                        const bdscan_params* params, void* y_n, void* stream);

/* ---------------------------------------------------------------------- */
/* Timestep-modulated active block (Appendix E, AdaLN factorization,         */
/* eq. cacheable-adaln): adaptive layer norm acts on the active block only,  */
/* so the cached prefix state stays timestep-free.                          */
/* ---------------------------------------------------------------------- */
/* Modulation of one denoising step: shift, scale, gate [Bt][D] fp32 (the
 * caller maps the timestep embedding e_t to them), eps of the layer norm. */
typedef struct bdscan_adaln {
  const float* shift;
  const float* scale;
  const float* gate;
  float eps;
} bdscan_adaln;

/* Bt * block * 8 bytes: the per-token layer-norm statistics. */
size_t bdscan_active_block_adaln_workspace_size(const bdscan_dims* dims);

/* As bdscan_active_block, with noisy->x = h [Bt][Bs][D], the block's hidden
 * input, normalised per token over the D channels (mean and biased variance;
 * no affine of its own) and modulated, u = (1 + scale) LN(h) + shift. The
 * block-restricted bidirectional scan runs on u from the read-only seed.
 * Writes out [Bt][Bs][D] (out_dtype) = h + gate * y_n, the gated residual.
 * Two launches: the statistics, then the scan. dt, B, C of the block are
 * given by the caller; nothing here touches the seed or any other cache. */
int bdscan_active_block_adaln(const bdscan_dims* dims, const float* seed, const bdscan_noisy* noisy,
                              const bdscan_params* params, const bdscan_adaln* mod, void* out, void* workspace,
                              size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* Full-sequence bidirectional layer (Sec. 4: the fully bidirectional Mamba */
/* denoiser of DiffuMamba, a forward scan and a reverse scan over the whole */
/* sequence, which the block partial-reverse design replaces). A comparator */
/* for the cache: its reverse states depend on every later token, so a     */
/* sampler must rerun it over the whole sequence at every denoising step.   */
/* ---------------------------------------------------------------------- */
size_t bdscan_full_bidir_workspace_size(const bdscan_dims* dims);

/* y [Bt][L][D] (out_dtype) = forward scan of (x, dt_f, B_f, C_f; A_f, D_f)
 * from a zero state at token 0 plus reverse scan of (x, dt_r, B_r, C_r;
 * A_r, D_r) from a zero state at token L-1, each with its own D x term;
 * noisy.x is the input of both directions. dims.block only sets the time
 * chunking of the scans (no block restriction applies); the usual block
 * limits hold. Each direction's output is kept in fp32 in the workspace
 * before the sum is rounded. */
int bdscan_full_bidir_forward(const bdscan_dims* dims, const bdscan_noisy* noisy, const bdscan_params* params,
                              void* y, void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------- */
/* Cache build for callers that cannot allocate device memory. The paper    */
/* has no counterpart: this is a deployment convenience of this library.   */
/* ---------------------------------------------------------------------- */
/* Some callers are not allowed to allocate device memory at the point
 * where they build or extend the cache: a plugin inside another inference
 * engine whose execution step may only use memory that engine planned
 * ahead of time, or a latency-critical serving loop where a cudaMalloc
 * (which can synchronise the device) is not acceptable. This entry point
 * takes the same arguments as bdscan_boundary_states minus the workspace
 * and computes the same result (bit for bit). Its scratch is a static device
 * array of BDSCAN_NOALLOC_SCRATCH_BYTES inside the library; every GPU on
 * which the library is used keeps that array until the process exits.
 *
 * Size limit: the call needs bdscan_boundary_states_workspace_size(dims,
 * emit_all) bytes of scratch; larger problems are rejected with
 * BDSCAN_ERR_UNSUPPORTED (use bdscan_boundary_states with a workspace).
 * First call per device: it looks up the array's device address with the
 * device current; make that first call before any stream capture begins.
 * Sharing: all calls use the same array. Calls whose GPU work overlaps (on
 * different streams or from different threads without ordering between
 * them) race on it and give wrong results; order them on one stream or with
 * events. Nothing in the array has to start at zero: each call writes every
 * scratch value before it reads it, so leftovers of a previous call are
 * never used. No allocation happens in this call (no cudaMalloc, cudaFree,
 * or allocating library routine). */
#define BDSCAN_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
int bdscan_boundary_states_noalloc(const bdscan_dims* dims, const bdscan_clean* clean, const float* A_f,
                                   const float* D_f, const float* init_state, void* y_c, float* states,
                                   int emit_all, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* BDSCAN_H */
