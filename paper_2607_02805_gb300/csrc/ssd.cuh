// ssd.cuh -- parameters of the SSD-form (Mamba-2, scalar decay per head)
// kernels of libbdscan. The recurrence, layouts and the block restriction are
// documented in include/bdscan_ssd.h.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace bds {

constexpr int kSsdP = 64;    // channels per head
constexpr int kSsdT = 128;   // tokens per tile (the tensor-core M)

struct SsdGeo {
  int64_t Bt, L, Bs;
  int H, N;
  int nb;  // blocks per stream
  int m;   // tiles per block, Bs / 128
};

// Block-local end state of every clean block (from a zero state), and the
// block sums of dt: T[b][k][h][p][n] = sum over the block's tokens s of
// exp(A[h] * sum_{r>s} dt_r) dt_s x_s[h, p] B_s[n].
struct SsdStateParams {
  SsdGeo g;
  const __nv_bfloat16 *x, *dt, *B;
  const float* A;
  float* T;      // [Bt][nb][H][P][N]
  float* sumdt;  // [Bt][nb][H]
  int hg;        // heads per CTA
  int* flag;     // wait flag
  int rev;       // 1: the stream is read right to left (token L-1-t of each batch row at position t)
};

// Sequential pass over blocks: S_k = exp(A sumdt_k) S_{k-1} + T_k.
struct SsdPassParams {
  SsdGeo g;
  const float* T;
  const float* sumdt;
  const float* A;
  const float* init;  // [Bt][H][P][N] or null
  float* states;      // emit_all: [Bt][nb][H][P][N] (may alias T); else [Bt][1][H][P][N]
  int emit_all;
  float* final_state; // [Bt][H][P][N] or null: the state after the last block
};

// Block scan of one stream: clean (forward part only) or noisy (seeded
// forward + block-local reverse), one 128-token tile of one block per CTA.
struct SsdScanParams {
  SsdGeo g;
  const __nv_bfloat16 *x, *dtf, *Bf, *Cf, *dtr, *Br, *Cr;
  const float *Af, *Df, *Ar, *Dr;
  const float* seed;  // seeds, slot stride H*P*N floats, batch stride seed_bstride; null = zero
  int64_t seed_bstride;
  int seed_shift;     // 1: block k reads slot k-1 (block 0: init_seed); 0: block k reads slot k
  const float* init_seed;  // [Bt][H][P][N] or null (zero): the seed of block 0 when seed_shift
  __nv_bfloat16* y;   // [Bt][L][H][P]
  int hg;
  int* flag;
  int rev;            // 1: the stream is read right to left (as in SsdStateParams)
  float* y32;         // non-null: write the output in fp32 here instead of y
  const float* y32_add;  // non-null: add this fp32 array to the output before rounding to y
  int tma;            // set by the launcher: x tiles and seeds arrive by TMA (left-to-right streams)
};

// Backward (ssd_bwd.cu). One stream and direction of the block-local
// backward: per (batch row, block, 128-token tile i, group of hg heads) the
// products G = C B^T (shared by the heads) and Q = dy x^T against every
// s-tile of the block the direction reaches, the masked decays, the
// contributions of tile i to dx (per head) and to dB and dC (summed over the
// group's heads) of every s-tile (partials over i and groups), the column
// sums of R' = Q o G o decay (partials over i) and its row sums with dt, and
// for the seeded forward direction the seed term's products (dC, the seed
// gradient partial over i, the row dot dy_t . seed term_t).
struct SsdBwdTileParams {
  SsdGeo g;
  const __nv_bfloat16 *x, *dy, *dt, *B, *C;  // x, dy [Bt][L][H][P] (dy null: zero); dt [Bt][L][H]; B, C [Bt][L][N]
  const float* A;       // [H]
  const float* states;  // seeded direction: block k reads states[b][k-1] ([Bt][nb][H][P][N])
  float* dx_part;       // [Bt*nb][H][m][Bs][P]
  float* dB_part;       // [Bt*nb][groups][m][Bs][N]
  float* dC_part;       // [Bt*nb][groups][Bs][N]
  float* col_part;      // [Bt*nb][H][m][Bs]
  float* rowsum;        // [Bt*nb][H][Bs]
  float* rowdot;        // [Bt*nb][H][Bs] (seeded direction)
  float* dS_part;       // [Bt*nb][H][m][P][N] (seeded direction)
  float* dd_part;       // [Bt*nb][H][m][8] or null: per warp, sum of dy . x over its rows of tile i
  int hg;               // heads per CTA (at most 16); groups = ceil(H / hg)
  int* flag;
  int tma;              // set by the launcher: x and dy tiles arrive by TMA
};

// The dt and A gradients of one stream and direction from the row and column
// sums: dc = A (rowsum - dt colsum' + rowdot), then a scan inside the block.
struct SsdBwdVecParams {
  SsdGeo g;
  const __nv_bfloat16* dt;
  const float* A;
  const float *col_part, *rowsum, *rowdot;  // rowdot null: zero
  int upper;
  float* ddt;                // [Bt][L][H] fp32, used when ddt_out is null
  __nv_bfloat16* ddt_out;    // [Bt][L][H] or null: the stream's final dt gradient (no other term adds to it)
  float* dA;                 // [Bt*nb][H]
  float* sumdt;              // [Bt*nb][H] or null: the block's sum of dt
};

// Reverse pass over the clean stream's block-end states: gS_k = dstates_k +
// seed gradients of block k+1 (both streams) + exp(A sumdt_{k+1}) gS_{k+1}.
struct SsdBwdPassParams {
  SsdGeo g;
  const float* A;
  const float *dS_c, *dS_f;  // [Bt*nb][H][m][P][N] seed gradient partials
  const float* dstates;      // [Bt][nb][H][P][N] or null
  const float* sumdt;        // [Bt*nb][H]
  float* gS;                 // [Bt][nb][H][P][N]
};

// Transpose of the clean block-state product T_k = sum_s w_s x_s B_s^T, and
// the gradient of the block decay exp(A sumdt_k) S_{k-1}.
struct SsdBwdStateParams {
  SsdGeo g;
  const __nv_bfloat16 *x, *dt, *B;
  const float* A;
  const float* gS;      // [Bt][nb][H][P][N]
  const float* states;  // [Bt][nb][H][P][N]
  const float* sumdt;   // [Bt*nb][H]
  float* dx_state;          // [Bt*nb][H][Bs][P]
  float* dB_state;          // [Bt*nb][H][Bs][N]
  const float* ddt_tile;    // [Bt][L][H] the tile side of the clean dt gradient
  __nv_bfloat16* ddt;       // [Bt][L][H] output: ddt_tile + this kernel's terms
  float* dA;                // [Bt*nb][H]
  int* flag;
};

cudaError_t launch_ssd_bwd_tile(bool upper, bool seeded, const SsdBwdTileParams& p, cudaStream_t s);
cudaError_t launch_ssd_bwd_vec(const SsdBwdVecParams& p, cudaStream_t s);
cudaError_t launch_ssd_bwd_pass(const SsdBwdPassParams& p, cudaStream_t s);
cudaError_t launch_ssd_bwd_state(const SsdBwdStateParams& p, cudaStream_t s);
// Fixed-order combines of the backward's partials into the outputs (bf16
// per-token gradients, fp32 parameter gradients); see ssd_bwd.cu.
cudaError_t launch_ssd_bwd_dx(const SsdGeo& g, const float* dxp_c, const float* dxs, const float* dxp_f,
                              const float* dxp_r, const __nv_bfloat16* dyc, const __nv_bfloat16* dyn, const float* Df,
                              const float* Dr, __nv_bfloat16* dxc, __nv_bfloat16* dxn, cudaStream_t s);
cudaError_t launch_ssd_bwd_dbc(const SsdGeo& g, int ngrp, const float* dBp_c, const float* dBs, const float* dCp_c,
                               const float* dBp_f, const float* dCp_f, const float* dBp_r, const float* dCp_r,
                               __nv_bfloat16* dBc, __nv_bfloat16* dCc, __nv_bfloat16* dBf, __nv_bfloat16* dCf,
                               __nv_bfloat16* dBr, __nv_bfloat16* dCr, cudaStream_t s);
// per-head sums of the partials: dA of both directions (clean, seeded,
// state and reverse terms), dD from the dy . x partials of both streams
// ([Bt*nb][H][m][8] each, from the tile kernels)
cudaError_t launch_ssd_bwd_params(const SsdGeo& g, const float* dd_c, const float* dd_n, const float* dA_c,
                                  const float* dA_f, const float* dA_s, const float* dA_r, float* dAf, float* dDf,
                                  float* dAr, float* dDr, cudaStream_t s);

cudaError_t launch_ssd_block_state(const SsdStateParams& p, cudaStream_t s);
cudaError_t launch_ssd_state_pass(const SsdPassParams& p, cudaStream_t s);
cudaError_t launch_ssd_block_scan(bool noisy, const SsdScanParams& p, cudaStream_t s);
int* ssd_wait_flag_ptr();  // device address of the wait flag (current device), or null
bool ssd_tma_enabled();    // the tensor-map encoder is available and TMA is allowed
void ssd_set_tma(bool on);  // allow (default) or forbid TMA operand loads
// A [rows][H][64] bf16 tensor (x, dy) as a 3-D tensor map with boxes of 64
// channels x 1 head x 128 tokens and 128-byte swizzle; false if unavailable.
bool encode_head_map(CUtensorMap* m, const __nv_bfloat16* base, int64_t rows, int H);
cudaError_t launch_ssd_wait_probe(uint32_t polls, cudaStream_t s);

}  // namespace bds
