// ssd.cuh -- parameters of the SSD-form (Mamba-2, scalar decay per head)
// kernels of libbdscan. The recurrence, layouts and the block restriction are
// documented in include/bdscan_ssd.h.
#pragma once
#include <cstdint>
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
};

cudaError_t launch_ssd_block_state(const SsdStateParams& p, cudaStream_t s);
cudaError_t launch_ssd_state_pass(const SsdPassParams& p, cudaStream_t s);
cudaError_t launch_ssd_block_scan(bool noisy, const SsdScanParams& p, cudaStream_t s);
int* ssd_wait_flag_ptr();  // device address of the wait flag (current device), or null
cudaError_t launch_ssd_wait_probe(uint32_t polls, cudaStream_t s);

}  // namespace bds
