// params.h -- kernel argument blocks and internal launcher declarations.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace bds {

constexpr int kCtaHost = 128;  // channels per CTA (one per thread); equals kCta in device.cuh
// Longest block whose backward segment checkpoints stay in shared memory.
constexpr int kCkSmemMaxBs = 128;

// Geometry shared by all kernels of one call.
struct Geo {
  int64_t Bt, L, Bs, D;
  int nb;       // blocks per stream, L / Bs
  int m;        // blocks per time chunk
  int nc;       // chunks, ceil(nb / m)
  int nc_full;  // chunks holding m blocks
  int G;        // channel groups of 128, ceil(D / 128)
};

// Forward-side kernels: chunk-local scan, chunk carry, block scan.
struct FwdParams {
  Geo g;
  const void *xc, *dtc, *Bc, *Cc;
  const void *xn, *dtf, *Bf, *Cf, *dtr, *Br, *Cr;
  const float *Af, *Df, *Ar, *Dr;
  void *yc, *yn;
  float* states;       // [Bt][nb][D][N] when emit_all
  int emit_all;
  float* final_state;  // [Bt][D][N] or null: state after the last token
  float* hst;          // workspace [Bt][nc+1][D][N]: chunk-local states, then chunk start states
  float* sdt;          // workspace [Bt][nc][D]: sum of dt over each chunk
  const float* init;   // [Bt][D][N] or null: state before token 0
  const float* seed;   // active block: [Bt][D][N]
  int c_begin;         // first chunk handled by a block-scan launch
  int stage_bufs;      // block scan: 2 = copy the next block while computing, 1 = synchronous
  int rev;             // chunk-local scan: right to left in time (with block-scan mode 2)
  // active block with adaptive layer norm: per batch row shift, scale, gate
  // [Bt][D] and per token (mean, 1/sqrt(var + eps)) of the block's input
  const float *shift, *scale, *gate;
  const float2* ln_stats;
};

// Backward-side kernels.
struct BwdParams {
  Geo g;
  const void *xc, *dtc, *Bc, *Cc;
  const void *xn, *dtf, *Bf, *Cf, *dtr, *Br, *Cr;
  const float *Af, *Df, *Ar, *Dr;
  const float* states;
  const void *dyc, *dyn;
  const float* dstates;
  void *dxc, *ddtc, *dBc, *dCc;
  void *dxn, *ddtf, *dBf, *dCf, *ddtr, *dBr, *dCr;
  float *dAf, *dDf, *dAr, *dDr;
  // workspace
  float* dS;        // [Bt][nb][D][N]  gradient of each noisy block's seed
  float* Lc;        // [Bt][nc][D][N]  local clean adjoint carry, then the carry into each chunk end
  float* sdtc;      // [Bt][nc][D]
  float* part_tok;  // [6][Bt][L][G][N] per channel-group sums of dB_c, dC_c, dB_f, dC_f, dB_r, dC_r
  float* part_A;    // [3][Bt*nc][D][N] dA partial sums: noisy fwd, noisy rev, clean
  float* part_D;    // [2][Bt*nc][D]    dD partial sums: noisy, clean
  int seg_resident;  // set per launch: blocks of several segments staged whole
  // segment checkpoints of blocks above kCkSmemMaxBs tokens, in global memory:
  // per CTA (linear block index) (Bs/16 - 1) x N x 128 floats; null otherwise
  float* ck_noisy;
  float* ck_clean;
};

// Launchers (fwd.cu / bwd.cu). dt: 0 = f32 in/out, 1 = bf16 in/out, 2 = bf16 in, f32 out.
cudaError_t launch_chunk_local(int dt, int N, const FwdParams& p, cudaStream_t s);
cudaError_t launch_chunk_carry(int N, const FwdParams& p, cudaStream_t s);
// mode 0: all-block forward, 1: clean scan only (cache build), 2: clean scan right to left
cudaError_t launch_block_scan(int dt, int N, int mode, int nchunks, const FwdParams& p, cudaStream_t s);
// One noisy block per batch row from p.seed (len == block).
cudaError_t launch_active_block(int dt, int N, const FwdParams& p, cudaStream_t s);
// Per-token layer-norm statistics of rows x D elements (dt: 0 f32, else bf16).
// State groups of the diagonal form (groups.cu): d_state split into groups
// of 16 (the last one 8 or 16, zero-padded) run one after another.
constexpr size_t kGroupScratchBytes = (size_t)16 << 20;  // scratch of the grouped active block
cudaError_t launch_group_gather(const void* src, int elt, int64_t rows, int N, int n0, int gs, void* dst,
                                cudaStream_t s);
cudaError_t launch_group_scatter(const float* src, int64_t rows, int N, int n0, int gs, void* dst, int out_elt,
                                 cudaStream_t s);
cudaError_t launch_group_add(float* acc, const float* add, int64_t n, cudaStream_t s);
cudaError_t launch_group_out(const float* acc, void* out, int out_elt, int64_t n, cudaStream_t s);
void* group_scratch();  // device address of the grouped active block's scratch, or null

cudaError_t launch_ln_stats(int dt, const void* h, int64_t rows, int64_t D, float eps, float2* stats, cudaStream_t s);
// The active block on the modulated input (1 + scale) LN(x) + shift, writing
// x + gate * y_n (p.shift, p.scale, p.gate, p.ln_stats set).
cudaError_t launch_active_block_adaln(int dt, int N, const FwdParams& p, cudaStream_t s);
// y = yf + yr elementwise (n elements, a multiple of 4), rounded to f32 or bf16.
cudaError_t launch_combine(int out_f32, const float* yf, const float* yr, void* y, int64_t n, cudaStream_t s);
cudaError_t launch_bwd_noisy(int dt, int N, const BwdParams& p, cudaStream_t s);
cudaError_t launch_bwd_carry(int N, const BwdParams& p, cudaStream_t s);
cudaError_t launch_bwd_clean(int dt, int N, const BwdParams& p, cudaStream_t s);
cudaError_t launch_bwd_reduce_tok(int dt, int N, const BwdParams& p, cudaStream_t s);
cudaError_t launch_bwd_reduce_par(int N, const BwdParams& p, cudaStream_t s);


// Helpers of api.cu for other translation units of the library.
int api_fail(int code, const char* msg);
int api_ok();
void api_begin();
cudaError_t api_launched(cudaError_t e, cudaStream_t s);
cudaError_t set_smem_cached(const void* fn, int bytes, int carveout);  // carveout < 0: leave it
int sm_count_cached();  // 0 if unknown
int api_check_forward_dims(const void* dims, Geo* g, int* dt, int* N, const char* fn);
size_t api_fwd_workspace(const Geo& g, int N);
size_t api_bwd_workspace(const Geo& g, int N);
// Launch sequences of bdscan_forward / bdscan_backward (counted by the
// launch hook) for other entry points of the library.
cudaError_t api_run_forward(int dt, int N, FwdParams& p, void* workspace, cudaStream_t s);
cudaError_t api_run_boundary(int dt, int N, FwdParams& p, float* states, int emit_all, cudaStream_t s);
cudaError_t api_run_backward(int dt, int N, BwdParams& p, void* workspace, cudaStream_t s);
int bwd_chunk_count(int dt, int N, const Geo& g);
// Upper bound of the backward's chunks per batch row (sizes its workspace
// independently of the device): twice the forward chunking, at most one
// chunk per block.
inline int bwd_max_chunks(const Geo& g) { return g.nb < 2 * g.nc ? g.nb : 2 * g.nc; }

}  // namespace bds
