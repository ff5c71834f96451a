#pragma once
// bwd_common.cuh -- shared parts of the backward-side kernels of libbdscan
// (sm_103a): bwd_noisy.cu, bwd_clean.cu and bwd.cu.
//
// Reverse-mode derivative of <dy_c,y_c> + <dy_n,y_n> + <dstates,states> for
// the all-block forward. For a scan h_t = a_t h_prev + dt_t B_t x_t with
// a_t = exp(dt_t A), the adjoint gbar_t = dLoss/dh_t obeys
//     gbar_t = C_t dy_t + a_next gbar_next (+ injections),
// and with p_t = a_t h_prev (the decayed previous state):
//     dx_t  += dt_t sum_n gbar B_t          ddt_t = x_t sum_n gbar B_t + sum_n A gbar p_t
//     dA    += sum_t dt_t gbar p_t          dB_t  += sum_d gbar dt_t x_t
//     dC_t  += sum_d dy_t h_t               seed gradient = a_first gbar_first.
// The gradient of a noisy block's seed flows into the clean scan at the end
// of the previous block (eq. prefix-cache-gradient).
//
// Kernels (grid (channel groups, time chunks, batch) unless noted):
//   k_bwd_noisy  per chunk, blocks last to first: the clean stream's local
//                adjoint over the block with a zero carry at the chunk end;
//                the reverse direction of the noisy block (recompute right to
//                left, adjoint left to right); the forward direction
//                (recompute from the seed left to right, adjoint right to
//                left), whose seed gradient feeds the clean adjoint of the
//                previous block and is saved for the clean backward.
//   k_bwd_carry  per (batch, channel, state), chunks last to first: the exact
//                adjoint entering each chunk's last token.
//   k_bwd_clean  per chunk, blocks last to first: recompute the clean state
//                from the saved boundary states, run the adjoint from the
//                exact carry, emit the clean-stream gradients.
//   k_reduce_*   sum the per-channel-group dB, dC and the per-chunk dA, dD
//                partials in a fixed order (deterministic results).
// The recompute keeps its values for up to 16 tokens per thread in tensor
// memory (TMEM): 16 x N fp32 per thread would not fit in registers next to
// the scan state, and TMEM is otherwise idle in this path. k_bwd_noisy holds
// p_t of every token; k_bwd_clean holds the state entering every other token
// and redoes one scan step for the rest (half the columns, three CTAs per SM).
// Blocks longer than 16 tokens are processed in 16-token segments from
// checkpointed states.
//
// Arithmetic is packed two state indices per FFMA2/FMUL2/FADD2, and per-thread
// state vectors use the group-swizzled order of device.cuh, which makes the
// channel reductions of dB and dC mostly select-free.
#include "device.cuh"
#include "params.h"

namespace bds {

namespace {

// checkpoint slots in shared memory: ck[slot][N][kCta], any (private) order
template <int N>
__device__ __forceinline__ void ck_store(float* ck, int slot, const float2 (&h)[N / 2]) {
#pragma unroll
  for (int j = 0; j < N / 2; ++j) {
    ck[((size_t)slot * N + 2 * j) * kCta + threadIdx.x] = h[j].x;
    ck[((size_t)slot * N + 2 * j + 1) * kCta + threadIdx.x] = h[j].y;
  }
}
template <int N>
__device__ __forceinline__ void ck_load(float2 (&h)[N / 2], const float* ck, int slot) {
#pragma unroll
  for (int j = 0; j < N / 2; ++j)
    h[j] = make_float2(ck[((size_t)slot * N + 2 * j) * kCta + threadIdx.x],
                       ck[((size_t)slot * N + 2 * j + 1) * kCta + threadIdx.x]);
}

// Tokens per backward segment; also the fixed stride of the staged tiles and
// of the reduction buffer, so that their addresses are immediates.
constexpr int kBwdTS = 16;

// red[slot][i][warp][lane] (i < kBwdTS): per direction a dB slot (adjoint
// pass) and the next one for dC (recompute pass); every lane stores its
// warp_reduce_swz_part value, a partial for state lane % N. `mine` is this
// thread's place, red + warp * 32 + lane.
constexpr int kRedRow = kWarps * 32;  // floats per (which, token)
template <int N>
__device__ __forceinline__ float* red_slot(float* red) {
  return red + threadIdx.x;
}
template <int N>
__device__ __forceinline__ void red_put(float* mine, int which, int i, float v) {
  mine[(which * kBwdTS + i) * kRedRow] = v;
}

// Sums the 4 warps' rows (32/N lane partials each, in a fixed order) of the
// slots sB (a dB) and sC (a dC) and stores the CTA's channel-group partials
// of the two token-by-state gradients for tokens [tstart, tstart+TS).
template <int N>
__device__ void red_flush(const BwdParams& p, const float* red, int sB, int sC, int tensB, int tensC, int64_t b,
                          int64_t tstart, int TS) {
  __syncthreads();
  const Geo& g = p.g;
#pragma unroll
  for (int j0 = 0; j0 < 2 * kBwdTS * N; j0 += kCta) {
    const int j = j0 + threadIdx.x;
    const int which = j / (kBwdTS * N), i = (j / N) % kBwdTS, n = j % N;
    if (i < TS) {
      const float* src = red + ((which == 0 ? sB : sC) * kBwdTS + i) * kRedRow + n;
      float s = 0.f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w)
#pragma unroll
        for (int r = 0; r < 32 / N; ++r) s += src[w * 32 + r * N];
      const int tensor = which == 0 ? tensB : tensC;
      p.part_tok[((((int64_t)tensor * g.Bt + b) * g.L + tstart + i) * g.G + blockIdx.x) * N + n] = s;
    }
  }
  __syncthreads();
}

__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }

// Copies states[k-1] of the CTA's 128 channels (the seed of block k) into
// dst, [kCta][N] fp32, in the caller's cp.async group; zeros for k = 0 and
// for channels past D. The clean backward stages it with the block's inputs,
// so the state its recompute starts from arrives with the prefetch.
template <int N>
__device__ __forceinline__ void issue_seed(float* dst, const float* states, const Geo& g, int64_t b, int k,
                                           int64_t d0) {
  constexpr int CPC = N / 4;  // 16-byte chunks per channel
  for (int q = threadIdx.x; q < kCta * CPC; q += kCta) {
    const bool ok = k > 0 && d0 + q / CPC < g.D;
    const float* src = ok ? states + ((b * g.nb + (k - 1)) * g.D + d0) * N + (int64_t)q * 4 : states;
    cp_async16(dst + q * 4, src, ok ? 16 : 0);
  }
}

// The backward splits each batch row's blocks into g.nc nearly equal chunks
// (its own partition, chosen per call so the last wave of CTAs is nearly
// full); chunk c holds blocks [chunk_lo(c), chunk_lo(c+1)).
__host__ __device__ inline int chunk_lo(const Geo& g, int c) { return (int)(((int64_t)c * g.nb) / g.nc); }

__host__ __device__ inline uint32_t pow2_cols(uint32_t need) {
  uint32_t c = 32;
  while (c < need) c <<= 1;
  return c;
}
// TMEM columns of one segment's held values: every state (noisy kernel) or
// every other one (clean kernel).
__host__ __device__ inline uint32_t full_cols(int TS, int N) { return pow2_cols((uint32_t)(TS * N)); }
__host__ __device__ inline uint32_t half_cols(int TS, int N) { return pow2_cols((uint32_t)(((TS + 1) / 2) * N)); }

// The state update alone on a group-swizzled packed state (checkpoint passes).
template <int N>
__device__ __forceinline__ void scan_state_swz(float2 (&h)[N / 2], const float2 (&A2)[N / 2], float dt, float x,
                                               const float* Brow, int sw) {
  const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x));
  float2 B[N / 2];
  vload2<N>(B, Brow, sw);
#pragma unroll
  for (int j = 0; j < N / 2; ++j) h[j] = fma2(ex2x2(mul2(dt2, A2[j])), h[j], mul2(u2, B[j]));
}

// Backward of one scan direction over one segment of TS tokens.
// FWDDIR: the scan runs left to right (recompute i = 0..TS-1, adjoint
// i = TS-1..0); otherwise right to left.
//   h   the state the segment's first scanned token continues (clobbered)
//   g   a_next gbar_next entering the segment's last scanned token (in/out)
//   dA  accumulated sum of dt * gbar * p (in/out)
//   epi(i, dt, x, dy, sum_n gbar B, sum_n A2 gbar p) writes the per-token results.
//   off  the segment's first token in the staged tile
// Channel sums of dy*h (dC) and gbar*dt*x (dB) go to red slots rb + 1 and rb
// through this thread's place `mine`.
template <int N, bool FWDDIR, typename St, typename Epi>
__device__ __forceinline__ void seg_bwd(const St& st, int TS, int jx, int jdt, int jdy, int rB, int rC,
                                        const float2 (&A2)[N / 2], int sw, float2 (&h)[N / 2],
                                        float2 (&g)[N / 2], float2 (&dA)[N / 2], uint32_t tb, float* mine, int off, int rb,
                                        Epi epi) {
#pragma unroll 2
  for (int k = 0; k < TS; ++k) {  // recompute, in scan order
    const int i = FWDDIR ? k : TS - 1 - k;
    const float dt = st.at(jdt, off + i), x = st.at(jx, off + i), dy = st.at(jdy, off + i);
    const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x)), dy2 = f2(dy);
    float2 B[N / 2], pv[N / 2], w[N / 2];
    vload2<N>(B, st.row(rB, off + i), sw);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      const float2 a = ex2x2(mul2(dt2, A2[j]));
      pv[j] = mul2(a, h[j]);
      h[j] = fma2(u2, B[j], pv[j]);
      w[j] = mul2(dy2, h[j]);
    }
    tmem_st2<N>(tb + (uint32_t)(i * N), pv);
    red_put<N>(mine, rb + 1, off + i, warp_reduce_swz_part<N>(w));
  }
  tmem_wait_st();
#pragma unroll 4
  for (int k = 0; k < TS; ++k) {  // adjoint, against scan order
    const int i = FWDDIR ? TS - 1 - k : k;
    float2 pv[N / 2];
    tmem_ld2<N>(tb + (uint32_t)(i * N), pv);
    const float dt = st.at(jdt, off + i), x = st.at(jx, off + i), dy = st.at(jdy, off + i);
    const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x)), dy2 = f2(dy);
    float2 B[N / 2], C[N / 2], w[N / 2];
    vload2<N>(B, st.row(rB, off + i), sw);
    vload2<N>(C, st.row(rC, off + i), sw);
    float2 sg[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    float2 sa[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      const float2 a = ex2x2(mul2(dt2, A2[j]));
      const float2 gb = fma2(C[j], dy2, g[j]);
      g[j] = mul2(a, gb);
      const float2 q = mul2(gb, pv[j]);
      sa[j & 1] = fma2(A2[j], q, sa[j & 1]);
      dA[j] = fma2(dt2, q, dA[j]);
      sg[j & 1] = fma2(gb, B[j], sg[j & 1]);
      w[j] = mul2(gb, u2);
    }
    red_put<N>(mine, rb, off + i, warp_reduce_swz_part<N>(w));
    const float2 sgs = add2(sg[0], sg[1]), sas = add2(sa[0], sa[1]);
    epi(i, dt, x, dy, __fadd_rn(sgs.x, sgs.y), __fadd_rn(sas.x, sas.y));
  }
}

// seg_bwd holding half of the states, for the clean kernel: its smaller TMEM
// footprint lets three CTAs share an SM. Arguments as for seg_bwd, except
//   tb   TMEM, (TS+1)/2 slots of N columns: the state entering every even
//        scan step.
// The adjoint takes the steps two at a time from the end. For steps k and
// k-1 it reloads the state entering k-1 and redoes step k-1 to get the state
// entering k, with the operations of the recompute (so the same bits); the
// decay a_{k-1} that this needs is the one the adjoint of step k-1 uses.
template <int N, bool FWDDIR, typename St, typename Epi>
__device__ __forceinline__ void seg_bwd_half(const St& st, int TS, int jx, int jdt, int jdy, int rB, int rC,
                                             const float2 (&A2)[N / 2], int sw, float2 (&h)[N / 2],
                                             float2 (&g)[N / 2], float2 (&dA)[N / 2], uint32_t tb, float* mine, int off, int rb,
                                             Epi epi) {
#pragma unroll 2
  for (int k = 0; k < TS; ++k) {  // recompute, in scan order
    const int i = FWDDIR ? k : TS - 1 - k;
    if ((k & 1) == 0) tmem_st2<N>(tb + (uint32_t)((k >> 1) * N), h);
    const float dt = st.at(jdt, off + i), x = st.at(jx, off + i), dy = st.at(jdy, off + i);
    const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x)), dy2 = f2(dy);
    float2 B[N / 2], w[N / 2];
    vload2<N>(B, st.row(rB, off + i), sw);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      const float2 a = ex2x2(mul2(dt2, A2[j]));
      h[j] = fma2(u2, B[j], mul2(a, h[j]));
      w[j] = mul2(dy2, h[j]);
    }
    red_put<N>(mine, rb + 1, off + i, warp_reduce_swz_part<N>(w));
  }
  tmem_wait_st();

  // one adjoint step at token i, given a = a_i and pv = a_i * (state entering i)
  auto step = [&](int i, const float2 (&a)[N / 2], const float2 (&pv)[N / 2]) {
    const float dt = st.at(jdt, off + i), x = st.at(jx, off + i), dy = st.at(jdy, off + i);
    const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x)), dy2 = f2(dy);
    float2 B[N / 2], C[N / 2], w[N / 2];
    vload2<N>(B, st.row(rB, off + i), sw);
    vload2<N>(C, st.row(rC, off + i), sw);
    float2 sg[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    float2 sa[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      const float2 gb = fma2(C[j], dy2, g[j]);
      g[j] = mul2(a[j], gb);
      const float2 q = mul2(gb, pv[j]);
      sa[j & 1] = fma2(A2[j], q, sa[j & 1]);
      dA[j] = fma2(dt2, q, dA[j]);
      sg[j & 1] = fma2(gb, B[j], sg[j & 1]);
      w[j] = mul2(gb, u2);
    }
    red_put<N>(mine, rb, off + i, warp_reduce_swz_part<N>(w));
    const float2 sgs = add2(sg[0], sg[1]), sas = add2(sa[0], sa[1]);
    epi(i, dt, x, dy, __fadd_rn(sgs.x, sgs.y), __fadd_rn(sas.x, sas.y));
  };

  int k = TS - 1;
  if ((TS & 1) != 0) {  // an odd count: the last step alone, its entering state is held
    const int i = FWDDIR ? k : TS - 1 - k;
    float2 S[N / 2], a[N / 2], pv[N / 2];
    tmem_ld2<N>(tb + (uint32_t)((k >> 1) * N), S);
    const float2 dt2 = f2(st.at(jdt, off + i));
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      a[j] = ex2x2(mul2(dt2, A2[j]));
      pv[j] = mul2(a[j], S[j]);
    }
    step(i, a, pv);
    --k;
  }
#pragma unroll 1
  for (; k > 0; k -= 2) {  // steps k (odd) and k-1
    const int i0 = FWDDIR ? k : TS - 1 - k, i1 = FWDDIR ? k - 1 : TS - k;
    float2 S[N / 2], a0[N / 2], pv0[N / 2], a1[N / 2], pv1[N / 2];
    tmem_ld2<N>(tb + (uint32_t)(((k - 1) >> 1) * N), S);  // state entering step k-1
    {
      const float dt1 = st.at(jdt, off + i1), x1 = st.at(jx, off + i1);
      const float2 dt12 = f2(dt1), u12 = f2(__fmul_rn(dt1, x1)), dt02 = f2(st.at(jdt, off + i0));
      float2 B1[N / 2];
      vload2<N>(B1, st.row(rB, off + i1), sw);
#pragma unroll
      for (int j = 0; j < N / 2; ++j) {
        a1[j] = ex2x2(mul2(dt12, A2[j]));
        pv1[j] = mul2(a1[j], S[j]);
        const float2 hk = fma2(u12, B1[j], pv1[j]);  // state entering step k
        a0[j] = ex2x2(mul2(dt02, A2[j]));
        pv0[j] = mul2(a0[j], hk);
      }
    }
    step(i0, a0, pv0);
    step(i1, a1, pv1);
  }
}


}  // namespace

// ---------------------------------------------------------------------------
// launch sizing shared by the backward kernels
// ---------------------------------------------------------------------------
namespace {

// Dynamic shared memory is padded so that no more CTAs share an SM than its
// 512 TMEM columns can hold at once.
inline size_t pad_for_tmem(size_t smem, uint32_t cols) {
  const int ctas = (int)(512 / cols);
  if (ctas >= 16) return smem;  // the thread limit already bounds residency
  const size_t cap = (size_t)(220 * 1024) / (size_t)ctas;
  const size_t need = cap > 2048 ? cap - 2048 : cap;
  return smem > need ? smem : need;
}

// Both attributes are set before every launch and before the occupancy query:
// the padded shared memory exceeds the 48 KB default, and without the largest
// carveout the driver may configure an SM for one such CTA instead of the two
// its TMEM can hold.
template <typename K>
cudaError_t set_bwd_attrs(K kernel, size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, (int)cudaSharedmemCarveoutMaxShared);
}

// Resident CTAs per SM of a backward kernel (0 on failure), from the per-SM
// limits: TMEM columns, registers (each of the four SM sub-partitions holds
// whole warps, registers allocated per thread in multiples of 8), shared
// memory with the per-CTA reserve, and threads. The runtime's occupancy
// calculator reports one CTA for the noisy kernel where the hardware admits
// two, so it is not used.
template <typename K>
int resident_ctas(K kernel, size_t smem, uint32_t tcols, int dev) {
  cudaFuncAttributes fa;
  int sm_smem = 0, sm_regs = 0, sm_threads = 0, reserve = 0;
  if (set_bwd_attrs(kernel, smem) != cudaSuccess || cudaFuncGetAttributes(&fa, kernel) != cudaSuccess ||
      cudaDeviceGetAttribute(&sm_smem, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sm_regs, cudaDevAttrMaxRegistersPerMultiprocessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sm_threads, cudaDevAttrMaxThreadsPerMultiProcessor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&reserve, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  const int by_tmem = (int)(512 / tcols);
  const int warp_regs = ((fa.numRegs + 7) / 8 * 8) * 32;
  const int by_regs = warp_regs > 0 ? (sm_regs / 4 / warp_regs) * 4 / kWarps : 0;
  const int by_smem = (int)((size_t)sm_smem / (smem + fa.sharedSizeBytes + (size_t)reserve));
  const int by_threads = sm_threads / kCta;
  int n = by_tmem;
  n = by_regs < n ? by_regs : n;
  n = by_smem < n ? by_smem : n;
  n = by_threads < n ? by_threads : n;
  return n;
}

// Shared memory of a launch, and whether a block of several segments is
// staged whole (one buffer per segment): only where that costs no resident CTA.
struct BwdLaunch {
  size_t smem;
  int resident;
};
template <typename L, typename K>
BwdLaunch bwd_launch(K kernel, int Bs, uint32_t cols, int dev) {
  const int TS = Bs < 16 ? Bs : 16, nseg = Bs / TS;
  if (nseg == 1) return {pad_for_tmem(L::bytes(2, TS, Bs), cols), 0};
  const size_t one = pad_for_tmem(L::bytes(1, TS, Bs), cols), all = pad_for_tmem(L::bytes(nseg, TS, Bs), cols);
  const int r1 = resident_ctas(kernel, one, cols, dev), ra = resident_ctas(kernel, all, cols, dev);
  return ra >= r1 && ra > 0 ? BwdLaunch{all, 1} : BwdLaunch{one, 0};
}
}  // namespace

#define BDS_DISPATCH_N(N, ...)                      \
  switch (N) {                                      \
    case 8: { constexpr int NN = 8; __VA_ARGS__ }   \
    case 16: { constexpr int NN = 16; __VA_ARGS__ } \
    default: return cudaErrorInvalidValue;          \
  }


// Resident CTAs per SM of the two TMEM kernels, as launched for this block
// size (0 on failure): bwd_noisy.cu and bwd_clean.cu.
int bwd_noisy_per_sm(int dt, int N, int Bs, int dev);
int bwd_clean_per_sm(int dt, int N, int Bs, int dev);

}  // namespace bds
