// bwd.cu -- backward-side kernels of libbdscan (sm_103a).
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
// The recompute stores p_t for up to 16 tokens per thread in tensor memory
// (TMEM): 16 x N fp32 per thread would not fit in registers next to the
// scan state, and TMEM is otherwise idle in this path. Blocks longer than 16
// tokens are processed in 16-token segments from checkpointed states.
#include "device.cuh"
#include "params.h"

namespace bds {

namespace {

template <int N>
__device__ __forceinline__ void ck_store(float* ck, int slot, const float (&h)[N]) {
#pragma unroll
  for (int n = 0; n < N; ++n) ck[((size_t)slot * N + n) * kCta + threadIdx.x] = h[n];
}
template <int N>
__device__ __forceinline__ void ck_load(float (&h)[N], const float* ck, int slot) {
#pragma unroll
  for (int n = 0; n < N; ++n) h[n] = ck[((size_t)slot * N + n) * kCta + threadIdx.x];
}

// red[which][i][warp][n]: which 0 = dB (adjoint pass), 1 = dC (recompute pass).
template <int N>
__device__ __forceinline__ void red_put(float* red, int which, int TS, int i, float v) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane < N) red[(((size_t)which * TS + i) * kWarps + warp) * N + lane] = v;
}

// Sums the 4 warps' rows and stores the CTA's channel-group partials of two
// token-by-state gradients for tokens [tstart, tstart+TS).
template <int N>
__device__ void red_flush(const BwdParams& p, const float* red, int tensB, int tensC, int64_t b,
                          int64_t tstart, int TS) {
  __syncthreads();
  const Geo& g = p.g;
  for (int j = threadIdx.x; j < 2 * TS * N; j += kCta) {
    const int which = j / (TS * N), r = j - which * TS * N, i = r / N, n = r - i * N;
    const float* src = red + (((size_t)which * TS + i) * kWarps) * N + n;
    float s = src[0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) s += src[w * N];
    const int tensor = which == 0 ? tensB : tensC;
    p.part_tok[((((int64_t)tensor * g.Bt + b) * g.L + tstart + i) * g.G + blockIdx.x) * N + n] = s;
  }
  __syncthreads();
}

__host__ __device__ inline size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }

// TMEM columns per CTA and the residency that allows (512 columns per SM).
__host__ __device__ inline uint32_t tcols_host(int TS, int N) {
  uint32_t need = (uint32_t)(TS * N), c = 32;
  while (c < need) c <<= 1;
  return c;
}

}  // namespace

// ---------------------------------------------------------------------------
// Noisy blocks (both directions) + the clean stream's chunk-local adjoint
// ---------------------------------------------------------------------------
template <typename T, int N>
struct NoisyBwdSmem {
  // token-by-channel: x_n, dt_f, dt_r, dy_n, dt_c, dy_c; token-by-state: B_f, C_f, B_r, C_r, C_c
  using St = Stage<T, N, 6, 5>;
  static __host__ __device__ size_t stage_off() { return 0; }
  static __host__ __device__ size_t dx_off(int TS) { return align16(St::bytes(TS)); }
  static __host__ __device__ size_t red_off(int TS, int Bs) { return dx_off(TS) + (size_t)Bs * kCta * 4; }
  static __host__ __device__ size_t ck_off(int TS, int Bs) { return red_off(TS, Bs) + (size_t)2 * TS * kWarps * N * 4; }
  static __host__ __device__ size_t slot_off(int TS, int Bs) {
    const int nseg = Bs / TS;
    return ck_off(TS, Bs) + (size_t)(nseg > 1 ? nseg - 1 : 1) * N * kCta * 4;
  }
  static __host__ __device__ size_t bytes(int TS, int Bs) { return slot_off(TS, Bs) + 16; }
};

template <typename T, typename TO, int N>
__global__ void __launch_bounds__(kCta, 1) k_bwd_noisy(const BwdParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  using L = NoisyBwdSmem<T, N>;
  const Geo& g = p.g;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  (void)lane;
  const int64_t b = blockIdx.z;
  const int c = blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + tid;
  const bool act = d < g.D;
  const int Bs = (int)g.Bs, TS = Bs < 16 ? Bs : 16, NSEG = Bs / TS;
  const int k_lo = c * g.m, k_hi = min(k_lo + g.m, g.nb) - 1;

  enum { XN = 0, DTF = 1, DTR = 2, DYN = 3, DTC = 4, DYC = 5 };
  enum { BF = 0, CF = 1, BR = 2, CR = 3, CC = 4 };
  typename L::St st;
  st.carve(smem, TS);
  st.td_src[XN] = (const T*)p.xn;
  st.td_src[DTF] = (const T*)p.dtf;
  st.td_src[DTR] = (const T*)p.dtr;
  st.td_src[DYN] = (const T*)p.dyn;
  st.td_src[DTC] = (const T*)p.dtc;
  st.td_src[DYC] = (const T*)p.dyc;
  st.row_src[BF] = (const T*)p.Bf;
  st.row_src[CF] = (const T*)p.Cf;
  st.row_src[BR] = (const T*)p.Br;
  st.row_src[CR] = (const T*)p.Cr;
  st.row_src[CC] = (const T*)p.Cc;
  float* dxbuf = reinterpret_cast<float*>(smem + L::dx_off(TS));
  float* red = reinterpret_cast<float*>(smem + L::red_off(TS, Bs));
  float* ck = reinterpret_cast<float*>(smem + L::ck_off(TS, Bs));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + L::slot_off(TS, Bs));

  const uint32_t tcols = tmem_cols_for((uint32_t)(TS * N));
  if (warp == 0) tmem_alloc(tslot, tcols);
  tmem_sync();
  const uint32_t tbase = *tslot;
  const uint32_t tb = tbase + ((uint32_t)(warp * 32) << 16);

  float A2f[N], A2r[N];
  vzero(A2f);
  vzero(A2r);
  float Dsum = 0.f;
  if (act) {
    vload(A2f, p.Af + d * N);
    vload(A2r, p.Ar + d * N);
#pragma unroll
    for (int n = 0; n < N; ++n) {
      A2f[n] = __fmul_rn(A2f[n], kLog2e);
      A2r[n] = __fmul_rn(A2r[n], kLog2e);
    }
    Dsum = __fadd_rn(p.Df[d], p.Dr[d]);
  }
  float dAf[N], dAr[N];
  vzero(dAf);
  vzero(dAr);
  float dDn = 0.f, sdt = 0.f;
  float carry[N];  // clean stream: a_{t+1} gbar_{t+1} (+ injections) entering token t from the right
  vzero(carry);
  float dSn[N];  // seed gradient of the block to the right of the current one
  vzero(dSn);

  for (int k = k_hi; k >= k_lo; --k) {
    const int64_t t0 = (int64_t)k * Bs;
    const int64_t row0 = b * g.L + t0;
    if (NSEG == 1) st.load(row0, TS, g.D, d0);

    // ---- clean stream: chunk-local adjoint over block k ----
    if (k < k_hi) {
#pragma unroll
      for (int n = 0; n < N; ++n) carry[n] = __fadd_rn(carry[n], dSn[n]);
      if (p.dstates != nullptr && act) {
        float e[N];
        vload(e, p.dstates + ((b * g.nb + k) * g.D + d) * N);
#pragma unroll
        for (int n = 0; n < N; ++n) carry[n] = __fadd_rn(carry[n], e[n]);
      }
    }
    for (int s = NSEG - 1; s >= 0; --s) {
      if (NSEG > 1) st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
      for (int i = TS - 1; i >= 0; --i) {
        const float dt = st.at(DTC, i), dy = st.at(DYC, i);
        float C[N];
        vload_row(C, st.row(CC, i));
#pragma unroll
        for (int n = 0; n < N; ++n) {
          const float gb = __fmaf_rn(C[n], dy, carry[n]);
          carry[n] = __fmul_rn(ex2(__fmul_rn(dt, A2f[n])), gb);
        }
        sdt = __fadd_rn(sdt, dt);
      }
    }

    // ---- noisy block k, reverse direction ----
    {
      if (NSEG > 1) {
        float h[N];
        vzero(h);
        for (int s = NSEG - 1; s >= 1; --s) {
          st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
          for (int i = TS - 1; i >= 0; --i) scan_state(h, A2r, st.at(DTR, i), st.at(XN, i), st.row(BR, i));
          ck_store(ck, s - 1, h);
        }
      }
      float gr[N];  // a_{t-1} gbar_{t-1}, entering token t from the left
      vzero(gr);
      for (int s = 0; s < NSEG; ++s) {
        if (NSEG > 1) st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
        float h[N];
        if (s == NSEG - 1)
          vzero(h);
        else
          ck_load(h, ck, s);
        for (int i = TS - 1; i >= 0; --i) {  // recompute, right to left
          const float dt = st.at(DTR, i), x = st.at(XN, i), dy = st.at(DYN, i);
          const float u = __fmul_rn(dt, x);
          float B[N], pv[N], w[N];
          vload_row(B, st.row(BR, i));
#pragma unroll
          for (int n = 0; n < N; ++n) {
            const float a = ex2(__fmul_rn(dt, A2r[n]));
            pv[n] = __fmul_rn(a, h[n]);
            h[n] = __fmaf_rn(u, B[n], pv[n]);
            w[n] = __fmul_rn(dy, h[n]);
          }
          Tmem<N>::st(tb + (uint32_t)(i * N), pv);
          red_put<N>(red, 1, TS, i, warp_reduce_scatter<N>(w));
        }
        tmem_wait_st();
        for (int i = 0; i < TS; ++i) {  // adjoint, left to right
          const float dt = st.at(DTR, i), x = st.at(XN, i), dy = st.at(DYN, i);
          const float u = __fmul_rn(dt, x);
          float B[N], C[N], pv[N], w[N];
          vload_row(B, st.row(BR, i));
          vload_row(C, st.row(CR, i));
          Tmem<N>::ld(tb + (uint32_t)(i * N), pv);
          float sgB = 0.f, sAq = 0.f;
#pragma unroll
          for (int n = 0; n < N; ++n) {
            const float a = ex2(__fmul_rn(dt, A2r[n]));
            const float gb = __fmaf_rn(C[n], dy, gr[n]);
            gr[n] = __fmul_rn(a, gb);
            const float q = __fmul_rn(gb, pv[n]);
            sAq = __fmaf_rn(A2r[n], q, sAq);
            dAr[n] = __fmaf_rn(dt, q, dAr[n]);
            sgB = __fmaf_rn(gb, B[n], sgB);
            w[n] = __fmul_rn(gb, u);
          }
          red_put<N>(red, 0, TS, i, warp_reduce_scatter<N>(w));
          const int ib = s * TS + i;
          if (act)
            reinterpret_cast<TO*>(p.ddtr)[(row0 + ib) * g.D + d] =
                to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
          dxbuf[ib * kCta + tid] = __fmul_rn(dt, sgB);
        }
        red_flush<N>(p, red, 4, 5, b, t0 + (int64_t)s * TS, TS);
      }
    }

    // ---- noisy block k, forward direction (seeded with states[k-1]) ----
    {
      float seed[N];
      vzero(seed);
      if (k > 0 && act) vload(seed, p.states + ((b * g.nb + (k - 1)) * g.D + d) * N);
      if (NSEG > 1) {
        float h[N];
#pragma unroll
        for (int n = 0; n < N; ++n) h[n] = seed[n];
        for (int s = 0; s < NSEG - 1; ++s) {
          st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
          for (int i = 0; i < TS; ++i) scan_state(h, A2f, st.at(DTF, i), st.at(XN, i), st.row(BF, i));
          ck_store(ck, s, h);
        }
      }
      float gf[N];  // a_{t+1} gbar_{t+1}, entering token t from the right
      vzero(gf);
      for (int s = NSEG - 1; s >= 0; --s) {
        if (NSEG > 1) st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
        float h[N];
        if (s == 0) {
#pragma unroll
          for (int n = 0; n < N; ++n) h[n] = seed[n];
        } else {
          ck_load(h, ck, s - 1);
        }
        for (int i = 0; i < TS; ++i) {  // recompute, left to right
          const float dt = st.at(DTF, i), x = st.at(XN, i), dy = st.at(DYN, i);
          const float u = __fmul_rn(dt, x);
          float B[N], pv[N], w[N];
          vload_row(B, st.row(BF, i));
#pragma unroll
          for (int n = 0; n < N; ++n) {
            const float a = ex2(__fmul_rn(dt, A2f[n]));
            pv[n] = __fmul_rn(a, h[n]);
            h[n] = __fmaf_rn(u, B[n], pv[n]);
            w[n] = __fmul_rn(dy, h[n]);
          }
          Tmem<N>::st(tb + (uint32_t)(i * N), pv);
          red_put<N>(red, 1, TS, i, warp_reduce_scatter<N>(w));
        }
        tmem_wait_st();
        for (int i = TS - 1; i >= 0; --i) {  // adjoint, right to left
          const float dt = st.at(DTF, i), x = st.at(XN, i), dy = st.at(DYN, i);
          const float u = __fmul_rn(dt, x);
          float B[N], C[N], pv[N], w[N];
          vload_row(B, st.row(BF, i));
          vload_row(C, st.row(CF, i));
          Tmem<N>::ld(tb + (uint32_t)(i * N), pv);
          float sgB = 0.f, sAq = 0.f;
#pragma unroll
          for (int n = 0; n < N; ++n) {
            const float a = ex2(__fmul_rn(dt, A2f[n]));
            const float gb = __fmaf_rn(C[n], dy, gf[n]);
            gf[n] = __fmul_rn(a, gb);
            const float q = __fmul_rn(gb, pv[n]);
            sAq = __fmaf_rn(A2f[n], q, sAq);
            dAf[n] = __fmaf_rn(dt, q, dAf[n]);
            sgB = __fmaf_rn(gb, B[n], sgB);
            w[n] = __fmul_rn(gb, u);
          }
          red_put<N>(red, 0, TS, i, warp_reduce_scatter<N>(w));
          const int ib = s * TS + i;
          const int64_t o = (row0 + ib) * g.D + d;
          if (act) {
            reinterpret_cast<TO*>(p.ddtf)[o] = to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
            const float dxv = __fmaf_rn(Dsum, dy, __fadd_rn(dxbuf[ib * kCta + tid], __fmul_rn(dt, sgB)));
            reinterpret_cast<TO*>(p.dxn)[o] = to_out<TO>(dxv);
          }
          dDn = __fmaf_rn(dy, x, dDn);
        }
        red_flush<N>(p, red, 2, 3, b, t0 + (int64_t)s * TS, TS);
      }
      // gradient of this block's seed, states[k-1]: a_{t0} gbar_{t0}
#pragma unroll
      for (int n = 0; n < N; ++n) dSn[n] = gf[n];
      if (k > 0 && act) vstore(p.dS + ((b * g.nb + (k - 1)) * g.D + d) * N, gf);
    }
  }

  if (act) {
    vstore(p.Lc + ((b * g.nc + c) * g.D + d) * N, carry);
    p.sdtc[(b * g.nc + c) * g.D + d] = sdt;
    const int64_t u = b * g.nc + c, U = g.Bt * g.nc;
    vstore(p.part_A + ((0 * U + u) * g.D + d) * N, dAf);
    vstore(p.part_A + ((1 * U + u) * g.D + d) * N, dAr);
    p.part_D[(0 * U + u) * g.D + d] = dDn;
  }
  tmem_sync();
  if (warp == 0) tmem_dealloc(tbase, tcols);
}

// ---------------------------------------------------------------------------
// Carry of the clean adjoint across chunks
// ---------------------------------------------------------------------------
template <int N>
__global__ void __launch_bounds__(256) k_bwd_carry(const BwdParams p) {
  const Geo& g = p.g;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= g.Bt * g.D * N) return;
  const int n = (int)(idx % N);
  const int64_t d = (idx / N) % g.D, b = idx / ((int64_t)N * g.D);
  const float A2 = __fmul_rn(p.Af[d * N + n], kLog2e);
  float G = 0.f;  // a_{t+1} gbar_{t+1} entering the current chunk's last token from the right
  for (int c = g.nc - 1; c >= 0; --c) {
    const int kl = min((c + 1) * g.m, g.nb) - 1;
    float gin = G;
    if (kl + 1 < g.nb) gin = __fadd_rn(gin, p.dS[((b * g.nb + kl) * g.D + d) * N + n]);
    if (p.dstates != nullptr) gin = __fadd_rn(gin, p.dstates[((b * g.nb + kl) * g.D + d) * N + n]);
    const int64_t o = ((b * g.nc + c) * g.D + d) * N + n;
    const float loc = p.Lc[o];
    const float s = p.sdtc[(b * g.nc + c) * g.D + d];
    p.Lc[o] = gin;
    G = __fmaf_rn(ex2(__fmul_rn(A2, s)), gin, loc);
  }
}

// ---------------------------------------------------------------------------
// Clean stream backward from the exact chunk carries
// ---------------------------------------------------------------------------
template <typename T, int N>
struct CleanBwdSmem {
  using St = Stage<T, N, 3, 2>;  // x_c, dt_c, dy_c; B_c, C_c
  static __host__ __device__ size_t red_off(int TS) { return align16(St::bytes(TS)); }
  static __host__ __device__ size_t ck_off(int TS) { return red_off(TS) + (size_t)2 * TS * kWarps * N * 4; }
  static __host__ __device__ size_t slot_off(int TS, int Bs) {
    const int nseg = Bs / TS;
    return ck_off(TS) + (size_t)(nseg > 1 ? nseg - 1 : 1) * N * kCta * 4;
  }
  static __host__ __device__ size_t bytes(int TS, int Bs) { return slot_off(TS, Bs) + 16; }
};

template <typename T, typename TO, int N>
__global__ void __launch_bounds__(kCta, 1) k_bwd_clean(const BwdParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  using L = CleanBwdSmem<T, N>;
  const Geo& g = p.g;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int64_t b = blockIdx.z;
  const int c = blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + tid;
  const bool act = d < g.D;
  const int Bs = (int)g.Bs, TS = Bs < 16 ? Bs : 16, NSEG = Bs / TS;
  const int k_lo = c * g.m, k_hi = min(k_lo + g.m, g.nb) - 1;

  enum { XC = 0, DTC = 1, DYC = 2 };
  enum { BC = 0, CC = 1 };
  typename L::St st;
  st.carve(smem, TS);
  st.td_src[XC] = (const T*)p.xc;
  st.td_src[DTC] = (const T*)p.dtc;
  st.td_src[DYC] = (const T*)p.dyc;
  st.row_src[BC] = (const T*)p.Bc;
  st.row_src[CC] = (const T*)p.Cc;
  float* red = reinterpret_cast<float*>(smem + L::red_off(TS));
  float* ck = reinterpret_cast<float*>(smem + L::ck_off(TS));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + L::slot_off(TS, Bs));

  const uint32_t tcols = tmem_cols_for((uint32_t)(TS * N));
  if (warp == 0) tmem_alloc(tslot, tcols);
  tmem_sync();
  const uint32_t tbase = *tslot;
  const uint32_t tb = tbase + ((uint32_t)(warp * 32) << 16);

  float A2[N];
  vzero(A2);
  float Df = 0.f;
  if (act) {
    vload(A2, p.Af + d * N);
#pragma unroll
    for (int n = 0; n < N; ++n) A2[n] = __fmul_rn(A2[n], kLog2e);
    Df = p.Df[d];
  }
  float dA[N];
  vzero(dA);
  float dDc = 0.f;
  float gc[N];  // a_{t+1} gbar_{t+1} (+ injections) entering token t from the right
  vzero(gc);

  for (int k = k_hi; k >= k_lo; --k) {
    const int64_t t0 = (int64_t)k * Bs;
    const int64_t row0 = b * g.L + t0;
    if (NSEG == 1) st.load(row0, TS, g.D, d0);
    if (k == k_hi) {
      if (act) vload(gc, p.Lc + ((b * g.nc + c) * g.D + d) * N);
    } else if (act) {
      float e[N];
      vload(e, p.dS + ((b * g.nb + k) * g.D + d) * N);
#pragma unroll
      for (int n = 0; n < N; ++n) gc[n] = __fadd_rn(gc[n], e[n]);
      if (p.dstates != nullptr) {
        vload(e, p.dstates + ((b * g.nb + k) * g.D + d) * N);
#pragma unroll
        for (int n = 0; n < N; ++n) gc[n] = __fadd_rn(gc[n], e[n]);
      }
    }
    float seed[N];
    vzero(seed);
    if (k > 0 && act) vload(seed, p.states + ((b * g.nb + (k - 1)) * g.D + d) * N);
    if (NSEG > 1) {
      float h[N];
#pragma unroll
      for (int n = 0; n < N; ++n) h[n] = seed[n];
      for (int s = 0; s < NSEG - 1; ++s) {
        st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
        for (int i = 0; i < TS; ++i) scan_state(h, A2, st.at(DTC, i), st.at(XC, i), st.row(BC, i));
        ck_store(ck, s, h);
      }
    }
    for (int s = NSEG - 1; s >= 0; --s) {
      if (NSEG > 1) st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
      float h[N];
      if (s == 0) {
#pragma unroll
        for (int n = 0; n < N; ++n) h[n] = seed[n];
      } else {
        ck_load(h, ck, s - 1);
      }
      for (int i = 0; i < TS; ++i) {  // recompute, left to right
        const float dt = st.at(DTC, i), x = st.at(XC, i), dy = st.at(DYC, i);
        const float u = __fmul_rn(dt, x);
        float B[N], pv[N], w[N];
        vload_row(B, st.row(BC, i));
#pragma unroll
        for (int n = 0; n < N; ++n) {
          const float a = ex2(__fmul_rn(dt, A2[n]));
          pv[n] = __fmul_rn(a, h[n]);
          h[n] = __fmaf_rn(u, B[n], pv[n]);
          w[n] = __fmul_rn(dy, h[n]);
        }
        Tmem<N>::st(tb + (uint32_t)(i * N), pv);
        red_put<N>(red, 1, TS, i, warp_reduce_scatter<N>(w));
      }
      tmem_wait_st();
      for (int i = TS - 1; i >= 0; --i) {  // adjoint, right to left
        const float dt = st.at(DTC, i), x = st.at(XC, i), dy = st.at(DYC, i);
        const float u = __fmul_rn(dt, x);
        float B[N], C[N], pv[N], w[N];
        vload_row(B, st.row(BC, i));
        vload_row(C, st.row(CC, i));
        Tmem<N>::ld(tb + (uint32_t)(i * N), pv);
        float sgB = 0.f, sAq = 0.f;
#pragma unroll
        for (int n = 0; n < N; ++n) {
          const float a = ex2(__fmul_rn(dt, A2[n]));
          const float gb = __fmaf_rn(C[n], dy, gc[n]);
          gc[n] = __fmul_rn(a, gb);
          const float q = __fmul_rn(gb, pv[n]);
          sAq = __fmaf_rn(A2[n], q, sAq);
          dA[n] = __fmaf_rn(dt, q, dA[n]);
          sgB = __fmaf_rn(gb, B[n], sgB);
          w[n] = __fmul_rn(gb, u);
        }
        red_put<N>(red, 0, TS, i, warp_reduce_scatter<N>(w));
        const int64_t o = (row0 + s * TS + i) * g.D + d;
        if (act) {
          reinterpret_cast<TO*>(p.ddtc)[o] = to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
          reinterpret_cast<TO*>(p.dxc)[o] = to_out<TO>(__fmaf_rn(Df, dy, __fmul_rn(dt, sgB)));
        }
        dDc = __fmaf_rn(dy, x, dDc);
      }
      red_flush<N>(p, red, 0, 1, b, t0 + (int64_t)s * TS, TS);
    }
  }
  if (act) {
    const int64_t u = b * g.nc + c, U = g.Bt * g.nc;
    vstore(p.part_A + ((2 * U + u) * g.D + d) * N, dA);
    p.part_D[(1 * U + u) * g.D + d] = dDc;
  }
  tmem_sync();
  if (warp == 0) tmem_dealloc(tbase, tcols);
}

// ---------------------------------------------------------------------------
// Deterministic reductions
// ---------------------------------------------------------------------------
template <typename TO, int N>
__global__ void __launch_bounds__(256) k_reduce_tok(const BwdParams p) {
  const Geo& g = p.g;
  const int64_t rows = g.Bt * g.L;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= 6 * rows * N) return;
  const int n = (int)(idx % N);
  const int64_t row = idx / N;
  const int tensor = (int)(row / rows);
  const int64_t bt = row - (int64_t)tensor * rows;
  const float* src = p.part_tok + row * g.G * N + n;
  float s = 0.f;
  for (int gi = 0; gi < g.G; ++gi) s += src[(int64_t)gi * N];
  void* dsts[6] = {p.dBc, p.dCc, p.dBf, p.dCf, p.dBr, p.dCr};
  reinterpret_cast<TO*>(dsts[tensor])[bt * N + n] = to_out<TO>(s);
}

template <int N>
__global__ void __launch_bounds__(256) k_reduce_par(const BwdParams p) {
  const Geo& g = p.g;
  const int64_t U = g.Bt * g.nc;
  const int64_t DN = g.D * N;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx < DN) {
    float sf = 0.f, sc = 0.f, sr = 0.f;
    for (int64_t u = 0; u < U; ++u) {
      sf += p.part_A[(0 * U + u) * DN + idx];
      sr += p.part_A[(1 * U + u) * DN + idx];
      sc += p.part_A[(2 * U + u) * DN + idx];
    }
    p.dAf[idx] = sf + sc;
    p.dAr[idx] = sr;
  } else if (idx < DN + g.D) {
    const int64_t d = idx - DN;
    float sn = 0.f, sc = 0.f;
    for (int64_t u = 0; u < U; ++u) {
      sn += p.part_D[(0 * U + u) * g.D + d];
      sc += p.part_D[(1 * U + u) * g.D + d];
    }
    p.dDf[d] = sn + sc;
    p.dDr[d] = sn;
  }
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
namespace {

// Dynamic shared memory is padded so that no more CTAs share an SM than its
// 512 TMEM columns can hold at once.
inline size_t pad_for_tmem(size_t smem, int TS, int N) {
  const uint32_t cols = tcols_host(TS, N);
  const int ctas = (int)(512 / cols);
  const size_t cap = (size_t)(220 * 1024) / (size_t)ctas;
  size_t need = cap > 2048 ? cap - 2048 : cap;
  if (ctas >= 16) need = 0;  // thread limit already bounds residency
  return smem > need ? smem : need;
}

template <typename T, typename TO, int N>
cudaError_t bwd_noisy_t(const BwdParams& p, cudaStream_t s) {
  const int Bs = (int)p.g.Bs, TS = Bs < 16 ? Bs : 16;
  const size_t smem = pad_for_tmem(NoisyBwdSmem<T, N>::bytes(TS, Bs), TS, N);
  cudaError_t e = cudaFuncSetAttribute(k_bwd_noisy<T, TO, N>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)p.g.G, (unsigned)p.g.nc, (unsigned)p.g.Bt);
  k_bwd_noisy<T, TO, N><<<grid, kCta, smem, s>>>(p);
  return cudaGetLastError();
}

template <typename T, typename TO, int N>
cudaError_t bwd_clean_t(const BwdParams& p, cudaStream_t s) {
  const int Bs = (int)p.g.Bs, TS = Bs < 16 ? Bs : 16;
  const size_t smem = pad_for_tmem(CleanBwdSmem<T, N>::bytes(TS, Bs), TS, N);
  cudaError_t e = cudaFuncSetAttribute(k_bwd_clean<T, TO, N>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)p.g.G, (unsigned)p.g.nc, (unsigned)p.g.Bt);
  k_bwd_clean<T, TO, N><<<grid, kCta, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

#define BDS_DISPATCH_N(N, ...)                      \
  switch (N) {                                      \
    case 8: { constexpr int NN = 8; __VA_ARGS__ }   \
    case 16: { constexpr int NN = 16; __VA_ARGS__ } \
    default: return cudaErrorInvalidValue;          \
  }

cudaError_t launch_bwd_noisy(int dt, int N, const BwdParams& p, cudaStream_t s) {
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return bwd_noisy_t<float, float, NN>(p, s);)
    case 1: BDS_DISPATCH_N(N, return bwd_noisy_t<bf16, bf16, NN>(p, s);)
    default: BDS_DISPATCH_N(N, return bwd_noisy_t<bf16, float, NN>(p, s);)
  }
}

cudaError_t launch_bwd_carry(int N, const BwdParams& p, cudaStream_t s) {
  const int64_t total = p.g.Bt * p.g.D * N;
  if (total == 0) return cudaSuccess;
  BDS_DISPATCH_N(N, k_bwd_carry<NN><<<(unsigned)((total + 255) / 256), 256, 0, s>>>(p); return cudaGetLastError();)
}

cudaError_t launch_bwd_clean(int dt, int N, const BwdParams& p, cudaStream_t s) {
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return bwd_clean_t<float, float, NN>(p, s);)
    case 1: BDS_DISPATCH_N(N, return bwd_clean_t<bf16, bf16, NN>(p, s);)
    default: BDS_DISPATCH_N(N, return bwd_clean_t<bf16, float, NN>(p, s);)
  }
}

cudaError_t launch_bwd_reduce_tok(int dt, int N, const BwdParams& p, cudaStream_t s) {
  const int64_t ntok = 6 * p.g.Bt * p.g.L * N;
  if (ntok == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)((ntok + 255) / 256);
  if (dt == 1) {
    BDS_DISPATCH_N(N, k_reduce_tok<bf16, NN><<<blocks, 256, 0, s>>>(p); return cudaGetLastError();)
  }
  BDS_DISPATCH_N(N, k_reduce_tok<float, NN><<<blocks, 256, 0, s>>>(p); return cudaGetLastError();)
}

cudaError_t launch_bwd_reduce_par(int N, const BwdParams& p, cudaStream_t s) {
  const int64_t npar = p.g.D * N + p.g.D;
  BDS_DISPATCH_N(N, k_reduce_par<NN><<<(unsigned)((npar + 255) / 256), 256, 0, s>>>(p); return cudaGetLastError();)
}

size_t bwd_noisy_smem(int dt, int N, int64_t Bs) {
  const int TS = Bs < 16 ? (int)Bs : 16;
  if (dt == 0) return N == 8 ? NoisyBwdSmem<float, 8>::bytes(TS, (int)Bs) : NoisyBwdSmem<float, 16>::bytes(TS, (int)Bs);
  return N == 8 ? NoisyBwdSmem<bf16, 8>::bytes(TS, (int)Bs) : NoisyBwdSmem<bf16, 16>::bytes(TS, (int)Bs);
}

size_t bwd_clean_smem(int dt, int N, int64_t Bs) {
  const int TS = Bs < 16 ? (int)Bs : 16;
  if (dt == 0) return N == 8 ? CleanBwdSmem<float, 8>::bytes(TS, (int)Bs) : CleanBwdSmem<float, 16>::bytes(TS, (int)Bs);
  return N == 8 ? CleanBwdSmem<bf16, 8>::bytes(TS, (int)Bs) : CleanBwdSmem<bf16, 16>::bytes(TS, (int)Bs);
}

}  // namespace bds
