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
// Noisy blocks (both directions) + the clean stream's chunk-local adjoint
// ---------------------------------------------------------------------------
template <typename T, int N>
struct NoisyBwdSmem {
  // token-by-channel: x_n, dt_f, dt_r, dy_n, dt_c, dy_c; token-by-state: B_f, C_f, B_r, C_r, C_c
  using St = Stage<T, N, 6, 5, 2, kBwdTS>;
  // `bufs` staging buffers: 2 for one-segment blocks (the next block is
  // copied while the current one is used); for longer blocks one per segment
  // (the whole block resident) or 1 (each segment copied when needed)
  static __host__ __device__ size_t dx_off(int bufs) { return align16(St::buf_bytes(kBwdTS) * bufs); }
  // dx partials of a tile (several short blocks) or of one long block
  static __host__ __device__ size_t red_off(int bufs, int Bs) { return dx_off(bufs) + (size_t)(Bs < kBwdTS ? kBwdTS : Bs) * kCta * 4; }
  // red slots: both directions of a tile at once for short blocks, one
  // direction's segment at a time otherwise
  static __host__ __device__ int red_slots(int Bs) { return Bs < kBwdTS ? 4 : 2; }
  static __host__ __device__ size_t ck_off(int bufs, int Bs) { return red_off(bufs, Bs) + (size_t)red_slots(Bs) * kBwdTS * kRedRow * 4; }
  static __host__ __device__ size_t slot_off(int bufs, int TS, int Bs) {
    return ck_off(bufs, Bs) + (size_t)(Bs / TS - 1) * N * kCta * 4;
  }
  static __host__ __device__ size_t bytes(int bufs, int TS, int Bs) { return slot_off(bufs, TS, Bs) + 16; }
};

// TILED (blocks shorter than kBwdTS tokens): several blocks per staged tile.
template <typename T, typename TO, int N, bool TILED>
__global__ void __launch_bounds__(kCta, 1) k_bwd_noisy(const BwdParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  using L = NoisyBwdSmem<T, N>;
  const Geo& g = p.g;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int sw = swz_of_lane<N>();
  const int64_t b = blockIdx.z;
  const int c = blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + tid;
  const bool act = d < g.D;
  const int Bs = (int)g.Bs, TS = Bs < 16 ? Bs : 16, NSEG = Bs / TS;
  const int k_lo = chunk_lo(g, c), k_hi = chunk_lo(g, c + 1) - 1;

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
  const bool resident = NSEG > 1 && p.seg_resident;
  const int bufs = NSEG == 1 ? 2 : (resident ? NSEG : 1);
  float* dxbuf = reinterpret_cast<float*>(smem + L::dx_off(bufs));
  float* red = reinterpret_cast<float*>(smem + L::red_off(bufs, Bs));
  float* mine = red_slot<N>(red);
  float* ck = reinterpret_cast<float*>(smem + L::ck_off(bufs, Bs));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + L::slot_off(bufs, TS, Bs));

  const uint32_t tcols = full_cols(TS, N);
  if (warp == 0) tmem_alloc(tslot, tcols);
  tmem_sync();
  const uint32_t tbase = *tslot;
  const uint32_t tb = tbase + ((uint32_t)(warp * 32) << 16);

  float2 A2f[N / 2], A2r[N / 2];
  vzero2<N>(A2f);
  vzero2<N>(A2r);
  float Dsum = 0.f;
  if (act) {
    vload2<N>(A2f, p.Af + d * N, sw);
    vload2<N>(A2r, p.Ar + d * N, sw);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      A2f[j] = mul2(A2f[j], f2(kLog2e));
      A2r[j] = mul2(A2r[j], f2(kLog2e));
    }
    Dsum = __fadd_rn(p.Df[d], p.Dr[d]);
  }
  float2 dAf[N / 2], dAr[N / 2];
  vzero2<N>(dAf);
  vzero2<N>(dAr);
  float dDn = 0.f, sdt = 0.f;
  float2 carry[N / 2];  // clean stream: a_{t+1} gbar_{t+1} (+ injections) entering token t from the right
  vzero2<N>(carry);
  float2 dSn[N / 2];  // seed gradient of the block to the right of the current one
  vzero2<N>(dSn);

  // everything for block k, whose tokens start at `off` in the staged tile
  auto block = [&](int k, int off) {
    const int64_t t0 = (int64_t)k * Bs;
    const int64_t row0 = b * g.L + t0;
    // make segment s current: staged now, or already resident
    auto stage_seg = [&](int s) {
      if (resident)
        st.select(s);
      else
        st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
    };

    // ---- clean stream: chunk-local adjoint over block k ----
    if (k < k_hi) {
#pragma unroll
      for (int j = 0; j < N / 2; ++j) carry[j] = add2(carry[j], dSn[j]);
      if (p.dstates != nullptr && act) {
        float2 e[N / 2];
        vload2<N>(e, p.dstates + ((b * g.nb + k) * g.D + d) * N, sw);
#pragma unroll
        for (int j = 0; j < N / 2; ++j) carry[j] = add2(carry[j], e[j]);
      }
    }
    for (int s = NSEG - 1; s >= 0; --s) {
      if (NSEG > 1) stage_seg(s);
#pragma unroll 4
      for (int i = TS - 1; i >= 0; --i) {
        const float dt = st.at(DTC, off + i), dy = st.at(DYC, off + i);
        const float2 dt2 = f2(dt), dy2 = f2(dy);
        float2 C[N / 2];
        vload2<N>(C, st.row(CC, off + i), sw);
#pragma unroll
        for (int j = 0; j < N / 2; ++j) carry[j] = mul2(ex2x2(mul2(dt2, A2f[j])), fma2(C[j], dy2, carry[j]));
        sdt = __fadd_rn(sdt, dt);
      }
    }

    // ---- noisy block k, reverse direction (zero state at the block end) ----
    {
      if (NSEG > 1) {
        float2 h[N / 2];
        vzero2<N>(h);
        for (int s = NSEG - 1; s >= 1; --s) {
          stage_seg(s);
#pragma unroll 4
          for (int i = TS - 1; i >= 0; --i) scan_state_swz<N>(h, A2r, st.at(DTR, i), st.at(XN, i), st.row(BR, i), sw);
          ck_store<N>(ck, s - 1, h);
        }
      }
      float2 gr[N / 2];  // a_{t-1} gbar_{t-1}, entering token t from the left
      vzero2<N>(gr);
      for (int s = 0; s < NSEG; ++s) {
        if (NSEG > 1) stage_seg(s);
        float2 h[N / 2];
        if (s == NSEG - 1)
          vzero2<N>(h);
        else
          ck_load<N>(h, ck, s);
        seg_bwd<N, false>(st, TS, XN, DTR, DYN, BR, CR, A2r, sw, h, gr, dAr, tb, mine, off, 0,
                          [&](int i, float dt, float x, float dy, float sgB, float sAq) {
                            const int ib = s * TS + i;
                            if (act)
                              reinterpret_cast<TO*>(p.ddtr)[(row0 + ib) * g.D + d] =
                                  to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
                            dxbuf[(off + ib) * kCta + tid] = __fmul_rn(dt, sgB);
                          });
        if (!TILED) red_flush<N>(p, red, 0, 1, 4, 5, b, t0 + (int64_t)s * TS, TS);
      }
    }

    // ---- noisy block k, forward direction (seeded with states[k-1]) ----
    {
      float2 seed[N / 2];
      vzero2<N>(seed);
      if (k > 0 && act) vload2<N>(seed, p.states + ((b * g.nb + (k - 1)) * g.D + d) * N, sw);
      if (NSEG > 1) {
        float2 h[N / 2];
#pragma unroll
        for (int j = 0; j < N / 2; ++j) h[j] = seed[j];
        for (int s = 0; s < NSEG - 1; ++s) {
          stage_seg(s);
#pragma unroll 4
          for (int i = 0; i < TS; ++i) scan_state_swz<N>(h, A2f, st.at(DTF, i), st.at(XN, i), st.row(BF, i), sw);
          ck_store<N>(ck, s, h);
        }
      }
      float2 gf[N / 2];  // a_{t+1} gbar_{t+1}, entering token t from the right
      vzero2<N>(gf);
      for (int s = NSEG - 1; s >= 0; --s) {
        if (NSEG > 1) stage_seg(s);
        float2 h[N / 2];
        if (s == 0) {
#pragma unroll
          for (int j = 0; j < N / 2; ++j) h[j] = seed[j];
        } else {
          ck_load<N>(h, ck, s - 1);
        }
        seg_bwd<N, true>(st, TS, XN, DTF, DYN, BF, CF, A2f, sw, h, gf, dAf, tb, mine, off, TILED ? 2 : 0,
                         [&](int i, float dt, float x, float dy, float sgB, float sAq) {
                           const int ib = s * TS + i;
                           const int64_t o = (row0 + ib) * g.D + d;
                           if (act) {
                             reinterpret_cast<TO*>(p.ddtf)[o] = to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
                             const float dxv =
                                 __fmaf_rn(Dsum, dy, __fadd_rn(dxbuf[(off + ib) * kCta + tid], __fmul_rn(dt, sgB)));
                             reinterpret_cast<TO*>(p.dxn)[o] = to_out<TO>(dxv);
                           }
                           dDn = __fmaf_rn(dy, x, dDn);
                         });
        if (!TILED) red_flush<N>(p, red, 0, 1, 2, 3, b, t0 + (int64_t)s * TS, TS);
      }
      // gradient of this block's seed, states[k-1]: a_{t0} gbar_{t0}
#pragma unroll
      for (int j = 0; j < N / 2; ++j) dSn[j] = gf[j];
      if (k > 0 && act) vstore2<N>(p.dS + ((b * g.nb + (k - 1)) * g.D + d) * N, gf, sw);
    }
  };

  if (TILED) {
    // Short blocks are staged in tiles of TB blocks (at most kBwdTS tokens),
    // the next tile copied while the current one is used, and the dB/dC
    // partials of a tile are flushed once for both directions.
    const int TB = kBwdTS / Bs;
    auto tile_lo = [&](int hi) { return hi - TB + 1 > k_lo ? hi - TB + 1 : k_lo; };
    st.issue(0, b * g.L + (int64_t)tile_lo(k_hi) * Bs, (k_hi - tile_lo(k_hi) + 1) * Bs, g.D, d0);
    int tile = 0;
    for (int kt_hi = k_hi; kt_hi >= k_lo; ++tile) {
      const int kt_lo = tile_lo(kt_hi), nbk = kt_hi - kt_lo + 1;
      const int buf = tile & 1;
      __syncthreads();  // the other buffer is no longer read
      if (kt_lo > k_lo) {
        const int nhi = kt_lo - 1, nlo = tile_lo(nhi);
        st.issue(buf ^ 1, b * g.L + (int64_t)nlo * Bs, (nhi - nlo + 1) * Bs, g.D, d0);
      }
      st.complete(buf, nbk * Bs, kt_lo > k_lo ? 1 : 0);
      for (int k = kt_hi; k >= kt_lo; --k) block(k, (k - kt_lo) * Bs);
      const int64_t ts0 = (int64_t)kt_lo * Bs;  // the tile's dB/dC partials, both directions
      red_flush<N>(p, red, 0, 1, 4, 5, b, ts0, nbk * Bs);
      red_flush<N>(p, red, 2, 3, 2, 3, b, ts0, nbk * Bs);
      kt_hi = kt_lo - 1;
    }
  } else {
    // one-segment blocks: block k-1 is copied while block k is processed
    if (NSEG == 1) st.issue(0, b * g.L + (int64_t)k_hi * Bs, TS, g.D, d0);
    for (int k = k_hi; k >= k_lo; --k) {
      const int64_t row0 = b * g.L + (int64_t)k * Bs;
      if (NSEG == 1) {
        const int buf = (k_hi - k) & 1;
        __syncthreads();  // the other buffer is no longer read
        if (k > k_lo) st.issue(buf ^ 1, row0 - Bs, TS, g.D, d0);
        st.complete(buf, TS, k > k_lo ? 1 : 0);
      } else if (resident) {  // every segment of the block, once
        __syncthreads();  // the previous block is no longer read
        for (int s = 0; s < NSEG; ++s) st.issue(s, row0 + (int64_t)s * TS, TS, g.D, d0);
        for (int s = 0; s < NSEG; ++s) st.complete(s, TS, 0);
      }
      block(k, 0);
    }
  }

  if (act) {
    vstore2<N>(p.Lc + ((b * g.nc + c) * g.D + d) * N, carry, sw);
    p.sdtc[(b * g.nc + c) * g.D + d] = sdt;
    const int64_t u = b * g.nc + c, U = g.Bt * g.nc;
    vstore2<N>(p.part_A + ((0 * U + u) * g.D + d) * N, dAf, sw);
    vstore2<N>(p.part_A + ((1 * U + u) * g.D + d) * N, dAr, sw);
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
  const float* dS = p.dS + (b * g.nb * g.D + d) * N + n;  // block k at [k * D * N]
  const float* ext = p.dstates != nullptr ? p.dstates + (b * g.nb * g.D + d) * N + n : nullptr;
  float* Lc = p.Lc + (b * g.nc * g.D + d) * N + n;        // chunk c at [c * D * N]
  const float* sdtc = p.sdtc + b * g.nc * g.D + d;         // chunk c at [c * D]
  const int64_t DN = g.D * N;
  // chunk_lo(c) = floor(c nb / nc), stepped down from c = nc by quotient and
  // remainder (no division per chunk)
  const int q0 = (int)(g.nb / g.nc), r0 = (int)(g.nb % g.nc);
  int lo = (int)g.nb, rem = 0;  // chunk_lo(c0 + 1) and its remainder
  float G = 0.f;  // a_{t+1} gbar_{t+1} entering the current chunk's last token from the right
  constexpr int U = 8;
  for (int c0 = g.nc - 1; c0 >= 0; c0 -= U) {
    // loads of up to U chunks first (they do not depend on the carry)
    float inj[U], loc[U], sd[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int c = c0 - j;
      const int kl = lo - 1;  // last block of chunk c
      lo -= q0;
      rem -= r0;
      if (rem < 0) {
        rem += (int)g.nc;
        lo -= 1;
      }
      const int cc = c >= 0 ? c : 0;
      const int64_t kk = c >= 0 ? kl : 0;
      const float vS = dS[kk * DN], vE = ext != nullptr ? ext[kk * DN] : 0.f;
      inj[j] = c >= 0 && kl + 1 < g.nb ? vS : 0.f;
      if (ext != nullptr) inj[j] = __fadd_rn(inj[j], c >= 0 ? vE : 0.f);
      loc[j] = Lc[cc * DN];
      sd[j] = sdtc[(int64_t)cc * g.D];
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const int c = c0 - j;
      if (c < 0) break;
      const float gin = __fadd_rn(G, inj[j]);
      Lc[c * DN] = gin;
      G = __fmaf_rn(ex2(__fmul_rn(A2, sd[j])), gin, loc[j]);
    }
  }
}

// ---------------------------------------------------------------------------
// Clean stream backward from the exact chunk carries
// ---------------------------------------------------------------------------
template <typename T, int N>
struct CleanBwdSmem {
  using St = Stage<T, N, 3, 2, 2, kBwdTS>;  // x_c, dt_c, dy_c; B_c, C_c
  // `bufs` staging buffers, as for the noisy kernel
  static __host__ __device__ size_t red_off(int bufs) { return align16(St::buf_bytes(kBwdTS) * bufs); }
  static __host__ __device__ size_t ck_off(int bufs) { return red_off(bufs) + (size_t)2 * kBwdTS * kRedRow * 4; }
  static __host__ __device__ size_t slot_off(int bufs, int TS, int Bs) {
    return ck_off(bufs) + (size_t)(Bs / TS - 1) * N * kCta * 4;
  }
  // one-segment blocks: the seeds of the current and the next block
  static __host__ __device__ size_t seed_off(int bufs, int TS, int Bs) { return slot_off(bufs, TS, Bs) + 16; }
  static __host__ __device__ size_t bytes(int bufs, int TS, int Bs) {
    return seed_off(bufs, TS, Bs) + (Bs / TS == 1 ? (size_t)2 * kCta * N * 4 : 0);
  }
};

template <typename T, typename TO, int N, bool TILED>
__global__ void __launch_bounds__(kCta, 3) k_bwd_clean(const BwdParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  using L = CleanBwdSmem<T, N>;
  const Geo& g = p.g;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int sw = swz_of_lane<N>();
  const int64_t b = blockIdx.z;
  const int c = blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + tid;
  const bool act = d < g.D;
  const int Bs = (int)g.Bs, TS = Bs < 16 ? Bs : 16, NSEG = Bs / TS;
  const int k_lo = chunk_lo(g, c), k_hi = chunk_lo(g, c + 1) - 1;

  enum { XC = 0, DTC = 1, DYC = 2 };
  enum { BC = 0, CC = 1 };
  typename L::St st;
  st.carve(smem, TS);
  st.td_src[XC] = (const T*)p.xc;
  st.td_src[DTC] = (const T*)p.dtc;
  st.td_src[DYC] = (const T*)p.dyc;
  st.row_src[BC] = (const T*)p.Bc;
  st.row_src[CC] = (const T*)p.Cc;
  const bool resident = NSEG > 1 && p.seg_resident;
  const int bufs = NSEG == 1 ? 2 : (resident ? NSEG : 1);
  float* red = reinterpret_cast<float*>(smem + L::red_off(bufs));
  float* mine = red_slot<N>(red);
  float* ck = reinterpret_cast<float*>(smem + L::ck_off(bufs));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + L::slot_off(bufs, TS, Bs));
  float* seedb = reinterpret_cast<float*>(smem + L::seed_off(bufs, TS, Bs));  // [2][kCta][N]

  const uint32_t tcols = half_cols(TS, N);  // held states of a segment
  if (warp == 0) tmem_alloc(tslot, tcols);
  tmem_sync();
  const uint32_t tbase = *tslot;
  const uint32_t tb = tbase + ((uint32_t)(warp * 32) << 16);

  float2 A2[N / 2];
  vzero2<N>(A2);
  float Df = 0.f;
  if (act) {
    vload2<N>(A2, p.Af + d * N, sw);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) A2[j] = mul2(A2[j], f2(kLog2e));
    Df = p.Df[d];
  }
  float2 dA[N / 2];
  vzero2<N>(dA);
  float dDc = 0.f;
  float2 gc[N / 2];  // a_{t+1} gbar_{t+1} (+ injections) entering token t from the right
  vzero2<N>(gc);

  // everything for block k, whose tokens start at `off` in the staged tile;
  // seed_staged: its seed is in seedb[buf]
  auto block = [&](int k, int off, int buf, bool seed_staged) {
    const int64_t t0 = (int64_t)k * Bs;
    const int64_t row0 = b * g.L + t0;
    // make segment s current: staged now, or already resident
    auto stage_seg = [&](int s) {
      if (resident)
        st.select(s);
      else
        st.load(row0 + (int64_t)s * TS, TS, g.D, d0);
    };
    if (k == k_hi) {
      if (act) vload2<N>(gc, p.Lc + ((b * g.nc + c) * g.D + d) * N, sw);
    } else if (act) {
      float2 e[N / 2];
      vload2<N>(e, p.dS + ((b * g.nb + k) * g.D + d) * N, sw);
#pragma unroll
      for (int j = 0; j < N / 2; ++j) gc[j] = add2(gc[j], e[j]);
      if (p.dstates != nullptr) {
        vload2<N>(e, p.dstates + ((b * g.nb + k) * g.D + d) * N, sw);
#pragma unroll
        for (int j = 0; j < N / 2; ++j) gc[j] = add2(gc[j], e[j]);
      }
    }
    float2 seed[N / 2];
    vzero2<N>(seed);
    if (seed_staged)
        vload2<N>(seed, seedb + (buf * kCta + tid) * N, sw);  // staged with the tile
      else if (NSEG == 1 && k > 0 && act)
        vload2<N>(seed, p.states + ((b * g.nb + (k - 1)) * g.D + d) * N, sw);
      else if (k > 0 && act)
        vload2<N>(seed, p.states + ((b * g.nb + (k - 1)) * g.D + d) * N, sw);
    if (NSEG > 1) {
      float2 h[N / 2];
#pragma unroll
      for (int j = 0; j < N / 2; ++j) h[j] = seed[j];
      for (int s = 0; s < NSEG - 1; ++s) {
        stage_seg(s);
#pragma unroll 4
        for (int i = 0; i < TS; ++i) scan_state_swz<N>(h, A2, st.at(DTC, i), st.at(XC, i), st.row(BC, i), sw);
        ck_store<N>(ck, s, h);
      }
    }
    for (int s = NSEG - 1; s >= 0; --s) {
      if (NSEG > 1) stage_seg(s);
      float2 h[N / 2];
      if (s == 0) {
#pragma unroll
        for (int j = 0; j < N / 2; ++j) h[j] = seed[j];
      } else {
        ck_load<N>(h, ck, s - 1);
      }
      seg_bwd_half<N, true>(st, TS, XC, DTC, DYC, BC, CC, A2, sw, h, gc, dA, tb, mine, off, 0,
                       [&](int i, float dt, float x, float dy, float sgB, float sAq) {
                         const int64_t o = (row0 + s * TS + i) * g.D + d;
                         if (act) {
                           reinterpret_cast<TO*>(p.ddtc)[o] = to_out<TO>(__fmaf_rn(x, sgB, __fmul_rn(kLn2, sAq)));
                           reinterpret_cast<TO*>(p.dxc)[o] = to_out<TO>(__fmaf_rn(Df, dy, __fmul_rn(dt, sgB)));
                         }
                         dDc = __fmaf_rn(dy, x, dDc);
                       });
      if (!TILED) red_flush<N>(p, red, 0, 1, 0, 1, b, t0 + (int64_t)s * TS, TS);
    }
  };

  if (TILED) {
    // Short blocks are staged in tiles of TB blocks (at most kBwdTS tokens)
    // together with the seed of the tile's last block, the next tile copied
    // while the current one is used, and the dB/dC partials of a tile are
    // flushed once.
    const int TB = kBwdTS / Bs;
    auto tile_lo = [&](int hi) { return hi - TB + 1 > k_lo ? hi - TB + 1 : k_lo; };
    issue_seed<N>(seedb, p.states, g, b, k_hi, d0);  // same cp.async group as the tile
    st.issue(0, b * g.L + (int64_t)tile_lo(k_hi) * Bs, (k_hi - tile_lo(k_hi) + 1) * Bs, g.D, d0);
    int tile = 0;
    for (int kt_hi = k_hi; kt_hi >= k_lo; ++tile) {
      const int kt_lo = tile_lo(kt_hi), nbk = kt_hi - kt_lo + 1;
      const int buf = tile & 1;
      __syncthreads();  // the other buffer is no longer read
      if (kt_lo > k_lo) {
        const int nhi = kt_lo - 1, nlo = tile_lo(nhi);
        issue_seed<N>(seedb + (buf ^ 1) * kCta * N, p.states, g, b, nhi, d0);
        st.issue(buf ^ 1, b * g.L + (int64_t)nlo * Bs, (nhi - nlo + 1) * Bs, g.D, d0);
      }
      st.complete(buf, nbk * Bs, kt_lo > k_lo ? 1 : 0);
      for (int k = kt_hi; k >= kt_lo; --k) block(k, (k - kt_lo) * Bs, buf, k == kt_hi);
      red_flush<N>(p, red, 0, 1, 0, 1, b, (int64_t)kt_lo * Bs, nbk * Bs);  // the tile's dB/dC
      kt_hi = kt_lo - 1;
    }
  } else {
    // one-segment blocks: block k-1 (and its seed) is copied while block k is processed
    if (NSEG == 1) {
      issue_seed<N>(seedb, p.states, g, b, k_hi, d0);  // same cp.async group as the block
      st.issue(0, b * g.L + (int64_t)k_hi * Bs, TS, g.D, d0);
    }
    for (int k = k_hi; k >= k_lo; --k) {
      const int64_t row0 = b * g.L + (int64_t)k * Bs;
      const int buf = (k_hi - k) & 1;
      if (NSEG == 1) {
        __syncthreads();  // the other buffer is no longer read
        if (k > k_lo) {
          issue_seed<N>(seedb + (buf ^ 1) * kCta * N, p.states, g, b, k - 1, d0);
          st.issue(buf ^ 1, row0 - Bs, TS, g.D, d0);
        }
        st.complete(buf, TS, k > k_lo ? 1 : 0);
      } else if (resident) {  // every segment of the block, once
        __syncthreads();  // the previous block is no longer read
        for (int s = 0; s < NSEG; ++s) st.issue(s, row0 + (int64_t)s * TS, TS, g.D, d0);
        for (int s = 0; s < NSEG; ++s) st.complete(s, TS, 0);
      }
      block(k, 0, buf, NSEG == 1);
    }
  }
  if (act) {
    const int64_t u = b * g.nc + c, U = g.Bt * g.nc;
    vstore2<N>(p.part_A + ((2 * U + u) * g.D + d) * N, dA, sw);
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
  void* dst = tensor == 0 ? p.dBc : tensor == 1 ? p.dCc : tensor == 2 ? p.dBf : tensor == 3 ? p.dCf
            : tensor == 4 ? p.dBr : p.dCr;
  reinterpret_cast<TO*>(dst)[bt * N + n] = to_out<TO>(s);
}

// One CTA sums 32 columns of the per-chunk partials: 8 slices of threads
// each add every 8th chunk (in order), then the slices are added in order.
template <int N>
__global__ void __launch_bounds__(256) k_reduce_par(const BwdParams p) {
  // 8 slices (warps) of the chunk partials; each lane sums 4 adjacent columns
  __shared__ float4 part[3][8][32];
  const Geo& g = p.g;
  const int64_t U = g.Bt * g.nc;
  const int64_t DN = g.D * N;
  const int lane = threadIdx.x & 31, slice = threadIdx.x >> 5;
  const int64_t col = ((int64_t)blockIdx.x * 32 + lane) * 4;  // D and D*N are multiples of 4
  float4 s0 = make_float4(0.f, 0.f, 0.f, 0.f), s1 = s0, s2 = s0;
  auto acc = [](float4& s, const float* src) {
    const float4 v = *reinterpret_cast<const float4*>(src);
    s.x += v.x;
    s.y += v.y;
    s.z += v.z;
    s.w += v.w;
  };
  if (col < DN) {
    const float* a0 = p.part_A + col;
    const float* a1 = p.part_A + U * DN + col;
    const float* a2 = p.part_A + 2 * U * DN + col;
#pragma unroll 4
    for (int64_t u = slice; u < U; u += 8) {
      acc(s0, a0 + u * DN);
      acc(s1, a1 + u * DN);
      acc(s2, a2 + u * DN);
    }
  } else if (col < DN + g.D) {
    const int64_t d = col - DN;
#pragma unroll 4
    for (int64_t u = slice; u < U; u += 8) {
      acc(s0, p.part_D + u * g.D + d);
      acc(s1, p.part_D + (U + u) * g.D + d);
    }
  }
  part[0][slice][lane] = s0;
  part[1][slice][lane] = s1;
  part[2][slice][lane] = s2;
  __syncthreads();
  if (slice == 0) {
    float4 t0 = part[0][0][lane], t1 = part[1][0][lane], t2 = part[2][0][lane];
#pragma unroll
    for (int k = 1; k < 8; ++k) {
      const float4 v0 = part[0][k][lane], v1 = part[1][k][lane], v2 = part[2][k][lane];
      t0 = make_float4(t0.x + v0.x, t0.y + v0.y, t0.z + v0.z, t0.w + v0.w);
      t1 = make_float4(t1.x + v1.x, t1.y + v1.y, t1.z + v1.z, t1.w + v1.w);
      t2 = make_float4(t2.x + v2.x, t2.y + v2.y, t2.z + v2.z, t2.w + v2.w);
    }
    if (col < DN) {
      // noisy forward direction + clean stream
      *reinterpret_cast<float4*>(p.dAf + col) = make_float4(t0.x + t2.x, t0.y + t2.y, t0.z + t2.z, t0.w + t2.w);
      *reinterpret_cast<float4*>(p.dAr + col) = t1;
    } else if (col < DN + g.D) {
      const int64_t d = col - DN;
      *reinterpret_cast<float4*>(p.dDf + d) = make_float4(t0.x + t1.x, t0.y + t1.y, t0.z + t1.z, t0.w + t1.w);  // noisy + clean
      *reinterpret_cast<float4*>(p.dDr + d) = t0;
    }
  }
}

// ---------------------------------------------------------------------------
// launchers
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
template <typename T, typename TO, int N, bool TILED>
BwdLaunch noisy_launch(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  return bwd_launch<NoisyBwdSmem<T, N>>(k_bwd_noisy<T, TO, N, TILED>, Bs, full_cols(TS, N), dev);
}
template <typename T, typename TO, int N, bool TILED>
BwdLaunch clean_launch(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  return bwd_launch<CleanBwdSmem<T, N>>(k_bwd_clean<T, TO, N, TILED>, Bs, half_cols(TS, N), dev);
}

template <typename T, typename TO, int N, bool TILED>
void bwd_per_sm_t(int Bs, int dev, int& noisy, int& clean) {
  const int TS = Bs < 16 ? Bs : 16;
  noisy = resident_ctas(k_bwd_noisy<T, TO, N, TILED>, noisy_launch<T, TO, N, TILED>(Bs, dev).smem,
                        full_cols(TS, N), dev);
  clean = resident_ctas(k_bwd_clean<T, TO, N, TILED>, clean_launch<T, TO, N, TILED>(Bs, dev).smem,
                        half_cols(TS, N), dev);
}
template <typename T, typename TO, int N>
void bwd_per_sm(int Bs, int dev, int& noisy, int& clean) {
  if (Bs < kBwdTS)
    bwd_per_sm_t<T, TO, N, true>(Bs, dev, noisy, clean);
  else
    bwd_per_sm_t<T, TO, N, false>(Bs, dev, noisy, clean);
}

template <typename T, typename TO, int N, bool TILED>
cudaError_t bwd_noisy_tt(const BwdParams& p_in, cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const BwdLaunch l = noisy_launch<T, TO, N, TILED>((int)p_in.g.Bs, dev);
  BwdParams p = p_in;
  p.seg_resident = l.resident;
  e = set_bwd_attrs(k_bwd_noisy<T, TO, N, TILED>, l.smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)p.g.G, (unsigned)p.g.nc, (unsigned)p.g.Bt);
  k_bwd_noisy<T, TO, N, TILED><<<grid, kCta, l.smem, s>>>(p);
  return cudaGetLastError();
}
template <typename T, typename TO, int N>
cudaError_t bwd_noisy_t(const BwdParams& p, cudaStream_t s) {
  return p.g.Bs < kBwdTS ? bwd_noisy_tt<T, TO, N, true>(p, s) : bwd_noisy_tt<T, TO, N, false>(p, s);
}

template <typename T, typename TO, int N, bool TILED>
cudaError_t bwd_clean_tt(const BwdParams& p_in, cudaStream_t s) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const BwdLaunch l = clean_launch<T, TO, N, TILED>((int)p_in.g.Bs, dev);
  BwdParams p = p_in;
  p.seg_resident = l.resident;
  e = set_bwd_attrs(k_bwd_clean<T, TO, N, TILED>, l.smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)p.g.G, (unsigned)p.g.nc, (unsigned)p.g.Bt);
  k_bwd_clean<T, TO, N, TILED><<<grid, kCta, l.smem, s>>>(p);
  return cudaGetLastError();
}
template <typename T, typename TO, int N>
cudaError_t bwd_clean_t(const BwdParams& p, cudaStream_t s) {
  return p.g.Bs < kBwdTS ? bwd_clean_tt<T, TO, N, true>(p, s) : bwd_clean_tt<T, TO, N, false>(p, s);
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
  const int64_t npar4 = (p.g.D * N + p.g.D) / 4;  // float4 columns
  BDS_DISPATCH_N(N, k_reduce_par<NN><<<(unsigned)((npar4 + 31) / 32), 256, 0, s>>>(p); return cudaGetLastError();)
}

// Backward chunks per batch row, between 1 and bwd_max_chunks(); both
// backward kernels use the same chunks. For each count, each kernel's time is
// modelled as (waves of CTAs over its resident slots) x (blocks in the longest
// chunk + a set-up of a quarter block) x (its work per block) x (CTAs sharing
// an SM): per token the noisy kernel makes five scan passes and four channel
// reductions, the clean kernel two and two. The count with the least modelled
// sum is taken. Falls back to the forward chunking if the attribute queries
// fail.
int bwd_chunk_count(int dt, int N, const Geo& g) {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return g.nc;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return g.nc;
  const int Bs = (int)g.Bs;
  int pn = 0, pc = 0;
  if (dt == 0) {
    if (N == 8) bwd_per_sm<float, float, 8>(Bs, dev, pn, pc); else bwd_per_sm<float, float, 16>(Bs, dev, pn, pc);
  } else if (dt == 1) {
    if (N == 8) bwd_per_sm<bf16, bf16, 8>(Bs, dev, pn, pc); else bwd_per_sm<bf16, bf16, 16>(Bs, dev, pn, pc);
  } else {
    if (N == 8) bwd_per_sm<bf16, float, 8>(Bs, dev, pn, pc); else bwd_per_sm<bf16, float, 16>(Bs, dev, pn, pc);
  }
  if (pn <= 0 || pc <= 0) return g.nc;
  constexpr double kNoisyWork = 9.0, kCleanWork = 4.0;  // scan passes + reductions per token
  const int64_t rows = g.Bt * g.G;
  const int cmax = bwd_max_chunks(g);
  int best = g.nc;
  double best_cost = 1e300;
  for (int nc = 1; nc <= cmax; ++nc) {
    const double blocks = (double)((g.nb + nc - 1) / nc) + 0.25;  // longest chunk + set-up
    const double wn = (double)((rows * nc + (int64_t)pn * sms - 1) / ((int64_t)pn * sms));
    const double wc = (double)((rows * nc + (int64_t)pc * sms - 1) / ((int64_t)pc * sms));
    const double cost = blocks * (wn * kNoisyWork * pn + wc * kCleanWork * pc);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = nc;
    }
  }
  return best;
}

}  // namespace bds
