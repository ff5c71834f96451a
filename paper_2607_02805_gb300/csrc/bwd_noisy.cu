// bwd_noisy.cu -- the noisy-block backward of libbdscan (sm_103a); see
// bwd_common.cuh for the derivative and the kernel sequence.
#include "bwd_common.cuh"

namespace bds {

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
  // checkpoints in shared memory up to kCkSmemMaxBs tokens, else in global memory
  static __host__ __device__ size_t slot_off(int bufs, int TS, int Bs) {
    return ck_off(bufs, Bs) + (Bs > kCkSmemMaxBs ? 0 : (size_t)(Bs / TS - 1) * N * kCta * 4);
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
  // debug build: the chunk's last token and the channel group lie inside the sizes
  if (!(dguard(kSiteBwdNoisy, b, g.Bt) && dguard(kSiteBwdNoisy, (int64_t)(k_hi + 1) * Bs - 1, g.L) &&
        dguard(kSiteBwdNoisy, d0, g.D)))
    return;

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
  float* ck = Bs > kCkSmemMaxBs
                  ? p.ck_noisy + (((size_t)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x) *
                                     (size_t)(NSEG - 1) * N * kCta
                  : reinterpret_cast<float*>(smem + L::ck_off(bufs, Bs));
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

namespace {

template <typename T, typename TO, int N, bool TILED>
BwdLaunch noisy_launch(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  return bwd_launch<NoisyBwdSmem<T, N>>(k_bwd_noisy<T, TO, N, TILED>, Bs, full_cols(TS, N), dev);
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

template <typename T, typename TO, int N>
int bwd_noisy_per_sm_t(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  if (Bs < kBwdTS)
    return resident_ctas(k_bwd_noisy<T, TO, N, true>, noisy_launch<T, TO, N, true>(Bs, dev).smem, full_cols(TS, N), dev);
  return resident_ctas(k_bwd_noisy<T, TO, N, false>, noisy_launch<T, TO, N, false>(Bs, dev).smem, full_cols(TS, N), dev);
}

}  // namespace

cudaError_t launch_bwd_noisy(int dt, int N, const BwdParams& p, cudaStream_t s) {
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return bwd_noisy_t<float, float, NN>(p, s);)
    case 1: BDS_DISPATCH_N(N, return bwd_noisy_t<bf16, bf16, NN>(p, s);)
    default: BDS_DISPATCH_N(N, return bwd_noisy_t<bf16, float, NN>(p, s);)
  }
}

int bwd_noisy_per_sm(int dt, int N, int Bs, int dev) {
  if (dt == 0) return N == 8 ? bwd_noisy_per_sm_t<float, float, 8>(Bs, dev) : bwd_noisy_per_sm_t<float, float, 16>(Bs, dev);
  if (dt == 1) return N == 8 ? bwd_noisy_per_sm_t<bf16, bf16, 8>(Bs, dev) : bwd_noisy_per_sm_t<bf16, bf16, 16>(Bs, dev);
  return N == 8 ? bwd_noisy_per_sm_t<bf16, float, 8>(Bs, dev) : bwd_noisy_per_sm_t<bf16, float, 16>(Bs, dev);
}

}  // namespace bds
