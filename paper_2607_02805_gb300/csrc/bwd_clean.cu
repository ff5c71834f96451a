// bwd_clean.cu -- the clean-stream backward of libbdscan (sm_103a); see
// bwd_common.cuh for the derivative and the kernel sequence.
#include "bwd_common.cuh"

namespace bds {

// ---------------------------------------------------------------------------
// Clean stream backward from the exact chunk carries
// ---------------------------------------------------------------------------
template <typename T, int N>
struct CleanBwdSmem {
  using St = Stage<T, N, 3, 2, 2, kBwdTS>;  // x_c, dt_c, dy_c; B_c, C_c
  // `bufs` staging buffers, as for the noisy kernel
  static __host__ __device__ size_t red_off(int bufs) { return align16(St::buf_bytes(kBwdTS) * bufs); }
  static __host__ __device__ size_t ck_off(int bufs) { return red_off(bufs) + (size_t)2 * kBwdTS * kRedRow * 4; }
  // checkpoints in shared memory up to kCkSmemMaxBs tokens, else in global memory
  static __host__ __device__ size_t slot_off(int bufs, int TS, int Bs) {
    return ck_off(bufs) + (Bs > kCkSmemMaxBs ? 0 : (size_t)(Bs / TS - 1) * N * kCta * 4);
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
  // debug build: the chunk's last token and the channel group lie inside the sizes
  if (!(dguard(kSiteBwdClean, b, g.Bt) && dguard(kSiteBwdClean, (int64_t)(k_hi + 1) * Bs - 1, g.L) &&
        dguard(kSiteBwdClean, d0, g.D)))
    return;

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
  float* ck = Bs > kCkSmemMaxBs
                  ? p.ck_clean + (((size_t)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x) *
                                     (size_t)(NSEG - 1) * N * kCta
                  : reinterpret_cast<float*>(smem + L::ck_off(bufs));
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

namespace {

template <typename T, typename TO, int N, bool TILED>
BwdLaunch clean_launch(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  return bwd_launch<CleanBwdSmem<T, N>>(k_bwd_clean<T, TO, N, TILED>, Bs, half_cols(TS, N), dev);
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

template <typename T, typename TO, int N>
int bwd_clean_per_sm_t(int Bs, int dev) {
  const int TS = Bs < 16 ? Bs : 16;
  if (Bs < kBwdTS)
    return resident_ctas(k_bwd_clean<T, TO, N, true>, clean_launch<T, TO, N, true>(Bs, dev).smem, half_cols(TS, N), dev);
  return resident_ctas(k_bwd_clean<T, TO, N, false>, clean_launch<T, TO, N, false>(Bs, dev).smem, half_cols(TS, N), dev);
}

}  // namespace

cudaError_t launch_bwd_clean(int dt, int N, const BwdParams& p, cudaStream_t s) {
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return bwd_clean_t<float, float, NN>(p, s);)
    case 1: BDS_DISPATCH_N(N, return bwd_clean_t<bf16, bf16, NN>(p, s);)
    default: BDS_DISPATCH_N(N, return bwd_clean_t<bf16, float, NN>(p, s);)
  }
}

int bwd_clean_per_sm(int dt, int N, int Bs, int dev) {
  if (dt == 0) return N == 8 ? bwd_clean_per_sm_t<float, float, 8>(Bs, dev) : bwd_clean_per_sm_t<float, float, 16>(Bs, dev);
  if (dt == 1) return N == 8 ? bwd_clean_per_sm_t<bf16, bf16, 8>(Bs, dev) : bwd_clean_per_sm_t<bf16, bf16, 16>(Bs, dev);
  return N == 8 ? bwd_clean_per_sm_t<bf16, float, 8>(Bs, dev) : bwd_clean_per_sm_t<bf16, float, 16>(Bs, dev);
}

}  // namespace bds
