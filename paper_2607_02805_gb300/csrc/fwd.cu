// fwd.cu -- forward-side kernels of libbdscan (sm_103a).
//
// The clean prefix scan (eq. boundary-state) is split into time chunks of
// m blocks (m = max(1, 128 / Bs)) so that Bt * D channels are not the only
// source of parallelism:
//   k_chunk_local  each (batch, chunk, 128 channels): scan the chunk from a
//                  zero state; keep the end state and the sum of dt.
//   k_chunk_carry  each (batch, channel, state): walk the chunks in order,
//                  H_{c+1} = exp(A * sum_c dt) * H_c + local_c, giving the
//                  exact state at every chunk start.
//   k_block_scan   each (batch, chunk, 128 channels): rescan the chunk from
//                  its start state, emitting y_c and the state at every
//                  block end; for every noisy block of the chunk, continue
//                  the state at its start through the noisy tokens (forward
//                  direction, eq. partial-reverse first line) and run the
//                  block-local reverse scan from zero (second line), and
//                  write their sum (third line).
//   k_active_block each (batch, 32 channels): one noisy block from a cached
//                  seed (the inference step), forward and reverse scans in
//                  two warps at once.
// The state at the end of a chunk's last block is taken from the carry
// kernel (the same value the next chunk starts from), so every consumer of
// a boundary state sees one value, and boundary states of a prefix equal
// those of any longer stream: chunking depends on Bs only.
#include "device.cuh"
#include "params.h"

namespace bds {

static_assert(kCta == kCtaHost, "host and device CTA widths differ");

constexpr int kLocalSpan = 32;  // tokens staged per step of the chunk-local scan
// Tokens the block scan stages at once: longer blocks are staged in segments
// of this many tokens (shared memory, and so residency, stays that of a
// 16-token block).
constexpr int kScanSeg = 16;

// REV: the scan runs right to left in time (logical token t is row L-1-t).
template <typename T, int N, bool REV>
__global__ void __launch_bounds__(kCta) k_chunk_local(const FwdParams p) {
  extern __shared__ __align__(16) unsigned char smem[];
  const Geo& g = p.g;
  const int64_t b = blockIdx.z;
  const int c = blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + threadIdx.x;
  const bool act = d < g.D;
  {  // debug build: the chunk's tokens, channels and state slot lie inside the sizes
    const int64_t tc = (int64_t)g.m * g.Bs, dl = (d0 + kCta < g.D ? d0 + kCta : g.D) - 1;
    if (!(dguard(kSiteChunkLocal, b, g.Bt) && dguard(kSiteChunkLocal, (c + 1) * tc - 1, g.L) &&
          dguard(kSiteChunkLocal, d0, g.D) &&
          dguard(kSiteChunkLocal, ((b * (g.nc + 1) + c) * g.D + dl) * N + N - 1, g.Bt * (g.nc + 1) * g.D * N)))
      return;
  }
  Stage<T, N, 2, 1, 2, 0, REV> st;
  st.carve(smem, kLocalSpan);
  auto prow = [&](int64_t t) { return b * g.L + (REV ? g.L - 1 - t : t); };  // row of logical token t
  st.td_src[0] = (const T*)p.xc;
  st.td_src[1] = (const T*)p.dtc;
  st.row_src[0] = (const T*)p.Bc;

  float2 A2[N / 2], h[N / 2];
  vzero2<N>(A2);
  vzero2<N>(h);
  if (act) {
    vload2<N>(A2, p.Af + d * N, 0);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) A2[j] = mul2(A2[j], f2(kLog2e));
  }
  float sdt = 0.f;
  const int64_t tc = (int64_t)g.m * g.Bs;
  const int64_t tbeg = (int64_t)c * tc;
  const int nspan = (int)((tc + kLocalSpan - 1) / kLocalSpan);
  st.issue(0, prow(tbeg), (int)(tc < kLocalSpan ? tc : kLocalSpan), g.D, d0);
  for (int sp = 0; sp < nspan; ++sp) {
    const int64_t t = (int64_t)sp * kLocalSpan;
    const int ns = (int)((tc - t) < kLocalSpan ? (tc - t) : kLocalSpan);
    __syncthreads();  // the other buffer is no longer read
    if (sp + 1 < nspan) {
      const int64_t tn = t + kLocalSpan;
      st.issue((sp + 1) & 1, prow(tbeg + tn), (int)((tc - tn) < kLocalSpan ? (tc - tn) : kLocalSpan), g.D, d0);
    }
    st.complete(sp & 1, ns, sp + 1 < nspan ? 1 : 0);
#pragma unroll 4
    for (int i = 0; i < ns; ++i) {
      const float dt = st.at(1, i);
      scan_state<N>(h, A2, dt, st.at(0, i), st.row(0, i));
      sdt = __fadd_rn(sdt, dt);
    }
  }
  if (act) {
    vstore2<N>(p.hst + ((b * (g.nc + 1) + c) * g.D + d) * N, h, 0);
    p.sdt[(b * g.nc + c) * g.D + d] = sdt;
  }
}

template <int N>
__global__ void __launch_bounds__(256) k_chunk_carry(const FwdParams p) {
  const Geo& g = p.g;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= g.Bt * g.D * N) return;
  const int n = (int)(idx % N);
  const int64_t d = (idx / N) % g.D, b = idx / ((int64_t)N * g.D);
  // debug build: the last state slot this thread writes (no barrier follows)
  if (!dguard(kSiteChunkCarry, ((b * (g.nc + 1) + g.nc_full) * g.D + d) * N + n, g.Bt * (g.nc + 1) * g.D * N)) return;
  const float A2 = __fmul_rn(p.Af[d * N + n], kLog2e);
  float H = p.init ? p.init[(b * g.D + d) * N + n] : 0.f;
  const int64_t hstride = g.D * N;
  float* hs = p.hst + b * (g.nc + 1) * hstride + d * N + n;
  const float* sd = p.sdt + b * g.nc * g.D + d;
  constexpr int U = 8;
  int c = 0;
  for (; c + U <= g.nc_full; c += U) {
    float hl[U], s[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {
      hl[j] = hs[(int64_t)(c + j) * hstride];
      s[j] = sd[(int64_t)(c + j) * g.D];
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      hs[(int64_t)(c + j) * hstride] = H;
      H = __fmaf_rn(ex2(__fmul_rn(A2, s[j])), H, hl[j]);
    }
  }
  for (; c < g.nc_full; ++c) {
    const float hl = hs[(int64_t)c * hstride], s = sd[(int64_t)c * g.D];
    hs[(int64_t)c * hstride] = H;
    H = __fmaf_rn(ex2(__fmul_rn(A2, s)), H, hl);
  }
  hs[(int64_t)g.nc_full * hstride] = H;
  dfinite(kSiteChunkCarry, H, idx);  // debug build: a non-finite cached state
}

// MODE 0: all-block forward (clean + noisy). MODE 1: clean scan only (cache
// build). MODE 2: clean scan only, right to left in time (logical token t is
// row L-1-t; the reverse direction of a full-sequence bidirectional layer).
// The active block has its own kernel (k_active_block).
template <int MODE>
struct ScanLayout {
  static_assert(MODE >= 0 && MODE <= 2, "block scan modes");
  static constexpr bool kClean = true;
  static constexpr bool kNoisy = MODE == 0;
  static constexpr int NTD = MODE == 0 ? 5 : 2;
  static constexpr int NROW = MODE == 0 ? 6 : 2;
  // token-by-channel slots
  static constexpr int XC = 0, DTC = 1;
  static constexpr int XN = 2, DTF = XN + 1, DTR = XN + 2;
  // token-by-state slots
  static constexpr int BC = 0, CC = 1;
  static constexpr int BF = 2, CF = BF + 1, BR = BF + 2, CR = BF + 3;
};

// TILED (blocks shorter than kScanSeg): several blocks per staged tile.
template <typename T, typename TO, int N, int MODE, bool TILED>
__global__ void __launch_bounds__(kCta, 4) k_block_scan(const FwdParams p) {
  using Ly = ScanLayout<MODE>;
  extern __shared__ __align__(16) unsigned char smem[];
  const Geo& g = p.g;
  const int64_t b = blockIdx.z;
  const int c = p.c_begin + blockIdx.y;
  const int64_t d0 = (int64_t)blockIdx.x * kCta, d = d0 + threadIdx.x;
  const bool act = d < g.D;
  // debug build: the chunk's first token and the channel group lie inside the sizes
  if (!(dguard(kSiteBlockScan, b, g.Bt) && dguard(kSiteBlockScan, (int64_t)c * g.m * g.Bs, g.L) &&
        dguard(kSiteBlockScan, d0, g.D)))
    return;
  const int Bs = (int)g.Bs;
  const int SEG = Bs < kScanSeg ? Bs : kScanSeg, NSEG = (Bs + SEG - 1) / SEG;
  // blocks shorter than kScanSeg are staged TB at a time (one tile of at most
  // kScanSeg tokens), so the staging and its barriers are paid per tile
  const int TB = TILED ? kScanSeg / Bs : 1;
  constexpr bool kRev = MODE == 2;
  Stage<T, N, Ly::NTD, Ly::NROW, 2, 0, kRev> st;
  st.carve(smem, NSEG == 1 ? TB * Bs : SEG);
  // the row holding logical row x = b L + t (t reversed in time for MODE 2)
  auto prow = [&](int64_t x) { return kRev ? 2 * b * g.L + g.L - 1 - x : x; };
  const bool dbuf = p.stage_bufs == 2 && NSEG == 1;
  float* yfbuf = reinterpret_cast<float*>(smem + decltype(st)::buf_bytes(st.stride()) *
                                                       (dbuf ? 2 : 1));
  if (Ly::kClean) {
    st.td_src[Ly::XC] = (const T*)p.xc;
    st.td_src[Ly::DTC] = (const T*)p.dtc;
    st.row_src[Ly::BC] = (const T*)p.Bc;
    st.row_src[Ly::CC] = (const T*)p.Cc;
  }
  if (Ly::kNoisy) {
    st.td_src[Ly::XN] = (const T*)p.xn;
    st.td_src[Ly::DTF] = (const T*)p.dtf;
    st.td_src[Ly::DTR] = (const T*)p.dtr;
    st.row_src[Ly::BF] = (const T*)p.Bf;
    st.row_src[Ly::CF] = (const T*)p.Cf;
    st.row_src[Ly::BR] = (const T*)p.Br;
    st.row_src[Ly::CR] = (const T*)p.Cr;
  }

  float2 A2f[N / 2], A2r[N / 2];
  float Df = 0.f, Dr = 0.f;
  vzero2<N>(A2f);
  vzero2<N>(A2r);
  if (act) {
    vload2<N>(A2f, p.Af + d * N, 0);
    Df = p.Df[d];
    if (Ly::kNoisy) {
      vload2<N>(A2r, p.Ar + d * N, 0);
      Dr = p.Dr[d];
    }
#pragma unroll
    for (int j = 0; j < N / 2; ++j) {
      A2f[j] = mul2(A2f[j], f2(kLog2e));
      A2r[j] = mul2(A2r[j], f2(kLog2e));
    }
  }

  const int k_lo = c * g.m, k_hi = min(k_lo + g.m, g.nb) - 1;
  const bool full = c < g.nc_full;
  float2 hc[N / 2];
  vzero2<N>(hc);
  if (act) vload2<N>(hc, p.hst + ((b * (g.nc + 1) + c) * g.D + d) * N, 0);

  auto tile_blocks = [&](int k0) { return k_hi - k0 + 1 < TB ? k_hi - k0 + 1 : TB; };
  if (dbuf) st.issue(0, prow(b * g.L + (int64_t)k_lo * Bs), tile_blocks(k_lo) * Bs, g.D, d0);
  for (int k0 = k_lo; k0 <= k_hi; k0 += TB) {
    const int nbk = tile_blocks(k0), tile = (k0 - k_lo) / TB;
    const int64_t trow = b * g.L + (int64_t)k0 * Bs;
    if (dbuf) {
      __syncthreads();  // the other buffer is no longer read
      const int k1 = k0 + TB;
      if (k1 <= k_hi) st.issue((tile + 1) & 1, prow(trow + (int64_t)nbk * Bs), tile_blocks(k1) * Bs, g.D, d0);
      st.complete(tile & 1, nbk * Bs, k1 <= k_hi ? 1 : 0);
    } else if (NSEG == 1) {
      st.load(prow(trow), nbk * Bs, g.D, d0);
    }
    for (int kk = 0; kk < nbk; ++kk) {
      const int k = k0 + kk;
      const int64_t row0 = trow + (int64_t)kk * Bs;
      const int toff = kk * Bs;  // the block's first token in the staged tile (0 for long blocks)
      float2 hs[N / 2];
#pragma unroll
      for (int j = 0; j < N / 2; ++j) hs[j] = hc[j];  // the block's seed: state before its first token
      for (int sg = 0; sg < NSEG; ++sg) {  // segments left to right
        const int i0 = sg * SEG, ns = Bs - i0 < SEG ? Bs - i0 : SEG;
        if (NSEG > 1) st.load(prow(row0 + i0), ns, g.D, d0);
#pragma unroll 2
        for (int ii = 0; ii < ns; ++ii) {
          const int i = i0 + ii;
          const int64_t o = prow(row0 + i) * g.D + d;
          if (Ly::kClean) {
            const float x = st.at(Ly::XC, toff + ii), dt = st.at(Ly::DTC, toff + ii);
            const float y = scan_step<N>(hc, A2f, dt, x, st.row(Ly::BC, toff + ii), st.row(Ly::CC, toff + ii));
            if (p.yc != nullptr && act) reinterpret_cast<TO*>(p.yc)[o] = to_out<TO>(with_skip(y, Df, x));
          }
          if (Ly::kNoisy) {
            const float x = st.at(Ly::XN, toff + ii), dt = st.at(Ly::DTF, toff + ii);
            const float y = scan_step<N>(hs, A2f, dt, x, st.row(Ly::BF, toff + ii), st.row(Ly::CF, toff + ii));
            yfbuf[i * kCta + threadIdx.x] = with_skip(y, Df, x);
          }
        }
      }
      if (Ly::kClean && p.emit_all && act) {
        float* dst = p.states + ((b * g.nb + k) * g.D + d) * N;
        if (k == k_hi && full) {
          float2 e[N / 2];
          vload2<N>(e, p.hst + ((b * (g.nc + 1) + c + 1) * g.D + d) * N, 0);
          vstore2<N>(dst, e, 0);
        } else {
          vstore2<N>(dst, hc, 0);
        }
      }
      if (Ly::kNoisy) {
        float2 hr[N / 2];
        vzero2<N>(hr);
        for (int sg = NSEG - 1; sg >= 0; --sg) {  // segments right to left; the last is still staged
          const int i0 = sg * SEG, ns = Bs - i0 < SEG ? Bs - i0 : SEG;
          if (sg < NSEG - 1) st.load(prow(row0 + i0), ns, g.D, d0);
#pragma unroll 2
          for (int ii = ns - 1; ii >= 0; --ii) {
            const int i = i0 + ii;
            const int64_t o = prow(row0 + i) * g.D + d;
            const float x = st.at(Ly::XN, toff + ii), dt = st.at(Ly::DTR, toff + ii);
            const float y = scan_step<N>(hr, A2r, dt, x, st.row(Ly::BR, toff + ii), st.row(Ly::CR, toff + ii));
            if (act)
              reinterpret_cast<TO*>(p.yn)[o] =
                  to_out<TO>(combine_dirs(yfbuf[i * kCta + threadIdx.x], with_skip(y, Dr, x)));
          }
        }
      }
    }
  }
  if (Ly::kClean && p.final_state != nullptr && c == g.nc - 1 && act) {
    float* dst = p.final_state + (b * g.D + d) * N;
    if (full) {
      float2 e[N / 2];
      vload2<N>(e, p.hst + ((b * (g.nc + 1) + c + 1) * g.D + d) * N, 0);
      vstore2<N>(dst, e, 0);
    } else {
      vstore2<N>(dst, hc, 0);
    }
  }
}

// ---------------------------------------------------------------------------
// Active block (the inference step): one noisy block per batch row from a
// read-only cached seed. A CTA covers 32 channels of one row; warp 0 runs the
// seeded forward scan and warp 1 the block-local reverse scan at the same
// time, each with the per-channel arithmetic of k_block_scan (scan_step,
// with_skip, combine_dirs), so the outputs equal those of the all-block
// forward bit for bit. The step is bound by the latency of the serial scan,
// so small CTAs spread it over many SMs.
// ---------------------------------------------------------------------------
constexpr int kActW = 32;  // channels per active-block CTA

template <typename T, int N>
struct ActiveLayout {
  // [3][Bs][32] x, dt_f, dt_r as stored; [4][Bs][N] B_f, C_f, B_r, C_r as
  // loaded and widened to fp32; [2][Bs][32] forward and reverse outputs
  static __host__ __device__ size_t td_bytes(int Bs) {
    return ((size_t)3 * Bs * kActW * sizeof(T) + 15) & ~(size_t)15;
  }
  static __host__ __device__ size_t raw_bytes(int Bs) {
    return is_f32<T>::value ? 0 : (((size_t)4 * Bs * N * sizeof(T) + 15) & ~(size_t)15);
  }
  static __host__ __device__ size_t rows_bytes(int Bs) { return (size_t)4 * Bs * N * 4; }
  static __host__ __device__ size_t bytes(int Bs) {
    return td_bytes(Bs) + raw_bytes(Bs) + rows_bytes(Bs) + (size_t)2 * Bs * kActW * 4;
  }
  // with adaptive layer norm: the modulated input [Bs][32] fp32 after the outputs
  static __host__ __device__ size_t bytes_ada(int Bs) { return bytes(Bs) + (size_t)Bs * kActW * 4; }
};

// ADA: adaptive layer norm on the block (Appendix E, eq. cacheable-adaln):
// the scans read u = (1 + scale) (x - mean) rstd + shift instead of x, and
// the output is x + gate * y_n. The seed, the cache, is never modulated.
template <typename T, typename TO, int N, bool ADA = false>
__global__ void __launch_bounds__(2 * kActW, 1) k_active_block(const FwdParams p) {
  using Ly = ActiveLayout<T, N>;
  extern __shared__ __align__(16) unsigned char smem[];
  const Geo& g = p.g;
  const int Bs = (int)g.Bs;
  const int64_t b = blockIdx.y, d0 = (int64_t)blockIdx.x * kActW;
  const int lane = threadIdx.x & 31, dir = threadIdx.x >> 5;  // dir 0: forward, 1: reverse
  const int64_t d = d0 + lane;
  const bool act = d < g.D;
  // debug build: the batch row and the channel group lie inside the sizes
  if (!(dguard(kSiteActiveBlock, b, g.Bt) && dguard(kSiteActiveBlock, d0, g.D))) return;
  T* td = reinterpret_cast<T*>(smem);
  float* rows = reinterpret_cast<float*>(smem + Ly::td_bytes(Bs) + Ly::raw_bytes(Bs));
  T* raw = is_f32<T>::value ? reinterpret_cast<T*>(rows) : reinterpret_cast<T*>(smem + Ly::td_bytes(Bs));
  float* ybuf = rows + (size_t)4 * Bs * N;

  // copies (16-byte chunks; channels past D read as zero)
  constexpr int E = 16 / (int)sizeof(T);
  constexpr int CPR = kActW / E;
  const int64_t row0 = b * g.L;
  for (int q = threadIdx.x; q < 3 * Bs * CPR; q += 2 * kActW) {
    const int j = q / (Bs * CPR), r = q - j * (Bs * CPR), t = r / CPR, cc = (r - t * CPR) * E;
    const T* src = (const T*)(j == 0 ? p.xn : (j == 1 ? p.dtf : p.dtr));
    const bool ok = d0 + cc < g.D;
    cp_async16(td + ((size_t)j * Bs + t) * kActW + cc,
               ok ? (const void*)(src + (row0 + t) * g.D + d0 + cc) : (const void*)src, ok ? 16 : 0);
  }
  const int rch = Bs * N / E;
  for (int q = threadIdx.x; q < 4 * rch; q += 2 * kActW) {
    const int j = q / rch, r = q - j * rch;
    const T* src = (const T*)(j == 0 ? p.Bf : (j == 1 ? p.Cf : (j == 2 ? p.Br : p.Cr)));
    cp_async16(raw + (size_t)j * Bs * N + r * E, src + row0 * N + (int64_t)r * E, 16);
  }
  cp_async_commit();

  // parameters and the seed while the copies are in flight
  float2 A2[N / 2], h[N / 2];
  vzero2<N>(A2);
  vzero2<N>(h);
  float Dd = 0.f;
  if (act) {
    vload2<N>(A2, (dir == 0 ? p.Af : p.Ar) + d * N, 0);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) A2[j] = mul2(A2[j], f2(kLog2e));
    Dd = dir == 0 ? p.Df[d] : p.Dr[d];
    if (dir == 0) vload2<N>(h, p.seed + (b * g.D + d) * N, 0);
  }
  cp_async_wait_all();
  __syncthreads();
  if (!is_f32<T>::value) {
    for (int q = threadIdx.x; q < 2 * Bs * N; q += 2 * kActW)
      reinterpret_cast<float2*>(rows)[q] = make_float2(cvt(raw[2 * q]), cvt(raw[2 * q + 1]));
    __syncthreads();
  }
  float* xmod = ybuf + (size_t)2 * Bs * kActW;  // [Bs][32], ADA only
  if (ADA) {
    for (int q = threadIdx.x; q < Bs * kActW; q += 2 * kActW) {
      const int i = q / kActW, c = q - i * kActW;
      const int64_t dc = d0 + c;
      float u = 0.f;
      if (dc < g.D) {
        const float2 st = p.ln_stats[b * Bs + i];
        const float z = __fmul_rn(__fsub_rn(cvt(td[q]), st.x), st.y);
        u = __fmaf_rn(__fadd_rn(1.f, p.scale[b * g.D + dc]), z, p.shift[b * g.D + dc]);
      }
      xmod[q] = u;
    }
    __syncthreads();
  }
  // this lane's input at token i: x as stored, or the modulated input
  auto xin = [&](int i) { return ADA ? xmod[i * kActW + lane] : cvt(td[i * kActW + lane]); };

  const T* xs = td;
  const T* dts = td + (size_t)(1 + dir) * Bs * kActW;
  const float* Brow = rows + (size_t)(2 * dir) * Bs * N;
  const float* Crow = Brow + (size_t)Bs * N;
  float* yb = ybuf + (size_t)dir * Bs * kActW;
  (void)xs;
  if (dir == 0) {
#pragma unroll 4
    for (int i = 0; i < Bs; ++i) {
      const float x = xin(i), dt = cvt(dts[i * kActW + lane]);
      const float y = scan_step<N>(h, A2, dt, x, Brow + i * N, Crow + i * N);
      yb[i * kActW + lane] = with_skip(y, Dd, x);
    }
  } else {
#pragma unroll 4
    for (int i = Bs - 1; i >= 0; --i) {
      const float x = xin(i), dt = cvt(dts[i * kActW + lane]);
      const float y = scan_step<N>(h, A2, dt, x, Brow + i * N, Crow + i * N);
      yb[i * kActW + lane] = with_skip(y, Dd, x);
    }
  }
  __syncthreads();
  for (int q = threadIdx.x; q < Bs * kActW; q += 2 * kActW) {
    const int i = q / kActW, c = q - i * kActW;
    if (d0 + c < g.D) {
      const float yv = combine_dirs(ybuf[q], ybuf[(size_t)Bs * kActW + q]);
      // gated residual of the modulated step: x + gate * y_n
      const float o = ADA ? __fmaf_rn(p.gate[b * g.D + d0 + c], yv, cvt(td[q])) : yv;
      reinterpret_cast<TO*>(p.yn)[(row0 + i) * g.D + d0 + c] = to_out<TO>(o);
    }
  }
}

// Layer-norm statistics of each token (one warp per row of D elements): the
// mean, then 1/sqrt(var + eps) from the centred second moment, in fp32.
template <typename T>
__global__ void __launch_bounds__(256) k_ln_stats(const T* h, int64_t rows, int64_t D, float eps, float2* stats) {
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const T* r = h + row * D;
  float s = 0.f;
  for (int64_t i = lane; i < D; i += 32) s = __fadd_rn(s, cvt(r[i]));
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xffffffffu, s, o));
  const float mu = __fdiv_rn(s, (float)D);
  float v = 0.f;
  for (int64_t i = lane; i < D; i += 32) {
    const float e = __fsub_rn(cvt(r[i]), mu);
    v = __fmaf_rn(e, e, v);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (lane == 0) stats[row] = make_float2(mu, __fdiv_rn(1.f, __fsqrt_rn(__fadd_rn(__fdiv_rn(v, (float)D), eps))));
}

// ---------------------------------------------------------------------------
// Sum of the two directions of a full-sequence bidirectional layer: each fp32
// input already holds its direction's output with its own skip term.
// ---------------------------------------------------------------------------
template <typename TO>
__global__ void __launch_bounds__(256) k_combine(const float* yf, const float* yr, TO* y, int64_t n4) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;  // four elements each
  if (i >= n4) return;
  const float4 a = reinterpret_cast<const float4*>(yf)[i], r = reinterpret_cast<const float4*>(yr)[i];
  TO* o = y + 4 * i;
  o[0] = to_out<TO>(combine_dirs(a.x, r.x));
  o[1] = to_out<TO>(combine_dirs(a.y, r.y));
  o[2] = to_out<TO>(combine_dirs(a.z, r.z));
  o[3] = to_out<TO>(combine_dirs(a.w, r.w));
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
namespace {

template <typename T, int N, bool REV>
cudaError_t chunk_local_rt(const FwdParams& p, cudaStream_t s) {
  const size_t smem = Stage<T, N, 2, 1, 2>::bytes(kLocalSpan);
  cudaError_t e =
      cudaFuncSetAttribute(k_chunk_local<T, N, REV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)p.g.G, (unsigned)p.g.nc_full, (unsigned)p.g.Bt);
  k_chunk_local<T, N, REV><<<grid, kCta, smem, s>>>(p);
  return cudaGetLastError();
}
template <typename T, int N>
cudaError_t chunk_local_t(const FwdParams& p, cudaStream_t s) {
  return p.rev ? chunk_local_rt<T, N, true>(p, s) : chunk_local_rt<T, N, false>(p, s);
}

// Above this much shared memory per CTA the block scan stages synchronously:
// at 16-token blocks a second buffer would cost a resident CTA per SM, which
// measured slower than the overlap it buys.
constexpr size_t kDoubleBufferLimit = 48 * 1024;

template <typename T, typename TO, int N, int MODE>
int block_scan_bufs_t(int64_t Bs) {
  using Ly = ScanLayout<MODE>;
  if (Bs > kScanSeg) return 1;  // segments are staged when needed
  const int tile = (int)(kScanSeg / Bs * Bs);
  const size_t extra = Ly::kNoisy ? (size_t)Bs * kCta * sizeof(float) : 0;
  return 2 * Stage<T, N, Ly::NTD, Ly::NROW, 2>::buf_bytes(tile) + extra <= kDoubleBufferLimit ? 2 : 1;
}

template <typename T, typename TO, int N, int MODE>
size_t block_scan_smem_t(int64_t Bs) {
  using Ly = ScanLayout<MODE>;
  const int seg = Bs < kScanSeg ? (int)(kScanSeg / Bs * Bs) : kScanSeg;  // staged tokens
  size_t b = Stage<T, N, Ly::NTD, Ly::NROW, 2>::buf_bytes(seg) * block_scan_bufs_t<T, TO, N, MODE>(Bs);
  if (Ly::kNoisy) b += (size_t)Bs * kCta * sizeof(float);
  return b;
}

template <typename T, typename TO, int N, int MODE>
cudaError_t block_scan_t(int nchunks, const FwdParams& p_in, cudaStream_t s) {
  FwdParams p = p_in;
  p.stage_bufs = block_scan_bufs_t<T, TO, N, MODE>(p.g.Bs);
  const size_t smem = block_scan_smem_t<T, TO, N, MODE>(p.g.Bs);
  dim3 grid((unsigned)p.g.G, (unsigned)nchunks, (unsigned)p.g.Bt);
  if (p.g.Bs < kScanSeg) {
    cudaError_t e = cudaFuncSetAttribute(k_block_scan<T, TO, N, MODE, true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_block_scan<T, TO, N, MODE, true><<<grid, kCta, smem, s>>>(p);
  } else {
    cudaError_t e = cudaFuncSetAttribute(k_block_scan<T, TO, N, MODE, false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_block_scan<T, TO, N, MODE, false><<<grid, kCta, smem, s>>>(p);
  }
  return cudaGetLastError();
}

template <typename T, typename TO, int N>
cudaError_t block_scan_mode(int mode, int nchunks, const FwdParams& p, cudaStream_t s) {
  switch (mode) {
    case 0: return block_scan_t<T, TO, N, 0>(nchunks, p, s);
    case 1: return block_scan_t<T, TO, N, 1>(nchunks, p, s);
    case 2: return block_scan_t<T, TO, N, 2>(nchunks, p, s);
    default: return cudaErrorInvalidValue;
  }
}

template <typename T, typename TO, int N, bool ADA = false>
cudaError_t active_block_t(const FwdParams& p, cudaStream_t s) {
  const size_t smem = ADA ? ActiveLayout<T, N>::bytes_ada((int)p.g.Bs) : ActiveLayout<T, N>::bytes((int)p.g.Bs);
  if (smem > 48 * 1024) {
    cudaError_t e =
        cudaFuncSetAttribute(k_active_block<T, TO, N, ADA>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((unsigned)((p.g.D + kActW - 1) / kActW), (unsigned)p.g.Bt);
  k_active_block<T, TO, N, ADA><<<grid, 2 * kActW, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

#define BDS_DISPATCH_N(N, ...)                      \
  switch (N) {                                      \
    case 8: { constexpr int NN = 8; __VA_ARGS__ }   \
    case 16: { constexpr int NN = 16; __VA_ARGS__ } \
    default: return cudaErrorInvalidValue;          \
  }

cudaError_t launch_chunk_local(int dt, int N, const FwdParams& p, cudaStream_t s) {
  if (p.g.nc_full == 0 || p.g.Bt == 0) return cudaSuccess;
  if (dt == 0) {
    BDS_DISPATCH_N(N, return chunk_local_t<float, NN>(p, s);)
  }
  BDS_DISPATCH_N(N, return chunk_local_t<bf16, NN>(p, s);)
}

cudaError_t launch_chunk_carry(int N, const FwdParams& p, cudaStream_t s) {
  const int64_t total = p.g.Bt * p.g.D * N;
  if (total == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)((total + 255) / 256);
  BDS_DISPATCH_N(N, k_chunk_carry<NN><<<blocks, 256, 0, s>>>(p); return cudaGetLastError();)
}

cudaError_t launch_block_scan(int dt, int N, int mode, int nchunks, const FwdParams& p, cudaStream_t s) {
  if (nchunks == 0 || p.g.Bt == 0) return cudaSuccess;
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return block_scan_mode<float, float, NN>(mode, nchunks, p, s);)
    case 1: BDS_DISPATCH_N(N, return block_scan_mode<bf16, bf16, NN>(mode, nchunks, p, s);)
    default: BDS_DISPATCH_N(N, return block_scan_mode<bf16, float, NN>(mode, nchunks, p, s);)
  }
}

cudaError_t launch_active_block(int dt, int N, const FwdParams& p, cudaStream_t s) {
  if (p.g.Bt == 0 || p.g.D == 0) return cudaSuccess;
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return active_block_t<float, float, NN>(p, s);)
    case 1: BDS_DISPATCH_N(N, return active_block_t<bf16, bf16, NN>(p, s);)
    default: BDS_DISPATCH_N(N, return active_block_t<bf16, float, NN>(p, s);)
  }
}

cudaError_t launch_active_block_adaln(int dt, int N, const FwdParams& p, cudaStream_t s) {
  if (p.g.Bt == 0 || p.g.D == 0) return cudaSuccess;
  switch (dt) {
    case 0: BDS_DISPATCH_N(N, return active_block_t<float, float, NN, true>(p, s);)
    case 1: BDS_DISPATCH_N(N, return active_block_t<bf16, bf16, NN, true>(p, s);)
    default: BDS_DISPATCH_N(N, return active_block_t<bf16, float, NN, true>(p, s);)
  }
}

cudaError_t launch_ln_stats(int dt, const void* h, int64_t rows, int64_t D, float eps, float2* stats, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)((rows + 7) / 8);
  if (dt == 0)
    k_ln_stats<float><<<blocks, 256, 0, s>>>(reinterpret_cast<const float*>(h), rows, D, eps, stats);
  else
    k_ln_stats<bf16><<<blocks, 256, 0, s>>>(reinterpret_cast<const bf16*>(h), rows, D, eps, stats);
  return cudaGetLastError();
}

cudaError_t launch_combine(int out_f32, const float* yf, const float* yr, void* y, int64_t n, cudaStream_t s) {
  const int64_t n4 = n / 4;  // D is a multiple of 4
  if (n4 == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)((n4 + 255) / 256);
  if (out_f32)
    k_combine<float><<<blocks, 256, 0, s>>>(yf, yr, reinterpret_cast<float*>(y), n4);
  else
    k_combine<bf16><<<blocks, 256, 0, s>>>(yf, yr, reinterpret_cast<bf16*>(y), n4);
  return cudaGetLastError();
}

}  // namespace bds
