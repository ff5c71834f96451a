// ssd.cu -- kernels of the SSD form (Mamba-2: one scalar decay per head,
// B and C shared by all channels) of the block-restricted bidirectional scan,
// on the tcgen05 tensor cores of sm_103a.
//
// Per block of Bs tokens (Bs = 128 m) and head h, with a_t = exp(dt_t A[h]):
//   * block-local end state (k_ssd_block_state):
//       T = sum_s w_s x_s B_s^T, w_s = exp(A sum_{r>s} dt_r) dt_s,
//     one MMA chain per head (M = 128 state rows, N = 64 channels, K = Bs
//     tokens): the block's B rows as stored are the MN-major A operand, the
//     weighted x (w o x, split into bf16 high and low parts) the B operand;
//   * the exact state at each block end (k_ssd_state_pass):
//       S_k = exp(A sum_block dt) S_{k-1} + T_k, in fp32, sequential in k;
//   * the block's output (k_ssd_block_scan), for a 128-token tile t of the block:
//       y_t = sum_s M[t, s] x_s + exp(A sum_{r<=t} dt_r) C_t . seed + D x_t,
//       M[t, s] = (C^f_t . B^f_s) exp(A_f sum_{s<r<=t} dt^f_r) dt^f_s  for s <= t
//               + (C^r_t . B^r_s) exp(A_r sum_{t<=r<s} dt^r_r) dt^r_s  for s >= t
//     (the reverse term only for noisy blocks). The Gram products C B^T are
//     shared by all heads and stay in TMEM; each head's decay-weighted M tile
//     is written to shared memory in bf16 and multiplied with x on the tensor
//     core; the seed term is a second MMA (seed split into bf16 high and low
//     parts); the epilogue adds the decayed seed term and D x.
#include <atomic>
#include <cstdio>
#include <cstring>
#include <mutex>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "device.cuh"
#include "params.h"
#include "ssd.cuh"
#include "ssd_common.cuh"
#include "umma.cuh"

namespace bds {
namespace {

using umma::sw128;

__device__ int g_ssd_wait_flag;

// Shared memory of k_ssd_block_state (offsets from a 1024-aligned base):
//   b     the block's B rows as the MN-major A operand: two 64-wide halves of
//         [Bs][64] bf16 (state rows 64..127 are zero when N = 64)
//   xr    two buffers of a head's x rows as loaded ([Bs][64] bf16, swizzled)
//   xs    the weighted x of the current head, bf16 high and low parts, each
//         [Bs][64] MN-major (the B operand)
//   w     per head of the CTA and token: exp(A sum_{r>s} dt_r) dt_s
struct StateSmem {
  uint32_t b, xr, xs, w, total;
  __host__ __device__ StateSmem(int Bs) {
    const uint32_t half = (uint32_t)Bs * 128u;
    b = 0;
    xr = b + 2u * half;
    xs = xr + 2u * half;
    w = xs + 2u * half;
    total = w + 8u * 256u * 4u + 1024u;
  }
};

constexpr int kStateThreads = 256;
constexpr int kStateIssuer = 64;  // the thread that issues a head's MMAs (k_ssd_block_state)

// One CTA of 8 warps per (batch row, block) and group of at most 8 heads.
// T^T[n][p] = sum_s B_s[n] (w_s x_s[p]): M = 128 state rows, N = 64
// channels, K = Bs tokens; warps w and w + 4 read TMEM lanes 32 (w % 4) and
// split the 64 channels. Head h's MMAs run while head h-1's accumulator is
// written out (two accumulators, TMEM columns 0..63 and 64..127).
template <int N>
__global__ void __launch_bounds__(kStateThreads, 1) k_ssd_block_state(const SsdStateParams p) {
  extern __shared__ unsigned char smraw[];
  unsigned char* sm = align1024(smraw);
  __shared__ uint64_t bar[2];
  __shared__ uint32_t tslot;
  const SsdGeo& g = p.g;
  const int Bs = (int)g.Bs, H = g.H, t = threadIdx.x, w = t >> 5, lane = t & 31;
  const StateSmem S(Bs);
  const uint32_t half = (uint32_t)Bs * 128u;
  const int64_t bk = blockIdx.x, b = bk / g.nb;
  const int k = (int)(bk % g.nb);
  const int h0 = blockIdx.y * p.hg, h1 = min(H, h0 + p.hg), hg = h1 - h0;
  // debug build: the block, the head group and its last state slot lie inside the sizes
  if (!(dguard(kSiteSsdBlockState, bk, g.Bt * g.nb) && dguard(kSiteSsdBlockState, h0, H) &&
        dguard(kSiteSsdBlockState, ((bk * H + h1 - 1) * kSsdP + kSsdP - 1) * N + N - 1, g.Bt * g.nb * H * kSsdP * N)))
    return;
  const RowMap tok(b, g.L, (int64_t)k * Bs, p.rev != 0);
  float* s_w = reinterpret_cast<float*>(sm + S.w);  // [hg][256]
  // B rows: chunk c of 8 state indices of token s goes to half c / 8
  for (int c = t; c < Bs * N / 8; c += kStateThreads) {
    const int s = c / (N / 8), ch = c % (N / 8);
    cp_async16(sm + S.b + (ch >> 3) * half + sw128(s, ch & 7), p.B + tok(s) * N + ch * 8, 16);
  }
  if (N == 64)
    for (int c = t; c < Bs * 8; c += kStateThreads)
      *reinterpret_cast<uint4*>(sm + S.b + half + c * 16) = make_uint4(0, 0, 0, 0);
  auto load_x = [&](int h, int buf) {
    for (int c = t; c < Bs * 8; c += kStateThreads) {
      const int s = c >> 3, ch = c & 7;
      cp_async16(sm + S.xr + buf * half + sw128(s, ch), p.x + (tok(s) * H + h) * kSsdP + ch * 8, 16);
    }
    cp_async_commit();
  };
  if (h0 < h1) load_x(h0, 0);
  // weights of every head of the CTA: warp hh scans head hh (suffix sums)
  if (w < hg) {
    const int h = h0 + w;
    const __nv_bfloat16* dth = p.dt + tok.base * H + h;  // position s at dth[s * dstep]
    const int64_t dstep = tok.step * H;
    float* suf = s_w + w * 256;
    const float tot = warp_scan_dt<true>(dth, dstep, Bs, suf);  // inclusive suffix sums
    __syncwarp();
    const float A2 = __fmul_rn(p.A[h], kLog2e);
    float wv[8];
    for (int q = 0, s = lane; s < Bs; s += 32, ++q) {
      const float after = s + 1 < Bs ? suf[s + 1] : 0.f;  // sum of dt over tokens after s
      wv[q] = __fmul_rn(ex2(__fmul_rn(A2, after)), __bfloat162float(dth[(int64_t)s * dstep]));
    }
    __syncwarp();
    for (int q = 0, s = lane; s < Bs; s += 32, ++q) suf[s] = wv[q];
    if (lane == 0) p.sumdt[bk * H + h] = tot;
  }
  if (t == 0) {
    umma::bar_init(&bar[0], 1);
    umma::bar_init(&bar[1], 1);
  }
  if (t < 32) tmem_alloc(&tslot, 128);
  umma::fence_before_sync();
  __syncthreads();
  umma::fence_after_sync();
  const uint32_t tm = tslot;
  const uint32_t lane_base = tm + ((uint32_t)(32 * (w & 3)) << 16);
  bool alive = true;
  // writes head (h0 + j)'s T from accumulator j & 1: lane n = state row n,
  // this warp's 32 of the 64 channels
  auto write_out = [&](int j) {
    const int n = 32 * (w & 3) + lane, pc = 32 * (w >> 2);
    if (32 * (w & 3) < N) {  // whole warps
      float v[32];
      umma::tmem_ld32(lane_base + 64u * (uint32_t)(j & 1) + (uint32_t)pc, v);
      float* dst = p.T + ((bk * H + h0 + j) * kSsdP + pc) * N + n;
#pragma unroll
      for (int e = 0; e < 32; ++e) dst[(int64_t)e * N] = v[e];
    }
  };
  for (int hh = 0; hh < hg && alive; ++hh) {
    const int h = h0 + hh;
    cp_async_wait_all();
    __syncthreads();  // head hh's x rows are in shared memory
    if (hh + 1 < hg) load_x(h + 1, (hh + 1) & 1);
    if (hh > 0) {  // head hh-1's MMAs are done reading the weighted x
      if (!cta_wait(&bar[(hh - 1) & 1], ((hh - 1) >> 1) & 1, p.flag)) {
        alive = false;
        break;
      }
      umma::fence_after_sync();
    }
    const unsigned char* xr = sm + S.xr + (hh & 1) * half;
    const float* wv = s_w + hh * 256;
    for (int c = t; c < Bs * 8; c += kStateThreads) {
      const int s = c >> 3, ch = c & 7;
      const uint32_t off = sw128(s, ch);
      const uint4 u = *reinterpret_cast<const uint4*>(xr + off);
      const __nv_bfloat162* xv = reinterpret_cast<const __nv_bfloat162*>(&u);
      const float ws = wv[s];
      uint32_t wh[4], wl[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __bfloat1622float2(xv[e]);
        const float v0 = __fmul_rn(ws, f.x), v1 = __fmul_rn(ws, f.y);
        const __nv_bfloat162 hv = __floats2bfloat162_rn(v0, v1);
        wh[e] = *reinterpret_cast<const uint32_t*>(&hv);
        wl[e] = pack_bf16(__fsub_rn(v0, __low2float(hv)), __fsub_rn(v1, __high2float(hv)));
      }
      *reinterpret_cast<uint4*>(sm + S.xs + off) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
      *reinterpret_cast<uint4*>(sm + S.xs + half + off) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
    }
    umma::fence_async_smem();
    umma::fence_before_sync();
    __syncthreads();
    // the issuing thread is held while the tensor pipe takes the MMAs: thread
    // 64's warp writes no output rows when N is 64 (only warps with
    // 32 (w mod 4) < N do), so the previous head's write-out runs beside it
    if (t == kStateIssuer) {
      umma::fence_after_sync();
      const uint32_t a0 = umma::smem_u32(sm + S.b), x0 = umma::smem_u32(sm + S.xs);
      constexpr uint32_t id = umma::idesc_bf16(128, 64, true, true);
      const uint32_t d = tm + 64u * (uint32_t)(hh & 1);
      const uint64_t da = umma::sdesc(a0, half, 1024), dh = umma::sdesc(x0, 1024, 1024),
                     dl = umma::sdesc(x0 + half, 1024, 1024);
      for (int kk = 0; kk < Bs / 16; ++kk) {
        const uint64_t a = umma::sdesc_adv(da, kk * 2048u);
        umma::mma_bf16(d, a, umma::sdesc_adv(dh, kk * 2048u), id, kk > 0);
        umma::mma_bf16(d, a, umma::sdesc_adv(dl, kk * 2048u), id, true);
      }
      umma::mma_commit(&bar[hh & 1]);
    }
    if (hh > 0) write_out(hh - 1);  // under head hh's MMAs
  }
  if (alive && hg > 0) {
    if (cta_wait(&bar[(hg - 1) & 1], ((hg - 1) >> 1) & 1, p.flag)) {
      umma::fence_after_sync();
      write_out(hg - 1);
    }
  }
  cp_async_wait_all();
  umma::fence_before_sync();
  __syncthreads();
  if (t < 32) tmem_dealloc(tm, 128);
}


// One thread per (batch row, head, channel, state index), sequential in k.
__global__ void __launch_bounds__(256) k_ssd_state_pass(const SsdPassParams p) {
  const SsdGeo& g = p.g;
  const int64_t per_b = (int64_t)g.H * kSsdP * g.N;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= g.Bt * per_b) return;
  const int64_t b = idx / per_b, r = idx - b * per_b;
  const int h = (int)(r / ((int64_t)kSsdP * g.N));
  // debug build: the last block-state slot this thread reads (no barrier follows)
  if (!dguard(kSiteSsdStatePass, (b * g.nb + g.nb - 1) * per_b + r, g.Bt * g.nb * per_b)) return;
  const float A2 = __fmul_rn(p.A[h], kLog2e);
  float S = p.init != nullptr ? p.init[idx] : 0.f;
  const float* T = p.T + b * g.nb * per_b + r;
  const float* sd = p.sumdt + b * g.nb * g.H + h;
  constexpr int U = 8;  // loads of U blocks first: they do not depend on the state
  for (int k0 = 0; k0 < g.nb; k0 += U) {
    float tv[U], dv[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int k = min(k0 + u, g.nb - 1);
      tv[u] = T[(int64_t)k * per_b];
      dv[u] = sd[(int64_t)k * g.H];
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (k0 + u >= g.nb) break;
      S = __fmaf_rn(ex2(__fmul_rn(A2, dv[u])), S, tv[u]);
      if (p.emit_all) p.states[(b * g.nb + k0 + u) * per_b + r] = S;
    }
  }
  if (!p.emit_all) p.states[b * per_b + r] = S;
  if (p.final_state != nullptr) p.final_state[b * per_b + r] = S;
  dfinite(kSiteSsdStatePass, S, idx);  // debug build: a non-finite cached state
}

// Copies one 128-token tile of a [tokens][N] bf16 tensor into K-major
// swizzled shared memory (N / 64 atom columns).
template <int N>
__device__ __forceinline__ void stage_rows(unsigned char* dst, const __nv_bfloat16* src, const RowMap& tok, int row0) {
  for (int c = threadIdx.x; c < 128 * N / 8; c += blockDim.x) {
    const int r = c / (N / 8), ch = c % (N / 8);
    cp_async16(dst + (ch >> 3) * kTile16 + sw128(r, ch & 7), src + tok(row0 + r) * N + ch * 8, 16);
  }
}

// Gram product D[128 x 128] = A_rows . B_rows^T over K = N (both K-major).
template <int N>
__device__ __forceinline__ void mma_gram(uint32_t d, uint32_t a, uint32_t b) {
  constexpr uint32_t id = umma::idesc_bf16(128, 128, false, false);
  const uint64_t da = umma::sdesc(a, 16, 1024), db = umma::sdesc(b, 16, 1024);
#pragma unroll
  for (int kk = 0; kk < N / 16; ++kk) {
    const uint32_t off = (kk >> 2) * kTile16 + (kk & 3) * 32u;
    umma::mma_bf16(d, umma::sdesc_adv(da, off), umma::sdesc_adv(db, off), id, kk > 0);
  }
}

// Shared memory of k_ssd_block_scan (offsets from a 1024-aligned base):
//   cf    the tile's C^f rows, K-major (N / 64 atom columns)
//   m0    decay-weighted mixing tile, buffer 0 (128 x 128 bf16, K-major)
//   m1    buffer 1; holds the tile's C^r rows until the Gram products are done
//   r     the B tiles of the Gram products; afterwards two buffers of a
//         head's x tiles (MN-major, 16 KB each; the current head and the next)
//         and the seed's bf16 high and low parts (64 rows x N, K-major).
//         The next head's seed, as loaded (fp32), waits in m1 (free between
//         a head's last mixing tile and the next head's second one).
//   dt    dt of every head of the CTA, per token, both directions (bf16)
//   vec   per token of the block, for the current head: A2 * cumulative dt,
//         dt and the column factors of both directions
struct ScanSmem {
  uint32_t cf, m0, m1, r, x, xsz, seed, raw, dt, vec, prm, total;
  __host__ __device__ ScanSmem(int N, int m) {
    const uint32_t tileC = 128u * (uint32_t)N * 2u;
    const uint32_t tileM = 32768u;
    cf = 0;
    m0 = cf + tileC;
    m1 = m0 + tileM;
    r = m1 + (tileC > tileM ? tileC : tileM);
    const uint32_t gram = (uint32_t)(m + 1) * tileC;
    x = r;
    xsz = (uint32_t)m * 16384u;
    seed = x + 2u * xsz;
    raw = m1;
    const uint32_t xs = 2u * xsz + 256u * (uint32_t)N;
    dt = r + (gram > xs ? gram : xs);
    vec = dt + 2u * 256u * 16u * 2u;
    prm = vec + 2u * 6u * 256u * 4u;
    total = prm + 4u * 16u * 4u + 1024u;  // + alignment slack of the dynamic base
  }
};

constexpr int kScanThreads = 256;
constexpr int kScanIssuer = 128;  // the thread that issues a head's MMAs
constexpr int kMaxHeadsPerCta = 16;

// Issues the cp.async copies of one head's x tiles (MN-major) and its seed
// (fp32, as stored) for a CTA of kScanThreads threads.
template <int N>
__device__ __forceinline__ void issue_head_loads(unsigned char* sm, const ScanSmem& L, const __nv_bfloat16* x,
                                                 const RowMap& tok, int H, int h, int ntile, const float* seed_h,
                                                 uint32_t xbuf) {
  for (int c = threadIdx.x; c < ntile * kSsdT * 8; c += kScanThreads) {
    const int s = c >> 3, ch = c & 7;
    cp_async16(sm + xbuf + (s >> 7) * 16384u + sw128(s & 127, ch), x + (tok(s) * H + h) * kSsdP + ch * 8, 16);
  }
  if (seed_h != nullptr)
    for (int c = threadIdx.x; c < kSsdP * N / 4; c += kScanThreads) cp_async16(sm + L.raw + c * 16, seed_h + c * 4, 16);
  cp_async_commit();
}

// Decay vectors of one direction of a head, by one warp, from the head's dt
// column in shared memory (bf16, stride `hs` between tokens): va = A2 times
// the inclusive cumulative dt (prefix sums forward, suffix sums reverse: each
// lane sums its tokens in order, then the lane totals are scanned), vw = dt,
// and the column factors
// vc = exp2(va_ref - va_s) vw_s with the reference at the last (forward) or
// first (reverse) token of s's 32-token column group. Lane l holds the
// tokens at scan positions l * per .. l * per + per - 1 in registers, so the
// reference is one shuffle away and every load is issued at once.
template <bool REV, typename T>
__device__ __forceinline__ void setup_dir(const T* dt, int hs, int n, float A2, float* va, float* vw, float* vc) {
  const int lane = threadIdx.x & 31, per = n / 32;  // 4 or 8
  float d[8], a[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const int pos = REV ? n - 1 - (lane * per + q) : lane * per + q;
    d[q] = q < per ? cvt(dt[pos * hs]) : 0.f;
  }
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    s = q < per ? __fadd_rn(s, d[q]) : s;
    a[q] = s;
  }
  float inc = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float v = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc = __fadd_rn(inc, v);
  }
  float base = __shfl_up_sync(0xffffffffu, inc, 1);
  if (lane == 0) base = 0.f;
#pragma unroll
  for (int q = 0; q < 8; ++q) a[q] = __fmul_rn(A2, __fadd_rn(base, a[q]));
  // the group's reference token is scan position 32 g + 31: lane (l | (32/per - 1)), slot per - 1
  const float ref = __shfl_sync(0xffffffffu, per == 8 ? a[7] : a[3], lane | (32 / per - 1));
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    if (q >= per) break;
    const int pos = REV ? n - 1 - (lane * per + q) : lane * per + q;
    va[pos] = a[q];
    vw[pos] = d[q];
    vc[pos] = __fmul_rn(ex2(__fsub_rn(ref, a[q])), d[q]);
  }
}

// One CTA of 8 warps per (batch row, block, 128-token tile i of the block)
// and group of at most 16 heads. Warp w serves token rows 32 (w % 4) .. +31 of
// the tile (TMEM lanes of its quarter) and column half w / 4 of each mixing
// tile and of the output.
// TMEM columns: Gram products at 128 q (forward products of s-tiles 0..i,
// then, for noisy blocks, reverse products of s-tiles i..m-1), the output
// accumulator at 384 and the seed term at 448.
// Decays: inside the block, exp(A sum dt) between rows and columns that are
// 32-token groups apart factors exactly into a row factor times a column
// factor, both at most 1 (referenced to the column group's last token for
// the forward direction and its first token for the reverse one); only the
// 32 x 32 blocks on the diagonal take one exp per element.
template <int N, bool NOISY>
__global__ void __launch_bounds__(kScanThreads, 1) k_ssd_block_scan(const SsdScanParams p,
                                                                    const __grid_constant__ CUtensorMap xmap) {
  extern __shared__ unsigned char smraw[];
  unsigned char* sm = align1024(smraw);
  __shared__ uint64_t bar[3];  // [0]: a head's MMAs, [1]: the Gram products, [2]: a head's loads (TMA)
  __shared__ uint32_t tslot;
  const SsdGeo& g = p.g;
  const int Bs = (int)g.Bs, H = g.H, m = g.m, t = threadIdx.x;
  const int w = t >> 5, lane = t & 31, q4 = w & 3, hf = w >> 2;
  const ScanSmem L(N, m);
  const int64_t idx = blockIdx.x;
  const int i = (int)(idx % m);
  const int64_t bk = idx / m, b = bk / g.nb;
  const int k = (int)(bk % g.nb);
  const int h0 = blockIdx.y * p.hg, h1 = min(H, h0 + p.hg), hg = h1 - h0;
  // debug build: the tile and the head group lie inside the sizes
  if (!(dguard(kSiteSsdBlockScan, idx, g.Bt * g.nb * m) && dguard(kSiteSsdBlockScan, h0, H))) return;
  const RowMap tok(b, g.L, (int64_t)k * Bs, p.rev != 0);
  const int row = 32 * q4 + lane, tt = i * kSsdT + row;  // token row in the tile / in the block
  const int rg = 4 * i + q4;                              // 32-token row group in the block
  __nv_bfloat16* s_dtf = reinterpret_cast<__nv_bfloat16*>(sm + L.dt);  // [Bs][hg], as stored
  __nv_bfloat16* s_dtr = s_dtf + 256 * kMaxHeadsPerCta;
  // per-head decay vectors, two buffers (the next head's are prepared while
  // the current head's MMAs run): A2_f * inclusive prefix sums of dt_f, dt_f,
  // forward column factors, A2_r * inclusive suffix sums of dt_r, dt_r,
  // reverse column factors; 256 floats each
  float* const vec0 = reinterpret_cast<float*>(sm + L.vec);
  const int nf = i + 1, nr = NOISY ? m - i : 0;           // Gram products per direction
  const int ntile = NOISY ? m : i + 1;                    // s-tiles whose x a head needs
  // this block's seed: slot k - 1 (or k) of p.seed; block 0 of a shifted
  // layout starts from init_seed
  const float* seed_src = nullptr;
  if (p.seed_shift && k == 0) {
    if (p.init_seed != nullptr) seed_src = p.init_seed + b * (int64_t)H * kSsdP * N;
  } else if (p.seed != nullptr) {
    seed_src = p.seed + b * p.seed_bstride + (int64_t)(p.seed_shift ? k - 1 : k) * H * kSsdP * N;
  }
  const bool has_seed = seed_src != nullptr;
  // --- Gram products C B^T of this tile against the block's s-tiles
  stage_rows<N>(sm + L.cf, p.Cf, tok, i * kSsdT);
  for (int j = 0; j < nf; ++j) stage_rows<N>(sm + L.r + j * 128u * N * 2u, p.Bf, tok, j * kSsdT);
  if (NOISY) {
    stage_rows<N>(sm + L.m1, p.Cr, tok, i * kSsdT);
    for (int j = i; j < m; ++j)
      stage_rows<N>(sm + L.r + (nf + j - i) * 128u * N * 2u, p.Br, tok, j * kSsdT);
  }
  cp_async_commit();
  float* s_prm = reinterpret_cast<float*>(sm + L.prm);  // [4][16]: A_f, D_f, A_r, D_r of the CTA's heads
  if (t < hg) {
    s_prm[t] = p.Af[h0 + t];
    s_prm[16 + t] = p.Df[h0 + t];
    if (NOISY) {
      s_prm[32 + t] = p.Ar[h0 + t];
      s_prm[48 + t] = p.Dr[h0 + t];
    }
  }
  {  // dt of the CTA's heads, bf16 as stored (Bs hg <= 256 * 16): every load issued before the stores
    __nv_bfloat16 vf[kMaxHeadsPerCta], vr[kMaxHeadsPerCta];
    const int ne = Bs * hg;
#pragma unroll
    for (int q = 0; q < kMaxHeadsPerCta; ++q) {
      const int e = t + q * kScanThreads, s = e / hg, hh = e - s * hg;
      if (e < ne) {
        vf[q] = p.dtf[tok(s) * H + h0 + hh];
        if (NOISY) vr[q] = p.dtr[tok(s) * H + h0 + hh];
      }
    }
#pragma unroll
    for (int q = 0; q < kMaxHeadsPerCta; ++q) {
      const int e = t + q * kScanThreads;
      if (e < ne) {
        s_dtf[e] = vf[q];
        if (NOISY) s_dtr[e] = vr[q];
      }
    }
  }
  if (t == 0) {
    umma::bar_init(&bar[0], 1);
    umma::bar_init(&bar[1], 1);
    umma::bar_init(&bar[2], 1);
  }
  if (t < 32) tmem_alloc(&tslot, 512);
  cp_async_wait_all();
  umma::fence_async_smem();
  umma::fence_before_sync();
  __syncthreads();
  umma::fence_after_sync();
  const uint32_t tm = tslot;
  const uint32_t lane_base = tm + ((uint32_t)(32 * q4) << 16);
  if (t == 0) {
    const uint32_t base = umma::smem_u32(sm);
    for (int qq = 0; qq < nf + nr; ++qq)
      mma_gram<N>(tm + 128u * qq, base + (qq < nf ? L.cf : L.m1), base + L.r + qq * 128u * N * 2u);
    umma::mma_commit(&bar[1]);
  }
  bool alive = cta_wait(&bar[1], 0, p.flag);
  umma::fence_after_sync();
  // one head's x tiles and raw seed into buffer xbuf: by TMA (thread 0; a
  // 128-token x tile is one box of the [tokens][heads][64] map, the seed one
  // contiguous run) when the launcher set up the map, else by cp.async
  bool ld_pending = false;  // a TMA phase issued and not yet waited for
  uint32_t ld_parity = 0;
  auto load_head = [&](int hd, uint32_t xbuf) {
    const float* seed_h = has_seed ? seed_src + (int64_t)hd * kSsdP * N : nullptr;
    if (p.tma) {
      ld_pending = true;
      ld_parity = (uint32_t)((hd - h0) & 1);
      if (t == 0) {
        umma::fence_async_smem();  // the buffers' earlier generic accesses before the async writes
        bar_expect_tx(&bar[2], (uint32_t)ntile * 16384u + (seed_h != nullptr ? (uint32_t)(kSsdP * N * 4) : 0u));
        const int row0 = (int)(b * g.L + (int64_t)k * Bs);
        for (int j = 0; j < ntile; ++j) tma_load_3d(sm + xbuf + (uint32_t)j * 16384u, &xmap, 0, hd, row0 + 128 * j, &bar[2]);
        if (seed_h != nullptr) bulk_load(sm + L.raw, seed_h, (uint32_t)(kSsdP * N * 4), &bar[2]);
      }
    } else {
      issue_head_loads<N>(sm, L, p.x, tok, H, hd, ntile, seed_h, xbuf);
    }
  };
  // the first head's x and seed (the B tiles are no longer read)
  if (alive && h0 < h1) load_head(h0, L.x);
  // decay vectors of head hh into buffer `buf`: warp 0 the forward direction,
  // warp 1 the reverse one (each scans, then fills its column factors;
  // forward referenced to the column group's last token, reverse to its first)
  auto setup = [&](int hh, int buf) {
    float* v = vec0 + buf * 1536;
    if (w == 0)
      setup_dir<false>(s_dtf + hh, hg, Bs, __fmul_rn(s_prm[hh], kLog2e), v, v + 256, v + 512);
    else if (NOISY && w == 1)
      setup_dir<true>(s_dtr + hh, hg, Bs, __fmul_rn(s_prm[32 + hh], kLog2e), v + 768, v + 1024, v + 1280);
  };
  if (alive && h0 < h1) setup(0, 0);
  // mixing tile j of head hh into shared buffer mt: this warp's two 32-column
  // groups (0: no term, 1: factored decay, 2: diagonal block; uniform per warp)
  auto build = [&](int j, const float* v, unsigned char* mt) {
    const float af_t = v[tt];
    const float ar_t = NOISY ? v[768 + tt] : 0.f;
    const uint32_t colf = 128u * j, colr = 128u * (nf + j - i);
#pragma unroll 1
    for (int c = 0; c < 2; ++c) {
      const int cg = 2 * hf + c, sg = 4 * j + cg, s0 = 32 * sg;  // column group of the tile / block
      const int fm = j > i ? 0 : (sg < rg ? 1 : (sg == rg ? 2 : 0));
      const int rm = !NOISY || j < i ? 0 : (sg > rg ? 1 : (sg == rg ? 2 : 0));
      // pairs of columns in packed fp32 (FMUL2 / FFMA2); decay vectors read 4 at a time
      float2 o[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) o[e] = make_float2(0.f, 0.f);
      const float4* va = reinterpret_cast<const float4*>(v + s0);           // A2 * cumulative dt (forward)
      const float4* vw = reinterpret_cast<const float4*>(v + 256 + s0);     // dt (forward)
      const float4* vc = reinterpret_cast<const float4*>(v + 512 + s0);     // column factors (forward)
      if (fm != 0) {
        float gv[32];
        umma::tmem_ld32(lane_base + colf + 32u * cg, gv);
        if (fm == 1) {
          const float2 rf = f2(ex2(__fsub_rn(af_t, v[s0 + 31])));
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float4 c4 = vc[e];
            o[2 * e] = mul2(mul2(make_float2(gv[4 * e], gv[4 * e + 1]), make_float2(c4.x, c4.y)), rf);
            o[2 * e + 1] = mul2(mul2(make_float2(gv[4 * e + 2], gv[4 * e + 3]), make_float2(c4.z, c4.w)), rf);
          }
        } else {
          const float2 at = f2(af_t), neg = f2(-1.f);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float4 a4 = va[e], w4 = vw[e];
            const float2 d0 = mul2(ex2x2(fma2(make_float2(a4.x, a4.y), neg, at)), make_float2(w4.x, w4.y));
            const float2 d1 = mul2(ex2x2(fma2(make_float2(a4.z, a4.w), neg, at)), make_float2(w4.z, w4.w));
            const float2 p0 = mul2(make_float2(gv[4 * e], gv[4 * e + 1]), d0);
            const float2 p1 = mul2(make_float2(gv[4 * e + 2], gv[4 * e + 3]), d1);
            const int sc = s0 + 4 * e;  // columns sc..sc+3
            o[2 * e] = make_float2(sc <= tt ? p0.x : 0.f, sc + 1 <= tt ? p0.y : 0.f);
            o[2 * e + 1] = make_float2(sc + 2 <= tt ? p1.x : 0.f, sc + 3 <= tt ? p1.y : 0.f);
          }
        }
      }
      if (rm != 0) {
        float gv[32];
        umma::tmem_ld32(lane_base + colr + 32u * cg, gv);
        const float4* ra = reinterpret_cast<const float4*>(v + 768 + s0);   // A2 * cumulative dt (reverse)
        const float4* rw = reinterpret_cast<const float4*>(v + 1024 + s0);  // dt (reverse)
        const float4* rc = reinterpret_cast<const float4*>(v + 1280 + s0);  // column factors (reverse)
        if (rm == 1) {
          const float2 rf = f2(ex2(__fsub_rn(ar_t, v[768 + s0])));
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float4 c4 = rc[e];
            o[2 * e] = fma2(mul2(make_float2(gv[4 * e], gv[4 * e + 1]), make_float2(c4.x, c4.y)), rf, o[2 * e]);
            o[2 * e + 1] = fma2(mul2(make_float2(gv[4 * e + 2], gv[4 * e + 3]), make_float2(c4.z, c4.w)), rf,
                                o[2 * e + 1]);
          }
        } else {
          const float2 at = f2(ar_t), neg = f2(-1.f);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float4 a4 = ra[e], w4 = rw[e];
            const float2 d0 = mul2(ex2x2(fma2(make_float2(a4.x, a4.y), neg, at)), make_float2(w4.x, w4.y));
            const float2 d1 = mul2(ex2x2(fma2(make_float2(a4.z, a4.w), neg, at)), make_float2(w4.z, w4.w));
            const float2 p0 = mul2(make_float2(gv[4 * e], gv[4 * e + 1]), d0);
            const float2 p1 = mul2(make_float2(gv[4 * e + 2], gv[4 * e + 3]), d1);
            const int sc = s0 + 4 * e;
            o[2 * e] = add2(o[2 * e], make_float2(sc >= tt ? p0.x : 0.f, sc + 1 >= tt ? p0.y : 0.f));
            o[2 * e + 1] = add2(o[2 * e + 1], make_float2(sc + 2 >= tt ? p1.x : 0.f, sc + 3 >= tt ? p1.y : 0.f));
          }
        }
      }
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) {
        const int col = 32 * cg + 8 * ch;  // s inside the tile
        *reinterpret_cast<uint4*>(mt + (col >> 6) * kTile16 + sw128(row, (col & 63) >> 3)) =
            make_uint4(pack_bf16(o[ch * 4].x, o[ch * 4].y), pack_bf16(o[ch * 4 + 1].x, o[ch * 4 + 1].y),
                       pack_bf16(o[ch * 4 + 2].x, o[ch * 4 + 2].y), pack_bf16(o[ch * 4 + 3].x, o[ch * 4 + 3].y));
      }
    }
  };
  // MMAs of mixing tile j (and, first, the seed term) by thread 0
  auto issue = [&](int j, uint32_t xcur, bool seed_term) {
    umma::fence_after_sync();
    const uint32_t base = umma::smem_u32(sm);
    if (seed_term) {  // C^f . seed^T into columns 448..511
      constexpr uint32_t id = umma::idesc_bf16(128, 64, false, false);
      const uint64_t dc = umma::sdesc(base + L.cf, 16, 1024), dh = umma::sdesc(base + L.seed, 16, 1024),
                     dl = umma::sdesc(base + L.seed + 128u * N, 16, 1024);
#pragma unroll
      for (int kk = 0; kk < N / 16; ++kk) {
        const uint32_t offc = (kk >> 2) * kTile16 + (kk & 3) * 32u;
        const uint32_t offs = (kk >> 2) * 8192u + (kk & 3) * 32u;
        const uint64_t a = umma::sdesc_adv(dc, offc);
        umma::mma_bf16(tm + 448, a, umma::sdesc_adv(dh, offs), id, kk > 0);
        umma::mma_bf16(tm + 448, a, umma::sdesc_adv(dl, offs), id, true);
      }
    }
    const uint64_t dm = umma::sdesc(base + (j ? L.m1 : L.m0), 16, 1024),
                   dx = umma::sdesc(base + xcur + (uint32_t)j * 16384u, 1024, 1024);
    constexpr uint32_t id = umma::idesc_bf16(128, 64, false, true);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk)
      umma::mma_bf16(tm + 384, umma::sdesc_adv(dm, (kk >> 2) * kTile16 + (kk & 3) * 32u),
                     umma::sdesc_adv(dx, kk * 2048u), id, j > 0 || kk > 0);
  };
  for (int hh = 0; hh < hg && alive; ++hh) {
    const int h = h0 + hh;
    const uint32_t xcur = L.x + (hh & 1) * L.xsz;  // this head's x tiles
    const float* v = vec0 + (hh & 1) * 1536;       // this head's decay vectors
    if (p.tma) {  // head hh's loads complete phase hh of the load barrier
      if (!cta_wait(&bar[2], (uint32_t)(hh & 1), p.flag)) {
        alive = false;
        break;
      }
      ld_pending = false;
    } else {
      cp_async_wait_all();
    }
    __syncthreads();  // the head's x and raw seed have landed, its decay vectors are ready
    if (has_seed) {   // seed (fp32, staged in m1) -> bf16 high + low parts, K-major
      for (int c = t; c < kSsdP * N / 8; c += kScanThreads) {
        const int pr = c / (N / 8), ch = c % (N / 8);
        const float4 u0 = *reinterpret_cast<const float4*>(sm + L.raw + (pr * N + ch * 8) * 4);
        const float4 u1 = *reinterpret_cast<const float4*>(sm + L.raw + (pr * N + ch * 8 + 4) * 4);
        const float vv[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
        uint32_t wh[4], wl[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat162 hv = __floats2bfloat162_rn(vv[2 * e], vv[2 * e + 1]);
          wh[e] = *reinterpret_cast<const uint32_t*>(&hv);
          wl[e] = pack_bf16(__fsub_rn(vv[2 * e], __low2float(hv)), __fsub_rn(vv[2 * e + 1], __high2float(hv)));
        }
        const uint32_t off = (ch >> 3) * 8192u + sw128(pr, ch & 7);
        *reinterpret_cast<uint4*>(sm + L.seed + off) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
        *reinterpret_cast<uint4*>(sm + L.seed + 128u * N + off) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
      }
    }
    build(0, v, sm + L.m0);
    umma::fence_async_smem();
    umma::fence_before_sync();
    __syncthreads();
    // The issuing thread is held while the tensor pipe takes the MMAs, so it
    // is thread 128: warp 4 (rows 0..31, right column half) has the least
    // mixing work on a diagonal tile (nothing for a clean block's, one term
    // per column group for a noisy block's)
    if (t == kScanIssuer) {
      issue(0, xcur, has_seed);
      if (ntile == 1) umma::mma_commit(&bar[0]);
    }
    if (ntile > 1) {  // the second tile is built while the first one's MMAs run
      build(1, v, sm + L.m1);
      umma::fence_async_smem();
      umma::fence_before_sync();
      __syncthreads();
      if (t == kScanIssuer) {
        issue(1, xcur, false);
        umma::mma_commit(&bar[0]);
      }
    }
    if (hh + 1 < hg) setup(hh + 1, (hh + 1) & 1);  // under this head's MMAs
    if (!cta_wait(&bar[0], hh & 1, p.flag)) {
      alive = false;
      break;
    }
    umma::fence_after_sync();
    // the next head's loads run under this head's epilogue
    if (hh + 1 < hg) load_head(h + 1, L.x + ((hh + 1) & 1) * L.xsz);
    // --- epilogue: y = mixing term + decayed seed term + D x, bf16 out;
    // this warp's 32 channels of its token row
    {
      float ya[32], yo[32];
      if (has_seed)
        umma::tmem_ld32x2(lane_base + 384u + 32u * hf, ya, lane_base + 448u + 32u * hf, yo);
      else
        umma::tmem_ld32(lane_base + 384u + 32u * hf, ya);
      const float dec = has_seed ? ex2(v[tt]) : 0.f;
      const float Dd = NOISY ? __fadd_rn(s_prm[16 + hh], s_prm[48 + hh]) : s_prm[16 + hh];
      const int64_t off = (tok(tt) * H + h) * kSsdP + 32 * hf;
      const unsigned char* xr = sm + xcur + (uint32_t)i * 16384u;
      // bf16 output: the warp's 32 rows x 64 bytes go through a 2 KB block of
      // m0 (free until the next head's mixing tile; 16-byte chunks XOR-swizzled
      // by row pair) and are stored as 64-byte row segments, 8 rows per store
      unsigned char* yb = sm + L.m0 + w * 2048u;
      const int lr = row & 31;
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) {
        const uint4 xv = *reinterpret_cast<const uint4*>(xr + sw128(row, 4 * hf + ch));
        const __nv_bfloat16* xe = reinterpret_cast<const __nv_bfloat16*>(&xv);
        float o[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          float acc = ya[ch * 8 + e];
          if (has_seed) acc = __fmaf_rn(dec, yo[ch * 8 + e], acc);
          o[e] = __fmaf_rn(Dd, __bfloat162float(xe[e]), acc);
        }
        if (p.y32 != nullptr) {  // fp32 output (one direction of a two-pass layer)
          float4* d4 = reinterpret_cast<float4*>(p.y32 + off + ch * 8);
          d4[0] = make_float4(o[0], o[1], o[2], o[3]);
          d4[1] = make_float4(o[4], o[5], o[6], o[7]);
          continue;
        }
        if (p.y32_add != nullptr) {  // the other direction's fp32 output, added before rounding
          const float4* a4 = reinterpret_cast<const float4*>(p.y32_add + off + ch * 8);
          const float4 u0 = a4[0], u1 = a4[1];
          o[0] = __fadd_rn(u0.x, o[0]); o[1] = __fadd_rn(u0.y, o[1]); o[2] = __fadd_rn(u0.z, o[2]);
          o[3] = __fadd_rn(u0.w, o[3]); o[4] = __fadd_rn(u1.x, o[4]); o[5] = __fadd_rn(u1.y, o[5]);
          o[6] = __fadd_rn(u1.z, o[6]); o[7] = __fadd_rn(u1.w, o[7]);
        }
        *reinterpret_cast<uint4*>(yb + lr * 64 + 16 * (ch ^ ((lr >> 1) & 3))) =
            make_uint4(pack_bf16(o[0], o[1]), pack_bf16(o[2], o[3]), pack_bf16(o[4], o[5]), pack_bf16(o[6], o[7]));
      }
      if (p.y32 == nullptr) {
        __syncwarp();
        const int ch = lane & 3;
#pragma unroll
        for (int rr = 0; rr < 32; rr += 8) {
          const int r2 = rr + (lane >> 2), tr = i * kSsdT + 32 * q4 + r2;  // row of the warp, token of the block
          *reinterpret_cast<uint4*>(p.y + (tok(tr) * H + h) * kSsdP + 32 * hf + 8 * ch) =
              *reinterpret_cast<const uint4*>(yb + r2 * 64 + 16 * (ch ^ ((r2 >> 1) & 3)));
        }
      }
    }
    umma::fence_before_sync();
    __syncthreads();
    umma::fence_after_sync();
  }
  cp_async_wait_all();
  if (ld_pending) umma::bar_wait(&bar[2], ld_parity);  // after a give-up: the copies in flight, bounded
  umma::fence_before_sync();
  __syncthreads();
  if (t < 32) tmem_dealloc(tm, 512);
}

}  // namespace

namespace {

// Failure-detection check of the bounded waits: thread 0 initialises an
// mbarrier that nothing ever completes; every thread waits on it through the
// same path as the tensor-core kernels, with `polls` polls, so the wait gives
// up, sets the flag and the kernel returns normally.
__global__ void __launch_bounds__(128) k_ssd_wait_probe(int* flag, uint32_t polls) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) umma::bar_init(&bar, 1);
  __syncthreads();
  const bool ok = umma::bar_wait(&bar, 0, polls);
  if (__syncthreads_or(ok ? 0 : 1) && threadIdx.x == 0) atomicExch(flag, 1);
}

}  // namespace

cudaError_t launch_ssd_wait_probe(uint32_t polls, cudaStream_t s) {
  int* flag = ssd_wait_flag_ptr();
  if (flag == nullptr) return cudaErrorInvalidSymbol;
  k_ssd_wait_probe<<<1, 128, 0, s>>>(flag, polls);
  return cudaGetLastError();
}

int* ssd_wait_flag_ptr() {
  // device address of the flag, looked up once per device (the symbol names
  // a different address on each device)
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return nullptr;
  static std::atomic<int*> addr[256];
  int* a = addr[dev].load(std::memory_order_acquire);
  if (a != nullptr) return a;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_ssd_wait_flag) != cudaSuccess) return nullptr;
  addr[dev].store(static_cast<int*>(p), std::memory_order_release);
  return static_cast<int*>(p);
}

namespace {

template <typename K>
cudaError_t set_smem(K kernel, uint32_t bytes) {
  return set_smem_cached(reinterpret_cast<const void*>(kernel), (int)bytes, 100);
}

}  // namespace

cudaError_t launch_ssd_block_state(const SsdStateParams& p, cudaStream_t s) {
  const int64_t rows = p.g.Bt * p.g.nb;
  if (rows == 0 || p.g.H == 0) return cudaSuccess;
  const dim3 grid((unsigned)rows, (unsigned)((p.g.H + p.hg - 1) / p.hg));
  if (p.hg < 1 || p.hg > 8) return cudaErrorInvalidValue;
  const uint32_t bytes = StateSmem((int)p.g.Bs).total;
  cudaError_t e;
  if (p.g.N == 64) {
    if ((e = set_smem(k_ssd_block_state<64>, bytes)) != cudaSuccess) return e;
    k_ssd_block_state<64><<<grid, kStateThreads, bytes, s>>>(p);
  } else {
    if ((e = set_smem(k_ssd_block_state<128>, bytes)) != cudaSuccess) return e;
    k_ssd_block_state<128><<<grid, kStateThreads, bytes, s>>>(p);
  }
  return cudaGetLastError();
}

cudaError_t launch_ssd_state_pass(const SsdPassParams& p, cudaStream_t s) {
  const int64_t n = p.g.Bt * p.g.H * kSsdP * p.g.N;
  if (n == 0) return cudaSuccess;
  k_ssd_state_pass<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(p);
  return cudaGetLastError();
}

// The driver's tensor-map encoder, looked up once through the runtime (no
// link against the driver library); null if unavailable.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// Whether the launchers may use TMA at all (bdscan_ssd_set_tma): the
// cp.async path stays callable on hardware that has TMA, for its tests.
static std::atomic<int> g_tma_allowed{1};
void ssd_set_tma(bool on) { g_tma_allowed.store(on ? 1 : 0); }

bool ssd_tma_enabled() { return g_tma_allowed.load() != 0 && tensor_map_encoder() != nullptr; }

// x [rows][H][64] bf16 as a 3-D map with boxes of 64 channels x 1 head x 128
// tokens, 128-byte swizzle (the layout the MMA descriptors read).
bool encode_head_map(CUtensorMap* m, const __nv_bfloat16* x, int64_t rows, int H) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (enc == nullptr || g_tma_allowed.load() == 0 || rows >= ((int64_t)1 << 31) || ((uintptr_t)x & 15u) != 0)
    return false;
  const cuuint64_t dims[3] = {(cuuint64_t)kSsdP, (cuuint64_t)H, (cuuint64_t)rows};
  const cuuint64_t strides[2] = {(cuuint64_t)kSsdP * 2, (cuuint64_t)H * kSsdP * 2};  // bytes, dims 1 and 2
  const cuuint32_t box[3] = {(cuuint32_t)kSsdP, 1u, (cuuint32_t)kSsdT};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(x), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int N, bool NOISY>
cudaError_t scan_t(const SsdScanParams& p_in, cudaStream_t s) {
  const int64_t tiles = p_in.g.Bt * p_in.g.nb * p_in.g.m;
  if (tiles == 0 || p_in.g.H == 0) return cudaSuccess;
  if (p_in.hg < 1 || p_in.hg > kMaxHeadsPerCta) return cudaErrorInvalidValue;
  const ScanSmem L(N, p_in.g.m);
  cudaError_t e = set_smem(k_ssd_block_scan<N, NOISY>, L.total);
  if (e != cudaSuccess) return e;
  SsdScanParams p = p_in;
  CUtensorMap xmap;
  memset(&xmap, 0, sizeof(xmap));
  // streams read right to left keep the cp.async path (a box cannot reverse rows)
  p.tma = !p.rev && encode_head_map(&xmap, p.x, p.g.Bt * p.g.L, p.g.H) ? 1 : 0;
  const dim3 grid((unsigned)tiles, (unsigned)((p.g.H + p.hg - 1) / p.hg));
  k_ssd_block_scan<N, NOISY><<<grid, kScanThreads, L.total, s>>>(p, xmap);
  return cudaGetLastError();
}

cudaError_t launch_ssd_block_scan(bool noisy, const SsdScanParams& p, cudaStream_t s) {
  if (p.g.N == 64) return noisy ? scan_t<64, true>(p, s) : scan_t<64, false>(p, s);
  return noisy ? scan_t<128, true>(p, s) : scan_t<128, false>(p, s);
}

}  // namespace bds
