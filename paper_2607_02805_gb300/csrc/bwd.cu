// bwd.cu -- backward-side kernels of libbdscan (sm_103a) between and after
// the two TMEM kernels: the exact carry of the clean adjoint across chunks,
// the deterministic reductions, and the backward chunk count. The derivative
// and the kernel sequence are described in bwd_common.cuh.
#include "bwd_common.cuh"

namespace bds {

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
  // debug build: the last seed gradient this thread reads (no barrier follows)
  if (!dguard(kSiteBwdCarry, ((b * g.nb + g.nb - 1) * g.D + d) * N + n, g.Bt * g.nb * g.D * N)) return;
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
// Deterministic reductions
// ---------------------------------------------------------------------------
// One thread per 4 consecutive state indices of one row of one tensor: the
// channel-group partials are summed in group order (16-byte loads).
template <typename TO, int N>
__global__ void __launch_bounds__(256) k_reduce_tok(const BwdParams p) {
  const Geo& g = p.g;
  const int64_t rows = g.Bt * g.L;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= 6 * rows * (N / 4)) return;
  const int n = (int)(idx % (N / 4)) * 4;
  const int64_t row = idx / (N / 4);
  const int tensor = (int)(row / rows);
  const int64_t bt = row - (int64_t)tensor * rows;
  // debug build: the last channel-group partial this thread reads (no barrier follows)
  if (!dguard(kSiteReduceTok, (row * g.G + g.G - 1) * N + n + 3, 6 * rows * g.G * N)) return;
  const float* src = p.part_tok + row * g.G * N + n;
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int gi = 0; gi < g.G; ++gi) {
    const float4 v = *reinterpret_cast<const float4*>(src + (int64_t)gi * N);
    s.x += v.x;
    s.y += v.y;
    s.z += v.z;
    s.w += v.w;
  }
  void* dst = tensor == 0 ? p.dBc : tensor == 1 ? p.dCc : tensor == 2 ? p.dBf : tensor == 3 ? p.dCf
            : tensor == 4 ? p.dBr : p.dCr;
  TO* d = reinterpret_cast<TO*>(dst) + bt * N + n;
  d[0] = to_out<TO>(s.x);
  d[1] = to_out<TO>(s.y);
  d[2] = to_out<TO>(s.z);
  d[3] = to_out<TO>(s.w);
}

// One CTA sums 128 columns (32 lanes x 4) of the per-chunk partials: 16
// slices of threads each add every 16th chunk (in order), then the slices
// are added in order.
constexpr int kParSlices = 16;
template <int N>
__global__ void __launch_bounds__(32 * kParSlices) k_reduce_par(const BwdParams p) {
  // kParSlices slices (warps) of the chunk partials; each lane sums 4 adjacent columns
  __shared__ float4 part[3][kParSlices][32];
  const Geo& g = p.g;
  const int64_t U = g.Bt * g.nc;
  const int64_t DN = g.D * N;
  const int lane = threadIdx.x & 31, slice = threadIdx.x >> 5;
  const int64_t col = ((int64_t)blockIdx.x * 32 + lane) * 4;  // D and D*N are multiples of 4
  // debug build: the CTA's first column lies inside the parameter columns
  if (!dguard(kSiteReducePar, (int64_t)blockIdx.x * 128, DN + g.D)) return;
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
    for (int64_t u = slice; u < U; u += kParSlices) {
      acc(s0, a0 + u * DN);
      acc(s1, a1 + u * DN);
      acc(s2, a2 + u * DN);
    }
  } else if (col < DN + g.D) {
    const int64_t d = col - DN;
#pragma unroll 4
    for (int64_t u = slice; u < U; u += kParSlices) {
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
    for (int k = 1; k < kParSlices; ++k) {
      const float4 v0 = part[0][k][lane], v1 = part[1][k][lane], v2 = part[2][k][lane];
      t0 = make_float4(t0.x + v0.x, t0.y + v0.y, t0.z + v0.z, t0.w + v0.w);
      t1 = make_float4(t1.x + v1.x, t1.y + v1.y, t1.z + v1.z, t1.w + v1.w);
      t2 = make_float4(t2.x + v2.x, t2.y + v2.y, t2.z + v2.z, t2.w + v2.w);
    }
    // debug build: a non-finite parameter gradient
    if (BDSCAN_DEBUG) {
      const float v[12] = {t0.x, t0.y, t0.z, t0.w, t1.x, t1.y, t1.z, t1.w, t2.x, t2.y, t2.z, t2.w};
#pragma unroll
      for (int q = 0; q < 12; ++q) dfinite(kSiteReducePar, v[q], col + (q & 3));
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

cudaError_t launch_bwd_carry(int N, const BwdParams& p, cudaStream_t s) {
  const int64_t total = p.g.Bt * p.g.D * N;
  if (total == 0) return cudaSuccess;
  BDS_DISPATCH_N(N, k_bwd_carry<NN><<<(unsigned)((total + 255) / 256), 256, 0, s>>>(p); return cudaGetLastError();)
}

cudaError_t launch_bwd_reduce_tok(int dt, int N, const BwdParams& p, cudaStream_t s) {
  const int64_t ntok = 6 * p.g.Bt * p.g.L * (N / 4);
  if (ntok == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)((ntok + 255) / 256);
  if (dt == 1) {
    BDS_DISPATCH_N(N, k_reduce_tok<bf16, NN><<<blocks, 256, 0, s>>>(p); return cudaGetLastError();)
  }
  BDS_DISPATCH_N(N, k_reduce_tok<float, NN><<<blocks, 256, 0, s>>>(p); return cudaGetLastError();)
}

cudaError_t launch_bwd_reduce_par(int N, const BwdParams& p, cudaStream_t s) {
  const int64_t npar4 = (p.g.D * N + p.g.D) / 4;  // float4 columns
  BDS_DISPATCH_N(N, k_reduce_par<NN><<<(unsigned)((npar4 + 31) / 32), 32 * kParSlices, 0, s>>>(p);
                 return cudaGetLastError();)
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
  const int pn = bwd_noisy_per_sm(dt, N, Bs, dev), pc = bwd_clean_per_sm(dt, N, Bs, dev);
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
