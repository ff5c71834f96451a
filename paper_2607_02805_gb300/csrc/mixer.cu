// mixer.cu -- the steps either side of the scan in a Mamba mixer (see
// include/bdscan_mixer.h): the width-4 causal depthwise convolution with
// SiLU (its last three inputs are part of the cache, Sec. 4.1 eq. cache-c4),
// the step size softplus(dt_raw + bias), and the SiLU-gated output; forward,
// backward, cache build and cached active block.
//
// These steps are elementwise per (token, channel), against the scan's work
// per (token, channel, state), and memory-bound: each runs as one fused pass
// over the tensors (convolution, SiLU and softplus together; gate and its
// derivative together) around the scan kernels of the library, which run in
// fp32 on intermediates kept in the workspace. The channel sums of the
// parameter gradients (taps, biases) are fixed-order two-level reductions,
// so results are deterministic.
#include <cstdio>
#include <cstring>

#include "bdscan_mixer.h"
#include "device.cuh"
#include "params.h"

namespace bds {
namespace {

constexpr int kW = 4;           // convolution width
constexpr int kParSplit = 256;  // token slices of the parameter-gradient reduction

// The logistic function and softplus on the fast hardware paths (__expf,
// __logf, __fdividef): relative errors of order 1e-6, far inside the
// tolerance of the path, and the same functions serve every entry point, so
// the cache paths stay bit-identical to the all-block ones.
__device__ __forceinline__ float sigm(float z) { return __fdividef(1.f, __fadd_rn(1.f, __expf(-z))); }
__device__ __forceinline__ float silu(float z) { return __fmul_rn(z, sigm(z)); }
// d SiLU / dz = s (1 + z (1 - s))
__device__ __forceinline__ float dsilu(float z) {
  const float s = sigm(z);
  return __fmul_rn(s, __fmaf_rn(z, __fsub_rn(1.f, s), 1.f));
}
__device__ __forceinline__ float softplus(float z) {
  return __fadd_rn(fmaxf(z, 0.f), __logf(__fadd_rn(1.f, __expf(-fabsf(z)))));
}

// Arguments of the input-side kernels. Token-by-channel tensors [Bt][L][D].
template <typename T>
struct MixIn {
  int64_t Bt, L, D, Bs;
  const T *xr_c, *dtr_c, *xr_n, *dtr_f, *dtr_r;
  const float *w, *cb, *bias_f, *bias_r;
  const float* conv_init;  // [Bt][3][D] or null
};

// Raw clean input at position u of batch row b, channel d (positions before 0
// read the initial convolution state).
template <typename T>
__device__ __forceinline__ float raw_c(const MixIn<T>& a, int64_t b, int64_t u, int64_t d) {
  if (u >= 0) return cvt(a.xr_c[(b * a.L + u) * a.D + d]);
  return a.conv_init != nullptr ? a.conv_init[(b * (kW - 1) + (kW - 1) + u) * a.D + d] : 0.f;
}
// Raw input seen by a noisy token of the block starting at k0, at position u:
// the noisy stream inside the block, the clean stream before it.
template <typename T>
__device__ __forceinline__ float raw_n(const MixIn<T>& a, int64_t b, int64_t u, int64_t k0, int64_t d) {
  return u >= k0 ? cvt(a.xr_n[(b * a.L + u) * a.D + d]) : raw_c(a, b, u, d);
}
template <typename T>
__device__ __forceinline__ float pre_c(const MixIn<T>& a, int64_t b, int64_t t, int64_t d) {
  float pre = a.cb[d];
#pragma unroll
  for (int j = 0; j < kW; ++j) pre = __fmaf_rn(a.w[d * kW + j], raw_c(a, b, t - (kW - 1) + j, d), pre);
  return pre;
}
template <typename T>
__device__ __forceinline__ float pre_n(const MixIn<T>& a, int64_t b, int64_t t, int64_t d) {
  const int64_t k0 = t - t % a.Bs;
  float pre = a.cb[d];
#pragma unroll
  for (int j = 0; j < kW; ++j) pre = __fmaf_rn(a.w[d * kW + j], raw_n(a, b, t - (kW - 1) + j, k0, d), pre);
  return pre;
}

// Vector access: V = 16 / sizeof(T) consecutive channels per thread (8 for
// bf16, 4 for fp32; d_inner is a multiple of V), so every token-by-channel
// load is 16 bytes per thread.
template <typename T>
struct Vec {
  static constexpr int V = 16 / (int)sizeof(T);
};
__device__ __forceinline__ void ld16(const bf16* p, float (&v)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 f = __bfloat1622float2(h[e]);
    v[2 * e] = f.x;
    v[2 * e + 1] = f.y;
  }
}
__device__ __forceinline__ void ld16(const float* p, float (&v)[4]) {
  const float4 u = *reinterpret_cast<const float4*>(p);
  v[0] = u.x;
  v[1] = u.y;
  v[2] = u.z;
  v[3] = u.w;
}
template <int V>
__device__ __forceinline__ void ldf(const float* p, float (&v)[V]) {
#pragma unroll
  for (int q = 0; q < V / 4; ++q) {
    const float4 u = *reinterpret_cast<const float4*>(p + 4 * q);
    v[4 * q] = u.x;
    v[4 * q + 1] = u.y;
    v[4 * q + 2] = u.z;
    v[4 * q + 3] = u.w;
  }
}
template <int V>
__device__ __forceinline__ void stv(float* p, const float (&v)[V]) {
#pragma unroll
  for (int q = 0; q < V / 4; ++q)
    *reinterpret_cast<float4*>(p + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}
template <int V>
__device__ __forceinline__ void stv(bf16* p, const float (&v)[V]) {
#pragma unroll
  for (int q = 0; q < V / 4; ++q) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(v[4 * q], v[4 * q + 1]);
    const __nv_bfloat162 c = __floats2bfloat162_rn(v[4 * q + 2], v[4 * q + 3]);
    *reinterpret_cast<uint2*>(p + 4 * q) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&c));
  }
}

// Raw inputs of window tap j (position u) for V channels from d: the clean
// stream, or the initial convolution state before token 0. u is the same for
// the whole CTA (one token row per CTA), so the branches are uniform.
template <typename T, int V>
__device__ __forceinline__ void raw_cv(const MixIn<T>& a, int64_t b, int64_t u, int64_t d, float (&r)[V]) {
  if (u >= 0) {
    ld16(a.xr_c + (b * a.L + u) * a.D + d, r);
  } else if (a.conv_init != nullptr) {
    ldf<V>(a.conv_init + (b * (kW - 1) + (kW - 1) + u) * a.D + d, r);
  } else {
#pragma unroll
    for (int v = 0; v < V; ++v) r[v] = 0.f;
  }
}
// The same for a noisy token of the block starting at k0: the noisy stream
// inside the block, the clean one (or the initial state) before it.
template <typename T, int V>
__device__ __forceinline__ void raw_nv(const MixIn<T>& a, int64_t b, int64_t u, int64_t k0, int64_t d, float (&r)[V]) {
  if (u >= k0)
    ld16(a.xr_n + (b * a.L + u) * a.D + d, r);
  else
    raw_cv<T, V>(a, b, u, d, r);
}
// Scan inputs in fp32: x = SiLU(conv), dt = softplus(dt_raw + bias), for the
// clean stream (if x_c) and the noisy stream (if x_n).
// Grid of the token-by-channel kernels: one CTA row per token (blockIdx.x,
// batch row b = token / L), 256 channels per CTA (blockIdx.y); no per-element
// division.
template <typename T>
__global__ void __launch_bounds__(256) k_mix_prep(const MixIn<T> a, float* x_c, float* dt_c, float* x_n, float* dt_f,
                                                  float* dt_r) {
  const int64_t d = (int64_t)blockIdx.y * 256 + threadIdx.x;
  if (d >= a.D) return;
  const int64_t bt = blockIdx.x, b = bt / a.L, t = bt - b * a.L, i = bt * a.D + d;
  if (x_c != nullptr) {
    x_c[i] = silu(pre_c(a, b, t, d));
    dt_c[i] = softplus(__fadd_rn(cvt(a.dtr_c[i]), a.bias_f[d]));
  }
  if (x_n != nullptr) {
    x_n[i] = silu(pre_n(a, b, t, d));
    dt_f[i] = softplus(__fadd_rn(cvt(a.dtr_f[i]), a.bias_f[d]));
    dt_r[i] = softplus(__fadd_rn(cvt(a.dtr_r[i]), a.bias_r[d]));
  }
}

// Backward through SiLU and softplus, in place on the scan's fp32 gradients:
// gx <- gx * SiLU'(pre), gdt <- gdt * sigmoid(dt_raw + bias); the step-size
// gradients also go out in the output type.
template <typename T, typename TO>
__global__ void __launch_bounds__(256) k_mix_dpre(const MixIn<T> a, float* gx_c, float* gdt_c, float* gx_n,
                                                  float* gdt_f, float* gdt_r, TO* ddtr_c, TO* ddtr_f, TO* ddtr_r) {
  const int64_t d = (int64_t)blockIdx.y * 256 + threadIdx.x;
  if (d >= a.D) return;
  const int64_t bt = blockIdx.x, b = bt / a.L, t = bt - b * a.L, i = bt * a.D + d;
  gx_c[i] = __fmul_rn(gx_c[i], dsilu(pre_c(a, b, t, d)));
  gx_n[i] = __fmul_rn(gx_n[i], dsilu(pre_n(a, b, t, d)));
  const float vc = __fmul_rn(gdt_c[i], sigm(__fadd_rn(cvt(a.dtr_c[i]), a.bias_f[d])));
  const float vf = __fmul_rn(gdt_f[i], sigm(__fadd_rn(cvt(a.dtr_f[i]), a.bias_f[d])));
  const float vr = __fmul_rn(gdt_r[i], sigm(__fadd_rn(cvt(a.dtr_r[i]), a.bias_r[d])));
  gdt_c[i] = vc;
  gdt_f[i] = vf;
  gdt_r[i] = vr;
  ddtr_c[i] = to_out<TO>(vc);
  ddtr_f[i] = to_out<TO>(vf);
  ddtr_r[i] = to_out<TO>(vr);
}

// Gradients of the raw inputs from the pre-activation gradients (the
// convolution's transpose): raw position u feeds tap j of token u + 3 - j; a
// noisy token's taps before its block feed the clean stream. V channels per
// thread (V = 16 / sizeof(TI), TI the input type).
template <typename TO, int V>
__global__ void __launch_bounds__(256) k_mix_dxr(int64_t Bt, int64_t L, int64_t D, int64_t Bs, const float* w,
                                                 const float* gp_c, const float* gp_n, TO* dxr_c, TO* dxr_n) {
  const int64_t d = ((int64_t)blockIdx.y * 256 + threadIdx.x) * V;
  if (d >= D) return;
  const int64_t bt = blockIdx.x, b = bt / L, u = bt - b * L, i = bt * D + d;
  float wv[kW * V], ac[V], an[V];
  ldf<kW * V>(w + d * kW, wv);
#pragma unroll
  for (int v = 0; v < V; ++v) ac[v] = an[v] = 0.f;
#pragma unroll
  for (int j = 0; j < kW; ++j) {
    const int64_t t = u + (kW - 1) - j;
    if (t >= L) continue;
    const int64_t o = (b * L + t) * D + d;
    float pc[V], pn[V];
    ldf<V>(gp_c + o, pc);
    ldf<V>(gp_n + o, pn);
    const bool inside = u >= t - t % Bs;  // the same block as the consuming noisy token
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float wj = wv[v * kW + j];
      ac[v] = __fmaf_rn(wj, pc[v], ac[v]);
      if (inside)
        an[v] = __fmaf_rn(wj, pn[v], an[v]);
      else
        ac[v] = __fmaf_rn(wj, pn[v], ac[v]);
    }
  }
  stv<V>(dxr_c + i, ac);
  stv<V>(dxr_n + i, an);
}

// Partial sums of the parameter gradients over a slice of the token rows:
// part[slice][v][d] for v = tap 0..3, conv bias, dt_bias_f, dt_bias_r; V
// channels per thread.
template <typename T>
__global__ void __launch_bounds__(128) k_mix_par_part(const MixIn<T> a, const float* gp_c, const float* gp_n,
                                                      const float* gdt_c, const float* gdt_f, const float* gdt_r,
                                                      float* part) {
  constexpr int V = Vec<T>::V;
  const int64_t d = ((int64_t)blockIdx.x * 128 + threadIdx.x) * V;
  const int slice = blockIdx.y;
  if (d >= a.D) return;
  float s[kW + 3][V];
#pragma unroll
  for (int q = 0; q < kW + 3; ++q)
#pragma unroll
    for (int v = 0; v < V; ++v) s[q][v] = 0.f;
  int64_t b = slice / a.L, t = slice - b * a.L;  // batch row and token of `row`, stepped without division
  for (int64_t row = slice; row < a.Bt * a.L; row += kParSplit) {
    const int64_t o = row * a.D + d, k0 = t - t % a.Bs;
    float pc[V], pn[V], g1[V], g2[V], g3[V];
    ldf<V>(gp_c + o, pc);
    ldf<V>(gp_n + o, pn);
    ldf<V>(gdt_c + o, g1);
    ldf<V>(gdt_f + o, g2);
    ldf<V>(gdt_r + o, g3);
#pragma unroll
    for (int j = 0; j < kW; ++j) {
      const int64_t u = t - (kW - 1) + j;
      float rc[V], rn[V];
      raw_cv<T, V>(a, b, u, d, rc);
      raw_nv<T, V>(a, b, u, k0, d, rn);
#pragma unroll
      for (int v = 0; v < V; ++v) {
        s[j][v] = __fmaf_rn(pc[v], rc[v], s[j][v]);
        s[j][v] = __fmaf_rn(pn[v], rn[v], s[j][v]);
      }
    }
#pragma unroll
    for (int v = 0; v < V; ++v) {
      s[kW][v] = __fadd_rn(s[kW][v], __fadd_rn(pc[v], pn[v]));
      s[kW + 1][v] = __fadd_rn(s[kW + 1][v], __fadd_rn(g1[v], g2[v]));
      s[kW + 2][v] = __fadd_rn(s[kW + 2][v], g3[v]);
    }
    t += kParSplit;
    while (t >= a.L) {
      t -= a.L;
      ++b;
    }
  }
#pragma unroll
  for (int q = 0; q < kW + 3; ++q) stv<V>(part + ((int64_t)slice * (kW + 3) + q) * a.D + d, s[q]);
}

// The slices summed in order: dconv_w [D][4], dconv_b, ddt_bias_f, ddt_bias_r [D].
__global__ void __launch_bounds__(256) k_mix_par_red(int64_t D, const float* part, float* dw, float* db, float* dbf,
                                                     float* dbr) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= D * (kW + 3)) return;
  const int v = (int)(i / D);
  const int64_t d = i % D;
  float s = 0.f;
  for (int sl = 0; sl < kParSplit; ++sl) s = __fadd_rn(s, part[((int64_t)sl * (kW + 3) + v) * D + d]);
  if (v < kW)
    dw[d * kW + v] = s;
  else if (v == kW)
    db[d] = s;
  else if (v == kW + 1)
    dbf[d] = s;
  else
    dbr[d] = s;
}

// out = y * SiLU(z), V elements per thread.
template <typename T, typename TO>
__global__ void __launch_bounds__(256) k_mix_gate(int64_t n, const float* y, const T* z, TO* out) {
  constexpr int V = Vec<T>::V;
  const int64_t i = ((int64_t)blockIdx.x * 256 + threadIdx.x) * V;
  if (i >= n) return;
  float yv[V], zv[V];
  ldf<V>(y + i, yv);
  ld16(z + i, zv);
#pragma unroll
  for (int v = 0; v < V; ++v) yv[v] = __fmul_rn(yv[v], silu(zv[v]));
  stv<V>(out + i, yv);
}

// The gate's backward: dy = dout * SiLU(z), dz = dout * y * SiLU'(z) (zero
// without dout), V elements per thread.
template <typename T, typename TO>
__global__ void __launch_bounds__(256) k_mix_gate_bwd(int64_t n, const float* y, const T* z, const T* dout, float* dy,
                                                      TO* dz) {
  constexpr int V = Vec<T>::V;
  const int64_t i = ((int64_t)blockIdx.x * 256 + threadIdx.x) * V;
  if (i >= n) return;
  float yv[V], zv[V], gv[V], a[V], c[V];
  ldf<V>(y + i, yv);
  ld16(z + i, zv);
  if (dout != nullptr) {
    ld16(dout + i, gv);
  } else {
#pragma unroll
    for (int v = 0; v < V; ++v) gv[v] = 0.f;
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    a[v] = __fmul_rn(gv[v], silu(zv[v]));
    c[v] = __fmul_rn(__fmul_rn(gv[v], yv[v]), dsilu(zv[v]));
  }
  stv<V>(dy + i, a);
  stv<V>(dz + i, c);
}

// Element type conversion (B, C to fp32 for the scan; their gradients back).
template <typename TI, typename TO>
__global__ void __launch_bounds__(256) k_mix_cvt(int64_t n, const TI* src, TO* dst) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i < n) dst[i] = to_out<TO>(cvt(src[i]));
}

// Convolution part of the cache: the raw clean inputs of the three tokens
// before each emitted boundary (every block end, or the end of the stream).
template <typename T>
__global__ void __launch_bounds__(256) k_mix_conv_states(const MixIn<T> a, int emit_all, float* cs) {
  const int64_t nS = emit_all ? a.L / a.Bs : 1;
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= a.Bt * nS * (kW - 1) * a.D) return;
  const int64_t d = i % a.D, r = i / a.D;
  const int q = (int)(r % (kW - 1));
  const int64_t k = (r / (kW - 1)) % nS, b = r / ((kW - 1) * nS);
  const int64_t end = emit_all ? (k + 1) * a.Bs : a.L;
  cs[i] = raw_c(a, b, end - (kW - 1) + q, d);
}

}  // namespace

// ---------------------------------------------------------------------------
// entry points
// ---------------------------------------------------------------------------
namespace {

size_t al(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace regions (byte offsets): fp32 scan inputs x_c, dt_c, x_n, dt_f,
// dt_r; fp32 B_c, C_c, B_f, C_f, B_r, C_r; fp32 scan outputs y_c, y_n; the
// scan's workspace. The backward adds the recomputed boundary states, the
// gate's fp32 gradients dy_c, dy_n, the scan's fp32 gradients (x, dt of the
// five streams, then B, C) and its workspace, and the parameter partials.
struct MixWs {
  size_t x[5], bc[6], y[2], scan, fwd_total;
  size_t states, dy[2], gx[5], gbc[6], bws, part, bwd_total;
};
MixWs mix_ws(const Geo& g, int N) {
  MixWs w;
  const size_t td = al((size_t)g.Bt * g.L * g.D * 4), tn = al((size_t)g.Bt * g.L * N * 4);
  size_t o = 0;
  for (int i = 0; i < 5; ++i, o += td) w.x[i] = o;
  for (int i = 0; i < 6; ++i, o += tn) w.bc[i] = o;
  for (int i = 0; i < 2; ++i, o += td) w.y[i] = o;
  w.scan = o;
  o += al(api_fwd_workspace(g, N));
  w.fwd_total = o;
  w.states = o;
  o += al((size_t)g.Bt * g.nb * g.D * N * 4);
  for (int i = 0; i < 2; ++i, o += td) w.dy[i] = o;
  for (int i = 0; i < 5; ++i, o += td) w.gx[i] = o;
  for (int i = 0; i < 6; ++i, o += tn) w.gbc[i] = o;
  w.bws = o;
  o += al(api_bwd_workspace(g, N));
  w.part = o;
  o += al((size_t)kParSplit * (kW + 3) * g.D * 4);
  w.bwd_total = o;
  return w;
}

bool a16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int bad_arg(const char* fn, const char* what) {
  char m[256];
  snprintf(m, sizeof(m), "%s: %s", fn, what);
  return api_fail(BDSCAN_ERR_ARG, m);
}
int cuda_err(const char* fn, cudaError_t e) {
  char m[256];
  snprintf(m, sizeof(m), "%s: %s", fn, cudaGetErrorString(e));
  return api_fail(BDSCAN_ERR_CUDA, m);
}

#define MIX_REQ(ptr, name) \
  if ((ptr) == nullptr || !a16(ptr)) return bad_arg(fn, name " is NULL or not 16-byte aligned")
#define MIX_OPT(ptr, name) \
  if ((ptr) != nullptr && !a16(ptr)) return bad_arg(fn, name " is not 16-byte aligned")

int check_mparams(const bdscan_mixer_params* m, const char* fn) {
  if (m == nullptr) return bad_arg(fn, "mparams is NULL");
  MIX_REQ(m->conv_w, "mparams.conv_w");
  MIX_REQ(m->conv_b, "mparams.conv_b");
  MIX_REQ(m->dt_bias_f, "mparams.dt_bias_f");
  MIX_REQ(m->dt_bias_r, "mparams.dt_bias_r");
  return BDSCAN_OK;
}

unsigned blocks_of(int64_t n) { return (unsigned)((n + 255) / 256); }
// one CTA row per token, 256 threads of V channels per CTA
dim3 rows_grid(const Geo& g, int V) {
  const int64_t span = 256 * (int64_t)V;
  return dim3((unsigned)(g.Bt * g.L), (unsigned)((g.D + span - 1) / span));
}
template <typename T>
unsigned vec_blocks(int64_t n) {
  constexpr int64_t span = 256 * Vec<T>::V;
  return (unsigned)((n + span - 1) / span);
}

template <typename T>
MixIn<T> mix_in(const Geo& g, const bdscan_clean* c, const bdscan_noisy* n, const bdscan_mixer_params* m,
                const float* conv_init) {
  MixIn<T> a;
  memset(&a, 0, sizeof(a));
  a.Bt = g.Bt;
  a.L = g.L;
  a.D = g.D;
  a.Bs = g.Bs;
  if (c != nullptr) {
    a.xr_c = (const T*)c->x;
    a.dtr_c = (const T*)c->dt;
  }
  if (n != nullptr) {
    a.xr_n = (const T*)n->x;
    a.dtr_f = (const T*)n->dt_f;
    a.dtr_r = (const T*)n->dt_r;
  }
  a.w = m->conv_w;
  a.cb = m->conv_b;
  a.bias_f = m->dt_bias_f;
  a.bias_r = m->dt_bias_r;
  a.conv_init = conv_init;
  return a;
}

// B and C of the given streams converted to fp32 into the workspace slots.
template <typename T>
cudaError_t to_f32(const void* const* src, const size_t* slot, int count, char* ws, int64_t n, cudaStream_t s) {
  cudaError_t e = cudaSuccess;
  for (int i = 0; i < count && e == cudaSuccess; ++i) {
    k_mix_cvt<T, float><<<blocks_of(n), 256, 0, s>>>(n, (const T*)src[i], (float*)(ws + slot[i]));
    e = api_launched(cudaGetLastError(), s);
  }
  return e;
}

// The forward of both streams up to the scan outputs: prep, B/C to fp32, the
// all-block scan in fp32 (states into `states`).
template <typename T>
cudaError_t mix_forward_core(const Geo& g, int N, const bdscan_clean* cl, const bdscan_noisy* nz,
                             const bdscan_params* pr, const bdscan_mixer_params* mp, float* states, char* ws,
                             const MixWs& w, cudaStream_t s) {
  const MixIn<T> a = mix_in<T>(g, cl, nz, mp, nullptr);
  const int64_t nn = g.Bt * g.L * N;
  float* X[5];
  for (int i = 0; i < 5; ++i) X[i] = (float*)(ws + w.x[i]);
  k_mix_prep<T><<<rows_grid(g, 1), 256, 0, s>>>(a, X[0], X[1], X[2], X[3], X[4]);
  cudaError_t e = api_launched(cudaGetLastError(), s);
  const void* bc[6] = {cl->B, cl->C, nz->B_f, nz->C_f, nz->B_r, nz->C_r};
  if (e == cudaSuccess) e = to_f32<T>(bc, w.bc, 6, ws, nn, s);
  if (e != cudaSuccess) return e;
  FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = g;
  p.xc = X[0];
  p.dtc = X[1];
  p.Bc = ws + w.bc[0];
  p.Cc = ws + w.bc[1];
  p.xn = X[2];
  p.dtf = X[3];
  p.Bf = ws + w.bc[2];
  p.Cf = ws + w.bc[3];
  p.dtr = X[4];
  p.Br = ws + w.bc[4];
  p.Cr = ws + w.bc[5];
  p.Af = pr->A_f;
  p.Df = pr->D_f;
  p.Ar = pr->A_r;
  p.Dr = pr->D_r;
  p.yc = ws + w.y[0];
  p.yn = ws + w.y[1];
  p.states = states;
  return api_run_forward(0, N, p, ws + w.scan, s);
}

template <typename T, typename TO>
cudaError_t gate(int64_t n, const char* ws, size_t yslot, const void* z, void* out, cudaStream_t s) {
  k_mix_gate<T, TO><<<vec_blocks<T>(n), 256, 0, s>>>(n, (const float*)(ws + yslot), (const T*)z, (TO*)out);
  return api_launched(cudaGetLastError(), s);
}

template <typename T, typename TO>
cudaError_t mix_forward_t(const Geo& g, int N, const bdscan_clean* cl, const void* z_c, const bdscan_noisy* nz,
                          const void* z_n, const bdscan_params* pr, const bdscan_mixer_params* mp, void* out_c,
                          void* out_n, float* states, char* ws, cudaStream_t s) {
  const MixWs w = mix_ws(g, N);
  cudaError_t e = mix_forward_core<T>(g, N, cl, nz, pr, mp, states, ws, w, s);
  const int64_t n = g.Bt * g.L * g.D;
  if (e == cudaSuccess) e = gate<T, TO>(n, ws, w.y[0], z_c, out_c, s);
  if (e == cudaSuccess) e = gate<T, TO>(n, ws, w.y[1], z_n, out_n, s);
  return e;
}

template <typename T, typename TO>
cudaError_t mix_backward_t(const Geo& g, int N, const bdscan_clean* cl, const void* z_c, const bdscan_noisy* nz,
                           const void* z_n, const bdscan_params* pr, const bdscan_mixer_params* mp,
                           const void* dout_c, const void* dout_n, const float* dstates,
                           const bdscan_clean_grads* gc, void* dz_c, const bdscan_noisy_grads* gn, void* dz_n,
                           const bdscan_param_grads* gp, const bdscan_mixer_grads* gm, char* ws, cudaStream_t s) {
  const MixWs w = mix_ws(g, N);
  float* states = (float*)(ws + w.states);
  // recompute the forward's scan inputs, outputs and boundary states
  cudaError_t e = mix_forward_core<T>(g, N, cl, nz, pr, mp, states, ws, w, s);
  if (e != cudaSuccess) return e;
  const int64_t n = g.Bt * g.L * g.D, nn = g.Bt * g.L * N;
  float* dy[2] = {(float*)(ws + w.dy[0]), (float*)(ws + w.dy[1])};
  k_mix_gate_bwd<T, TO><<<vec_blocks<T>(n), 256, 0, s>>>(n, (const float*)(ws + w.y[0]), (const T*)z_c, (const T*)dout_c,
                                                     dy[0], (TO*)dz_c);
  e = api_launched(cudaGetLastError(), s);
  if (e != cudaSuccess) return e;
  k_mix_gate_bwd<T, TO><<<vec_blocks<T>(n), 256, 0, s>>>(n, (const float*)(ws + w.y[1]), (const T*)z_n, (const T*)dout_n,
                                                     dy[1], (TO*)dz_n);
  e = api_launched(cudaGetLastError(), s);
  if (e != cudaSuccess) return e;
  float* G[5];
  for (int i = 0; i < 5; ++i) G[i] = (float*)(ws + w.gx[i]);
  BwdParams q;
  memset(&q, 0, sizeof(q));
  q.g = g;
  q.xc = ws + w.x[0];
  q.dtc = ws + w.x[1];
  q.Bc = ws + w.bc[0];
  q.Cc = ws + w.bc[1];
  q.xn = ws + w.x[2];
  q.dtf = ws + w.x[3];
  q.Bf = ws + w.bc[2];
  q.Cf = ws + w.bc[3];
  q.dtr = ws + w.x[4];
  q.Br = ws + w.bc[4];
  q.Cr = ws + w.bc[5];
  q.Af = pr->A_f;
  q.Df = pr->D_f;
  q.Ar = pr->A_r;
  q.Dr = pr->D_r;
  q.states = states;
  q.dyc = dy[0];
  q.dyn = dy[1];
  q.dstates = dstates;
  q.dxc = G[0];
  q.ddtc = G[1];
  q.dBc = ws + w.gbc[0];
  q.dCc = ws + w.gbc[1];
  q.dxn = G[2];
  q.ddtf = G[3];
  q.dBf = ws + w.gbc[2];
  q.dCf = ws + w.gbc[3];
  q.ddtr = G[4];
  q.dBr = ws + w.gbc[4];
  q.dCr = ws + w.gbc[5];
  q.dAf = gp->dA_f;
  q.dDf = gp->dD_f;
  q.dAr = gp->dA_r;
  q.dDr = gp->dD_r;
  e = api_run_backward(0, N, q, ws + w.bws, s);
  if (e != cudaSuccess) return e;
  // through SiLU, softplus and the convolution
  const MixIn<T> a = mix_in<T>(g, cl, nz, mp, nullptr);
  k_mix_dpre<T, TO><<<rows_grid(g, 1), 256, 0, s>>>(a, G[0], G[1], G[2], G[3], G[4], (TO*)gc->ddt, (TO*)gn->ddt_f,
                                                 (TO*)gn->ddt_r);
  e = api_launched(cudaGetLastError(), s);
  if (e != cudaSuccess) return e;
  k_mix_dxr<TO, Vec<T>::V><<<rows_grid(g, Vec<T>::V), 256, 0, s>>>(g.Bt, g.L, g.D, g.Bs, mp->conv_w, G[0], G[2], (TO*)gc->dx, (TO*)gn->dx);
  e = api_launched(cudaGetLastError(), s);
  if (e != cudaSuccess) return e;
  void* gbc_out[6] = {gc->dB, gc->dC, gn->dB_f, gn->dC_f, gn->dB_r, gn->dC_r};
  for (int i = 0; i < 6 && e == cudaSuccess; ++i) {
    k_mix_cvt<float, TO><<<blocks_of(nn), 256, 0, s>>>(nn, (const float*)(ws + w.gbc[i]), (TO*)gbc_out[i]);
    e = api_launched(cudaGetLastError(), s);
  }
  if (e != cudaSuccess) return e;
  float* part = (float*)(ws + w.part);
  k_mix_par_part<T><<<dim3((unsigned)((g.D + 128 * Vec<T>::V - 1) / (128 * Vec<T>::V)), kParSplit), 128, 0, s>>>(a, G[0], G[2], G[1], G[3], G[4],
                                                                                  part);
  e = api_launched(cudaGetLastError(), s);
  if (e != cudaSuccess) return e;
  k_mix_par_red<<<blocks_of(g.D * (kW + 3)), 256, 0, s>>>(g.D, part, gm->dconv_w, gm->dconv_b, gm->ddt_bias_f,
                                                          gm->ddt_bias_r);
  return api_launched(cudaGetLastError(), s);
}

template <typename T, typename TO>
cudaError_t mix_boundary_t(const Geo& g, int N, const bdscan_clean* cl, const void* z_c, const float* A_f,
                           const float* D_f, const bdscan_mixer_params* mp, const float* init_state,
                           const float* conv_init, void* out_c, float* states, float* conv_states, int emit_all,
                           char* ws, cudaStream_t s) {
  const MixWs w = mix_ws(g, N);
  const MixIn<T> a = mix_in<T>(g, cl, nullptr, mp, conv_init);
  const int64_t n = g.Bt * g.L * g.D, nn = g.Bt * g.L * N;
  k_mix_prep<T><<<rows_grid(g, 1), 256, 0, s>>>(a, (float*)(ws + w.x[0]), (float*)(ws + w.x[1]), nullptr, nullptr,
                                             nullptr);
  cudaError_t e = api_launched(cudaGetLastError(), s);
  const void* bc[2] = {cl->B, cl->C};
  if (e == cudaSuccess) e = to_f32<T>(bc, w.bc, 2, ws, nn, s);
  if (e != cudaSuccess) return e;
  FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = g;
  p.xc = ws + w.x[0];
  p.dtc = ws + w.x[1];
  p.Bc = ws + w.bc[0];
  p.Cc = ws + w.bc[1];
  p.Af = A_f;
  p.Df = D_f;
  p.init = init_state;
  p.yc = out_c != nullptr ? (void*)(ws + w.y[0]) : nullptr;
  p.hst = (float*)(ws + w.scan);
  p.sdt = (float*)(ws + w.scan + al((size_t)g.Bt * (g.nc + 1) * g.D * N * 4));
  e = api_run_boundary(0, N, p, states, emit_all, s);
  if (e == cudaSuccess && out_c != nullptr) e = gate<T, TO>(n, ws, w.y[0], z_c, out_c, s);
  if (e != cudaSuccess) return e;
  const int64_t nc = g.Bt * (emit_all ? g.nb : 1) * (kW - 1) * g.D;
  k_mix_conv_states<T><<<blocks_of(nc), 256, 0, s>>>(a, emit_all, conv_states);
  return api_launched(cudaGetLastError(), s);
}

template <typename T, typename TO>
cudaError_t mix_active_t(const Geo& g, int N, const float* seed, const float* conv_seed, const bdscan_noisy* nz,
                         const void* z_n, const bdscan_params* pr, const bdscan_mixer_params* mp, void* out_n,
                         char* ws, cudaStream_t s) {
  const MixWs w = mix_ws(g, N);
  // one block: every window position before its first token reads the cached
  // convolution state
  const MixIn<T> a = mix_in<T>(g, nullptr, nz, mp, conv_seed);
  const int64_t n = g.Bt * g.L * g.D, nn = g.Bt * g.L * N;
  k_mix_prep<T><<<rows_grid(g, 1), 256, 0, s>>>(a, nullptr, nullptr, (float*)(ws + w.x[2]), (float*)(ws + w.x[3]),
                                             (float*)(ws + w.x[4]));
  cudaError_t e = api_launched(cudaGetLastError(), s);
  const void* bc[4] = {nz->B_f, nz->C_f, nz->B_r, nz->C_r};
  if (e == cudaSuccess) e = to_f32<T>(bc, w.bc + 2, 4, ws, nn, s);
  if (e != cudaSuccess) return e;
  FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = g;
  p.xn = ws + w.x[2];
  p.dtf = ws + w.x[3];
  p.Bf = ws + w.bc[2];
  p.Cf = ws + w.bc[3];
  p.dtr = ws + w.x[4];
  p.Br = ws + w.bc[4];
  p.Cr = ws + w.bc[5];
  p.Af = pr->A_f;
  p.Df = pr->D_f;
  p.Ar = pr->A_r;
  p.Dr = pr->D_r;
  p.yn = ws + w.y[1];
  p.seed = seed;
  e = api_launched(launch_active_block(0, N, p, s), s);
  if (e == cudaSuccess) e = gate<T, TO>(n, ws, w.y[1], z_n, out_n, s);
  return e;
}

// dt code: 0 f32 in and out, 1 bf16 in and out, 2 bf16 in, f32 out
#define MIX_DISPATCH(dt, CALL)                      \
  switch (dt) {                                     \
    case 0: { using T = float; using TO = float; return CALL; } \
    case 1: { using T = bf16; using TO = bf16; return CALL; }   \
    default: { using T = bf16; using TO = float; return CALL; } \
  }

}  // namespace
}  // namespace bds

using bds::Geo;
using bds::a16;
using bds::bad_arg;
using bds::bf16;

namespace {

template <typename F>
int mix_run(const char* fn, F f) {
  const cudaError_t e = f();
  if (e != cudaSuccess) return bds::cuda_err(fn, e);
  return bds::api_ok();
}

int mix_check_streams(const char* fn, const bdscan_clean* cl, const bdscan_noisy* nz) {
  if (cl != nullptr) {
    MIX_REQ(cl->x, "clean.x");
    MIX_REQ(cl->dt, "clean.dt");
    MIX_REQ(cl->B, "clean.B");
    MIX_REQ(cl->C, "clean.C");
  }
  if (nz != nullptr) {
    MIX_REQ(nz->x, "noisy.x");
    MIX_REQ(nz->dt_f, "noisy.dt_f");
    MIX_REQ(nz->B_f, "noisy.B_f");
    MIX_REQ(nz->C_f, "noisy.C_f");
    MIX_REQ(nz->dt_r, "noisy.dt_r");
    MIX_REQ(nz->B_r, "noisy.B_r");
    MIX_REQ(nz->C_r, "noisy.C_r");
  }
  return BDSCAN_OK;
}
int mix_check_params(const char* fn, const bdscan_params* pr) {
  if (pr == nullptr) return bds::bad_arg(fn, "params is NULL");
  MIX_REQ(pr->A_f, "params.A_f");
  MIX_REQ(pr->D_f, "params.D_f");
  MIX_REQ(pr->A_r, "params.A_r");
  MIX_REQ(pr->D_r, "params.D_r");
  return BDSCAN_OK;
}
int mix_check_ws(const char* fn, void* ws, size_t have, size_t need) {
  MIX_REQ(ws, "workspace");
  if (have < need) {
    char m[200];
    snprintf(m, sizeof(m), "workspace of %zu bytes, %zu needed", have, need);
    return bds::bad_arg(fn, m);
  }
  return BDSCAN_OK;
}

}  // namespace

extern "C" {

size_t bdscan_mixer_forward_workspace_size(const bdscan_dims* dims) {
  Geo g;
  int dt = 0, N = 0;
  if (bds::api_check_forward_dims(dims, &g, &dt, &N, "bdscan_mixer_forward_workspace_size")) return 0;
  return bds::mix_ws(g, N).fwd_total;
}
size_t bdscan_mixer_backward_workspace_size(const bdscan_dims* dims) {
  Geo g;
  int dt = 0, N = 0;
  if (bds::api_check_forward_dims(dims, &g, &dt, &N, "bdscan_mixer_backward_workspace_size")) return 0;
  return bds::mix_ws(g, N).bwd_total;
}
size_t bdscan_mixer_boundary_states_workspace_size(const bdscan_dims* dims) {
  return bdscan_mixer_forward_workspace_size(dims);
}
size_t bdscan_mixer_active_block_workspace_size(const bdscan_dims* dims) {
  return bdscan_mixer_forward_workspace_size(dims);
}

int bdscan_mixer_forward(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                         const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                         const bdscan_mixer_params* mparams, void* out_c, void* out_n, float* states,
                         void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_mixer_forward";
  Geo g;
  int dt = 0, N = 0;
  int rc = bds::api_check_forward_dims(dims, &g, &dt, &N, fn);
  if (rc) return rc;
  if (g.Bt == 0 || g.L == 0) return bds::api_ok();
  if (clean == nullptr || noisy == nullptr) return bds::bad_arg(fn, "clean or noisy is NULL");
  if ((rc = mix_check_streams(fn, clean, noisy)) || (rc = mix_check_params(fn, params)) ||
      (rc = bds::check_mparams(mparams, fn)))
    return rc;
  MIX_REQ(z_c, "z_c");
  MIX_REQ(z_n, "z_n");
  MIX_REQ(out_c, "out_c");
  MIX_REQ(out_n, "out_n");
  MIX_REQ(states, "states");
  if ((rc = mix_check_ws(fn, workspace, workspace_bytes, bds::mix_ws(g, N).fwd_total))) return rc;
  char* ws = (char*)workspace;
  cudaStream_t s = (cudaStream_t)stream;
  return mix_run(fn, [&]() -> cudaError_t {
    MIX_DISPATCH(dt, (bds::mix_forward_t<T, TO>(g, N, clean, z_c, noisy, z_n, params, mparams, out_c, out_n, states,
                                               ws, s)))
  });
}

int bdscan_mixer_backward(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                          const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                          const bdscan_mixer_params* mparams, const void* dout_c, const void* dout_n,
                          const float* dstates, const bdscan_clean_grads* gclean, void* dz_c,
                          const bdscan_noisy_grads* gnoisy, void* dz_n, const bdscan_param_grads* gparams,
                          const bdscan_mixer_grads* gmparams, void* workspace, size_t workspace_bytes,
                          void* stream) {
  const char* fn = "bdscan_mixer_backward";
  Geo g;
  int dt = 0, N = 0;
  int rc = bds::api_check_forward_dims(dims, &g, &dt, &N, fn);
  if (rc) return rc;
  if (g.Bs > 256)
    return bds::api_fail(BDSCAN_ERR_UNSUPPORTED, "bdscan_mixer_backward: backward block above 256");
  if (g.Bs > 16 && g.Bs % 16 != 0)
    return bds::api_fail(BDSCAN_ERR_UNSUPPORTED, "bdscan_mixer_backward: backward needs block <= 16 or a multiple of 16");
  if (gparams == nullptr || gmparams == nullptr) return bds::bad_arg(fn, "gparams or gmparams is NULL");
  MIX_REQ(gparams->dA_f, "dA_f");
  MIX_REQ(gparams->dD_f, "dD_f");
  MIX_REQ(gparams->dA_r, "dA_r");
  MIX_REQ(gparams->dD_r, "dD_r");
  MIX_REQ(gmparams->dconv_w, "dconv_w");
  MIX_REQ(gmparams->dconv_b, "dconv_b");
  MIX_REQ(gmparams->ddt_bias_f, "ddt_bias_f");
  MIX_REQ(gmparams->ddt_bias_r, "ddt_bias_r");
  if (g.Bt == 0 || g.L == 0) return bds::api_fail(BDSCAN_ERR_UNSUPPORTED, "bdscan_mixer_backward: empty problem");
  if (clean == nullptr || noisy == nullptr) return bds::bad_arg(fn, "clean or noisy is NULL");
  if ((rc = mix_check_streams(fn, clean, noisy)) || (rc = mix_check_params(fn, params)) ||
      (rc = bds::check_mparams(mparams, fn)))
    return rc;
  MIX_REQ(z_c, "z_c");
  MIX_REQ(z_n, "z_n");
  MIX_OPT(dout_c, "dout_c");
  MIX_REQ(dout_n, "dout_n");
  MIX_OPT(dstates, "dstates");
  MIX_REQ(dz_c, "dz_c");
  MIX_REQ(dz_n, "dz_n");
  if (gclean == nullptr || gnoisy == nullptr) return bds::bad_arg(fn, "gradient struct is NULL");
  MIX_REQ(gclean->dx, "gclean.dx");
  MIX_REQ(gclean->ddt, "gclean.ddt");
  MIX_REQ(gclean->dB, "gclean.dB");
  MIX_REQ(gclean->dC, "gclean.dC");
  MIX_REQ(gnoisy->dx, "gnoisy.dx");
  MIX_REQ(gnoisy->ddt_f, "gnoisy.ddt_f");
  MIX_REQ(gnoisy->dB_f, "gnoisy.dB_f");
  MIX_REQ(gnoisy->dC_f, "gnoisy.dC_f");
  MIX_REQ(gnoisy->ddt_r, "gnoisy.ddt_r");
  MIX_REQ(gnoisy->dB_r, "gnoisy.dB_r");
  MIX_REQ(gnoisy->dC_r, "gnoisy.dC_r");
  if ((rc = mix_check_ws(fn, workspace, workspace_bytes, bds::mix_ws(g, N).bwd_total))) return rc;
  char* ws = (char*)workspace;
  cudaStream_t s = (cudaStream_t)stream;
  return mix_run(fn, [&]() -> cudaError_t {
    MIX_DISPATCH(dt, (bds::mix_backward_t<T, TO>(g, N, clean, z_c, noisy, z_n, params, mparams, dout_c, dout_n,
                                                dstates, gclean, dz_c, gnoisy, dz_n, gparams, gmparams, ws, s)))
  });
}

int bdscan_mixer_boundary_states(const bdscan_dims* dims, const bdscan_clean* clean, const void* z_c,
                                 const float* A_f, const float* D_f, const bdscan_mixer_params* mparams,
                                 const float* init_state, const float* conv_init, void* out_c, float* states,
                                 float* conv_states, int emit_all, void* workspace, size_t workspace_bytes,
                                 void* stream) {
  const char* fn = "bdscan_mixer_boundary_states";
  Geo g;
  int dt = 0, N = 0;
  int rc = bds::api_check_forward_dims(dims, &g, &dt, &N, fn);
  if (rc) return rc;
  if (g.Bt == 0) return bds::api_ok();
  MIX_OPT(init_state, "init_state");
  MIX_OPT(conv_init, "conv_init");
  cudaStream_t s = (cudaStream_t)stream;
  if (g.L == 0) {  // the cache is the initial state
    if (emit_all) return bds::api_ok();
    MIX_REQ(states, "states");
    MIX_REQ(conv_states, "conv_states");
    const size_t sb = (size_t)g.Bt * g.D * N * 4, cb = (size_t)g.Bt * 3 * g.D * 4;
    cudaError_t e = init_state ? cudaMemcpyAsync(states, init_state, sb, cudaMemcpyDeviceToDevice, s)
                               : cudaMemsetAsync(states, 0, sb, s);
    if (e == cudaSuccess)
      e = conv_init ? cudaMemcpyAsync(conv_states, conv_init, cb, cudaMemcpyDeviceToDevice, s)
                    : cudaMemsetAsync(conv_states, 0, cb, s);
    return e == cudaSuccess ? bds::api_ok() : bds::cuda_err(fn, e);
  }
  if (clean == nullptr) return bds::bad_arg(fn, "clean is NULL");
  if ((rc = mix_check_streams(fn, clean, nullptr)) || (rc = bds::check_mparams(mparams, fn))) return rc;
  MIX_REQ(A_f, "A_f");
  MIX_REQ(D_f, "D_f");
  MIX_REQ(states, "states");
  MIX_REQ(conv_states, "conv_states");
  MIX_OPT(out_c, "out_c");
  MIX_OPT(z_c, "z_c");
  if ((out_c == nullptr) != (z_c == nullptr)) return bds::bad_arg(fn, "give both z_c and out_c, or neither");
  if ((rc = mix_check_ws(fn, workspace, workspace_bytes, bds::mix_ws(g, N).fwd_total))) return rc;
  char* ws = (char*)workspace;
  return mix_run(fn, [&]() -> cudaError_t {
    MIX_DISPATCH(dt, (bds::mix_boundary_t<T, TO>(g, N, clean, z_c, A_f, D_f, mparams, init_state, conv_init, out_c,
                                                states, conv_states, emit_all ? 1 : 0, ws, s)))
  });
}

int bdscan_mixer_active_block(const bdscan_dims* dims, const float* seed, const float* conv_seed,
                              const bdscan_noisy* noisy, const void* z_n, const bdscan_params* params,
                              const bdscan_mixer_params* mparams, void* out_n, void* workspace,
                              size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_mixer_active_block";
  Geo g;
  int dt = 0, N = 0;
  int rc = bds::api_check_forward_dims(dims, &g, &dt, &N, fn);
  if (rc) return rc;
  if (dims->len != dims->block && dims->len != 0) return bds::bad_arg(fn, "len must equal block");
  if (g.Bt == 0 || g.L == 0) return bds::api_ok();
  MIX_REQ(seed, "seed");
  MIX_REQ(conv_seed, "conv_seed");
  if (noisy == nullptr) return bds::bad_arg(fn, "noisy is NULL");
  if ((rc = mix_check_streams(fn, nullptr, noisy)) || (rc = mix_check_params(fn, params)) ||
      (rc = bds::check_mparams(mparams, fn)))
    return rc;
  MIX_REQ(z_n, "z_n");
  MIX_REQ(out_n, "out_n");
  if ((rc = mix_check_ws(fn, workspace, workspace_bytes, bds::mix_ws(g, N).fwd_total))) return rc;
  char* ws = (char*)workspace;
  cudaStream_t s = (cudaStream_t)stream;
  return mix_run(fn, [&]() -> cudaError_t {
    MIX_DISPATCH(dt, (bds::mix_active_t<T, TO>(g, N, seed, conv_seed, noisy, z_n, params, mparams, out_n, ws, s)))
  });
}

}  // extern "C"
