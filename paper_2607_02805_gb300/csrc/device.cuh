// device.cuh -- device-side building blocks of libbdscan (sm_103a).
//
// Thread mapping used by every scan kernel: one CTA of 128 threads covers 128
// consecutive channels d of one batch row; each thread owns one channel and
// keeps all N state elements of that channel in registers, so the sum over
// the state index (y = C.h, and dx, ddt in the backward) never leaves the
// thread. Inputs are staged per block of tokens into shared memory with
// cp.async: token-by-channel tiles stay in their storage type (one 2- or
// 4-byte read per thread and step), token-by-state rows (B, C) are widened
// to fp32 once per stage and read by all threads as broadcasts.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "debug.cuh"

namespace bds {

constexpr int kCta = 128;
constexpr int kWarps = kCta / 32;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.69314718055994531f;

typedef __nv_bfloat16 bf16;

// 2^x on the MUFU unit (ex2.approx.ftz.f32). exp(dt*A) is evaluated as
// 2^(dt * A*log2(e)) with A*log2(e) formed once per kernel.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float cvt(float v) { return v; }
__device__ __forceinline__ float cvt(bf16 v) { return __bfloat162float(v); }

template <typename TO>
__device__ __forceinline__ TO to_out(float v);
template <>
__device__ __forceinline__ float to_out<float>(float v) { return v; }
template <>
__device__ __forceinline__ bf16 to_out<bf16>(float v) { return __float2bfloat16_rn(v); }

template <typename T>
struct is_f32 { static constexpr bool value = false; };
template <>
struct is_f32<float> { static constexpr bool value = true; };

// ---------------------------------------------------------------------------
// cp.async staging
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, int src_bytes) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(src_bytes)
               : "memory");
}
// one 4-byte word, through L1 (the .cg form takes 16-byte copies only)
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// Copies `nsteps` token rows of a token-by-channel tensor g [.., D] for the
// channels [d0, d0+128) into tile[step][128]: step r is row row0 + r, or
// row0 - r with REV (a span staged in reversed time). Channels >= D read as
// zero; a null tensor stages zeros. Row starts are 16-byte aligned because D
// is a multiple of 16/sizeof(T) (checked on the host).
template <typename T, bool REV = false>
__device__ __forceinline__ void issue_td(T* tile, const T* g, int64_t row0, int nsteps, int64_t D,
                                         int64_t d0) {
  constexpr int E = 16 / (int)sizeof(T);
  constexpr int CPR = kCta / E;
  const int total = nsteps * CPR;
  for (int i = threadIdx.x; i < total; i += kCta) {
    const int r = i / CPR, q = i - r * CPR;
    const int64_t d = d0 + (int64_t)q * E;
    T* dst = tile + r * kCta + q * E;
    if (g == nullptr) {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
    } else {
      const bool ok = d < D;
      cp_async16(dst, ok ? (const void*)(g + (REV ? row0 - r : row0 + r) * D + d) : (const void*)g, ok ? 16 : 0);
    }
  }
}

// Copies nsteps token-by-state rows [N] into dst[step][N]: step r is row
// row0 + r, or row0 - r with REV.
template <typename T, int N, bool REV = false>
__device__ __forceinline__ void issue_rows(T* dst, const T* g, int64_t row0, int nsteps) {
  constexpr int E = 16 / (int)sizeof(T);
  static_assert((N * sizeof(T)) % 16 == 0, "state rows must be whole 16-byte chunks");
  constexpr int RPC = N / E;  // 16-byte chunks per row
  const int total = nsteps * RPC;
  for (int i = threadIdx.x; i < total; i += kCta) {
    if (g == nullptr) {
      *reinterpret_cast<uint4*>(dst + i * E) = make_uint4(0u, 0u, 0u, 0u);
    } else if (REV) {
      const int r = i / RPC, q = i - r * RPC;
      cp_async16(dst + i * E, g + (row0 - r) * N + q * E, 16);
    } else {
      cp_async16(dst + i * E, g + row0 * N + (int64_t)i * E, 16);
    }
  }
}

__device__ __forceinline__ void cp_async_wait_one() { asm volatile("cp.async.wait_group 1;\n" ::: "memory"); }

// A set of staged tensors for one span of up to `tsmax` tokens, in NBUF
// shared-memory buffers. With two buffers the next span is copied while the
// current one is processed: issue(next) ... complete(current, pending = 1).
// TSMAX > 0 fixes the span stride at compile time (every staged address is
// then a base plus an immediate); 0 takes it from carve(). REV stages spans in
// reversed time: issue's row0 is the row of the span's first step and the
// following steps are the rows below it.
template <typename T, int N, int NTD, int NROW, int NBUF = 1, int TSMAX = 0, bool REV = false>
struct Stage {
  unsigned char* base;
  int tsmax;
  const T* cur_td;       // token-by-channel tiles of the current buffer, this thread's channel
  const float* cur_rows;  // fp32 rows of the current buffer
  const T* td_src[NTD];
  const T* row_src[NROW];

  static __host__ __device__ size_t td_bytes(int ts) { return ((size_t)NTD * ts * kCta * sizeof(T) + 15) & ~(size_t)15; }
  static __host__ __device__ size_t raw_bytes(int ts) {
    return is_f32<T>::value ? 0 : (((size_t)NROW * ts * N * sizeof(T) + 15) & ~(size_t)15);
  }
  static __host__ __device__ size_t rows_bytes(int ts) { return (size_t)NROW * ts * N * sizeof(float); }
  static __host__ __device__ size_t buf_bytes(int ts) { return td_bytes(ts) + raw_bytes(ts) + rows_bytes(ts); }
  static __host__ __device__ size_t bytes(int ts) { return (size_t)NBUF * buf_bytes(ts); }

  __device__ __forceinline__ int stride() const { return TSMAX > 0 ? TSMAX : tsmax; }
  __device__ void carve(unsigned char* b, int ts) {
    base = b;
    tsmax = TSMAX > 0 ? TSMAX : ts;
    select(0);
  }
  __device__ __forceinline__ void select(int buf) {
    cur_td = td(buf) + threadIdx.x;
    cur_rows = rows(buf);
  }
  __device__ __forceinline__ T* td(int buf) const { return reinterpret_cast<T*>(base + (size_t)buf * buf_bytes(stride())); }
  __device__ __forceinline__ float* rows(int buf) const {
    return reinterpret_cast<float*>(base + (size_t)buf * buf_bytes(stride()) + td_bytes(stride()) + raw_bytes(stride()));
  }
  __device__ __forceinline__ T* raw(int buf) const {
    return is_f32<T>::value ? reinterpret_cast<T*>(rows(buf))
                            : reinterpret_cast<T*>(base + (size_t)buf * buf_bytes(stride()) + td_bytes(stride()));
  }
  // Starts the copies of tokens [row0, row0+nsteps) into buffer `buf` (one
  // cp.async group per thread). The caller guarantees no thread still reads it.
  __device__ void issue(int buf, int64_t row0, int nsteps, int64_t D, int64_t d0) {
    T* t = td(buf);
    T* r = raw(buf);
#pragma unroll
    for (int j = 0; j < NTD; ++j) issue_td<T, REV>(t + (size_t)j * stride() * kCta, td_src[j], row0, nsteps, D, d0);
#pragma unroll
    for (int j = 0; j < NROW; ++j) issue_rows<T, N, REV>(r + (size_t)j * stride() * N, row_src[j], row0, nsteps);
    cp_async_commit();
  }
  // Waits for the copies of buffer `buf` (with `pending` newer groups still in
  // flight), widens its B/C rows to fp32 and makes it the current buffer.
  __device__ void complete(int buf, int nsteps, int pending) {
    if (pending)
      cp_async_wait_one();
    else
      cp_async_wait_all();
    __syncthreads();
    if (!is_f32<T>::value) {
      const int half = nsteps * N / 2;  // element pairs per row
      const T* r = raw(buf);
      float* f = rows(buf);
#pragma unroll
      for (int j = 0; j < NROW; ++j) {
        const T* rj = r + (size_t)j * stride() * N;
        float* fj = f + (size_t)j * stride() * N;
        for (int q = threadIdx.x; q < half; q += kCta)
          reinterpret_cast<float2*>(fj)[q] = make_float2(cvt(rj[2 * q]), cvt(rj[2 * q + 1]));
      }
      __syncthreads();
    }
    select(buf);
  }
  // Synchronous load into buffer 0 (starts with a barrier so no thread still
  // reads the previous contents).
  __device__ void load(int64_t row0, int nsteps, int64_t D, int64_t d0) {
    __syncthreads();
    issue(0, row0, nsteps, D, d0);
    complete(0, nsteps, 0);
  }
  __device__ __forceinline__ float at(int j, int step) const {
    return cvt(cur_td[(j * stride() + step) * kCta]);
  }
  __device__ __forceinline__ const float* row(int j, int step) const {
    return cur_rows + (j * stride() + step) * N;
  }
};

// ---------------------------------------------------------------------------
// Per-thread state vectors
// ---------------------------------------------------------------------------
template <int N>
__device__ __forceinline__ void vload(float (&v)[N], const float* g) {
#pragma unroll
  for (int n = 0; n < N; n += 4) {
    const float4 q = *reinterpret_cast<const float4*>(g + n);
    v[n] = q.x;
    v[n + 1] = q.y;
    v[n + 2] = q.z;
    v[n + 3] = q.w;
  }
}
template <int N>
__device__ __forceinline__ void vstore(float* g, const float (&v)[N]) {
#pragma unroll
  for (int n = 0; n < N; n += 4) *reinterpret_cast<float4*>(g + n) = make_float4(v[n], v[n + 1], v[n + 2], v[n + 3]);
}
template <int N>
__device__ __forceinline__ void vzero(float (&v)[N]) {
#pragma unroll
  for (int n = 0; n < N; ++n) v[n] = 0.f;
}
template <int N>
__device__ __forceinline__ void vload_row(float (&v)[N], const float* s) {  // shared-memory row
#pragma unroll
  for (int n = 0; n < N; n += 4) {
    const float4 q = *reinterpret_cast<const float4*>(s + n);
    v[n] = q.x;
    v[n + 1] = q.y;
    v[n + 2] = q.z;
    v[n + 3] = q.w;
  }
}

// y of one direction with its D term, and the two-direction sum of a noisy
// token (eq. partial-reverse). Shared by the all-block forward and the
// active-block step so both round identically.
__device__ __forceinline__ float with_skip(float y_scan, float Dd, float x) { return __fmaf_rn(Dd, x, y_scan); }
__device__ __forceinline__ float combine_dirs(float y_fwd, float y_rev) { return __fadd_rn(y_fwd, y_rev); }

// ---------------------------------------------------------------------------
// Warp reduction over channels: v[0..N) summed over the 32 lanes; afterwards
// every lane l holds the total for state index l % N. Halving exchange
// (each level keeps half the values and adds the partner's other half),
// then a butterfly over the remaining lane bits. Fixed order: deterministic.
// ---------------------------------------------------------------------------
template <int N>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[N]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = N / 2; o >= 1; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float send = up ? v[i] : v[i + o];
      const float keep = up ? v[i + o] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
#pragma unroll
  for (int o = N; o < 32; o <<= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
  return v[0];
}

// ---------------------------------------------------------------------------
// Packed FP32: two state indices per FFMA2/FMUL2/FADD2 (sm_100 family). Each
// half is rounded exactly as the scalar __fmaf_rn/__fmul_rn/__fadd_rn.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 f2(float v) { return make_float2(v, v); }
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 mul2(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 ex2x2(float2 v) { return make_float2(ex2(v.x), ex2(v.y)); }

// Per-thread state vectors of N floats held as N/2 float2. In the backward
// kernels the 4-float groups of a vector are stored in a lane-dependent
// order: slot group j holds state group j ^ sw with sw = (lane >> 2) & (N/4 - 1).
// This makes the first halving levels of the channel reduction select-free
// (see warp_reduce_swz_part). The forward kernels use the natural order (sw = 0).
template <int N>
__device__ __forceinline__ int swz_of_lane() {
  return (int)((threadIdx.x >> 2) & (N / 4 - 1));
}
// global or shared memory -> registers, group-swizzled
template <int N>
__device__ __forceinline__ void vload2(float2 (&v)[N / 2], const float* src, int sw) {
#pragma unroll
  for (int j = 0; j < N / 4; ++j) {
    const float4 q = *reinterpret_cast<const float4*>(src + 4 * (j ^ sw));
    v[2 * j] = make_float2(q.x, q.y);
    v[2 * j + 1] = make_float2(q.z, q.w);
  }
}
template <int N>
__device__ __forceinline__ void vstore2(float* dst, const float2 (&v)[N / 2], int sw) {
#pragma unroll
  for (int j = 0; j < N / 4; ++j)
    *reinterpret_cast<float4*>(dst + 4 * (j ^ sw)) = make_float4(v[2 * j].x, v[2 * j].y, v[2 * j + 1].x, v[2 * j + 1].y);
}
template <int N>
__device__ __forceinline__ void vzero2(float2 (&v)[N / 2]) {
#pragma unroll
  for (int j = 0; j < N / 2; ++j) v[j] = make_float2(0.f, 0.f);
}

// Channel reduction of a group-swizzled vector, stopped before the last
// butterfly: afterwards lane l holds a partial sum for state index l % N,
// and the 32/N lanes l' with l' % N == l % N hold partials that add up to the
// total over the 32 lanes. The levels over lane bits 3 and 2 exchange whole
// slot halves without selects (the partner's matching state sits in the
// complementary slot); the levels over lane bits 1 and 0 exchange within a
// 4-group with selects. Fixed order: deterministic.
template <int N>
__device__ __forceinline__ float warp_reduce_swz_part(float2 (&v)[N / 2]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = N / 4; o >= 2; o >>= 1) {
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float2 r = make_float2(__shfl_xor_sync(0xffffffffu, v[i + o].x, 2 * o),
                                   __shfl_xor_sync(0xffffffffu, v[i + o].y, 2 * o));
      v[i] = add2(v[i], r);
    }
  }
  const bool up1 = (lane & 2) != 0;
  float k0 = up1 ? v[1].x : v[0].x, k1 = up1 ? v[1].y : v[0].y;
  const float s0 = up1 ? v[0].x : v[1].x, s1 = up1 ? v[0].y : v[1].y;
  k0 += __shfl_xor_sync(0xffffffffu, s0, 2);
  k1 += __shfl_xor_sync(0xffffffffu, s1, 2);
  const bool up0 = (lane & 1) != 0;
  float k = up0 ? k1 : k0;
  const float s = up0 ? k0 : k1;
  k += __shfl_xor_sync(0xffffffffu, s, 1);
  return k;
}

// ---------------------------------------------------------------------------
// The selective-scan step (eq. mamba-scan-background with A_t = exp(dt A)):
//     a[n] = 2^(dt * A2[n]),  h[n] = a[n] h[n] + (dt x) B[n],
// returning sum_n C[n] h[n] (without the D term), on a packed state in the
// natural order. The operation order is fixed with explicit round-to-nearest
// intrinsics, so every kernel that uses it (all-block forward, cache build,
// cache tail, active block) produces the same bits from the same state and
// inputs.
// ---------------------------------------------------------------------------
template <int N>
__device__ __forceinline__ float scan_step(float2 (&h)[N / 2], const float2 (&A2)[N / 2], float dt, float x,
                                           const float* Bs, const float* Cs) {
  const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x));
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int q = 0; q < N / 4; ++q) {
    const float4 b = *reinterpret_cast<const float4*>(Bs + 4 * q);
    const float4 c = *reinterpret_cast<const float4*>(Cs + 4 * q);
    h[2 * q] = fma2(ex2x2(mul2(dt2, A2[2 * q])), h[2 * q], mul2(u2, make_float2(b.x, b.y)));
    acc0 = fma2(make_float2(c.x, c.y), h[2 * q], acc0);
    h[2 * q + 1] = fma2(ex2x2(mul2(dt2, A2[2 * q + 1])), h[2 * q + 1], mul2(u2, make_float2(b.z, b.w)));
    acc1 = fma2(make_float2(c.z, c.w), h[2 * q + 1], acc1);
  }
  const float2 s = add2(acc0, acc1);
  return __fadd_rn(s.x, s.y);
}

// The state update alone (no output), same arithmetic as scan_step.
template <int N>
__device__ __forceinline__ void scan_state(float2 (&h)[N / 2], const float2 (&A2)[N / 2], float dt, float x,
                                           const float* Bs) {
  const float2 dt2 = f2(dt), u2 = f2(__fmul_rn(dt, x));
#pragma unroll
  for (int q = 0; q < N / 4; ++q) {
    const float4 b = *reinterpret_cast<const float4*>(Bs + 4 * q);
    h[2 * q] = fma2(ex2x2(mul2(dt2, A2[2 * q])), h[2 * q], mul2(u2, make_float2(b.x, b.y)));
    h[2 * q + 1] = fma2(ex2x2(mul2(dt2, A2[2 * q + 1])), h[2 * q + 1], mul2(u2, make_float2(b.z, b.w)));
  }
}

// ---------------------------------------------------------------------------
// Tensor memory (TMEM) as per-thread scratch for the backward recompute.
// A CTA of 4 warps allocates `cols` 32-bit columns; warp w owns TMEM lanes
// 32w..32w+31 (one lane per thread), so each thread has `cols` private fp32
// slots. tcgen05.st/ld move 16 (or 8) consecutive columns of the thread's
// lane; a wait orders them before the registers are used.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t tmem_cols_for(uint32_t need) {
  uint32_t c = 32;
  while (c < need) c <<= 1;
  return c;
}
__device__ __forceinline__ void tmem_alloc(uint32_t* smem_slot, uint32_t cols) {
  const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem_slot);
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(s), "r"(cols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(cols) : "memory");
}
__device__ __forceinline__ void tmem_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;\n" ::); }

template <int N>
struct Tmem;

// float2-array views of the TMEM row copies
template <int N>
__device__ __forceinline__ void tmem_st2(uint32_t ta, const float2 (&v)[N / 2]) {
  Tmem<N>::st(ta, *reinterpret_cast<const float(*)[N]>(&v[0]));
}
template <int N>
__device__ __forceinline__ void tmem_ld2(uint32_t ta, float2 (&v)[N / 2]) {
  Tmem<N>::ld(ta, *reinterpret_cast<float(*)[N]>(&v[0]));
}
template <>
struct Tmem<16> {
  static __device__ __forceinline__ void st(uint32_t ta, const float (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
        "%13, %14, %15, %16};\n" ::"r"(ta),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15])));
  }
  static __device__ __forceinline__ void ld(uint32_t ta, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
        "%13, %14, %15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(ta));
    // the wait names the destination registers so no use moves above it
    asm volatile("tcgen05.wait::ld.sync.aligned;\n"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                   "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                   "+r"(r[14]), "+r"(r[15])
                 :);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
  }
};

template <>
struct Tmem<8> {
  static __device__ __forceinline__ void st(uint32_t ta, const float (&v)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};\n" ::"r"(ta),
                 "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
                 "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
                 "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])));
  }
  static __device__ __forceinline__ void ld(uint32_t ta, float (&v)[8]) {
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(ta));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7])
                 :);
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
  }
};

}  // namespace bds
