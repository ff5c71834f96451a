// ssd_common.cuh -- device helpers shared by the SSD-form kernels of
// libbdscan (ssd.cu: forward side; ssd_bwd.cu: backward).
#pragma once
#include <cuda_bf16.h>
#include <cstdint>

#include "device.cuh"
#include "ssd.cuh"
#include "umma.cuh"

namespace bds {
namespace {

constexpr uint32_t kTile16 = 16384;  // one atom column of a 128-row operand tile

// Bulk copies by the tensor memory accelerator, completing on an mbarrier:
// the issuing thread first announces the bytes the phase will receive.
__device__ __forceinline__ void bar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(umma::smem_u32(bar)), "r"(bytes)
               : "memory");
}
// One box of a 3-D tensor map (coordinates innermost first) into shared memory.
__device__ __forceinline__ void tma_load_3d(void* dst, const void* map, int c0, int c1, int c2, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];\n" ::"r"(umma::smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(umma::smem_u32(bar))
      : "memory");
}
// A contiguous run of `bytes` (a multiple of 16, both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
                   umma::smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(umma::smem_u32(bar))
               : "memory");
}

// Bounded wait shared by all threads of the CTA; a give-up sets the flag and
// makes every thread see the failure.
__device__ __forceinline__ bool cta_wait(uint64_t* bar, uint32_t parity, int* flag) {
  const bool ok = umma::bar_wait(bar, parity);
  const int bad = __syncthreads_or(ok ? 0 : 1);
  if (bad && threadIdx.x == 0) atomicExch(flag, 1);
  return bad == 0;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Inclusive scan of dt over `n` tokens by one warp (n a multiple of 32):
// lane l sums tokens [l*n/32, (l+1)*n/32) in order, then the lane totals are
// scanned. REV = true scans from the last token (suffix sums). `raw`, if not
// null, receives dt itself (fp32) at the same positions.
template <bool REV>
__device__ __forceinline__ float warp_scan_dt(const __nv_bfloat16* dt, int64_t stride, int n, float* out,
                                              float* raw = nullptr) {
  const int lane = threadIdx.x & 31, per = n / 32;
  float loc[8];
  // all of the lane's loads are issued before the first add (n <= 256)
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const int pos = REV ? n - 1 - (lane * per + q) : lane * per + q;
    loc[q] = q < per ? __bfloat162float(dt[pos * stride]) : 0.f;
  }
  if (raw != nullptr) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int pos = REV ? n - 1 - (lane * per + q) : lane * per + q;
      if (q < per) raw[pos] = loc[q];
    }
  }
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    s = q < per ? __fadd_rn(s, loc[q]) : s;
    loc[q] = s;
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
  for (int q = 0; q < 8; ++q) {
    const int pos = REV ? n - 1 - (lane * per + q) : lane * per + q;
    if (q < per) out[pos] = __fadd_rn(base, loc[q]);
  }
  return __shfl_sync(0xffffffffu, inc, 31);  // total
}


// Token index of position s of block k in batch row b: left to right, or
// right to left (position t of the reversed stream is token L-1-t).
struct RowMap {
  int64_t base, step;
  __device__ __forceinline__ RowMap(int64_t b, int64_t L, int64_t k0, bool rev)
      : base(rev ? b * L + L - 1 - k0 : b * L + k0), step(rev ? -1 : 1) {}
  __device__ __forceinline__ int64_t operator()(int64_t s) const { return base + step * s; }
};

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
  return reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~(uintptr_t)1023);
}


}  // namespace
}  // namespace bds
