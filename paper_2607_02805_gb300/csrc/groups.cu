// groups.cu -- state groups of the diagonal form: d_state above 16 (or not 8
// or 16) runs the scan kernels once per group of 16 states (the last group 8
// or 16, zero-padded). The state index is separable in the recurrence of
// Sec. 3 (eq. mamba-scan-background): every (channel, state) element has its
// own decay, and only y = C h (forward) and dx, ddt (backward) sum over the
// states, so the per-group results add up to the full ones. These kernels
// move B, C, A and the states between the caller's [..][N] layout and the
// per-group [..][gs] layout, and add the groups' fp32 outputs in a fixed
// order (group 0 first).
#include "device.cuh"
#include "params.h"

namespace bds {
namespace {

// dst[r][k] = src[r][n0 + k] for k < gs (zero where n0 + k >= N); T is the
// element type of both.
template <typename T>
__global__ void __launch_bounds__(256) k_group_gather(const T* src, int64_t rows, int N, int n0, int gs, T* dst) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= rows * gs) return;
  const int64_t r = i / gs;
  const int k = (int)(i - r * gs), n = n0 + k;
  dst[i] = n < N ? src[r * N + n] : T(0.f);
}

// dst[r][n0 + k] = src[r][k] (fp32 to the output type) for k < gs, n0 + k < N.
template <typename TO>
__global__ void __launch_bounds__(256) k_group_scatter(const float* src, int64_t rows, int N, int n0, int gs, TO* dst) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= rows * gs) return;
  const int64_t r = i / gs;
  const int k = (int)(i - r * gs), n = n0 + k;
  if (n < N) dst[r * N + n] = to_out<TO>(src[i]);
}

// acc += add (fp32)
__global__ void __launch_bounds__(256) k_group_add(float* acc, const float* add, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i < n) acc[i] = __fadd_rn(acc[i], add[i]);
}

// out = acc in the output type
template <typename TO>
__global__ void __launch_bounds__(256) k_group_out(const float* acc, TO* out, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i < n) out[i] = to_out<TO>(acc[i]);
}

unsigned nblk(int64_t n) { return (unsigned)((n + 255) / 256); }

}  // namespace

cudaError_t launch_group_gather(const void* src, int elt, int64_t rows, int N, int n0, int gs, void* dst,
                                cudaStream_t s) {
  if (rows * gs == 0) return cudaSuccess;
  if (elt == 2)
    k_group_gather<bf16><<<nblk(rows * gs), 256, 0, s>>>((const bf16*)src, rows, N, n0, gs, (bf16*)dst);
  else
    k_group_gather<float><<<nblk(rows * gs), 256, 0, s>>>((const float*)src, rows, N, n0, gs, (float*)dst);
  return cudaGetLastError();
}

cudaError_t launch_group_scatter(const float* src, int64_t rows, int N, int n0, int gs, void* dst, int out_elt,
                                 cudaStream_t s) {
  if (rows * gs == 0) return cudaSuccess;
  if (out_elt == 2)
    k_group_scatter<bf16><<<nblk(rows * gs), 256, 0, s>>>(src, rows, N, n0, gs, (bf16*)dst);
  else
    k_group_scatter<float><<<nblk(rows * gs), 256, 0, s>>>(src, rows, N, n0, gs, (float*)dst);
  return cudaGetLastError();
}

cudaError_t launch_group_add(float* acc, const float* add, int64_t n, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  k_group_add<<<nblk(n), 256, 0, s>>>(acc, add, n);
  return cudaGetLastError();
}

cudaError_t launch_group_out(const float* acc, void* out, int out_elt, int64_t n, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  if (out_elt == 2)
    k_group_out<bf16><<<nblk(n), 256, 0, s>>>(acc, (bf16*)out, n);
  else
    k_group_out<float><<<nblk(n), 256, 0, s>>>(acc, (float*)out, n);
  return cudaGetLastError();
}

// Scratch of the grouped active block (the entry point has no workspace
// argument): a static device array, as the no-alloc cache build's; calls
// that overlap in time on one device race on it.
static __device__ __align__(256) unsigned char g_group_scratch[kGroupScratchBytes];

void* group_scratch() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_group_scratch) != cudaSuccess) return nullptr;
  return p;
}

}  // namespace bds
