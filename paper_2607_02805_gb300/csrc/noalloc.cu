// noalloc.cu -- cache build (bdscan_boundary_states) for callers that may not
// allocate device memory: the scratch of the chunked clean scan lives in a
// static device array of this file instead of a caller workspace. The
// kernels and their launch order are those of bdscan_boundary_states, so
// the results are the same bits.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "bdscan.h"
#include "params.h"

namespace {

// Scratch of bdscan_boundary_states_noalloc: chunk start states followed by
// the per-chunk sums of dt (the same layout as the caller workspace of
// bdscan_boundary_states). Every GPU that loads the library holds it until
// the process exits; all calls share it.
static __device__ __align__(256) unsigned char g_scratch[BDSCAN_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device. Host code cannot use
// the symbol itself (on the host it names a stand-in, not device memory), so
// the address is looked up once per device, with that device current.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

int cuda_error(cudaError_t e) {
  char msg[256];
  snprintf(msg, sizeof(msg), "bdscan_boundary_states_noalloc: %s", cudaGetErrorString(e));
  return bds::api_fail(BDSCAN_ERR_CUDA, msg);
}

}  // namespace

extern "C" int bdscan_boundary_states_noalloc(const bdscan_dims* dims, const bdscan_clean* clean,
                                              const float* A_f, const float* D_f, const float* init_state,
                                              void* y_c, float* states, int emit_all, void* stream) {
  const char* fn = "bdscan_boundary_states_noalloc";
  bds::Geo g;
  int dt = 0, N = 0;
  int rc = bds::api_check_forward_dims(dims, &g, &dt, &N, fn);
  if (rc) return rc;
  if (g.Bt == 0) return bds::api_ok();
  if (init_state != nullptr && !aligned16(init_state))
    return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: init_state is not 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  if (g.L == 0) {  // the cache is the initial state
    if (emit_all) return bds::api_ok();
    if (states == nullptr || !aligned16(states))
      return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: states is NULL or not 16-byte aligned");
    const size_t bytes = (size_t)g.Bt * g.D * N * 4;
    cudaError_t e = init_state ? cudaMemcpyAsync(states, init_state, bytes, cudaMemcpyDeviceToDevice, s)
                               : cudaMemsetAsync(states, 0, bytes, s);
    return e == cudaSuccess ? bds::api_ok() : cuda_error(e);
  }
  if (clean == nullptr || clean->x == nullptr || clean->dt == nullptr || clean->B == nullptr || clean->C == nullptr ||
      !aligned16(clean->x) || !aligned16(clean->dt) || !aligned16(clean->B) || !aligned16(clean->C))
    return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: clean inputs NULL or not 16-byte aligned");
  if (A_f == nullptr || D_f == nullptr || !aligned16(A_f) || !aligned16(D_f))
    return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: A_f/D_f NULL or not 16-byte aligned");
  if (states == nullptr || !aligned16(states))
    return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: states is NULL or not 16-byte aligned");
  if (y_c != nullptr && !aligned16(y_c))
    return bds::api_fail(BDSCAN_ERR_ARG, "bdscan_boundary_states_noalloc: y_c is not 16-byte aligned");
  const size_t need = bds::api_fwd_workspace(g, N);
  if (need > BDSCAN_NOALLOC_SCRATCH_BYTES) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "bdscan_boundary_states_noalloc: needs %zu bytes of scratch, the static scratch holds %zu; "
             "use bdscan_boundary_states with a workspace",
             need, (size_t)BDSCAN_NOALLOC_SCRATCH_BYTES);
    return bds::api_fail(BDSCAN_ERR_UNSUPPORTED, msg);
  }
  void* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) return cuda_error(e);

  bds::FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = g;
  p.xc = clean->x;
  p.dtc = clean->dt;
  p.Bc = clean->B;
  p.Cc = clean->C;
  p.Af = A_f;
  p.Df = D_f;
  p.yc = y_c;
  p.init = init_state;
  p.hst = (float*)scratch;
  p.sdt = (float*)((char*)scratch + al256((size_t)g.Bt * (g.nc + 1) * g.D * N * 4));
  // every launch is counted (and timed by the profiling hook) as in
  // bdscan_boundary_states
  if (g.nc_full > 0) e = bds::api_launched(bds::launch_chunk_local(dt, N, p, s), s);
  if (e == cudaSuccess) e = bds::api_launched(bds::launch_chunk_carry(N, p, s), s);
  if (e == cudaSuccess) {
    if (emit_all || y_c != nullptr) {
      p.emit_all = emit_all ? 1 : 0;
      p.states = emit_all ? states : nullptr;
      p.final_state = emit_all ? nullptr : states;
      e = bds::api_launched(bds::launch_block_scan(dt, N, 1, g.nc, p, s), s);
    } else if (g.nc_full == g.nc) {
      const size_t row = (size_t)g.D * N * 4;
      e = cudaMemcpy2DAsync(states, row, p.hst + (size_t)g.nc * g.D * N, (size_t)(g.nc + 1) * row, row,
                            (size_t)g.Bt, cudaMemcpyDeviceToDevice, s);
    } else {
      p.emit_all = 0;
      p.final_state = states;
      p.c_begin = g.nc - 1;
      e = bds::api_launched(bds::launch_block_scan(dt, N, 1, 1, p, s), s);
    }
  }
  return e == cudaSuccess ? bds::api_ok() : cuda_error(e);
}
