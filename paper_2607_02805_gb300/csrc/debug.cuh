// debug.cuh -- device status words of the debug build of libbdscan.
//
// Built with -DBDSCAN_DEBUG=1 (lib/libbdscan_debug.so), every kernel first
// checks, for each buffer it touches, that the last element its CTA reads or
// writes lies inside the extent the call's sizes give that buffer. The check
// depends on blockIdx and the sizes only, so it is uniform over the CTA and
// runs before the first barrier, TMEM allocation or access. A failed check
// records (site, offset, extent) in this translation unit's device status word
// (the first failure wins) and the CTA returns without touching memory: the
// debug build never makes the access it flags and never traps. The cached
// states and the parameter gradients are also checked for non-finite values.
// At the end of each entry point the debug build synchronizes the device,
// reads every status word, and returns BDSCAN_ERR_DEVICE naming the first
// failed site (then clears them). In the release build every check is the
// constant `true` and compiles away.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#ifndef BDSCAN_DEBUG
#define BDSCAN_DEBUG 0
#endif

namespace bds {

// Sites of the device checks (named in the error message).
enum DebugSite : int {
  kSiteChunkLocal = 1,
  kSiteChunkCarry,
  kSiteBlockScan,
  kSiteActiveBlock,
  kSiteBwdNoisy,
  kSiteBwdCarry,
  kSiteBwdClean,
  kSiteReduceTok,
  kSiteReducePar,
  kSiteSsdBlockState,
  kSiteSsdStatePass,
  kSiteSsdBlockScan,
  kSiteSsdBwdTile,
  kSiteSsdBwdState,
  kSiteCount
};

constexpr int kStatusRange = 1;      // an extent check failed
constexpr int kStatusNonFinite = 2;  // a state or parameter gradient is NaN or infinite

struct DevStatus {
  int code;  // 0: no failure
  int site;
  long long value;  // the offending offset, or the flat index of the non-finite value
  long long limit;  // the extent checked against (range failures)
};

namespace dbg {
// Reads (and, if `clear`, resets) one translation unit's status word, and
// sets its slack: extents are taken `slack` elements shorter than the sizes
// give, so a test can make a check fail on an in-range access (the CTA then
// skips it). Returns a cudaError_t.
typedef int (*StatusIo)(DevStatus* out, int clear, long long slack);
int add_status_io(StatusIo io);  // host: registers a translation unit (api.cu)
}  // namespace dbg

#if BDSCAN_DEBUG

static __device__ DevStatus g_dev_status;
static __device__ long long g_dev_slack;

__device__ __forceinline__ void dev_record(int code, int site, long long value, long long limit) {
  if (atomicCAS(&g_dev_status.code, 0, code) == 0) {
    g_dev_status.site = site;
    g_dev_status.value = value;
    g_dev_status.limit = limit;
  }
}

// true when [0, last] lies inside an extent of `limit` elements
__device__ __forceinline__ bool dguard(int site, long long last, long long limit) {
  const long long lim = limit - g_dev_slack;
  if (last >= 0 && last < lim) return true;
  dev_record(kStatusRange, site, last, lim);
  return false;
}

__device__ __forceinline__ void dfinite(int site, float v, long long where) {
  if (!isfinite(v)) dev_record(kStatusNonFinite, site, where, 0);
}

static int dev_status_io(DevStatus* out, int clear, long long slack) {
  cudaError_t e = cudaMemcpyFromSymbol(out, g_dev_status, sizeof(DevStatus));
  if (e == cudaSuccess && clear) {
    const DevStatus zero = {0, 0, 0, 0};
    e = cudaMemcpyToSymbol(g_dev_status, &zero, sizeof(DevStatus));
  }
  if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_dev_slack, &slack, sizeof(long long));
  return (int)e;
}
static const int g_dev_status_registered = dbg::add_status_io(&dev_status_io);

#else

__device__ __forceinline__ constexpr bool dguard(int, long long, long long) { return true; }
__device__ __forceinline__ void dfinite(int, float, long long) {}

#endif

}  // namespace bds
