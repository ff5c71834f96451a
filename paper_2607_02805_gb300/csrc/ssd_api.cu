// ssd_api.cu -- the C ABI of the SSD-form scan (include/bdscan_ssd.h):
// argument validation, workspace layout and the launch sequence.
#include <cstdio>
#include <cstring>

#include "bdscan_ssd.h"
#include "params.h"
#include "ssd.cuh"

namespace {

// "<function>: <message>" as the thread's last error; returns `code`.
int fail_msg(int code, const char* fn, const char* what) {
  char msg[384];
  snprintf(msg, sizeof(msg), "%s: %s", fn, what);
  return bds::api_fail(code, msg);
}

// "<function>: <argument> <problem>" as the thread's last error; returns `code`.
int fail_arg(int code, const char* fn, const char* name, const char* problem) {
  char msg[384];
  snprintf(msg, sizeof(msg), "%s: %s %s", fn, name, problem);
  return bds::api_fail(code, msg);
}

int cuda_fail(cudaError_t e, const char* fn) {
  char msg[384];
  snprintf(msg, sizeof(msg), "%s: %s", fn, cudaGetErrorString(e));
  return bds::api_fail(BDSCAN_ERR_CUDA, msg);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }
size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

#define SSD_REQ(ptr, fn, name)                                                              \
  do {                                                                                      \
    if ((ptr) == nullptr) return fail_arg(BDSCAN_ERR_ARG, fn, name, "is NULL");         \
    if (!aligned16(ptr)) return fail_arg(BDSCAN_ERR_ARG, fn, name, "is not 16-byte aligned"); \
  } while (0)
#define SSD_OPT(ptr, fn, name)                                                              \
  do {                                                                                      \
    if ((ptr) != nullptr && !aligned16(ptr))                                                \
      return fail_arg(BDSCAN_ERR_ARG, fn, name, "is not 16-byte aligned");              \
  } while (0)

// Validates the dimensions and fills the geometry.
int check(const bdscan_ssd_dims* d, bds::SsdGeo* g, const char* fn) {
  bds::api_begin();
  if (d == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "dims is NULL");
  if (d->batch < 0 || d->len < 0 || d->heads < 0) return fail_msg(BDSCAN_ERR_ARG, fn, "negative batch, len or heads");
  if (d->block <= 0) return fail_msg(BDSCAN_ERR_ARG, fn, "block must be positive");
  if (d->len % d->block != 0) return fail_msg(BDSCAN_ERR_ARG, fn, "len is not a multiple of block");
  if (d->dtype != BDSCAN_BF16) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "dtype must be bf16");
  if (d->head_dim != 64) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "head_dim must be 64");
  if (d->d_state != 64 && d->d_state != 128) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "d_state must be 64 or 128");
  if (d->block != 128 && d->block != 256) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "block must be 128 or 256");
  if (d->heads > 65535 * 8) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "too many heads");
  const int64_t nb = d->len / d->block;
  if (d->batch * nb * (d->block / 128) > 0x7fffffffLL) return fail_msg(BDSCAN_ERR_UNSUPPORTED, fn, "too many blocks");
  g->Bt = d->batch;
  g->L = d->len;
  g->Bs = d->block;
  g->H = (int)d->heads;
  g->N = (int)d->d_state;
  g->nb = (int)nb;
  g->m = (int)(d->block / 128);
  return BDSCAN_OK;
}

int sm_count() {
  const int n = bds::sm_count_cached();
  return n > 0 ? n : 1;
}

// Heads per CTA. A CTA pays a fixed set-up (the block's B/C rows; in the
// block scan the Gram products, shared by all its heads) and then about the
// same time per head. Over the group counts g from ceil(H / maxg) to H, the
// model (waves of g * units CTAs over the SMs) x (1 set-up + ceil(H / g)
// heads) is minimised; ties keep the smaller g. With few `units` (an active
// block) this reaches one head per CTA; with many it keeps large groups.
int heads_per_cta(int H, int64_t units, int maxg) {
  if (H <= 0 || units <= 0) return 1;
  const int64_t sms = sm_count();
  int best = (H + maxg - 1) / maxg;
  int64_t best_cost = -1;
  for (int g = (H + maxg - 1) / maxg; g <= H; ++g) {
    const int hg = (H + g - 1) / g;
    if (g > (H + maxg - 1) / maxg && (H + g - 2) / (g - 1) == hg) continue;  // same heads per CTA, more CTAs
    const int64_t waves = (units * g + sms - 1) / sms;
    const int64_t cost = waves * (1 + hg);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = g;
    }
  }
  return (H + best - 1) / best;
}

size_t sumdt_bytes(const bds::SsdGeo& g) { return al256((size_t)g.Bt * g.nb * g.H * 4); }
size_t states_bytes(const bds::SsdGeo& g) { return al256((size_t)g.Bt * g.nb * g.H * 64 * g.N * 4); }

int check_clean(const bdscan_clean* c, const char* fn) {
  if (c == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "clean is NULL");
  SSD_REQ(c->x, fn, "clean.x");
  SSD_REQ(c->dt, fn, "clean.dt");
  SSD_REQ(c->B, fn, "clean.B");
  SSD_REQ(c->C, fn, "clean.C");
  return BDSCAN_OK;
}

int check_noisy(const bdscan_noisy* n, const bdscan_params* pr, const char* fn) {
  if (n == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "noisy is NULL");
  if (pr == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "params is NULL");
  SSD_REQ(n->x, fn, "noisy.x");
  SSD_REQ(n->dt_f, fn, "noisy.dt_f");
  SSD_REQ(n->B_f, fn, "noisy.B_f");
  SSD_REQ(n->C_f, fn, "noisy.C_f");
  SSD_REQ(n->dt_r, fn, "noisy.dt_r");
  SSD_REQ(n->B_r, fn, "noisy.B_r");
  SSD_REQ(n->C_r, fn, "noisy.C_r");
  SSD_REQ(pr->A_f, fn, "params.A_f");
  SSD_REQ(pr->D_f, fn, "params.D_f");
  SSD_REQ(pr->A_r, fn, "params.A_r");
  SSD_REQ(pr->D_r, fn, "params.D_r");
  return BDSCAN_OK;
}

using bf = __nv_bfloat16;

}  // namespace

namespace {

bds::SsdScanParams clean_scan(const bds::SsdGeo& g, const bdscan_clean* c, const float* A_f, const float* D_f,
                              const float* seeds, const float* init, void* y, int* flag) {
  bds::SsdScanParams p{};
  p.g = g;
  p.x = (const bf*)c->x;
  p.dtf = (const bf*)c->dt;
  p.Bf = (const bf*)c->B;
  p.Cf = (const bf*)c->C;
  p.Af = A_f;
  p.Df = D_f;
  p.seed = seeds;
  p.seed_bstride = (int64_t)g.nb * g.H * 64 * g.N;
  p.seed_shift = 1;
  p.init_seed = init;
  p.y = (bf*)y;
  p.hg = heads_per_cta(g.H, g.Bt * g.nb * g.m, 16);
  p.flag = flag;
  return p;
}

bds::SsdScanParams noisy_scan(const bds::SsdGeo& g, const bdscan_noisy* n, const bdscan_params* pr, void* y,
                              int* flag) {
  bds::SsdScanParams p{};
  p.g = g;
  p.x = (const bf*)n->x;
  p.dtf = (const bf*)n->dt_f;
  p.Bf = (const bf*)n->B_f;
  p.Cf = (const bf*)n->C_f;
  p.dtr = (const bf*)n->dt_r;
  p.Br = (const bf*)n->B_r;
  p.Cr = (const bf*)n->C_r;
  p.Af = pr->A_f;
  p.Df = pr->D_f;
  p.Ar = pr->A_r;
  p.Dr = pr->D_r;
  p.y = (bf*)y;
  p.hg = heads_per_cta(g.H, g.Bt * g.nb * g.m, 16);
  p.flag = flag;
  return p;
}

// Block-local states into T, then the exact states (in place when T is the
// emitted states array).
cudaError_t build_states(const bds::SsdGeo& g, const bdscan_clean* c, const float* A_f, const float* init,
                         float* T, float* sumdt, float* final_state, int* flag, cudaStream_t s, int rev = 0) {
  bds::SsdStateParams sp{};
  sp.g = g;
  sp.x = (const bf*)c->x;
  sp.dt = (const bf*)c->dt;
  sp.B = (const bf*)c->B;
  sp.A = A_f;
  sp.T = T;
  sp.sumdt = sumdt;
  sp.hg = heads_per_cta(g.H, g.Bt * g.nb, 8);
  sp.flag = flag;
  sp.rev = rev;
  cudaError_t e = bds::api_launched(bds::launch_ssd_block_state(sp, s), s);
  if (e != cudaSuccess) return e;
  bds::SsdPassParams pp{};
  pp.g = g;
  pp.T = T;
  pp.sumdt = sumdt;
  pp.A = A_f;
  pp.init = init;
  pp.states = T;
  pp.emit_all = 1;
  pp.final_state = final_state;
  return bds::api_launched(bds::launch_ssd_state_pass(pp, s), s);
}

}  // namespace

extern "C" {

size_t bdscan_ssd_forward_workspace_size(const bdscan_ssd_dims* dims) {
  bds::SsdGeo g{};
  if (check(dims, &g, "bdscan_ssd_forward_workspace_size") != BDSCAN_OK) return 0;
  return sumdt_bytes(g);
}

int bdscan_ssd_forward(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                       const bdscan_params* params, void* y_c, void* y_n, float* states, void* workspace,
                       size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_ssd_forward";
  bds::SsdGeo g{};
  int rc = check(dims, &g, fn);
  if (rc) return rc;
  if (g.Bt == 0 || g.nb == 0 || g.H == 0) return bds::api_ok();
  if ((rc = check_clean(clean, fn)) || (rc = check_noisy(noisy, params, fn))) return rc;
  SSD_REQ(y_c, fn, "y_c");
  SSD_REQ(y_n, fn, "y_n");
  SSD_REQ(states, fn, "states");
  SSD_REQ(workspace, fn, "workspace");
  if (workspace_bytes < sumdt_bytes(g)) return fail_msg(BDSCAN_ERR_ARG, fn, "workspace too small");
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return cuda_fail(cudaGetLastError(), fn);
  cudaStream_t s = (cudaStream_t)stream;
  float* sumdt = (float*)workspace;
  cudaError_t e = build_states(g, clean, params->A_f, nullptr, states, sumdt, nullptr, flag, s);
  if (e == cudaSuccess) {
    const bds::SsdScanParams cp = clean_scan(g, clean, params->A_f, params->D_f, states, nullptr, y_c, flag);
    e = bds::api_launched(bds::launch_ssd_block_scan(false, cp, s), s);
  }
  if (e == cudaSuccess) {
    bds::SsdScanParams np = noisy_scan(g, noisy, params, y_n, flag);
    np.seed = states;
    np.seed_bstride = (int64_t)g.nb * g.H * 64 * g.N;
    np.seed_shift = 1;
    e = bds::api_launched(bds::launch_ssd_block_scan(true, np, s), s);
  }
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return bds::api_ok();
}

size_t bdscan_ssd_boundary_states_workspace_size(const bdscan_ssd_dims* dims, int emit_all) {
  bds::SsdGeo g{};
  if (check(dims, &g, "bdscan_ssd_boundary_states_workspace_size") != BDSCAN_OK) return 0;
  return sumdt_bytes(g) + (emit_all ? 0 : states_bytes(g));
}

int bdscan_ssd_boundary_states(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const float* A_f,
                               const float* D_f, const float* init_state, void* y_c, float* states,
                               int emit_all, void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_ssd_boundary_states";
  bds::SsdGeo g{};
  int rc = check(dims, &g, fn);
  if (rc) return rc;
  if (g.Bt == 0 || g.nb == 0 || g.H == 0) return bds::api_ok();
  if ((rc = check_clean(clean, fn))) return rc;
  SSD_REQ(A_f, fn, "A_f");
  SSD_REQ(states, fn, "states");
  SSD_REQ(workspace, fn, "workspace");
  SSD_OPT(init_state, fn, "init_state");
  SSD_OPT(y_c, fn, "y_c");
  if (y_c != nullptr) SSD_REQ(D_f, fn, "D_f");
  if (workspace_bytes < sumdt_bytes(g) + (emit_all ? 0 : states_bytes(g)))
    return fail_msg(BDSCAN_ERR_ARG, fn, "workspace too small");
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return cuda_fail(cudaGetLastError(), fn);
  cudaStream_t s = (cudaStream_t)stream;
  float* sumdt = (float*)workspace;
  // every block-end state goes to `states` (emit_all) or to the workspace,
  // with the final one copied out
  float* all = emit_all ? states : (float*)((char*)workspace + sumdt_bytes(g));
  cudaError_t e = build_states(g, clean, A_f, init_state, all, sumdt, emit_all ? nullptr : states, flag, s);
  if (e == cudaSuccess && y_c != nullptr) {
    const bds::SsdScanParams cp = clean_scan(g, clean, A_f, D_f, all, init_state, y_c, flag);
    e = bds::api_launched(bds::launch_ssd_block_scan(false, cp, s), s);
  }
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return bds::api_ok();
}

int bdscan_ssd_active_block(const bdscan_ssd_dims* dims, const float* seed, const bdscan_noisy* noisy,
                            const bdscan_params* params, void* y_n, void* stream) {
  const char* fn = "bdscan_ssd_active_block";
  bds::SsdGeo g{};
  int rc = check(dims, &g, fn);
  if (rc) return rc;
  if (dims->len != dims->block) return fail_msg(BDSCAN_ERR_ARG, fn, "len must equal block");
  if (g.Bt == 0 || g.H == 0) return bds::api_ok();
  if ((rc = check_noisy(noisy, params, fn))) return rc;
  SSD_OPT(seed, fn, "seed");
  SSD_REQ(y_n, fn, "y_n");
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return cuda_fail(cudaGetLastError(), fn);
  cudaStream_t s = (cudaStream_t)stream;
  bds::SsdScanParams np = noisy_scan(g, noisy, params, y_n, flag);
  np.seed = seed;
  np.seed_bstride = (int64_t)g.H * 64 * g.N;
  np.seed_shift = 0;
  const cudaError_t e = bds::api_launched(bds::launch_ssd_block_scan(true, np, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return bds::api_ok();
}

int bdscan_ssd_wait_flag(int reset) {
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return -1;
  int v = 0;
  if (cudaMemcpy(&v, flag, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
  if (reset && cudaMemset(flag, 0, sizeof(int)) != cudaSuccess) return -1;
  return v;
}

int bdscan_ssd_tma_enabled(void) { return bds::ssd_tma_enabled() ? 1 : 0; }

int bdscan_ssd_set_tma(int enable) {
  bds::ssd_set_tma(enable != 0);
  return bds::ssd_tma_enabled() ? 1 : 0;
}

int bdscan_ssd_wait_selftest(uint32_t polls) {
  const char* fn = "bdscan_ssd_wait_selftest";
  bds::api_begin();
  if (polls == 0 || polls > (1u << 20)) return fail_msg(BDSCAN_ERR_ARG, fn, "polls must be in 1..2^20");
  if (bdscan_ssd_wait_flag(1) < 0) return cuda_fail(cudaGetLastError(), fn);
  cudaError_t e = bds::api_launched(bds::launch_ssd_wait_probe(polls, nullptr), nullptr);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, fn);
  const int v = bdscan_ssd_wait_flag(1);
  if (v < 0) return cuda_fail(cudaGetLastError(), fn);
  bds::api_ok();
  return v;
}

size_t bdscan_ssd_full_bidir_workspace_size(const bdscan_ssd_dims* dims) {
  bds::SsdGeo g{};
  if (check(dims, &g, "bdscan_ssd_full_bidir_workspace_size") != BDSCAN_OK) return 0;
  return sumdt_bytes(g) + states_bytes(g) + al256((size_t)g.Bt * g.L * g.H * 64 * 4);
}

int bdscan_ssd_full_bidir_forward(const bdscan_ssd_dims* dims, const bdscan_noisy* noisy, const bdscan_params* params,
                                  void* y, void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_ssd_full_bidir_forward";
  bds::SsdGeo g{};
  int rc = check(dims, &g, fn);
  if (rc) return rc;
  if (g.Bt == 0 || g.nb == 0 || g.H == 0) return bds::api_ok();
  if ((rc = check_noisy(noisy, params, fn))) return rc;
  SSD_REQ(y, fn, "y");
  SSD_REQ(workspace, fn, "workspace");
  const size_t need = sumdt_bytes(g) + states_bytes(g) + al256((size_t)g.Bt * g.L * g.H * 64 * 4);
  if (workspace_bytes < need) return fail_msg(BDSCAN_ERR_ARG, fn, "workspace too small");
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return cuda_fail(cudaGetLastError(), fn);
  cudaStream_t s = (cudaStream_t)stream;
  float* sumdt = (float*)workspace;
  float* st = (float*)((char*)workspace + sumdt_bytes(g));
  float* y32 = (float*)((char*)st + states_bytes(g));
  // each direction is the clean-stream scan over the whole sequence: left to
  // right with the forward parameters, then right to left with the reverse
  // ones; the first writes fp32, the second adds it and rounds once
  cudaError_t e = cudaSuccess;
  for (int dir = 0; dir < 2 && e == cudaSuccess; ++dir) {
    const bdscan_clean c{noisy->x, dir ? noisy->dt_r : noisy->dt_f, dir ? noisy->B_r : noisy->B_f,
                         dir ? noisy->C_r : noisy->C_f};
    const float* A = dir ? params->A_r : params->A_f;
    const float* D = dir ? params->D_r : params->D_f;
    e = build_states(g, &c, A, nullptr, st, sumdt, nullptr, flag, s, dir);
    if (e != cudaSuccess) break;
    bds::SsdScanParams cp = clean_scan(g, &c, A, D, st, nullptr, y, flag);
    cp.rev = dir;
    if (dir == 0) cp.y32 = y32;
    else cp.y32_add = y32;
    e = bds::api_launched(bds::launch_ssd_block_scan(false, cp, s), s);
  }
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return bds::api_ok();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// backward
// ---------------------------------------------------------------------------
namespace {

// Workspace regions of the SSD backward (byte offsets), per stream s = clean,
// noisy forward direction, noisy reverse direction: the tile partials of dx,
// dB, dC, the column and row sums, the row dots and seed-gradient partials
// (seeded directions), the dt and A gradients; then the block sums of dt,
// the state gradients, the clean block-state terms and the dD partials.
struct SsdBwdWs {
  size_t dxp[3], dBp[3], dCp[3], colp[3], rows[3], rowdot[3], dSp[3], ddtv[3], dAv[3];
  size_t sumdt, gS, dxs, dBs, dAs, dd, total;
  int hg, ngrp;  // heads per tile CTA, head groups
};
// Head groups of the tile kernel: enough CTAs for about 1024 (several waves
// over the SMs), at most 16 heads per CTA; a function of the dimensions only,
// so the workspace size does not depend on the device.
void ssd_bwd_groups(const bds::SsdGeo& g, int* hg, int* ngrp) {
  const int64_t units = g.Bt * g.nb * g.m;
  int64_t want = units > 0 ? (1024 + units - 1) / units : 1;
  const int64_t lo = (g.H + 15) / 16;
  if (want < lo) want = lo;
  if (want > g.H) want = g.H;
  if (want < 1) want = 1;
  *hg = (int)((g.H + want - 1) / want);
  *ngrp = g.H > 0 ? (g.H + *hg - 1) / *hg : 1;
}
SsdBwdWs ssd_bwd_ws(const bds::SsdGeo& g) {
  SsdBwdWs w;
  ssd_bwd_groups(g, &w.hg, &w.ngrp);
  const size_t bkg = (size_t)g.Bt * g.nb * w.ngrp;
  const size_t bkh = (size_t)g.Bt * g.nb * g.H, P = 64, N = (size_t)g.N, m = (size_t)g.m, Bs = (size_t)g.Bs;
  size_t o = 0;
  auto take = [&](size_t floats) {
    const size_t at = o;
    o += al256(floats * 4);
    return at;
  };
  for (int s = 0; s < 3; ++s) {
    w.dxp[s] = take(bkh * m * Bs * P);
    w.dBp[s] = take(bkg * m * Bs * N);
    w.dCp[s] = take(bkg * Bs * N);
    w.colp[s] = take(bkh * m * Bs);
    w.rows[s] = take(bkh * Bs);
    w.rowdot[s] = s < 2 ? take(bkh * Bs) : 0;
    w.dSp[s] = s < 2 ? take(bkh * m * P * N) : 0;
    w.ddtv[s] = s == 0 ? take((size_t)g.Bt * g.L * g.H) : 0;  // the noisy directions write their outputs
    w.dAv[s] = take(bkh);
  }
  w.sumdt = take(bkh);
  w.gS = take(bkh * P * N);
  w.dxs = take(bkh * Bs * P);
  w.dBs = take(bkh * Bs * N);
  w.dAs = take(bkh);
  w.dd = take(bkh * m * 8 * 2);  // dy . x partials of the clean, then the noisy stream
  w.total = o;
  return w;
}

}  // namespace

extern "C" size_t bdscan_ssd_backward_workspace_size(const bdscan_ssd_dims* dims) {
  bds::SsdGeo g{};
  if (check(dims, &g, "bdscan_ssd_backward_workspace_size") != BDSCAN_OK) return 0;
  return ssd_bwd_ws(g).total;
}

extern "C" int bdscan_ssd_backward(const bdscan_ssd_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                                   const bdscan_params* params, const float* states, const void* dy_c, const void* dy_n,
                                   const float* dstates, const bdscan_clean_grads* gclean,
                                   const bdscan_noisy_grads* gnoisy, const bdscan_param_grads* gparams,
                                   void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_ssd_backward";
  bds::SsdGeo g{};
  int rc = check(dims, &g, fn);
  if (rc) return rc;
  if (gparams == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "gparams is NULL");
  SSD_REQ(gparams->dA_f, fn, "gparams.dA_f");
  SSD_REQ(gparams->dD_f, fn, "gparams.dD_f");
  SSD_REQ(gparams->dA_r, fn, "gparams.dA_r");
  SSD_REQ(gparams->dD_r, fn, "gparams.dD_r");
  cudaStream_t s = (cudaStream_t)stream;
  if (g.Bt == 0 || g.L == 0 || g.H == 0) {
    cudaError_t e = cudaSuccess;
    const size_t hb = (size_t)g.H * 4;
    if (hb > 0) {
      e = cudaMemsetAsync(gparams->dA_f, 0, hb, s);
      if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dA_r, 0, hb, s);
      if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dD_f, 0, hb, s);
      if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dD_r, 0, hb, s);
    }
    return e == cudaSuccess ? bds::api_ok() : cuda_fail(e, fn);
  }
  if ((rc = check_clean(clean, fn)) || (rc = check_noisy(noisy, params, fn))) return rc;
  SSD_REQ(states, fn, "states");
  SSD_OPT(dy_c, fn, "dy_c");
  SSD_REQ(dy_n, fn, "dy_n");
  SSD_OPT(dstates, fn, "dstates");
  if (gclean == nullptr || gnoisy == nullptr) return fail_msg(BDSCAN_ERR_ARG, fn, "gradient struct is NULL");
  SSD_REQ(gclean->dx, fn, "gclean.dx");
  SSD_REQ(gclean->ddt, fn, "gclean.ddt");
  SSD_REQ(gclean->dB, fn, "gclean.dB");
  SSD_REQ(gclean->dC, fn, "gclean.dC");
  SSD_REQ(gnoisy->dx, fn, "gnoisy.dx");
  SSD_REQ(gnoisy->ddt_f, fn, "gnoisy.ddt_f");
  SSD_REQ(gnoisy->dB_f, fn, "gnoisy.dB_f");
  SSD_REQ(gnoisy->dC_f, fn, "gnoisy.dC_f");
  SSD_REQ(gnoisy->ddt_r, fn, "gnoisy.ddt_r");
  SSD_REQ(gnoisy->dB_r, fn, "gnoisy.dB_r");
  SSD_REQ(gnoisy->dC_r, fn, "gnoisy.dC_r");
  const SsdBwdWs w = ssd_bwd_ws(g);
  SSD_REQ(workspace, fn, "workspace");
  if (workspace_bytes < w.total) {
    char msg[160];
    snprintf(msg, sizeof(msg), "workspace of %zu bytes, %zu needed", workspace_bytes, w.total);
    return fail_msg(BDSCAN_ERR_ARG, fn, msg);
  }
  int* flag = bds::ssd_wait_flag_ptr();
  if (flag == nullptr) return fail_msg(BDSCAN_ERR_CUDA, fn, "cannot locate the device wait flag");
  char* ws = (char*)workspace;
  auto F = [&](size_t off) { return (float*)(ws + off); };
  using bf = __nv_bfloat16;
  const bf* xs[3] = {(const bf*)clean->x, (const bf*)noisy->x, (const bf*)noisy->x};
  const bf* dys[3] = {(const bf*)dy_c, (const bf*)dy_n, (const bf*)dy_n};
  const bf* dts[3] = {(const bf*)clean->dt, (const bf*)noisy->dt_f, (const bf*)noisy->dt_r};
  const bf* Bsrc[3] = {(const bf*)clean->B, (const bf*)noisy->B_f, (const bf*)noisy->B_r};
  const bf* Csrc[3] = {(const bf*)clean->C, (const bf*)noisy->C_f, (const bf*)noisy->C_r};
  const float* As[3] = {params->A_f, params->A_f, params->A_r};
  cudaError_t e = cudaSuccess;
  // 1. block-local products of the three streams (clean and noisy forward
  //    seeded with the clean state before each block, noisy reverse unseeded)
  for (int st = 0; st < 3 && e == cudaSuccess; ++st) {
    bds::SsdBwdTileParams p;
    memset(&p, 0, sizeof(p));
    p.g = g;
    p.x = xs[st];
    p.dy = dys[st];
    p.dt = dts[st];
    p.B = Bsrc[st];
    p.C = Csrc[st];
    p.A = As[st];
    p.states = st < 2 ? states : nullptr;
    p.dx_part = F(w.dxp[st]);
    p.dB_part = F(w.dBp[st]);
    p.dC_part = F(w.dCp[st]);
    p.col_part = F(w.colp[st]);
    p.rowsum = F(w.rows[st]);
    p.rowdot = st < 2 ? F(w.rowdot[st]) : nullptr;
    p.dS_part = st < 2 ? F(w.dSp[st]) : nullptr;
    p.dd_part = st < 2 ? F(w.dd) + (size_t)st * g.Bt * g.nb * g.H * g.m * 8 : nullptr;
    p.hg = w.hg;
    p.flag = flag;
    e = bds::api_launched(bds::launch_ssd_bwd_tile(st == 2, st < 2, p, s), s);
  }
  // 2. dt and A gradients of each stream from the row and column sums
  for (int st = 0; st < 3 && e == cudaSuccess; ++st) {
    bds::SsdBwdVecParams v;
    memset(&v, 0, sizeof(v));
    v.g = g;
    v.dt = dts[st];
    v.A = As[st];
    v.col_part = F(w.colp[st]);
    v.rowsum = F(w.rows[st]);
    v.rowdot = st < 2 ? F(w.rowdot[st]) : nullptr;
    v.upper = st == 2;
    v.ddt = st == 0 ? F(w.ddtv[0]) : nullptr;
    v.ddt_out = st == 1 ? (bf*)gnoisy->ddt_f : st == 2 ? (bf*)gnoisy->ddt_r : nullptr;
    v.dA = F(w.dAv[st]);
    v.sumdt = st == 0 ? F(w.sumdt) : nullptr;
    e = bds::api_launched(bds::launch_ssd_bwd_vec(v, s), s);
  }
  // 3. reverse pass over the clean block-end states
  if (e == cudaSuccess) {
    bds::SsdBwdPassParams q;
    memset(&q, 0, sizeof(q));
    q.g = g;
    q.A = params->A_f;
    q.dS_c = F(w.dSp[0]);
    q.dS_f = F(w.dSp[1]);
    q.dstates = dstates;
    q.sumdt = F(w.sumdt);
    q.gS = F(w.gS);
    e = bds::api_launched(bds::launch_ssd_bwd_pass(q, s), s);
  }
  // 4. transpose of the clean block-state products
  if (e == cudaSuccess) {
    bds::SsdBwdStateParams r;
    memset(&r, 0, sizeof(r));
    r.g = g;
    r.x = xs[0];
    r.dt = dts[0];
    r.B = Bsrc[0];
    r.A = params->A_f;
    r.gS = F(w.gS);
    r.states = states;
    r.sumdt = F(w.sumdt);
    r.dx_state = F(w.dxs);
    r.dB_state = F(w.dBs);
    r.ddt_tile = F(w.ddtv[0]);
    r.ddt = (bf*)gclean->ddt;
    r.dA = F(w.dAs);
    r.flag = flag;
    e = bds::api_launched(bds::launch_ssd_bwd_state(r, s), s);
  }
  // 5. fixed-order combines into the outputs
  if (e == cudaSuccess)
    e = bds::api_launched(bds::launch_ssd_bwd_dx(g, F(w.dxp[0]), F(w.dxs), F(w.dxp[1]), F(w.dxp[2]), dys[0], dys[1],
                                                 params->D_f, params->D_r, (bf*)gclean->dx, (bf*)gnoisy->dx, s),
                          s);
  if (e == cudaSuccess)
    e = bds::api_launched(bds::launch_ssd_bwd_dbc(g, w.ngrp, F(w.dBp[0]), F(w.dBs), F(w.dCp[0]), F(w.dBp[1]), F(w.dCp[1]),
                                                  F(w.dBp[2]), F(w.dCp[2]), (bf*)gclean->dB, (bf*)gclean->dC,
                                                  (bf*)gnoisy->dB_f, (bf*)gnoisy->dC_f, (bf*)gnoisy->dB_r,
                                                  (bf*)gnoisy->dC_r, s),
                          s);
  if (e == cudaSuccess)
    e = bds::api_launched(bds::launch_ssd_bwd_params(g, F(w.dd), F(w.dd) + (size_t)g.Bt * g.nb * g.H * g.m * 8,
                                                     F(w.dAv[0]), F(w.dAv[1]), F(w.dAs), F(w.dAv[2]), gparams->dA_f,
                                                     gparams->dD_f, gparams->dA_r, gparams->dD_r, s),
                          s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return bds::api_ok();
}
