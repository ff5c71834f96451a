// api.cu -- the C ABI of libbdscan: argument validation, workspace layout
// and the launch sequence of each entry point. No exception crosses the ABI;
// every error is a return code plus a thread-local message.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>
#include <vector>

#include "bdscan.h"
#include "debug.cuh"
#include "params.h"

namespace bds {
namespace dbg {
// Status words of the translation units of the debug build (registered at
// load time, before any call).
std::vector<StatusIo>& status_ios() {
  static std::vector<StatusIo> v;
  return v;
}
std::mutex& status_mu() {
  static std::mutex mu;
  return mu;
}
int add_status_io(StatusIo io) {
  std::lock_guard<std::mutex> lk(status_mu());
  status_ios().push_back(io);
  return (int)status_ios().size();
}
long long g_slack = 0;
}  // namespace dbg
}  // namespace bds

namespace {

thread_local char g_err[512] = "";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

// timing hook state (per host thread)
thread_local void* const* g_prof_ev = nullptr;
thread_local int g_prof_n = 0;
thread_local int g_launches = 0;
thread_local int g_last_launches = 0;

const char* site_name(int site) {
  static const char* names[] = {"?", "k_chunk_local", "k_chunk_carry", "k_block_scan", "k_active_block",
                                "k_bwd_noisy", "k_bwd_carry", "k_bwd_clean", "k_reduce_tok", "k_reduce_par",
                                "k_ssd_block_state", "k_ssd_state_pass", "k_ssd_block_scan", "k_ssd_bwd_tile",
                                "k_ssd_bwd_state"};
  static_assert(sizeof(names) / sizeof(names[0]) == bds::kSiteCount, "one name per debug site");
  return site > 0 && site < bds::kSiteCount ? names[site] : names[0];
}

// Debug build: after an entry point's launches, wait for them and read every
// translation unit's status word (clearing it). Returns BDSCAN_OK or the code.
int debug_check(int launches) {
  if (!BDSCAN_DEBUG || launches == 0) return BDSCAN_OK;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return fail(BDSCAN_ERR_CUDA, "debug status check: %s", cudaGetErrorString(e));
  bds::DevStatus first = {0, 0, 0, 0};
  std::lock_guard<std::mutex> lk(bds::dbg::status_mu());
  for (bds::dbg::StatusIo io : bds::dbg::status_ios()) {
    bds::DevStatus st;
    const int r = io(&st, 1, bds::dbg::g_slack);
    if (r != 0) return fail(BDSCAN_ERR_CUDA, "debug status read: %s", cudaGetErrorString((cudaError_t)r));
    if (st.code != 0 && first.code == 0) first = st;
  }
  if (first.code == bds::kStatusRange)
    return fail(BDSCAN_ERR_DEVICE, "device status: %s: offset %lld outside the extent %lld its sizes give (the CTA skipped its work)",
                site_name(first.site), first.value, first.limit);
  if (first.code != 0)
    return fail(BDSCAN_ERR_DEVICE, "device status: %s: non-finite value at index %lld", site_name(first.site), first.value);
  return BDSCAN_OK;
}

int ok() {
  const int rc = debug_check(g_launches);
  if (rc != BDSCAN_OK) return rc;
  g_err[0] = '\0';
  g_last_launches = g_launches;
  return BDSCAN_OK;
}

// Called after every kernel launch of an entry point.
cudaError_t launched(cudaError_t e, cudaStream_t s) {
  if (e != cudaSuccess) return e;
  if (g_prof_ev != nullptr && g_launches < g_prof_n) e = cudaEventRecord((cudaEvent_t)g_prof_ev[g_launches], s);
  ++g_launches;
  return e;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(BDSCAN_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int64_t blocks_per_chunk(int64_t Bs) { return Bs >= 128 ? 1 : 128 / Bs; }

struct Call {
  bds::Geo g;
  int dt;  // 0 f32/f32, 1 bf16/bf16, 2 bf16/f32
  int N;
  size_t in_elt;
};

// d_state of the kernels themselves; other sizes run in state groups
bool direct_N(int N) { return N == 8 || N == 16; }

// Validates the dimensions common to every entry point; d_state is any
// multiple of 4 up to 64 (state groups above, see check_dims).
int check_dims_any(const bdscan_dims* dm, Call* c, const char* fn) {
  g_launches = 0;
  if (dm == nullptr) return fail(BDSCAN_ERR_ARG, "%s: dims is NULL", fn);
  if (dm->batch < 0 || dm->len < 0) return fail(BDSCAN_ERR_ARG, "%s: negative batch or len", fn);
  if (dm->block <= 0) return fail(BDSCAN_ERR_ARG, "%s: block must be positive", fn);
  if (dm->d_inner <= 0 || dm->d_state <= 0) return fail(BDSCAN_ERR_ARG, "%s: d_inner and d_state must be positive", fn);
  if (dm->len % dm->block != 0)
    return fail(BDSCAN_ERR_ARG, "%s: len (%lld) is not a multiple of block (%lld)", fn, (long long)dm->len,
                (long long)dm->block);
  if (dm->dtype != BDSCAN_F32 && dm->dtype != BDSCAN_BF16) return fail(BDSCAN_ERR_ARG, "%s: bad dtype %d", fn, dm->dtype);
  if (dm->out_dtype != BDSCAN_F32 && dm->out_dtype != BDSCAN_BF16)
    return fail(BDSCAN_ERR_ARG, "%s: bad out_dtype %d", fn, dm->out_dtype);
  if (dm->dtype == BDSCAN_F32 && dm->out_dtype == BDSCAN_BF16)
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: f32 inputs with bf16 outputs are not supported", fn);
  if (dm->d_state > 64 || dm->d_state % 4 != 0)
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: d_state %lld not supported (a multiple of 4 up to 64)", fn,
                (long long)dm->d_state);
  const int64_t vec = dm->dtype == BDSCAN_BF16 ? 8 : 4;
  if (dm->d_inner % vec != 0)
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: d_inner %lld must be a multiple of %lld for this dtype", fn,
                (long long)dm->d_inner, (long long)vec);
  if (dm->batch > 65535) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: batch above 65535", fn);
  const int64_t nb = dm->len / dm->block;
  if (nb > (int64_t)1 << 30) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: too many blocks", fn);
  const int64_t m = blocks_per_chunk(dm->block);
  const int64_t nc = (nb + m - 1) / m;
  if (nc > 65535) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: len too long for one call (more than 65535 chunks)", fn);
  c->g.Bt = dm->batch;
  c->g.L = dm->len;
  c->g.Bs = dm->block;
  c->g.D = dm->d_inner;
  c->g.nb = (int)nb;
  c->g.m = (int)m;
  c->g.nc = (int)nc;
  c->g.nc_full = (int)(nb / m);
  c->g.G = (int)((dm->d_inner + bds::kCtaHost - 1) / bds::kCtaHost);
  c->dt = dm->dtype == BDSCAN_F32 ? 0 : (dm->out_dtype == BDSCAN_BF16 ? 1 : 2);
  c->N = (int)dm->d_state;
  c->in_elt = dm->dtype == BDSCAN_F32 ? 4 : 2;
  return BDSCAN_OK;
}

// The same for entry points without state groups: d_state 8 or 16.
int check_dims(const bdscan_dims* dm, Call* c, const char* fn) {
  const int rc = check_dims_any(dm, c, fn);
  if (rc != BDSCAN_OK) return rc;
  if (!direct_N(c->N)) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: d_state %d not supported here (8 or 16)", fn, c->N);
  return BDSCAN_OK;
}

#define REQ(ptr, fn, name)                                                              \
  do {                                                                                  \
    if ((ptr) == nullptr) return fail(BDSCAN_ERR_ARG, "%s: %s is NULL", fn, name);      \
    if (!aligned16(ptr)) return fail(BDSCAN_ERR_ARG, "%s: %s is not 16-byte aligned", fn, name); \
  } while (0)
#define OPT(ptr, fn, name)                                                              \
  do {                                                                                  \
    if ((ptr) != nullptr && !aligned16(ptr))                                            \
      return fail(BDSCAN_ERR_ARG, "%s: %s is not 16-byte aligned", fn, name);           \
  } while (0)

size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t fwd_ws(const bds::Geo& g, int N) {
  return al256((size_t)g.Bt * (g.nc + 1) * g.D * N * 4) + al256((size_t)g.Bt * g.nc * g.D * 4);
}

struct BwdWs {
  size_t dS, Lc, sdtc, part_tok, part_A, part_D, ck, total;
};
BwdWs bwd_ws(const bds::Geo& g, int N) {
  BwdWs w;
  size_t o = 0;
  w.dS = o;
  o += al256((size_t)g.Bt * g.nb * g.D * N * 4);
  w.Lc = o;
  o += al256((size_t)g.Bt * g.nc * g.D * N * 4);
  w.sdtc = o;
  o += al256((size_t)g.Bt * g.nc * g.D * 4);
  w.part_tok = o;
  o += al256((size_t)6 * g.Bt * g.L * g.G * N * 4);
  w.part_A = o;
  o += al256((size_t)3 * g.Bt * g.nc * g.D * N * 4);
  w.part_D = o;
  o += al256((size_t)2 * g.Bt * g.nc * g.D * 4);
  // segment checkpoints of long blocks: one region per CTA of each TMEM kernel
  // (grid G x nc x Bt), (Bs/16 - 1) x N x 128 floats each
  w.ck = o;
  if (g.Bs > bds::kCkSmemMaxBs) o += 2 * al256((size_t)g.G * g.nc * g.Bt * (g.Bs / 16 - 1) * N * bds::kCtaHost * 4);
  w.total = o;
  return w;
}

// Blocks up to 256 tokens (the paper's block, hyperparameter table); the
// backward keeps the segment checkpoints of blocks above kCkSmemMaxBs in
// global memory.
int check_block_limits(const Call& c, bool backward, const char* fn) {
  if (backward && c.g.Bs > 256) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: backward block %lld above 256", fn, (long long)c.g.Bs);
  if (c.g.Bs > 256) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: block %lld above 256", fn, (long long)c.g.Bs);
  if (backward && c.g.Bs > 16 && c.g.Bs % 16 != 0)
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: backward needs block <= 16 or a multiple of 16", fn);
  return BDSCAN_OK;
}

void fill_clean(bds::FwdParams& p, const bdscan_clean* cl) {
  p.xc = cl->x;
  p.dtc = cl->dt;
  p.Bc = cl->B;
  p.Cc = cl->C;
}
void fill_noisy(bds::FwdParams& p, const bdscan_noisy* nz) {
  p.xn = nz->x;
  p.dtf = nz->dt_f;
  p.Bf = nz->B_f;
  p.Cf = nz->C_f;
  p.dtr = nz->dt_r;
  p.Br = nz->B_r;
  p.Cr = nz->C_r;
}

int check_clean(const bdscan_clean* cl, const char* fn) {
  if (cl == nullptr) return fail(BDSCAN_ERR_ARG, "%s: clean is NULL", fn);
  REQ(cl->x, fn, "clean.x");
  REQ(cl->dt, fn, "clean.dt");
  REQ(cl->B, fn, "clean.B");
  REQ(cl->C, fn, "clean.C");
  return BDSCAN_OK;
}
int check_noisy(const bdscan_noisy* nz, const char* fn) {
  if (nz == nullptr) return fail(BDSCAN_ERR_ARG, "%s: noisy is NULL", fn);
  REQ(nz->x, fn, "noisy.x");
  REQ(nz->dt_f, fn, "noisy.dt_f");
  REQ(nz->B_f, fn, "noisy.B_f");
  REQ(nz->C_f, fn, "noisy.C_f");
  REQ(nz->dt_r, fn, "noisy.dt_r");
  REQ(nz->B_r, fn, "noisy.B_r");
  REQ(nz->C_r, fn, "noisy.C_r");
  return BDSCAN_OK;
}
int check_params(const bdscan_params* pr, const char* fn) {
  if (pr == nullptr) return fail(BDSCAN_ERR_ARG, "%s: params is NULL", fn);
  REQ(pr->A_f, fn, "params.A_f");
  REQ(pr->D_f, fn, "params.D_f");
  REQ(pr->A_r, fn, "params.A_r");
  REQ(pr->D_r, fn, "params.D_r");
  return BDSCAN_OK;
}

// Runs the chunk-local scan and the chunk carry: hst then holds every chunk
// start state (slot nc_full: the state after the last full chunk).
int run_chunk_states(const Call& c, bds::FwdParams& p, cudaStream_t s, const char* fn) {
  cudaError_t e = cudaSuccess;
  if (c.g.nc_full > 0) e = launched(bds::launch_chunk_local(c.dt, c.N, p, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  e = launched(bds::launch_chunk_carry(c.N, p, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return BDSCAN_OK;
}


// ---------------------------------------------------------------------------
// State groups: d_state other than 8 or 16 (a multiple of 4 up to 64). The
// scan kernels run once per group of 16 states (the last one 8 or 16,
// zero-padded: zero B, C and A add nothing), on gathered copies of the
// group's B, C, A and states, with fp32 outputs that are added in group
// order; the D terms come from group 0 only (the others get D = 0).
// ---------------------------------------------------------------------------
struct GroupPlan {
  int G;
  int n0[4], gs[4];
};
GroupPlan group_plan(int N) {
  GroupPlan q;
  q.G = (N + 15) / 16;
  for (int g = 0; g < q.G; ++g) {
    q.n0[g] = 16 * g;
    const int rem = N - 16 * g;
    q.gs[g] = rem >= 16 ? 16 : (rem <= 8 ? 8 : 16);
  }
  return q;
}

struct Carve {
  size_t o = 0;
  size_t take(size_t bytes) {
    const size_t at = o;
    o += al256(bytes);
    return at;
  }
};

// the per-group calls write fp32 outputs: dt code 0 (f32 inputs) or 2 (bf16
// inputs, f32 outputs); the caller's outputs have element size out_elt
int group_dt(const Call& c) { return c.dt == 0 ? 0 : 2; }
int out_elt(const Call& c) { return c.dt == 1 ? 2 : 4; }

struct FwdGroupWs {
  size_t scan, bc[6], a[2], dzero, st, acc[2], tmp[2], total;
};
FwdGroupWs fwd_group_ws(const Call& c) {
  const bds::Geo& g = c.g;
  FwdGroupWs w;
  Carve k;
  w.scan = k.take(fwd_ws(g, 16));
  for (int i = 0; i < 6; ++i) w.bc[i] = k.take((size_t)g.Bt * g.L * 16 * c.in_elt);
  for (int i = 0; i < 2; ++i) w.a[i] = k.take((size_t)g.D * 16 * 4);
  w.dzero = k.take((size_t)g.D * 4);
  w.st = k.take((size_t)g.Bt * g.nb * g.D * 16 * 4);
  for (int i = 0; i < 2; ++i) w.acc[i] = k.take((size_t)g.Bt * g.L * g.D * 4);
  for (int i = 0; i < 2; ++i) w.tmp[i] = k.take((size_t)g.Bt * g.L * g.D * 4);
  w.total = k.o;
  return w;
}

struct BndGroupWs {
  size_t scan, bc[2], a, dzero, st, init, acc, tmp, total;
};
BndGroupWs bnd_group_ws(const Call& c, int emit_all) {
  const bds::Geo& g = c.g;
  BndGroupWs w;
  Carve k;
  w.scan = k.take(fwd_ws(g, 16));
  for (int i = 0; i < 2; ++i) w.bc[i] = k.take((size_t)g.Bt * g.L * 16 * c.in_elt);
  w.a = k.take((size_t)g.D * 16 * 4);
  w.dzero = k.take((size_t)g.D * 4);
  w.st = k.take((size_t)g.Bt * (emit_all ? g.nb : 1) * g.D * 16 * 4);
  w.init = k.take((size_t)g.Bt * g.D * 16 * 4);
  w.acc = k.take((size_t)g.Bt * g.L * g.D * 4);
  w.tmp = k.take((size_t)g.Bt * g.L * g.D * 4);
  w.total = k.o;
  return w;
}

struct BwdGroupWs {
  size_t scan, bc[6], a[2], dzero, st, dst, acc[5], tmp[5], gbc[6], ga[2], gd[2], total;
};
BwdGroupWs bwd_group_ws(const Call& c) {
  const bds::Geo& g = c.g;
  bds::Geo gmax = g;
  gmax.nc = bds::bwd_max_chunks(g);
  BwdGroupWs w;
  Carve k;
  w.scan = k.take(bwd_ws(gmax, 16).total);
  for (int i = 0; i < 6; ++i) w.bc[i] = k.take((size_t)g.Bt * g.L * 16 * c.in_elt);
  for (int i = 0; i < 2; ++i) w.a[i] = k.take((size_t)g.D * 16 * 4);
  w.dzero = k.take((size_t)g.D * 4);
  w.st = k.take((size_t)g.Bt * g.nb * g.D * 16 * 4);
  w.dst = k.take((size_t)g.Bt * g.nb * g.D * 16 * 4);
  for (int i = 0; i < 5; ++i) w.acc[i] = k.take((size_t)g.Bt * g.L * g.D * 4);
  for (int i = 0; i < 5; ++i) w.tmp[i] = k.take((size_t)g.Bt * g.L * g.D * 4);
  for (int i = 0; i < 6; ++i) w.gbc[i] = k.take((size_t)g.Bt * g.L * 16 * 4);
  for (int i = 0; i < 2; ++i) w.ga[i] = k.take((size_t)g.D * 16 * 4);
  for (int i = 0; i < 2; ++i) w.gd[i] = k.take((size_t)g.D * 4);
  w.total = k.o;
  return w;
}

struct ActGroupWs {
  size_t bc[4], a[2], dzero, seed, acc, tmp, total;
};
ActGroupWs act_group_ws(const Call& c) {
  const bds::Geo& g = c.g;
  ActGroupWs w;
  Carve k;
  for (int i = 0; i < 4; ++i) w.bc[i] = k.take((size_t)g.Bt * g.L * 16 * c.in_elt);
  for (int i = 0; i < 2; ++i) w.a[i] = k.take((size_t)g.D * 16 * 4);
  w.dzero = k.take((size_t)g.D * 4);
  w.seed = k.take((size_t)g.Bt * g.D * 16 * 4);
  w.acc = k.take((size_t)g.Bt * g.L * g.D * 4);
  w.tmp = k.take((size_t)g.Bt * g.L * g.D * 4);
  w.total = k.o;
  return w;
}

// gathers of one group (B/C rows of the tokens, A rows of the channels)
cudaError_t gather(const void* src, int elt, int64_t rows, int N, int n0, int gs, char* dst, cudaStream_t s) {
  return launched(bds::launch_group_gather(src, elt, rows, N, n0, gs, dst, s), s);
}

int grouped_forward(const Call& c, const bdscan_clean* clean, const bdscan_noisy* noisy, const bdscan_params* pr,
                    void* y_c, void* y_n, float* states, char* ws, cudaStream_t s, const char* fn) {
  const bds::Geo& g = c.g;
  const FwdGroupWs w = fwd_group_ws(c);
  const GroupPlan q = group_plan(c.N);
  const int64_t tok = g.Bt * g.L, n = g.Bt * g.L * g.D;
  cudaError_t e = cudaMemsetAsync(ws + w.dzero, 0, (size_t)g.D * 4, s);
  const void* bc[6] = {clean->B, clean->C, noisy->B_f, noisy->C_f, noisy->B_r, noisy->C_r};
  for (int gi = 0; gi < q.G && e == cudaSuccess; ++gi) {
    const int n0 = q.n0[gi], gs = q.gs[gi];
    for (int i = 0; i < 6 && e == cudaSuccess; ++i) e = gather(bc[i], (int)c.in_elt, tok, c.N, n0, gs, ws + w.bc[i], s);
    if (e == cudaSuccess) e = gather(pr->A_f, 4, g.D, c.N, n0, gs, ws + w.a[0], s);
    if (e == cudaSuccess) e = gather(pr->A_r, 4, g.D, c.N, n0, gs, ws + w.a[1], s);
    if (e != cudaSuccess) break;
    bds::FwdParams p;
    memset(&p, 0, sizeof(p));
    p.g = g;
    p.xc = clean->x;
    p.dtc = clean->dt;
    p.Bc = ws + w.bc[0];
    p.Cc = ws + w.bc[1];
    p.xn = noisy->x;
    p.dtf = noisy->dt_f;
    p.Bf = ws + w.bc[2];
    p.Cf = ws + w.bc[3];
    p.dtr = noisy->dt_r;
    p.Br = ws + w.bc[4];
    p.Cr = ws + w.bc[5];
    p.Af = (const float*)(ws + w.a[0]);
    p.Ar = (const float*)(ws + w.a[1]);
    p.Df = gi == 0 ? pr->D_f : (const float*)(ws + w.dzero);
    p.Dr = gi == 0 ? pr->D_r : (const float*)(ws + w.dzero);
    p.yc = ws + (gi == 0 ? w.acc[0] : w.tmp[0]);
    p.yn = ws + (gi == 0 ? w.acc[1] : w.tmp[1]);
    p.states = (float*)(ws + w.st);
    e = bds::api_run_forward(group_dt(c), gs, p, ws + w.scan, s);
    for (int i = 0; i < 2 && gi > 0 && e == cudaSuccess; ++i)
      e = launched(bds::launch_group_add((float*)(ws + w.acc[i]), (const float*)(ws + w.tmp[i]), n, s), s);
    if (e == cudaSuccess)
      e = launched(bds::launch_group_scatter((const float*)(ws + w.st), g.Bt * g.nb * g.D, c.N, n0, gs, states, 4, s), s);
  }
  if (e == cudaSuccess) e = launched(bds::launch_group_out((const float*)(ws + w.acc[0]), y_c, out_elt(c), n, s), s);
  if (e == cudaSuccess) e = launched(bds::launch_group_out((const float*)(ws + w.acc[1]), y_n, out_elt(c), n, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int grouped_boundary(const Call& c, const bdscan_clean* clean, const float* A_f, const float* D_f,
                     const float* init_state, void* y_c, float* states, int emit_all, char* ws, cudaStream_t s,
                     const char* fn) {
  const bds::Geo& g = c.g;
  const BndGroupWs w = bnd_group_ws(c, emit_all);
  const GroupPlan q = group_plan(c.N);
  const int64_t tok = g.Bt * g.L, n = g.Bt * g.L * g.D, srows = g.Bt * (emit_all ? g.nb : 1) * g.D;
  cudaError_t e = cudaMemsetAsync(ws + w.dzero, 0, (size_t)g.D * 4, s);
  for (int gi = 0; gi < q.G && e == cudaSuccess; ++gi) {
    const int n0 = q.n0[gi], gs = q.gs[gi];
    e = gather(clean->B, (int)c.in_elt, tok, c.N, n0, gs, ws + w.bc[0], s);
    if (e == cudaSuccess) e = gather(clean->C, (int)c.in_elt, tok, c.N, n0, gs, ws + w.bc[1], s);
    if (e == cudaSuccess) e = gather(A_f, 4, g.D, c.N, n0, gs, ws + w.a, s);
    if (e == cudaSuccess && init_state != nullptr) e = gather(init_state, 4, g.Bt * g.D, c.N, n0, gs, ws + w.init, s);
    if (e != cudaSuccess) break;
    bds::FwdParams p;
    memset(&p, 0, sizeof(p));
    p.g = g;
    p.xc = clean->x;
    p.dtc = clean->dt;
    p.Bc = ws + w.bc[0];
    p.Cc = ws + w.bc[1];
    p.Af = (const float*)(ws + w.a);
    p.Df = gi == 0 ? D_f : (const float*)(ws + w.dzero);
    p.yc = y_c != nullptr ? (void*)(ws + (gi == 0 ? w.acc : w.tmp)) : nullptr;
    p.init = init_state != nullptr ? (const float*)(ws + w.init) : nullptr;
    p.hst = (float*)(ws + w.scan);
    p.sdt = (float*)(ws + w.scan + al256((size_t)g.Bt * (g.nc + 1) * g.D * 16 * 4));
    e = bds::api_run_boundary(group_dt(c), gs, p, (float*)(ws + w.st), emit_all, s);
    if (e == cudaSuccess && y_c != nullptr && gi > 0)
      e = launched(bds::launch_group_add((float*)(ws + w.acc), (const float*)(ws + w.tmp), n, s), s);
    if (e == cudaSuccess)
      e = launched(bds::launch_group_scatter((const float*)(ws + w.st), srows, c.N, n0, gs, states, 4, s), s);
  }
  if (e == cudaSuccess && y_c != nullptr)
    e = launched(bds::launch_group_out((const float*)(ws + w.acc), y_c, out_elt(c), n, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int grouped_backward(const Call& c, const bdscan_clean* clean, const bdscan_noisy* noisy, const bdscan_params* pr,
                     const float* states, const void* dy_c, const void* dy_n, const float* dstates,
                     const bdscan_clean_grads* gc, const bdscan_noisy_grads* gn, const bdscan_param_grads* gp,
                     char* ws, cudaStream_t s, const char* fn) {
  const bds::Geo& g = c.g;
  const BwdGroupWs w = bwd_group_ws(c);
  const GroupPlan q = group_plan(c.N);
  const int64_t tok = g.Bt * g.L, n = g.Bt * g.L * g.D, srows = g.Bt * g.nb * g.D;
  cudaError_t e = cudaMemsetAsync(ws + w.dzero, 0, (size_t)g.D * 4, s);
  const void* bc[6] = {clean->B, clean->C, noisy->B_f, noisy->C_f, noisy->B_r, noisy->C_r};
  void* gbc_out[6] = {gc->dB, gc->dC, gn->dB_f, gn->dC_f, gn->dB_r, gn->dC_r};
  void* acc_out[5] = {gc->dx, gc->ddt, gn->dx, gn->ddt_f, gn->ddt_r};
  for (int gi = 0; gi < q.G && e == cudaSuccess; ++gi) {
    const int n0 = q.n0[gi], gs = q.gs[gi];
    for (int i = 0; i < 6 && e == cudaSuccess; ++i) e = gather(bc[i], (int)c.in_elt, tok, c.N, n0, gs, ws + w.bc[i], s);
    if (e == cudaSuccess) e = gather(pr->A_f, 4, g.D, c.N, n0, gs, ws + w.a[0], s);
    if (e == cudaSuccess) e = gather(pr->A_r, 4, g.D, c.N, n0, gs, ws + w.a[1], s);
    if (e == cudaSuccess) e = gather(states, 4, srows, c.N, n0, gs, ws + w.st, s);
    if (e == cudaSuccess && dstates != nullptr) e = gather(dstates, 4, srows, c.N, n0, gs, ws + w.dst, s);
    if (e != cudaSuccess) break;
    bds::BwdParams p;
    memset(&p, 0, sizeof(p));
    p.g = g;
    p.xc = clean->x;
    p.dtc = clean->dt;
    p.Bc = ws + w.bc[0];
    p.Cc = ws + w.bc[1];
    p.xn = noisy->x;
    p.dtf = noisy->dt_f;
    p.Bf = ws + w.bc[2];
    p.Cf = ws + w.bc[3];
    p.dtr = noisy->dt_r;
    p.Br = ws + w.bc[4];
    p.Cr = ws + w.bc[5];
    p.Af = (const float*)(ws + w.a[0]);
    p.Ar = (const float*)(ws + w.a[1]);
    p.Df = gi == 0 ? pr->D_f : (const float*)(ws + w.dzero);
    p.Dr = gi == 0 ? pr->D_r : (const float*)(ws + w.dzero);
    p.states = (const float*)(ws + w.st);
    p.dyc = dy_c;
    p.dyn = dy_n;
    p.dstates = dstates != nullptr ? (const float*)(ws + w.dst) : nullptr;
    const size_t* dst = gi == 0 ? w.acc : w.tmp;
    p.dxc = ws + dst[0];
    p.ddtc = ws + dst[1];
    p.dxn = ws + dst[2];
    p.ddtf = ws + dst[3];
    p.ddtr = ws + dst[4];
    p.dBc = ws + w.gbc[0];
    p.dCc = ws + w.gbc[1];
    p.dBf = ws + w.gbc[2];
    p.dCf = ws + w.gbc[3];
    p.dBr = ws + w.gbc[4];
    p.dCr = ws + w.gbc[5];
    p.dAf = (float*)(ws + w.ga[0]);
    p.dAr = (float*)(ws + w.ga[1]);
    p.dDf = gi == 0 ? gp->dD_f : (float*)(ws + w.gd[0]);  // the D gradients do not depend on the group
    p.dDr = gi == 0 ? gp->dD_r : (float*)(ws + w.gd[1]);
    e = bds::api_run_backward(group_dt(c), gs, p, ws + w.scan, s);
    for (int i = 0; i < 5 && gi > 0 && e == cudaSuccess; ++i)
      e = launched(bds::launch_group_add((float*)(ws + w.acc[i]), (const float*)(ws + w.tmp[i]), n, s), s);
    for (int i = 0; i < 6 && e == cudaSuccess; ++i)
      e = launched(bds::launch_group_scatter((const float*)(ws + w.gbc[i]), tok, c.N, n0, gs, gbc_out[i], out_elt(c), s), s);
    if (e == cudaSuccess)
      e = launched(bds::launch_group_scatter((const float*)(ws + w.ga[0]), g.D, c.N, n0, gs, gp->dA_f, 4, s), s);
    if (e == cudaSuccess)
      e = launched(bds::launch_group_scatter((const float*)(ws + w.ga[1]), g.D, c.N, n0, gs, gp->dA_r, 4, s), s);
  }
  for (int i = 0; i < 5 && e == cudaSuccess; ++i)
    e = launched(bds::launch_group_out((const float*)(ws + w.acc[i]), acc_out[i], out_elt(c), n, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int grouped_active(const Call& c, const float* seed, const bdscan_noisy* noisy, const bdscan_params* pr, void* y_n,
                   cudaStream_t s, const char* fn) {
  const bds::Geo& g = c.g;
  const ActGroupWs w = act_group_ws(c);
  if (w.total > bds::kGroupScratchBytes)
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: d_state %d needs %zu bytes of group scratch (%zu available)", fn, c.N,
                w.total, bds::kGroupScratchBytes);
  char* ws = (char*)bds::group_scratch();
  if (ws == nullptr) return cuda_fail(cudaGetLastError(), fn);
  const GroupPlan q = group_plan(c.N);
  const int64_t tok = g.Bt * g.L, n = g.Bt * g.L * g.D;
  cudaError_t e = cudaMemsetAsync(ws + w.dzero, 0, (size_t)g.D * 4, s);
  const void* bc[4] = {noisy->B_f, noisy->C_f, noisy->B_r, noisy->C_r};
  for (int gi = 0; gi < q.G && e == cudaSuccess; ++gi) {
    const int n0 = q.n0[gi], gs = q.gs[gi];
    for (int i = 0; i < 4 && e == cudaSuccess; ++i) e = gather(bc[i], (int)c.in_elt, tok, c.N, n0, gs, ws + w.bc[i], s);
    if (e == cudaSuccess) e = gather(pr->A_f, 4, g.D, c.N, n0, gs, ws + w.a[0], s);
    if (e == cudaSuccess) e = gather(pr->A_r, 4, g.D, c.N, n0, gs, ws + w.a[1], s);
    if (e == cudaSuccess) e = gather(seed, 4, g.Bt * g.D, c.N, n0, gs, ws + w.seed, s);
    if (e != cudaSuccess) break;
    bds::FwdParams p;
    memset(&p, 0, sizeof(p));
    p.g = g;
    p.xn = noisy->x;
    p.dtf = noisy->dt_f;
    p.Bf = ws + w.bc[0];
    p.Cf = ws + w.bc[1];
    p.dtr = noisy->dt_r;
    p.Br = ws + w.bc[2];
    p.Cr = ws + w.bc[3];
    p.Af = (const float*)(ws + w.a[0]);
    p.Ar = (const float*)(ws + w.a[1]);
    p.Df = gi == 0 ? pr->D_f : (const float*)(ws + w.dzero);
    p.Dr = gi == 0 ? pr->D_r : (const float*)(ws + w.dzero);
    p.yn = ws + (gi == 0 ? w.acc : w.tmp);
    p.seed = (const float*)(ws + w.seed);
    e = launched(bds::launch_active_block(group_dt(c), gs, p, s), s);
    if (e == cudaSuccess && gi > 0)
      e = launched(bds::launch_group_add((float*)(ws + w.acc), (const float*)(ws + w.tmp), n, s), s);
  }
  if (e == cudaSuccess) e = launched(bds::launch_group_out((const float*)(ws + w.acc), y_n, out_elt(c), n, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

}  // namespace

extern "C" {

const char* bdscan_last_error(void) { return g_err; }

int bdscan_version(void) { return 100; }

int bdscan_profile_events(void* const* events, int n) {
  g_prof_ev = (n > 0) ? events : nullptr;
  g_prof_n = (events != nullptr && n > 0) ? n : 0;
  return BDSCAN_OK;
}

int bdscan_last_launch_count(void) { return g_last_launches; }

int bdscan_debug_build(void) { return BDSCAN_DEBUG; }

int bdscan_debug_set_slack(long long elements) {
  const char* fn = "bdscan_debug_set_slack";
  if (!BDSCAN_DEBUG) return fail(BDSCAN_ERR_UNSUPPORTED, "%s: this is the release build (no device checks)", fn);
  if (elements < 0) return fail(BDSCAN_ERR_ARG, "%s: negative slack %lld", fn, elements);
  std::lock_guard<std::mutex> lk(bds::dbg::status_mu());
  bds::dbg::g_slack = elements;
  for (bds::dbg::StatusIo io : bds::dbg::status_ios()) {
    bds::DevStatus st;
    const int r = io(&st, 0, elements);
    if (r != 0) return fail(BDSCAN_ERR_CUDA, "%s: %s", fn, cudaGetErrorString((cudaError_t)r));
  }
  g_err[0] = '\0';
  return BDSCAN_OK;
}

int64_t bdscan_chunk_tokens(int64_t block) { return block <= 0 ? 0 : blocks_per_chunk(block) * block; }

size_t bdscan_forward_workspace_size(const bdscan_dims* dims) {
  Call c{};
  if (check_dims_any(dims, &c, "bdscan_forward_workspace_size") != BDSCAN_OK) return 0;
  if (!direct_N(c.N)) return fwd_group_ws(c).total;
  return fwd_ws(c.g, c.N);
}

size_t bdscan_boundary_states_workspace_size(const bdscan_dims* dims, int emit_all) {
  (void)emit_all;
  Call c{};
  if (check_dims_any(dims, &c, "bdscan_boundary_states_workspace_size") != BDSCAN_OK) return 0;
  if (!direct_N(c.N)) return bnd_group_ws(c, emit_all).total;
  return fwd_ws(c.g, c.N);
}

size_t bdscan_backward_workspace_size(const bdscan_dims* dims) {
  Call c{};
  if (check_dims_any(dims, &c, "bdscan_backward_workspace_size") != BDSCAN_OK) return 0;
  if (!direct_N(c.N)) return bwd_group_ws(c).total;
  bds::Geo gmax = c.g;
  gmax.nc = bds::bwd_max_chunks(c.g);
  return bwd_ws(gmax, c.N).total;
}

int bdscan_forward(const bdscan_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                   const bdscan_params* params, void* y_c, void* y_n, float* states, void* workspace,
                   size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_forward";
  Call c{};
  int rc = check_dims_any(dims, &c, fn);
  if (rc) return rc;
  if ((rc = check_block_limits(c, false, fn))) return rc;
  if (c.g.Bt == 0 || c.g.L == 0) return ok();
  if ((rc = check_clean(clean, fn)) || (rc = check_noisy(noisy, fn)) || (rc = check_params(params, fn))) return rc;
  REQ(y_c, fn, "y_c");
  REQ(y_n, fn, "y_n");
  REQ(states, fn, "states");
  const size_t need = direct_N(c.N) ? fwd_ws(c.g, c.N) : fwd_group_ws(c).total;
  REQ(workspace, fn, "workspace");
  if (workspace_bytes < need)
    return fail(BDSCAN_ERR_ARG, "%s: workspace of %zu bytes, %zu needed", fn, workspace_bytes, need);
  cudaStream_t s = (cudaStream_t)stream;
  if (!direct_N(c.N)) return grouped_forward(c, clean, noisy, params, y_c, y_n, states, (char*)workspace, s, fn);
  bds::FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = c.g;
  fill_clean(p, clean);
  fill_noisy(p, noisy);
  p.Af = params->A_f;
  p.Df = params->D_f;
  p.Ar = params->A_r;
  p.Dr = params->D_r;
  p.yc = y_c;
  p.yn = y_n;
  p.states = states;
  p.emit_all = 1;
  p.hst = (float*)workspace;
  p.sdt = (float*)((char*)workspace + al256((size_t)c.g.Bt * (c.g.nc + 1) * c.g.D * c.N * 4));
  if ((rc = run_chunk_states(c, p, s, fn))) return rc;
  cudaError_t e = launched(bds::launch_block_scan(c.dt, c.N, 0, c.g.nc, p, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int bdscan_boundary_states(const bdscan_dims* dims, const bdscan_clean* clean, const float* A_f,
                           const float* D_f, const float* init_state, void* y_c, float* states, int emit_all,
                           void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_boundary_states";
  Call c{};
  int rc = check_dims_any(dims, &c, fn);
  if (rc) return rc;
  if ((rc = check_block_limits(c, false, fn))) return rc;
  if (c.g.Bt == 0) return ok();
  cudaStream_t s = (cudaStream_t)stream;
  OPT(init_state, fn, "init_state");
  if (c.g.L == 0) {
    if (emit_all) return ok();
    REQ(states, fn, "states");
    const size_t bytes = (size_t)c.g.Bt * c.g.D * c.N * 4;
    cudaError_t e = init_state ? cudaMemcpyAsync(states, init_state, bytes, cudaMemcpyDeviceToDevice, s)
                               : cudaMemsetAsync(states, 0, bytes, s);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
  }
  if ((rc = check_clean(clean, fn))) return rc;
  REQ(A_f, fn, "A_f");
  REQ(D_f, fn, "D_f");
  REQ(states, fn, "states");
  OPT(y_c, fn, "y_c");
  const size_t need = direct_N(c.N) ? fwd_ws(c.g, c.N) : bnd_group_ws(c, emit_all).total;
  REQ(workspace, fn, "workspace");
  if (workspace_bytes < need)
    return fail(BDSCAN_ERR_ARG, "%s: workspace of %zu bytes, %zu needed", fn, workspace_bytes, need);
  if (!direct_N(c.N))
    return grouped_boundary(c, clean, A_f, D_f, init_state, y_c, states, emit_all, (char*)workspace, s, fn);
  bds::FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = c.g;
  fill_clean(p, clean);
  p.Af = A_f;
  p.Df = D_f;
  p.yc = y_c;
  p.init = init_state;
  p.hst = (float*)workspace;
  p.sdt = (float*)((char*)workspace + al256((size_t)c.g.Bt * (c.g.nc + 1) * c.g.D * c.N * 4));
  cudaError_t e = bds::api_run_boundary(c.dt, c.N, p, states, emit_all, s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int bdscan_active_block(const bdscan_dims* dims, const float* seed, const bdscan_noisy* noisy,
                        const bdscan_params* params, void* y_n, void* stream) {
  const char* fn = "bdscan_active_block";
  Call c{};
  int rc = check_dims_any(dims, &c, fn);
  if (rc) return rc;
  if (dims->len != dims->block && dims->len != 0)
    return fail(BDSCAN_ERR_ARG, "%s: len (%lld) must equal block (%lld)", fn, (long long)dims->len,
                (long long)dims->block);
  if ((rc = check_block_limits(c, false, fn))) return rc;
  if (c.g.Bt == 0 || c.g.L == 0) return ok();
  REQ(seed, fn, "seed");
  if ((rc = check_noisy(noisy, fn)) || (rc = check_params(params, fn))) return rc;
  REQ(y_n, fn, "y_n");
  if (!direct_N(c.N)) return grouped_active(c, seed, noisy, params, y_n, (cudaStream_t)stream, fn);
  bds::FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = c.g;
  fill_noisy(p, noisy);
  p.Af = params->A_f;
  p.Df = params->D_f;
  p.Ar = params->A_r;
  p.Dr = params->D_r;
  p.yn = y_n;
  p.seed = seed;
  cudaError_t e = launched(bds::launch_active_block(c.dt, c.N, p, (cudaStream_t)stream), (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

size_t bdscan_active_block_adaln_workspace_size(const bdscan_dims* dims) {
  Call c{};
  if (check_dims(dims, &c, "bdscan_active_block_adaln_workspace_size") != BDSCAN_OK) return 0;
  return al256((size_t)c.g.Bt * c.g.L * sizeof(float2));
}

int bdscan_active_block_adaln(const bdscan_dims* dims, const float* seed, const bdscan_noisy* noisy,
                              const bdscan_params* params, const bdscan_adaln* mod, void* out, void* workspace,
                              size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_active_block_adaln";
  Call c{};
  int rc = check_dims(dims, &c, fn);
  if (rc) return rc;
  if (dims->len != dims->block && dims->len != 0)
    return fail(BDSCAN_ERR_ARG, "%s: len (%lld) must equal block (%lld)", fn, (long long)dims->len,
                (long long)dims->block);
  if ((rc = check_block_limits(c, false, fn))) return rc;
  if (c.g.Bs > 128)  // the modulated block is kept in shared memory next to the scan's
    return fail(BDSCAN_ERR_UNSUPPORTED, "%s: block %lld above 128", fn, (long long)c.g.Bs);
  if (c.g.Bt == 0 || c.g.L == 0) return ok();
  REQ(seed, fn, "seed");
  if ((rc = check_noisy(noisy, fn)) || (rc = check_params(params, fn))) return rc;
  if (mod == nullptr) return fail(BDSCAN_ERR_ARG, "%s: mod is NULL", fn);
  REQ(mod->shift, fn, "mod.shift");
  REQ(mod->scale, fn, "mod.scale");
  REQ(mod->gate, fn, "mod.gate");
  if (!(mod->eps >= 0.f)) return fail(BDSCAN_ERR_ARG, "%s: eps must be a non-negative number", fn);
  REQ(out, fn, "out");
  const size_t need = al256((size_t)c.g.Bt * c.g.L * sizeof(float2));
  REQ(workspace, fn, "workspace");
  if (workspace_bytes < need)
    return fail(BDSCAN_ERR_ARG, "%s: workspace of %zu bytes, %zu needed", fn, workspace_bytes, need);
  cudaStream_t s = (cudaStream_t)stream;
  bds::FwdParams p;
  memset(&p, 0, sizeof(p));
  p.g = c.g;
  fill_noisy(p, noisy);
  p.Af = params->A_f;
  p.Df = params->D_f;
  p.Ar = params->A_r;
  p.Dr = params->D_r;
  p.yn = out;
  p.seed = seed;
  p.shift = mod->shift;
  p.scale = mod->scale;
  p.gate = mod->gate;
  p.ln_stats = (const float2*)workspace;
  cudaError_t e = launched(
      bds::launch_ln_stats(c.dt, noisy->x, c.g.Bt * c.g.L, c.g.D, mod->eps, (float2*)workspace, s), s);
  if (e == cudaSuccess) e = launched(bds::launch_active_block_adaln(c.dt, c.N, p, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

size_t bdscan_full_bidir_workspace_size(const bdscan_dims* dims) {
  Call c{};
  if (check_dims(dims, &c, "bdscan_full_bidir_workspace_size") != BDSCAN_OK) return 0;
  const size_t y32 = al256((size_t)c.g.Bt * c.g.L * c.g.D * 4);
  return fwd_ws(c.g, c.N) + 2 * y32;
}

int bdscan_full_bidir_forward(const bdscan_dims* dims, const bdscan_noisy* noisy, const bdscan_params* params,
                              void* y, void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_full_bidir_forward";
  Call c{};
  int rc = check_dims(dims, &c, fn);
  if (rc) return rc;
  if ((rc = check_block_limits(c, false, fn))) return rc;
  if (c.g.Bt == 0 || c.g.L == 0) return ok();
  if ((rc = check_noisy(noisy, fn)) || (rc = check_params(params, fn))) return rc;
  REQ(y, fn, "y");
  const size_t y32 = al256((size_t)c.g.Bt * c.g.L * c.g.D * 4), fws = fwd_ws(c.g, c.N);
  REQ(workspace, fn, "workspace");
  if (workspace_bytes < fws + 2 * y32)
    return fail(BDSCAN_ERR_ARG, "%s: workspace of %zu bytes, %zu needed", fn, workspace_bytes, fws + 2 * y32);
  cudaStream_t s = (cudaStream_t)stream;
  float* yf = (float*)((char*)workspace + fws);
  float* yr = (float*)((char*)workspace + fws + y32);
  const int dt_scan = c.dt == 0 ? 0 : 2;  // fp32 outputs of each direction
  for (int dir = 0; dir < 2; ++dir) {
    bds::FwdParams p;
    memset(&p, 0, sizeof(p));
    p.g = c.g;
    p.xc = noisy->x;
    p.dtc = dir == 0 ? noisy->dt_f : noisy->dt_r;
    p.Bc = dir == 0 ? noisy->B_f : noisy->B_r;
    p.Cc = dir == 0 ? noisy->C_f : noisy->C_r;
    p.Af = dir == 0 ? params->A_f : params->A_r;
    p.Df = dir == 0 ? params->D_f : params->D_r;
    p.yc = dir == 0 ? yf : yr;
    p.rev = dir;
    p.hst = (float*)workspace;  // the chunk states of one direction, then of the other
    p.sdt = (float*)((char*)workspace + al256((size_t)c.g.Bt * (c.g.nc + 1) * c.g.D * c.N * 4));
    if ((rc = run_chunk_states(c, p, s, fn))) return rc;
    cudaError_t e = launched(bds::launch_block_scan(dt_scan, c.N, dir == 0 ? 1 : 2, c.g.nc, p, s), s);
    if (e != cudaSuccess) return cuda_fail(e, fn);
  }
  cudaError_t e = launched(bds::launch_combine(c.dt != 1, yf, yr, y, c.g.Bt * c.g.L * c.g.D, s), s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

int bdscan_backward(const bdscan_dims* dims, const bdscan_clean* clean, const bdscan_noisy* noisy,
                    const bdscan_params* params, const float* states, const void* dy_c, const void* dy_n,
                    const float* dstates, const bdscan_clean_grads* gclean, const bdscan_noisy_grads* gnoisy,
                    const bdscan_param_grads* gparams, void* workspace, size_t workspace_bytes, void* stream) {
  const char* fn = "bdscan_backward";
  Call c{};
  int rc = check_dims_any(dims, &c, fn);
  if (rc) return rc;
  if ((rc = check_block_limits(c, true, fn))) return rc;
  if (gparams == nullptr) return fail(BDSCAN_ERR_ARG, "%s: gparams is NULL", fn);
  REQ(gparams->dA_f, fn, "dA_f");
  REQ(gparams->dD_f, fn, "dD_f");
  REQ(gparams->dA_r, fn, "dA_r");
  REQ(gparams->dD_r, fn, "dD_r");
  cudaStream_t s = (cudaStream_t)stream;
  if (c.g.Bt == 0 || c.g.L == 0) {
    const size_t an = (size_t)c.g.D * c.N * 4, dn = (size_t)c.g.D * 4;
    cudaError_t e = cudaMemsetAsync(gparams->dA_f, 0, an, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dA_r, 0, an, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dD_f, 0, dn, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(gparams->dD_r, 0, dn, s);
    if (e != cudaSuccess) return cuda_fail(e, fn);
    return ok();
  }
  if ((rc = check_clean(clean, fn)) || (rc = check_noisy(noisy, fn)) || (rc = check_params(params, fn))) return rc;
  REQ(states, fn, "states");
  OPT(dy_c, fn, "dy_c");
  REQ(dy_n, fn, "dy_n");
  OPT(dstates, fn, "dstates");
  if (gclean == nullptr || gnoisy == nullptr) return fail(BDSCAN_ERR_ARG, "%s: gradient struct is NULL", fn);
  REQ(gclean->dx, fn, "gclean.dx");
  REQ(gclean->ddt, fn, "gclean.ddt");
  REQ(gclean->dB, fn, "gclean.dB");
  REQ(gclean->dC, fn, "gclean.dC");
  REQ(gnoisy->dx, fn, "gnoisy.dx");
  REQ(gnoisy->ddt_f, fn, "gnoisy.ddt_f");
  REQ(gnoisy->dB_f, fn, "gnoisy.dB_f");
  REQ(gnoisy->dC_f, fn, "gnoisy.dC_f");
  REQ(gnoisy->ddt_r, fn, "gnoisy.ddt_r");
  REQ(gnoisy->dB_r, fn, "gnoisy.dB_r");
  REQ(gnoisy->dC_r, fn, "gnoisy.dC_r");
  bds::Geo gmax = c.g;
  gmax.nc = bds::bwd_max_chunks(c.g);
  const size_t need = direct_N(c.N) ? bwd_ws(gmax, c.N).total : bwd_group_ws(c).total;
  REQ(workspace, fn, "workspace");
  if (workspace_bytes < need)
    return fail(BDSCAN_ERR_ARG, "%s: workspace of %zu bytes, %zu needed", fn, workspace_bytes, need);
  if (!direct_N(c.N))
    return grouped_backward(c, clean, noisy, params, states, dy_c, dy_n, dstates, gclean, gnoisy, gparams,
                            (char*)workspace, s, fn);
  bds::BwdParams p;
  memset(&p, 0, sizeof(p));
  p.xc = clean->x;
  p.dtc = clean->dt;
  p.Bc = clean->B;
  p.Cc = clean->C;
  p.xn = noisy->x;
  p.dtf = noisy->dt_f;
  p.Bf = noisy->B_f;
  p.Cf = noisy->C_f;
  p.dtr = noisy->dt_r;
  p.Br = noisy->B_r;
  p.Cr = noisy->C_r;
  p.Af = params->A_f;
  p.Df = params->D_f;
  p.Ar = params->A_r;
  p.Dr = params->D_r;
  p.states = states;
  p.dyc = dy_c;
  p.dyn = dy_n;
  p.dstates = dstates;
  p.dxc = gclean->dx;
  p.ddtc = gclean->ddt;
  p.dBc = gclean->dB;
  p.dCc = gclean->dC;
  p.dxn = gnoisy->dx;
  p.ddtf = gnoisy->ddt_f;
  p.dBf = gnoisy->dB_f;
  p.dCf = gnoisy->dC_f;
  p.ddtr = gnoisy->ddt_r;
  p.dBr = gnoisy->dB_r;
  p.dCr = gnoisy->dC_r;
  p.dAf = gparams->dA_f;
  p.dDf = gparams->dD_f;
  p.dAr = gparams->dA_r;
  p.dDr = gparams->dD_r;
  p.g = c.g;
  cudaError_t e = bds::api_run_backward(c.dt, c.N, p, workspace, s);
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return ok();
}

}  // extern "C"

namespace bds {

int api_fail(int code, const char* msg) { return fail(code, "%s", msg); }

int api_ok() { return ok(); }

// Kernel-launch bookkeeping for entry points defined in other files: reset at
// the start of a call, then every launch goes through api_launched.
void api_begin() { g_launches = 0; }

cudaError_t api_launched(cudaError_t e, cudaStream_t s) { return launched(e, s); }

// Kernel attributes are set once per (kernel, device, size): repeated calls
// (an active-block loop) then skip the runtime calls on their host path.
cudaError_t set_smem_cached(const void* fn, int bytes, int carveout) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  struct Entry {
    const void* fn;
    int dev, bytes, carveout;
  };
  static std::mutex mu;
  static Entry tab[256];
  static int n = 0;
  {
    std::lock_guard<std::mutex> lk(mu);
    for (int i = 0; i < n; ++i)
      if (tab[i].fn == fn && tab[i].dev == dev && tab[i].bytes >= bytes && tab[i].carveout == carveout)
        return cudaSuccess;
  }
  if ((e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess) return e;
  if (carveout >= 0 && (e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, carveout)) !=
                           cudaSuccess)
    return e;
  std::lock_guard<std::mutex> lk(mu);
  for (int i = 0; i < n; ++i)
    if (tab[i].fn == fn && tab[i].dev == dev && tab[i].carveout == carveout) {
      if (bytes > tab[i].bytes) tab[i].bytes = bytes;
      return cudaSuccess;
    }
  if (n < 256) tab[n++] = Entry{fn, dev, bytes, carveout};
  return cudaSuccess;
}

// Multiprocessor count of the current device, looked up once per device.
int sm_count_cached() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return 0;
  static std::atomic<int> counts[256];
  int v = counts[dev].load(std::memory_order_relaxed);
  if (v > 0) return v;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) return 0;
  counts[dev].store(v, std::memory_order_relaxed);
  return v;
}

// Validation shared with other entry points that take forward-side dims.
int api_check_forward_dims(const void* dims, Geo* g, int* dt, int* N, const char* fn) {
  Call c{};
  int rc = check_dims((const bdscan_dims*)dims, &c, fn);
  if (rc) return rc;
  if ((rc = check_block_limits(c, false, fn))) return rc;
  *g = c.g;
  *dt = c.dt;
  *N = c.N;
  return BDSCAN_OK;
}

size_t api_fwd_workspace(const Geo& g, int N) { return fwd_ws(g, N); }

size_t api_bwd_workspace(const Geo& g, int N) {
  Geo gm = g;
  gm.nc = bwd_max_chunks(g);
  return bwd_ws(gm, N).total;
}

// The cache build's launches with p's clean tensors, hst/sdt (the workspace)
// and init set: every block-end state or the final one into `states`, and
// p.yc if set.
cudaError_t api_run_boundary(int dt, int N, FwdParams& p, float* states, int emit_all, cudaStream_t s) {
  const Geo& g = p.g;
  cudaError_t e = cudaSuccess;
  if (g.nc_full > 0) e = launched(launch_chunk_local(dt, N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_chunk_carry(N, p, s), s);
  if (e != cudaSuccess) return e;
  if (emit_all || p.yc != nullptr) {
    p.emit_all = emit_all ? 1 : 0;
    p.states = emit_all ? states : nullptr;
    p.final_state = emit_all ? nullptr : states;
    return launched(launch_block_scan(dt, N, 1, g.nc, p, s), s);
  }
  if (g.nc_full == g.nc) {
    // the state after the last chunk is the carry kernel's final value
    const size_t row = (size_t)g.D * N * 4;
    return cudaMemcpy2DAsync(states, row, p.hst + (size_t)g.nc * g.D * N, (size_t)(g.nc + 1) * row, row,
                             (size_t)g.Bt, cudaMemcpyDeviceToDevice, s);
  }
  // a partial last chunk: rescan it from its start state
  p.emit_all = 0;
  p.final_state = states;
  p.c_begin = g.nc - 1;
  return launched(launch_block_scan(dt, N, 1, 1, p, s), s);
}

// The all-block forward's launches (chunk-local scan, chunk carry, block
// scan) with p's tensors set; the workspace holds the chunk states.
cudaError_t api_run_forward(int dt, int N, FwdParams& p, void* workspace, cudaStream_t s) {
  p.hst = (float*)workspace;
  p.sdt = (float*)((char*)workspace + al256((size_t)p.g.Bt * (p.g.nc + 1) * p.g.D * N * 4));
  p.emit_all = 1;
  cudaError_t e = cudaSuccess;
  if (p.g.nc_full > 0) e = launched(launch_chunk_local(dt, N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_chunk_carry(N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_block_scan(dt, N, 0, p.g.nc, p, s), s);
  return e;
}

// The backward's launches with p's tensors set (p.g the forward geometry):
// its own chunking of each batch row, the workspace layout, five kernels.
cudaError_t api_run_backward(int dt, int N, BwdParams& p, void* workspace, cudaStream_t s) {
  Geo gb = p.g;
  gb.nc = bwd_chunk_count(dt, N, p.g);
  const BwdWs w = bwd_ws(gb, N);
  p.g = gb;
  char* ws = (char*)workspace;
  p.dS = (float*)(ws + w.dS);
  p.Lc = (float*)(ws + w.Lc);
  p.sdtc = (float*)(ws + w.sdtc);
  p.part_tok = (float*)(ws + w.part_tok);
  p.part_A = (float*)(ws + w.part_A);
  p.part_D = (float*)(ws + w.part_D);
  if (gb.Bs > kCkSmemMaxBs) {
    const size_t ckb = al256((size_t)gb.G * gb.nc * gb.Bt * (gb.Bs / 16 - 1) * N * kCtaHost * 4);
    p.ck_noisy = (float*)(ws + w.ck);
    p.ck_clean = (float*)(ws + w.ck + ckb);
  }
  cudaError_t e = launched(launch_bwd_noisy(dt, N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_bwd_carry(N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_bwd_clean(dt, N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_bwd_reduce_tok(dt, N, p, s), s);
  if (e == cudaSuccess) e = launched(launch_bwd_reduce_par(N, p, s), s);
  return e;
}

}  // namespace bds
