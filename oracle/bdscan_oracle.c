/*
 * bdscan_oracle.c -- plain fp64 CPU oracle for the block-restricted
 * bidirectional selective state-space scan of BDLM Mamba-H
 * (arXiv 2607.02805, "Training Hybrid Block Diffusion Language Models with
 * Partial Bidirectionality").
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the CPU
 * baseline of the benchmark load this library. It shares no source, header,
 * table or constant with the CUDA library, and it never calls it.
 *
 * What it computes, in the paper's terms:
 *
 *  - The selective update of Sec. 3 (eq. mamba-scan-background),
 *        s_t = A_t s_{t-1} + B_t x_t,   y_t = C_t s_t + D x_t,
 *    with the Mamba-1 discretisation A_t = exp(dt_t * A) for a diagonal A
 *    holding one decay per (channel d, state n), and B_t x_t read as
 *    dt_t * B_t[n] * x_t[d].  dt is given after its softplus.
 *  - The forward prefix scan over the clean stream, whose state at every
 *    block end is the reusable boundary state s_k = F_fwd(c^(k))
 *    (Sec. 4, eq. boundary-state; eq. cache-c4).
 *  - For every noisy block: a forward scan seeded from the boundary state at
 *    its start, a reverse scan confined to the block and started from zero,
 *    and the sum of the two directions (Sec. 4, eq. partial-reverse). Each
 *    direction has its own dt, B, C and its own A and D; the forward
 *    direction of the noisy block shares A_f, D_f with the clean scan
 *    because both are the same layer's forward scan.
 *  - All blocks at once, as in the all-block objective (Sec. 4.1), and the
 *    gradient that flows from each noisy block through its cached seed into
 *    the clean prefix scan (eq. prefix-cache-gradient).
 *
 * Readings where the paper is silent (each listed in the design notes):
 *  - states[k] is the clean state after token (k+1)*Bs-1; noisy block k is
 *    seeded with states[k-1], block 0 with zero.
 *  - The reverse direction starts from zero at the block end and includes
 *    the token's own input (a causal scan of the reversed block).
 *  - Each direction adds its own D term, so the sum carries (D_f+D_r)*x.
 *  - The clean stream is scanned forward only.
 *
 * Layouts (row-major, all fp64 here):
 *   token-by-channel tensors x, dt, dy, y:  [Bt][L][D]
 *   token-by-state tensors   B, C:          [Bt][L][N]
 *   A: [D][N]   D: [D]   states: [Bt][nS][D][N]   seed: [Bt][D][N]
 *
 * Parallelism: OpenMP over independent channels (forward) and over batch
 * rows (backward, so that the sums over channels stay in a fixed order).
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
  long batch; /* Bt */
  long len;   /* L, tokens per stream */
  long block; /* Bs */
  long d;     /* D, channels (d_inner) */
  long n;     /* N, state size (d_state) */
} bdo_dims;

static int g_threads = 1;

void bdo_set_threads(int t) { g_threads = t > 0 ? t : 1; }
int bdo_get_threads(void) { return g_threads; }
int bdo_has_openmp(void) {
#ifdef _OPENMP
  return 1;
#else
  return 0;
#endif
}

#define TD(m, b, t, c) ((((b) * (m)->len) + (t)) * (m)->d + (c))
#define TN(m, b, t, s) ((((b) * (m)->len) + (t)) * (m)->n + (s))

/* ---------------------------------------------------------------------- */
/* Forward                                                                  */
/* ---------------------------------------------------------------------- */

/* Causal forward scan of one channel of the clean stream (eq.
 * mamba-scan-background), starting from h0 (or zero). Writes y (if given),
 * the state at every block end (emit_all) or only the final state
 * (states_final), following eq. boundary-state. */
static void clean_scan_channel(const bdo_dims* m, long b, long c, const double* x, const double* dt,
                               const double* B, const double* C, const double* A, const double* Dv,
                               const double* h0, double* y, double* states, long nS, int emit_all,
                               double* h_final) {
  const long N = m->n;
  double* h = (double*)calloc((size_t)N, sizeof(double));
  if (h0)
    for (long s = 0; s < N; ++s) h[s] = h0[s];
  for (long t = 0; t < m->len; ++t) {
    const double dtt = dt[TD(m, b, t, c)];
    const double xt = x[TD(m, b, t, c)];
    double yt = 0.0;
    for (long s = 0; s < N; ++s) {
      const double a = exp(dtt * A[c * N + s]);
      h[s] = a * h[s] + dtt * B[TN(m, b, t, s)] * xt;
      yt += C[TN(m, b, t, s)] * h[s];
    }
    if (y) y[TD(m, b, t, c)] = yt + Dv[c] * xt;
    if (emit_all && states && (t + 1) % m->block == 0) {
      const long k = (t + 1) / m->block - 1;
      for (long s = 0; s < N; ++s) states[((b * nS + k) * m->d + c) * N + s] = h[s];
    }
  }
  if (h_final)
    for (long s = 0; s < N; ++s) h_final[s] = h[s];
  free(h);
}

/* One noisy block of one channel (eq. partial-reverse): a forward scan over
 * positions t0..t0+Bs-1 seeded with `seed` (zero if NULL), a reverse scan over
 * the same positions started from zero, and the sum of both outputs. */
static void noisy_block_channel(const bdo_dims* m, long b, long t0, long c, const double* seed,
                                const double* xn, const double* dtf, const double* Bf,
                                const double* Cf, const double* dtr, const double* Br,
                                const double* Cr, const double* Af, const double* Df,
                                const double* Ar, const double* Dr, double* yn) {
  const long N = m->n, Bs = m->block;
  double* h = (double*)calloc((size_t)N, sizeof(double));
  double* yf = (double*)calloc((size_t)Bs, sizeof(double));
  /* forward direction, continuing the cached state */
  if (seed)
    for (long s = 0; s < N; ++s) h[s] = seed[s];
  for (long i = 0; i < Bs; ++i) {
    const long t = t0 + i;
    const double dtt = dtf[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)];
    double yt = 0.0;
    for (long s = 0; s < N; ++s) {
      const double a = exp(dtt * Af[c * N + s]);
      h[s] = a * h[s] + dtt * Bf[TN(m, b, t, s)] * xt;
      yt += Cf[TN(m, b, t, s)] * h[s];
    }
    yf[i] = yt + Df[c] * xt;
  }
  /* reverse direction: rev(F_rev(rev(block))), zero state at the block end */
  for (long s = 0; s < N; ++s) h[s] = 0.0;
  for (long i = Bs - 1; i >= 0; --i) {
    const long t = t0 + i;
    const double dtt = dtr[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)];
    double yt = 0.0;
    for (long s = 0; s < N; ++s) {
      const double a = exp(dtt * Ar[c * N + s]);
      h[s] = a * h[s] + dtt * Br[TN(m, b, t, s)] * xt;
      yt += Cr[TN(m, b, t, s)] * h[s];
    }
    yn[TD(m, b, t, c)] = yf[i] + (yt + Dr[c] * xt);
  }
  free(h);
  free(yf);
}

static int dims_ok(const bdo_dims* m) {
  if (!m || m->batch < 0 || m->len < 0 || m->block <= 0 || m->d < 0 || m->n <= 0) return 0;
  if (m->len % m->block != 0) return 0;
  return 1;
}

/* All-block forward: clean scan with every boundary state, then every noisy
 * block seeded from the state at its start. states: [Bt][L/Bs][D][N]. */
int bdo_forward(const bdo_dims* m, const double* xc, const double* dtc, const double* Bc,
                const double* Cc, const double* xn, const double* dtf, const double* Bf,
                const double* Cf, const double* dtr, const double* Br, const double* Cr,
                const double* Af, const double* Df, const double* Ar, const double* Dr,
                double* yc, double* yn, double* states) {
  if (!dims_ok(m)) return -1;
  const long nb = m->len / m->block, Bt = m->batch, D = m->d, N = m->n;
  long jobs = Bt * D;
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
  for (long j = 0; j < jobs; ++j) {
    const long b = j / D, c = j % D;
    clean_scan_channel(m, b, c, xc, dtc, Bc, Cc, Af, Df, NULL, yc, states, nb, 1, NULL);
  }
  jobs = Bt * nb * D;
#pragma omp parallel for schedule(dynamic, 16) num_threads(g_threads)
  for (long j = 0; j < jobs; ++j) {
    const long b = j / (nb * D), k = (j / D) % nb, c = j % D;
    const double* seed = k > 0 ? &states[((b * nb + (k - 1)) * D + c) * N] : NULL;
    noisy_block_channel(m, b, k * m->block, c, seed, xn, dtf, Bf, Cf, dtr, Br, Cr, Af, Df, Ar, Dr, yn);
  }
  return 0;
}

/* Cache build: the clean forward scan only, optionally continued from an
 * initial state (cache append after a block is finalised). emit_all != 0
 * writes every block-end state ([Bt][L/Bs][D][N]); otherwise only the final
 * state ([Bt][1][D][N]). y (nullable) receives the clean outputs. */
int bdo_boundary_states(const bdo_dims* m, const double* xc, const double* dtc, const double* Bc,
                        const double* Cc, const double* Af, const double* Df,
                        const double* init_state, double* yc, double* states, int emit_all) {
  if (!dims_ok(m)) return -1;
  const long nb = m->len / m->block, Bt = m->batch, D = m->d, N = m->n;
  const long nS = emit_all ? nb : 1;
  const long jobs = Bt * D;
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
  for (long j = 0; j < jobs; ++j) {
    const long b = j / D, c = j % D;
    const double* h0 = init_state ? &init_state[(b * D + c) * N] : NULL;
    double* fin = emit_all ? NULL : &states[(b * D + c) * N];
    clean_scan_channel(m, b, c, xc, dtc, Bc, Cc, Af, Df, h0, yc, states, nS, emit_all, fin);
  }
  return 0;
}

/* Cached active-block step: one noisy block (m->len == m->block) seeded from a
 * read-only cached state seed[Bt][D][N]. */
int bdo_active_block(const bdo_dims* m, const double* seed, const double* xn, const double* dtf,
                     const double* Bf, const double* Cf, const double* dtr, const double* Br,
                     const double* Cr, const double* Af, const double* Df, const double* Ar,
                     const double* Dr, double* yn) {
  if (!dims_ok(m) || m->len != m->block) return -1;
  const long Bt = m->batch, D = m->d, N = m->n;
  const long jobs = Bt * D;
#pragma omp parallel for schedule(dynamic, 16) num_threads(g_threads)
  for (long j = 0; j < jobs; ++j) {
    const long b = j / D, c = j % D;
    noisy_block_channel(m, b, 0, c, &seed[(b * D + c) * N], xn, dtf, Bf, Cf, dtr, Br, Cr, Af, Df,
                        Ar, Dr, yn);
  }
  return 0;
}

/* ---------------------------------------------------------------------- */
/* Backward                                                                 */
/* ---------------------------------------------------------------------- */
/*
 * Reverse-mode derivative of
 *     Loss = <dy_c, y_c> + <dy_n, y_n> + <dstates, states>
 * with respect to every input, for the recurrences above. For a scan
 * h_t = a_t h_prev + dt_t B_t x_t, y_t = C_t h_t + D x_t, with
 * a_t = exp(dt_t A) and g_t = dLoss/dh_t (the adjoint, summed over every
 * later use of h_t):
 *     g_t        = C_t dy_t + a_next g_next (+ any direct injection at t)
 *     dx_t      += D dy_t + dt_t sum_n g_t B_t
 *     ddt_t      = sum_n g_t (B_t x_t + A a_t h_prev)
 *     dA        += sum_t g_t dt_t a_t h_prev
 *     dB_t[n]   += sum_d g_t dt_t x_t
 *     dC_t[n]   += sum_d dy_t h_t
 *     dD        += sum_t dy_t x_t
 *     dh_prev    = a_t g_t at the first step (gradient of the seed).
 * "next" follows the scan order: t+1 for forward scans, t-1 for the reverse
 * scan. The clean stream receives, at every block end t = (k+1)Bs-1, the
 * gradient of the seed of noisy block k+1 plus dstates[k] (the path
 * l_k -> C_k -> F(b_<k) -> theta of eq. prefix-cache-gradient).
 */
int bdo_backward(const bdo_dims* m, const double* xc, const double* dtc, const double* Bc,
                 const double* Cc, const double* xn, const double* dtf, const double* Bf,
                 const double* Cf, const double* dtr, const double* Br, const double* Cr,
                 const double* Af, const double* Df, const double* Ar, const double* Dr,
                 const double* states, const double* dyc, const double* dyn, const double* dstates,
                 double* dxc, double* ddtc, double* dBc, double* dCc, double* dxn, double* ddtf,
                 double* dBf, double* dCf, double* ddtr, double* dBr, double* dCr, double* dAf,
                 double* dDf, double* dAr, double* dDr) {
  if (!dims_ok(m)) return -1;
  const long Bt = m->batch, L = m->len, Bs = m->block, D = m->d, N = m->n, nb = L / Bs;
  const size_t tokN = (size_t)(Bt * L * N);
  memset(dBc, 0, tokN * sizeof(double));
  memset(dCc, 0, tokN * sizeof(double));
  memset(dBf, 0, tokN * sizeof(double));
  memset(dCf, 0, tokN * sizeof(double));
  memset(dBr, 0, tokN * sizeof(double));
  memset(dCr, 0, tokN * sizeof(double));
  /* per batch row partial sums of the parameter gradients, added in row order */
  double* pAf = (double*)calloc((size_t)(Bt * D * N), sizeof(double));
  double* pAr = (double*)calloc((size_t)(Bt * D * N), sizeof(double));
  double* pDf = (double*)calloc((size_t)(Bt * D), sizeof(double));
  double* pDr = (double*)calloc((size_t)(Bt * D), sizeof(double));

#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
  for (long b = 0; b < Bt; ++b) {
    double* hc = (double*)malloc((size_t)(L * N) * sizeof(double)); /* clean h_t */
    double* ac = (double*)malloc((size_t)(L * N) * sizeof(double)); /* clean a_t */
    double* hb = (double*)malloc((size_t)(Bs * N) * sizeof(double)); /* block h_t */
    double* hp = (double*)malloc((size_t)(Bs * N) * sizeof(double)); /* block h_prev */
    double* ab = (double*)malloc((size_t)(Bs * N) * sizeof(double)); /* block a_t */
    double* dS = (double*)malloc((size_t)(nb * N) * sizeof(double)); /* seed grads */
    double* g = (double*)malloc((size_t)N * sizeof(double));
    for (long c = 0; c < D; ++c) {
      double* gAf = &pAf[(b * D + c) * N];
      double* gAr = &pAr[(b * D + c) * N];
      double dDf_acc = 0.0, dDr_acc = 0.0;
      for (long q = 0; q < nb * N; ++q) dS[q] = 0.0;

      for (long k = 0; k < nb; ++k) {
        const long t0 = k * Bs;
        /* --- noisy block k, forward direction (seeded) --- */
        /* hp[i] holds the state the step at position t0+i continues from */
        for (long s = 0; s < N; ++s)
          hp[s] = k > 0 ? states[((b * nb + (k - 1)) * D + c) * N + s] : 0.0;
        for (long i = 0; i < Bs; ++i) {
          const long t = t0 + i;
          const double dtt = dtf[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)];
          for (long s = 0; s < N; ++s) {
            const double prev = hp[i * N + s];
            const double a = exp(dtt * Af[c * N + s]);
            ab[i * N + s] = a;
            hb[i * N + s] = a * prev + dtt * Bf[TN(m, b, t, s)] * xt;
            if (i + 1 < Bs) hp[(i + 1) * N + s] = hb[i * N + s];
          }
        }
        for (long s = 0; s < N; ++s) g[s] = 0.0;
        for (long i = Bs - 1; i >= 0; --i) {
          const long t = t0 + i;
          const double dtt = dtf[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)], dy = dyn[TD(m, b, t, c)];
          double sum_gB = 0.0, sum_dt = 0.0;
          for (long s = 0; s < N; ++s) {
            const double anext = i + 1 < Bs ? ab[(i + 1) * N + s] : 0.0;
            g[s] = Cf[TN(m, b, t, s)] * dy + anext * g[s];
            const double prev = hp[i * N + s];
            sum_gB += g[s] * Bf[TN(m, b, t, s)];
            sum_dt += g[s] * (Bf[TN(m, b, t, s)] * xt + Af[c * N + s] * ab[i * N + s] * prev);
            gAf[s] += g[s] * dtt * ab[i * N + s] * prev;
            dBf[TN(m, b, t, s)] += g[s] * dtt * xt;
            dCf[TN(m, b, t, s)] += dy * hb[i * N + s];
          }
          dxn[TD(m, b, t, c)] = dtt * sum_gB;
          ddtf[TD(m, b, t, c)] = sum_dt;
        }
        if (k > 0)
          for (long s = 0; s < N; ++s) dS[(k - 1) * N + s] = ab[s] * g[s];

        /* --- noisy block k, reverse direction (zero state at the block end) --- */
        /* here hp[i] holds h^r_{t+1} (the state the step at t continues) */
        for (long i = Bs - 1; i >= 0; --i) {
          const long t = t0 + i;
          const double dtt = dtr[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)];
          for (long s = 0; s < N; ++s) {
            const double nxt = i + 1 < Bs ? hb[(i + 1) * N + s] : 0.0;
            const double a = exp(dtt * Ar[c * N + s]);
            ab[i * N + s] = a;
            hp[i * N + s] = nxt;
            hb[i * N + s] = a * nxt + dtt * Br[TN(m, b, t, s)] * xt;
          }
        }
        for (long s = 0; s < N; ++s) g[s] = 0.0;
        for (long i = 0; i < Bs; ++i) {
          const long t = t0 + i;
          const double dtt = dtr[TD(m, b, t, c)], xt = xn[TD(m, b, t, c)], dy = dyn[TD(m, b, t, c)];
          double sum_gB = 0.0, sum_dt = 0.0;
          for (long s = 0; s < N; ++s) {
            const double aprev = i > 0 ? ab[(i - 1) * N + s] : 0.0;
            g[s] = Cr[TN(m, b, t, s)] * dy + aprev * g[s];
            const double nxt = hp[i * N + s];
            sum_gB += g[s] * Br[TN(m, b, t, s)];
            sum_dt += g[s] * (Br[TN(m, b, t, s)] * xt + Ar[c * N + s] * ab[i * N + s] * nxt);
            gAr[s] += g[s] * dtt * ab[i * N + s] * nxt;
            dBr[TN(m, b, t, s)] += g[s] * dtt * xt;
            dCr[TN(m, b, t, s)] += dy * hb[i * N + s];
          }
          dxn[TD(m, b, t, c)] += dtt * sum_gB + (Df[c] + Dr[c]) * dy;
          ddtr[TD(m, b, t, c)] = sum_dt;
          dDf_acc += dy * xt;
          dDr_acc += dy * xt;
        }
      }

      /* --- clean stream: recompute, then the adjoint over the whole stream --- */
      for (long t = 0; t < L; ++t) {
        const double dtt = dtc[TD(m, b, t, c)], xt = xc[TD(m, b, t, c)];
        for (long s = 0; s < N; ++s) {
          const double prev = t > 0 ? hc[(t - 1) * N + s] : 0.0;
          const double a = exp(dtt * Af[c * N + s]);
          ac[t * N + s] = a;
          hc[t * N + s] = a * prev + dtt * Bc[TN(m, b, t, s)] * xt;
        }
      }
      for (long s = 0; s < N; ++s) g[s] = 0.0;
      for (long t = L - 1; t >= 0; --t) {
        const double dtt = dtc[TD(m, b, t, c)], xt = xc[TD(m, b, t, c)];
        const double dy = dyc ? dyc[TD(m, b, t, c)] : 0.0;
        const int at_end = ((t + 1) % Bs) == 0;
        const long k = (t + 1) / Bs - 1;
        double sum_gB = 0.0, sum_dt = 0.0;
        for (long s = 0; s < N; ++s) {
          const double anext = t + 1 < L ? ac[(t + 1) * N + s] : 0.0;
          double inj = 0.0;
          if (at_end) {
            if (k + 1 < nb) inj += dS[k * N + s];
            if (dstates) inj += dstates[((b * nb + k) * D + c) * N + s];
          }
          g[s] = Cc[TN(m, b, t, s)] * dy + inj + anext * g[s];
          const double prev = t > 0 ? hc[(t - 1) * N + s] : 0.0;
          sum_gB += g[s] * Bc[TN(m, b, t, s)];
          sum_dt += g[s] * (Bc[TN(m, b, t, s)] * xt + Af[c * N + s] * ac[t * N + s] * prev);
          gAf[s] += g[s] * dtt * ac[t * N + s] * prev;
          dBc[TN(m, b, t, s)] += g[s] * dtt * xt;
          dCc[TN(m, b, t, s)] += dy * hc[t * N + s];
        }
        dxc[TD(m, b, t, c)] = dtt * sum_gB + Df[c] * dy;
        ddtc[TD(m, b, t, c)] = sum_dt;
        dDf_acc += dy * xt;
      }
      pDf[b * D + c] = dDf_acc;
      pDr[b * D + c] = dDr_acc;
    }
    free(hc);
    free(ac);
    free(hb);
    free(hp);
    free(ab);
    free(dS);
    free(g);
  }

  for (long q = 0; q < D * N; ++q) {
    double sf = 0.0, sr = 0.0;
    for (long b = 0; b < Bt; ++b) {
      sf += pAf[b * D * N + q];
      sr += pAr[b * D * N + q];
    }
    dAf[q] = sf;
    dAr[q] = sr;
  }
  for (long c = 0; c < D; ++c) {
    double sf = 0.0, sr = 0.0;
    for (long b = 0; b < Bt; ++b) {
      sf += pDf[b * D + c];
      sr += pDr[b * D + c];
    }
    dDf[c] = sf;
    dDr[c] = sr;
  }
  free(pAf);
  free(pAr);
  free(pDf);
  free(pDr);
  return 0;
}
