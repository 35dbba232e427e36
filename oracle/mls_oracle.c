/*
 * CPU oracle for the Matryoshka-suite output stage (LM heads + next-token
 * cross-entropy + integrated distillation), forward and backward.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the tests, the package's smoke check and the CPU
 * baseline leg of the benchmark do.  It shares no code, header, table or
 * helper with the CUDA library.
 *
 * Everything is computed in IEEE double precision with the logits
 * materialised in full, one token at a time, exactly as the definitions in
 * the paper read:
 *
 *   heads           z_m = W^m o^m,  W^m in R^{V x D_m}          (Sec. 2, "Modeling"
 *                                                               and "Inter-model Junction")
 *   cross-entropy   CE_m = logsumexp(z_m) - z_m[y]               (Sec. 2, "Modeling")
 *   distillation    Ld_m = - sum_v q_v log softmax(z_m / tau)_v,
 *                   q = stop_grad(softmax(z_T / tau)), T = teacher  (Eq. 2)
 *   sub-model loss  L_m = (1 - alpha) CE_m + alpha Ld_m, m != T (Eq. 3);
 *                   L_T = CE_T (Eq. 2 defines the term only for m < M)
 *   total           loss = sum_m w_m * (1/N) sum_{t valid} L_m[t]   (sum after Eq. 3;
 *                   per-size weights w_m of App. G, default 1)
 *
 * Readings of the paper (each one is listed in the design notes):
 *   - Eq. 2 has no temperature.  tau divides both the teacher's and the
 *     student's logits inside the distillation term only; CE stays at tau = 1;
 *     no tau^2 factor.  At tau = 1 this is Eq. 2 exactly.
 *   - KL_m = Ld_m - H(q) is reported as a diagnostic; it does not enter the loss.
 *   - The (1 - alpha) factor of Eq. 3 multiplies CE for every student.
 *   - Tokens whose target is negative are ignored: they contribute nothing to
 *     the loss, to N or to the gradients, and their per-token losses are 0.
 *     Targets >= V are rejected (return code 3).
 *   - argmax ties resolve to the lowest vocabulary index.
 *   - N = 0 (every token ignored) gives loss 0 and zero gradients.
 *
 * Gradient (backward) with g = grad_scale, c_m = g w_m / N, p = softmax(z):
 *   student:  dL/dz_m = c_m [ (1 - alpha)(p_m - e_y) + (alpha/tau)(softmax(z_m/tau) - q) ]
 *   teacher:  dL/dz_T = c_T (p_T - e_y)          (stop-grad on q in Eq. 2)
 *   dH_m = G_m W_m,   dW_m = G_m^T H_m.
 *
 * Inputs are passed with their storage type (bf16 bit patterns, fp32 or fp64) and
 * upcast to double element by element; all arithmetic is double.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_MAX_M 16

typedef struct {
  int M;                /* number of sub-models */
  long long T;          /* tokens */
  long long V;          /* vocabulary size */
  const int* d;         /* d[M]: width D_m of sub-model m */
  int teacher;          /* index of the distillation teacher (paper: M-1) */
  double tau;           /* distillation temperature (paper: 1) */
  double alpha;         /* alpha_d of Eq. 3 */
  const double* w;      /* per-sub-model weights w[M] (App. G); NULL means all 1 */
  int in_dtype;         /* 0 = bf16 bit patterns (uint16), 1 = fp32, 2 = fp64 */
} mls_oracle_problem;

/* One stored element as a double: bf16 is the top half of an fp32. */
static double elem(const void* base, int dtype, long long i) {
  if (dtype == 0) {
    uint32_t bits = ((uint32_t)((const uint16_t*)base)[i]) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
  }
  if (dtype == 1) return (double)((const float*)base)[i];
  return ((const double*)base)[i];
}

static int check_problem(const mls_oracle_problem* p) {
  if (!p || p->M < 1 || p->M > ORACLE_MAX_M || p->T < 0 || p->V < 1 || !p->d) return 1;
  if (p->teacher < 0 || p->teacher >= p->M) return 1;
  if (!(p->tau > 0.0) || !(p->alpha >= 0.0 && p->alpha <= 1.0)) return 1;
  if (p->in_dtype < 0 || p->in_dtype > 2) return 1;
  for (int m = 0; m < p->M; ++m)
    if (p->d[m] < 1) return 1;
  return 0;
}

static double weight(const mls_oracle_problem* p, int m) { return p->w ? p->w[m] : 1.0; }

/* z[v] = sum_k H[t,k] W[v,k] for every v: the full logit row of one token.
   (The storage type is switched on outside the loops; every product and the
   order of the sum over k are the same as elem(H) * elem(W) summed k = 0..d-1.) */
static void logits_row(const mls_oracle_problem* p, const void* H, const void* W, int dm,
                       long long t, double* z) {
  double h[dm > 0 ? dm : 1];
  for (int k = 0; k < dm; ++k) h[k] = elem(H, p->in_dtype, t * dm + k);
  for (long long v = 0; v < p->V; ++v) {
    double acc = 0.0;
    if (p->in_dtype == 0) {
      const uint16_t* w = (const uint16_t*)W + v * dm;
      for (int k = 0; k < dm; ++k) {
        uint32_t bits = ((uint32_t)w[k]) << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        acc += h[k] * (double)f;
      }
    } else if (p->in_dtype == 1) {
      const float* w = (const float*)W + v * dm;
      for (int k = 0; k < dm; ++k) acc += h[k] * (double)w[k];
    } else {
      const double* w = (const double*)W + v * dm;
      for (int k = 0; k < dm; ++k) acc += h[k] * w[k];
    }
    z[v] = acc;
  }
}

/* log sum_v exp(z[v] / s) with the maximum factored out. */
static double logsumexp_scaled(const double* z, long long V, double s) {
  double mx = -INFINITY;
  for (long long v = 0; v < V; ++v)
    if (z[v] / s > mx) mx = z[v] / s;
  double sum = 0.0;
  for (long long v = 0; v < V; ++v) sum += exp(z[v] / s - mx);
  return mx + log(sum);
}

static int argmax_lowest(const double* z, long long V) {
  long long best = 0;
  for (long long v = 1; v < V; ++v)
    if (z[v] > z[best]) best = v;
  return (int)best;
}

static long long count_valid(const mls_oracle_problem* p, const int* y) {
  long long n = 0;
  for (long long t = 0; t < p->T; ++t)
    if (y[t] >= 0) ++n;
  return n;
}

static int check_targets(const mls_oracle_problem* p, const int* y) {
  for (long long t = 0; t < p->T; ++t)
    if (y[t] >= p->V) return 3;
  return 0;
}

/*
 * Everything one token needs, from its materialised logits z[m][v]:
 * per-token losses, diagnostics, argmax, lse statistics and, when G is
 * non-NULL, the logit gradients G[m][v] (already scaled by c_m).
 */
static void token_terms(const mls_oracle_problem* p, double* const* z, int y, double inv_n,
                        double grad_scale, double* L, double* CE, double* Ld, double* KL,
                        int* amax, double* lse, double* lse_tau, double* const* G) {
  const int M = p->M, Tm = p->teacher;
  const long long V = p->V;
  const double tau = p->tau, alpha = p->alpha;

  for (int m = 0; m < M; ++m) {
    lse[m] = logsumexp_scaled(z[m], V, 1.0);
    lse_tau[m] = logsumexp_scaled(z[m], V, tau);
    amax[m] = argmax_lowest(z[m], V);
  }

  /* q = softmax(z_T / tau), log q and the teacher entropy H(q). */
  double Hq = 0.0;
  for (long long v = 0; v < V; ++v) {
    double logq = z[Tm][v] / tau - lse_tau[Tm];
    Hq -= exp(logq) * logq;
  }

  for (int m = 0; m < M; ++m) {
    /* Eq. 2: Ld = -sum_v q_v log softmax(z_m/tau)_v;  KL = Ld - H(q). */
    double ld = 0.0;
    for (long long v = 0; v < V; ++v) {
      double q = exp(z[Tm][v] / tau - lse_tau[Tm]);
      double logp_tau = z[m][v] / tau - lse_tau[m];
      ld -= q * logp_tau;
    }
    const int valid = y >= 0;
    const double ce = valid ? lse[m] - z[m][y] : 0.0;
    CE[m] = ce;
    Ld[m] = valid ? ld : 0.0;
    KL[m] = valid ? ld - Hq : 0.0;
    if (m == Tm)
      L[m] = ce;                                  /* teacher: CE only */
    else
      L[m] = valid ? (1.0 - alpha) * ce + alpha * ld : 0.0;   /* Eq. 3 */

    if (G) {
      const double c = valid ? grad_scale * weight(p, m) * inv_n : 0.0;
      for (long long v = 0; v < V; ++v) {
        double pm = exp(z[m][v] - lse[m]);
        double onehot = (v == y) ? 1.0 : 0.0;
        double g;
        if (m == Tm) {
          g = pm - onehot;
        } else {
          double pm_tau = exp(z[m][v] / tau - lse_tau[m]);
          double q = exp(z[Tm][v] / tau - lse_tau[Tm]);
          g = (1.0 - alpha) * (pm - onehot) + (alpha / tau) * (pm_tau - q);
        }
        G[m][v] = c * g;
      }
    }
  }
}

/*
 * Forward over all tokens.
 *   loss      [1]        scalar objective
 *   tok_loss  [M*T]      L_m[t]  (model-major)
 *   tok_diag  [3*M*T]    CE, Ld, KL (each [M*T]); may be NULL
 *   argmax    [M*T]      may be NULL
 *   stats     [2*M*T]    logsumexp(z_m), logsumexp(z_m/tau); may be NULL
 * Returns 0, 1 for bad arguments, 3 for a target >= V, 4 for out of memory.
 */
int mls_oracle_fwd(const mls_oracle_problem* p, const void* const* H, const void* const* W,
                   const int* y, double* loss, double* tok_loss, double* tok_diag, int* argmax,
                   double* stats) {
  if (check_problem(p) || !H || !W || !y || !loss || !tok_loss) return 1;
  if (check_targets(p, y)) return 3;
  const int M = p->M;
  const long long T = p->T, V = p->V;
  const long long n_valid = count_valid(p, y);
  const double inv_n = n_valid > 0 ? 1.0 / (double)n_valid : 0.0;
  int err = 0;

#pragma omp parallel
  {
    double* zbuf = (double*)malloc(sizeof(double) * (size_t)M * (size_t)V);
    double* z[ORACLE_MAX_M];
    if (!zbuf) {
#pragma omp atomic write
      err = 4;
    } else {
      for (int m = 0; m < M; ++m) z[m] = zbuf + (size_t)m * V;
    }
#pragma omp for schedule(dynamic, 1)
    for (long long t = 0; t < T; ++t) {
      if (!zbuf) continue;
      double L[ORACLE_MAX_M], CE[ORACLE_MAX_M], Ld[ORACLE_MAX_M], KL[ORACLE_MAX_M];
      double lse[ORACLE_MAX_M], lse_tau[ORACLE_MAX_M];
      int am[ORACLE_MAX_M];
      for (int m = 0; m < M; ++m) logits_row(p, H[m], W[m], p->d[m], t, z[m]);
      token_terms(p, z, y[t], inv_n, 1.0, L, CE, Ld, KL, am, lse, lse_tau, NULL);
      for (int m = 0; m < M; ++m) {
        tok_loss[m * T + t] = L[m];
        if (tok_diag) {
          tok_diag[(0 * M + m) * T + t] = CE[m];
          tok_diag[(1 * M + m) * T + t] = Ld[m];
          tok_diag[(2 * M + m) * T + t] = KL[m];
        }
        if (argmax) argmax[m * T + t] = am[m];
        if (stats) {
          stats[(0 * M + m) * T + t] = lse[m];
          stats[(1 * M + m) * T + t] = lse_tau[m];
        }
      }
    }
    free(zbuf);
  }
  if (err) return err;

  double total = 0.0;
  for (int m = 0; m < M; ++m) {
    double s = 0.0;
    for (long long t = 0; t < T; ++t)
      if (y[t] >= 0) s += tok_loss[m * T + t];
    total += weight(p, m) * s * inv_n;
  }
  *loss = total;
  return 0;
}

/*
 * Backward over all tokens: dH[m] [T*d_m] = G_m W_m and dW[m] [V*d_m] = G_m^T H_m,
 * both overwritten.  G_m (T x V doubles per model) is materialised.
 */
int mls_oracle_bwd(const mls_oracle_problem* p, const void* const* H, const void* const* W,
                   const int* y, double grad_scale, double* const* dH, double* const* dW) {
  if (check_problem(p) || !H || !W || !y || !dH || !dW) return 1;
  if (check_targets(p, y)) return 3;
  const int M = p->M;
  const long long T = p->T, V = p->V;
  const long long n_valid = count_valid(p, y);
  const double inv_n = n_valid > 0 ? 1.0 / (double)n_valid : 0.0;

  double* Gall = (double*)malloc(sizeof(double) * (size_t)M * (size_t)(T > 0 ? T : 1) * (size_t)V);
  if (!Gall) return 4;
  int err = 0;

#pragma omp parallel
  {
    double* zbuf = (double*)malloc(sizeof(double) * (size_t)M * (size_t)V);
    double* z[ORACLE_MAX_M];
    if (!zbuf) {
#pragma omp atomic write
      err = 4;
    } else {
      for (int m = 0; m < M; ++m) z[m] = zbuf + (size_t)m * V;
    }
#pragma omp for schedule(dynamic, 1)
    for (long long t = 0; t < T; ++t) {
      if (!zbuf) continue;
      double L[ORACLE_MAX_M], CE[ORACLE_MAX_M], Ld[ORACLE_MAX_M], KL[ORACLE_MAX_M];
      double lse[ORACLE_MAX_M], lse_tau[ORACLE_MAX_M];
      int am[ORACLE_MAX_M];
      double* G[ORACLE_MAX_M];
      for (int m = 0; m < M; ++m) {
        logits_row(p, H[m], W[m], p->d[m], t, z[m]);
        G[m] = Gall + ((size_t)m * T + t) * V;
      }
      token_terms(p, z, y[t], inv_n, grad_scale, L, CE, Ld, KL, am, lse, lse_tau, G);
    }
    free(zbuf);

    /* dH_m[t,k] = sum_v G_m[t,v] W_m[v,k] */
    for (int m = 0; m < M; ++m) {
      const int dm = p->d[m];
#pragma omp for schedule(static)
      for (long long t = 0; t < T; ++t) {
        const double* g = Gall + ((size_t)m * T + t) * V;
        for (int k = 0; k < dm; ++k) {
          double acc = 0.0;
          for (long long v = 0; v < V; ++v) acc += g[v] * elem(W[m], p->in_dtype, v * dm + k);
          dH[m][t * dm + k] = acc;
        }
      }
      /* dW_m[v,k] = sum_t G_m[t,v] H_m[t,k] */
#pragma omp for schedule(static)
      for (long long v = 0; v < V; ++v) {
        for (int k = 0; k < dm; ++k) {
          double acc = 0.0;
          for (long long t = 0; t < T; ++t)
            acc += Gall[((size_t)m * T + t) * V + v] * elem(H[m], p->in_dtype, t * dm + k);
          dW[m][v * dm + k] = acc;
        }
      }
    }
  }
  free(Gall);
  return err;
}

/*
 * Selected tokens only (for sampling a large problem): per-token outputs and
 * the dH rows of the tokens in rows[0..nrows).  n_valid is N for the whole
 * problem (the count of targets >= 0), which the caller computes from the
 * targets.  Outputs are laid out [M*nrows] (model-major) like the forward's
 * [M*T]; dH_rows[m] is [nrows*d_m].  Any output may be NULL.
 */
int mls_oracle_rows(const mls_oracle_problem* p, const void* const* H, const void* const* W,
                    const int* y, const long long* rows, int nrows, long long n_valid,
                    double grad_scale, double* tok_loss, double* tok_diag, int* argmax,
                    double* stats, double* const* dH_rows) {
  if (check_problem(p) || !H || !W || !y || !rows || nrows < 0 || n_valid < 0) return 1;
  for (int r = 0; r < nrows; ++r)
    if (rows[r] < 0 || rows[r] >= p->T) return 1;
  const int M = p->M;
  const long long V = p->V;
  const double inv_n = n_valid > 0 ? 1.0 / (double)n_valid : 0.0;
  int err = 0;

#pragma omp parallel
  {
    double* buf = (double*)malloc(sizeof(double) * 2 * (size_t)M * (size_t)V);
    double* z[ORACLE_MAX_M];
    double* G[ORACLE_MAX_M];
    if (!buf) {
#pragma omp atomic write
      err = 4;
    } else {
      for (int m = 0; m < M; ++m) {
        z[m] = buf + (size_t)m * V;
        G[m] = buf + (size_t)(M + m) * V;
      }
    }
#pragma omp for schedule(dynamic, 1)
    for (int r = 0; r < nrows; ++r) {
      if (!buf) continue;
      const long long t = rows[r];
      if (y[t] >= p->V) {
#pragma omp atomic write
        err = 3;
        continue;
      }
      double L[ORACLE_MAX_M], CE[ORACLE_MAX_M], Ld[ORACLE_MAX_M], KL[ORACLE_MAX_M];
      double lse[ORACLE_MAX_M], lse_tau[ORACLE_MAX_M];
      int am[ORACLE_MAX_M];
      for (int m = 0; m < M; ++m) logits_row(p, H[m], W[m], p->d[m], t, z[m]);
      token_terms(p, z, y[t], inv_n, grad_scale, L, CE, Ld, KL, am, lse, lse_tau,
                  dH_rows ? G : NULL);
      for (int m = 0; m < M; ++m) {
        if (tok_loss) tok_loss[(long long)m * nrows + r] = L[m];
        if (tok_diag) {
          tok_diag[(long long)(0 * M + m) * nrows + r] = CE[m];
          tok_diag[(long long)(1 * M + m) * nrows + r] = Ld[m];
          tok_diag[(long long)(2 * M + m) * nrows + r] = KL[m];
        }
        if (argmax) argmax[(long long)m * nrows + r] = am[m];
        if (stats) {
          stats[(long long)(0 * M + m) * nrows + r] = lse[m];
          stats[(long long)(1 * M + m) * nrows + r] = lse_tau[m];
        }
        if (dH_rows) {
          const int dm = p->d[m];
          for (int k = 0; k < dm; ++k) {
            double acc = 0.0;
            for (long long v = 0; v < V; ++v) acc += G[m][v] * elem(W[m], p->in_dtype, v * dm + k);
            dH_rows[m][(long long)r * dm + k] = acc;
          }
        }
      }
    }
    free(buf);
  }
  return err;
}

/* Threads the oracle will use (OpenMP), for reporting. */
int mls_oracle_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/*
 * Evaluation metrics between sub-models (Sec. 3.2.2: pairwise KL divergence
 * and top-1 next-token agreement across the suite's sub-models; App. A plots
 * KL(p_student || p_teacher)).  For every token and every ordered pair (i, j),
 * with p = softmax(z) at temperature 1:
 *   kl[(i*M + j)*T + t] = KL(p_i || p_j) = sum_v p_i[v] (log p_i[v] - log p_j[v])
 *   agree[(i*M + j)*T + t] = 1 if argmax z_i == argmax z_j (lowest index on ties)
 * The diagonal is 0 (kl) and 1 (agree).  tau, alpha, w and the teacher index
 * of the problem are not used.
 */
int mls_oracle_pairwise(const mls_oracle_problem* p, const void* const* H, const void* const* W,
                        double* kl, int* agree) {
  if (check_problem(p) || !H || !W || !kl) return 1;
  const int M = p->M;
  const long long T = p->T, V = p->V;
  int err = 0;
#pragma omp parallel
  {
    double* buf = (double*)malloc(sizeof(double) * 2 * (size_t)M * (size_t)V);
    if (!buf) {
#pragma omp atomic write
      err = 4;
    }
#pragma omp for schedule(dynamic, 1)
    for (long long t = 0; t < T; ++t) {
      if (!buf) continue;
      double* logp[ORACLE_MAX_M];
      int am[ORACLE_MAX_M];
      for (int m = 0; m < M; ++m) {
        double* z = buf + (size_t)m * V;
        logits_row(p, H[m], W[m], p->d[m], t, z);
        am[m] = argmax_lowest(z, V);
        const double lse = logsumexp_scaled(z, V, 1.0);
        logp[m] = buf + (size_t)(M + m) * V;
        for (long long v = 0; v < V; ++v) logp[m][v] = z[v] - lse;
      }
      for (int i = 0; i < M; ++i) {
        for (int j = 0; j < M; ++j) {
          double k = 0.0;
          if (i != j)
            for (long long v = 0; v < V; ++v) k += exp(logp[i][v]) * (logp[i][v] - logp[j][v]);
          kl[((long long)i * M + j) * T + t] = k;
          if (agree) agree[((long long)i * M + j) * T + t] = am[i] == am[j];
        }
      }
    }
    free(buf);
  }
  return err;
}

/*
 * Inter-model junction (Eq. 1).  Per token t, with o = o^m[t] (D_m values) the
 * output of sub-model m and e = e^{m+1}[t] (D_{m+1} - D_m values) the fresh
 * embedding of sub-model m+1:
 *   o~ = o * ||e||_2 / ||o||_2          (o~ = 0 when ||o|| = 0)
 *   x  = concat(o~, e)                  embed_first = 0: the first D_m channels
 *                                       carry sub-model m (the reading of the prose)
 *   x  = concat(e, o~)                  embed_first = 1: Eq. 1's written order
 * Storage types as for the heads (in_dtype 0 bf16 bits, 1 fp32, 2 fp64); the
 * output x is double.  The backward takes g = dL/dx and returns
 *   dL/do = s (g_o - o (g_o . o) / ||o||^2),  dL/de = g_e + s (g_o . o) e / ||e||^2,
 * with s = ||e|| / ||o|| (both 0 when ||o|| = 0; the e term is 0 when ||e|| = 0),
 * written out from the chain rule of o~ = o ||e|| / ||o||.
 */
static double row_norm(const void* a, int dtype, long long t, int n) {
  double s = 0.0;
  for (int k = 0; k < n; ++k) {
    const double v = elem(a, dtype, t * n + k);
    s += v * v;
  }
  return sqrt(s);
}

int mls_oracle_junction_fwd(long long T, int d_prev, int d_next, int dtype, int embed_first,
                            const void* o, const void* e, double* x) {
  const int de = d_next - d_prev;
  if (T < 0 || d_prev < 1 || de < 1 || dtype < 0 || dtype > 2 || !o || !e || !x) return 1;
#pragma omp parallel for schedule(static)
  for (long long t = 0; t < T; ++t) {
    const double no = row_norm(o, dtype, t, d_prev), ne = row_norm(e, dtype, t, de);
    const double s = no > 0.0 ? ne / no : 0.0;
    double* xr = x + t * d_next;
    const int oo = embed_first ? de : 0, eo = embed_first ? 0 : d_prev;
    for (int k = 0; k < d_prev; ++k) xr[oo + k] = elem(o, dtype, t * d_prev + k) * s;
    for (int k = 0; k < de; ++k) xr[eo + k] = elem(e, dtype, t * de + k);
  }
  return 0;
}

int mls_oracle_junction_bwd(long long T, int d_prev, int d_next, int dtype, int embed_first,
                            const void* o, const void* e, const void* g, double* d_o, double* d_e) {
  const int de = d_next - d_prev;
  if (T < 0 || d_prev < 1 || de < 1 || dtype < 0 || dtype > 2 || !o || !e || !g || !d_o || !d_e)
    return 1;
#pragma omp parallel for schedule(static)
  for (long long t = 0; t < T; ++t) {
    const double no = row_norm(o, dtype, t, d_prev), ne = row_norm(e, dtype, t, de);
    const int oo = embed_first ? de : 0, eo = embed_first ? 0 : d_prev;
    double go_dot_o = 0.0;
    for (int k = 0; k < d_prev; ++k)
      go_dot_o += elem(g, dtype, t * d_next + oo + k) * elem(o, dtype, t * d_prev + k);
    if (no > 0.0) {
      const double s = ne / no;
      for (int k = 0; k < d_prev; ++k)
        d_o[t * d_prev + k] = s * (elem(g, dtype, t * d_next + oo + k) -
                                   elem(o, dtype, t * d_prev + k) * go_dot_o / (no * no));
      for (int k = 0; k < de; ++k) {
        const double ge = elem(g, dtype, t * d_next + eo + k);
        const double ek = elem(e, dtype, t * de + k);
        d_e[t * de + k] = ge + (ne > 0.0 ? s * go_dot_o * ek / (ne * ne) : 0.0);
      }
    } else {
      for (int k = 0; k < d_prev; ++k) d_o[t * d_prev + k] = 0.0;
      for (int k = 0; k < de; ++k) d_e[t * de + k] = elem(g, dtype, t * d_next + eo + k);
    }
  }
  return 0;
}

/*
 * Speculative-decoding verify step for a nested draft / verifier pair
 * (Sec. 2 "Speculative Decoding", Sec. 3.2.3: greedy and nucleus p = 0.9,
 * temperature 0.4), written from the standard speculative sampling rule.
 * Sequence b has gamma drafted tokens x_i, draft logits zd_i (i < gamma) and
 * verifier logits zv_i (i <= gamma), both materialised from hidden states and
 * heads.  For sampling, a distribution is nucleus(softmax(z / temperature)):
 * tokens sorted by probability (descending, then by index) are kept up to and
 * including the first one at which the cumulative probability reaches top_p,
 * then renormalised.  With q_i (draft) and p_i (verifier):
 *   x_i is accepted iff q_i(x_i) > 0 and u[b,i,0] * q_i(x_i) < p_i(x_i);
 *   at the first rejection k: next = sample(norm(max(0, p_k - q_k)), u[b,k,1])
 *     (sample(p_k, u[b,k,1]) if that is all zero);
 *   if all gamma are accepted: next = sample(p_gamma, u[b,gamma,1]);
 *   sample(r, u) = the smallest index v with sum_{w<=v} r_w > u * sum_w r_w.
 * Greedy: x_i is accepted iff x_i == argmax zv_i (lowest index on ties) and
 * next = argmax zv_k at the first rejection (or at gamma).
 * u is [B][gamma+1][2].  Outputs n_accepted[b] and next_token[b].
 */
static void logits_of(const void* H, const void* W, int d, long long V, int dtype, long long row,
                      double* z) {
  for (long long v = 0; v < V; ++v) {
    double acc = 0.0;
    for (int k = 0; k < d; ++k) acc += elem(H, dtype, row * d + k) * elem(W, dtype, v * d + k);
    z[v] = acc;
  }
}

static double* g_sort_p;  /* comparator context (single-threaded use) */
static int by_prob_then_index(const void* a, const void* b) {
  const long long i = *(const long long*)a, j = *(const long long*)b;
  if (g_sort_p[i] > g_sort_p[j]) return -1;
  if (g_sort_p[i] < g_sort_p[j]) return 1;
  return (i > j) - (i < j);
}

/* p <- nucleus(softmax(z / temperature)); order is scratch of V indices */
static void nucleus_probs(const double* z, long long V, double temperature, double top_p, double* p,
                          long long* order) {
  double mx = -INFINITY;
  for (long long v = 0; v < V; ++v)
    if (z[v] > mx) mx = z[v];
  double s = 0.0;
  for (long long v = 0; v < V; ++v) s += exp((z[v] - mx) / temperature);
  for (long long v = 0; v < V; ++v) p[v] = exp((z[v] - mx) / temperature) / s;
  for (long long v = 0; v < V; ++v) order[v] = v;
  g_sort_p = p;
  qsort(order, (size_t)V, sizeof(long long), by_prob_then_index);
  double cum = 0.0, kept = 0.0;
  long long k = 0;
  while (k < V) {
    cum += p[order[k]];
    ++k;
    if (cum >= top_p) break;
  }
  for (long long i = 0; i < k; ++i) kept += p[order[i]];
  for (long long i = k; i < V; ++i) p[order[i]] = 0.0;
  for (long long i = 0; i < k; ++i) p[order[i]] /= kept;
}

static long long sample_index(const double* r, long long V, double u) {
  double tot = 0.0;
  for (long long v = 0; v < V; ++v) tot += r[v];
  double cum = 0.0;
  for (long long v = 0; v < V; ++v) {
    cum += r[v];
    if (cum > u * tot) return v;
  }
  return V - 1;
}

int mls_oracle_spec_verify(int B, int gamma, long long V, int d_draft, int d_verify, int dtype,
                           double temperature, double top_p, int greedy, const void* Hd,
                           const void* Wd, const void* Hv, const void* Wv, const int* draft,
                           const double* u, int* n_accepted, int* next_token) {
  if (B < 0 || gamma < 0 || V < 1 || d_draft < 1 || d_verify < 1 || !(temperature > 0.0) ||
      !(top_p > 0.0 && top_p <= 1.0) || dtype < 0 || dtype > 2)
    return 1;
  double* zd = (double*)malloc(sizeof(double) * (size_t)V * 4);
  long long* order = (long long*)malloc(sizeof(long long) * (size_t)V);
  if (!zd || !order) {
    free(zd);
    free(order);
    return 4;
  }
  double *zv = zd + V, *q = zd + 2 * V, *p = zd + 3 * V;
  for (int b = 0; b < B; ++b) {
    int k = 0, next = -1;
    for (; k < gamma; ++k) {
      const long long pos_d = (long long)b * gamma + k, pos_v = (long long)b * (gamma + 1) + k;
      const int x = draft[pos_d];
      logits_of(Hv, Wv, d_verify, V, dtype, pos_v, zv);
      if (greedy) {
        const int best = argmax_lowest(zv, V);
        if (x != best) {
          next = best;
          break;
        }
        continue;
      }
      logits_of(Hd, Wd, d_draft, V, dtype, pos_d, zd);
      nucleus_probs(zd, V, temperature, top_p, q, order);
      nucleus_probs(zv, V, temperature, top_p, p, order);
      const double uacc = u[((long long)b * (gamma + 1) + k) * 2 + 0];
      const int ok = x >= 0 && x < V && q[x] > 0.0 && uacc * q[x] < p[x];
      if (!ok) {
        double any = 0.0;
        for (long long v = 0; v < V; ++v) {
          q[v] = p[v] - q[v] > 0.0 ? p[v] - q[v] : 0.0;
          any += q[v];
        }
        next = (int)sample_index(any > 0.0 ? q : p, V, u[((long long)b * (gamma + 1) + k) * 2 + 1]);
        break;
      }
    }
    if (next < 0) {
      const long long pos_v = (long long)b * (gamma + 1) + gamma;
      logits_of(Hv, Wv, d_verify, V, dtype, pos_v, zv);
      if (greedy) {
        next = argmax_lowest(zv, V);
      } else {
        nucleus_probs(zv, V, temperature, top_p, p, order);
        next = (int)sample_index(p, V, u[((long long)b * (gamma + 1) + gamma) * 2 + 1]);
      }
    }
    n_accepted[b] = k;
    next_token[b] = next;
  }
  free(zd);
  free(order);
  return 0;
}
