/*
 * relation_oracle.c -- plain, slow fp64 CPU oracle for the causal Self-Exchange
 * Relation (SER) / Multi-Head Relation (MHR) operator of
 * "Ask Self, Ask Others: Relation Is All You Need" (arxiv 2608.20172).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent checker of the CUDA
 * path.  Only the test suite, the package's smoke check and the benchmark's CPU
 * baseline leg may build, load or call it.  It shares no code, header, table or
 * constant with the CUDA library, and the CUDA library never calls it.
 *
 * Every routine works on ONE head with contiguous row-major [T][d] fp64 arrays
 * (rows are tokens, zero-based r; the paper's one-based index is i = r + 1),
 * except the rel_oracle_mhr_* wrappers, which loop over the (b, h) heads of a
 * strided [B][T][H][d] tensor (Sec. 3.2 / App. A.2.1: heads are independent).
 *
 * Definitions followed (paper section / equation):
 *   U_ij = p1_i . p2_j / sqrt(d_h)                       Eq. (relation-projections)
 *   S_i  = sigmoid(U_ii / tau_S), E_ij = SiLU(U_ij)       Eq. (causal-relation)
 *   R_ii = S_i; R_ij = E_ij - lambda log i (j<i); -inf (j>i)
 *   F_i  = Softmax(R_i), Y_i = sum_j F_ij I~_j            Eq. (relation-flow)
 *   factorisation L^E, A, Z, F_ii, g, pi^E, Ibar, Delta  Eqs. (aggregate-exchange-logit),
 *                                                        (self-flow-mass), (conditional-
 *                                                        exchange-distribution), (information-
 *                                                        space-form); App. A.1.2-A.1.6, A.1.8
 *   tiled Exchange scan (m, l, z)                         Eqs. (flashrelation-*); App. A.3
 *   backward, generic softmax gradient                    App. A.1.7 ("general Relation transport")
 *   backward, Self-Exchange credit decomposition          App. A.1.7 (first part)
 *
 * Readings where the paper leaves a choice: natural logarithm everywhere; the
 * count index i is one-based and restarts at 1 for every sequence; R_ii is the
 * sigmoid value itself (not its log); the Exchange map of the diagonal, E_ii, is
 * never used; tau_S carries no gradient.  logZ_i = log sum_j exp(R_ij) is the
 * per-row statistic the GPU path saves for its backward.
 *
 * Return value of every entry point: 0 on success, -1 on a bad argument.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

static double sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }
static double silu(double x) { return x * sigmoid(x); }
/* d SiLU(u) / du = sigma(u) + u sigma(u) (1 - sigma(u))            (App. A.1.7) */
static double silu_grad(double x) {
  double s = sigmoid(x);
  return s + x * s * (1.0 - s);
}

static double dot(const double* a, const double* b, int d) {
  double acc = 0.0;
  for (int c = 0; c < d; ++c) acc += a[c] * b[c];
  return acc;
}

static int bad_args(int T, int d, const void* q, const void* k, const void* v) {
  return T < 1 || d < 1 || !q || !k || !v;
}

/* ------------------------------------------------------------------------ */
/* Materialised Full Relation, one row.                                      */
/* Builds R_r[0..T-1] exactly as Eq. (causal-relation) states (including the */
/* -inf entries above the diagonal), then F_r = Softmax(R_r) with the usual  */
/* max subtraction, logZ_r = log sum_j exp(R_rj) and Y_r = sum_j F_rj I~_j.  */
/* Work arrays: Rrow, Frow of length T, Urow of length T.                    */
/* ------------------------------------------------------------------------ */
static void relation_row(int r, int T, int d, const double* q, const double* k, const double* v,
                         double lambda, double tau_s, double* Urow, double* Rrow, double* Frow,
                         double* y_r, double* logz_r) {
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  const double count_shift = lambda * log((double)(r + 1)); /* lambda_l log i, i one-based */
  for (int j = 0; j < T; ++j) {
    if (j <= r) {
      Urow[j] = dot(q + (size_t)r * d, k + (size_t)j * d, d) * inv_sqrt_d;
    } else {
      Urow[j] = NAN; /* U_ij for j > i never enters R */
    }
    if (j == r) {
      Rrow[j] = sigmoid(Urow[j] / tau_s);        /* Self      */
    } else if (j < r) {
      Rrow[j] = silu(Urow[j]) - count_shift;     /* Exchange  */
    } else {
      Rrow[j] = -INFINITY;                       /* causal    */
    }
  }
  double mx = -INFINITY;
  for (int j = 0; j < T; ++j) mx = Rrow[j] > mx ? Rrow[j] : mx;
  double sum = 0.0;
  for (int j = 0; j < T; ++j) {
    Frow[j] = exp(Rrow[j] - mx); /* exp(-inf) = 0 */
    sum += Frow[j];
  }
  for (int j = 0; j < T; ++j) Frow[j] /= sum;
  *logz_r = mx + log(sum);
  for (int c = 0; c < d; ++c) y_r[c] = 0.0;
  for (int j = 0; j < T; ++j) {
    if (Frow[j] == 0.0) continue;
    for (int c = 0; c < d; ++c) y_r[c] += Frow[j] * v[(size_t)j * d + c];
  }
}

/* Forward of one head, materialised (Eqs. causal-relation, relation-flow).
 * y: [T][d]; logz: [T]; R, F: optional [T][T] outputs (may be NULL). */
int rel_oracle_fwd(int T, int d, const double* q, const double* k, const double* v,
                   double lambda, double tau_s, double* y, double* logz, double* R, double* F) {
  if (bad_args(T, d, q, k, v) || !y || !logz || !(tau_s > 0.0)) return -1;
  double* U = (double*)malloc(sizeof(double) * (size_t)T);
  double* Rr = (double*)malloc(sizeof(double) * (size_t)T);
  double* Fr = (double*)malloc(sizeof(double) * (size_t)T);
  if (!U || !Rr || !Fr) { free(U); free(Rr); free(Fr); return -1; }
  for (int r = 0; r < T; ++r) {
    relation_row(r, T, d, q, k, v, lambda, tau_s, U, Rr, Fr, y + (size_t)r * d, logz + r);
    if (R) memcpy(R + (size_t)r * T, Rr, sizeof(double) * (size_t)T);
    if (F) memcpy(F + (size_t)r * T, Fr, sizeof(double) * (size_t)T);
  }
  free(U); free(Rr); free(Fr);
  return 0;
}

/* Forward restricted to a list of rows (same row definition as above); used to
 * check long sequences at sampled rows.  y: [nrows][d]; logz: [nrows]. */
int rel_oracle_fwd_rows(int T, int d, const double* q, const double* k, const double* v,
                        double lambda, double tau_s, int nrows, const int* rows,
                        double* y, double* logz) {
  if (bad_args(T, d, q, k, v) || !y || !logz || !rows || nrows < 0 || !(tau_s > 0.0)) return -1;
  for (int n = 0; n < nrows; ++n)
    if (rows[n] < 0 || rows[n] >= T) return -1;
  int fail = 0;
#pragma omp parallel
  {
    double* U = (double*)malloc(sizeof(double) * (size_t)T);
    double* Rr = (double*)malloc(sizeof(double) * (size_t)T);
    double* Fr = (double*)malloc(sizeof(double) * (size_t)T);
    const int ok = U && Rr && Fr;
    if (!ok) {
#pragma omp atomic write
      fail = 1;
    }
#pragma omp for schedule(dynamic, 1)
    for (int n = 0; n < nrows; ++n)
      if (ok)
        relation_row(rows[n], T, d, q, k, v, lambda, tau_s, U, Rr, Fr, y + (size_t)n * d,
                     logz + n);
    free(U); free(Rr); free(Fr);
  }
  return fail ? -1 : 0;
}

/* ------------------------------------------------------------------------ */
/* Factorised Self-Exchange form (App. A.1.2-A.1.6, boundary A.1.8).        */
/* Computes, per row, S_i, E_ij (j<i), L^E_i = LSE_{j<i} E_ij,             */
/* A_i = L^E_i - lambda log i, g_i = sigma(A_i - S_i), F_ii = sigma(S_i-A_i),*/
/* pi^E_ij = Softmax_{j<i}(E_ij), Ibar_i = sum_{j<i} pi^E_ij I~_j,          */
/* Y_i = (1 - g_i) I~_i + g_i Ibar_i and logZ_i = log(e^S_i + e^A_i).       */
/* Row 1 (r = 0): the historical set is empty, L^E = A = -inf, g = 0,       */
/* F_11 = 1, Y_1 = I~_1; Ibar_1 is undefined and reported as 0.             */
/* Every output except y may be NULL.  pi: optional [T][T] (0 for j >= i).  */
/* ------------------------------------------------------------------------ */
int rel_oracle_fwd_factorized(int T, int d, const double* q, const double* k, const double* v,
                              double lambda, double tau_s, double* y, double* logz, double* S,
                              double* LE, double* A, double* g, double* Fii, double* Ibar,
                              double* pi) {
  if (bad_args(T, d, q, k, v) || !y || !(tau_s > 0.0)) return -1;
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* E = (double*)malloc(sizeof(double) * (size_t)T);
  double* p = (double*)malloc(sizeof(double) * (size_t)T);
  double* ib = (double*)malloc(sizeof(double) * (size_t)d);
  if (!E || !p || !ib) { free(E); free(p); free(ib); return -1; }
  for (int r = 0; r < T; ++r) {
    const double* qr = q + (size_t)r * d;
    double s_i = sigmoid(dot(qr, k + (size_t)r * d, d) * inv_sqrt_d / tau_s);
    double le = -INFINITY, a = -INFINITY, g_i = 0.0;
    for (int c = 0; c < d; ++c) ib[c] = 0.0;
    if (r > 0) {
      double mx = -INFINITY;
      for (int j = 0; j < r; ++j) {
        E[j] = silu(dot(qr, k + (size_t)j * d, d) * inv_sqrt_d);
        mx = E[j] > mx ? E[j] : mx;
      }
      double sum = 0.0;
      for (int j = 0; j < r; ++j) sum += exp(E[j] - mx);
      le = mx + log(sum);                            /* L^E_i */
      a = le - lambda * log((double)(r + 1));        /* A_i   */
      g_i = sigmoid(a - s_i);                        /* g_i   */
      for (int j = 0; j < r; ++j) {
        p[j] = exp(E[j] - mx) / sum;                 /* pi^E_ij */
        for (int c = 0; c < d; ++c) ib[c] += p[j] * v[(size_t)j * d + c];
      }
    }
    for (int c = 0; c < d; ++c)
      y[(size_t)r * d + c] = (1.0 - g_i) * v[(size_t)r * d + c] + g_i * ib[c];
    if (logz) {
      if (r == 0) {
        logz[r] = s_i;
      } else { /* log(e^S + e^A) evaluated without overflow */
        double hi = s_i > a ? s_i : a, lo = s_i > a ? a : s_i;
        logz[r] = hi + log1p(exp(lo - hi));
      }
    }
    if (S) S[r] = s_i;
    if (LE) LE[r] = le;
    if (A) A[r] = a;
    if (g) g[r] = g_i;
    if (Fii) Fii[r] = r == 0 ? 1.0 : sigmoid(s_i - a);
    if (Ibar)
      for (int c = 0; c < d; ++c) Ibar[(size_t)r * d + c] = ib[c];
    if (pi)
      for (int j = 0; j < T; ++j) pi[(size_t)r * T + j] = (j < r) ? p[j] : 0.0;
  }
  free(E); free(p); free(ib);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* FlashRelation tiled Exchange scan (Sec. 5.1, App. A.3), in fp64.          */
/* For each row the historical keys j < i are visited in tiles of `tile`     */
/* consecutive keys.  The state (m, l, z) starts empty (-inf, 0, 0) and is   */
/* updated per tile by m' = max(m, max_B E), l' = e^{m-m'} l + sum_B e^{E-m'},*/
/* z' = e^{m-m'} z + sum_B e^{E-m'} I~_j.  The terminal state gives          */
/* L^E = m + log l and Ibar = z / l, and the row is completed by             */
/* A = L^E - lambda log i, g = sigma(A - S), Y = (1 - g) I~_i + g Ibar.      */
/* `reverse` != 0 visits the tiles from the newest to the oldest, to check   */
/* that the result does not depend on tile order (App. A.3.2 invariant).     */
/* ------------------------------------------------------------------------ */
int rel_oracle_fwd_scan(int T, int d, const double* q, const double* k, const double* v,
                        double lambda, double tau_s, int tile, int reverse, double* y,
                        double* logz) {
  if (bad_args(T, d, q, k, v) || !y || tile < 1 || !(tau_s > 0.0)) return -1;
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* z = (double*)malloc(sizeof(double) * (size_t)d);
  if (!z) return -1;
  for (int r = 0; r < T; ++r) {
    const double* qr = q + (size_t)r * d;
    double m = -INFINITY, l = 0.0;
    for (int c = 0; c < d; ++c) z[c] = 0.0;
    int ntiles = (r + tile - 1) / tile; /* tiles covering keys 0..r-1 */
    for (int t = 0; t < ntiles; ++t) {
      int tb = reverse ? (ntiles - 1 - t) : t;
      int j0 = tb * tile, j1 = j0 + tile < r ? j0 + tile : r;
      double mb = -INFINITY;
      for (int j = j0; j < j1; ++j) {
        double e = silu(dot(qr, k + (size_t)j * d, d) * inv_sqrt_d);
        mb = e > mb ? e : mb;
      }
      double mnew = m > mb ? m : mb;
      double scale = exp(m - mnew); /* exp(-inf) = 0 for the empty state */
      l *= scale;
      for (int c = 0; c < d; ++c) z[c] *= scale;
      for (int j = j0; j < j1; ++j) {
        double w = exp(silu(dot(qr, k + (size_t)j * d, d) * inv_sqrt_d) - mnew);
        l += w;
        for (int c = 0; c < d; ++c) z[c] += w * v[(size_t)j * d + c];
      }
      m = mnew;
    }
    double s_i = sigmoid(dot(qr, k + (size_t)r * d, d) * inv_sqrt_d / tau_s);
    if (r == 0) { /* empty history: App. A.1.8 */
      for (int c = 0; c < d; ++c) y[c] = v[c];
      if (logz) logz[0] = s_i;
      continue;
    }
    double a = m + log(l) - lambda * log((double)(r + 1));
    double g_i = sigmoid(a - s_i);
    for (int c = 0; c < d; ++c)
      y[(size_t)r * d + c] = (1.0 - g_i) * v[(size_t)r * d + c] + g_i * z[c] / l;
    if (logz) {
      double hi = s_i > a ? s_i : a, lo = s_i > a ? a : s_i;
      logz[r] = hi + log1p(exp(lo - hi));
    }
  }
  free(z);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Backward, generic softmax gradient (App. A.1.7, general transport).       */
/* With G = dL/dY: H_ij = G_i . I~_j, dL/dR_ij = F_ij (H_ij - sum_k F_ik H_ik),*/
/* dU_ii = dR_ii S_i (1 - S_i) / tau_S, dU_ij = dR_ij SiLU'(U_ij) (j < i),   */
/* dP1 = dU P2 / sqrt(d), dP2 = dU^T P1 / sqrt(d), dI~ = F^T G and           */
/* dL/dlambda = sum_{i, j<i} dR_ij (-log i).  Rows are processed one at a    */
/* time with the full materialised row R_i, F_i of relation_row().           */
/* dq, dk, dv: [T][d]; dlambda: scalar.  Any of the four may be NULL.        */
/* ------------------------------------------------------------------------ */
/* rel_oracle_bwd_tail: the same computation restricted to the rows r >= row_begin.
 * Rows are independent in this form, so the outputs are exact for dq rows
 * r >= row_begin and for dk, dv rows j >= row_begin (only rows i >= j feed key j);
 * dq rows below row_begin are set to 0, and dlambda sums the processed rows only.
 * rel_oracle_bwd is the case row_begin = 0. */
int rel_oracle_bwd_tail(int T, int d, const double* q, const double* k, const double* v,
                        const double* dy, double lambda, double tau_s, int row_begin,
                        double* dq, double* dk, double* dv, double* dlambda) {
  if (bad_args(T, d, q, k, v) || !dy || !(tau_s > 0.0) || row_begin < 0 || row_begin >= T)
    return -1;
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* U = (double*)malloc(sizeof(double) * (size_t)T);
  double* Rr = (double*)malloc(sizeof(double) * (size_t)T);
  double* Fr = (double*)malloc(sizeof(double) * (size_t)T);
  double* Hr = (double*)malloc(sizeof(double) * (size_t)T);
  double* yr = (double*)malloc(sizeof(double) * (size_t)d);
  double* gk = (double*)calloc((size_t)T * d, sizeof(double));
  double* gv = (double*)calloc((size_t)T * d, sizeof(double));
  if (!U || !Rr || !Fr || !Hr || !yr || !gk || !gv) {
    free(U); free(Rr); free(Fr); free(Hr); free(yr); free(gk); free(gv);
    return -1;
  }
  double dlam = 0.0;
  if (dq)
    for (size_t n = 0; n < (size_t)row_begin * d; ++n) dq[n] = 0.0;
  for (int r = row_begin; r < T; ++r) {
    double lz;
    relation_row(r, T, d, q, k, v, lambda, tau_s, U, Rr, Fr, yr, &lz);
    const double* G = dy + (size_t)r * d;
    double FH = 0.0;
    for (int j = 0; j <= r; ++j) {
      Hr[j] = dot(G, v + (size_t)j * d, d);
      FH += Fr[j] * Hr[j];
    }
    double log_i = log((double)(r + 1));
    if (dq)
      for (int c = 0; c < d; ++c) dq[(size_t)r * d + c] = 0.0;
    for (int j = 0; j <= r; ++j) {
      double dR = Fr[j] * (Hr[j] - FH);
      double dU;
      if (j == r) {
        double s = Rr[r]; /* R_ii = S_i */
        dU = dR * s * (1.0 - s) / tau_s;
      } else {
        dU = dR * silu_grad(U[j]);
        dlam += -log_i * dR;
      }
      for (int c = 0; c < d; ++c) {
        if (dq) dq[(size_t)r * d + c] += dU * k[(size_t)j * d + c] * inv_sqrt_d;
        gk[(size_t)j * d + c] += dU * q[(size_t)r * d + c] * inv_sqrt_d;
        gv[(size_t)j * d + c] += Fr[j] * G[c];
      }
    }
  }
  if (dk) memcpy(dk, gk, sizeof(double) * (size_t)T * d);
  if (dv) memcpy(dv, gv, sizeof(double) * (size_t)T * d);
  if (dlambda) *dlambda = dlam;
  free(U); free(Rr); free(Fr); free(Hr); free(yr); free(gk); free(gv);
  return 0;
}

int rel_oracle_bwd(int T, int d, const double* q, const double* k, const double* v,
                   const double* dy, double lambda, double tau_s, double* dq, double* dk,
                   double* dv, double* dlambda) {
  return rel_oracle_bwd_tail(T, d, q, k, v, dy, lambda, tau_s, 0, dq, dk, dv, dlambda);
}

/* ------------------------------------------------------------------------ */
/* Backward, Self-Exchange credit decomposition (App. A.1.7, first part).    */
/* From the factorised quantities (S, E, pi^E, g, Ibar, Delta = Ibar - I~_i):*/
/*   dI~_j   = (1 - g_j) G_j + sum_{i>j} g_i pi^E_ij G_i                     */
/*   c_i     = G_i . Delta_i                                                 */
/*   dL/dS_i = -g_i (1 - g_i) c_i                                            */
/*   dL/dE_ij = g_i pi^E_ij [ (1 - g_i) c_i + G_i . (I~_j - Ibar_i) ]       */
/*   dL/dlambda = - sum_{i>1} g_i (1 - g_i) c_i log i                        */
/* and the role-map derivatives chain dS, dE to U and then to P1, P2.       */
/* Row 1 has g = 0 and contributes only (1 - g_1) G_1 = G_1 to dI~_1 and its */
/* Self term (zero, since dS_1 = 0).                                         */
/* ------------------------------------------------------------------------ */
int rel_oracle_bwd_credit(int T, int d, const double* q, const double* k, const double* v,
                          const double* dy, double lambda, double tau_s, double* dq, double* dk,
                          double* dv, double* dlambda) {
  if (bad_args(T, d, q, k, v) || !dy || !(tau_s > 0.0)) return -1;
  const double inv_sqrt_d = 1.0 / sqrt((double)d);
  double* yy = (double*)malloc(sizeof(double) * (size_t)T * d);
  double* S = (double*)malloc(sizeof(double) * (size_t)T);
  double* g = (double*)malloc(sizeof(double) * (size_t)T);
  double* Ib = (double*)malloc(sizeof(double) * (size_t)T * d);
  double* pi = (double*)malloc(sizeof(double) * (size_t)T * T);
  double* gq = (double*)calloc((size_t)T * d, sizeof(double));
  double* gk = (double*)calloc((size_t)T * d, sizeof(double));
  double* gv = (double*)calloc((size_t)T * d, sizeof(double));
  int rc = -1;
  if (!yy || !S || !g || !Ib || !pi || !gq || !gk || !gv) goto done;
  if (rel_oracle_fwd_factorized(T, d, q, k, v, lambda, tau_s, yy, NULL, S, NULL, NULL, g, NULL,
                                Ib, pi) != 0)
    goto done;
  double dlam = 0.0;
  for (int r = 0; r < T; ++r) {
    const double* G = dy + (size_t)r * d;
    const double* qr = q + (size_t)r * d;
    /* dI~_r += (1 - g_r) G_r  (Self share) */
    for (int c = 0; c < d; ++c) gv[(size_t)r * d + c] += (1.0 - g[r]) * G[c];
    if (r == 0) continue; /* g_1 = 0: no Exchange, no Self-Exchange credit */
    double c_i = 0.0;
    for (int c = 0; c < d; ++c) c_i += G[c] * (Ib[(size_t)r * d + c] - v[(size_t)r * d + c]);
    double gg = g[r] * (1.0 - g[r]);
    /* Self: dL/dS_i = -g(1-g)c, then dS/dU_ii = S(1-S)/tau_S */
    double dU_self = -gg * c_i * S[r] * (1.0 - S[r]) / tau_s;
    for (int c = 0; c < d; ++c) {
      gq[(size_t)r * d + c] += dU_self * k[(size_t)r * d + c] * inv_sqrt_d;
      gk[(size_t)r * d + c] += dU_self * qr[c] * inv_sqrt_d;
    }
    dlam += -gg * c_i * log((double)(r + 1));
    for (int j = 0; j < r; ++j) {
      double p = pi[(size_t)r * T + j];
      /* dI~_j += g_i pi_ij G_i (Exchange share) */
      for (int c = 0; c < d; ++c) gv[(size_t)j * d + c] += g[r] * p * G[c];
      double gdiff = 0.0;
      for (int c = 0; c < d; ++c) gdiff += G[c] * (v[(size_t)j * d + c] - Ib[(size_t)r * d + c]);
      double dE = g[r] * p * ((1.0 - g[r]) * c_i + gdiff);
      double u = dot(qr, k + (size_t)j * d, d) * inv_sqrt_d;
      double dU = dE * silu_grad(u);
      for (int c = 0; c < d; ++c) {
        gq[(size_t)r * d + c] += dU * k[(size_t)j * d + c] * inv_sqrt_d;
        gk[(size_t)j * d + c] += dU * qr[c] * inv_sqrt_d;
      }
    }
  }
  if (dq) memcpy(dq, gq, sizeof(double) * (size_t)T * d);
  if (dk) memcpy(dk, gk, sizeof(double) * (size_t)T * d);
  if (dv) memcpy(dv, gv, sizeof(double) * (size_t)T * d);
  if (dlambda) *dlambda = dlam;
  rc = 0;
done:
  free(yy); free(S); free(g); free(Ib); free(pi); free(gq); free(gk); free(gv);
  return rc;
}

/* ------------------------------------------------------------------------ */
/* Multi-Head Relation wrappers (Sec. 3.2, App. A.2.1): every (b, h) head is */
/* an independent SER problem.  Tensors are [B][T][H][d] with element strides*/
/* sB, sT, sH (d contiguous); logz is [B][H][T].  Heads run in parallel      */
/* (OpenMP) when the library was built with it; nthreads <= 0 keeps the     */
/* runtime default.  dlambda (bwd) sums over all heads (lambda is shared).   */
/* ------------------------------------------------------------------------ */
static void gather_head(const double* src, double* dst, int T, int d, long long sT,
                        long long off) {
  for (int t = 0; t < T; ++t)
    for (int c = 0; c < d; ++c) dst[(size_t)t * d + c] = src[off + (long long)t * sT + c];
}
static void scatter_head(const double* src, double* dst, int T, int d, long long sT,
                         long long off) {
  for (int t = 0; t < T; ++t)
    for (int c = 0; c < d; ++c) dst[off + (long long)t * sT + c] = src[(size_t)t * d + c];
}

int rel_oracle_mhr_fwd(int B, int T, int H, int d, long long sB, long long sT, long long sH,
                       const double* q, const double* k, const double* v, double lambda,
                       double tau_s, double* y, double* logz, int nthreads) {
  if (B < 1 || H < 1 || bad_args(T, d, q, k, v) || !y || !logz) return -1;
  int fail = 0;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
  for (int bh = 0; bh < B * H; ++bh) {
    int b = bh / H, h = bh % H;
    long long off = (long long)b * sB + (long long)h * sH;
    size_t n = (size_t)T * d;
    double* buf = (double*)malloc(sizeof(double) * n * 4);
    if (!buf) {
#pragma omp atomic write
      fail = 1;
      continue;
    }
    double *hq = buf, *hk = buf + n, *hv = buf + 2 * n, *hy = buf + 3 * n;
    gather_head(q, hq, T, d, sT, off);
    gather_head(k, hk, T, d, sT, off);
    gather_head(v, hv, T, d, sT, off);
    if (rel_oracle_fwd(T, d, hq, hk, hv, lambda, tau_s, hy, logz + (size_t)bh * T, NULL,
                       NULL) != 0) {
#pragma omp atomic write
      fail = 1;
    }
    scatter_head(hy, y, T, d, sT, off);
    free(buf);
  }
  return fail ? -1 : 0;
}

int rel_oracle_mhr_bwd(int B, int T, int H, int d, long long sB, long long sT, long long sH,
                       const double* q, const double* k, const double* v, const double* dy,
                       double lambda, double tau_s, double* dq, double* dk, double* dv,
                       double* dlambda, int nthreads) {
  if (B < 1 || H < 1 || bad_args(T, d, q, k, v) || !dy || !dq || !dk || !dv || !dlambda)
    return -1;
  int fail = 0;
  double* dl = (double*)calloc((size_t)B * H, sizeof(double));
  if (!dl) return -1;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
  for (int bh = 0; bh < B * H; ++bh) {
    int b = bh / H, h = bh % H;
    long long off = (long long)b * sB + (long long)h * sH;
    size_t n = (size_t)T * d;
    double* buf = (double*)malloc(sizeof(double) * n * 7);
    if (!buf) {
#pragma omp atomic write
      fail = 1;
      continue;
    }
    double *hq = buf, *hk = buf + n, *hv = buf + 2 * n, *hg = buf + 3 * n;
    double *gq = buf + 4 * n, *gk = buf + 5 * n, *gv = buf + 6 * n;
    gather_head(q, hq, T, d, sT, off);
    gather_head(k, hk, T, d, sT, off);
    gather_head(v, hv, T, d, sT, off);
    gather_head(dy, hg, T, d, sT, off);
    if (rel_oracle_bwd(T, d, hq, hk, hv, hg, lambda, tau_s, gq, gk, gv, dl + bh) != 0) {
#pragma omp atomic write
      fail = 1;
    }
    scatter_head(gq, dq, T, d, sT, off);
    scatter_head(gk, dk, T, d, sT, off);
    scatter_head(gv, dv, T, d, sT, off);
    free(buf);
  }
  double tot = 0.0;
  for (int bh = 0; bh < B * H; ++bh) tot += dl[bh]; /* fixed order: deterministic */
  *dlambda = tot;
  free(dl);
  return fail ? -1 : 0;
}

/* Threads an OpenMP parallel region of this library would use (1 without OpenMP). */
int rel_oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
