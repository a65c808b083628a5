/*
 * linear_oracle.c -- plain, slow fp64 CPU oracle for Linear Relation, the recurrent
 * Exchange form of "Ask Self, Ask Others: Relation Is All You Need" (arxiv 2608.20172).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the package's smoke check and the
 * benchmark's CPU baseline leg may build, load or call it.  It shares no code, header,
 * table or constant with the CUDA library, and the CUDA library never calls it.
 *
 * Every routine works on ONE head with contiguous row-major [T][d] fp64 arrays (rows are
 * tokens t = 1..T in the paper's notation, zero-based here).  Inputs: the relation
 * coordinates p1_t, p2_t (after RoPE, which is upstream), the information I~_t (v), and
 * the channel-wise retention alpha_t in (0, 1]^d (produced upstream by the KDA-style
 * parameterisation of Eq. (retention-vector); it is an input here).
 *
 * Definitions followed (paper section / equation):
 *   S_t = sigmoid(p1_t . p2_t / (tau_S sqrt(d)))        Eq. (linear-self-relation), App. A.4.1
 *   ^p1_t = p1_t / |p1_t|,  ^p2_t = p2_t / |p2_t|        Eq. (linear-self-relation)
 *   C_0 = 0;  C_t^- = Diag(alpha_t) C_{t-1}              App. A.4.2 (recurrent step)
 *   E_t = S_t (C_t^-)^T ^p1_t;  Y_t = I~_t + E_t          Eq. (decayed-relation-state)
 *   C_t = C_t^- + S_t ^p2_t I~_t^T                        (Ask Self -> Ask Others -> Answer
 *                                                          -> Become Others)
 *   unrolled: E_t = sum_{j<t} S_t S_j [^p2_j^T (prod_{u=j+1..t} Diag(alpha_u)) ^p1_t] I~_j
 *                                                        App. A.4.4-A.4.5
 * C is d x d with the row index on the coordinate (^p) side and the column index on
 * the information side.
 *
 * Readings where the paper leaves a choice: tau_S = 2 as for the Self relation of
 * Sec. 3.1, which Linear Relation keeps; the state starts at zero for every sequence;
 * the L2 normalisation has no epsilon (a zero p1 or p2 row is outside the operator's
 * domain); tau_S carries no gradient.  The backward (not written out in the paper) is
 * the reverse-mode derivative of the recurrent step above, taken in reverse token order.
 *
 * Return value of every entry point: 0 on success, -1 on a bad argument.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

static double lsig(double x) { return 1.0 / (1.0 + exp(-x)); }

static double ldot(const double* a, const double* b, int d) {
  double s = 0.0;
  for (int c = 0; c < d; ++c) s += a[c] * b[c];
  return s;
}

static int lbad(int T, int d, const void* p1, const void* p2, const void* v, const void* alpha) {
  return T < 1 || d < 1 || !p1 || !p2 || !v || !alpha;
}

/* Ask Self: S_t, ^p1_t, ^p2_t of one token. */
static void ask_self(int d, const double* p1, const double* p2, double tau_s, double* S,
                     double* q, double* k) {
  const double n1 = sqrt(ldot(p1, p1, d)), n2 = sqrt(ldot(p2, p2, d));
  *S = lsig(ldot(p1, p2, d) / (tau_s * sqrt((double)d)));
  for (int c = 0; c < d; ++c) {
    q[c] = p1[c] / n1;
    k[c] = p2[c] / n2;
  }
}

/* Recurrent forward (App. A.4.2).  y [T][d]; S (optional) [T]; states (optional)
 * [T + 1][d][d] receives C_0 .. C_T. */
int rel_linear_fwd(int T, int d, const double* p1, const double* p2, const double* v,
                   const double* alpha, double tau_s, double* y, double* S, double* states) {
  if (lbad(T, d, p1, p2, v, alpha) || !y || !(tau_s > 0.0)) return -1;
  double* C = (double*)calloc((size_t)d * d, sizeof(double));
  double* q = (double*)malloc(sizeof(double) * (size_t)d);
  double* k = (double*)malloc(sizeof(double) * (size_t)d);
  if (!C || !q || !k) { free(C); free(q); free(k); return -1; }
  if (states) memcpy(states, C, sizeof(double) * (size_t)d * d);
  for (int t = 0; t < T; ++t) {
    const double* I = v + (size_t)t * d;
    const double* a = alpha + (size_t)t * d;
    double s_t;
    ask_self(d, p1 + (size_t)t * d, p2 + (size_t)t * d, tau_s, &s_t, q, k);
    /* C_t^- = Diag(alpha_t) C_{t-1} */
    for (int c = 0; c < d; ++c)
      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] *= a[c];
    /* Ask Others: E_t = S_t (C_t^-)^T ^p1_t;  Answer: Y_t = I~_t + E_t */
    for (int j = 0; j < d; ++j) {
      double e = 0.0;
      for (int c = 0; c < d; ++c) e += C[(size_t)c * d + j] * q[c];
      y[(size_t)t * d + j] = I[j] + s_t * e;
    }
    /* Become Others: C_t = C_t^- + S_t ^p2_t I~_t^T */
    for (int c = 0; c < d; ++c)
      for (int j = 0; j < d; ++j) C[(size_t)c * d + j] += s_t * k[c] * I[j];
    if (S) S[t] = s_t;
    if (states) memcpy(states + (size_t)(t + 1) * d * d, C, sizeof(double) * (size_t)d * d);
  }
  free(C); free(q); free(k);
  return 0;
}

/* Unrolled forward (App. A.4.4-A.4.5), O(T^2 d^2 + T^2 d): each historical token j
 * contributes S_t S_j [^p2_j^T (prod_{u=j+1..t} Diag(alpha_u)) ^p1_t] I~_j. */
int rel_linear_fwd_unrolled(int T, int d, const double* p1, const double* p2, const double* v,
                            const double* alpha, double tau_s, double* y) {
  if (lbad(T, d, p1, p2, v, alpha) || !y || !(tau_s > 0.0)) return -1;
  double* S = (double*)malloc(sizeof(double) * (size_t)T);
  double* Q = (double*)malloc(sizeof(double) * (size_t)T * d);
  double* K = (double*)malloc(sizeof(double) * (size_t)T * d);
  double* prod = (double*)malloc(sizeof(double) * (size_t)d);
  if (!S || !Q || !K || !prod) { free(S); free(Q); free(K); free(prod); return -1; }
  for (int t = 0; t < T; ++t)
    ask_self(d, p1 + (size_t)t * d, p2 + (size_t)t * d, tau_s, &S[t], Q + (size_t)t * d,
             K + (size_t)t * d);
  for (int t = 0; t < T; ++t) {
    double* yt = y + (size_t)t * d;
    for (int j = 0; j < d; ++j) yt[j] = v[(size_t)t * d + j];
    for (int c = 0; c < d; ++c) prod[c] = 1.0;
    for (int j = t - 1; j >= 0; --j) {
      /* prod = prod_{u=j+1..t} alpha_u, built from u = t downwards */
      for (int c = 0; c < d; ++c) prod[c] *= alpha[(size_t)(j + 1) * d + c];
      double w = 0.0;
      for (int c = 0; c < d; ++c) w += K[(size_t)j * d + c] * prod[c] * Q[(size_t)t * d + c];
      w *= S[t] * S[j];
      for (int c = 0; c < d; ++c) yt[c] += w * v[(size_t)j * d + c];
    }
  }
  free(S); free(Q); free(K); free(prod);
  return 0;
}

/* Backward: reverse-mode derivative of the recurrent step, tokens in reverse order, with
 * dy = dL/dY.  Writes dp1, dp2, dv, dalpha (all [T][d]). */
int rel_linear_bwd(int T, int d, const double* p1, const double* p2, const double* v,
                   const double* alpha, const double* dy, double tau_s, double* dp1,
                   double* dp2, double* dv, double* dalpha) {
  if (lbad(T, d, p1, p2, v, alpha) || !dy || !dp1 || !dp2 || !dv || !dalpha ||
      !(tau_s > 0.0))
    return -1;
  const size_t dd = (size_t)d * d;
  double* states = (double*)malloc(sizeof(double) * (size_t)(T + 1) * dd);
  double* y = (double*)malloc(sizeof(double) * (size_t)T * d);
  double* dC = (double*)calloc(dd, sizeof(double));
  double* Cm = (double*)malloc(sizeof(double) * dd);
  double* q = (double*)malloc(sizeof(double) * (size_t)d);
  double* k = (double*)malloc(sizeof(double) * (size_t)d);
  double* dq = (double*)malloc(sizeof(double) * (size_t)d);
  double* dk = (double*)malloc(sizeof(double) * (size_t)d);
  if (!states || !y || !dC || !Cm || !q || !k || !dq || !dk) {
    free(states); free(y); free(dC); free(Cm); free(q); free(k); free(dq); free(dk);
    return -1;
  }
  rel_linear_fwd(T, d, p1, p2, v, alpha, tau_s, y, NULL, states);
  const double rsd = 1.0 / sqrt((double)d);
  for (int t = T - 1; t >= 0; --t) {
    const double* P1 = p1 + (size_t)t * d;
    const double* P2 = p2 + (size_t)t * d;
    const double* I = v + (size_t)t * d;
    const double* a = alpha + (size_t)t * d;
    const double* G = dy + (size_t)t * d;
    const double* Cprev = states + (size_t)t * dd;  /* C_{t-1} */
    double s_t;
    ask_self(d, P1, P2, tau_s, &s_t, q, k);
    for (int c = 0; c < d; ++c)
      for (int j = 0; j < d; ++j) Cm[(size_t)c * d + j] = a[c] * Cprev[(size_t)c * d + j];
    double dS = 0.0;
    /* Become Others: C_t = C_t^- + S k I^T */
    for (int j = 0; j < d; ++j) {
      double kdc = 0.0;  /* (dC^T k)_j */
      for (int c = 0; c < d; ++c) kdc += dC[(size_t)c * d + j] * k[c];
      dv[(size_t)t * d + j] = G[j] + s_t * kdc;  /* Answer: Y = I + E;  write */
      dS += kdc * I[j];
    }
    for (int c = 0; c < d; ++c) {
      double dci = 0.0;  /* (dC I)_c */
      for (int j = 0; j < d; ++j) dci += dC[(size_t)c * d + j] * I[j];
      dk[c] = s_t * dci;
    }
    /* Ask Others: E = S (C_t^-)^T q */
    for (int j = 0; j < d; ++j) {
      double h = 0.0;
      for (int c = 0; c < d; ++c) h += Cm[(size_t)c * d + j] * q[c];
      dS += G[j] * h;
    }
    for (int c = 0; c < d; ++c) {
      double cg = 0.0;
      for (int j = 0; j < d; ++j) cg += Cm[(size_t)c * d + j] * G[j];
      dq[c] = s_t * cg;
    }
    /* dL/dC_t^- = dC + S q G^T; then C_t^- = Diag(alpha) C_{t-1} */
    for (int c = 0; c < d; ++c) {
      double da = 0.0;
      for (int j = 0; j < d; ++j) {
        const double dcm = dC[(size_t)c * d + j] + s_t * q[c] * G[j];
        da += dcm * Cprev[(size_t)c * d + j];
        dC[(size_t)c * d + j] = a[c] * dcm;  /* becomes dL/dC_{t-1} */
      }
      dalpha[(size_t)t * d + c] = da;
    }
    /* Ask Self: S = sigmoid(p1 . p2 / (tau sqrt d)), q = p1 / |p1|, k = p2 / |p2| */
    const double du = dS * s_t * (1.0 - s_t) / tau_s * rsd;
    const double n1 = sqrt(ldot(P1, P1, d)), n2 = sqrt(ldot(P2, P2, d));
    const double qdq = ldot(q, dq, d), kdk = ldot(k, dk, d);
    for (int c = 0; c < d; ++c) {
      dp1[(size_t)t * d + c] = du * P2[c] + (dq[c] - q[c] * qdq) / n1;
      dp2[(size_t)t * d + c] = du * P1[c] + (dk[c] - k[c] * kdk) / n2;
    }
  }
  free(states); free(y); free(dC); free(Cm); free(q); free(k); free(dq); free(dk);
  return 0;
}
