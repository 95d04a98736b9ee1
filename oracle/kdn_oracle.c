/*
 * kdn_oracle.c -- plain fp64 CPU oracle for the Kalman Delta Network (KDN)
 * token mixers.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * reference that the CUDA path is checked against.  Only the test suite,
 * the smoke check and the benchmark's CPU-baseline leg may load it; the
 * product library never links, loads or calls it, and it shares no code,
 * header, table or helper with the CUDA path.
 *
 * Everything is a direct token-by-token transcription of the paper's
 * equations in float64, with no chunking, blocking or reordering:
 *
 *   Diagonal KDN, Prop. 3 ("Diagonal Kalman Delta Network"):
 *     alpha_t = exp(g_t)                       (g = log alpha is the input)
 *     phat_t  = alpha_t^2 * p_{t-1} + omega_t  (eq. diag-covariance-prediction)
 *     kappa_t = phat_t * k_t / (r_t + sum_i phat_ti k_ti^2)   (eq. kla-box-gain)
 *     Shat_t  = diag(alpha_t) S_{t-1}
 *     S_t     = Shat_t + kappa_t (v_t - Shat_t^T k_t)^T         (eq. kla-box-memory)
 *     o_t     = tau * S_t^T q_t   (read of the post-write state; App. F.2
 *                                  keeps the diagonal of A_qk for this reason)
 *     u_t     = mu * k_t * k_t / r_t                            (eq. diag-cov-update)
 *     p_t     = phat_t / (1 + u_t * phat_t)           (eq. prefix-diag-uncertainty)
 *
 *   Isotropic KDN, Prop. 5 ("Isotropic Kalman Delta Network", App. E):
 *     a_t    = (1/d_k) sum_i alpha_ti^2   (alpha_t^2 when the decay is one
 *                                          scalar per head)
 *     bhat_t = a_t b_{t-1} + omega_t
 *     beta_t = bhat_t / (r_t + bhat_t |k_t|^2),  kappa_t = beta_t k_t
 *     memory as above with D_t = diag(alpha_t)
 *     u_t    = mu |k_t|^2 / (d_k r_t),  b_t = bhat_t / (1 + u_t bhat_t)
 *
 * Surrogate mode (isotropic only): when a per-token predicted variance
 * bhat_t is supplied, it replaces the tracked one.  This is the fixed-gain
 * surrogate of eq. fixed-gain-approx (Sec. 3.3) under which the update is the
 * textbook delta rule of eq. unified-delta-rule.
 *
 * The backward pass is not given in the paper.  It is the adjoint of the
 * token loop above, derived by hand (reverse-mode differentiation of each
 * assignment, in reverse order) and run with (S, p) checkpoints every
 * CKPT tokens and forward recomputation inside each segment.
 *
 * Layouts (row-major, the same ones the C ABI uses):
 *   q, k           [B, T, H, dk]      v, o           [B, T, H, dv]
 *   g, omega (diag)[B, T, H, dk]      r              [B, T, H]
 *   omega (iso)    [B, T, H]          g (iso)        [B, T, H, dk] or [B, T, H]
 *   S0, ST         [B, H, dk, dv]     p0, pT  diag   [B, H, dk];  iso [B, H]
 */
#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define CKPT 64

typedef struct {
  int variant;           /* 0 = Diagonal KDN, 1 = Isotropic KDN */
  int B, T, H, dk, dv;
  double mu, tau;
  int per_channel_decay; /* isotropic: 1 -> g is [B,T,H,dk]; 0 -> [B,T,H] */
  const double *q, *k, *v, *g, *omega, *r, *S0, *p0;
  const double *bhat_in; /* isotropic surrogate mode, [B,T,H]; NULL = tracked */
  double *o, *ST, *pT;
  double *kappa_out, *phat_out, *p_out; /* optional per-token traces */
  /* backward */
  const double *dO, *dST, *dpT;
  double *dq, *dk_, *dv_, *dg, *domega, *dr, *dS0, *dp0;
  double *dmu; /* [B,H] dL/dmu of each sequence (mu enters only through u), or NULL */
} job_t;

/* Per-token intermediates of one forward step, kept for the adjoint. */
typedef struct {
  double *alpha;  /* [dk] */
  double *phat;   /* [dk] diag; [1] iso */
  double *kappa;  /* [dk] */
  double *u;      /* [dk] diag; [1] iso */
  double *delta;  /* [dv] innovation v - Shat^T k */
  double s;       /* diag: r + sum phat k^2 */
  double a, n2, beta; /* iso */
} step_t;

static size_t tok(const job_t *J, int b, int t, int h) {
  return ((size_t)b * J->T + t) * J->H + h;
}

static int pdim(const job_t *J) { return J->variant == 0 ? J->dk : 1; }

/*
 * One token of Prop. 3 (variant 0) or Prop. 5 (variant 1), in place on
 * (S, p).  S is [dk, dv], p is [dk] (diag) or [1] (iso).  Writes o_t.
 */
static void fwd_step(const job_t *J, int b, int t, int h, double *S, double *p,
                     double *o_t, step_t *st) {
  const int dk = J->dk, dv = J->dv;
  const size_t th = tok(J, b, t, h);
  const double *kt = J->k + th * dk;
  const double *qt = J->q + th * dk;
  const double *vt = J->v + th * dv;
  const double rt = J->r[th];

  /* transition D_t = diag(alpha_t), alpha = exp(g) */
  for (int i = 0; i < dk; ++i) {
    double gi;
    if (J->variant == 1 && !J->per_channel_decay) gi = J->g[th];
    else gi = J->g[th * dk + i];
    st->alpha[i] = exp(gi);
  }

  if (J->variant == 0) {
    /* eq. diag-covariance-prediction and eq. kla-box-gain */
    double s = rt;
    for (int i = 0; i < dk; ++i) {
      st->phat[i] = st->alpha[i] * st->alpha[i] * p[i] + J->omega[th * dk + i];
      s += st->phat[i] * kt[i] * kt[i];
    }
    st->s = s;
    for (int i = 0; i < dk; ++i) st->kappa[i] = st->phat[i] * kt[i] / s;
  } else {
    /* eq. iso-kla-box-cov-update and eq. iso-kla-box-gain */
    double a = 0.0, n2 = 0.0;
    for (int i = 0; i < dk; ++i) {
      a += st->alpha[i] * st->alpha[i];
      n2 += kt[i] * kt[i];
    }
    a /= dk;
    st->a = a;
    st->n2 = n2;
    double bhat = J->bhat_in ? J->bhat_in[th] : a * p[0] + J->omega[th];
    st->phat[0] = bhat;
    st->beta = bhat / (rt + bhat * n2);
    for (int i = 0; i < dk; ++i) st->kappa[i] = st->beta * kt[i];
  }

  /* prediction Shat = D S and innovation delta = v - Shat^T k */
  for (int i = 0; i < dk; ++i)
    for (int j = 0; j < dv; ++j) S[(size_t)i * dv + j] *= st->alpha[i];
  for (int j = 0; j < dv; ++j) {
    double acc = 0.0;
    for (int i = 0; i < dk; ++i) acc += S[(size_t)i * dv + j] * kt[i];
    st->delta[j] = vt[j] - acc;
  }
  /* residual write S = Shat + kappa delta^T */
  for (int i = 0; i < dk; ++i)
    for (int j = 0; j < dv; ++j) S[(size_t)i * dv + j] += st->kappa[i] * st->delta[j];
  /* read of the post-write state */
  for (int j = 0; j < dv; ++j) {
    double acc = 0.0;
    for (int i = 0; i < dk; ++i) acc += S[(size_t)i * dv + j] * qt[i];
    o_t[j] = J->tau * acc;
  }
  /* information-scaled posterior variance (eq. diag-cov-update / Prop. 5) */
  if (J->variant == 0) {
    for (int i = 0; i < dk; ++i) {
      st->u[i] = J->mu * kt[i] * kt[i] / rt;
      p[i] = st->phat[i] / (1.0 + st->u[i] * st->phat[i]);
    }
  } else {
    st->u[0] = J->mu * st->n2 / (dk * rt);
    p[0] = st->phat[0] / (1.0 + st->u[0] * st->phat[0]);
  }
}

static void step_alloc(step_t *st, int dk, int dv) {
  st->alpha = calloc(dk, sizeof(double));
  st->phat = calloc(dk, sizeof(double));
  st->kappa = calloc(dk, sizeof(double));
  st->u = calloc(dk, sizeof(double));
  st->delta = calloc(dv, sizeof(double));
}

static void step_free(step_t *st) {
  free(st->alpha); free(st->phat); free(st->kappa); free(st->u); free(st->delta);
}

static void init_state(const job_t *J, int b, int h, double *S, double *p) {
  const int dk = J->dk, dv = J->dv, np = pdim(J);
  const size_t sd = ((size_t)b * J->H + h) * dk * dv;
  if (J->S0) memcpy(S, J->S0 + sd, sizeof(double) * dk * dv);
  else memset(S, 0, sizeof(double) * dk * dv);
  for (int i = 0; i < np; ++i)
    p[i] = J->p0 ? J->p0[((size_t)b * J->H + h) * np + i] : 1.0;
}

static void fwd_one(const job_t *J, int b, int h) {
  const int dk = J->dk, dv = J->dv, np = pdim(J);
  double *S = malloc(sizeof(double) * dk * dv);
  double *p = malloc(sizeof(double) * np);
  step_t st;
  step_alloc(&st, dk, dv);
  init_state(J, b, h, S, p);
  for (int t = 0; t < J->T; ++t) {
    const size_t th = tok(J, b, t, h);
    fwd_step(J, b, t, h, S, p, J->o + th * dv, &st);
    if (J->kappa_out) memcpy(J->kappa_out + th * dk, st.kappa, sizeof(double) * dk);
    if (J->phat_out) memcpy(J->phat_out + th * np, st.phat, sizeof(double) * np);
    if (J->p_out) memcpy(J->p_out + th * np, p, sizeof(double) * np);
  }
  const size_t bh = (size_t)b * J->H + h;
  if (J->ST) memcpy(J->ST + bh * dk * dv, S, sizeof(double) * dk * dv);
  if (J->pT) memcpy(J->pT + bh * np, p, sizeof(double) * np);
  step_free(&st);
  free(S);
  free(p);
}

/*
 * Adjoint of one forward step.  On entry dS = dL/dS_t (all later uses
 * included), dp = dL/dp_t; Sprev/pprev are the state before token t, Scur the
 * state after it.  On exit dS = dL/dS_{t-1}, dp = dL/dp_{t-1}, and this
 * token's input gradients are written.
 */
static void bwd_step(const job_t *J, int b, int t, int h, const double *Sprev,
                     const double *pprev, const double *Scur, const step_t *st,
                     double *dS, double *dp, double *dalpha, double *dkap,
                     double *dphat, double *dkt) {
  const int dk = J->dk, dv = J->dv;
  const size_t th = tok(J, b, t, h);
  const double *kt = J->k + th * dk;
  const double *qt = J->q + th * dk;
  const double *dot = J->dO + th * dv;
  const double rt = J->r[th];
  double dr = 0.0;

  for (int i = 0; i < dk; ++i) { dalpha[i] = 0.0; dkap[i] = 0.0; dphat[i] = 0.0; dkt[i] = 0.0; }

  /* read o_t = tau S_t^T q_t */
  for (int i = 0; i < dk; ++i) {
    double acc = 0.0;
    for (int j = 0; j < dv; ++j) {
      acc += Scur[(size_t)i * dv + j] * dot[j];
      dS[(size_t)i * dv + j] += J->tau * qt[i] * dot[j];
    }
    J->dq[th * dk + i] = J->tau * acc;
  }

  /* posterior variance p_t = phat/(1 + u phat):  dp/dphat = 1/(1+u phat)^2,
     dp/du = -p_t^2 */
  if (J->variant == 0) {
    for (int i = 0; i < dk; ++i) {
      const double den = 1.0 + st->u[i] * st->phat[i];
      const double pt = st->phat[i] / den;
      dphat[i] += dp[i] / (den * den);
      const double du = -dp[i] * pt * pt;
      /* u = mu k^2 / r */
      dkt[i] += du * 2.0 * J->mu * kt[i] / rt;
      dr += -du * st->u[i] / rt;
      if (J->dmu) J->dmu[(size_t)b * J->H + h] += du * kt[i] * kt[i] / rt;
    }
  }
  double dbhat = 0.0, dn2 = 0.0;
  if (J->variant == 1) {
    const double den = 1.0 + st->u[0] * st->phat[0];
    const double bt = st->phat[0] / den;
    dbhat += dp[0] / (den * den);
    const double du = -dp[0] * bt * bt;
    /* u = mu n2 / (dk r) */
    dn2 += du * J->mu / (dk * rt);
    dr += -du * st->u[0] / rt;
    if (J->dmu) J->dmu[(size_t)b * J->H + h] += du * st->n2 / (dk * rt);
  }

  /* residual write S_t = Shat + kappa delta^T, delta = v - Shat^T k */
  double *ddelta = calloc(dv, sizeof(double));
  for (int i = 0; i < dk; ++i) {
    double acc = 0.0;
    for (int j = 0; j < dv; ++j) acc += dS[(size_t)i * dv + j] * st->delta[j];
    dkap[i] = acc;
  }
  for (int j = 0; j < dv; ++j) {
    double acc = 0.0;
    for (int i = 0; i < dk; ++i) acc += dS[(size_t)i * dv + j] * st->kappa[i];
    ddelta[j] = acc;
    J->dv_[th * dv + j] = acc;
  }
  /* dShat = dS - k ddelta^T; dk -= Shat ddelta; Shat = diag(alpha) Sprev */
  for (int i = 0; i < dk; ++i) {
    double acc_k = 0.0, acc_a = 0.0;
    for (int j = 0; j < dv; ++j) {
      const double shat = st->alpha[i] * Sprev[(size_t)i * dv + j];
      const double dshat = dS[(size_t)i * dv + j] - kt[i] * ddelta[j];
      acc_k += shat * ddelta[j];
      acc_a += dshat * Sprev[(size_t)i * dv + j];
      dS[(size_t)i * dv + j] = st->alpha[i] * dshat; /* now dL/dS_{t-1} (memory path) */
    }
    dkt[i] -= acc_k;
    dalpha[i] += acc_a;
  }
  free(ddelta);

  if (J->variant == 0) {
    /* gain kappa = phat k / s, s = r + sum phat k^2 */
    double c = 0.0;
    for (int i = 0; i < dk; ++i) c += dkap[i] * st->kappa[i];
    const double ds = -c / st->s;
    for (int i = 0; i < dk; ++i) {
      dphat[i] += dkap[i] * kt[i] / st->s + ds * kt[i] * kt[i];
      dkt[i] += dkap[i] * st->phat[i] / st->s + 2.0 * ds * st->phat[i] * kt[i];
    }
    dr += ds;
    /* prediction phat = alpha^2 pprev + omega */
    for (int i = 0; i < dk; ++i) {
      J->domega[th * dk + i] = dphat[i];
      dalpha[i] += 2.0 * st->alpha[i] * pprev[i] * dphat[i];
      dp[i] = st->alpha[i] * st->alpha[i] * dphat[i];
    }
  } else {
    /* gain kappa = beta k, beta = bhat / (r + bhat n2) */
    double dbeta = 0.0;
    for (int i = 0; i < dk; ++i) {
      dbeta += dkap[i] * kt[i];
      dkt[i] += st->beta * dkap[i];
    }
    const double bhat = st->phat[0];
    const double den = rt + bhat * st->n2;
    dbhat += dbeta * rt / (den * den);
    dr += -dbeta * st->beta / den;
    dn2 += -dbeta * st->beta * st->beta;
    for (int i = 0; i < dk; ++i) dkt[i] += 2.0 * kt[i] * dn2;
    if (J->bhat_in) {
      /* surrogate mode: bhat is an input, nothing flows to omega or b */
      J->domega[th] = 0.0;
      dp[0] = 0.0;
    } else {
      /* bhat = a bprev + omega, a = mean alpha^2 */
      J->domega[th] = dbhat;
      const double da = pprev[0] * dbhat;
      for (int i = 0; i < dk; ++i) dalpha[i] += da * 2.0 * st->alpha[i] / dk;
      dp[0] = st->a * dbhat;
    }
  }

  /* alpha = exp(g) */
  if (J->variant == 1 && !J->per_channel_decay) {
    double acc = 0.0;
    for (int i = 0; i < dk; ++i) acc += st->alpha[i] * dalpha[i];
    J->dg[th] = acc;
  } else {
    for (int i = 0; i < dk; ++i) J->dg[th * dk + i] = st->alpha[i] * dalpha[i];
  }
  for (int i = 0; i < dk; ++i) J->dk_[th * dk + i] = dkt[i];
  J->dr[th] = dr;
}

static void bwd_one(const job_t *J, int b, int h) {
  const int dk = J->dk, dv = J->dv, np = pdim(J), T = J->T;
  const size_t sz = (size_t)dk * dv;
  const int nseg = (T + CKPT - 1) / CKPT;
  double *ckS = malloc(sizeof(double) * sz * (nseg > 0 ? nseg : 1));
  double *ckp = malloc(sizeof(double) * np * (nseg > 0 ? nseg : 1));
  double *S = malloc(sizeof(double) * sz);
  double *p = malloc(sizeof(double) * np);
  double *o_scratch = malloc(sizeof(double) * dv);
  /* states inside one segment: index m holds the state after m tokens */
  double *segS = malloc(sizeof(double) * sz * (CKPT + 1));
  double *segp = malloc(sizeof(double) * np * (CKPT + 1));
  step_t *steps = malloc(sizeof(step_t) * CKPT);
  for (int m = 0; m < CKPT; ++m) step_alloc(&steps[m], dk, dv);
  double *dS = malloc(sizeof(double) * sz);
  double *dp = malloc(sizeof(double) * np);
  double *dalpha = malloc(sizeof(double) * dk), *dkap = malloc(sizeof(double) * dk);
  double *dphat = malloc(sizeof(double) * dk), *dkt = malloc(sizeof(double) * dk);

  /* forward sweep that records a checkpoint at the start of each segment */
  init_state(J, b, h, S, p);
  for (int t = 0; t < T; ++t) {
    if (t % CKPT == 0) {
      memcpy(ckS + (size_t)(t / CKPT) * sz, S, sizeof(double) * sz);
      memcpy(ckp + (size_t)(t / CKPT) * np, p, sizeof(double) * np);
    }
    fwd_step(J, b, t, h, S, p, o_scratch, &steps[0]);
  }

  const size_t bh = (size_t)b * J->H + h;
  if (J->dmu) J->dmu[bh] = 0.0;
  for (size_t e = 0; e < sz; ++e) dS[e] = J->dST ? J->dST[bh * sz + e] : 0.0;
  for (int i = 0; i < np; ++i) dp[i] = J->dpT ? J->dpT[bh * np + i] : 0.0;

  for (int sgi = nseg - 1; sgi >= 0; --sgi) {
    const int t0 = sgi * CKPT;
    const int t1 = (t0 + CKPT < T) ? t0 + CKPT : T;
    memcpy(segS, ckS + (size_t)sgi * sz, sizeof(double) * sz);
    memcpy(segp, ckp + (size_t)sgi * np, sizeof(double) * np);
    for (int t = t0; t < t1; ++t) {
      const int m = t - t0;
      memcpy(segS + (size_t)(m + 1) * sz, segS + (size_t)m * sz, sizeof(double) * sz);
      memcpy(segp + (size_t)(m + 1) * np, segp + (size_t)m * np, sizeof(double) * np);
      fwd_step(J, b, t, h, segS + (size_t)(m + 1) * sz, segp + (size_t)(m + 1) * np,
               o_scratch, &steps[m]);
    }
    for (int t = t1 - 1; t >= t0; --t) {
      const int m = t - t0;
      bwd_step(J, b, t, h, segS + (size_t)m * sz, segp + (size_t)m * np,
               segS + (size_t)(m + 1) * sz, &steps[m], dS, dp, dalpha, dkap, dphat, dkt);
    }
  }
  if (J->dS0) memcpy(J->dS0 + bh * sz, dS, sizeof(double) * sz);
  if (J->dp0) memcpy(J->dp0 + bh * np, dp, sizeof(double) * np);

  for (int m = 0; m < CKPT; ++m) step_free(&steps[m]);
  free(steps); free(ckS); free(ckp); free(S); free(p); free(o_scratch);
  free(segS); free(segp); free(dS); free(dp); free(dalpha); free(dkap); free(dphat); free(dkt);
}

/* ---- threading over independent (b, h) sequences --------------------- */

typedef struct {
  const job_t *J;
  int bwd;
  int next; /* shared work counter, protected by lock */
  pthread_mutex_t lock;
} pool_t;

static void *worker(void *arg) {
  pool_t *P = (pool_t *)arg;
  const job_t *J = P->J;
  for (;;) {
    pthread_mutex_lock(&P->lock);
    int w = P->next++;
    pthread_mutex_unlock(&P->lock);
    if (w >= J->B * J->H) break;
    if (P->bwd) bwd_one(J, w / J->H, w % J->H);
    else fwd_one(J, w / J->H, w % J->H);
  }
  return NULL;
}

static int run(const job_t *J, int bwd, int nthreads) {
  const int units = J->B * J->H;
  if (nthreads <= 0) {
    long n = sysconf(_SC_NPROCESSORS_ONLN);
    nthreads = (int)(n > 0 ? n : 1);
  }
  if (nthreads > units) nthreads = units;
  if (nthreads < 1) nthreads = 1;
  pool_t P;
  P.J = J;
  P.bwd = bwd;
  P.next = 0;
  pthread_mutex_init(&P.lock, NULL);
  pthread_t *th = malloc(sizeof(pthread_t) * nthreads);
  for (int i = 0; i < nthreads; ++i) pthread_create(&th[i], NULL, worker, &P);
  for (int i = 0; i < nthreads; ++i) pthread_join(th[i], NULL);
  free(th);
  pthread_mutex_destroy(&P.lock);
  return nthreads;
}

static int check(int variant, int B, int T, int H, int dk, int dv) {
  if (variant != 0 && variant != 1) return -1;
  if (B < 0 || T < 0 || H < 0 || dk < 1 || dv < 1) return -1;
  return 0;
}

/* ---- exported entry points (called through ctypes) ------------------- */

/* Forward over T tokens (Prop. 3 / Prop. 5).  Returns the number of threads
   used, or -1 on bad arguments.  The decode step is this call with T = 1. */
int kdn_oracle_fwd(int variant, int B, int T, int H, int dk, int dv, double mu,
                   double tau, int per_channel_decay, const double *q,
                   const double *k, const double *v, const double *g,
                   const double *omega, const double *r, const double *S0,
                   const double *p0, const double *bhat_in, double *o,
                   double *ST, double *pT, double *kappa_out, double *phat_out,
                   double *p_out, int nthreads) {
  if (check(variant, B, T, H, dk, dv)) return -1;
  job_t J;
  memset(&J, 0, sizeof J);
  J.variant = variant; J.B = B; J.T = T; J.H = H; J.dk = dk; J.dv = dv;
  J.mu = mu; J.tau = tau; J.per_channel_decay = variant == 0 ? 1 : per_channel_decay;
  J.q = q; J.k = k; J.v = v; J.g = g; J.omega = omega; J.r = r; J.S0 = S0; J.p0 = p0;
  J.bhat_in = variant == 1 ? bhat_in : NULL;
  J.o = o; J.ST = ST; J.pT = pT;
  J.kappa_out = kappa_out; J.phat_out = phat_out; J.p_out = p_out;
  return run(&J, 0, nthreads);
}

/* Backward (adjoint of the forward token loop).  dST / dpT may be NULL (zero
   cotangent).  dS0 / dp0 may be NULL.  dmu (may be NULL) [B,H] receives dL/dmu of each
   sequence: mu enters only through u, so dmu = sum_t sum_i du_{t,i} u_{t,i} / mu. */
int kdn_oracle_bwd(int variant, int B, int T, int H, int dk, int dv, double mu,
                   double tau, int per_channel_decay, const double *q,
                   const double *k, const double *v, const double *g,
                   const double *omega, const double *r, const double *S0,
                   const double *p0, const double *bhat_in, const double *dO,
                   const double *dST, const double *dpT, double *dq, double *dk_,
                   double *dv_, double *dg, double *domega, double *dr,
                   double *dS0, double *dp0, double *dmu, int nthreads) {
  if (check(variant, B, T, H, dk, dv)) return -1;
  job_t J;
  memset(&J, 0, sizeof J);
  J.variant = variant; J.B = B; J.T = T; J.H = H; J.dk = dk; J.dv = dv;
  J.mu = mu; J.tau = tau; J.per_channel_decay = variant == 0 ? 1 : per_channel_decay;
  J.q = q; J.k = k; J.v = v; J.g = g; J.omega = omega; J.r = r; J.S0 = S0; J.p0 = p0;
  J.bhat_in = variant == 1 ? bhat_in : NULL;
  J.dO = dO; J.dST = dST; J.dpT = dpT;
  J.dq = dq; J.dk_ = dk_; J.dv_ = dv_; J.dg = dg; J.domega = domega; J.dr = dr;
  J.dS0 = dS0; J.dp0 = dp0; J.dmu = dmu;
  return run(&J, 1, nthreads);
}
