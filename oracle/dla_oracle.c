/*
 * dla_oracle.c -- plain fp64 CPU oracle of Dynamic Linear Attention (DLA,
 * arXiv 2606.10650).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark load this file's library.  The CUDA
 * library never links, includes or calls it, and it includes nothing of the
 * CUDA library.
 *
 * It is deliberately slow and literal: every memory state is an explicit
 * d_v x d_k matrix of doubles, the score is evaluated element by element
 * from its definition, merges really add the two matrices and shift the
 * list, and the read-out loops over every cached state.  There is no
 * blocking, no Gram identity and no reordering beyond what the paper states.
 *
 * Notation and passages followed (paper sections / equations / algorithms):
 *   token state          s_t = v_t k_t^T (d_v x d_k)          Sec. 2 (recurrent
 *                        linear attention, S_t = S_{t-1} + v_t k_t^T), phi = id
 *   state information    I_t = ||N(A) - N(B)||_F / (||N(B)||_F + eps)
 *     score_mode 0       A = s_t, B = S (last state)           Algorithm 1
 *     score_mode 1       A = S + s_t, B = S                     Eq. (importance_score)
 *     N = RMSNorm over the whole matrix, gain 1                Sec. 3.1 ("we apply
 *                        RMSNorm to both ... prior to score computation")
 *   boundary             b_t = 1[I_t >= tau]                    Sec. 3.1
 *   state update         b_t=0: S_cur += s_t ; b_t=1: new state  Sec. 3.1 update rule
 *   capacity bound       if |M| = C: merge adjacent pair of lowest density
 *                        (Ibar_i + Ibar_{i+1}) / (n_i + n_{i+1}), sum S, n, Ibar,
 *                        remove i*+1, shift, then append       Algorithm 2, Sec. 3.2
 *   read-out             o_t = sum_i lambda_{t,i} S_i q_t over the cache after
 *                        token t                                Eq. (capacity_bounded_output)
 *
 * Readings taken where the paper is silent or inconsistent:
 *   first token opens state 0 with I_0 = 0; the boundary token's score goes to
 *   the state it opens; the capacity counts the open state; the argmin takes
 *   the lowest index on exact ties; lambda NULL means all ones; the state a
 *   boundary token opens holds s_t only (Sec. 3.1 update rule, not the
 *   merge-then-append of Algorithm 1's pseudo-code).
 *
 * Build: gcc -O2 -fPIC -shared -ffp-contract=off (no FMA contraction, so that
 * x86 and Arm hosts round identically).
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int C, dk, dv, score_mode;
  double tau, eps, rms_eps;
  int m;                 /* live states (including the open one)            */
  double **S;            /* S[i]: logical state i, row-major [dv][dk]       */
  double *store;         /* C matrices backing S                            */
  long long *n;          /* tokens summarised by state i                    */
  double *ibar;          /* sum of the per-token scores of state i          */
  long long *first, *last; /* token range [first, last] of state i          */
  long long t;           /* tokens processed so far                         */
  double *s_tok;         /* scratch: current token state                    */
  double *s_tmp;         /* scratch: S + s for score_mode 1                 */
} orc_stream;

static long long dsize(const orc_stream *st) { return (long long)st->dk * st->dv; }

orc_stream *orc_new(int C, int dk, int dv, double tau, double eps,
                    double rms_eps, int score_mode) {
  if (C < 2 || dk < 1 || dv < 1) return NULL;
  orc_stream *st = (orc_stream *)calloc(1, sizeof(orc_stream));
  st->C = C; st->dk = dk; st->dv = dv; st->score_mode = score_mode;
  st->tau = tau; st->eps = eps; st->rms_eps = rms_eps;
  long long D = (long long)dk * dv;
  st->store = (double *)calloc((size_t)(C * D), sizeof(double));
  st->S = (double **)calloc((size_t)C, sizeof(double *));
  for (int i = 0; i < C; ++i) st->S[i] = st->store + (long long)i * D;
  st->n = (long long *)calloc((size_t)C, sizeof(long long));
  st->ibar = (double *)calloc((size_t)C, sizeof(double));
  st->first = (long long *)calloc((size_t)C, sizeof(long long));
  st->last = (long long *)calloc((size_t)C, sizeof(long long));
  st->s_tok = (double *)calloc((size_t)D, sizeof(double));
  st->s_tmp = (double *)calloc((size_t)D, sizeof(double));
  return st;
}

void orc_free(orc_stream *st) {
  if (!st) return;
  free(st->store); free(st->S); free(st->n); free(st->ibar);
  free(st->first); free(st->last); free(st->s_tok); free(st->s_tmp);
  free(st);
}

/* Deep copy of src into dst (same C, dk, dv).  The pointer array S is
 * rebuilt so that dst's logical order matches src's. */
int orc_copy(orc_stream *dst, const orc_stream *src) {
  if (dst->C != src->C || dst->dk != src->dk || dst->dv != src->dv) return -1;
  long long D = dsize(src);
  dst->score_mode = src->score_mode;
  dst->tau = src->tau; dst->eps = src->eps; dst->rms_eps = src->rms_eps;
  dst->m = src->m; dst->t = src->t;
  for (int i = 0; i < src->C; ++i) {
    dst->S[i] = dst->store + (long long)i * D;
    memcpy(dst->S[i], src->S[i], (size_t)D * sizeof(double));
    dst->n[i] = src->n[i]; dst->ibar[i] = src->ibar[i];
    dst->first[i] = src->first[i]; dst->last[i] = src->last[i];
  }
  return 0;
}

/* s = v k^T, row j, column kk. */
static void token_state(const orc_stream *st, const double *k, const double *v,
                        double *s) {
  for (int j = 0; j < st->dv; ++j)
    for (int kk = 0; kk < st->dk; ++kk) s[(long long)j * st->dk + kk] = v[j] * k[kk];
}

/* RMSNorm scale of a whole matrix: sqrt(mean(X o X) + rms_eps), gain 1. */
static double rms_of(const double *X, long long D, double rms_eps) {
  double ss = 0.0;
  for (long long e = 0; e < D; ++e) ss += X[e] * X[e];
  return sqrt(ss / (double)D + rms_eps);
}

/* I = ||N(A) - N(B)||_F / (||N(B)||_F + eps), evaluated element by element. */
static double info_score(const double *A, const double *B, long long D,
                         double eps, double rms_eps) {
  double ra = rms_of(A, D, rms_eps), rb = rms_of(B, D, rms_eps);
  double diff = 0.0, nb = 0.0;
  for (long long e = 0; e < D; ++e) {
    double na = A[e] / ra, nbv = B[e] / rb;
    diff += (na - nbv) * (na - nbv);
    nb += nbv * nbv;
  }
  return sqrt(diff) / (sqrt(nb) + eps);
}

/* Score of token state s against the last (open) state; requires m >= 1. */
static double score_token(orc_stream *st, const double *s) {
  long long D = dsize(st);
  const double *S = st->S[st->m - 1];
  if (st->score_mode == 1) {
    for (long long e = 0; e < D; ++e) st->s_tmp[e] = S[e] + s[e];
    return info_score(st->s_tmp, S, D, st->eps, st->rms_eps);
  }
  return info_score(s, S, D, st->eps, st->rms_eps);
}

static double pair_density(const orc_stream *st, int i) {
  return (st->ibar[i] + st->ibar[i + 1]) / (double)(st->n[i] + st->n[i + 1]);
}

/* argmin over adjacent pairs i = 0..m-2 of the pair density; strict '<' so
 * the lowest index wins an exact tie.  Also reports the runner-up. */
static int argmin_pair(const orc_stream *st, double *best_d, int *second,
                       double *second_d) {
  int best = -1, sec = -1;
  double bd = 0.0, sd = 0.0;
  for (int i = 0; i + 1 < st->m; ++i) {
    double d = pair_density(st, i);
    if (best < 0 || d < bd) {
      sec = best; sd = bd;
      best = i; bd = d;
    } else if (sec < 0 || d < sd) {
      sec = i; sd = d;
    }
  }
  if (best_d) *best_d = bd;
  if (second) *second = sec;
  if (second_d) *second_d = sd;
  return best;
}

/* Merge logical states j and j+1 into j, remove j+1 and shift the rest. */
static void merge_pair(orc_stream *st, int j) {
  long long D = dsize(st);
  double *Sj = st->S[j], *Sn = st->S[j + 1];
  for (long long e = 0; e < D; ++e) Sj[e] += Sn[e];
  st->n[j] += st->n[j + 1];
  st->ibar[j] += st->ibar[j + 1];
  st->last[j] = st->last[j + 1];
  for (int i = j + 1; i + 1 < st->m; ++i) {
    st->S[i] = st->S[i + 1];
    st->n[i] = st->n[i + 1]; st->ibar[i] = st->ibar[i + 1];
    st->first[i] = st->first[i + 1]; st->last[i] = st->last[i + 1];
  }
  st->m -= 1;
  st->S[st->m] = Sn; /* its buffer is free again */
}

static void append_state(orc_stream *st, const double *s, double I) {
  long long D = dsize(st);
  memcpy(st->S[st->m], s, (size_t)D * sizeof(double));
  st->n[st->m] = 1; st->ibar[st->m] = I;
  st->first[st->m] = st->t; st->last[st->m] = st->t;
  st->m += 1;
}

/*
 * Process one token (Algorithm 1 step + Algorithm 2 insertion).
 * Outputs: *I_out the score (0 for the first token), *b_out the boundary
 * indicator, *j_out the merged pair index i* (or -1).
 */
int orc_step(orc_stream *st, const double *k, const double *v, double *I_out,
             int *b_out, int *j_out) {
  double *s = st->s_tok;
  token_state(st, k, v, s);
  double I = 0.0;
  int b = 1, j = -1;
  if (st->m == 0) {
    append_state(st, s, 0.0);
  } else {
    I = score_token(st, s);
    b = (I >= st->tau) ? 1 : 0;
    if (b) {
      if (st->m == st->C) {
        j = argmin_pair(st, NULL, NULL, NULL);
        merge_pair(st, j);
      }
      append_state(st, s, I);
    } else {
      long long D = dsize(st);
      double *S = st->S[st->m - 1];
      for (long long e = 0; e < D; ++e) S[e] += s[e];
      st->n[st->m - 1] += 1;
      st->ibar[st->m - 1] += I;
      st->last[st->m - 1] = st->t;
    }
  }
  st->t += 1;
  if (I_out) *I_out = I;
  if (b_out) *b_out = b;
  if (j_out) *j_out = j;
  return 0;
}

/*
 * What orc_step would decide for (k, v), without changing the stream.
 * out[0] I, out[1] boundary, out[2] merge index (-1 none), out[3] best pair
 * density, out[4] runner-up density (or +inf), out[5] relative threshold
 * margin |I - tau| / tau (inf for the first token), out[6] relative gap
 * (runner-up - best) / |best| (inf when no merge happens), out[7] first token
 * of the newest state among the best and runner-up pairs (-1 when no merge),
 * out[8] the last token of that state (-1 when no merge).  out must hold 9.
 */
int orc_probe(orc_stream *st, const double *k, const double *v, double *out) {
  double *s = st->s_tok;
  token_state(st, k, v, s);
  for (int e = 0; e < 9; ++e) out[e] = 0.0;
  out[2] = -1.0; out[4] = INFINITY; out[5] = INFINITY; out[6] = INFINITY;
  out[7] = -1.0; out[8] = -1.0;
  if (st->m == 0) { out[1] = 1.0; return 0; }
  double I = score_token(st, s);
  int b = (I >= st->tau) ? 1 : 0;
  out[0] = I; out[1] = (double)b;
  out[5] = fabs(I - st->tau) / fabs(st->tau);
  if (b && st->m == st->C) {
    double bd, sd; int sec;
    int j = argmin_pair(st, &bd, &sec, &sd);
    out[2] = (double)j; out[3] = bd;
    if (sec >= 0) {
      out[4] = sd;
      double scale = fabs(bd) > 0.0 ? fabs(bd) : 1e-300;
      out[6] = (sd - bd) / scale;
      int newest = (j > sec ? j : sec) + 1;
      out[7] = (double)st->first[newest];
      out[8] = (double)st->last[newest];
    }
  }
  return 0;
}

/* o = sum_{i<m} lambda_i S_i q ; lam may be NULL (all ones). */
int orc_readout(const orc_stream *st, const double *q, const double *lam,
                double *o) {
  for (int j = 0; j < st->dv; ++j) o[j] = 0.0;
  for (int i = 0; i < st->m; ++i) {
    double w = lam ? lam[i] : 1.0;
    const double *S = st->S[i];
    for (int j = 0; j < st->dv; ++j) {
      double acc = 0.0;
      for (int kk = 0; kk < st->dk; ++kk) acc += S[(long long)j * st->dk + kk] * q[kk];
      o[j] += w * acc;
    }
  }
  return 0;
}

/*
 * Run T tokens through the stream.  Token t's vectors start at
 * q + t*row_stride (same for k, v); lambda row t at lam + t*lam_stride.
 * want_o (optional) selects the tokens whose output is computed; o row t
 * is written at o + t*o_stride.  boundary / merge_log / itrace (optional)
 * receive the per-token decisions and scores.
 */
int orc_forward(orc_stream *st, long long T, const double *q, const double *k,
                const double *v, long long row_stride, const double *lam,
                long long lam_stride, const unsigned char *want_o, double *o,
                long long o_stride, unsigned char *boundary, int *merge_log,
                double *itrace) {
  for (long long t = 0; t < T; ++t) {
    double I; int b, j;
    orc_step(st, k + t * row_stride, v + t * row_stride, &I, &b, &j);
    if (boundary) boundary[t] = (unsigned char)b;
    if (merge_log) merge_log[t] = j;
    if (itrace) itrace[t] = I;
    if (o && (!want_o || want_o[t]))
      orc_readout(st, q + t * row_stride, lam ? lam + t * lam_stride : NULL,
                  o + t * o_stride);
  }
  return 0;
}

/* Export the cache in logical order: states [m][dv][dk], n, ibar, first, last. */
int orc_export(const orc_stream *st, double *states, long long *n, double *ibar,
               long long *first, long long *last, int *m, long long *t) {
  long long D = dsize(st);
  for (int i = 0; i < st->m; ++i) {
    if (states) memcpy(states + (long long)i * D, st->S[i], (size_t)D * sizeof(double));
    if (n) n[i] = st->n[i];
    if (ibar) ibar[i] = st->ibar[i];
    if (first) first[i] = st->first[i];
    if (last) last[i] = st->last[i];
  }
  if (m) *m = st->m;
  if (t) *t = st->t;
  return 0;
}

int orc_get_m(const orc_stream *st) { return st->m; }
long long orc_get_t(const orc_stream *st) { return st->t; }
