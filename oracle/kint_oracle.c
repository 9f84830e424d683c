/*
 * K-interval attention -- plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the package smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no code with
 * the CUDA path and is written for a reader who checks it against the paper
 * ("Pretraining Transformers with Quantized Softmax in Attention"):
 *
 *   Sec. 3 "Objects and calibration" and App. A  -> scores, MinMax / FWM grids,
 *                                                  interval index r, position t
 *   Sec. 3 "Reconstruction" and App. A LERP/Nearest -> w^L, w^N, bin index l
 *   App. A "Normalization"                        -> P = w / sum w, O = P V
 *   App. B "Normalization Jacobian"               -> gamma = (g - <g>_P) / W
 *   App. B "LERP own-score slope"                 -> Delta (secant)
 *   Eq. (calgrad), Eq. (full), App. B "Full calibration gradient (MinMax)"
 *   App. B "FWM" paragraph                        -> FWM calibration gradient
 *   App. "Tail policy in the MinMax -> FWM change" -> the resolved grid (FWM's
 *                                                  step and origin, continued
 *                                                  below -tau, no zero tail)
 *   Eq. (wste) / Eq. (pste), App. B Weight-STE / Prob-STE paragraphs
 *   App. B "Detach (legacy)"                      -> detached extrema, and its P1
 *                                                  control (zero-sum projection)
 *   supplement "Single-channel ablation" and "Local gradient decomposition"
 *                                                 -> max_only / min_only modes
 *                                                  (g_self + g_M, g_self + g_m)
 *   App. B "Softmax", App. A "Softmax"            -> the comparator
 *   App. "Reduced-precision exponential baselines" -> FP8-rounded exponential
 *                                                  (E4M3 forward, fp32-exp backward)
 *                                                  and BF16 exponential (bf16 casts
 *                                                  and bf16 chain rule)
 *   App. "Geometry probe"                         -> per-row probes: span, width,
 *                                                  softmax entropy, mass below -6,
 *                                                  top-bucket mass, effective buckets,
 *                                                  total variation to softmax
 *   Table "Edge cases" (App. A)                   -> degenerate rows, ties,
 *                                                  midpoint rounding, window edge
 *
 * Everything is computed per causal row in fp64 from the fp32 inputs (fp64
 * inputs in the -DKOR_F64_INPUT build), with
 * plain loops and no blocking.  Rows are independent; heads (b, h) are spread
 * over POSIX threads, one head per thread at a time.
 *
 * Readings of points the paper leaves open (each is listed with its reason in
 * the design notes of the repository):
 *   - the score scale 1/sqrt(d) is applied once, inside the operator;
 *   - tau is a parameter (the paper trains only tau = 6);
 *   - ties among extrema split the extremum gradient evenly over the tie set;
 *   - the Nearest midpoint t = 1/2 rounds up; the FWM cutoff is strict (z < -tau);
 *   - the degenerate MinMax branch is M - m <= 1e-12 (fp64 here);
 *   - the forward of Nearest returns P^N = w^N / W^N directly (strict hard forward).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#include "kint_oracle.h"

#define DEGENERATE_EPS 1e-12

typedef struct {
  const kor_params* p;
  const kor_in *Q, *K, *V, *dO;
  const kor_fwd_out* fo;
  const kor_bwd_out* bo;
  const kor_override* ov;
  int do_bwd;
  int next_bh;
  pthread_mutex_t lock;
} job_t;

/* Per-thread row workspace, sized T. */
typedef struct {
  double *s, *z, *t, *wL, *wN, *P, *Pst, *g, *dS;
  double *er0, *er1; /* per key: the grid values e^{b_r}, e^{b_{r+1}} of its interval */
  int *r, *l, *tail, *code_l, *code_r;
  double* e; /* K+1 grid values e^{b_r} */
  double* margin;
  /* scalars of the current row */
  double M, m, h, b0, W_N, W_L, Wst;
  int amax, amin, nmax, nmin, degenerate, n;
} row_t;

static double dot_in(const kor_in* a, const kor_in* b, int d) {
  double acc = 0.0;
  for (int k = 0; k < d; ++k) acc += (double)a[k] * (double)b[k];
  return acc;
}

static double clampd(double x, double lo, double hi) { return x < lo ? lo : (x > hi ? hi : x); }

/* Distance from u to the nearest point of {n + 1/2 : n = 0..K-1} (Nearest bin
 * edges) and of {1..K-1} (LERP interval switches). */
static double decision_distance_u(double u, int K) {
  double best = INFINITY;
  for (int n = 0; n < K; ++n) {
    double dh = fabs(u - (n + 0.5));
    if (dh < best) best = dh;
    if (n >= 1) {
      double di = fabs(u - n);
      if (di < best) best = di;
    }
  }
  return best;
}

/* The same for the resolved grid, whose switches continue below u = 0: every
 * n / 2 with n <= 2K - 1 (bin edges n + 1/2, interval switches n <= K - 1). */
static double decision_distance_resolved(double u, int K) {
  if (u >= K - 0.5) return u - (K - 0.5);
  return fabs(u - floor(2.0 * u + 0.5) / 2.0);
}

/* Stored decision code of an index under the resolved policy. */
static int resolved_code(int idx) {
  const int c = idx + KOR_CODE_OFFSET;
  return c < 0 ? 0 : (c > 252 ? 252 : c);
}

/* OCP E4M3 ("fn": bias 7, 3 mantissa bits, no infinities).  Codes 0..0x3F in
 * increasing order cover [0, 1.875]: code = (exponent field << 3) | mantissa,
 * subnormals (exponent field 0) m * 2^-9, normals (1 + m/8) 2^(e - 7). */
static double e4m3_value(int code) {
  const int e = code >> 3, m = code & 7;
  return e == 0 ? ldexp((double)m, -9) : ldexp(1.0 + m / 8.0, e - 7);
}

/* Round 0 <= w <= 1 to the nearest E4M3 value, ties to the even code (even
 * mantissa), by scanning every code.  Returns the code; *mg receives the
 * distance, in z = ln w units, from w to the nearer edge of its rounding cell. */
static int e4m3_round(double w, double* mg) {
  int best = 0;
  for (int c = 1; c <= 0x3F; ++c) {
    const double dc = fabs(w - e4m3_value(c)), db = fabs(w - e4m3_value(best));
    if (dc < db || (dc == db && (c & 1) == 0)) best = c;
  }
  const double lo = best > 0 ? 0.5 * (e4m3_value(best - 1) + e4m3_value(best)) : 0.0;
  const double hi = 0.5 * (e4m3_value(best) + e4m3_value(best + 1));
  const double lz = log(w);
  const double dlo = lo > 0.0 ? lz - log(lo) : INFINITY, dhi = log(hi) - lz;
  *mg = dlo < dhi ? dlo : dhi;
  return best;
}

/* bfloat16: 8 significant bits, fp32's exponent range.  Round to nearest, ties to
 * even (x = f 2^e with f in [1/2, 1): the significand is f 2^8 in [128, 256)), and
 * flush magnitudes below 2^-126 to zero. */
static double bf16_rne(double x) {
  if (fabs(x) < ldexp(1.0, -126)) return 0.0;
  int e;
  const double f = frexp(x, &e);
  double r = f * 256.0;
  const double fl = floor(r), fr = r - fl;
  r = (fr > 0.5 || (fr == 0.5 && fmod(fl, 2.0) != 0.0)) ? fl + 1.0 : fl;
  return ldexp(r, e - 8);
}

/* Low byte of the bfloat16 bit pattern of a bfloat16 value v (0 for zero):
 * bits = sign | (E + 127) << 7 | m for v = +-(1 + m/128) 2^E. */
static int bf16_low_byte(double v) {
  if (v == 0.0) return 0;
  int e;
  const double f = frexp(fabs(v), &e); /* |v| = f 2^e, f in [1/2, 1) */
  const int E = e - 1, m = (int)(f * 256.0) - 128;
  return (((E + 127) & 1) << 7) | m;
}

/* The bfloat16 neighbour of x (the rounded value or the next one either way)
 * whose low byte is c; the rounded value itself when none matches. */
static double bf16_with_low_byte(double x, int c) {
  const double r = bf16_rne(x);
  if (r == 0.0 || bf16_low_byte(r) == c) return r;
  int e;
  frexp(fabs(r), &e);
  const double ulp = ldexp(1.0, e - 8);
  const double cand[2] = {r - ulp, r + ulp};
  for (int k = 0; k < 2; ++k)
    if (bf16_low_byte(bf16_rne(cand[k])) == c) return bf16_rne(cand[k]);
  return r;
}

/* Distance from x to the nearest bfloat16 rounding midpoint (x != 0). */
static double bf16_margin(double x) {
  int e;
  frexp(fabs(x), &e);
  const double half = ldexp(1.0, e - 9); /* half an ulp of x's binade */
  const double r = bf16_rne(x);
  return fabs(half - fabs(x - r));
}

/*
 * Forward quantities of causal row i of head bh (App. A).  Fills R.
 */
static void row_forward(const job_t* J, int bh, int i, row_t* R) {
  const kor_params* p = J->p;
  const int T = p->T, d = p->d, K = p->Kint;
  const kor_in* Qi = J->Q + ((size_t)bh * T + i) * d;
  const kor_in* Kh = J->K + (size_t)bh * T * d;
  const double scale = 1.0 / sqrt((double)d);
  const int n = i + 1; /* causal: keys 0..i are valid, later keys get w = 0 */
  R->n = n;

  /* Scores S = Q K^T / sqrt(d_h)  (Sec. 3, App. A) */
  for (int j = 0; j < n; ++j) R->s[j] = dot_in(Qi, Kh + (size_t)j * d, d) * scale;

  /* Row extrema; lowest index among ties, and the size of the tie set. */
  int amax = 0, amin = 0;
  for (int j = 1; j < n; ++j) {
    if (R->s[j] > R->s[amax]) amax = j;
    if (R->s[j] < R->s[amin]) amin = j;
  }
  if (J->ov && J->ov->amax) amax = J->ov->amax[(size_t)bh * T + i];
  if (J->ov && J->ov->amin) amin = J->ov->amin[(size_t)bh * T + i];
  R->M = R->s[amax];
  R->m = R->s[amin];
  R->amax = amax;
  R->amin = amin;
  R->nmax = 0;
  R->nmin = 0;
  for (int j = 0; j < n; ++j) {
    if (R->s[j] == R->M) R->nmax++;
    if (R->s[j] == R->m) R->nmin++;
  }

  R->degenerate = 0;
  R->h = 0.0;
  R->b0 = 0.0;
  for (int j = 0; j < n; ++j) {
    R->z[j] = R->s[j] - R->M;
    R->tail[j] = 0;
    R->r[j] = 0;
    R->l[j] = 0;
    R->t[j] = 0.0;
    R->margin[j] = INFINITY;
    R->code_l[j] = KOR_CODE_NOGRID;
    R->code_r[j] = KOR_CODE_NOGRID;
    R->er0[j] = 0.0;
    R->er1[j] = 0.0;
  }

  if (p->calib == KOR_SOFTMAX) {
    /* w^E_j = e^{z_j} (App. A, Softmax) */
    for (int j = 0; j < n; ++j) {
      R->wL[j] = exp(R->z[j]);
      R->wN[j] = R->wL[j];
    }
  } else if (p->calib == KOR_EXP_FP8) {
    /* w^exp_j = e^{z_j}, rounded to E4M3 and returned to full precision: the
     * forward weight (App. "Reduced-precision exponential baselines").  The
     * exponential itself is kept for the backward. */
    for (int j = 0; j < n; ++j) {
      const double we = exp(R->z[j]);
      double mg;
      int code = e4m3_round(we, &mg);
      if (J->ov && J->ov->bins) code = J->ov->bins[((size_t)bh * T + i) * T + j]; /* decision-aligned re-run */
      R->er0[j] = we;
      R->wL[j] = R->wN[j] = e4m3_value(code);
      R->code_l[j] = R->code_r[j] = code;
      R->margin[j] = mg;
    }
  } else if (p->calib == KOR_EXP_BF16) {
    /* z rounded to bfloat16, its exponential rounded to bfloat16: the forward weight
     * (App. "Reduced-precision exponential baselines").  Both roundings are decisions:
     * their codes are the low bytes, their margin the distance (in z) to a midpoint. */
    /* The row max key has z = 0 exactly; its code moves only if another key takes over as
     * the row max, i.e. by the gap between the maximum and the runner-up score. */
    double top_gap = INFINITY;
    for (int j = 0; j < n; ++j)
      if (R->s[j] != R->M && R->M - R->s[j] < top_gap) top_gap = R->M - R->s[j];
    for (int j = 0; j < n; ++j) {
      const size_t idx = ((size_t)bh * T + i) * T + j;
      const int ov = J->ov && J->ov->bins;
      const double zb = ov ? bf16_with_low_byte(R->z[j], J->ov->bins[idx]) : bf16_rne(R->z[j]);
      const double ez = exp(zb);
      const double w = (ov && J->ov->ivals) ? bf16_with_low_byte(ez, J->ov->ivals[idx]) : bf16_rne(ez);
      R->er0[j] = w;
      R->wL[j] = R->wN[j] = w;
      R->code_l[j] = bf16_low_byte(zb);
      R->code_r[j] = bf16_low_byte(w);
      /* z = 0 (the row max) is a boundary in its own way: every z of either sign near 0 has
       * its own bfloat16 code, so the row max key's code moves when a runner-up within
       * rounding takes over as the maximum: its margin is the top-two gap */
      double mg = top_gap;
      if (R->z[j] != 0.0) mg = bf16_margin(R->z[j]);
      if (ez > 0.0 && ez != 1.0) {
        const double me = bf16_margin(ez) / ez; /* relative: in z units */
        if (me < mg) mg = me;
      }
      R->margin[j] = mg;
    }
  } else if (p->calib == KOR_MINMAX && (R->M - R->m) <= DEGENERATE_EPS) {
    /* Degenerate MinMax row: weights 1, P uniform (Table "Edge cases"). */
    R->degenerate = 1;
    for (int j = 0; j < n; ++j) {
      R->wL[j] = 1.0;
      R->wN[j] = 1.0;
    }
  } else {
    /* Grid.  MinMax: z_min = m - M, h = (M - m)/K, b_r = z_min + r h.
     *        FWM:    h = tau/K, b_r = -tau + r h  (resolved: the same
     *                grid for every integer r <= K, no tail).           */
    const int resolved = (p->calib == KOR_FWM_RESOLVED);
    if (p->calib == KOR_MINMAX) {
      R->b0 = R->m - R->M;
      R->h = (R->M - R->m) / K;
    } else {
      R->b0 = -p->tau;
      R->h = p->tau / K;
    }
    const double h = R->h, b0 = R->b0;
    for (int rr = 0; rr <= K; ++rr) R->e[rr] = exp(b0 + rr * h);

    for (int j = 0; j < n; ++j) {
      const double z = R->z[j];
      int tail = 0;
      double zc = z;
      if (p->calib == KOR_FWM) {
        tail = (z < -p->tau);        /* zero tail below the window, strict */
        zc = clampd(z, -p->tau, 0.0); /* z~ = clip(z, -tau, 0) */
      }
      /* r = clip(floor((z - b_0)/h), 0, K-1), t = clip((z - b_r)/h, 0, 1);
       * resolved: r = min(floor(u), K-1), unbounded below */
      const double u = (zc - b0) / h;
      int r = (int)floor(u);
      if (r < 0 && !resolved) r = 0;
      if (r > K - 1) r = K - 1;
      double t = clampd((zc - (b0 + r * h)) / h, 0.0, 1.0);
      /* Nearest grid centre: l = r + [t >= 1/2] (midpoint rounds up) */
      int l = r + (t >= 0.5 ? 1 : 0);

      /* Distance to the nearest decision boundary, in score units. */
      double mg = INFINITY;
      if (p->calib == KOR_FWM) mg = fabs(z + p->tau);
      if (!tail) {
        double du = (resolved ? decision_distance_resolved(u, K) : decision_distance_u(u, K)) * h;
        if (du < mg) mg = du;
      }
      R->margin[j] = mg;

      if (J->ov && J->ov->bins) {
        /* Decision-aligned re-run: take the given bin / interval / tail choice
         * (resolved: a saturated code 0 keeps this row's own choice). */
        const size_t idx = ((size_t)bh * T + i) * T + j;
        const int cb = J->ov->bins[idx];
        tail = !resolved && (cb == KOR_CODE_TAIL);
        if (resolved) {
          if (cb != 0) {
            l = cb - KOR_CODE_OFFSET;
            if (J->ov->ivals) r = J->ov->ivals[idx] - KOR_CODE_OFFSET;
            t = clampd((zc - (b0 + r * h)) / h, 0.0, 1.0);
          }
        } else if (!tail) {
          l = cb;
          if (J->ov->ivals) r = J->ov->ivals[idx];
          t = clampd((zc - (b0 + r * h)) / h, 0.0, 1.0);
        }
      }
      R->tail[j] = tail;
      R->r[j] = r;
      R->t[j] = t;
      R->l[j] = l;
      if (tail) {
        R->wL[j] = 0.0;
        R->wN[j] = 0.0;
        R->code_l[j] = KOR_CODE_TAIL;
        R->code_r[j] = KOR_CODE_TAIL;
      } else {
        /* grid values e^{b_r}: the table, or for the resolved grid below the
         * window the same expression at the negative index */
        R->er0[j] = r >= 0 ? R->e[r] : exp(b0 + r * h);
        R->er1[j] = r + 1 >= 0 ? R->e[r + 1] : exp(b0 + (r + 1) * h);
        const double eN = l >= 0 ? R->e[l] : exp(b0 + l * h);
        R->wL[j] = (1.0 - t) * R->er0[j] + t * R->er1[j]; /* LERP */
        R->wN[j] = eN;                                   /* Nearest */
        R->code_l[j] = resolved ? resolved_code(l) : l;
        R->code_r[j] = resolved ? resolved_code(r) : r;
      }
    }
  }

  /* Normalization: W = sum_l w_l, P = w / W (App. A). */
  double WN = 0.0, WL = 0.0;
  for (int j = 0; j < n; ++j) {
    WN += R->wN[j];
    WL += R->wL[j];
  }
  R->W_N = WN;
  R->W_L = WL;
  const int hard = (p->calib != KOR_SOFTMAX && p->recon == KOR_NEAREST);
  for (int j = 0; j < n; ++j) R->P[j] = hard ? R->wN[j] / WN : R->wL[j] / WL;
}

static void fwd_row_outputs(const job_t* J, int bh, int i, row_t* R) {
  const kor_params* p = J->p;
  const kor_fwd_out* fo = J->fo;
  const int T = p->T, d = p->d, n = R->n, K = p->Kint;
  const size_t row = (size_t)bh * T + i;
  const kor_in* Vh = J->V + (size_t)bh * T * d;
  const int hard = (p->calib != KOR_SOFTMAX && p->recon == KOR_NEAREST);
  if (fo->O) {
    double* O = fo->O + row * d;
    for (int k = 0; k < d; ++k) O[k] = 0.0;
    for (int j = 0; j < n; ++j)
      for (int k = 0; k < d; ++k) O[k] += R->P[j] * (double)Vh[(size_t)j * d + k];
  }
  if (fo->OL) {
    double* OL = fo->OL + row * d;
    for (int k = 0; k < d; ++k) OL[k] = 0.0;
    for (int j = 0; j < n; ++j)
      for (int k = 0; k < d; ++k) OL[k] += (R->wL[j] / R->W_L) * (double)Vh[(size_t)j * d + k];
  }
  if (fo->M) fo->M[row] = R->M;
  if (fo->m) fo->m[row] = R->m;
  if (fo->amax) fo->amax[row] = R->amax;
  if (fo->amin) fo->amin[row] = R->amin;
  if (fo->nmax) fo->nmax[row] = R->nmax;
  if (fo->nmin) fo->nmin[row] = R->nmin;
  if (fo->W) fo->W[row] = hard ? R->W_N : R->W_L;
  if (fo->WL) fo->WL[row] = R->W_L;
  if (fo->bins || fo->ivals || fo->margin) {
    for (int j = 0; j < T; ++j) {
      const size_t idx = row * T + j;
      const int valid = j < n;
      if (fo->bins) fo->bins[idx] = (uint8_t)(valid ? R->code_l[j] : KOR_CODE_MASKED);
      if (fo->ivals) fo->ivals[idx] = (uint8_t)(valid ? R->code_r[j] : KOR_CODE_MASKED);
      if (fo->margin) fo->margin[idx] = valid ? R->margin[j] : INFINITY;
    }
  }
  if (fo->probe) {
    /* Geometry probe (App. "Geometry probe"), on the operator's own fp64 scores:
     * P^E = softmax(s); buckets are the operator's levels (Nearest: l in 0..K;
     * LERP: interval r in 0..K-1), with FWM's tail keys as one more bucket and a
     * degenerate MinMax row as a single bucket; the top bucket is l = K (Nearest)
     * or r = K-1 (LERP). */
    const size_t plane = (size_t)p->B * p->H * T;
    double Z = 0.0;
    for (int j = 0; j < n; ++j) Z += exp(R->z[j]);
    double H = 0.0, below = 0.0, top = 0.0, tv = 0.0;
    double* mass = (double*)calloc((size_t)K + 3, sizeof(double));
    const int nearest = (p->recon == KOR_NEAREST);
    for (int j = 0; j < n; ++j) {
      const double pe = exp(R->z[j]) / Z;
      if (pe > 0.0) H -= pe * log(pe);
      if (R->z[j] < -6.0) below += 1.0;
      tv += fabs(R->P[j] - pe);
      int bkt, is_top;
      if (R->degenerate) {
        bkt = 0;
        is_top = 1;
      } else if (R->tail[j]) {
        bkt = K + 1;
        is_top = 0;
      } else {
        bkt = nearest ? R->l[j] : R->r[j];
        is_top = nearest ? (R->l[j] == K) : (R->r[j] == K - 1);
      }
      if (mass) mass[bkt] += pe;
      if (is_top) top += pe;
    }
    double Hq = 0.0;
    for (int b = 0; b <= K + 1 && mass; ++b)
      if (mass[b] > 0.0) Hq -= mass[b] * log(mass[b]);
    free(mass);
    const double vals[KOR_PROBES] = {R->degenerate ? 0.0 : R->M - R->m, R->degenerate ? 0.0 : R->h, H, below / n,
                                     top, exp(Hq), 0.5 * tv};
    for (int k = 0; k < KOR_PROBES; ++k) fo->probe[k * plane + row] = vals[k];
  }
  if (fo->row_margin) {
    /* Gap between the extremum and the runner-up (a different score value),
     * i.e. how far the arg-extremum decision is from flipping. */
    double gmax = INFINITY, gmin = INFINITY;
    for (int j = 0; j < n; ++j) {
      if (R->s[j] != R->M && R->M - R->s[j] < gmax) gmax = R->M - R->s[j];
      if (R->s[j] != R->m && R->s[j] - R->m < gmin) gmin = R->s[j] - R->m;
    }
    fo->row_margin[row] = gmax < gmin ? gmax : gmin;
  }
}

/*
 * Backward of causal row i (App. B).  Adds this row's contributions to
 * dK, dV (rows 0..i of the head) and writes dQ_i.
 */
static void bwd_row(const job_t* J, int bh, int i, row_t* R) {
  const kor_params* p = J->p;
  const kor_bwd_out* bo = J->bo;
  const int T = p->T, d = p->d, K = p->Kint, n = R->n;
  const size_t row = (size_t)bh * T + i;
  const kor_in* Qi = J->Q + row * d;
  const kor_in* dOi = J->dO + row * d;
  const kor_in* Kh = J->K + (size_t)bh * T * d;
  const kor_in* Vh = J->V + (size_t)bh * T * d;
  const double scale = 1.0 / sqrt((double)d);

  /* Upstream gradient at the probabilities: g_j = dO_i . V_j */
  for (int j = 0; j < n; ++j) R->g[j] = dot_in(dOi, Vh + (size_t)j * d, d);

  double cM = 0.0, cm = 0.0;
  if (p->calib == KOR_SOFTMAX) {
    /* dL/ds_j = P_j (g_j - sum_i P_i g_i)  (App. B, Softmax) */
    double D = 0.0;
    for (int j = 0; j < n; ++j) D += R->P[j] * R->g[j];
    for (int j = 0; j < n; ++j) R->dS[j] = R->P[j] * (R->g[j] - D);
  } else if (p->calib == KOR_EXP_BF16) {
    /* The chain rule through the casts in bfloat16: the gradient reaching the bfloat16
     * weight is bf16(gamma_j), gamma_j = (g_j - <g>_P) / W; the exponential's backward
     * multiplies it by its bfloat16 output, rounded to bfloat16; the cast of z passes it
     * on.  The row max collects -sum_j dL/dz_j (split among ties). */
    double D = 0.0;
    for (int j = 0; j < n; ++j) D += R->P[j] * R->g[j];
    double own = 0.0;
    for (int j = 0; j < n; ++j) {
      R->dS[j] = bf16_rne(bf16_rne((R->g[j] - D) / R->W_N) * R->er0[j]);
      own += R->dS[j];
    }
    if (p->grad == KOR_DETACH_PROJ) {
      for (int j = 0; j < n; ++j) R->dS[j] -= own / n;
    } else if (p->grad != KOR_DETACH) {
      cM = -own;
      if (p->grad == KOR_FULL || p->grad == KOR_MAX_ONLY)
        for (int j = 0; j < n; ++j)
          if (R->s[j] == R->M) R->dS[j] += cM / R->nmax;
    }
  } else if (p->calib == KOR_EXP_FP8) {
    /* Normalization Jacobian at the rounded weights, gamma_j = (g_j - <g>_P) / W;
     * the rounding passes the gradient unchanged and dw_j/dz_j = e^{z_j}.  With
     * z = s - M the row max collects -sum_j dL/dz_j (split among ties); it has no
     * minimum channel. */
    double D = 0.0;
    for (int j = 0; j < n; ++j) D += R->P[j] * R->g[j];
    double own = 0.0;
    for (int j = 0; j < n; ++j) {
      R->dS[j] = (R->g[j] - D) / R->W_N * R->er0[j];
      own += R->dS[j];
    }
    if (p->grad == KOR_DETACH_PROJ) {
      for (int j = 0; j < n; ++j) R->dS[j] -= own / n;
    } else if (p->grad != KOR_DETACH) {
      cM = -own;
      if (p->grad == KOR_FULL || p->grad == KOR_MAX_ONLY)
        for (int j = 0; j < n; ++j)
          if (R->s[j] == R->M) R->dS[j] += cM / R->nmax;
    }
  } else if (R->degenerate) {
    /* Degenerate MinMax row: zero gradient (Table "Edge cases"). */
    for (int j = 0; j < n; ++j) R->dS[j] = 0.0;
  } else {
    /* Point of the normalization Jacobian:
     *   Nearest + Weight-STE: (P^N, W^N)   Eq. (wste)
     *   Nearest + Prob-STE:   (P^L, W^L)   Eq. (pste)
     *   LERP:                 (P^L, W^L)   exact Jacobian                 */
    const int at_hard = (p->recon == KOR_NEAREST && p->ste == KOR_WEIGHT);
    const double Wst = at_hard ? R->W_N : R->W_L;
    double D = 0.0;
    for (int j = 0; j < n; ++j) {
      R->Pst[j] = at_hard ? R->wN[j] / R->W_N : R->wL[j] / R->W_L;
      D += R->Pst[j] * R->g[j];
    }
    const double h = R->h;
    for (int j = 0; j < n; ++j) {
      if (R->tail[j]) {
        R->dS[j] = 0.0; /* mask and clamp: zero gradient */
        continue;
      }
      const int r = R->r[j];
      const double t = R->t[j];
      const double gamma = (R->g[j] - D) / Wst;           /* normalization Jacobian */
      const double Delta = (R->er1[j] - R->er0[j]) / h;   /* secant slope */
      R->dS[j] = gamma * Delta;                           /* own-score term */
      if (p->grad != KOR_DETACH && p->grad != KOR_DETACH_PROJ) {
        if (p->calib == KOR_MINMAX) {
          /* Eq. (calgrad) */
          const double rho = (r + t) / K;
          const double X = ((1.0 - t) * r * R->er0[j] + t * (r + 1) * R->er1[j]) / K;
          const double dwdM = -R->wL[j] - Delta * rho + X;
          const double dwdm = -Delta * (1.0 - rho) + R->wL[j] - X;
          cM += gamma * dwdM;
          cm += gamma * dwdm;
        } else {
          /* FWM: dw/dM = -Delta for in-window keys (resolved: every key), no m term. */
          cM += gamma * (-Delta);
        }
      }
    }
    if (p->grad == KOR_DETACH_PROJ) {
      /* P1 control (App. B, "Detach (legacy)"): keep the detached terms and subtract their
       * mean over the causal row, g'_ij = g_ij - (1/(i+1)) sum_{k<=i} g_ik, so that every
       * row sums to zero.  The mean is taken over all n = i + 1 causal keys, FWM tail keys
       * (detached term 0) included. */
      double mean = 0.0;
      for (int j = 0; j < n; ++j) mean += R->dS[j];
      mean /= n;
      for (int j = 0; j < n; ++j) R->dS[j] -= mean;
    } else if (p->grad != KOR_DETACH) {
      /* Eq. (full): the extremum terms go to the arg-max / arg-min keys, split
       * evenly among ties; the single-channel modes keep one of the two. */
      const int use_M = p->grad == KOR_FULL || p->grad == KOR_MAX_ONLY;
      const int use_m = p->grad == KOR_FULL || p->grad == KOR_MIN_ONLY;
      for (int j = 0; j < n; ++j) {
        if (use_M && R->s[j] == R->M) R->dS[j] += cM / R->nmax;
        if (use_m && p->calib == KOR_MINMAX && R->s[j] == R->m) R->dS[j] += cm / R->nmin;
      }
    }
  }

  /* dQ_i = sum_j dS_j K_j / sqrt(d); dK_j += dS_j Q_i / sqrt(d); dV_j += P_j dO_i */
  double* dQi = bo->dQ ? bo->dQ + row * d : NULL;
  if (dQi)
    for (int k = 0; k < d; ++k) dQi[k] = 0.0;
  double dsum = 0.0, dabs = 0.0;
  for (int j = 0; j < n; ++j) {
    const double ds = R->dS[j];
    dsum += ds;
    dabs += fabs(ds);
    const kor_in* Kj = Kh + (size_t)j * d;
    if (dQi)
      for (int k = 0; k < d; ++k) dQi[k] += ds * (double)Kj[k] * scale;
    if (bo->dK) {
      double* dKj = bo->dK + ((size_t)bh * T + j) * d;
      for (int k = 0; k < d; ++k) dKj[k] += ds * (double)Qi[k] * scale;
    }
    if (bo->dV) {
      double* dVj = bo->dV + ((size_t)bh * T + j) * d;
      for (int k = 0; k < d; ++k) dVj[k] += R->P[j] * (double)dOi[k];
    }
  }
  if (bo->dS) {
    double* out = bo->dS + row * T;
    for (int j = 0; j < T; ++j) out[j] = j < n ? R->dS[j] : 0.0;
  }
  if (bo->cM) bo->cM[row] = cM;
  if (bo->cm) bo->cm[row] = cm;
  if (bo->dsum) bo->dsum[row] = dsum;
  if (bo->dabs) bo->dabs[row] = dabs;
}

static int row_alloc(row_t* R, int T, int K) {
  memset(R, 0, sizeof(*R));
  double** dptrs[] = {&R->s, &R->z, &R->t, &R->wL, &R->wN, &R->P, &R->Pst, &R->g, &R->dS, &R->margin,
                      &R->er0, &R->er1};
  for (size_t k = 0; k < sizeof(dptrs) / sizeof(dptrs[0]); ++k) {
    *dptrs[k] = (double*)calloc((size_t)T, sizeof(double));
    if (!*dptrs[k]) return -1;
  }
  int** iptrs[] = {&R->r, &R->l, &R->tail, &R->code_l, &R->code_r};
  for (size_t k = 0; k < sizeof(iptrs) / sizeof(iptrs[0]); ++k) {
    *iptrs[k] = (int*)calloc((size_t)T, sizeof(int));
    if (!*iptrs[k]) return -1;
  }
  R->e = (double*)calloc((size_t)K + 2, sizeof(double));
  return R->e ? 0 : -1;
}

static void row_free(row_t* R) {
  double* dp[] = {R->s, R->z, R->t, R->wL, R->wN, R->P, R->Pst, R->g, R->dS, R->margin, R->e, R->er0, R->er1};
  for (size_t k = 0; k < sizeof(dp) / sizeof(dp[0]); ++k) free(dp[k]);
  int* ip[] = {R->r, R->l, R->tail, R->code_l, R->code_r};
  for (size_t k = 0; k < sizeof(ip) / sizeof(ip[0]); ++k) free(ip[k]);
}

static void* worker(void* arg) {
  job_t* J = (job_t*)arg;
  const kor_params* p = J->p;
  row_t R;
  if (row_alloc(&R, p->T, p->Kint) != 0) {
    row_free(&R);
    return (void*)1;
  }
  const int nbh = p->B * p->H;
  for (;;) {
    pthread_mutex_lock(&J->lock);
    const int bh = J->next_bh++;
    pthread_mutex_unlock(&J->lock);
    if (bh >= nbh) break;
    if (J->do_bwd) {
      const size_t base = (size_t)bh * p->T * p->d;
      if (J->bo->dK) memset(J->bo->dK + base, 0, sizeof(double) * p->T * p->d);
      if (J->bo->dV) memset(J->bo->dV + base, 0, sizeof(double) * p->T * p->d);
    }
    for (int i = 0; i < p->T; ++i) {
      row_forward(J, bh, i, &R);
      if (J->do_bwd)
        bwd_row(J, bh, i, &R);
      else
        fwd_row_outputs(J, bh, i, &R);
    }
  }
  row_free(&R);
  return NULL;
}

static int check_params(const kor_params* p) {
  if (!p || p->B < 1 || p->H < 1 || p->T < 1 || p->d < 1) return -1;
  if (p->calib < 0 || p->calib > 5) return -1;
  if (p->calib != KOR_SOFTMAX && p->calib != KOR_EXP_FP8 && p->calib != KOR_EXP_BF16 &&
      (p->Kint < 1 || p->Kint > (1 << 20)))
    return -1;
  if ((p->calib == KOR_FWM || p->calib == KOR_FWM_RESOLVED) && !(p->tau > 0.0)) return -1;
  if (p->recon < 0 || p->recon > 1 || p->ste < 0 || p->ste > 1 || p->grad < 0 || p->grad > 4) return -1;
  return 0;
}

static int run(const kor_params* p, const kor_in* Q, const kor_in* K, const kor_in* V, const kor_in* dO,
               const kor_fwd_out* fo, const kor_bwd_out* bo, const kor_override* ov) {
  if (check_params(p) != 0) return -1;
  /* the uint8 decision codes hold l in 0..K and need K + 1 < KOR_CODE_NOGRID */
  if (fo && (fo->bins || fo->ivals) && p->Kint >= KOR_CODE_NOGRID - 1) return -1;
  /* the probes are defined for the grid calibrations MinMax and FWM */
  if (fo && fo->probe && p->calib != KOR_MINMAX && p->calib != KOR_FWM) return -1;
  /* resolved: codes l + KOR_CODE_OFFSET <= 252 */
  if (p->calib == KOR_FWM_RESOLVED && ((fo && (fo->bins || fo->ivals)) || (ov && ov->bins)) &&
      p->Kint > 252 - KOR_CODE_OFFSET)
    return -1;
  job_t J;
  memset(&J, 0, sizeof(J));
  J.p = p;
  J.Q = Q;
  J.K = K;
  J.V = V;
  J.dO = dO;
  J.fo = fo;
  J.bo = bo;
  J.ov = ov;
  J.do_bwd = bo != NULL;
  pthread_mutex_init(&J.lock, NULL);
  int nt = p->nthreads > 0 ? p->nthreads : (int)sysconf(_SC_NPROCESSORS_ONLN);
  if (nt < 1) nt = 1;
  if (nt > p->B * p->H) nt = p->B * p->H;
  pthread_t* th = (pthread_t*)calloc((size_t)nt, sizeof(pthread_t));
  int rc = 0;
  for (int k = 0; k < nt; ++k) pthread_create(&th[k], NULL, worker, &J);
  for (int k = 0; k < nt; ++k) {
    void* ret = NULL;
    pthread_join(th[k], &ret);
    if (ret) rc = -2;
  }
  free(th);
  pthread_mutex_destroy(&J.lock);
  return rc;
}

int kor_forward(const kor_params* p, const kor_in* Q, const kor_in* K, const kor_in* V, const kor_fwd_out* out,
                const kor_override* ov) {
  if (!Q || !K || !V || !out) return -1;
  return run(p, Q, K, V, NULL, out, NULL, ov);
}

int kor_backward(const kor_params* p, const kor_in* Q, const kor_in* K, const kor_in* V, const kor_in* dO,
                 const kor_bwd_out* out, const kor_override* ov) {
  if (!Q || !K || !V || !dO || !out) return -1;
  return run(p, Q, K, V, dO, NULL, out, ov);
}

int kor_hardware_threads(void) { return (int)sysconf(_SC_NPROCESSORS_ONLN); }
