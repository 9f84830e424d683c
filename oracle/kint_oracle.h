/*
 * K-interval attention -- fp64 CPU oracle (TEST INFRASTRUCTURE ONLY).
 * Interface of oracle/kint_oracle.c.  Not used by, and not sharing anything
 * with, the CUDA library.
 *
 * Inputs are row-major [B, H, T, d] arrays (Q, K, V, dO); every output is
 * fp64 (or int32 / uint8 for decisions), row-major, caller-allocated.  Any
 * output pointer may be NULL.  Attention is causal: row i sees keys 0..i.
 */
#ifndef KINT_ORACLE_H
#define KINT_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element type of Q, K, V, dO.  The default build takes fp32 (the operator's
 * input type); building with -DKOR_F64_INPUT gives an otherwise identical
 * library taking fp64 inputs, used by the finite-difference checks. */
#ifdef KOR_F64_INPUT
typedef double kor_in;
#else
typedef float kor_in;
#endif

/* Calibrations: MinMax, FWM, the softmax comparator, and FWM's "resolved" tail policy
 * (App. "Tail policy in the MinMax -> FWM change"): FWM's step tau/K and origin -tau,
 * with the grid continued below -tau (negative indices) instead of a zero tail. */
/* KOR_EXP_FP8 is the FP8-rounded exponential baseline (App. "Reduced-precision
 * exponential baselines"): w = E4M3(e^{z}) forward, the fp32 exponential's derivative
 * backward (identity surrogate on the rounding), the row max on the gradient path;
 * K, tau, the reconstruction and the STE placement do not apply to it. */
/* KOR_EXP_BF16 is the BF16 exponential baseline of the same appendix: z = s - M rounded to
 * bfloat16, its exponential rounded to bfloat16 (w), P = w / sum w; the backward is the
 * chain rule through those casts in bfloat16 arithmetic: dL/dz_j = bf16(bf16(gamma_j) w_j),
 * the row max on the gradient path.  bfloat16 rounding is to nearest even; magnitudes
 * below 2^-126 flush to zero. */
enum { KOR_MINMAX = 0, KOR_FWM = 1, KOR_SOFTMAX = 2, KOR_FWM_RESOLVED = 3, KOR_EXP_FP8 = 4, KOR_EXP_BF16 = 5 };
enum { KOR_LERP = 0, KOR_NEAREST = 1 };
enum { KOR_WEIGHT = 0, KOR_PROB = 1 };
/* Backward modes: the full calibration gradient (Eq. full), detached extrema (App. B
 * "Detach (legacy)"), and the single-channel ablations that keep only the maximum's or
 * only the minimum's calibration term (App. "Single-channel ablation":
 * g_max_only = g_self + g_M, g_min_only = g_self + g_m), and the P1 control of App. B
 * "Detach (legacy)": the detached score gradient projected, per causal row, onto the
 * zero-sum subspace (g'_ij = g_ij - (1/(i+1)) sum_{k<=i} g_ik). */
enum { KOR_FULL = 0, KOR_DETACH = 1, KOR_MAX_ONLY = 2, KOR_MIN_ONLY = 3, KOR_DETACH_PROJ = 4 };

/* Codes of the per-key decision arrays (bins: Nearest index l in 0..K,
 * ivals: interval index r in 0..K-1).  Under the resolved policy the indices run
 * below zero and are stored as index + KOR_CODE_OFFSET, saturated to [0, 252]
 * (code 0 stands for every index <= -128; such keys carry weights below
 * e^{-tau - 128 tau/K}).  Under KOR_EXP_FP8 both arrays hold the E4M3 byte of
 * the rounded weight (0x00 = 0 .. 0x38 = 1).  Under KOR_EXP_BF16 bins holds the low
 * byte of the bfloat16 bits of the rounded z and ivals that of the rounded weight
 * (the low byte tells apart the two bfloat16 neighbours of a value). */
enum { KOR_CODE_NOGRID = 253, KOR_CODE_TAIL = 254, KOR_CODE_MASKED = 255, KOR_CODE_OFFSET = 128 };

typedef struct {
  int B, H, T, d;
  int Kint;   /* K, number of intervals */
  int calib;  /* KOR_MINMAX / KOR_FWM / KOR_SOFTMAX / KOR_FWM_RESOLVED / KOR_EXP_FP8 / KOR_EXP_BF16 */
  double tau; /* FWM window in nats (also the resolved grid's origin) */
  int recon;  /* KOR_LERP / KOR_NEAREST */
  int ste;    /* KOR_WEIGHT / KOR_PROB (ignored for LERP) */
  int grad;   /* KOR_FULL / KOR_DETACH / KOR_MAX_ONLY / KOR_MIN_ONLY / KOR_DETACH_PROJ */
  int nthreads; /* <= 0: all online cores */
} kor_params;

typedef struct {
  double* O;          /* [B,H,T,d] forward output */
  double* M;          /* [B,H,T] row max */
  double* m;          /* [B,H,T] row min */
  int32_t* amax;      /* [B,H,T] lowest arg-max */
  int32_t* amin;      /* [B,H,T] lowest arg-min */
  int32_t* nmax;      /* [B,H,T] size of the arg-max tie set */
  int32_t* nmin;      /* [B,H,T] size of the arg-min tie set */
  double* W;          /* [B,H,T] W^N (Nearest) or W^L (LERP); softmax: sum e^z */
  double* WL;         /* [B,H,T] W^L */
  double* OL;         /* [B,H,T,d] P^L V */
  uint8_t* bins;      /* [B,H,T,T] Nearest index l / codes */
  uint8_t* ivals;     /* [B,H,T,T] interval index r / codes */
  double* margin;     /* [B,H,T,T] distance (score units) to the nearest decision boundary */
  double* row_margin; /* [B,H,T] gap between an extremum and its runner-up */
  double* probe;      /* [7][B,H,T] geometry probe of each row (MinMax / FWM only), in order:
                         span M - m; native width h; softmax entropy H(P^E); fraction of keys
                         with z < -6; top-bucket mass; effective buckets exp H(q); TV(P, P^E) */
} kor_fwd_out;

enum { KOR_PROBES = 7 };

typedef struct {
  double* dQ;   /* [B,H,T,d] */
  double* dK;   /* [B,H,T,d] */
  double* dV;   /* [B,H,T,d] */
  double* cM;   /* [B,H,T] sum_j gamma_j dw_j/dM (0 under detach; computed in every other mode) */
  double* cm;   /* [B,H,T] sum_j gamma_j dw_j/dm (MinMax; 0 under detach) */
  double* dsum; /* [B,H,T] sum_j dL/ds_ij */
  double* dabs; /* [B,H,T] sum_j |dL/ds_ij| */
  double* dS;   /* [B,H,T,T] dL/ds (optional, small cases) */
} kor_bwd_out;

/* Decision-aligned re-run: where given, the oracle takes these decisions
 * instead of its own (used only for keys whose own decision lies within the
 * rounding guard band of a boundary). */
typedef struct {
  const uint8_t* bins;  /* [B,H,T,T] */
  const uint8_t* ivals; /* [B,H,T,T] */
  const int32_t* amax;  /* [B,H,T] */
  const int32_t* amin;  /* [B,H,T] */
} kor_override;

int kor_forward(const kor_params* p, const kor_in* Q, const kor_in* K, const kor_in* V, const kor_fwd_out* out,
                const kor_override* ov);
int kor_backward(const kor_params* p, const kor_in* Q, const kor_in* K, const kor_in* V, const kor_in* dO,
                 const kor_bwd_out* out, const kor_override* ov);
int kor_hardware_threads(void);

#ifdef __cplusplus
}
#endif
#endif
