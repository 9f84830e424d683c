/*
 * kint_attn.h -- C ABI of libkint, K-interval attention (forward and backward)
 * on one NVIDIA GB300 (sm_103a).
 *
 * K-interval attention replaces the softmax of causal attention (paper: Sec. 3,
 * App. A): scores S = Q K^T / sqrt(d) are calibrated per row (MinMax: the grid
 * spans the row's own [m, M]; FWM: a fixed window [M - tau, M] anchored at the
 * row maximum, zero weight below it), the exponential is rebuilt on K intervals
 * from K + 1 grid values e^{b_r} (LERP interpolation or Nearest rounding), the
 * weights are normalised, P = w / sum w, and O = P V.  The backward is the
 * closed form of App. B: normalization Jacobian, LERP secant slope, and the
 * calibration derivatives through the row extrema (Eqs. calgrad and full),
 * placed by Weight-STE (Eq. wste) or Prob-STE (Eq. pste); the detached-extrema
 * mode keeps only the own-score term.
 *
 * Conventions shared by every entry point
 *   - Tensors are fp32, row-major, contiguous [B, H, T, d]; row statistics are
 *     [B, H, T].  All tensor pointers are DEVICE pointers owned by the caller;
 *     the library never allocates, frees or synchronises (except
 *     kint_get_status, which synchronises the given stream).  Work is enqueued
 *     on `stream` (a cudaStream_t; 0 = legacy default stream).
 *   - Attention is causal (row i sees keys 0..i, App. A); causal must be 1.
 *   - d must be 64 or 128; T >= 1 is arbitrary (ragged final tiles are masked);
 *     B * H * ceil(T / 128) <= 2^31 - 1.
 *   - Every device pointer must be 16-byte aligned.
 *   - The score scale 1/sqrt(d) is applied inside the operator.
 *   - Errors are returned as negative codes BEFORE any work is enqueued; no
 *     output is touched then.  Faults detected on the device (a bounded wait
 *     that ran out) are reported by kint_get_status().
 *   - Calls on different streams that share a workspace race.
 */
#ifndef KINT_ATTN_H
#define KINT_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes. */
#define KINT_OK 0
#define KINT_ERR_ARG (-1)          /* null pointer, size < 1, K out of [1, 64], tau <= 0, bad enum, causal != 1 */
#define KINT_ERR_UNSUPPORTED (-2)  /* d not in {64, 128}; 3xTF32 with d != 64; MinMax with K > 32 unless
                                      TF32 at d = 64; sizes beyond the limits above */
#define KINT_ERR_ALIGN (-3)        /* a device pointer is not 16-byte aligned */
#define KINT_ERR_WORKSPACE (-4)    /* workspace NULL or smaller than kint_attn_workspace_bytes() */
#define KINT_ERR_LAUNCH (-5)       /* the CUDA runtime refused a launch or a tensor-map encoding */
#define KINT_ERR_DEVICE (-6)       /* kint_get_status: a kernel flagged a device-side fault */
#define KINT_ERR_NO_DEVICE (-7)    /* no sm_103 device current, or the driver lacks tensor maps */
#define KINT_ERR_SCRATCH_LIMIT (-8) /* kint_attn_fwd_noalloc: problem needs more than KINT_NOALLOC_SCRATCH_BYTES */

/* Calibration (Sec. 3 "Objects and calibration"; App. A "MinMax grid", "FWM";
 * App. A "Softmax" is the exact-exponential comparator).  FWM_RESOLVED is the
 * "resolved" tail policy of App. "Tail policy in the MinMax -> FWM change": FWM's
 * step tau/K and origin -tau, with the grid continued below -tau (negative indices)
 * instead of a zero tail; its grid values below the window come from the exponential
 * unit (ex2.approx), in-window values from the same table as FWM. */
typedef enum {
  KINT_CALIB_MINMAX = 0,
  KINT_CALIB_FWM = 1,
  KINT_CALIB_SOFTMAX = 2,
  KINT_CALIB_FWM_RESOLVED = 3,
  KINT_CALIB_EXP_FP8 = 4,
  KINT_CALIB_EXP_BF16 = 5
} kint_calib;
/* KINT_CALIB_EXP_BF16 is the BF16 exponential baseline of the same appendix: z = s - M
 * rounded to bfloat16, w = e^z rounded to bfloat16 (round to nearest even; the exponential
 * is ex2.approx, flushing below 2^-126), P = w / sum w; the backward is the chain rule
 * through the casts in bfloat16 arithmetic, dL/dz_j = bf16(bf16(gamma_j) w_j), with the
 * row max on the gradient path as for EXP_FP8.  Kint, tau, recon, ste: as for EXP_FP8. */
/* KINT_CALIB_EXP_FP8 is the FP8-rounded exponential baseline of App. "Reduced-precision
 * exponential baselines": w = E4M3(e^{s - M}) (round to nearest even) in the forward, the
 * exponential's own derivative e^{s - M} in the backward (identity surrogate on the
 * rounding, normalization Jacobian at the rounded weights), the row max M on the gradient
 * path as the maximum channel (full / max_only keep it; detach, min_only drop it).  Kint,
 * tau, recon and ste are not used (they must still be valid values); the exponential is
 * ex2.approx, as for the softmax comparator. */
/* Reconstruction (Sec. 3 "Reconstruction"; App. A "LERP", "Nearest"). */
typedef enum { KINT_RECON_LERP = 0, KINT_RECON_NEAREST = 1 } kint_recon;
/* Surrogate placement (Sec. 3 Eqs. wste / pste).  Ignored under LERP, where the
 * two placements coincide (w^N = w^L). */
typedef enum { KINT_STE_WEIGHT = 0, KINT_STE_PROB = 1 } kint_ste;
/* Backward mode: full calibration gradient (Eq. full), detached extrema
 * (App. B "Detach (legacy)"), or one extremum channel only (supplement
 * "Single-channel ablation": max_only keeps the c_M term, min_only the c_m term;
 * for FWM, which has no minimum channel, max_only equals full and min_only
 * equals detach), or the P1 control of App. B "Detach (legacy)": the detached score
 * gradient projected onto the zero-sum subspace of each causal row,
 * dS'_ij = dS_ij - (1/(i+1)) sum_{k<=i} dS_ik (tail keys included).  The forward does not
 * depend on it; softmax ignores it. */
typedef enum {
  KINT_GRAD_FULL = 0,
  KINT_GRAD_DETACH = 1,
  KINT_GRAD_MAX_ONLY = 2,
  KINT_GRAD_MIN_ONLY = 3,
  KINT_GRAD_DETACH_PROJ = 4
} kint_grad;
/* Tensor-core arithmetic: plain TF32 products (the precision the paper trains
 * with, App. C "Numerics and hardware"), or 3xTF32 (hi/lo operand splitting,
 * fp32-level accuracy). */
typedef enum { KINT_PREC_TF32 = 0, KINT_PREC_3XTF32 = 1 } kint_prec;

/* Row statistics written by kint_attn_fwd and read by kint_attn_bwd.  All
 * arrays are caller-owned device memory of B*H*T elements unless noted. */
typedef struct {
  float* row_max;    /* M_i = max_j s_ij over valid keys (App. A) */
  float* row_min;    /* m_i = min_j s_ij; MinMax only (the FWM and softmax grids are
                        anchored at M_i alone): otherwise set to +inf */
  int32_t* arg_max;  /* lowest j with s_ij == M_i */
  int32_t* arg_min;  /* lowest j with s_ij == m_i; -1 when row_min is not computed */
  int32_t* n_max;    /* number of keys tied at M_i (the extremum gradient is split evenly) */
  int32_t* n_min;    /* number of keys tied at m_i; 0 when row_min is not computed */
  float* W;          /* W^N = sum w^N (Nearest) or W^L (LERP); softmax: sum e^{s - M};
                        EXP_FP8: sum E4M3(e^{s - M}) */
  float* W_lerp;     /* W^L; required for Prob-STE, may be NULL otherwise */
  float* O_lerp;     /* [B,H,T,d] P^L V; required for Prob-STE, may be NULL otherwise */
  float* c_M;        /* optional side output of kint_attn_bwd (NULL: not written): the row's
                        calibration sum c_M = sum_j gamma_j dw_j/dM (supplement "Local gradient
                        decomposition", the M channel; EXP_FP8: -sum_j gamma_j e^{z_j}); 0 under
                        detach, detach_proj and for softmax */
  float* c_m;        /* optional side output of kint_attn_bwd: c_m = sum_j gamma_j dw_j/dm
                        (MinMax; 0 otherwise) */
  /* Optional side outputs of kint_attn_bwd (NULL: not written), [B,H,T] each: the row sums
   * sum_j dS_ij (dS_sum) and sum_j |dS_ij| (dS_abs) of the score gradient that the dK
   * contraction uses, extremum terms, tie split and the P1 projection included.  Eq. (full)
   * makes sum_j dS_ij zero in exact arithmetic in every full mode (the three per-key terms
   * cancel, Sec. 3 after Eq. full); the detached mode breaks it (App. B "Detach (legacy)").
   * |dS_sum| / dS_abs per row is the zero-sum residual of the paper's gradient-consistency
   * diagnostics.  Accumulated with fp32 atomics in an order that is not fixed; the call
   * zeroes them first.  Either may be NULL; giving one selects a slower diagnostic variant
   * of the dK/dV kernel.  16-byte aligned. */
  float* dS_sum;
  float* dS_abs;
} kint_rowstats;

/*
 * Workspace needed by kint_attn_fwd (is_bwd = 0) or kint_attn_bwd (is_bwd = 1)
 * for these sizes and precision.  0 for invalid sizes.
 */
size_t kint_attn_workspace_bytes(int B, int H, int T, int d, kint_prec prec, int is_bwd);

/*
 * Forward: O = P V with P the K-interval probabilities (App. A).  For Nearest
 * the forward returns the hard probabilities P^N = w^N / W^N directly
 * (the strict hard forward of App. C.2 (iii)); for LERP P^L = w^L / W^L.
 *   Q, K, V  in:  [B,H,T,d]
 *   O        out: [B,H,T,d]
 *   st       out: row statistics (struct itself is host memory, read during the call)
 *   Kint     number of intervals K, 1..64 (ignored for softmax and EXP_FP8)
 *   tau      FWM window in nats, > 0 (FWM and FWM_RESOLVED; ignored otherwise)
 *   workspace, workspace_bytes: device scratch of at least
 *            kint_attn_workspace_bytes(B, H, T, d, prec, 0) bytes
 */
int kint_attn_fwd(const float* Q, const float* K, const float* V, float* O, const kint_rowstats* st, int B, int H,
                  int T, int d, int Kint, kint_calib calib, float tau, kint_recon recon, kint_ste ste,
                  kint_grad grad, int causal, kint_prec prec, void* workspace, size_t workspace_bytes,
                  void* stream);

/*
 * Backward (App. B): dQ, dK, dV of L given dO = dL/dO, with the row statistics
 * of the forward of the same inputs and configuration.
 *   gamma_j = (g_j - <g>_{P*}) / W*, g_j = dO_i . V_j, where (P*, W*) is
 *     (P^N, W^N) for Nearest + Weight-STE and (P^L, W^L) otherwise;
 *   dS_ij = gamma_j Delta_j + [j tied at M_i] c_M / n_max + [j tied at m_i] c_m / n_min
 *     (c_m only for MinMax; both dropped under detach, c_m under max_only, c_M under
 *      min_only; FWM tail keys get 0; degenerate MinMax rows get 0; FWM_RESOLVED has no
 *      tail; EXP_FP8 uses gamma at the rounded weights and e^{z_j} in place of Delta_j);
 *     under detach_proj each causal row of the detached dS then loses its mean;
 *   st->c_M, st->c_m, when non-NULL, receive the per-row sums c_M, c_m (16-byte aligned;
 *     the sums are written whether or not the mode applies them, 0 under detach and
 *     detach_proj);
 *   dQ = dS K / sqrt(d), dK = dS^T Q / sqrt(d), dV = P^T dO with the forward P.
 * dQ, dK, dV are overwritten.
 * Two implementations (kint_set_backward_path): TF32 at d = 64 with any calibration but
 * MinMax and any mode but detach_proj, and without dS_sum / dS_abs, runs a single pass
 * over the (key block, query tile) pairs that adds its dQ partial sums, and then the
 * extremum terms, in fp32 in global memory: the order of those additions is not fixed,
 * so dQ (and dK under the extremum terms) may differ in the last bits from call to call.
 * Everything else, and calls whose rows hold more tied maximum keys in all than the call
 * has rows (the single pass lists each tied key), runs two passes (dQ, then dK/dV) whose
 * results are bit-reproducible.
 *   O        in:  forward output
 *   dO       in:  [B,H,T,d]
 *   st       in:  row statistics written by kint_attn_fwd
 */
int kint_attn_bwd(const float* Q, const float* K, const float* V, const float* O, const float* dO,
                  const kint_rowstats* st, float* dQ, float* dK, float* dV, int B, int H, int T, int d, int Kint,
                  kint_calib calib, float tau, kint_recon recon, kint_ste ste, kint_grad grad, int causal,
                  kint_prec prec, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Geometry probe (App. "Geometry probe"), MinMax and FWM only: pass 1 on Q, K (into st,
 * as kint_attn_fwd writes it), then per causal row i of every head, from the fp32 scores
 * the operator uses, into probe[k * B*H*T + (b*H + h)*T + i] for k =
 *   0  span M - m (0 for a degenerate MinMax row)
 *   1  native width h: (M - m)/K (MinMax), tau/K (FWM); 0 for a degenerate row
 *   2  softmax entropy H(P^E), P^E = softmax of the row's scores
 *   3  share of the row's i + 1 keys with z = s - M < -6
 *   4  top-bucket mass: P^E mass on keys in the top level (Nearest, l = K) or the top
 *      interval (LERP, r = K - 1); 1 for a degenerate row
 *   5  effective buckets exp H(q), q_b the P^E mass of bucket b: the Nearest levels l or the
 *      LERP intervals r, FWM tail keys as one more bucket, a degenerate row as one bucket
 *   6  total variation 1/2 sum_j |P_j - P^E_j| to the operator's forward P
 * probe: device, [7][B,H,T] fp32, 16-byte aligned, caller-owned.  The workspace is the
 * forward's (kint_attn_workspace_bytes(..., 0)).  The per-CTA bucket masses take
 * 1 KB x (K + 2) of shared memory: TF32 at d = 64 supports every K, 3xTF32 and d = 128
 * K <= 27 (KINT_ERR_UNSUPPORTED above).  Diagnostic: not on the training path.
 */
int kint_attn_probe(const float* Q, const float* K, const kint_rowstats* st, float* probe, int B, int H, int T,
                    int d, int Kint, kint_calib calib, float tau, kint_recon recon, int causal, kint_prec prec,
                    void* workspace, size_t workspace_bytes, void* stream);

/*
 * Decision dump for parity checks: for every (b, h, i, j) the Nearest index
 * l_ij = r + [t >= 1/2] in 0..K (bins) and the interval index r_ij in 0..K-1
 * (ivals), with 254 for FWM tail keys (z < -tau), 255 for masked keys (j > i)
 * and 253 where no grid exists (degenerate MinMax rows, softmax); under
 * FWM_RESOLVED both indices run below zero and are stored as index + 128,
 * saturated to [0, 252] (0: index <= -128); under EXP_FP8 both hold the E4M3
 * byte of the rounded weight (0x00 = 0 .. 0x38 = 1); under EXP_BF16 bins holds the low
 * byte of the bfloat16 bits of z and ivals that of the weight.  Either
 * output may be NULL.  Needs the row statistics of kint_attn_fwd on the same
 * inputs and the forward's workspace size.  bins, ivals: [B,H,T,T] uint8.
 */
int kint_attn_debug_bins(const float* Q, const float* K, const float* V, const kint_rowstats* st, uint8_t* bins,
                         uint8_t* ivals, int B, int H, int T, int d, int Kint, kint_calib calib, float tau,
                         kint_recon recon, kint_ste ste, int causal, kint_prec prec, void* workspace,
                         size_t workspace_bytes, void* stream);

/*
 * Synchronises `stream`, then returns KINT_OK, or KINT_ERR_DEVICE if any kernel
 * of this library flagged a device-side fault since the last call (the flag
 * word is cleared).  *detail (may be NULL) receives the raw flag bits:
 * 1 = TMA wait timed out, 2 = MMA wait timed out, 4 = CTA sync timed out.
 */
int kint_get_status(void* stream, unsigned* detail);

/* Human-readable text for a return code (static storage). */
const char* kint_strerror(int code);

/* Wall-clock limit, in nanoseconds, of every bounded device-side wait
 * (default 2e9).  Values < 1000 are clamped to 1000. */
void kint_set_wait_timeout_ns(unsigned long long ns);

/*
 * Test hook of the bounded waits (the paper has no counterpart).  The next `count`
 * calls that run the row-statistics pass (kint_attn_fwd, kint_attn_fwd_noalloc,
 * kint_attn_debug_bins, kint_attn_probe) make that kernel's first wait, which comes
 * before it issues any copy or product, wait on a barrier that nothing completes.  The
 * wait gives up after the kint_set_wait_timeout_ns limit: the kernel sets bit 4 (CTA
 * sync timed out) in the status word, releases its tensor memory and leaves, so
 * kint_get_status then returns KINT_ERR_DEVICE and the context stays usable.  The
 * outputs of such a call are not defined.  Nothing faults, traps or hangs.  count <= 0
 * cancels pending requests.  Process-wide.
 */
void kint_test_expire_next_wait(int count);

/*
 * Backward implementation choice (process-wide; the paper has no counterpart): 0 (default)
 * uses the single-pass backward wherever kint_attn_bwd describes it as applying, 1 always
 * the two-pass kernels (bit-reproducible).  Other values act as 0.  Do not change it
 * while another thread is inside an entry point.
 */
void kint_set_backward_path(int path);

/*
 * Launch tracing (a profiling aid with no counterpart in the paper).  When set,
 * cb(kernel_name, phase, stream, user) is called on the host immediately before
 * (phase 0) and after (phase 1) every kernel launch this library makes, with
 * the stream the kernel is enqueued on, so a caller can record CUDA events
 * around single kernels.  NULL disables it.  Process-wide setting; do not
 * change it while another thread is inside an entry point.
 */
typedef void (*kint_launch_cb)(const char* kernel_name, int phase, void* stream, void* user);
void kint_set_launch_callback(kint_launch_cb cb, void* user);

/*
 * Forward without a caller-supplied workspace (the paper has no counterpart).
 *
 * Some callers cannot hand the library scratch memory: code that runs while a
 * stream is being captured into a CUDA graph (where cudaMalloc is not allowed),
 * serving loops that forbid any device allocation after start-up, and plug-in
 * hosts that pass only input and output buffers.  This entry point behaves like
 * kint_attn_fwd but takes its scratch from a fixed array of
 * KINT_NOALLOC_SCRATCH_BYTES that the library keeps in device memory (every GPU
 * that loads the library holds it until the process exits).  It allocates
 * nothing.  The caller still provides Q, K, V, O and the row statistics.
 *   - The first call on a device (with that device current) looks up the
 *     array's device address; make that first call before any stream capture.
 *   - Problems whose forward workspace, kint_attn_workspace_bytes(..., 0),
 *     exceeds KINT_NOALLOC_SCRATCH_BYTES return KINT_ERR_SCRATCH_LIMIT before
 *     any work is enqueued.  That workspace is B*H*d*round_up(T, 32)*4 bytes in
 *     TF32 (so at d = 64 the limit is B*H*round_up(T, 32) <= 131072) and about
 *     four times as much in 3xTF32; compare kint_attn_workspace_bytes(..., 0)
 *     with KINT_NOALLOC_SCRATCH_BYTES to know in advance.
 *   - All calls share the one array: calls whose work overlaps on the GPU
 *     (different streams, or concurrent host threads) race and must be
 *     serialised by the caller.  The array keeps the previous call's contents;
 *     nothing in it needs to start at zero, because every forward writes the
 *     whole region it later reads.
 */
#define KINT_NOALLOC_SCRATCH_BYTES (32u << 20)
int kint_attn_fwd_noalloc(const float* Q, const float* K, const float* V, float* O, const kint_rowstats* st, int B,
                          int H, int T, int d, int Kint, kint_calib calib, float tau, kint_recon recon,
                          kint_ste ste, kint_grad grad, int causal, kint_prec prec, void* stream);

#ifdef __cplusplus
}
#endif
#endif
