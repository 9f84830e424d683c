// Launch parameters shared by the host launcher and the kernels of libkint.
// Plain data only; the tensor maps travel separately as __grid_constant__.
#pragma once
#include <cstdint>
#include <cuda.h>

namespace kint {

enum Calib : int { CAL_MINMAX = 0, CAL_FWM = 1, CAL_SOFTMAX = 2, CAL_FWMR = 3, CAL_EXP8 = 4, CAL_EXPB = 5 };
// FWM's grid (step tau/K, origin -tau), with a zero tail below the window (FWM) or
// continued below it with negative indices (CAL_FWMR, the "resolved" tail policy)
__host__ __device__ constexpr bool fwm_like(int cal) { return cal == CAL_FWM || cal == CAL_FWMR; }
// weights from the exponential unit instead of a grid: the softmax comparator, and
// CAL_EXP8, the FP8-rounded exponential baseline (E4M3(e^z) forward, e^z backward)
__host__ __device__ constexpr bool exp_like(int cal) { return cal == CAL_SOFTMAX || cal == CAL_EXP8; }
// no grid at all (no reconstruction, no surrogate placement): the above and CAL_EXPB, the
// BF16 exponential baseline (z and e^z rounded to bfloat16, bfloat16 chain rule backward)
__host__ __device__ constexpr bool gridless(int cal) { return exp_like(cal) || cal == CAL_EXPB; }
enum Recon : int { REC_LERP = 0, REC_NEAREST = 1 };
enum Grad : int { GRAD_FULL = 0, GRAD_DETACH = 1, GRAD_MAX_ONLY = 2, GRAD_MIN_ONLY = 3, GRAD_DETACH_PROJ = 4 };

constexpr int KMAX = 64;  // largest number of intervals K

// Which weights a forward main-pass launch feeds to the P V contraction.
enum PvSel : int {
  PV_MAIN = 0,       // forward weights (w^N, w^L or e^z) -> O, W
  PV_MAIN_LERP = 1,  // both: forward weights -> O, w^L -> O_lerp (TF32 only)
  PV_LERP = 2,       // w^L -> O_lerp, W_lerp (second launch of 3xTF32 Prob-STE)
};
// Which products a dK/dV launch computes.
enum DkvSel : int { DKV_BOTH = 0, DKV_DV = 1, DKV_DK = 2 };

// Every TMA descriptor a launch may use.  Natural maps view X as [BH][T][d]
// (box 32 x rows); transposed maps view X^T as [BH][d][Tp] (box 32 x d).
struct Maps {
  CUtensorMap q, q_lo, k, k_lo, v, v_lo, dout, dout_lo;  // natural
  CUtensorMap kt, kt_lo, vt, vt_lo, qt, qt_lo, dot, dot_lo;  // transposed
  CUtensorMap out, out_lerp, dq, dk, dv;  // outputs (natural, box 32 x 64 rows) for TMA stores
  CUtensorMap dq16, dk32, dv32;  // single-pass backward: 16-column boxes (64-byte swizzle), dQ reduces of 16 rows, dK / dV stores of 32
};

// Static item schedule of a persistent kernel, computed on the host (longest processing
// time first over the launch's CTAs): CTA c takes the items idx[off[c]] .. idx[off[c+1] - 1]
// in that order.  n == 0: no schedule, the snake order (snake_item) instead.
constexpr int SCHED_MAX_CTAS = 304, SCHED_MAX_ITEMS = 1536;
struct Sched {
  int n;
  uint16_t off[SCHED_MAX_CTAS + 1];
  uint16_t idx[SCHED_MAX_ITEMS];
};

struct Params {
  int B, H, T, d, Kint, calib, recon, ste, grad, x3;
  int BH, nqb;  // number of 128-row query blocks
  float tau, scale;       // scale = 1/sqrt(d)
  float fwm_inv_h;        // K / tau (FWM), host-rounded
  float fwm_hl, fwm_b0l;  // (tau / K) log2 e and -tau log2 e (resolved grid below the window)
  float fwm_e[KMAX + 2];  // FWM grid values e^{-tau + r tau/K}, r = 0..K (host fp64 -> fp32)
  int pv_sel, dkv_sel, debug;
  int expire_wait;  // test hook: the launch's first wait is on a barrier that nothing completes
  unsigned long long wait_ns;
  unsigned* status;

  // smem plan (byte offsets from the 1024-aligned base), set by the host
  int sm_a, sm_stage0, sm_stage_bytes, nstage, sm_table, sm_rows, sm_bars;
  int sm_rstat;  // dQ kernel: the next item's row statistics, [9][256] words
  int nbuf;  // score buffers in TMEM (2: the next tile's product runs under this tile's element work)
  int nitems;     // work items (128-row query or key block, head), longest first
  int ngrid;      // CTAs launched: nitems, or one per SM when the kernel loops over items
  int sm_ostage;  // smem tile(s) the epilogue stages outputs in for TMA stores
  int ops_smem;  // backward: the 128-row TMEM operands (Q, dO / K, V) are staged in smem by TMA first
  int sm_v, sm_kt;  // single-pass backward: the V tile (A operand of g^T) and the K^T tile (B operand of dQ)
  // Launch gate of the backward kernels that run on one side of a device-side decision:
  // with gate set, the kernel does its work only if (*gate != 0) == (gate_on != 0)
  const int* gate;
  int gate_on;

  // tensors (device pointers)
  const float *Q, *K, *V, *O, *dO, *Ostar;
  float* Out;
  float *row_max, *row_min, *W, *W_lerp, *O_lerp;
  int32_t *arg_max, *arg_min, *n_max, *n_min;
  float *dQ, *dK, *dV;
  void* rec;                // [B*H*T] per-query-row records (RowRec) written by the dQ kernel
  float* rtab;              // [B*H*T][Kp] (e_r, e_{r+1}) MinMax grid pairs per row (workspace)
  int Kp;                   // K rounded up to even (pair-table row stride in pairs)
  int* tileflags;           // [B*H][nqt] 1 where a 64-row query tile holds a row with tied extrema
  int nqt;                  // ceil(T / 64)
  float* tie_acc;           // [2][BH*T][d] sums of tied keys (workspace, touched only on ties)
  const float* gbar;        // [BH*T] <g>_{P*} = dO_i . O*_i (workspace, written by the dO prep)
  float *cM_out, *cm_out;   // optional [BH*T] side outputs of the backward: c_M, c_m per row
  float *dsum_out, *dabs_out;  // optional [BH*T] side outputs of the backward: sum_j dS_ij, sum_j |dS_ij|
  void* frec;               // [B*H*T] 16-byte row records of the single-pass backward (RecJob of k_prep)
  float* rsum;              // [B*H*T] single-pass backward: sum_j gamma_ij Delta_ij per row
  int* tie_any;             // single-pass backward: set when the rows' ties exceed the tie list
  int* tie_count;           // single-pass backward: entries in tie_list; tie_total: the ties the rows hold
  int* tie_total;
  int2* tie_list;           // [tie_cap] (row, key) pairs of tied maxima found by k_bwd_fused
  int tie_cap;
  float* kt_out;            // [BH][d][Tp] K^T for the two-pass kernels, written by k_bwd_ext when the
                            // single pass gives way to them (the single pass forms its K^T tiles itself)
  float* probe;             // [7][BH*T] geometry probe outputs
  uint8_t *bins, *ivals;
};

}  // namespace kint
