// Backward of K-interval attention on sm_103a (App. B).
//
// k_bwd_dq   (one CTA per 128-row query block, thread = query row): recomputes
//   S = Q K^T and g = dO V^T per 64-key tile, forms the own-score term
//   dS_own = gamma Delta, accumulates the row's calibration sums, and
//   dQ = dS_own K.  At the end of the row it knows c_M and c_m (Eq. full) and
//   adds their contribution at the arg-max / arg-min keys; it also leaves the
//   row scalars <g>_{P*}, c_M / n_max, c_m / n_min for the second kernel.
// k_bwd_dkdv (one CTA per 128-key block, thread = key): recomputes S^T and
//   g^T per 64-query tile, forms the full dS (calibration terms included, now
//   that c_M, c_m are known) and the forward P, and accumulates
//   dV = P^T dO, dK = dS^T Q.
#include <cfloat>
#include "kint_dev.cuh"
#include "kint_launch.h"

namespace kint {

constexpr int BKEY = 64;  // keys per tile in k_bwd_dq
constexpr int BQRY = 64;  // queries per tile in k_bwd_dkdv

// Quantities of one score element needed by the backward.
struct BwdElem {
  float p;    // forward probability P_ij
  float ds;   // dL/ds_ij without the extremum terms
  float dm;   // gamma * dw/dm (MinMax calibration sum term)
};

// Row-level constants of query row i.
struct RowB {
  RowGrid g;
  float M, m, invWf, invWs, D;
};

// Own-score gradient and forward probability of one valid key (App. B):
//   gamma = (g - <g>_{P*}) / W*, Delta = (e_{r+1} - e_r) / h, dS_own = gamma Delta,
//   dw/dm = A_r + t B_r with A_r = (1 - r/K)(e_r - Delta), B_r = (1-(r+1)/K) e_{r+1} - (1 - r/K) e_r + Delta/K
//   (Eq. calgrad rewritten per interval; dw/dM = -Delta - dw/dm).
__device__ __forceinline__ BwdElem bwd_elem(const Params& p, const RowB& R, float s, float gval, float er_tab_r,
                                            float er_tab_r1, float el_tab, const KeyPos& kp) {
  BwdElem e{0.f, 0.f, 0.f};
  if (p.calib == CAL_SOFTMAX) {
    e.p = expf(__fsub_rn(s, R.M)) * R.invWf;
    e.ds = e.p * (gval - R.D);  // P (g - <g>_P)  (App. B, Softmax)
    return e;
  }
  if (R.g.nogrid) {  // degenerate MinMax row: uniform P, zero gradient
    e.p = R.invWf;
    return e;
  }
  if (kp.tail) return e;  // FWM zero tail: weight and gradient 0
  const float wl = __fmaf_rn(kp.t, __fsub_rn(er_tab_r1, er_tab_r), er_tab_r);
  const float wf = (p.recon == REC_NEAREST) ? el_tab : wl;
  e.p = wf * R.invWf;
  const float gam = (gval - R.D) * R.invWs;
  const float dlt = __fsub_rn(er_tab_r1, er_tab_r) * R.g.inv_h;
  e.ds = gam * dlt;
  if (p.calib == CAL_MINMAX && p.grad == 0) {
    const float fk = 1.0f / (float)p.Kint;
    const float ar = 1.0f - (float)kp.r * fk;
    const float ar1 = ar - fk;
    const float A = ar * (er_tab_r - dlt);
    const float Bc = ar1 * er_tab_r1 - ar * er_tab_r + dlt * fk;
    e.dm = gam * (A + kp.t * Bc);
  }
  return e;
}

// ---------------------------------------------------------------------------
// k_bwd_dq.  TMEM columns: Q [0, dp), dO [dp, 2dp), S [2dp, 2dp+64),
// g [2dp+64, 2dp+128), dQ [2dp+128, 2dp+128+d), dp = d (TF32) or 2d (3xTF32:
// hi then lo).  dS overwrites S (and, as the lo part under 3xTF32, g).
// smem: stages {K [64 x d], V [64 x d], K^T [d x 64]} (hi[, lo] each);
// per-thread grid table [K+1][128] at sm_table.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(NT, 1) k_bwd_dq(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1;
  const int ktile = BKEY * D * 4;  // [64 x D] natural or [D x 64] transposed
  float* tab = reinterpret_cast<float*>(sm + p.sm_table);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_st = bars;
  uint64_t* bar_mma = bars + p.nstage;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 1 + p.nstage);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int bh = blockIdx.y, qb = p.nqb - 1 - blockIdx.x;
  const int i = qb * 128 + tid;
  const bool row_ok = i < p.T;
  const int nkt = min(2 * qb + 2, (p.T + BKEY - 1) / BKEY);
  const int dp = D * parts;
  const int cQ = 0, cdO = dp, cS = 2 * dp, cG = 2 * dp + 64, cdQ = 2 * dp + 128;

  if (tid == 0) {
    for (int s = 0; s < p.nstage; ++s) mbar_init(&bar_st[s], 1);
    mbar_init(bar_mma, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  auto stage_ptr = [&](int kt) { return sm + p.sm_stage0 + (kt % p.nstage) * p.sm_stage_bytes; };
  auto load_stage = [&](int kt) {
    uint64_t* b = &bar_st[kt % p.nstage];
    uint8_t* dst = stage_ptr(kt);
    mbar_arrive_expect_tx(b, 3 * parts * ktile);
    load_rows_tile(dst, &maps.k, b, D, BKEY, 0, kt * BKEY, bh);
    load_rows_tile(dst + parts * ktile, &maps.v, b, D, BKEY, 0, kt * BKEY, bh);
    load_rows_tile(dst + 2 * parts * ktile, &maps.kt, b, BKEY, D, kt * BKEY, 0, bh);
    if (p.x3) {
      load_rows_tile(dst + ktile, &maps.k_lo, b, D, BKEY, 0, kt * BKEY, bh);
      load_rows_tile(dst + parts * ktile + ktile, &maps.v_lo, b, D, BKEY, 0, kt * BKEY, bh);
      load_rows_tile(dst + 2 * parts * ktile + ktile, &maps.kt_lo, b, BKEY, D, kt * BKEY, 0, bh);
    }
  };
  if (tid == 0)
    for (int kt = 0; kt < min(p.nstage, nkt); ++kt) load_stage(kt);

  // Operands A = Q and dO of this thread's row into TMEM.
  row_to_tmem(tmem, cQ, p.Q, bh * p.T + i, row_ok ? (bh + 1) * p.T : 0, D, p.x3 != 0);
  row_to_tmem(tmem, cdO, p.dO, bh * p.T + i, row_ok ? (bh + 1) * p.T : 0, D, p.x3 != 0);

  // Row constants.
  const size_t row = (size_t)bh * p.T + (row_ok ? i : 0);
  RowB R;
  R.M = row_ok ? p.row_max[row] : 0.f;
  R.m = row_ok ? p.row_min[row] : 0.f;
  R.g = row_grid(p, R.M, R.m);
  const float Wf = row_ok ? p.W[row] : 1.f;
  const bool prob = (p.recon == REC_NEAREST && p.ste == 1 && p.calib != CAL_SOFTMAX);
  const float Ws = prob ? (row_ok ? p.W_lerp[row] : 1.f) : Wf;
  R.invWf = 1.0f / Wf;
  R.invWs = 1.0f / Ws;
  // <g>_{P*} = dO_i . O*_i  with O* = P* V (P* = P^L for Prob-STE, else the forward P)
  {
    float acc = 0.f;
    if (row_ok) {
      const float4* a = reinterpret_cast<const float4*>(p.dO + row * D);
      const float4* b = reinterpret_cast<const float4*>(p.Ostar + row * D);
      for (int q = 0; q < D / 4; ++q) {
        const float4 x = __ldg(a + q), y = __ldg(b + q);
        acc = __fmaf_rn(x.x, y.x, acc);
        acc = __fmaf_rn(x.y, y.y, acc);
        acc = __fmaf_rn(x.z, y.z, acc);
        acc = __fmaf_rn(x.w, y.w, acc);
      }
    }
    R.D = acc;
  }
  const int nmax = row_ok ? p.n_max[row] : 1, nmin = row_ok ? p.n_min[row] : 1;
  const int amax = row_ok ? p.arg_max[row] : 0, amin = row_ok ? p.arg_min[row] : 0;
  const bool full = p.grad == 0 && p.calib != CAL_SOFTMAX && !R.g.nogrid;
  const bool minmax = p.calib == CAL_MINMAX;
  if (p.calib != CAL_SOFTMAX)
    for (int r = 0; r <= Kq; ++r) tab[r * NT + tid] = grid_value(p, R.g, r);
  float* tie_max = p.tie_acc + row * D;
  float* tie_min = p.tie_acc + ((size_t)p.BH * p.T + row) * D;
  const bool track_ties = row_ok && full && (nmax > 1 || (minmax && nmin > 1));
  if (track_ties)
    for (int k = 0; k < D; ++k) {
      tie_max[k] = 0.f;
      tie_min[k] = 0.f;
    }

  tmem_st_wait();
  tc_fence_before();
  __syncthreads();

  float own_acc = 0.f, cm_acc = 0.f;
  bool failed = false;
  uint32_t mph = 0;
  for (int kt = 0; kt < nkt; ++kt) {
    const uint8_t* st = stage_ptr(kt);
    if (tid == 0) {
      const bool ok =
          mbar_wait(&bar_st[kt % p.nstage], (kt / p.nstage) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      if (ok) {
        tc_fence_after();
        const uint8_t* sk = st;
        const uint8_t* sv = st + parts * ktile;
        if (p.x3) {
          mma_tmem_smem(tmem + cS, tmem + cQ + D, sk, BKEY, D, false);   // Q_lo K_hi
          mma_tmem_smem(tmem + cS, tmem + cQ, sk + ktile, BKEY, D, true); // Q_hi K_lo
          mma_tmem_smem(tmem + cS, tmem + cQ, sk, BKEY, D, true);         // Q_hi K_hi
          mma_tmem_smem(tmem + cG, tmem + cdO + D, sv, BKEY, D, false);
          mma_tmem_smem(tmem + cG, tmem + cdO, sv + ktile, BKEY, D, true);
          mma_tmem_smem(tmem + cG, tmem + cdO, sv, BKEY, D, true);
        } else {
          mma_tmem_smem(tmem + cS, tmem + cQ, sk, BKEY, D, false);
          mma_tmem_smem(tmem + cG, tmem + cdO, sv, BKEY, D, false);
        }
        mma_commit(bar_mma);
      }
    }
    bool ok = mbar_wait(bar_mma, mph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
    mph ^= 1;
    if (cta_any(!ok)) {
      failed = true;
      break;
    }
    tc_fence_after();
#pragma unroll 1
    for (int c = 0; c < BKEY / 32; ++c) {
      float sv[32], gv[32], a1[32], a2[32];
      tmem_ld32(lane_addr(tmem, cS + c * 32), sv);
      tmem_ld32(lane_addr(tmem, cG + c * 32), gv);
      tmem_ld_wait();
      const int j0 = kt * BKEY + c * 32;
#pragma unroll
      for (int jj = 0; jj < 32; ++jj) {
        const int j = j0 + jj;
        const bool valid = row_ok && j <= i;
        float ds = 0.f;
        if (valid) {
          const float s = __fmul_rn(sv[jj], p.scale);
          KeyPos kp{0, 0, 0.f, false};
          float er = 0.f, er1 = 0.f, el = 0.f;
          if (p.calib != CAL_SOFTMAX && !R.g.nogrid) {
            kp = key_pos(p, __fmaf_rn(sv[jj], R.g.k1, R.g.c0));
            if (!kp.tail) {
              er = tab[kp.r * NT + tid];
              er1 = tab[(kp.r + 1) * NT + tid];
              el = tab[kp.l * NT + tid];
            }
          }
          const BwdElem e = bwd_elem(p, R, s, gv[jj], er, er1, el, kp);
          ds = e.ds;
          if (full) {
            own_acc += e.ds;
            cm_acc += e.dm;
            if (track_ties) {
              if (nmax > 1 && s == R.M)
                for (int k = 0; k < D; ++k) tie_max[k] += p.K[((size_t)bh * p.T + j) * D + k];
              if (minmax && nmin > 1 && s == R.m)
                for (int k = 0; k < D; ++k) tie_min[k] += p.K[((size_t)bh * p.T + j) * D + k];
            }
          }
        }
        if (p.x3) {
          const float h = tf32_rna(ds);
          a1[jj] = h;
          a2[jj] = __fsub_rn(ds, h);
        } else {
          a1[jj] = ds;
        }
      }
      tmem_st32(lane_addr(tmem, cS + c * 32), a1);
      if (p.x3) tmem_st32(lane_addr(tmem, cG + c * 32), a2);
    }
    tmem_st_wait();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint8_t* skt = st + 2 * parts * ktile;
      const bool acc = kt > 0;
      if (p.x3) {
        mma_tmem_smem(tmem + cdQ, tmem + cS, skt, D, BKEY, acc);           // dS_hi K_hi
        mma_tmem_smem(tmem + cdQ, tmem + cS, skt + ktile, D, BKEY, true);  // dS_hi K_lo
        mma_tmem_smem(tmem + cdQ, tmem + cG, skt, D, BKEY, true);          // dS_lo K_hi
      } else {
        mma_tmem_smem(tmem + cdQ, tmem + cS, skt, D, BKEY, acc);
      }
      mma_commit(bar_mma);
    }
    ok = mbar_wait(bar_mma, mph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
    mph ^= 1;
    if (cta_any(!ok)) {
      failed = true;
      break;
    }
    tc_fence_after();
    if (tid == 0 && kt + p.nstage < nkt) load_stage(kt + p.nstage);
  }

  if (!failed) {
    // Extremum terms of Eq. (full): c_m = sum_j gamma_j dw_j/dm; c_M = -sum_j gamma_j Delta_j - c_m
    // (App. B: Delta + dw/dM + dw/dm = 0); FWM: c_M = -sum_window gamma Delta, no m term.
    const float cm = (full && minmax) ? cm_acc : 0.f;
    const float cM = full ? (-own_acc - cm) : 0.f;
    const float cMn = cM / (float)nmax, cmn = cm / (float)nmin;
    const float* kmax = (nmax == 1) ? p.K + ((size_t)bh * p.T + amax) * D : tie_max;
    const float* kmin = (nmin == 1) ? p.K + ((size_t)bh * p.T + amin) * D : tie_min;
    float* dst = p.dQ + row * D;
    for (int c = 0; c < D; c += 32) {
      float v[32];
      tmem_ld32(lane_addr(tmem, cdQ + c), v);
      tmem_ld_wait();
      if (row_ok) {
#pragma unroll 4
        for (int q = 0; q < 32; ++q) {
          float x = v[q];
          if (full) {
            x = __fmaf_rn(cMn, kmax[c + q], x);
            if (minmax) x = __fmaf_rn(cmn, kmin[c + q], x);
          }
          dst[c + q] = x * p.scale;
        }
      }
    }
    if (row_ok) {
      p.Drow[row] = R.D;
      p.cMn[row] = cMn;
      p.cmn[row] = cmn;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

cudaError_t launch_bwd_dq(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_bwd_dq, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  k_bwd_dq<<<dim3(p.nqb, p.BH), NT, smem_bytes, s>>>(maps, p);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// k_bwd_dkdv.  Thread t owns key j = kb*128 + t (TMEM lane t).  TMEM columns:
// K [0, dp), V [dp, 2dp) (dK launches), then S^T (64), g^T (64), dV (d), dK (d).
// P^T overwrites S^T and dS^T overwrites g^T; under 3xTF32 (one product per
// launch) the hi part goes to the first and the lo part to the second.
// smem: stages {Q [64 x d], dO [64 x d], Q^T [d x 64], dO^T [d x 64]} (hi[, lo]);
// per-query-row constants and grid tables of the current query tile.
// ---------------------------------------------------------------------------
struct QRows {  // per query row of the current tile, in shared memory
  float M[BQRY], m[BQRY], inv_h[BQRY], c0[BQRY], invWf[BQRY], invWs[BQRY], D[BQRY], cMn[BQRY], cmn[BQRY];
  int amax[BQRY], amin[BQRY], nmax[BQRY], nmin[BQRY], nogrid[BQRY];
};

__global__ void __launch_bounds__(NT, 1) k_bwd_dkdv(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1;
  const int qtile = BQRY * D * 4;
  const bool do_dv = p.dkv_sel != DKV_DK, do_dk = p.dkv_sel != DKV_DV;
  QRows* qr = reinterpret_cast<QRows*>(sm + p.sm_rows);
  float* tab = reinterpret_cast<float*>(sm + p.sm_table);  // [BQRY][K+2]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_st = bars;
  uint64_t* bar_mma = bars + p.nstage;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 1 + p.nstage);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int bh = blockIdx.y, kb = blockIdx.x;
  const int j = kb * 128 + tid;
  const int dp = D * parts;
  const int cK = 0, cV = dp;
  const int cS = do_dk ? 2 * dp : dp;
  const int cG = cS + 64, cdV = cS + 128, cdK = cdV + (do_dv ? D : 0);
  const int qt0 = (kb * 128) / BQRY;
  const int nqt = (p.T + BQRY - 1) / BQRY;
  const int tstride = Kq + 2;
  // Stage layout: Q | dO | Q^T | dO^T, each `parts` tiles; only the needed ones are loaded.
  const int oQ = 0, odO = parts * qtile, oQT = 2 * parts * qtile, odOT = 3 * parts * qtile;
  const bool need_dO = do_dk, need_QT = do_dk, need_dOT = do_dv;

  if (tid == 0) {
    for (int s = 0; s < p.nstage; ++s) mbar_init(&bar_st[s], 1);
    mbar_init(bar_mma, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  auto stage_ptr = [&](int it) { return sm + p.sm_stage0 + (it % p.nstage) * p.sm_stage_bytes; };
  auto load_stage = [&](int it) {
    const int q0 = (qt0 + it) * BQRY;
    uint64_t* b = &bar_st[it % p.nstage];
    uint8_t* dst = stage_ptr(it);
    const int ntiles = 1 + (need_dO ? 1 : 0) + (need_QT ? 1 : 0) + (need_dOT ? 1 : 0);
    mbar_arrive_expect_tx(b, ntiles * parts * qtile);
    load_rows_tile(dst + oQ, &maps.q, b, D, BQRY, 0, q0, bh);
    if (p.x3) load_rows_tile(dst + oQ + qtile, &maps.q_lo, b, D, BQRY, 0, q0, bh);
    if (need_dO) {
      load_rows_tile(dst + odO, &maps.dout, b, D, BQRY, 0, q0, bh);
      if (p.x3) load_rows_tile(dst + odO + qtile, &maps.dout_lo, b, D, BQRY, 0, q0, bh);
    }
    if (need_QT) {
      load_rows_tile(dst + oQT, &maps.qt, b, BQRY, D, q0, 0, bh);
      if (p.x3) load_rows_tile(dst + oQT + qtile, &maps.qt_lo, b, BQRY, D, q0, 0, bh);
    }
    if (need_dOT) {
      load_rows_tile(dst + odOT, &maps.dot, b, BQRY, D, q0, 0, bh);
      if (p.x3) load_rows_tile(dst + odOT + qtile, &maps.dot_lo, b, BQRY, D, q0, 0, bh);
    }
  };
  const int nit = nqt - qt0;
  if (tid == 0)
    for (int it = 0; it < min(p.nstage, nit); ++it) load_stage(it);

  const bool key_ok = j < p.T;
  row_to_tmem(tmem, cK, p.K, bh * p.T + j, key_ok ? (bh + 1) * p.T : 0, D, p.x3 != 0);
  if (do_dk) row_to_tmem(tmem, cV, p.V, bh * p.T + j, key_ok ? (bh + 1) * p.T : 0, D, p.x3 != 0);
  tmem_st_wait();

  const bool prob = (p.recon == REC_NEAREST && p.ste == 1 && p.calib != CAL_SOFTMAX);
  const bool minmax = p.calib == CAL_MINMAX;
  const bool fullg = p.grad == 0 && p.calib != CAL_SOFTMAX;
  bool failed = false;
  uint32_t mph = 0;
  for (int it = 0; it < nit; ++it) {
    const int q0 = (qt0 + it) * BQRY;
    // Per-query-row constants of this tile (the previous tile's readers have
    // passed the CTA barrier that closed their iteration).
    if (tid < BQRY) {
      const int iq = q0 + tid;
      const bool ok = iq < p.T;
      const size_t rw = (size_t)bh * p.T + (ok ? iq : 0);
      const float M = ok ? p.row_max[rw] : 0.f, m = ok ? p.row_min[rw] : 0.f;
      const RowGrid g = row_grid(p, M, m);
      const float Wf = ok ? p.W[rw] : 1.f;
      const float Ws = prob ? (ok ? p.W_lerp[rw] : 1.f) : Wf;
      qr->M[tid] = M;
      qr->m[tid] = m;
      qr->inv_h[tid] = g.inv_h;
      qr->c0[tid] = g.c0;
      qr->invWf[tid] = 1.0f / Wf;
      qr->invWs[tid] = 1.0f / Ws;
      qr->D[tid] = ok ? p.Drow[rw] : 0.f;
      qr->cMn[tid] = ok ? p.cMn[rw] : 0.f;
      qr->cmn[tid] = ok ? p.cmn[rw] : 0.f;
      qr->amax[tid] = ok ? p.arg_max[rw] : -1;
      qr->amin[tid] = ok ? p.arg_min[rw] : -1;
      qr->nmax[tid] = ok ? p.n_max[rw] : 1;
      qr->nmin[tid] = ok ? p.n_min[rw] : 1;
      qr->nogrid[tid] = g.nogrid ? 1 : 0;
    }
    if (p.calib != CAL_SOFTMAX) {
      // grid tables: row (tid % 64), entries r = tid/64, tid/64 + 2, ...
      const int rr = tid % BQRY, iq = q0 + rr;
      const bool ok = iq < p.T;
      const size_t rw = (size_t)bh * p.T + (ok ? iq : 0);
      const float M = ok ? p.row_max[rw] : 0.f, m = ok ? p.row_min[rw] : 0.f;
      const RowGrid g = row_grid(p, M, m);
      for (int r = tid / BQRY; r <= Kq; r += NT / BQRY) tab[rr * tstride + r] = grid_value(p, g, r);
    }
    __syncthreads();

    const uint8_t* st = stage_ptr(it);
    if (tid == 0) {
      const bool ok =
          mbar_wait(&bar_st[it % p.nstage], (it / p.nstage) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      if (ok) {
        tc_fence_after();
        if (p.x3) {
          mma_tmem_smem(tmem + cS, tmem + cK + D, st + oQ, BQRY, D, false);
          mma_tmem_smem(tmem + cS, tmem + cK, st + oQ + qtile, BQRY, D, true);
          mma_tmem_smem(tmem + cS, tmem + cK, st + oQ, BQRY, D, true);
          if (do_dk) {
            mma_tmem_smem(tmem + cG, tmem + cV + D, st + odO, BQRY, D, false);
            mma_tmem_smem(tmem + cG, tmem + cV, st + odO + qtile, BQRY, D, true);
            mma_tmem_smem(tmem + cG, tmem + cV, st + odO, BQRY, D, true);
          }
        } else {
          mma_tmem_smem(tmem + cS, tmem + cK, st + oQ, BQRY, D, false);
          if (do_dk) mma_tmem_smem(tmem + cG, tmem + cV, st + odO, BQRY, D, false);
        }
        mma_commit(bar_mma);
      }
    }
    bool ok = mbar_wait(bar_mma, mph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
    mph ^= 1;
    if (cta_any(!ok)) {
      failed = true;
      break;
    }
    tc_fence_after();
#pragma unroll 1
    for (int c = 0; c < BQRY / 32; ++c) {
      float sv[32], gv[32], pa[32], da[32];
      tmem_ld32(lane_addr(tmem, cS + c * 32), sv);
      if (do_dk) tmem_ld32(lane_addr(tmem, cG + c * 32), gv);
      tmem_ld_wait();
#pragma unroll
      for (int ii = 0; ii < 32; ++ii) {
        const int r_ = c * 32 + ii;  // query row within the tile
        const int iq = q0 + r_;
        const bool valid = key_ok && iq < p.T && iq >= j;
        float pv = 0.f, ds = 0.f;
        if (valid) {
          RowB R;
          R.M = qr->M[r_];
          R.m = qr->m[r_];
          R.g.inv_h = qr->inv_h[r_];
          R.g.k1 = __fmul_rn(p.scale, R.g.inv_h);
          R.g.c0 = qr->c0[r_];
          R.g.nogrid = qr->nogrid[r_] != 0;
          R.invWf = qr->invWf[r_];
          R.invWs = qr->invWs[r_];
          R.D = qr->D[r_];
          const float s = __fmul_rn(sv[ii], p.scale);
          KeyPos kp{0, 0, 0.f, false};
          float er = 0.f, er1 = 0.f, el = 0.f;
          if (p.calib != CAL_SOFTMAX && !R.g.nogrid) {
            kp = key_pos(p, __fmaf_rn(sv[ii], R.g.k1, R.g.c0));
            if (!kp.tail) {
              const float* t_ = tab + r_ * tstride;
              er = t_[kp.r];
              er1 = t_[kp.r + 1];
              el = t_[kp.l];
            }
          }
          const BwdElem e = bwd_elem(p, R, s, do_dk ? gv[ii] : 0.f, er, er1, el, kp);
          pv = e.p;
          ds = e.ds;
          if (fullg && !R.g.nogrid) {
            const int nM = qr->nmax[r_];
            if (nM == 1 ? (j == qr->amax[r_]) : (s == R.M)) ds += qr->cMn[r_];
            if (minmax) {
              const int nm = qr->nmin[r_];
              if (nm == 1 ? (j == qr->amin[r_]) : (s == R.m)) ds += qr->cmn[r_];
            }
          }
        }
        if (p.x3) {
          const float x = do_dv ? pv : ds;
          const float h = tf32_rna(x);
          pa[ii] = h;
          da[ii] = __fsub_rn(x, h);
        } else {
          pa[ii] = pv;
          da[ii] = ds;
        }
      }
      if (p.x3 || do_dv) tmem_st32(lane_addr(tmem, cS + c * 32), pa);
      if (p.x3 || do_dk) tmem_st32(lane_addr(tmem, cG + c * 32), da);
    }
    tmem_st_wait();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const bool acc = it > 0;
      if (p.x3) {
        // one product per launch: A_hi at cS, A_lo at cG
        const int cacc = do_dv ? cdV : cdK;
        const uint8_t* b = st + (do_dv ? odOT : oQT);
        mma_tmem_smem(tmem + cacc, tmem + cS, b, D, BQRY, acc);
        mma_tmem_smem(tmem + cacc, tmem + cS, b + qtile, D, BQRY, true);
        mma_tmem_smem(tmem + cacc, tmem + cG, b, D, BQRY, true);
      } else {
        if (do_dv) mma_tmem_smem(tmem + cdV, tmem + cS, st + odOT, D, BQRY, acc);
        if (do_dk) mma_tmem_smem(tmem + cdK, tmem + cG, st + oQT, D, BQRY, acc);
      }
      mma_commit(bar_mma);
    }
    ok = mbar_wait(bar_mma, mph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
    mph ^= 1;
    if (cta_any(!ok)) {
      failed = true;
      break;
    }
    tc_fence_after();
    if (tid == 0 && it + p.nstage < nit) load_stage(it + p.nstage);
  }

  if (!failed) {
    const size_t krow = (size_t)bh * p.T + (key_ok ? j : 0);
    for (int pass = 0; pass < 2; ++pass) {
      const bool want = pass == 0 ? do_dv : do_dk;
      if (!want) continue;
      const int col = pass == 0 ? cdV : cdK;
      const float mul = pass == 0 ? 1.0f : p.scale;
      float* dst = (pass == 0 ? p.dV : p.dK) + krow * D;
      for (int c = 0; c < D; c += 32) {
        float v[32];
        tmem_ld32(lane_addr(tmem, col + c), v);
        tmem_ld_wait();
        if (key_ok) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            reinterpret_cast<float4*>(dst + c)[q] =
                make_float4(v[4 * q] * mul, v[4 * q + 1] * mul, v[4 * q + 2] * mul, v[4 * q + 3] * mul);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

cudaError_t launch_bwd_dkdv(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_bwd_dkdv, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  k_bwd_dkdv<<<dim3((p.T + 127) / 128, p.BH), NT, smem_bytes, s>>>(maps, p);
  return cudaGetLastError();
}

}  // namespace kint
