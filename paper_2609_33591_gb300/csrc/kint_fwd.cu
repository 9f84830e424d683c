// Forward of K-interval attention on sm_103a: operand preparation, pass 1
// (row extrema) and pass 2 (grid reconstruction, normalization, P V).
//
// Two passes are needed because the grid of a row depends on its final
// extrema (Sec. 3: MinMax spans [m, M]; FWM is anchored at M), so partial
// results cannot be rescaled online the way a softmax running maximum can.
#include <cfloat>
#include "kint_dev.cuh"
#include "kint_launch.h"

namespace kint {

// ---------------------------------------------------------------------------
// Operand preparation (HBM-bound).  tcgen05.mma kind::tf32 reads both operands
// K-major, so every second-stage product (P V, dS K, P^T dO, dS^T Q) reads a
// transposed copy X^T [BH][d][Tp].  3xTF32 also needs tf32 hi/lo splits.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_prep(const float* __restrict__ X, float* __restrict__ nat_hi,
                                              float* __restrict__ nat_lo, float* __restrict__ tr_hi,
                                              float* __restrict__ tr_lo, int T, int Tp, int d, int split) {
  __shared__ float hi_s[32][33];
  __shared__ float lo_s[32][33];
  const int t0 = blockIdx.x * 32, k0 = blockIdx.y * 32, bh = blockIdx.z;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const size_t nat = (size_t)bh * T * d;
  for (int r = ty; r < 32; r += 8) {
    const int t = t0 + r;
    float x = (t < T) ? X[nat + (size_t)t * d + k0 + tx] : 0.0f;
    float lo = 0.0f;
    if (split) {
      const float h = tf32_rna(x);
      lo = __fsub_rn(x, h);
      x = h;
      if (t < T && nat_hi) {
        nat_hi[nat + (size_t)t * d + k0 + tx] = x;
        nat_lo[nat + (size_t)t * d + k0 + tx] = lo;
      }
    }
    hi_s[r][tx] = x;
    lo_s[r][tx] = lo;
  }
  __syncthreads();
  const size_t tr = (size_t)bh * d * Tp;
  for (int r = ty; r < 32; r += 8) {
    const int k = k0 + r, t = t0 + tx;  // t < Tp by construction of the grid
    if (tr_hi) tr_hi[tr + (size_t)k * Tp + t] = hi_s[tx][r];
    if (split && tr_lo) tr_lo[tr + (size_t)k * Tp + t] = lo_s[tx][r];
  }
}

cudaError_t launch_prep(const float* X, float* nat_hi, float* nat_lo, float* tr_hi, float* tr_lo, int BH, int T,
                        int Tp, int d, bool split, cudaStream_t s) {
  dim3 grid(Tp / 32, d / 32, BH), block(32, 8);
  k_prep<<<grid, block, 0, s>>>(X, nat_hi, nat_lo, tr_hi, tr_lo, T, Tp, d, split ? 1 : 0);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Pass 1: row extrema (App. A: M = max_j s_j, m = min_j s_j over valid keys,
// lowest index among ties and the tie counts of Table "Edge cases").
// CTA = one 128-row query block of one head; thread t owns query row
// qb*128 + t, which is TMEM lane t of the score tile S = Q K^T (M = N = 128).
// Thread 0 issues TMA and MMA; S is double-buffered in TMEM so the product of
// key tile kb+1 runs while tile kb is reduced.
// smem: Q tile (hi[, lo]) at sm_a; nstage key stages (K hi[, lo]).
// TMEM: S buffers at columns [0,128) and [128,256).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(NT, 1) k_fwd_stats(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  const int D = p.d, tile = D * 512, parts = p.x3 ? 2 : 1;
  uint8_t* sQ = sm + p.sm_a;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_q = bars;
  uint64_t* bar_st = bars + 1;               // [nstage]
  uint64_t* bar_mma = bars + 1 + p.nstage;   // [2], one per S buffer
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 3 + p.nstage);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int bh = blockIdx.y, qb = p.nqb - 1 - blockIdx.x;
  const int i = qb * 128 + tid;
  const int nkb = qb + 1;

  if (tid == 0) {
    mbar_init(bar_q, 1);
    for (int s = 0; s < p.nstage; ++s) mbar_init(&bar_st[s], 1);
    mbar_init(&bar_mma[0], 1);
    mbar_init(&bar_mma[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  auto stage_ptr = [&](int kb) { return sm + p.sm_stage0 + (kb % p.nstage) * p.sm_stage_bytes; };
  auto load_k = [&](int kb) {
    uint64_t* b = &bar_st[kb % p.nstage];
    uint8_t* dst = stage_ptr(kb);
    mbar_arrive_expect_tx(b, parts * tile);
    load_rows_tile(dst, &maps.k, b, D, 128, 0, kb * 128, bh);
    if (p.x3) load_rows_tile(dst + tile, &maps.k_lo, b, D, 128, 0, kb * 128, bh);
  };
  // Thread 0: wait for key tile kb and issue S[kb & 1] = Q K_kb^T.
  auto issue_s = [&](int kb) -> bool {
    if (kb == 0 && !mbar_wait(bar_q, 0, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) return false;
    if (!mbar_wait(&bar_st[kb % p.nstage], (kb / p.nstage) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA))
      return false;
    tc_fence_after();
    const uint8_t* sk = stage_ptr(kb);
    const uint32_t dcol = tmem + (kb & 1) * 128;
    if (p.x3) {
      mma_smem_smem(dcol, sQ + tile, sk, 128, D, false);  // Q_lo K_hi
      mma_smem_smem(dcol, sQ, sk + tile, 128, D, true);   // Q_hi K_lo
      mma_smem_smem(dcol, sQ, sk, 128, D, true);          // Q_hi K_hi
    } else {
      mma_smem_smem(dcol, sQ, sk, 128, D, false);
    }
    mma_commit(&bar_mma[kb & 1]);
    return true;
  };

  if (tid == 0) {
    mbar_arrive_expect_tx(bar_q, parts * tile);
    load_rows_tile(sQ, &maps.q, bar_q, D, 128, 0, qb * 128, bh);
    if (p.x3) load_rows_tile(sQ + tile, &maps.q_lo, bar_q, D, 128, 0, qb * 128, bh);
    for (int kb = 0; kb < min(p.nstage, nkb); ++kb) load_k(kb);
    issue_s(0);
  }

  float M = -FLT_MAX, m = FLT_MAX;
  int amax = 0, amin = 0, nmax = 0, nmin = 0;
  bool failed = false;
  for (int kb = 0; kb < nkb; ++kb) {
    if (tid == 0 && kb + 1 < nkb) {
      // S[(kb+1)&1] was last read in iteration kb-1 (closed by a CTA barrier).
      // Its key tile sits in stage (kb+1)%nstage; with one stage that stage is
      // refilled below only after S[kb] completed, so wait for it here first.
      if (p.nstage == 1) {
        // single stage: tile kb+1 is loaded after MMA kb completes (below)
      } else {
        issue_s(kb + 1);
      }
    }
    const bool ok = mbar_wait(&bar_mma[kb & 1], (kb >> 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
    if (cta_any(!ok)) {
      failed = true;
      break;
    }
    tc_fence_after();
    if (tid == 0) {
      if (kb + p.nstage < nkb) load_k(kb + p.nstage);  // this stage's product has completed
      if (p.nstage == 1 && kb + 1 < nkb) issue_s(kb + 1);
    }
    const uint32_t scol = (kb & 1) * 128;
#pragma unroll 1
    for (int c = 0; c < 4; ++c) {
      float v[32];
      tmem_ld32(lane_addr(tmem, scol + c * 32), v);
      tmem_ld_wait();
      const int j0 = kb * 128 + c * 32;
#pragma unroll
      for (int jj = 0; jj < 32; ++jj) {
        const int j = j0 + jj;
        if (j <= i) {
          const float sc = __fmul_rn(v[jj], p.scale);
          if (sc > M) {
            M = sc;
            amax = j;
            nmax = 1;
          } else if (sc == M) {
            ++nmax;
          }
          if (sc < m) {
            m = sc;
            amin = j;
            nmin = 1;
          } else if (sc == m) {
            ++nmin;
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
  }
  if (!failed && i < p.T) {
    const size_t row = (size_t)bh * p.T + i;
    p.row_max[row] = M;
    p.row_min[row] = m;
    p.arg_max[row] = amax;
    p.arg_min[row] = amin;
    p.n_max[row] = nmax;
    p.n_min[row] = nmin;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

cudaError_t launch_fwd_stats(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_fwd_stats, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  k_fwd_stats<<<dim3(p.nqb, p.BH), NT, smem_bytes, s>>>(maps, p);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Pass 2: per key, the grid position u, the decisions (r, t, l, tail) and the
// reconstructed weight (App. A "LERP": w^L = (1-t) e_r + t e_{r+1};
// "Nearest": w^N = e_l; FWM tail: 0), by shared-memory table lookup and FMA in
// place of the exponential; W = sum w; O = (sum_j w_j V_j) / W.
// TMEM: S / A (weights as MMA operand A) at [0,128); A2 (second weights, or
// the lo part of A under 3xTF32) at [128,256); O at [256, 256+d); O_lerp at
// [256+d, 256+2d).
// smem: Q (hi[, lo]) at sm_a; stages {K tile, V^T tile} (hi[, lo] each);
// per-thread grid table [K+1][128] fp32 at sm_table.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(NT, 1) k_fwd_main(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1;
  const int qtile = D * 512;       // [128 x D]
  const int vtile = D * 512;       // [D x 128] transposed
  uint8_t* sQ = sm + p.sm_a;
  float* tab = reinterpret_cast<float*>(sm + p.sm_table);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_q = bars;
  uint64_t* bar_st = bars + 1;
  uint64_t* bar_mma = bars + 1 + p.nstage;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2 + p.nstage);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int bh = blockIdx.y, qb = p.nqb - 1 - blockIdx.x;
  const int i = qb * 128 + tid;
  const bool row_ok = i < p.T;
  const int nkb = qb + 1;
  const bool nearest = p.recon == REC_NEAREST;
  const int sel = p.pv_sel;

  if (tid == 0) {
    mbar_init(bar_q, 1);
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

  auto stage_ptr = [&](int kb) { return sm + p.sm_stage0 + (kb % p.nstage) * p.sm_stage_bytes; };
  auto load_kv = [&](int kb) {
    uint64_t* b = &bar_st[kb % p.nstage];
    uint8_t* dst = stage_ptr(kb);
    mbar_arrive_expect_tx(b, parts * (qtile + vtile));
    load_rows_tile(dst, &maps.k, b, D, 128, 0, kb * 128, bh);
    load_rows_tile(dst + parts * qtile, &maps.vt, b, 128, D, kb * 128, 0, bh);
    if (p.x3) {
      load_rows_tile(dst + qtile, &maps.k_lo, b, D, 128, 0, kb * 128, bh);
      load_rows_tile(dst + parts * qtile + vtile, &maps.vt_lo, b, 128, D, kb * 128, 0, bh);
    }
  };
  if (tid == 0) {
    mbar_arrive_expect_tx(bar_q, parts * qtile);
    load_rows_tile(sQ, &maps.q, bar_q, D, 128, 0, qb * 128, bh);
    if (p.x3) load_rows_tile(sQ + qtile, &maps.q_lo, bar_q, D, 128, 0, qb * 128, bh);
    for (int kb = 0; kb < min(p.nstage, nkb); ++kb) load_kv(kb);
  }

  // Row set-up: extrema from pass 1, grid, per-thread table of e_r.
  const size_t row = (size_t)bh * p.T + (row_ok ? i : 0);
  const float M = row_ok ? p.row_max[row] : 0.0f;
  const float m = row_ok ? p.row_min[row] : 0.0f;
  const RowGrid g = row_grid(p, M, m);
  if (p.calib != CAL_SOFTMAX)
    for (int r = 0; r <= Kq; ++r) tab[r * NT + tid] = grid_value(p, g, r);

  float Wm = 0.0f, Wl = 0.0f;
  bool failed = false;
  uint32_t mph = 0;
  for (int kb = 0; kb < nkb; ++kb) {
    const uint8_t* st = stage_ptr(kb);
    if (tid == 0) {
      bool ok = (kb > 0 || mbar_wait(bar_q, 0, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) &&
                mbar_wait(&bar_st[kb % p.nstage], (kb / p.nstage) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      if (ok) {
        tc_fence_after();
        if (p.x3) {
          mma_smem_smem(tmem, sQ + qtile, st, 128, D, false);
          mma_smem_smem(tmem, sQ, st + qtile, 128, D, true);
          mma_smem_smem(tmem, sQ, st, 128, D, true);
        } else {
          mma_smem_smem(tmem, sQ, st, 128, D, false);
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
    for (int c = 0; c < 4; ++c) {
      float v[32], a1[32], a2[32];
      tmem_ld32(lane_addr(tmem, c * 32), v);
      tmem_ld_wait();
      const int j0 = kb * 128 + c * 32;
      float wm_part = 0.0f, wl_part = 0.0f;
#pragma unroll
      for (int jj = 0; jj < 32; ++jj) {
        const int j = j0 + jj;
        const bool valid = row_ok && j <= i;
        const float s = __fmul_rn(v[jj], p.scale);
        float wmain = 0.0f, wlerp = 0.0f;
        uint8_t cb = 255, ci = 255;
        if (valid) {
          if (p.calib == CAL_SOFTMAX) {
            wmain = expf(__fsub_rn(s, M));
            cb = ci = 253;
          } else if (g.nogrid) {
            wmain = wlerp = 1.0f;
            cb = ci = 253;
          } else {
            const KeyPos kp = key_pos(p, __fmaf_rn(s, g.inv_h, g.c0));
            if (kp.tail) {
              cb = ci = 254;
            } else {
              const float er = tab[kp.r * NT + tid];
              const float er1 = tab[(kp.r + 1) * NT + tid];
              wlerp = __fmaf_rn(kp.t, __fsub_rn(er1, er), er);
              wmain = nearest ? tab[kp.l * NT + tid] : wlerp;
              cb = (uint8_t)kp.l;
              ci = (uint8_t)kp.r;
            }
          }
        }
        wm_part += wmain;
        wl_part += wlerp;
        const float a = (sel == PV_LERP) ? wlerp : wmain;
        if (p.x3) {
          const float h = tf32_rna(a);
          a1[jj] = h;
          a2[jj] = __fsub_rn(a, h);
        } else {
          a1[jj] = a;
          a2[jj] = wlerp;
        }
        if (p.debug && row_ok && j < p.T) {
          const size_t idx = ((size_t)bh * p.T + i) * p.T + j;
          if (p.bins) p.bins[idx] = cb;
          if (p.ivals) p.ivals[idx] = ci;
        }
      }
      Wm += wm_part;
      Wl += wl_part;
      tmem_st32(lane_addr(tmem, c * 32), a1);
      if (p.x3 || sel == PV_MAIN_LERP) tmem_st32(lane_addr(tmem, 128 + c * 32), a2);
    }
    tmem_st_wait();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint8_t* vt = st + parts * qtile;
      const bool acc = kb > 0;
      if (p.x3) {
        mma_tmem_smem(tmem + 256, tmem + 0, vt, D, 128, acc);            // A_hi V_hi
        mma_tmem_smem(tmem + 256, tmem + 0, vt + vtile, D, 128, true);   // A_hi V_lo
        mma_tmem_smem(tmem + 256, tmem + 128, vt, D, 128, true);         // A_lo V_hi
      } else {
        mma_tmem_smem(tmem + 256, tmem + 0, vt, D, 128, acc);
        if (sel == PV_MAIN_LERP) mma_tmem_smem(tmem + 256 + D, tmem + 128, vt, D, 128, acc);
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
    if (tid == 0 && kb + p.nstage < nkb) load_kv(kb + p.nstage);
  }

  if (!failed && !p.debug) {
    // Normalization (App. A): O = (sum_j w_j V_j) / W.  Every lane runs the
    // warp-collective TMEM loads; only rows < T store.
    const float Wout = (sel == PV_LERP) ? Wl : Wm;
    const float inv = row_ok ? 1.0f / Wout : 0.0f;
    float* dst = (sel == PV_LERP ? p.O_lerp : p.Out) + row * D;
    for (int c = 0; c < D; c += 32) {
      float v[32];
      tmem_ld32(lane_addr(tmem, 256 + c), v);
      tmem_ld_wait();
      if (row_ok) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          reinterpret_cast<float4*>(dst + c)[q] =
              make_float4(v[4 * q] * inv, v[4 * q + 1] * inv, v[4 * q + 2] * inv, v[4 * q + 3] * inv);
      }
    }
    if (sel == PV_MAIN_LERP) {
      const float invl = row_ok ? 1.0f / Wl : 0.0f;
      float* dl = p.O_lerp + row * D;
      for (int c = 0; c < D; c += 32) {
        float v[32];
        tmem_ld32(lane_addr(tmem, 256 + D + c), v);
        tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            reinterpret_cast<float4*>(dl + c)[q] =
                make_float4(v[4 * q] * invl, v[4 * q + 1] * invl, v[4 * q + 2] * invl, v[4 * q + 3] * invl);
        }
      }
    }
    if (row_ok) {
      if (sel != PV_LERP) p.W[row] = Wm;
      if (sel != PV_MAIN && p.W_lerp) p.W_lerp[row] = Wl;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

cudaError_t launch_fwd_main(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_fwd_main, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  k_fwd_main<<<dim3(p.nqb, p.BH), NT, smem_bytes, s>>>(maps, p);
  return cudaGetLastError();
}

}  // namespace kint
