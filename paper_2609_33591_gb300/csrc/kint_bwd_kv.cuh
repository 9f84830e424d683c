// dK/dV kernel of the backward (App. B), as a template: included by the
// translation unit of the plain kernels and by the one of the kernels that also
// accumulate the per-row score-gradient sums (RS), so the two compile in parallel.
#pragma once
#include "kint_bwd_common.cuh"

namespace kint {

// ---------------------------------------------------------------------------
// dK/dV kernel element work on one 32-query chunk of one key j: the forward
// probability P_ij and dS_ij = gamma_ij Delta_ij plus, at the arg-max / arg-min
// key of row i, c_M / n_max and c_m / n_min (Eq. full).  Row constants come
// from the RowRec array of the tile in shared memory (broadcast loads).
// ---------------------------------------------------------------------------
template <int CAL, int REC, bool FULLG, bool PROJ, bool MASKED, bool TIES, int W>
__device__ __forceinline__ void kv_chunk(const float (&sv)[W], const float (&gv)[W], float (&pa)[W],
                                         float (&da)[W], int j, int i0, int T, uint32_t recs, uint32_t tabs,
                                         uint32_t fwtab, uint32_t tstride, float Kf, float fwm_inv_h,
                                         float scale, float hl, float b0l) {
#pragma unroll
  for (int ii = 0; ii < W; ++ii) {
    const uint32_t ra = recs + ii * 64u;  // RowRec of query row i0 + ii
    const float4 r0 = lds_f4(ra);          // c0, k1, invWf, ga
    const float4 r1 = lds_f4(ra + 16);     // gb, cMn, amax, flags
    float4 r2 = make_float4(0.f, 0.f, 0.f, 0.f);
    if constexpr (CAL == CAL_MINMAX) r2 = lds_f4(ra + 32);  // inv_h, cmn, amin, -
    const float gam = __fmaf_rn(gv[ii], r0.w, r1.x);
    float pv, ds;
    if constexpr (CAL == CAL_SOFTMAX) {
      pv = ex2_approx(__fmaf_rn(sv[ii], r0.y, r0.x)) * r0.z;
      ds = pv * gam;
    } else if constexpr (CAL == CAL_EXP8) {
      // forward P from the E4M3-rounded weight; dS from the exponential itself
      const float we = ex2_approx(__fmaf_rn(sv[ii], r0.y, r0.x));
      pv = e4m3_rn(we) * r0.z;
      ds = gam * we;
    } else if constexpr (CAL == CAL_EXPB) {
      // record holds -M, scale: z = acc * scale - M; the bfloat16 chain rule
      float zb;
      const float w = bf16_exp_weight(__fadd_rn(__fmul_rn(sv[ii], r0.y), r0.x), zb);
      pv = w * r0.z;
      ds = bf16_rn(__fmul_rn(bf16_rn(gam), w));
    } else if constexpr (fwm_like(CAL) && REC == REC_NEAREST) {
      // record holds 2k1, 2c0; Kf = 2K; fwtab: the half-bin table of (w^N, Delta_r / h)
      const float v = __fmaf_rn(sv[ii], r0.y, r0.x);
      const uint32_t qb = fwm_half_bits(v, Kf);
      float2 e = lds_f2(fwtab + qb * 8u);
      if constexpr (CAL == CAL_FWMR) {
        // resolved: below the window, (w^N, Delta_r / h) of the continued grid (u = v / 2 exactly)
        const BelowPair bp = resolved_below(__fmul_rn(v, 0.5f), hl, b0l);
        const float2 eb = make_float2(bp.t >= 0.5f ? bp.e1 : bp.e0, __fmul_rn(__fsub_rn(bp.e1, bp.e0), fwm_inv_h));
        e = v < 0.0f ? eb : e;
      }
      pv = e.x * r0.z;
      ds = gam * e.y;
    } else {
      const float u = __fmaf_rn(sv[ii], r0.y, r0.x);
      float t, rf;
      uint32_t rb;
      decode_u(u, Kf, t, rb, rf);
      float2 e = lds_f2(fwm_like(CAL) ? fwtab + rb * 8u : tabs + ii * tstride + rb * 8u);
      if constexpr (CAL == CAL_FWMR) {
        const BelowPair bp = resolved_below(u, hl, b0l);
        const bool below = u < 0.0f;
        t = below ? bp.t : t;
        e = below ? make_float2(bp.e0, bp.e1) : e;
      }
      const float de = __fsub_rn(e.y, e.x);
      const float wl = __fmaf_rn(t, de, e.x);
      const float wn = (t >= 0.5f) ? e.y : e.x;
      float w = (REC == REC_NEAREST) ? wn : wl;
      ds = gam * (de * (CAL == CAL_MINMAX ? r2.x : fwm_inv_h));
      if constexpr (CAL == CAL_FWM) {
        const bool tail = u < 0.0f;
        w = tail ? 0.f : w;
        ds = tail ? 0.f : ds;
      }
      if constexpr (CAL == CAL_MINMAX) {
        const bool ng = (__float_as_int(r1.w) & REC_NOGRID) != 0;
        w = ng ? 1.f : w;
        ds = ng ? 0.f : ds;
      }
      pv = w * r0.z;
    }
    if constexpr (FULLG && CAL != CAL_SOFTMAX) {
      ds += (j == __float_as_int(r1.z)) ? r1.y : 0.f;
      if constexpr (CAL == CAL_MINMAX) ds += (j == __float_as_int(r2.z)) ? r2.y : 0.f;
    } else if constexpr (PROJ && CAL != CAL_SOFTMAX) {
      ds = __fsub_rn(ds, r1.y);  // detached, P1 projection: minus the row mean
    }
    if constexpr (MASKED) {
      const int iq = i0 + ii;
      const bool ok = iq >= j && iq < T;
      pv = ok ? pv : 0.f;
      ds = ok ? ds : 0.f;
    }
    if constexpr (FULLG && TIES && CAL != CAL_SOFTMAX) {
      // rows with tied extrema (flagged per 64-row query tile by the dQ kernel): the tie set
      // is found by equality on the recomputed scores (rare, kept off the common path)
      const int fl = __float_as_int(r1.w);
      const int iq = i0 + ii;
      const bool okr = (!MASKED || (iq >= j && iq < T)) && (fl & (REC_TIEMAX | REC_TIEMIN)) && !(fl & REC_NOGRID);
      if (okr) {
        const float2 ext = lds_f2(ra + 48);  // M, m
        const float sc = __fmul_rn(sv[ii], scale);
        if ((fl & REC_TIEMAX) && sc == ext.x) ds += r1.y;
        if (CAL == CAL_MINMAX && (fl & REC_TIEMIN) && sc == ext.y) ds += r2.y;
      }
    }
    pa[ii] = pv;
    da[ii] = ds;
  }
}

// Per-row score-gradient sums (a diagnostic side output of the backward): the calling
// warp holds dS for 16 query rows (v[c], row r0 + c) at 32 keys (one per lane).  A
// butterfly reduce-scatter leaves the 32-key sum of row c = (lane >> 1) & 15 in lanes
// 2c and 2c + 1 (the xor-16 step keeps rows 8..15 in the upper half-warp, xor-8 rows
// +4, xor-4 rows +2, xor-2 rows +1, and xor-1 adds the pair); the even lane adds it to
// the row's global sums (fp32 atomics: the order of the additions is not fixed).
__device__ __forceinline__ void rowsum_add(const float (&v)[16], float* dsum, float* dabs, size_t r0, int nvalid) {
  const int lane = threadIdx.x & 31;
  float s[16], a[16];
#pragma unroll
  for (int c = 0; c < 16; ++c) {
    s[c] = v[c];
    a[c] = fabsf(v[c]);
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1) {
    const bool up = (lane & (2 * w)) != 0;
#pragma unroll
    for (int k = 0; k < w; ++k) {
      const float ss = up ? s[k] : s[k + w], sa = up ? a[k] : a[k + w];
      const float ks = up ? s[k + w] : s[k], ka = up ? a[k + w] : a[k];
      s[k] = ks + __shfl_xor_sync(0xffffffffu, ss, 2 * w);
      a[k] = ka + __shfl_xor_sync(0xffffffffu, sa, 2 * w);
    }
  }
  s[0] += __shfl_xor_sync(0xffffffffu, s[0], 1);
  a[0] += __shfl_xor_sync(0xffffffffu, a[0], 1);
  const int c = (lane >> 1) & 15;
  if ((lane & 1) == 0 && c < nvalid) {
    if (dsum) atomicAdd(dsum + r0 + c, s[0]);
    if (dabs) atomicAdd(dabs + r0 + c, a[0]);
  }
}

// MMA thread of k_bwd_dkdv: wait for the query tile in stage st (ring position), then
// S^T_b = K Q^T and (dK launches) g^T_b = V dO^T into score buffer b.
__device__ __forceinline__ bool kv_issue_sg(const Params& p, RingPos stg, int b, uint64_t* bar_full,
                                            uint64_t* bar_sfull, const uint8_t* st0, uint32_t cKa, uint32_t cVa,
                                            uint32_t cSG, int qtile, bool needV, int oQ, int odO) {
  const int D = p.d, s = stg.i;
  if (!mbar_wait_warp(&bar_full[s], stg.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) return false;
  tc_fence_after();
  const uint8_t* st = st0 + s * p.sm_stage_bytes;
  const uint32_t cS = cSG + 128 * b, cG = cS + 64;
  if (p.x3) {
    mma_tmem_smem(cS, cKa + D, st + oQ, BT, D, false);
    mma_tmem_smem(cS, cKa, st + oQ + qtile, BT, D, true);
    mma_tmem_smem(cS, cKa, st + oQ, BT, D, true);
    if (needV) {
      mma_tmem_smem(cG, cVa + D, st + odO, BT, D, false);
      mma_tmem_smem(cG, cVa, st + odO + qtile, BT, D, true);
      mma_tmem_smem(cG, cVa, st + odO, BT, D, true);
    }
  } else {
    mma_tmem_smem(cS, cKa, st + oQ, BT, D, false);
    if (needV) mma_tmem_smem(cG, cVa, st + odO, BT, D, false);
  }
  mma_commit(&bar_sfull[b]);
  return true;
}

// Producer warp of k_bwd_dkdv: TMA-stores the dV / dK tiles of its k-th item, which the
// compute warps staged at `tile` (dV, then dK), and returns once they have been read out.
__device__ __forceinline__ bool store_staged_dkdv(const Maps& maps, const Params& p, uint64_t* bar_ostg, int k,
                                                  const uint8_t* tile, bool doDV, bool doDK) {
  if (!mbar_wait_warp(bar_ostg, k & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) return false;
  const int item = snake_item(k), kb = item / p.BH, bh = item % p.BH;
  if (doDV) store_rows_tile_boxed(tile, &maps.dv, p.d, 64, kb * 128, bh, false);
  if (doDK) store_rows_tile_boxed(tile + 128 * p.d * 4, &maps.dk, p.d, 64, kb * 128, bh, false);
  tma_store_wait_read();
  return true;
}

// ---------------------------------------------------------------------------
// k_bwd_dkdv.  Thread t (< 256) owns key j = kb*128 + t%128 and the query half
// t/128 of each 64-query tile.  TMEM: K [0, dp), V [dp, 2dp) (dK launches),
// then per buffer b: S^T_b (64 columns) and g^T_b (64 columns) from `base`,
// dV, dK.  P^T overwrites S^T_b and dS^T overwrites g^T_b (3xTF32: the single
// product's hi part goes to S^T_b, its lo part to g^T_b).
// smem stage: Q | dO | Q^T | dO^T tiles (hi[, lo]), the 64 RowRecs of the tile,
// and (MinMax) their grid pair tables; FWM's shared table at sm_table.
// ---------------------------------------------------------------------------
template <int CAL, int REC, bool FULLG, bool PROJ = false, bool RS = false>
__global__ void __launch_bounds__(NTHR, 1) k_bwd_dkdv(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  if (p.gate != nullptr) {
    // launched on one side of a device-side decision: when the single-pass backward ran
    // instead, leave before any set-up (no barrier, no tensor memory)
    pdl_wait();
    if (gated_off(p)) return;
  }
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1, NS = p.nstage, nbuf = p.nbuf;
  const int qtile = BT * D * 4;
  const bool doDV = p.dkv_sel != DKV_DK, doDK = p.dkv_sel != DKV_DV, needV = doDK;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_full = bars;
  uint64_t* bar_empty = bars + NS;
  uint64_t* bar_sfull = bars + 2 * NS;
  uint64_t* bar_pready = bars + 2 * NS + 2;
  uint64_t* bar_done = bars + 2 * NS + 4;
  uint64_t* bar_ops = bars + 2 * NS + 5;  // K / V rows stored in TMEM by every compute warp
  uint64_t* bar_stg = bars + 2 * NS + 6;   // K / V tiles staged in smem by TMA
  uint64_t* bar_ostg = bars + 2 * NS + 7;  // an item's dV / dK tiles staged in the K / V area
  // a stage's transposed tiles (Q^T, dO^T) complete on their own barrier, so the products
  // S^T, g^T wait only for the first half of the stage's bytes
  uint64_t* bar_fullT = bars + 2 * NS + 8;  // [NS]
  // the first half of a stage (Q, dO, row records) is free once the compute warps are done
  // with the tile (S^T, g^T completed before they started); the transposed half once the
  // products dV, dK that read it complete (bar_empty)
  uint64_t* bar_emptyA = bars + 3 * NS + 8;  // [NS]
  uint64_t* bar_drain = bars + 4 * NS + 8;   // the MMA warp's clean-up commit
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4 * NS + 9);
  const int tid = threadIdx.x, warp = warp_id_uniform();
  const int dp = D * parts;
  const int cK = 0, cV = dp, base = needV ? 2 * dp : dp;
  const int cdV = base + 128 * nbuf, cdK = cdV + (doDV ? D : 0);
  // 3xTF32 (one product per launch): the two cross terms accumulate apart from hi x hi.
  // The tensor core rounds each accumulation step toward zero, so a dK / dV row summed
  // over a whole causal column (up to T / 8 x 3 steps) drifts by about one unit in the
  // last place per step; keeping the cross terms out of the main accumulator cuts its
  // steps by three, and the two sums meet in fp32 in the epilogue.
  const int cdC = cdK + (doDK ? D : 0);
  const int nqt = (p.T + BT - 1) / BT;
  const int oQ = 0, odO = parts * qtile, oQT = 2 * parts * qtile, odOT = 3 * parts * qtile;
  const int oRec = 4 * parts * qtile, oTab = oRec + BT * 64;
  const uint32_t tstride = (uint32_t)p.Kp * 8u;
  constexpr int W = BT / NCG;  // query columns per thread per tile
  constexpr int WS = 16;       // columns per register chunk

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_fullT[s], 1);
      mbar_init(&bar_empty[s], 1);
      mbar_init(&bar_emptyA[s], NCOMP / 32);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar_sfull[b], 1);
      mbar_init(&bar_pready[b], NCOMP / 32);
    }
    mbar_init(bar_done, 1);
    mbar_init(bar_ops, NCOMP / 32);
    mbar_init(bar_stg, 1);
    mbar_init(bar_ostg, NCOMP / 32);
    mbar_init(bar_drain, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_trigger();
  pdl_wait();  // everything below may read what the previous kernel wrote
  // All 512 columns are allocated, so the allocation starts at lane 0, column 0; a
  // compile-time base keeps the TMEM addresses of the issue paths in uniform registers.
  if (threadIdx.x == 0 && *tslot != 0u) dev_flag(p.status, DEV_ERR_BOUNDS);
  constexpr uint32_t tmem = 0;

  // Work items are (128-key block kb, head) pairs, longest first (kb = 0 meets every
  // query tile); a CTA takes the items snake_item(0), snake_item(1), ...  Tile counters
  // (stage ring, score buffers) run on across items.
  if (warp == PRODUCER_WARP) {
    int gt = 0, n = 0;
    RingPos ld;  // stage of the next tile loaded
    RingPos nf, nT;  // ring positions after the last first-half and transposed-half loads issued
    int cf = 0, cT = 0;  // how many of each were issued
    bool ok = true;
    // K / V of this CTA's k-th item into the staging area (TF32 at d = 64)
    int staged = 0;  // staging loads issued
    auto stage_ops = [&](int k) {
      const int it_ = snake_item(k), kb_ = it_ / p.BH, bh_ = it_ % p.BH;
      mbar_arrive_expect_tx(bar_stg, (needV ? 2 : 1) * 128 * D * 4);
      load_rows_tile_boxed(sm + p.sm_a, &maps.k, bar_stg, D, 128, BT, 0, kb_ * 128, bh_);
      if (needV) load_rows_tile_boxed(sm + p.sm_a + 128 * D * 4, &maps.v, bar_stg, D, 128, BT, 0, kb_ * 128, bh_);
      staged = k + 1;
    };
    if (p.ops_smem && snake_item(0) < p.nitems) stage_ops(0);
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int kb = item / p.BH, bh = item % p.BH;
      const int qt0 = (kb * 128) / BT, nit = nqt - qt0;
      for (int it = 0; it < nit; ++it, ++gt, ld.next(NS)) {
        const int s = ld.i, q0 = (qt0 + it) * BT;
        if (gt >= NS && !mbar_wait_warp(&bar_emptyA[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        // first the operands of S^T, g^T and the row records, then the transposed tiles
        uint64_t* b = &bar_full[s];
        const int nrows = min(BT, p.T - q0);
        uint32_t bytes = (1 + (needV ? 1 : 0)) * parts * qtile + nrows * 64;
        if (CAL == CAL_MINMAX) bytes += nrows * tstride;
        mbar_arrive_expect_tx(b, bytes);
        load_rows_tile(dst + oQ, &maps.q, b, D, BT, 0, q0, bh);
        if (p.x3) load_rows_tile(dst + oQ + qtile, &maps.q_lo, b, D, BT, 0, q0, bh);
        if (needV) {
          load_rows_tile(dst + odO, &maps.dout, b, D, BT, 0, q0, bh);
          if (p.x3) load_rows_tile(dst + odO + qtile, &maps.dout_lo, b, D, BT, 0, q0, bh);
        }
        const size_t r0 = (size_t)bh * p.T + q0;
        bulk_load(dst + oRec, reinterpret_cast<const RowRec*>(p.rec) + r0, nrows * 64, b);
        if (CAL == CAL_MINMAX) bulk_load(dst + oTab, p.rtab + r0 * p.Kp * 2, nrows * tstride, b);
        nf.next(NS);
        ++cf;
        if (gt >= NS && !mbar_wait_warp(&bar_empty[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        uint64_t* bt = &bar_fullT[s];
        mbar_arrive_expect_tx(bt, ((doDK ? 1 : 0) + (doDV ? 1 : 0)) * parts * qtile);
        if (doDK) {
          load_rows_tile(dst + oQT, &maps.qt, bt, BT, D, q0, 0, bh);
          if (p.x3) load_rows_tile(dst + oQT + qtile, &maps.qt_lo, bt, BT, D, q0, 0, bh);
        }
        if (doDV) {
          load_rows_tile(dst + odOT, &maps.dot, bt, BT, D, q0, 0, bh);
          if (p.x3) load_rows_tile(dst + odOT + qtile, &maps.dot_lo, bt, BT, D, q0, 0, bh);
        }
        nT.next(NS);
        ++cT;
        // The next item's K / V, as soon as the stage ring holds this item's first tiles: it needs
        // this item's K / V copied out into TMEM and the previous item's dV / dK tiles, staged in
        // the same area since, stored; both happen at the end of the previous item, so the load
        // has this whole item to land.
        if (p.ops_smem && it == min(nit, NS) - 1 && snake_item(n + 1) < p.nitems) {
          if (!mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) ||
              (n >= 1 && !store_staged_dkdv(maps, p, bar_ostg, n - 1, sm + p.sm_a, doDV, doDK))) {
            ok = false;
            break;
          }
          stage_ops(n + 1);
        }
      }
    }
    // the last-but-one item's tiles (the last item's are stored by the compute warps)
    if (p.ops_smem && ok && n >= 2) store_staged_dkdv(maps, p, bar_ostg, n - 2, sm + p.sm_a, doDV, doDK);
    tma_store_wait_all();
    // clean-up: the last tiles issued have landed
    drain_ring(bar_full, nf, cf, NS, p.wait_ns, p.status);
    drain_ring(bar_fullT, nT, cT, NS, p.wait_ns, p.status);
    if (staged > 0) mbar_wait_warp(bar_stg, (staged - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
  } else if (warp == MMA_WARP) {
    const uint8_t* st0 = sm + p.sm_stage0;
    const uint32_t cKa = tmem + cK, cVa = tmem + cV, cSG = tmem + base;
    int n = 0;
    RingPos is, ib, cs, cb;  // stage / buffer of the next S^T, g^T product and of the tile being finished
    bool ok = true;
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int kb = item / p.BH, nit = nqt - (kb * 128) / BT;
      // K / V of the item in TMEM (the compute warps copy them only after the previous
      // item's last S, g were read)
      ok = mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC);
      if (ok) tc_fence_after();
      ok = ok && kv_issue_sg(p, is, ib.i, bar_full, bar_sfull, st0, cKa, cVa, cSG, qtile, needV, oQ, odO);
      is.next(NS);
      ib.next(nbuf);
      for (int it = 0; it < nit && ok; ++it, cs.next(NS), cb.next(nbuf)) {
        const int b = cb.i, s = cs.i;
        if (nbuf == 2 && it + 1 < nit) {
          ok = kv_issue_sg(p, is, ib.i, bar_full, bar_sfull, st0, cKa, cVa, cSG, qtile, needV, oQ, odO);
          is.next(NS);
          ib.next(nbuf);
        }
        if (!ok) break;
        if (!mbar_wait_warp(&bar_pready[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) ||
            !mbar_wait_warp(&bar_fullT[s], cs.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* st = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        const uint32_t cS = tmem + base + 128 * b, cG = cS + 64;
        const bool acc = it > 0;
        if (p.x3) {
          const uint32_t cacc = tmem + (doDV ? cdV : cdK);
          const uint8_t* bt = st + (doDV ? odOT : oQT);
          mma_tmem_smem(cacc, cS, bt, D, BT, acc);                   // hi x hi
          mma_tmem_smem(tmem + cdC, cS, bt + qtile, D, BT, acc);     // hi x lo
          mma_tmem_smem(tmem + cdC, cG, bt, D, BT, true);            // lo x hi
        } else {
          if (doDV) mma_tmem_smem(tmem + cdV, cS, st + odOT, D, BT, acc);
          if (doDK) mma_tmem_smem(tmem + cdK, cG, st + oQT, D, BT, acc);
        }
        mma_commit(&bar_empty[s]);
        if (nbuf == 1 && it + 1 < nit) {
          ok = kv_issue_sg(p, is, ib.i, bar_full, bar_sfull, st0, cKa, cVa, cSG, qtile, needV, oQ, odO);
          is.next(NS);
          ib.next(nbuf);
        }
      }
      mma_commit(bar_done);
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else {
    const int row = tid & 127, cg = (tid >> 7) & (NCG - 1);
    // K / V rows of the n-th item into TMEM (column group 0 takes K, group 1 takes V),
    // handed to the MMA warp through bar_ops: TF32 at d = 64 from the tiles the producer
    // staged in smem, otherwise from global rows.  The next item's rows go in as soon as
    // the current item's last S^T, g^T have been read, so its first products run under
    // the current item's epilogue.
    auto ops_to_tmem = [&](int n) {
      const int item = snake_item(n), kb = item / p.BH, bh = item % p.BH, j = kb * 128 + row;
      if (p.ops_smem) {
        if (mbar_wait(bar_stg, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA) && (cg == 0 || needV))
          staged_row_to_tmem(tmem, cg == 0 ? cK : cV, sm + p.sm_a + (cg == 0 ? 0 : 128 * D * 4), row, D);
      } else {
        const size_t lim = j < p.T ? (size_t)(bh + 1) * p.T : 0;
        if (cg == 0) row_to_tmem(tmem, cK, p.K, bh * p.T + j, lim, D, p.x3 != 0);
        else if (needV) row_to_tmem(tmem, cV, p.V, bh * p.T + j, lim, D, p.x3 != 0);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if ((tid & 31) == 0) mbar_arrive(bar_ops);
    };
    if (snake_item(0) < p.nitems) ops_to_tmem(0);
    // FWM Nearest: the half-bin table (entry q at sm_table + 8 (q + 2)) and the doubled
    // position; FWM LERP: the pair table, entry r at sm_table + 8 r (0x4B000000 * 8 =
    // 0x58000000 mod 2^32)
    constexpr bool half = fwm_like(CAL) && REC == REC_NEAREST;
    if constexpr (fwm_like(CAL)) {
      if (half && tid < 2 * Kq + 1 + kHalfTail)
        *reinterpret_cast<float2*>(sm + p.sm_table + tid * 8) = fwm_half_entry(p, tid - kHalfTail);
      if (!half && tid < Kq)
        *reinterpret_cast<float2*>(sm + p.sm_table + tid * 8) = make_float2(p.fwm_e[tid], p.fwm_e[tid + 1]);
    }
    const float Kf = (float)(half ? 2 * Kq : Kq);
    const uint32_t fwtab = smem_u32(sm + p.sm_table) + (half ? 8u * kHalfTail : 0u) - 0x58000000u;
    group_sync(BAR_COMPUTE, NCOMP);  // the FWM table
    bool failed = false;
    int n = 0;
    RingPos cs, cb;  // stage and score buffer of the current tile
    for (int item = snake_item(n); item < p.nitems && !failed; item = snake_item(++n)) {
      const int kb = item / p.BH, bh = item % p.BH;
      const int qt0 = (kb * 128) / BT, nit = nqt - qt0;
      const int j = kb * 128 + row;
      const int* tflags = p.tileflags + (size_t)bh * p.nqt + qt0;
      int tie_next = (FULLG && CAL != CAL_SOFTMAX) ? __ldg(tflags) : 0;
      for (int it = 0; it < nit; ++it, cs.next(NS), cb.next(nbuf)) {
        // the tie flag of this 64-row query tile, loaded one tile ahead
        const int tie_here = tie_next;
        if (FULLG && CAL != CAL_SOFTMAX && it + 1 < nit) tie_next = __ldg(tflags + it + 1);
        const int b = cb.i, s = cs.i;
        const int q0 = (qt0 + it) * BT;
        const bool ok1 = mbar_wait(&bar_sfull[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
        // the stage's row records arrived with its tiles (bar_full), before the products were issued
        const bool ok2 = ok1 && mbar_wait(&bar_full[s], cs.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
        if (!ok2) {
          failed = true;
          break;
        }
        tc_fence_after();
        const uint8_t* st = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        // two 16-column halves of the thread's W columns (bounds the live registers)
#pragma unroll 1
        for (int h = 0; h < W / WS; ++h) {
          const int c0 = cg * W + h * WS, i0h = q0 + c0;
          const uint32_t recs = smem_u32(st + oRec) + c0 * 64;
          const uint32_t tabs = smem_u32(st + oTab) + c0 * tstride - 0x58000000u;
          const int cS = base + 128 * b + c0, cG = cS + 64;
          float sv[WS], gv[WS], pa[WS], da[WS];
          tmem_ldw<WS>(lane_addr(tmem, cS), sv);
          if (needV) {
            tmem_ldw<WS>(lane_addr(tmem, cG), gv);
          } else {
#pragma unroll
            for (int q = 0; q < WS; ++q) gv[q] = 0.f;
          }
          tmem_ld_wait();
          const bool masked = (i0h < kb * 128 + 128) || (i0h + WS > p.T);
          if (FULLG && CAL != CAL_SOFTMAX && tie_here)
            kv_chunk<CAL, REC, FULLG, PROJ, true, true, WS>(sv, gv, pa, da, j, i0h, p.T, recs, tabs, fwtab, tstride, Kf,
                                                      p.fwm_inv_h, p.scale, p.fwm_hl, p.fwm_b0l);
          else if (masked)
            kv_chunk<CAL, REC, FULLG, PROJ, true, false, WS>(sv, gv, pa, da, j, i0h, p.T, recs, tabs, fwtab, tstride,
                                                       Kf, p.fwm_inv_h, p.scale, p.fwm_hl, p.fwm_b0l);
          else
            kv_chunk<CAL, REC, FULLG, PROJ, false, false, WS>(sv, gv, pa, da, j, i0h, p.T, recs, tabs, fwtab, tstride,
                                                        Kf, p.fwm_inv_h, p.scale, p.fwm_hl, p.fwm_b0l);
          // optional side outputs: per-query-row sums of dS and |dS| over this warp's 32 keys
          if constexpr (RS) {
            if (doDK) rowsum_add(da, p.dsum_out, p.dabs_out, (size_t)bh * p.T + i0h, min(WS, p.T - i0h));
          }
          if (p.x3) {
#pragma unroll
            for (int q = 0; q < WS; ++q) {
              const float x = doDV ? pa[q] : da[q];
              const float hh = tf32_rna(x);
              pa[q] = hh;
              da[q] = __fsub_rn(x, hh);
            }
            tmem_stw<WS>(lane_addr(tmem, cS), pa);
            tmem_stw<WS>(lane_addr(tmem, cG), da);
          } else {
            if (doDV) tmem_stw<WS>(lane_addr(tmem, cS), pa);
            if (doDK) tmem_stw<WS>(lane_addr(tmem, cG), da);
          }
        }
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_emptyA[s]);  // the stage's records are read
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_pready[b]);
      }
      // the next item's K / V (this item's S^T, g^T have all been read: the last tile's were)
      if (!failed && snake_item(n + 1) < p.nitems) ops_to_tmem(n + 1);
      const bool dok = !failed && mbar_wait(bar_done, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
      failed = group_any(BAR_COMPUTE, NCOMP, !dok);
      if (!failed) {
        tc_fence_after();
        // dV, dK rows into swizzled tiles for TMA stores: in the K / V staging area (free now
        // that the next item's K / V are in TMEM; the producer stores them before it stages
        // the item after next), or, for the last item, in the idle stage ring (stored here).
        // Without the staging area (3xTF32, d = 128, one-product launches) straight to
        // global memory.
        const bool last = snake_item(n + 1) >= p.nitems;
        uint8_t* stg = last ? sm + p.sm_stage0 : sm + p.sm_a;
        for (int pass = 0; pass < 2; ++pass) {
          if (pass == 0 ? !doDV : !doDK) continue;
          const int col = pass == 0 ? cdV : cdK;
          const float mul = pass == 0 ? 1.0f : p.scale;
          float* out = (pass == 0 ? p.dV : p.dK) + ((size_t)bh * p.T + j) * D;
          for (int c = cg * (D / NCG); c < (cg + 1) * (D / NCG); c += 32) {
            float v[32];
            tmem_ld32(lane_addr(tmem, col + c), v);
            if (p.x3) {
              float w[32];
              tmem_ld32(lane_addr(tmem, cdC + c), w);
              tmem_ld_wait();
#pragma unroll
              for (int q = 0; q < 32; ++q) v[q] += w[q];
            }
            tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < 32; ++q) v[q] *= mul;
            if (p.ops_smem) {
              row_to_staged(stg + pass * 128 * D * 4, row, c / 32, v);
            } else if (j < p.T) {
              float4* dst = reinterpret_cast<float4*>(out + c);
#pragma unroll
              for (int q = 0; q < 8; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            }
          }
        }
        if (p.ops_smem) {
          fence_async_smem();
          if (last) {
            group_sync(BAR_COMPUTE, NCOMP);
            if (warp == 0 && doDV) store_rows_tile_boxed(stg, &maps.dv, D, 64, kb * 128, bh, false);
            if (warp == 1 && doDK) store_rows_tile_boxed(stg + 128 * D * 4, &maps.dk, D, 64, kb * 128, bh, false);
          } else {
            __syncwarp();
            if ((tid & 31) == 0) mbar_arrive(bar_ostg);
          }
        }
      }
    }
    if (warp < 2) tma_store_wait_all();
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

// Every backward mode of one calibration and reconstruction; softmax ignores the mode.
template <int CAL, int REC, bool RS>
cudaError_t launch_dkdv_modes(dim3 grid, const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  if constexpr (CAL == CAL_SOFTMAX) {
    return launch3(k_bwd_dkdv<CAL_SOFTMAX, REC_LERP, false, false, RS>, grid, maps, p, smem_bytes, s);
  } else {
    const bool proj = p.grad == GRAD_DETACH_PROJ, full = p.grad != GRAD_DETACH && !proj;
    return full ? launch3(k_bwd_dkdv<CAL, REC, true, false, RS>, grid, maps, p, smem_bytes, s)
           : proj ? launch3(k_bwd_dkdv<CAL, REC, false, true, RS>, grid, maps, p, smem_bytes, s)
                  : launch3(k_bwd_dkdv<CAL, REC, false, false, RS>, grid, maps, p, smem_bytes, s);
  }
}

// The dK/dV launch of p's configuration; RS: the instantiation that also accumulates the
// per-row sums of dS and |dS| (p.dsum_out, p.dabs_out).
template <bool RS>
cudaError_t launch_bwd_dkdv_t(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  const dim3 grid((unsigned)p.ngrid);
  const bool near = p.recon == REC_NEAREST;
  switch (p.calib) {
    case CAL_SOFTMAX: return launch_dkdv_modes<CAL_SOFTMAX, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
    case CAL_EXP8: return launch_dkdv_modes<CAL_EXP8, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
    case CAL_EXPB: return launch_dkdv_modes<CAL_EXPB, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
    case CAL_MINMAX:
      return near ? launch_dkdv_modes<CAL_MINMAX, REC_NEAREST, RS>(grid, maps, p, smem_bytes, s)
                  : launch_dkdv_modes<CAL_MINMAX, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
    case CAL_FWMR:
      return near ? launch_dkdv_modes<CAL_FWMR, REC_NEAREST, RS>(grid, maps, p, smem_bytes, s)
                  : launch_dkdv_modes<CAL_FWMR, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
    default:
      return near ? launch_dkdv_modes<CAL_FWM, REC_NEAREST, RS>(grid, maps, p, smem_bytes, s)
                  : launch_dkdv_modes<CAL_FWM, REC_LERP, RS>(grid, maps, p, smem_bytes, s);
  }
}

}  // namespace kint
