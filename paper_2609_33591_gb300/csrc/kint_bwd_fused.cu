// Single-pass backward (App. B) for TF32 at d = 64: one key-block-major pass forms
// S^T, g^T and the element work once per (key block, query tile) pair and feeds all
// three contractions from it:
//   dV_j += sum_i P_ij dO_i,   dK_j += s sum_i dS_ij Q_i   (TMEM accumulators per key block)
//   dQ_i += s sum_j dS_ij K_j                              (a 64-query partial per tile,
//                                                           added to global memory)
// with dS_ij = gamma_ij Delta_ij, the own-score term.  The extremum terms of Eq. (full)
// (c_M / n_max at the arg-max key of each row) need the whole row's sum
// c_M = -sum_j gamma_ij Delta_ij (FWM: dw/dM = -Delta in the window; the FP8 / BF16
// exponentials keep the same maximum channel), which is complete only after every key
// block has passed, so this pass accumulates that row sum and k_bwd_ext adds
//   dQ_i += s (c_M / n_max) K_amax(i),   dK_amax(i) += s (c_M / n_max) Q_i
// afterwards.  Rows with tied maxima would need the tie set, which only the scores
// themselves give: when any row has one, the gated two-pass kernels (k_bwd_dq,
// k_bwd_dkdv) run instead and these kernels leave at once.
//
// The partial dQ sums and the extremum scatter are fp32 additions whose order is not
// fixed, so this path is not bit-reproducible from run to run; the two-pass path is.
#include "kint_bwd_common.cuh"

namespace kint {

// 16-byte row record of this pass (written by the backward's dO prep job, RecJob):
// u = acc * k1 + c0 with k1 the same for every row of a launch (FWM, the exponentials),
// forward 1/W, gamma = g * ga + gb.
struct FRec {
  float c0, invWf, ga, gb;
};

// acc -> position multiplier of every row, formed as the dQ kernel forms it
__device__ __forceinline__ float fused_k1(const Params& p) {
  const RowGrid g = row_grid(p, 0.0f, 0.0f);
  if (exp_like(p.calib)) return p.scale * kLog2e;
  return (fwm_like(p.calib) && p.recon == REC_NEAREST) ? 2.0f * g.k1 : g.k1;
}

// ---------------------------------------------------------------------------
// Element work on 16 query columns of key j: the forward probability P_ij and the
// own-score term dS_ij = gamma_ij Delta_ij, with the decisions and roundings of the
// dK/dV kernel's (App. A "LERP", "Nearest"; the exponential baselines).
// ---------------------------------------------------------------------------
template <int CAL, int REC, bool MASKED, int W>
__device__ __forceinline__ void fused_chunk(const float (&sv)[W], const float (&gv)[W], float (&pa)[W],
                                            float (&da)[W], int j, int i0, int T, uint32_t recs, uint32_t fwtab,
                                            float Kf, float k1, float fwm_inv_h, float hl, float b0l) {
#pragma unroll
  for (int ii = 0; ii < W; ++ii) {
    const float4 r = lds_f4(recs + ii * 16u);  // c0, invWf, ga, gb
    const float gam = __fmaf_rn(gv[ii], r.z, r.w);
    float pv, ds;
    if constexpr (CAL == CAL_SOFTMAX) {
      pv = ex2_approx(__fmaf_rn(sv[ii], k1, r.x)) * r.y;
      ds = pv * gam;
    } else if constexpr (CAL == CAL_EXP8) {
      const float we = ex2_approx(__fmaf_rn(sv[ii], k1, r.x));
      pv = e4m3_rn(we) * r.y;
      ds = gam * we;
    } else if constexpr (CAL == CAL_EXPB) {
      float zb;
      const float w = bf16_exp_weight(__fadd_rn(__fmul_rn(sv[ii], k1), r.x), zb);
      pv = w * r.y;
      ds = bf16_rn(__fmul_rn(bf16_rn(gam), w));
    } else if constexpr (REC == REC_NEAREST) {
      // FWM Nearest: v = 2u indexes the half-bin table of (w^N, Delta_r / h)
      const float v = __fmaf_rn(sv[ii], k1, r.x);
      const uint32_t qb = fwm_half_bits(v, Kf);
      float2 e = lds_f2(fwtab + qb * 8u);
      if constexpr (CAL == CAL_FWMR) {
        const BelowPair bp = resolved_below(__fmul_rn(v, 0.5f), hl, b0l);
        const float2 eb = make_float2(bp.t >= 0.5f ? bp.e1 : bp.e0, __fmul_rn(__fsub_rn(bp.e1, bp.e0), fwm_inv_h));
        e = v < 0.0f ? eb : e;
      }
      pv = e.x * r.y;
      ds = gam * e.y;
    } else {
      // FWM LERP: the pair table (e_r, e_{r+1})
      const float u = __fmaf_rn(sv[ii], k1, r.x);
      float t, rf;
      uint32_t rb;
      decode_u(u, Kf, t, rb, rf);
      float2 e = lds_f2(fwtab + rb * 8u);
      if constexpr (CAL == CAL_FWMR) {
        const BelowPair bp = resolved_below(u, hl, b0l);
        const bool below = u < 0.0f;
        t = below ? bp.t : t;
        e = below ? make_float2(bp.e0, bp.e1) : e;
      }
      const float de = __fsub_rn(e.y, e.x);
      float w = __fmaf_rn(t, de, e.x);
      ds = gam * (de * fwm_inv_h);
      if constexpr (CAL == CAL_FWM) {
        const bool tail = u < 0.0f;
        w = tail ? 0.f : w;
        ds = tail ? 0.f : ds;
      }
      pv = w * r.y;
    }
    if constexpr (MASKED) {
      const int iq = i0 + ii;
      const bool ok = iq >= j && iq < T;
      pv = ok ? pv : 0.f;
      ds = ok ? ds : 0.f;
    }
    pa[ii] = pv;
    da[ii] = ds;
  }
}

// The calling warp holds v[c] for 16 query rows r0 + c at 32 keys (one per lane): the
// 32-key sum of each row is added to dst[r0 + c] (butterfly reduce-scatter: the xor-16
// step keeps rows 8..15 in the upper half-warp, xor-8 rows +4, xor-4 +2, xor-2 +1, and
// xor-1 adds the pair; the even lane of each pair adds it).
__device__ __forceinline__ void rowsum_red(const float (&v)[16], float* dst, size_t r0, int nvalid) {
  const int lane = threadIdx.x & 31;
  float s[16];
#pragma unroll
  for (int c = 0; c < 16; ++c) s[c] = v[c];
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1) {
    const bool up = (lane & (2 * w)) != 0;
#pragma unroll
    for (int k = 0; k < w; ++k) {
      const float send = up ? s[k] : s[k + w];
      const float keep = up ? s[k + w] : s[k];
      s[k] = keep + __shfl_xor_sync(0xffffffffu, send, 2 * w);
    }
  }
  s[0] += __shfl_xor_sync(0xffffffffu, s[0], 1);
  const int c = (lane >> 1) & 15;
  if ((lane & 1) == 0 && c < nvalid) red_add_f32(dst + r0 + c, s[0]);
}


// ---------------------------------------------------------------------------
// k_bwd_fused (640 threads: 16 compute warps, the MMA warp, two producer warps, an idle warp).  Work
// items are (128-key block kb, head) pairs, longest first; a CTA
// takes sched_item(sch, 0), sched_item(sch, 1), ...  Thread t (< 512) owns key j = kb*128 + t%128
// (TMEM lane t%128) and the 16 query columns 16 (t/128) .. +15 of each 64-query tile:
// four compute warps per SM sub-partition, so that one warp's latencies (TMEM and
// shared-memory loads, shuffles) hide under the others' element work.
// TMEM: K [0, 64) (A operand of S^T), per buffer b: S^T_b at 64 + 128 b and g^T_b 64
// columns further (P^T overwrites S^T_b, dS^T overwrites g^T_b: the A operands of dV, dK),
// dV [320, 384), dK [384, 448), the 64-query dQ partial [448, 512) (M = 64: query row r
// of the tile in lane 32 (r / 16) + r % 16).
// smem: two stages, each Q | dO | Q^T | dO^T tiles and the tile's 64 FRecs.  Tile u
// (counted over the CTA's whole run) uses stage u % 2; its dS (64 query rows x 128 keys,
// K-major: the A operand of the dQ product) goes into the Q^T | dO^T half of the other
// stage once the products dV, dK of tile u - 1 have read it, so the Q | dO half is free
// for tile u + 2 as soon as the element work of tile u is done, and that stage's Q^T | dO^T
// half takes tile u + 1's tiles once dQ of tile u has read dS.  The item's V tile (A
// operand of g^T) also stages the next item's K rows on their way into TMEM; its K^T tile
// (B operand of dQ), which the compute warps write from the K rows in TMEM, stages the dV,
// dK rows of the epilogue (32 keys x 16 columns per warp, 64-byte swizzle) for TMA stores,
// after which each warp writes its part of the next item's K^T there; each compute warp
// has a 1 KB slice for its 16 rows x 16 columns of the dQ partial (64-byte swizzle), added
// to dQ by a TMA reduce.
// ---------------------------------------------------------------------------
constexpr int NCOMP_F = 512;  // compute threads
constexpr int MMA_WARP_F = NCOMP_F / 32, PRODUCER_WARP_F = NCOMP_F / 32 + 1, PRODUCER2_WARP_F = NCOMP_F / 32 + 2;
// The MMA warp, the two producer warps and a fourth, idle warp form the fifth warpgroup, which
// gives registers to the four compute warpgroups: launched at 96 per thread (640 threads),
// it keeps 64 and the compute warps take 104 (512 x 104 + 128 x 64 = 640 x 96).
constexpr int NTHR_FUSED = NCOMP_F + 128;
constexpr int REG_LAUNCH_F = 96, REG_COMP_F = 104, REG_AUX_F = 64;
static_assert(NCOMP_F * REG_COMP_F + (NTHR_FUSED - NCOMP_F) * REG_AUX_F <= NTHR_FUSED * REG_LAUNCH_F,
              "register shares exceed the launch allocation");

// Byte offset of 16-byte chunk c of row r in a tile of 64-byte rows under the 64-byte
// swizzle (chunk index XOR bits 1..2 of the row), the layout TMA reads for the dQ reduce
// and the dV / dK stores.
__device__ __forceinline__ uint32_t sw64_off(int r, int c) {
  return (uint32_t)r * 64u + (uint32_t)((c ^ ((r >> 1) & 3)) << 4);
}

template <int CAL, int REC, bool FULLG>
__global__ void __launch_bounds__(NTHR_FUSED, 1) k_bwd_fused(const __grid_constant__ Maps maps, const Params p,
                                                           const __grid_constant__ Sched sch) {
  uint8_t* sm = smem_base();
  constexpr int D = 64, NS = 2;
  constexpr int qtile = BT * D * 4;
  constexpr int oQ = 0, odO = qtile, oQT = 2 * qtile, odOT = 3 * qtile, oRec = 4 * qtile;
  constexpr int cK = 0, cSG = 64, cdV = 320, cdK = 384, cdQ = 448;
  constexpr int PNL_DS = 64 * SW;  // one 32-key panel of the dS tile
  const int Kq = p.Kint;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_full = bars;                 // [NS] Q, dO, records landed
  uint64_t* bar_emptyA = bars + NS;          // [NS] Q | dO half free (the element work is done)
  uint64_t* bar_fullT = bars + 2 * NS;       // [NS] Q^T, dO^T landed
  uint64_t* bar_empty = bars + 3 * NS;       // [NS] Q^T | dO^T half free for the producer (dQ read the dS there)
  uint64_t* bar_tfree = bars + 4 * NS;       // [NS] Q^T, dO^T read by dV, dK (dS may go there)
  uint64_t* bar_sfull = bars + 5 * NS;       // [2] S^T_b, g^T_b computed
  uint64_t* bar_pready = bars + 5 * NS + 2;  // [2] P^T, dS^T, dS of buffer b written
  uint64_t* bar_dqfull = bars + 5 * NS + 4;  // the tile's dQ partial computed
  uint64_t* bar_done = bars + 5 * NS + 5;    // every product of the item completed
  uint64_t* bar_kst = bars + 5 * NS + 6;     // the item's K rows staged in the V buffer
  uint64_t* bar_ops = bars + 5 * NS + 7;     // the item's K rows in TMEM (the V buffer free)
  uint64_t* bar_v = bars + 5 * NS + 8;       // the item's V tile landed
  uint64_t* bar_vfree = bars + 5 * NS + 9;   // the item's last g^T completed
  uint64_t* bar_kt = bars + 5 * NS + 10;     // the item's K^T tile written by every compute warp
  uint64_t* bar_drain = bars + 5 * NS + 12;  // the MMA warp's clean-up commit
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 5 * NS + 13);
  const int tid = threadIdx.x, warp = warp_id_uniform();
  const int nqt = (p.T + BT - 1) / BT;

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_emptyA[s], NCOMP_F / 32);
      mbar_init(&bar_fullT[s], 1);
      mbar_init(&bar_empty[s], 1);
      mbar_init(&bar_tfree[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar_sfull[b], 1);
      mbar_init(&bar_pready[b], NCOMP_F / 32);
    }
    mbar_init(bar_dqfull, 1);
    mbar_init(bar_done, 1);
    mbar_init(bar_kst, 1);
    mbar_init(bar_ops, NCOMP_F / 32);
    mbar_init(bar_v, 1);
    mbar_init(bar_vfree, 1);
    mbar_init(bar_kt, NCOMP_F / 32);
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
  pdl_wait();
  // All 512 columns are allocated: the allocation starts at lane 0, column 0.
  if (threadIdx.x == 0 && *tslot != 0u) dev_flag(p.status, DEV_ERR_BOUNDS);
  constexpr uint32_t tmem = 0;
  if (gated_off(p)) {
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp < NCOMP_F / 32)
    setmaxnreg_inc<REG_COMP_F>();
  else
    setmaxnreg_dec<REG_AUX_F>();

  // Two producer warps: PRODUCER_WARP_F loads the Q | dO halves with their records and the
  // items' K rows and V tiles, PRODUCER2_WARP_F the Q^T | dO^T halves, so that neither kind
  // of load waits behind the other's condition.
  auto item_of = [&](int k, int& kb_, int& bh_) {
    const int it_ = sched_item(sch, k);
    kb_ = it_ / p.BH;
    bh_ = it_ % p.BH;
  };
  if (warp == PRODUCER_WARP_F) {
    int gt = 0, n = 0;
    RingPos ld, nf;
    int cf = 0, nks = 0, nv = 0;
    bool ok = true;
    auto load_k = [&](int k) {  // K rows of item k into the V buffer
      int kb_, bh_;
      item_of(k, kb_, bh_);
      mbar_arrive_expect_tx(bar_kst, 128 * D * 4);
      load_rows_tile_boxed(sm + p.sm_v, &maps.k, bar_kst, D, 128, BT, 0, kb_ * 128, bh_);
      ++nks;
    };
    auto load_v = [&](int k) {
      int kb_, bh_;
      item_of(k, kb_, bh_);
      mbar_arrive_expect_tx(bar_v, 128 * D * 4);
      load_rows_tile_boxed(sm + p.sm_v, &maps.v, bar_v, D, 128, BT, 0, kb_ * 128, bh_);
      ++nv;
    };
    if (sched_item(sch, 0) < p.nitems) load_k(0);
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int kb = item / p.BH, bh = item % p.BH;
      const int qt0 = (kb * 128) / BT, nit = nqt - qt0;
      for (int it = 0; it < nit; ++it, ++gt, ld.next(NS)) {
        const int s = ld.i, q0 = (qt0 + it) * BT;
        if (gt >= NS && !mbar_wait_warp(&bar_emptyA[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        uint64_t* b = &bar_full[s];
        const int nrows = min(BT, p.T - q0);
        mbar_arrive_expect_tx(b, 2 * qtile + nrows * 16);
        load_rows_tile(dst + oQ, &maps.q, b, D, BT, 0, q0, bh);
        load_rows_tile(dst + odO, &maps.dout, b, D, BT, 0, q0, bh);
        bulk_load(dst + oRec, reinterpret_cast<const FRec*>(p.frec) + (size_t)bh * p.T + q0, nrows * 16, b);
        nf.next(NS);
        ++cf;
        // this item's V, once its K rows have gone from the V buffer into TMEM (after the
        // item's first tiles, whose loads need only the previous item's element work)
        if (it == min(nit, NS) - 1) {
          if (!mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
            ok = false;
            break;
          }
          load_v(n);
        }
      }
      // the next item's K rows, once this item's last g^T has read V
      if (ok && sched_item(sch, n + 1) < p.nitems) {
        if (!mbar_wait_warp(bar_vfree, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          ok = false;
          break;
        }
        load_k(n + 1);
      }
    }
    // clean-up: the last loads issued have landed
    drain_ring(bar_full, nf, cf, NS, p.wait_ns, p.status);
    if (nks > 0) mbar_wait_warp(bar_kst, (nks - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
    if (nv > 0) mbar_wait_warp(bar_v, (nv - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
  } else if (warp == PRODUCER2_WARP_F) {
    int gt = 0, n = 0;
    RingPos ld, nT;
    int cT = 0;
    bool ok = true;
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int kb = item / p.BH, bh = item % p.BH;
      const int qt0 = (kb * 128) / BT, nit = nqt - qt0;
      for (int it = 0; it < nit; ++it, ++gt, ld.next(NS)) {
        const int s = ld.i, q0 = (qt0 + it) * BT;
        // the Q^T | dO^T half holds dS of the previous tile until its dQ product has read it
        if (gt >= 1 &&
            !mbar_wait_warp(&bar_empty[s], (uint32_t)((gt - 1) >> 1) & 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        uint64_t* bt = &bar_fullT[s];
        mbar_arrive_expect_tx(bt, 2 * qtile);
        load_rows_tile(dst + oQT, &maps.qt, bt, BT, D, q0, 0, bh);
        load_rows_tile(dst + odOT, &maps.dot, bt, BT, D, q0, 0, bh);
        nT.next(NS);
        ++cT;
      }
    }
    // clean-up: the last loads issued have landed
    drain_ring(bar_fullT, nT, cT, NS, p.wait_ns, p.status);
  } else if (warp == MMA_WARP_F) {
    const uint8_t* st0 = sm + p.sm_stage0;
    const uint32_t idq = idesc_tf32(64, D, 0, 0);
    int n = 0;
    RingPos is, ib, cs, cb;  // stage / buffer of the next S^T, g^T product and of the tile being finished
    bool ok = true;
    // S^T_b = K Q^T (A in TMEM) and g^T_b = V dO^T (A in smem) of the next tile
    auto issue_sg = [&]() -> bool {
      const int s = is.i;
      if (!mbar_wait_warp(&bar_full[s], is.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) return false;
      tc_fence_after();
      const uint8_t* st = st0 + s * p.sm_stage_bytes;
      const uint32_t cS = tmem + cSG + 128 * ib.i, cG = cS + 64;
      mma_tmem_smem(cS, tmem + cK, st + oQ, BT, D, false);
      mma_smem_smem(cG, sm + p.sm_v, st + odO, BT, D, false);
      mma_commit(&bar_sfull[ib.i]);
      is.next(NS);
      ib.next(2);
      return true;
    };
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int kb = item / p.BH, nit = nqt - (kb * 128) / BT;
      ok = mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) &&
           mbar_wait_warp(bar_v, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      if (ok) tc_fence_after();
      ok = ok && issue_sg();
      if (ok && nit == 1) mma_commit(bar_vfree);
      for (int it = 0; it < nit && ok; ++it, cs.next(NS), cb.next(2)) {
        if (it + 1 < nit) {
          ok = issue_sg();
          if (ok && it + 2 == nit) mma_commit(bar_vfree);
          if (!ok) break;
        }
        const int b = cb.i, s = cs.i;
        if (!mbar_wait_warp(&bar_pready[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) ||
            (it == 0 && !mbar_wait_warp(bar_kt, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* st = st0 + s * p.sm_stage_bytes;
        const uint8_t* so = st0 + (s ^ 1) * p.sm_stage_bytes;  // the other stage: this tile's dS
        const uint32_t cS = tmem + cSG + 128 * b, cG = cS + 64;
        // dQ partial (64 queries x 64) = dS K, first: its completion frees the other stage's
        // Q^T | dO^T half for the next tile's transposed tiles
        mma_ss_k<16>(tmem + cdQ, so + oQT, sm + p.sm_kt, PNL_DS, 64 * SW, idq, false);
        mma_commit(&bar_empty[s ^ 1]);
        mma_commit(bar_dqfull);
        if (!mbar_wait_warp(&bar_fullT[s], cs.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        mma_tmem_smem(tmem + cdV, cS, st + odOT, D, BT, it > 0);
        mma_tmem_smem(tmem + cdK, cG, st + oQT, D, BT, it > 0);
        mma_commit(&bar_tfree[s]);
      }
      mma_commit(bar_done);
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else if (warp < NCOMP_F / 32) {
    const int row = tid & 127, cq = tid >> 7, q4 = warp & 3, lane = tid & 31;
    uint8_t* dqs = sm + p.sm_ostage + warp * 1024;      // this warp's dQ reduce slice (16 rows x 16)
    uint8_t* ostg = sm + p.sm_kt + (q4 * 4 + cq) * 2048;  // its epilogue slice (32 rows x 16)
    // the k-th item's K rows from the V buffer into TMEM (each warp 16 of its keys' 64
    // columns), handed to the MMA warp (and the producer) through bar_ops
    auto ops_to_tmem = [&](int k) {
      const bool okk = mbar_wait(bar_kst, k & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      if (okk) {
        const uint32_t base = smem_u32(sm + p.sm_v) + (uint32_t)(cq >> 1) * 128u * SW + (uint32_t)row * SW;
        float v[16];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int chunk = (cq & 1) * 4 + c;
          const float4 x = lds_f4(base + (uint32_t)((chunk ^ (row & 7)) << 4));
          v[4 * c] = x.x;
          v[4 * c + 1] = x.y;
          v[4 * c + 2] = x.z;
          v[4 * c + 3] = x.w;
        }
        tmem_st16(lane_addr(tmem, cK + 16 * cq), v);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_ops);
    };
    // The item's K^T tile (the B operand of every dQ product: 64 rows d, 128 keys, four 32-key
    // panels under the 128-byte swizzle) from its K rows in TMEM: this thread's key (TMEM lane)
    // at its 16 columns d = 16 cq .. 16 cq + 15, which in that layout are rows 16 cq + k of panel
    // q4, the 2 KB of the warp's own epilogue slice.  Handed to the MMA warp through bar_kt.
    auto kt_out = [&]() {
      float v[16];
      tmem_ld16(lane_addr(tmem, cK + 16 * cq), v);
      tmem_ld_wait();
      const uint32_t base = smem_u32(ostg) + (uint32_t)(lane & 3) * 4u;
#pragma unroll
      for (int k = 0; k < 16; ++k)
        asm volatile("st.shared.f32 [%0], %1;" ::"r"(base + (uint32_t)k * (uint32_t)SW +
                                                     ((((uint32_t)lane >> 2) ^ (uint32_t)(k & 7)) << 4)),
                     "f"(v[k])
                     : "memory");
      fence_async_smem();  // read by the tensor core
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_kt);
    };
    // the dQ partial of tile q0 (this warp's 16 rows in its lanes 0..15, its 16 columns),
    // scaled, staged in the warp's slice and added to dQ by a TMA reduce
    auto dq_out = [&](int bh_, int q0) {
      float v[16];
      tmem_ld16(lane_addr(tmem, cdQ + 16 * cq), v);
      tmem_ld_wait();
      tma_store_wait_read();  // the slice's previous reduce has read it
      if (lane < 16) {
        const uint32_t base = smem_u32(dqs);
#pragma unroll
        for (int c = 0; c < 4; ++c)
          asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(base + sw64_off(lane, c)),
                       "f"(v[4 * c] * p.scale), "f"(v[4 * c + 1] * p.scale), "f"(v[4 * c + 2] * p.scale),
                       "f"(v[4 * c + 3] * p.scale)
                       : "memory");
      }
      fence_async_smem();
      __syncwarp();
      tma_reduce_add_3d(&maps.dq16, dqs, 16 * cq, q0 + 16 * q4, bh_);
      tma_store_commit();
    };
    // (i, j) pairs of a row with tied maxima whose score at key j equals its maximum, into the
    // tie list (rows i0 .. i0 + 15 of this thread's chunk, key j)
    auto tie_search = [&](const float (&sv)[16], int j_, int i0, int bh_) {
#pragma unroll
      for (int ii = 0; ii < 16; ++ii) {
        const int i = i0 + ii;
        if (i >= p.T || j_ > i) continue;
        const size_t rw = (size_t)bh_ * p.T + i;
        if (__ldg(p.n_max + rw) > 1 && __fmul_rn(sv[ii], p.scale) == __ldg(p.row_max + rw)) {
          const int slot = atomicAdd(p.tie_count, 1);
          if (slot < p.tie_cap) p.tie_list[slot] = make_int2((int)rw, j_);
          else dev_flag(p.status, DEV_ERR_BOUNDS);
        }
      }
    };
    if (sched_item(sch, 0) < p.nitems) {
      ops_to_tmem(0);
      kt_out();
    }
    constexpr bool half = fwm_like(CAL) && REC == REC_NEAREST;
    if constexpr (fwm_like(CAL)) {
      if (half && tid < 2 * Kq + 1 + kHalfTail)
        *reinterpret_cast<float2*>(sm + p.sm_table + tid * 8) = fwm_half_entry(p, tid - kHalfTail);
      if (!half && tid < Kq)
        *reinterpret_cast<float2*>(sm + p.sm_table + tid * 8) = make_float2(p.fwm_e[tid], p.fwm_e[tid + 1]);
    }
    const float Kf = (float)(half ? 2 * Kq : Kq), k1 = fused_k1(p);
    const uint32_t fwtab = smem_u32(sm + p.sm_table) + (half ? 8u * kHalfTail : 0u) - 0x58000000u;
    group_sync(BAR_COMPUTE, NCOMP_F);  // the FWM table
    bool failed = false;
    int n = 0, gu = 0;  // gu: tiles so far over the CTA's run (stage parity, bar_dqfull, bar_tfree)
    RingPos cs, cb;
    const int c0 = cq * 16;  // this thread's query columns in every tile
    for (int item = sched_item(sch, n); item < p.nitems && !failed; item = sched_item(sch, ++n)) {
      const int kb = item / p.BH, bh = item % p.BH;
      const int qt0 = (kb * 128) / BT, nit = nqt - qt0;
      const int j = kb * 128 + row;
      const int* tflags = p.tileflags + (size_t)bh * p.nqt + qt0;
      int tie_next = FULLG ? __ldg(tflags) : 0;
      for (int it = 0; it < nit; ++it, cs.next(NS), cb.next(2), ++gu) {
        const int b = cb.i, s = cs.i;
        const int q0 = (qt0 + it) * BT;
        // the tie flag of this 64-row query tile, loaded one tile ahead
        const int tie_here = tie_next;
        if (FULLG && it + 1 < nit) tie_next = __ldg(tflags + it + 1);
        const bool ok1 = mbar_wait(&bar_sfull[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
        const bool ok2 = ok1 && mbar_wait(&bar_full[s], cs.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
        if (!ok2) {
          failed = true;
          break;
        }
        tc_fence_after();
        const uint8_t* st = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        // this lane's key in the dS tile (the other stage's Q^T | dO^T half): panel q4, 4-byte
        // slot lane % 4 of chunk lane / 4
        const uint32_t dsb = smem_u32(sm + p.sm_stage0 + (s ^ 1) * p.sm_stage_bytes + oQT) + (uint32_t)q4 * PNL_DS +
                             (uint32_t)(lane & 3) * 4u;
        const uint32_t dchunk = (uint32_t)(lane >> 2);
        const int i0h = q0 + c0;
        {
          const uint32_t recs = smem_u32(st + oRec) + c0 * 16;
          const int cS = cSG + 128 * b + c0, cG = cS + 64;
          float sv[16], gv[16], pa[16], da[16];
          tmem_ldw<16>(lane_addr(tmem, cS), sv);
          tmem_ldw<16>(lane_addr(tmem, cG), gv);
          tmem_ld_wait();
          // rows with tied maxima in this tile (rare): list every causal key whose score equals
          // the row maximum, the equality the forward's tie count was taken with
          if (FULLG && tie_here) tie_search(sv, j, i0h, bh);
          const bool masked = (i0h < kb * 128 + 128) || (i0h + 16 > p.T);
          if (masked)
            fused_chunk<CAL, REC, true, 16>(sv, gv, pa, da, j, i0h, p.T, recs, fwtab, Kf, k1, p.fwm_inv_h, p.fwm_hl,
                                            p.fwm_b0l);
          else
            fused_chunk<CAL, REC, false, 16>(sv, gv, pa, da, j, i0h, p.T, recs, fwtab, Kf, k1, p.fwm_inv_h, p.fwm_hl,
                                             p.fwm_b0l);
          if constexpr (FULLG) rowsum_red(da, p.rsum, (size_t)bh * p.T + i0h, min(16, p.T - i0h));
          tmem_stw<16>(lane_addr(tmem, cS), pa);
          tmem_stw<16>(lane_addr(tmem, cG), da);
          // dS goes where the previous tile's Q^T, dO^T were, once dV, dK have read them
          if (gu >= 1 &&
              !mbar_wait(&bar_tfree[s ^ 1], (uint32_t)((gu - 1) >> 1) & 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
            failed = true;
            break;
          }
#pragma unroll
          for (int ii = 0; ii < 16; ++ii) {
            const uint32_t i = (uint32_t)(c0 + ii);
            asm volatile("st.shared.f32 [%0], %1;" ::"r"(dsb + i * (uint32_t)SW + (((dchunk ^ (i & 7u)) << 4))),
                         "f"(da[ii])
                         : "memory");
          }
        }
        // the tile's records and Q, dO are no longer needed
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar_emptyA[s]);
        // the previous tile's dQ partial (its product was issued after that tile's element work)
        if (it > 0) {
          if (!mbar_wait(bar_dqfull, (uint32_t)(gu - 1) & 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
            failed = true;
            break;
          }
          tc_fence_after();
          dq_out(bh, q0 - BT);
        }
        tmem_st_wait();
        fence_async_smem();  // dS, written here, is read by the tensor core
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar_pready[b]);
        // the item's last S^T has completed: the next item's K rows may replace these
        if (it + 1 == nit && sched_item(sch, n + 1) < p.nitems) ops_to_tmem(n + 1);
      }
      const bool dok = !failed && mbar_wait(bar_done, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
      failed = group_any(BAR_COMPUTE, NCOMP_F, !dok);
      if (!failed) {
        tc_fence_after();
        dq_out(bh, (qt0 + nit - 1) * BT);
        // dV, then dK (scaled): this warp's 32 rows x 16 columns through its slice of the
        // K^T buffer (every product of the item has completed) and a TMA store
        for (int pass = 0; pass < 2; ++pass) {
          float v[16];
          tmem_ld16(lane_addr(tmem, (pass == 0 ? cdV : cdK) + 16 * cq), v);
          tmem_ld_wait();
          const float mul = pass == 0 ? 1.0f : p.scale;
          if (pass == 1) tma_store_wait_read();  // dV has left the slice
          const uint32_t base = smem_u32(ostg);
#pragma unroll
          for (int c = 0; c < 4; ++c)
            asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(base + sw64_off(lane, c)),
                         "f"(v[4 * c] * mul), "f"(v[4 * c + 1] * mul), "f"(v[4 * c + 2] * mul),
                         "f"(v[4 * c + 3] * mul)
                         : "memory");
          fence_async_smem();
          __syncwarp();
          tma_store_3d(pass == 0 ? &maps.dv32 : &maps.dk32, ostg, 16 * cq, kb * 128 + 32 * q4, bh);
          tma_store_commit();
        }
        tma_store_wait_read();
        // the next item's K^T into the slice the stores have read (its K rows are in TMEM)
        if (sched_item(sch, n + 1) < p.nitems) kt_out();
        tc_fence_before();
      }
    }
    tma_store_wait_all();  // every reduce and store of this warp is complete
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// The extremum terms of Eq. (full) after the single pass: c_M = -sum_j gamma_ij Delta_ij
// (the row sums k_bwd_fused accumulated), split over the n_max arg-max keys:
//   dQ_i += s (c_M / n_max) K_j,   dK_j += s (c_M / n_max) Q_i   for each arg-max key j
// (USE_M: not in min_only, where FWM-like grids have no minimum channel), both as fp32
// additions at L2, and the c_M / c_m side outputs.  The first blocks take rows with one
// maximum (arg_max), 64 rows per block, 16 threads per row with four columns each and
// four rows per thread, all loads issued before the additions; the last EXT_TIE_BLOCKS
// blocks take the tied maxima that k_bwd_fused listed as (row, key) pairs.
// ---------------------------------------------------------------------------
constexpr int EXT_TIE_BLOCKS = 64;

// K^T [BH][64][Tp] (keys past T zero) for the two-pass kernels that run in place of the
// single pass: 32-key blocks through a padded shared tile, grid-stride.
__device__ void ext_kt_fallback(const Params& p) {
  __shared__ float ts[32][65];
  const int Tp = (p.T + 31) & ~31, ntb = Tp / 32, tid = threadIdx.x;
  for (int u = blockIdx.x; u < p.BH * ntb; u += gridDim.x) {
    const int bh = u / ntb, t0 = (u % ntb) * 32;
    const int r = tid >> 3, c8 = (tid & 7) * 8;
    const int t = t0 + r;
#pragma unroll
    for (int k = 0; k < 8; ++k) ts[r][c8 + k] = t < p.T ? p.K[((size_t)bh * p.T + t) * 64 + c8 + k] : 0.f;
    __syncthreads();
    const int dd = tid >> 2, k8 = (tid & 3) * 8;
#pragma unroll
    for (int k = 0; k < 8; ++k) p.kt_out[((size_t)bh * 64 + dd) * Tp + t0 + k8 + k] = ts[k8 + k][dd];
    __syncthreads();
  }
}

template <bool USE_M>
__global__ void __launch_bounds__(256) k_bwd_ext(const Params p) {
  pdl_wait();
  pdl_trigger();
  if (gated_off(p)) {
    // the two-pass kernels run instead of this pass's result: they read K^T
    if (p.kt_out) ext_kt_fallback(p);
    return;
  }
  const int nrows = p.BH * p.T, l = threadIdx.x & 15, grp = threadIdx.x >> 4;
  const int nrb = (nrows + 63) / 64;
  if ((int)blockIdx.x < nrb) {
    int r[4], am[4];
    float c[4];
    bool act[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      r[k] = blockIdx.x * 64 + 16 * k + grp;
      act[k] = r[k] < nrows;
      c[k] = 0.f;
      am[k] = 0;
      if (act[k]) {
        const float cM = -p.rsum[r[k]];
        if (l == 0) {
          if (p.cM_out) p.cM_out[r[k]] = cM;
          if (p.cm_out) p.cm_out[r[k]] = 0.f;
        }
        c[k] = cM * p.scale;
        act[k] = USE_M && p.n_max[r[k]] == 1;  // tied rows' keys come from the tie list
        am[k] = p.arg_max[r[k]];
      }
    }
    if constexpr (USE_M) {
      float4 k4[4], q4[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (act[k]) {
          const int bh = r[k] / p.T;
          k4[k] = __ldg(reinterpret_cast<const float4*>(p.K + ((size_t)bh * p.T + am[k]) * 64 + 4 * l));
          q4[k] = __ldg(reinterpret_cast<const float4*>(p.Q + (size_t)r[k] * 64 + 4 * l));
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (act[k]) {
          const int bh = r[k] / p.T;
          red_add_v4(p.dQ + (size_t)r[k] * 64 + 4 * l, c[k] * k4[k].x, c[k] * k4[k].y, c[k] * k4[k].z,
                     c[k] * k4[k].w);
          red_add_v4(p.dK + ((size_t)bh * p.T + am[k]) * 64 + 4 * l, c[k] * q4[k].x, c[k] * q4[k].y,
                     c[k] * q4[k].z, c[k] * q4[k].w);
        }
      }
    }
  } else if constexpr (USE_M) {
    // the tied maxima: c_M / n_max of row i at each listed key j
    const int cnt = min(*p.tie_count, p.tie_cap);
    for (int e = (blockIdx.x - nrb) * 16 + grp; e < cnt; e += EXT_TIE_BLOCKS * 16) {
      const int2 rj = p.tie_list[e];
      const int rr = rj.x, bh = rr / p.T;
      const float cc = -p.rsum[rr] / (float)p.n_max[rr] * p.scale;
      const size_t kr = ((size_t)bh * p.T + rj.y) * 64 + 4 * l, qr = (size_t)rr * 64 + 4 * l;
      const float4 k4 = __ldg(reinterpret_cast<const float4*>(p.K + kr));
      const float4 q4 = __ldg(reinterpret_cast<const float4*>(p.Q + qr));
      red_add_v4(p.dQ + qr, cc * k4.x, cc * k4.y, cc * k4.z, cc * k4.w);
      red_add_v4(p.dK + kr, cc * q4.x, cc * q4.y, cc * q4.z, cc * q4.w);
    }
  }
}

template <class K>
static cudaError_t launch_fused_k(K kern, dim3 grid, const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s,
                                  const Sched& sch) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, grid, dim3(NTHR_FUSED), smem_bytes, s, maps, p, sch);
}

template <int CAL, int REC>
static cudaError_t launch_fused_modes(dim3 grid, const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s,
                                      const Sched& sch) {
  const bool full = p.grad != GRAD_DETACH && p.grad != GRAD_DETACH_PROJ;
  if constexpr (CAL == CAL_SOFTMAX) {
    return launch_fused_k(k_bwd_fused<CAL_SOFTMAX, REC_LERP, false>, grid, maps, p, smem_bytes, s, sch);
  } else {
    return full ? launch_fused_k(k_bwd_fused<CAL, REC, true>, grid, maps, p, smem_bytes, s, sch)
                : launch_fused_k(k_bwd_fused<CAL, REC, false>, grid, maps, p, smem_bytes, s, sch);
  }
}

cudaError_t launch_bwd_fused(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch) {
  const dim3 grid((unsigned)p.ngrid);
  const bool near = p.recon == REC_NEAREST;
  switch (p.calib) {
    case CAL_SOFTMAX: return launch_fused_modes<CAL_SOFTMAX, REC_LERP>(grid, maps, p, smem_bytes, s, sch);
    case CAL_EXP8: return launch_fused_modes<CAL_EXP8, REC_LERP>(grid, maps, p, smem_bytes, s, sch);
    case CAL_EXPB: return launch_fused_modes<CAL_EXPB, REC_LERP>(grid, maps, p, smem_bytes, s, sch);
    case CAL_FWMR:
      return near ? launch_fused_modes<CAL_FWMR, REC_NEAREST>(grid, maps, p, smem_bytes, s, sch)
                  : launch_fused_modes<CAL_FWMR, REC_LERP>(grid, maps, p, smem_bytes, s, sch);
    case CAL_FWM:
      return near ? launch_fused_modes<CAL_FWM, REC_NEAREST>(grid, maps, p, smem_bytes, s, sch)
                  : launch_fused_modes<CAL_FWM, REC_LERP>(grid, maps, p, smem_bytes, s, sch);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_bwd_ext(const Params& p, cudaStream_t s) {
  const int nrb = (int)(((size_t)p.BH * p.T + 63) / 64);
  const bool use_M = p.grad != GRAD_MIN_ONLY;
  const dim3 grid((unsigned)(nrb + (use_M ? EXT_TIE_BLOCKS : 0))), block(256);
  return use_M ? launch_pdl(k_bwd_ext<true>, grid, block, 0, s, p) : launch_pdl(k_bwd_ext<false>, grid, block, 0, s, p);
}

}  // namespace kint
