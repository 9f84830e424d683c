// Backward of K-interval attention on sm_103a (App. B).
//
// k_bwd_dq   (one CTA per 128-row query block, a thread per query row and
//   column half): per 64-key tile, S = Q K^T and g = dO V^T on the tensor
//   cores, then the own-score term dS_own = gamma Delta with
//   gamma = (g - <g>_{P*}) / W* (normalization Jacobian) and Delta the LERP
//   secant (e_{r+1} - e_r) / h, and dQ += dS_own K.  The row's calibration sums
//   complete at the end of the row; it then adds c_M / n_max (and c_m / n_min)
//   times the arg-extremum keys to dQ (Eq. full) and writes a 64-byte record of
//   the row's constants for the second kernel.
// k_bwd_dkdv (one CTA per 128-key block, a thread per key and column half): per
//   64-query tile, S^T and g^T, the forward P and the full dS (extremum terms
//   now known), and dV += P^T dO, dK += dS^T Q.
// Both: compute warps 0-7, an MMA-issuing warp 8, a TMA/bulk-copy producer warp
// 9; tiles change hands through mbarriers only.
#include "kint_bwd_common.cuh"

namespace kint {

// ---------------------------------------------------------------------------
// dQ kernel element work on one 32-key chunk of one row.
// Returns dS_own in out[]; accumulates sum dS_own and sum gamma dw/dm.
//   dw/dm = A_r + t B_r, A_r = (1 - r/K)(e_r - Delta),
//   B_r = (1 - r/K)(e_{r+1} - e_r) - (e_{r+1} - Delta)/K   (Eq. calgrad per interval)
// ---------------------------------------------------------------------------
template <int CAL, bool FULLG, bool DIAG, int W>
__device__ __forceinline__ void dq_chunk(const float (&sv)[W], const float (&gv)[W], float (&out)[W], int j0,
                                         int i, float k1, float c0, float inv_h, float ga, float gb, bool nogrid,
                                         float Kf, float fk, uint32_t tab, float sk1, float sc0, float invWf,
                                         float hl, float b0l, float& own, float& cm) {
#pragma unroll
  for (int jj = 0; jj < W; ++jj) {
    float ds, dm = 0.f;
    if constexpr (CAL == CAL_SOFTMAX) {
      const float pr = ex2_approx(__fmaf_rn(sv[jj], sk1, sc0)) * invWf;
      ds = pr * __fmaf_rn(gv[jj], ga, gb);  // P (g - <g>_P)
    } else if constexpr (CAL == CAL_EXP8) {
      // gamma e^{z}: the exponential's derivative through the rounding's identity surrogate
      ds = ex2_approx(__fmaf_rn(sv[jj], sk1, sc0)) * __fmaf_rn(gv[jj], ga, gb);
    } else if constexpr (CAL == CAL_EXPB) {
      // the bfloat16 chain rule: bf16(bf16(gamma) w), w = bf16(e^{bf16(z)}); k1, c0 = scale, -M
      float zb;
      const float w = bf16_exp_weight(__fadd_rn(__fmul_rn(sv[jj], k1), c0), zb);
      ds = bf16_rn(__fmul_rn(bf16_rn(__fmaf_rn(gv[jj], ga, gb)), w));
    } else if constexpr (fwm_like(CAL)) {
      // k1, c0 doubled (v = 2u), Kf = 2K, tab: the half-bin table of Delta_r / h (4-byte entries)
      const float v = __fmaf_rn(sv[jj], k1, c0);
      const uint32_t qb = fwm_half_bits(v, Kf);
      float dl = lds_f32(tab + qb * 4u);
      if constexpr (CAL == CAL_FWMR) {
        // resolved: below the window the secant of the continued grid (u = v / 2 exactly)
        const BelowPair bp = resolved_below(__fmul_rn(v, 0.5f), hl, b0l);
        dl = v < 0.0f ? __fmul_rn(__fsub_rn(bp.e1, bp.e0), inv_h) : dl;
      }
      ds = __fmaf_rn(gv[jj], ga, gb) * dl;
    } else {
      const float u = __fmaf_rn(sv[jj], k1, c0);
      float t, rf;
      uint32_t rb;
      decode_u(u, Kf, t, rb, rf);
      const float2 e = lds_f2(tab + rb * 1024u);
      const float de = __fsub_rn(e.y, e.x);
      const float dlt = de * inv_h;
      const float gam = __fmaf_rn(gv[jj], ga, gb);
      ds = gam * dlt;
      if constexpr (FULLG) {
        const float ar = __fmaf_rn(rf, -fk, 1.0f);
        const float A = ar * __fsub_rn(e.x, dlt);
        const float Bc = __fmaf_rn(ar, de, -fk * __fsub_rn(e.y, dlt));
        dm = gam * __fmaf_rn(t, Bc, A);
        dm = nogrid ? 0.f : dm;
      }
      ds = nogrid ? 0.f : ds;
    }
    if constexpr (DIAG) {
      const bool ok = (j0 + jj) <= i;
      ds = ok ? ds : 0.f;
      dm = ok ? dm : 0.f;
    }
    if constexpr (CAL != CAL_SOFTMAX) own += ds;  // (detached too: the P1 row mean)
    if constexpr (FULLG && CAL == CAL_MINMAX) cm += dm;
    out[jj] = ds;
  }
}

// Warp-cooperative gather of one 128-byte row segment per lane into the warp's 4 KB smem
// slot: lane l passes the address of its segment (null: zeros).  Each asynchronous copy
// instruction moves four whole segments (eight lanes each, 16 bytes per lane); 16-byte
// chunks are swizzled by row, so both the copies and the reads are conflict-free.
// gather_rows128_issue starts the copies; gather_rows128_read waits for them and hands
// lane l its segment.
__device__ __forceinline__ void gather_rows128_issue(const float* mine, float4* slot) {
  const int l = threadIdx.x & 31;
  const unsigned long long mp = reinterpret_cast<unsigned long long>(mine);
  __syncwarp();  // the slot's previous contents have been read
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int r = 4 * k + (l >> 3), ch = l & 7;
    const unsigned long long src = __shfl_sync(0xffffffffu, mp, r);
    const uint32_t dst = smem_u32(slot + r * 8 + (ch ^ (r & 7)));
    const unsigned long long gsrc = src ? src + 16ull * ch : mp;  // any valid address when zero-filled
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(gsrc), "r"(src ? 16 : 0)
                 : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void gather_rows128_read(const float4* slot, float4 (&out)[8]) {
  const int l = threadIdx.x & 31;
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncwarp();
#pragma unroll
  for (int q = 0; q < 8; ++q) out[q] = slot[l * 8 + (q ^ (l & 7))];
}

// Adds key rows j0 + b (b a set bit of `mask`) of K (rows of d floats from `k0`) to
// the tie sum `acc` (rare path, kept rolled).
__device__ __forceinline__ void add_tied_keys(uint32_t mask, float* acc, const float* k0, int d) {
#pragma unroll 1
  while (mask) {
    const int b = __ffs(mask) - 1;
    mask &= mask - 1;
    const float* kr = k0 + (size_t)b * d;
#pragma unroll 1
    for (int k = 0; k < d; ++k) atomicAdd(&acc[k], kr[k]);
  }
}

// MMA thread of k_bwd_dq: wait for key tile kt, then S_b = Q K^T and g_b = dO V^T
// into score buffer b = kt % nbuf.
__device__ __forceinline__ bool dq_issue_sg(const Params& p, RingPos stg, int b, uint64_t* bar_full,
                                            uint64_t* bar_sfull, const uint8_t* st0, uint32_t cQa, uint32_t cdOa,
                                            uint32_t cSG, int ktile) {
  const int D = p.d, s = stg.i, parts = p.x3 ? 2 : 1;
  if (!mbar_wait_warp(&bar_full[s], stg.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) return false;
  tc_fence_after();
  const uint8_t* sk = st0 + s * p.sm_stage_bytes;
  const uint8_t* sv = sk + parts * ktile;
  const uint32_t cS = cSG + 128 * b, cG = cS + 64;
  if (p.x3) {
    mma_tmem_smem(cS, cQa + D, sk, BT, D, false);     // Q_lo K_hi
    mma_tmem_smem(cS, cQa, sk + ktile, BT, D, true);  // Q_hi K_lo
    mma_tmem_smem(cS, cQa, sk, BT, D, true);          // Q_hi K_hi
    mma_tmem_smem(cG, cdOa + D, sv, BT, D, false);
    mma_tmem_smem(cG, cdOa, sv + ktile, BT, D, true);
    mma_tmem_smem(cG, cdOa, sv, BT, D, true);
  } else {
    mma_tmem_smem(cS, cQa, sk, BT, D, false);
    mma_tmem_smem(cG, cdOa, sv, BT, D, false);
  }
  mma_commit(&bar_sfull[b]);
  return true;
}

// ---------------------------------------------------------------------------
// k_bwd_dq.
// TMEM: Q [0, dp), dO [dp, 2dp) (dp = d, or 2d for 3xTF32 hi|lo; loaded by the
// compute threads), then per score buffer b: S_b at 2dp + 128 b (64 columns), g_b
// right after it (64 columns); dQ at 2dp + 128 nbuf.  dS overwrites S_b (its tf32
// lo part, under 3xTF32, overwrites g_b).
// smem: stages {K [64 x d], V [64 x d], K^T [d x 64]} (hi[, lo] each) at
// sm_stage0; the grid pair table at sm_table; exchange words at sm_rows.
// ---------------------------------------------------------------------------
// Producer warp of k_bwd_dq: TMA-stores the dQ tile of its k-th item, which the compute
// warps staged at `tile`, and returns once it has been read out.
__device__ __forceinline__ bool store_staged_dq(const Maps& maps, const Params& p, uint64_t* bar_ostg, int k,
                                                const uint8_t* tile) {
  if (!mbar_wait_warp(bar_ostg, k & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) return false;
  const int item = snake_item(k), qb = p.nqb - 1 - item / p.BH, bh = item % p.BH;
  store_rows_tile_boxed(tile, &maps.dq, p.d, 64, qb * 128, bh, false);
  tma_store_wait_read();
  return true;
}

template <int CAL, bool FULLG>
__global__ void __launch_bounds__(NTHR_DQ, 1) k_bwd_dq(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  if (p.gate != nullptr) {
    // launched on one side of a device-side decision: when the single-pass backward ran
    // instead, leave before any set-up (no barrier, no tensor memory)
    pdl_wait();
    if (gated_off(p)) return;
  }
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1, NS = p.nstage, nbuf = p.nbuf;
  const int ktile = BT * D * 4;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_full = bars;               // [NS]
  uint64_t* bar_empty = bars + NS;         // [NS]
  uint64_t* bar_sfull = bars + 2 * NS;     // [2]
  uint64_t* bar_pready = bars + 2 * NS + 2;  // [2]
  uint64_t* bar_done = bars + 2 * NS + 4;
  uint64_t* bar_ops = bars + 2 * NS + 5;  // Q / dO rows stored in TMEM by every compute warp (per item)
  uint64_t* bar_stg = bars + 2 * NS + 6;   // Q / dO tiles staged in smem by TMA (per item)
  uint64_t* bar_ostg = bars + 2 * NS + 7;  // an item's dQ tile staged in the Q / dO area
  // K and V of a stage are free once S, g of the tile completed (the compute warps, which
  // waited for them, arrive); K^T once the dQ product reading it completes (bar_empty)
  uint64_t* bar_emptyA = bars + 2 * NS + 8;  // [NS]
  // score buffer b free again: the dQ product that read its dS completed (MMA2 -> MMA warp)
  uint64_t* bar_dqdone = bars + 3 * NS + 8;  // [2]
  uint64_t* bar_drain = bars + 3 * NS + 10;  // the clean-up commits of the two MMA warps
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 3 * NS + 11);
  float* xch = reinterpret_cast<float*>(sm + p.sm_rows);  // [8][128]
  const int tid = threadIdx.x, warp = warp_id_uniform();
  constexpr int W = BT / NCG;  // key columns per thread per tile
  const int dp = D * parts;
  const int cQ = 0, cdO = dp, cSG0 = 2 * dp, cdQ = cSG0 + 128 * nbuf;

  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_empty[s], 1);
      mbar_init(&bar_emptyA[s], NCOMP / 32);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar_sfull[b], 1);
      mbar_init(&bar_pready[b], NCOMP / 32);
      mbar_init(&bar_dqdone[b], 1);
    }
    mbar_init(bar_done, 1);
    mbar_init(bar_ops, NCOMP / 32);
    mbar_init(bar_stg, 1);
    mbar_init(bar_ostg, NCOMP / 32);
    mbar_init(bar_drain, 2);
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

  if (warp == PRODUCER_WARP) {
    int gt = 0, n = 0;
    RingPos ld;  // stage of the next tile loaded
    bool ok = true;
    // Q / dO of this CTA's k-th item into the staging area (TF32 at d = 64)
    int staged = 0;  // staging loads issued
    auto stage_ops = [&](int k) {
      const int it_ = snake_item(k), qb_ = p.nqb - 1 - it_ / p.BH, bh_ = it_ % p.BH;
      mbar_arrive_expect_tx(bar_stg, 2 * 128 * D * 4);
      load_rows_tile_boxed(sm + p.sm_a, &maps.q, bar_stg, D, 128, BT, 0, qb_ * 128, bh_);
      load_rows_tile_boxed(sm + p.sm_a + 128 * D * 4, &maps.dout, bar_stg, D, 128, BT, 0, qb_ * 128, bh_);
      staged = k + 1;
    };
    if (p.ops_smem && snake_item(0) < p.nitems) stage_ops(0);
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH;
      const int nkt = min(2 * qb + 2, (p.T + BT - 1) / BT);
      for (int kt = 0; kt < nkt; ++kt, ++gt, ld.next(NS)) {
        const int s = ld.i;
        if (gt >= NS && !mbar_wait_warp(&bar_emptyA[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        uint64_t* b = &bar_full[s];
        mbar_arrive_expect_tx(b, 3 * parts * ktile);
        load_rows_tile(dst, &maps.k, b, D, BT, 0, kt * BT, bh);
        load_rows_tile(dst + parts * ktile, &maps.v, b, D, BT, 0, kt * BT, bh);
        if (p.x3) {
          load_rows_tile(dst + ktile, &maps.k_lo, b, D, BT, 0, kt * BT, bh);
          load_rows_tile(dst + parts * ktile + ktile, &maps.v_lo, b, D, BT, 0, kt * BT, bh);
        }
        if (gt >= NS && !mbar_wait_warp(&bar_empty[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        load_rows_tile(dst + 2 * parts * ktile, &maps.kt, b, BT, D, kt * BT, 0, bh);
        if (p.x3) load_rows_tile(dst + 2 * parts * ktile + ktile, &maps.kt_lo, b, BT, D, kt * BT, 0, bh);
        // The next item's Q / dO, as soon as the stage ring holds this item's first tiles: it needs
        // this item's Q / dO copied out into TMEM and the previous item's dQ tile, staged in the
        // same area since, stored; both happen at the end of the previous item, so the load has
        // this whole item to land.
        if (p.ops_smem && kt == min(nkt, NS) - 1 && snake_item(n + 1) < p.nitems) {
          if (!mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) ||
              (n >= 1 && !store_staged_dq(maps, p, bar_ostg, n - 1, sm + p.sm_a))) {
            ok = false;
            break;
          }
          stage_ops(n + 1);
        }
      }
    }
    // the last-but-one item's tile (the last item's is stored by the compute warps)
    if (p.ops_smem && ok && n >= 2) store_staged_dq(maps, p, bar_ostg, n - 2, sm + p.sm_a);
    tma_store_wait_all();
    // clean-up: the last tiles issued have landed
    drain_ring(bar_full, ld, gt, NS, p.wait_ns, p.status);
    if (staged > 0) mbar_wait_warp(bar_stg, (staged - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
  } else if (warp == MMA_WARP) {
    // S, g of every tile, into score buffer b once the dQ product that read the buffer's
    // previous dS has completed (bar_dqdone)
    const uint8_t* st0 = sm + p.sm_stage0;
    const uint32_t cQa = tmem + cQ, cdOa = tmem + cdO, cSG = tmem + cSG0;
    int n = 0, g = 0;
    RingPos is, ib;  // stage and buffer of the next S, g product
    bool ok = true;
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH;
      const int nkt = min(2 * qb + 2, (p.T + BT - 1) / BT);
      // Q / dO of the item in TMEM (copied by the compute warps once the previous item's
      // last S, g were read)
      ok = mbar_wait_warp(bar_ops, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC);
      if (ok) tc_fence_after();
      for (int kt = 0; kt < nkt && ok; ++kt, ++g, is.next(NS), ib.next(nbuf)) {
        if (g >= nbuf &&
            !mbar_wait_warp(&bar_dqdone[ib.i], ib.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          ok = false;
          break;
        }
        ok = dq_issue_sg(p, is, ib.i, bar_full, bar_sfull, st0, cQa, cdOa, cSG, ktile);
      }
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else if (warp == MMA2_WARP) {
    // dQ += dS K of every tile once the compute warps wrote its dS
    RingPos cs, cb;  // stage and buffer of the tile being finished
    int n = 0;
    bool ok = true;
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH;
      const int nkt = min(2 * qb + 2, (p.T + BT - 1) / BT);
      for (int kt = 0; kt < nkt && ok; ++kt, cs.next(NS), cb.next(nbuf)) {
        const int b = cb.i, s = cs.i;
        if (!mbar_wait_warp(&bar_pready[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* skt = sm + p.sm_stage0 + s * p.sm_stage_bytes + 2 * parts * ktile;
        const uint32_t cS = tmem + cSG0 + 128 * b, cG = cS + 64;
        const bool acc = kt > 0;
        if (p.x3) {
          mma_tmem_smem(tmem + cdQ, cS, skt, D, BT, acc);           // dS_hi K_hi
          mma_tmem_smem(tmem + cdQ, cS, skt + ktile, D, BT, true);  // dS_hi K_lo
          mma_tmem_smem(tmem + cdQ, cG, skt, D, BT, true);          // dS_lo K_hi
        } else {
          mma_tmem_smem(tmem + cdQ, cS, skt, D, BT, acc);
        }
        mma_commit(&bar_empty[s]);
        mma_commit(&bar_dqdone[b]);
      }
      mma_commit(bar_done);
    }
    drain_mma(bar_drain, p.wait_ns, p.status);
  } else {
    // ---- compute warps: items one after the other ----
    const int row = tid & 127, cg = (tid >> 7) & (NCG - 1);
    // Operand rows of the n-th item into TMEM (column group 0 takes Q, group 1 takes dO),
    // handed to the MMA warp through bar_ops.  TF32 at d = 64: from the tiles the producer
    // staged in smem; otherwise from global rows.  The next item's rows go in as soon as
    // the current item's last S, g have been read (before its dQ epilogue), so the next
    // item's first products run under that epilogue.
    auto ops_to_tmem = [&](int n) {
      const int item = snake_item(n);
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, i = qb * 128 + row;
      if (p.ops_smem) {
        if (mbar_wait(bar_stg, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA))
          staged_row_to_tmem(tmem, cg == 0 ? cQ : cdO, sm + p.sm_a + (cg == 0 ? 0 : 128 * D * 4), row, D);
      } else {
        row_to_tmem(tmem, cg == 0 ? cQ : cdO, cg == 0 ? p.Q : p.dO, bh * p.T + i, i < p.T ? (bh + 1) * p.T : 0, D,
                    p.x3 != 0);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if ((tid & 31) == 0) mbar_arrive(bar_ops);
    };
    // The row statistics of an item, loaded one item ahead (under the previous item's epilogue).
    struct RowIn {
      float M = 0.f, m = 0.f, Wf = 1.f, Ws = 1.f, Dg = 0.f;
      int nmax = 1, nmin = 1, amax = 0, amin = 0;
    };
    // They arrive by asynchronous copies into this thread's slot of a [9][NCOMP] word array,
    // issued at the start of the previous item, so their latency hides under its tiles.
    const bool prob = (p.recon == REC_NEAREST && p.ste == 1 && !gridless(CAL));
    const uint32_t rslot = smem_u32(sm + p.sm_rstat) + 4u * (uint32_t)tid;
    auto prefetch_row_stats = [&](int n) {
      const int item = snake_item(n);
      const int i = (p.nqb - 1 - item / p.BH) * 128 + row;
      if (i < p.T) {
        const size_t rw = (size_t)(item % p.BH) * p.T + i;
        const void* src[9] = {p.row_max + rw, p.row_min + rw, p.W + rw, p.n_max + rw, p.n_min + rw,
                              p.arg_max + rw, p.arg_min + rw, p.gbar + rw, (prob ? p.W_lerp : p.W) + rw};
#pragma unroll
        for (int k = 0; k < 9; ++k)
          asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(rslot + (uint32_t)k * 4u * NCOMP),
                       "l"(src[k])
                       : "memory");
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    };
    auto load_row_stats = [&](int n) {
      RowIn r;
      const int item = snake_item(n);
      const int i = (p.nqb - 1 - item / p.BH) * 128 + row;
      asm volatile("cp.async.wait_all;" ::: "memory");
      if (i < p.T) {
        r.M = lds_f32(rslot);
        r.m = lds_f32(rslot + 4u * NCOMP);
        r.Wf = lds_f32(rslot + 8u * NCOMP);
        r.nmax = __float_as_int(lds_f32(rslot + 12u * NCOMP));
        r.nmin = __float_as_int(lds_f32(rslot + 16u * NCOMP));
        r.amax = __float_as_int(lds_f32(rslot + 20u * NCOMP));
        r.amin = __float_as_int(lds_f32(rslot + 24u * NCOMP));
        r.Dg = lds_f32(rslot + 28u * NCOMP);  // <g>_{P*} = dO_i . O*_i
        r.Ws = lds_f32(rslot + 32u * NCOMP);
      }
      return r;
    };
    int n = 0;
    RingPos cb, cs;  // score buffer and stage of the current tile
    bool failed = false;
    RowIn nx;
    if (snake_item(0) < p.nitems) {
      prefetch_row_stats(0);
      ops_to_tmem(0);
      nx = load_row_stats(0);
    }
    for (int item = snake_item(n); item < p.nitems && !failed; item = snake_item(++n)) {
      // ---- set-up: row constants, grid table (the operands are in TMEM already) ----
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH;
      const int nkt = min(2 * qb + 2, (p.T + BT - 1) / BT);
      const int i = qb * 128 + row;
      const bool row_ok = i < p.T;
      const size_t rw = (size_t)bh * p.T + (row_ok ? i : 0);
      const float M = nx.M, m = nx.m, Wf = nx.Wf, Ws = nx.Ws, Dg = nx.Dg;
      const int nmax = nx.nmax, nmin = nx.nmin, amax = nx.amax, amin = nx.amin;
      if (snake_item(n + 1) < p.nitems) prefetch_row_stats(n + 1);  // (the slot was just read)
      const RowGrid g = row_grid(p, M, m);
      if constexpr (fwm_like(CAL)) {  // the same for every item
        if (n == 0 && tid < 2 * Kq + 1 + kHalfTail)
          *reinterpret_cast<float*>(sm + p.sm_table + tid * 4) = fwm_half_entry(p, tid - kHalfTail).y;
      } else if constexpr (CAL == CAL_MINMAX) {
        for (int r = cg; r < Kq; r += NCG) {
          const float2 e = make_float2(grid_value(p, g, r), grid_value(p, g, r + 1));
          *reinterpret_cast<float2*>(sm + p.sm_table + (size_t)r * 1024 + row * 8) = e;
          if (row_ok) *reinterpret_cast<float2*>(p.rtab + (rw * p.Kp + r) * 2) = e;
        }
      }
      // the arg-extremum key rows the epilogue reads, into L2 ahead of it
      if (FULLG && CAL != CAL_SOFTMAX && row_ok) {
        prefetch_l2(p.K + ((size_t)bh * p.T + amax) * D + cg * (D / NCG));
        if (CAL == CAL_MINMAX) prefetch_l2(p.K + ((size_t)bh * p.T + amin) * D + cg * (D / NCG));
      }
      const float ga = CAL == CAL_SOFTMAX ? 1.0f : 1.0f / Ws;
      const float gb = CAL == CAL_SOFTMAX ? -Dg : -Dg * ga;
      const float invWf = 1.0f / Wf;
      const float sk1 = p.scale * kLog2e, sc0 = -M * kLog2e;
      // FWM: the half-bin table, entry q at sm_table + 4 (q + 2), addressed by the bits
      // 0x4B000000 + q of floor(2u) (0x4B000000 * 4 = 0x2C000000 mod 2^32), and the doubled
      // position v = 2u; MinMax: this row's pair table, r * 1024 apart
      const float Kf = (float)(fwm_like(CAL) ? 2 * Kq : Kq), fk = 1.0f / (float)Kq;
      const float k1q = fwm_like(CAL) ? 2.0f * g.k1 : g.k1, c0q = fwm_like(CAL) ? 2.0f * g.c0 : g.c0;
      const uint32_t tab = fwm_like(CAL) ? smem_u32(sm + p.sm_table) + 4u * kHalfTail - 0x2C000000u
                                            : smem_u32(sm + p.sm_table) + (uint32_t)row * 8u;
      const bool minmax = CAL == CAL_MINMAX;
      const bool track = FULLG && CAL != CAL_SOFTMAX && row_ok && !g.nogrid && (nmax > 1 || (minmax && nmin > 1));
      float* tie_max = p.tie_acc + rw * D;
      float* tie_min = p.tie_acc + ((size_t)p.BH * p.T + rw) * D;
      if (track && cg == 0) {
        for (int k = 0; k < D; ++k) tie_max[k] = tie_min[k] = 0.f;
        atomicOr(p.tileflags + (size_t)bh * p.nqt + i / BT, 1);
      }
      // the grid table, and the zeroed tie sums (every column group of a row may add to them)
      group_sync(BAR_COMPUTE, NCOMP);
      float own = 0.f, cm = 0.f;
      for (int kt = 0; kt < nkt; ++kt, cb.next(nbuf)) {
        const int b = cb.i;
        const bool ok = mbar_wait(&bar_sfull[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
        if (!ok) {
          failed = true;
          break;
        }
        // S, g of the tile completed: its K and V may be reloaded
        if ((tid & 31) == 0) mbar_arrive(&bar_emptyA[cs.i]);
        cs.next(NS);
        tc_fence_after();
        const int cS = cSG0 + 128 * b + cg * W, cG = cS + 64;
        float sv[W], gv[W], out[W];
        tmem_ldw<W>(lane_addr(tmem, cS), sv);
        tmem_ldw<W>(lane_addr(tmem, cG), gv);
        tmem_ld_wait();
        const int j0 = kt * BT + cg * W;
        if (j0 + W - 1 > qb * 128)
          dq_chunk<CAL, FULLG, true, W>(sv, gv, out, j0, i, k1q, c0q, g.inv_h, ga, gb, g.nogrid, Kf, fk, tab, sk1,
                                        sc0, invWf, g.hl, g.b0l, own, cm);
        else
          dq_chunk<CAL, FULLG, false, W>(sv, gv, out, j0, i, k1q, c0q, g.inv_h, ga, gb, g.nogrid, Kf, fk, tab,
                                         sk1, sc0, invWf, g.hl, g.b0l, own, cm);
        if (__any_sync(0xffffffffu, track)) {
          // rare: tied extrema, the tie set is found by equality on the recomputed scores
          uint32_t mk_max = 0, mk_min = 0;
  #pragma unroll
          for (int jj = 0; jj < W; ++jj) {
            const float s = __fmul_rn(sv[jj], p.scale);
            const bool okj = track && j0 + jj <= i;
            mk_max |= (okj && nmax > 1 && s == M) ? (1u << jj) : 0u;
            mk_min |= (okj && minmax && nmin > 1 && s == m) ? (1u << jj) : 0u;
          }
          add_tied_keys(mk_max, tie_max, p.K + ((size_t)bh * p.T + j0) * D, D);
          add_tied_keys(mk_min, tie_min, p.K + ((size_t)bh * p.T + j0) * D, D);
        }
        if (p.x3) {
          float lo[W];
  #pragma unroll
          for (int q = 0; q < W; ++q) {
            const float h = tf32_rna(out[q]);
            lo[q] = __fsub_rn(out[q], h);
            out[q] = h;
          }
          tmem_stw<W>(lane_addr(tmem, cG), lo);
        }
        tmem_stw<W>(lane_addr(tmem, cS), out);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_pready[b]);
      }
      // the next item's Q / dO (this item's S, g have all been read: the last tile's were)
      // and its row statistics
      if (!failed && snake_item(n + 1) < p.nitems) {
        ops_to_tmem(n + 1);
        nx = load_row_stats(n + 1);
      }
      if (p.ops_smem && FULLG && CAL != CAL_SOFTMAX) {
        // the epilogue's arg-max key rows (this thread's column half), gathered into the dO half
        // of the staging area (read by every warp's copy above: hence the barrier) while the
        // item's last product completes
        group_sync(BAR_COMPUTE, NCOMP);
        const bool own_row = !failed && row_ok && !g.nogrid && nmax == 1;
        gather_rows128_issue(own_row ? p.K + ((size_t)bh * p.T + amax) * D + cg * (D / NCG) : nullptr,
                             reinterpret_cast<float4*>(sm + p.sm_a + 128 * D * 4) + warp * 256);
      }
      const bool dok = !failed && mbar_wait(bar_done, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
      failed = group_any(BAR_COMPUTE, NCOMP, !dok);
      if (!failed) {
        tc_fence_after();
        xch[cg * 128 + row] = own;
        xch[(NCG + cg) * 128 + row] = cm;
        group_sync(BAR_COMPUTE, NCOMP);
        float own_t = 0.f, cm_t = 0.f;
  #pragma unroll
        for (int q = 0; q < NCG; ++q) {
          own_t += xch[q * 128 + row];
          cm_t += xch[(NCG + q) * 128 + row];
        }
        // Eq. (full): c_m = sum gamma dw/dm; c_M = -sum gamma Delta - c_m (Delta + dw/dM + dw/dm = 0);
        // FWM: c_M = -sum_window gamma Delta.  Split evenly over tied keys; the single-channel
        // modes (max_only, min_only) apply one of the two sums.
        const bool full = FULLG && CAL != CAL_SOFTMAX && !g.nogrid;
        const float cmv = (full && minmax) ? cm_t : 0.f;
        const float cMv = full ? (-own_t - cmv) : 0.f;
        const bool use_M = p.grad != GRAD_MIN_ONLY, use_m = p.grad != GRAD_MAX_ONLY;
        // P1 control (detached, App. B): dS_ij - mu_i over the causal row, mu_i = sum_j dS_ij / (i + 1),
        // adds -mu_i C_i to dQ_i, C_i = sum_{j<=i} K_j (prefix sums, in the tie-sum buffer, which
        // the detached modes do not use); the dK/dV pass subtracts mu_i from every causal dS_ij
        const bool p1 = !FULLG && CAL != CAL_SOFTMAX && p.grad == GRAD_DETACH_PROJ;
        const float mu = p1 ? own_t / (float)(i + 1) : 0.f;
        // (n_min is 0 where the minimum side was not computed, and c_m is 0 there)
        const float cMn = p1 ? -mu : (use_M ? cMv / (float)nmax : 0.f);
        const float cmn = (use_m && minmax && nmin > 0) ? cmv / (float)nmin : 0.f;
        const float* kmax = p1 ? tie_max : (nmax == 1) ? p.K + ((size_t)bh * p.T + amax) * D : tie_max;
        const float* kmin = (nmin == 1) ? p.K + ((size_t)bh * p.T + amin) * D : tie_min;
        // dQ rows into a swizzled tile for a TMA store: in the Q / dO staging area (free now
        // that the next item's Q / dO are in TMEM; the producer stores it before it stages
        // the item after next), or, for the last item, in the idle stage ring (stored here).
        // Without the staging area (3xTF32, d = 128) straight to global memory.
        const bool last = snake_item(n + 1) >= p.nitems;
        uint8_t* stg = last ? sm + p.sm_stage0 : sm + p.sm_a;
        for (int c = cg * (D / NCG); c < (cg + 1) * (D / NCG); c += 32) {
          // the arg-extremum key rows (128 bytes of each: this column half).  With the staging
          // area, the warp gathers its 32 rows cooperatively (four whole lines per load) into
          // its 4 KB slot of the free dO half of that area, then each thread reads its row back;
          // otherwise every thread loads its own row (32 lines per load).
          float4 km[8], kn[8];
          if (p.ops_smem && FULLG && CAL != CAL_SOFTMAX) {
            // the arg-max rows were requested before the wait for the item's last product
            // (tie sums, complete only now, are read directly)
            float4* slot = reinterpret_cast<float4*>(sm + p.sm_a + 128 * D * 4) + warp * 256;
            gather_rows128_read(slot, km);
            if (row_ok && full && nmax > 1) {
  #pragma unroll
              for (int q = 0; q < 8; ++q) km[q] = reinterpret_cast<const float4*>(tie_max + c)[q];
            }
            if (minmax) {
              gather_rows128_issue(full && row_ok ? kmin + c : nullptr, slot);
              gather_rows128_read(slot, kn);
            }
          } else {
  #pragma unroll
            for (int q = 0; q < 8; ++q) {
              km[q] = (row_ok && (full || p1)) ? __ldg(reinterpret_cast<const float4*>(kmax + c) + q)
                                               : make_float4(0.f, 0.f, 0.f, 0.f);
              kn[q] = (row_ok && full && minmax) ? __ldg(reinterpret_cast<const float4*>(kmin + c) + q)
                                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            }
          }
          if (!minmax) {
  #pragma unroll
            for (int q = 0; q < 8; ++q) kn[q] = make_float4(0.f, 0.f, 0.f, 0.f);
          }
          float v[32];
          tmem_ld32(lane_addr(tmem, cdQ + c), v);
          tmem_ld_wait();
  #pragma unroll
          for (int q = 0; q < 8; ++q) {
            v[4 * q] = __fmaf_rn(cmn, kn[q].x, __fmaf_rn(cMn, km[q].x, v[4 * q])) * p.scale;
            v[4 * q + 1] = __fmaf_rn(cmn, kn[q].y, __fmaf_rn(cMn, km[q].y, v[4 * q + 1])) * p.scale;
            v[4 * q + 2] = __fmaf_rn(cmn, kn[q].z, __fmaf_rn(cMn, km[q].z, v[4 * q + 2])) * p.scale;
            v[4 * q + 3] = __fmaf_rn(cmn, kn[q].w, __fmaf_rn(cMn, km[q].w, v[4 * q + 3])) * p.scale;
          }
          if (p.ops_smem) {
            row_to_staged(stg, row, c / 32, v);
          } else if (row_ok) {
            float4* dst = reinterpret_cast<float4*>(p.dQ + rw * D + c);
  #pragma unroll
            for (int q = 0; q < 8; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
        if (p.ops_smem) {
          fence_async_smem();
          if (last) {
            group_sync(BAR_COMPUTE, NCOMP);
            if (warp == 0) store_rows_tile_boxed(stg, &maps.dq, D, 64, qb * 128, bh, false);
          } else {
            __syncwarp();
            if ((tid & 31) == 0) mbar_arrive(bar_ostg);
          }
        }
        if (row_ok && cg == 0) {
          if (p.cM_out) p.cM_out[rw] = cMv;
          if (p.cm_out) p.cm_out[rw] = cmv;
          // the position as the dK/dV pass forms it: softmax log2 e^{s-M}, FWM Nearest 2u, else u
          const bool half = fwm_like(CAL) && p.recon == REC_NEAREST;
          RowRec r;
          r.c0 = exp_like(CAL) ? sc0 : (half ? 2.0f * g.c0 : g.c0);
          r.k1 = exp_like(CAL) ? sk1 : (half ? 2.0f * g.k1 : g.k1);
          r.invWf = invWf;
          r.ga = ga;
          r.gb = gb;
          r.cMn = full ? cMn : mu;  // detached: the P1 row mean (0 without the projection)
          r.amax = (nmax == 1) ? amax : -1;
          r.flags = (g.nogrid ? REC_NOGRID : 0) | (nmax > 1 ? REC_TIEMAX : 0) | (nmin > 1 ? REC_TIEMIN : 0);
          r.inv_h = g.inv_h;
          r.cmn = (full && minmax) ? cmn : 0.f;
          r.amin = (nmin == 1) ? amin : -1;
          r.pad0 = 0;
          r.M = M;
          r.m = m;
          r.pad1 = r.pad2 = 0.f;
          reinterpret_cast<RowRec*>(p.rec)[rw] = r;
        }
      }
    }
    if (warp == 0) tma_store_wait_all();
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------
// Key prefix sums C_i = sum_{j<=i} K_j of every head ([BH][T][d], fp32), for the P1
// control of App. B ("Detach (legacy)"): projecting the detached dS onto the zero-sum
// subspace of each causal row adds -mu_i C_i to dQ_i.  One CTA per (head, 32-column
// slice): its warps take consecutive row segments (lane = column, 128-byte rows), sum
// them, exchange the segment totals through shared memory and write running sums (the
// second pass re-reads the segment, from L2).
// ---------------------------------------------------------------------------
constexpr int KCUM_WARPS = 16;
__global__ void __launch_bounds__(KCUM_WARPS * 32) k_kcum(const float* __restrict__ K, float* __restrict__ C,
                                                          int T, int d) {
  __shared__ float part[KCUM_WARPS][32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nsl = d / 32;
  const int bh = blockIdx.x / nsl, col = (blockIdx.x % nsl) * 32 + lane;
  const int seg = (T + KCUM_WARPS - 1) / KCUM_WARPS;
  const int t0 = min(T, w * seg), t1 = min(T, t0 + seg);
  const float* src = K + (size_t)bh * T * d + col;
  float* dst = C + (size_t)bh * T * d + col;
  pdl_wait();  // (the dQ kernel's wait on this launch then also covers the operand prep)
  float sum = 0.f;
#pragma unroll 4
  for (int t = t0; t < t1; ++t) sum += __ldg(src + (size_t)t * d);
  part[w][lane] = sum;
  __syncthreads();
  pdl_trigger();
  float run = 0.f;
  for (int q = 0; q < w; ++q) run += part[q][lane];
#pragma unroll 4
  for (int t = t0; t < t1; ++t) {
    run += __ldg(src + (size_t)t * d);
    dst[(size_t)t * d] = run;
  }
}

cudaError_t launch_kcum(const float* K, float* C, int BH, int T, int d, cudaStream_t s) {
  return launch_pdl(k_kcum, dim3((unsigned)(BH * (d / 32))), dim3(KCUM_WARPS * 32), 0, s, K, C, T, d);
}

cudaError_t launch_bwd_dq(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  const dim3 grid((unsigned)p.ngrid);
  const bool full = p.grad != GRAD_DETACH && p.grad != GRAD_DETACH_PROJ;
  if (p.calib == CAL_SOFTMAX) return launch3(k_bwd_dq<CAL_SOFTMAX, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
  if (p.calib == CAL_EXP8)
    return full ? launch3(k_bwd_dq<CAL_EXP8, true>, grid, maps, p, smem_bytes, s, NTHR_DQ)
                : launch3(k_bwd_dq<CAL_EXP8, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
  if (p.calib == CAL_EXPB)
    return full ? launch3(k_bwd_dq<CAL_EXPB, true>, grid, maps, p, smem_bytes, s, NTHR_DQ)
                : launch3(k_bwd_dq<CAL_EXPB, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
  if (p.calib == CAL_MINMAX)
    return full ? launch3(k_bwd_dq<CAL_MINMAX, true>, grid, maps, p, smem_bytes, s, NTHR_DQ)
                : launch3(k_bwd_dq<CAL_MINMAX, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
  if (p.calib == CAL_FWMR)
    return full ? launch3(k_bwd_dq<CAL_FWMR, true>, grid, maps, p, smem_bytes, s, NTHR_DQ)
                : launch3(k_bwd_dq<CAL_FWMR, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
  return full ? launch3(k_bwd_dq<CAL_FWM, true>, grid, maps, p, smem_bytes, s, NTHR_DQ)
              : launch3(k_bwd_dq<CAL_FWM, false>, grid, maps, p, smem_bytes, s, NTHR_DQ);
}

}  // namespace kint
