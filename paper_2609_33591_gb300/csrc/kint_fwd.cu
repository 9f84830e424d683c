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

// Row record of the single-pass backward for row rw (position t of head bh) from its row
// max M, forward normalizer Wf, the W* of gamma Ws, tie count nm and <g>_{P*} = dg;
// returns whether this row's tied keys overflow the tie list.
__device__ __forceinline__ bool prep_row_record(const RecJob& R, size_t rw, int bh, int t, float M, float Wf, float Ws,
                                                int nm, float dg) {
  float4 f;
  f.z = R.softmax ? 1.0f : 1.0f / Ws;  // gamma = g * f.z + f.w
  f.w = R.softmax ? -dg : -dg * f.z;
  f.y = 1.0f / Wf;
  if (R.c0_kind == 0) {
    f.x = -M * kLog2e;
  } else if (R.c0_kind == 1) {
    const float c0 = __fmul_rn(__fsub_rn(R.tau, M), R.inv_h);
    f.x = R.half ? 2.0f * c0 : c0;
  } else {
    f.x = -M;
  }
  R.frec[rw] = f;
  R.rsum[rw] = 0.0f;
  // the calibration-sum outputs stay 0 in the modes whose extremum pass does not write them
  if (R.cM_out) R.cM_out[rw] = 0.0f;
  if (R.cm_out) R.cm_out[rw] = 0.0f;
  if (nm <= 1) return false;
  // a row with tied maxima: its 64-row query tile takes the single pass's tie search
  R.tileflags[(size_t)bh * R.nqt + t / 64] = 1;
  return atomicAdd(R.tie_total, nm) + nm > R.tie_cap;
}

// ---------------------------------------------------------------------------
// Operand preparation (HBM-bound).  tcgen05.mma kind::tf32 reads both operands
// K-major, so every second-stage product (P V, dS K, P^T dO, dS^T Q) reads a
// transposed copy X^T [BH][d][Tp].  3xTF32 also needs tf32 hi/lo splits.  A job
// with Y also forms the row dot products dot[t] = X_t . Y_t (the backward's
// <g>_{P*} = dO_i . O*_i, App. B) from the rows it already holds.
// One launch serves up to four tensors.  The work units (job, head, 32-row block)
// are spread over a grid of sixteen CTAs per SM that loop over them, so the launch
// has no partial last wave; a unit moves all d columns in 64-column steps through a
// padded 32 x 65 shared tile (128 threads, four float4 loads and stores each).
// ---------------------------------------------------------------------------
template <bool SPLIT>
__global__ void __launch_bounds__(128) k_prep(const __grid_constant__ PrepJobs jobs, int T, int Tp, int d,
                                              int BH) {
  __shared__ float hs[32][65];
  __shared__ float ls[SPLIT ? 32 : 1][65];
  __shared__ float dots[32];
  const int tid = threadIdx.x;
  const int r = tid >> 4, c4 = tid & 15;  // load phase: rows r + 8 q, columns 4 c4 .. 4 c4 + 3
  const int k = tid >> 3, tq = tid & 7;   // store phase: output rows k + 16 q, keys 4 tq .. 4 tq + 3
  const int ntb = Tp / 32, per_job = BH * ntb, units = jobs.n * per_job;
  pdl_wait();
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const PrepJob& J = jobs.j[u / per_job];
    const int bh = (u % per_job) / ntb, t0 = (u % ntb) * 32;
    const size_t nat = (size_t)bh * T * d, tr = (size_t)bh * d * Tp;
    const bool dotj = J.Y != nullptr;
    const RecJob& R = jobs.rec;
    const bool recj = dotj && R.frec != nullptr;
    // single-pass set-up: this unit's row statistics load under the transposes, and its dQ
    // rows start at zero (the single pass adds its partial sums to them)
    float rM = 0.f, rW = 1.f, rWs = 1.f;
    int rnm = 0;
    if (recj) {
      const int t = t0 + tid;
      if (tid < 32 && t < T) {
        const size_t rw = (size_t)bh * T + t;
        rM = R.row_max[rw];
        rW = R.W[rw];
        rWs = R.Ws[rw];
        rnm = R.n_max[rw];
      }
      const int nr = min(32, T - t0);
      float4* dq = reinterpret_cast<float4*>(R.dQ + nat + (size_t)t0 * d);
      for (int k4 = tid; k4 < nr * d / 4; k4 += 128) dq[k4] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float dacc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int k0 = 0; k0 < d; k0 += 64) {
      float4 x[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int t = t0 + r + 8 * q;
        x[q] = t < T ? __ldg(reinterpret_cast<const float4*>(J.X + nat + (size_t)t * d + k0 + 4 * c4))
                     : make_float4(0.f, 0.f, 0.f, 0.f);
      }
      if (dotj) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int t = t0 + r + 8 * q;
          if (t < T) {
            const float4 y = __ldg(reinterpret_cast<const float4*>(J.Y + nat + (size_t)t * d + k0 + 4 * c4));
            dacc[q] = __fmaf_rn(x[q].x, y.x, dacc[q]);
            dacc[q] = __fmaf_rn(x[q].y, y.y, dacc[q]);
            dacc[q] = __fmaf_rn(x[q].z, y.z, dacc[q]);
            dacc[q] = __fmaf_rn(x[q].w, y.w, dacc[q]);
          }
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int rr = r + 8 * q, t = t0 + rr;
        float4 v = x[q];
        if constexpr (SPLIT) {
          float4 h, l;
          h.x = tf32_rna(v.x); l.x = __fsub_rn(v.x, h.x);
          h.y = tf32_rna(v.y); l.y = __fsub_rn(v.y, h.y);
          h.z = tf32_rna(v.z); l.z = __fsub_rn(v.z, h.z);
          h.w = tf32_rna(v.w); l.w = __fsub_rn(v.w, h.w);
          if (t < T && J.nat_hi) {
            const size_t off = nat + (size_t)t * d + k0 + 4 * c4;
            *reinterpret_cast<float4*>(J.nat_hi + off) = h;
            *reinterpret_cast<float4*>(J.nat_lo + off) = l;
          }
          v = h;
          ls[rr][4 * c4] = l.x; ls[rr][4 * c4 + 1] = l.y; ls[rr][4 * c4 + 2] = l.z; ls[rr][4 * c4 + 3] = l.w;
        }
        hs[rr][4 * c4] = v.x; hs[rr][4 * c4 + 1] = v.y; hs[rr][4 * c4 + 2] = v.z; hs[rr][4 * c4 + 3] = v.w;
      }
      __syncthreads();
      if (J.tr_hi) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int kk = k + 16 * q, t = t0 + 4 * tq;
          const size_t off = tr + (size_t)(k0 + kk) * Tp + t;
          *reinterpret_cast<float4*>(J.tr_hi + off) =
              make_float4(hs[4 * tq][kk], hs[4 * tq + 1][kk], hs[4 * tq + 2][kk], hs[4 * tq + 3][kk]);
          if constexpr (SPLIT) {
            if (J.tr_lo)
              *reinterpret_cast<float4*>(J.tr_lo + off) =
                  make_float4(ls[4 * tq][kk], ls[4 * tq + 1][kk], ls[4 * tq + 2][kk], ls[4 * tq + 3][kk]);
          }
        }
      }
      __syncthreads();
    }
    if (dotj) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float v = dacc[q];
#pragma unroll
        for (int o = 8; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        const int t = t0 + r + 8 * q;
        if (c4 == 0 && t < T) {
          J.dot[(size_t)bh * T + t] = v;
          dots[r + 8 * q] = v;
        }
      }
      if (recj) {
        __syncthreads();  // dots[] (the next unit writes it only after the syncs of its own loop)
        const int t = t0 + tid;
        if (tid < 32 && t < T &&
            prep_row_record(R, (size_t)bh * T + t, bh, t, rM, rW, rWs, rnm, dots[tid]))
          atomicOr(R.tie_any, 1);
      }
    }
  }
}

cudaError_t launch_prep(const PrepJobs& jobs, int BH, int T, int Tp, int d, bool split, int nsm, cudaStream_t s) {
  if (jobs.n <= 0) return cudaSuccess;
  const int units = jobs.n * BH * (Tp / 32);
  // sixteen 128-thread CTAs per SM (the most that are resident): a unit's loads, transpose
  // and stores run one after the other, so the SM hides their latency with other CTAs' units
  dim3 grid((unsigned)(units < 16 * nsm ? units : 16 * nsm)), block(128);
  return launch_pdl(split ? k_prep<true> : k_prep<false>, grid, block, 0, s, jobs, T, Tp, d, BH);
}

// ---------------------------------------------------------------------------
// Pass 1: row extrema (App. A: M = max_j s_j, m = min_j s_j over valid keys,
// lowest index among ties and the tie counts of Table "Edge cases").
// CTA = one 128-row query block of one head.  Compute thread t owns query row
// qb*128 + t%128 (TMEM lane t%128) and the column half t/128 of every 128-key
// score tile S = Q K^T.  The MMA warp computes S into two TMEM buffers
// (columns [0,128) and [128,256)), so the product of tile kb+1 runs while tile
// kb is reduced; the producer warp streams K tiles through a TMA ring.
// ---------------------------------------------------------------------------

// One 32-key chunk: chunk extrema by a max/min tree, then (warp-uniform branch,
// taken while a lane's running extremum can still move) the lanes whose chunk
// reaches their running extremum count the chunk's equal keys with a bit mask;
// its lowest set bit is the lowest index.  Masked keys (j > i) take -inf / +inf.
// MIN: also the minimum side, which only the MinMax grid spans (FWM and the softmax
// comparator are anchored at M alone).  RAW: the scale is a power of two (d = 64: 2^-3), so
// the chunk compares the unscaled dot products, whose order and equalities are those of
// the scaled scores (exact scaling: only scores below 2^-123 in magnitude, subnormal after
// scaling, could merge), and M, m are scaled once when the row is stored.
template <bool DIAG, bool MIN, bool RAW>
__device__ __forceinline__ void stats_chunk(float (&v)[32], int j0, int i, float scale, float& M, float& m,
                                            int& amax, int& amin, int& nmax, int& nmin) {
  float hi[16], lo[16];
  if constexpr (!RAW) {
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) v[jj] = __fmul_rn(v[jj], scale);
  }
#pragma unroll
  for (int jj = 0; jj < 16; ++jj) {
    float a = v[jj], b = v[jj + 16], a2 = a, b2 = b;
    if constexpr (DIAG) {
      const bool oa = j0 + jj <= i, ob = j0 + jj + 16 <= i;
      a = oa ? a : -INFINITY;
      b = ob ? b : -INFINITY;
      a2 = oa ? a2 : INFINITY;
      b2 = ob ? b2 : INFINITY;
    }
    hi[jj] = fmaxf(a, b);
    if constexpr (MIN) lo[jj] = fminf(a2, b2);
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int jj = 0; jj < w; ++jj) {
      hi[jj] = fmaxf(hi[jj], hi[jj + w]);
      if constexpr (MIN) lo[jj] = fminf(lo[jj], lo[jj + w]);
    }
  const float cmax = hi[0];
  float cmin = 0.f;
  if constexpr (MIN) cmin = lo[0];
  const bool um = cmax >= M, un = MIN && cmin <= m;
  if (__any_sync(0xffffffffu, um)) {
    uint32_t mk = 0;
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
      const bool e = (v[jj] == cmax) && (!DIAG || j0 + jj <= i);
      mk |= e ? (1u << jj) : 0u;
    }
    if (um) {
      if (cmax > M) {
        M = cmax;
        amax = j0 + __ffs(mk) - 1;
        nmax = __popc(mk);
      } else {
        nmax += __popc(mk);
      }
    }
  }
  if (MIN && __any_sync(0xffffffffu, un)) {
    uint32_t mk = 0;
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
      const bool e = (v[jj] == cmin) && (!DIAG || j0 + jj <= i);
      mk |= e ? (1u << jj) : 0u;
    }
    if (un) {
      if (cmin < m) {
        m = cmin;
        amin = j0 + __ffs(mk) - 1;
        nmin = __popc(mk);
      } else {
        nmin += __popc(mk);
      }
    }
  }
}

static dim3 launch_grid(const Params& p) { return dim3((unsigned)p.ngrid); }

template <bool MIN, bool RAW>
__global__ void __launch_bounds__(NTHR, 2) k_fwd_stats(const __grid_constant__ Maps maps, const Params p,
                                                         const __grid_constant__ Sched sch) {
  uint8_t* sm = smem_base();
  const int D = p.d, tile = D * 512, parts = p.x3 ? 2 : 1, NS = p.nstage;
  uint8_t* sQ = sm + p.sm_a;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_q = bars;
  uint64_t* bar_full = bars + 1;
  uint64_t* bar_empty = bars + 1 + NS;
  uint64_t* bar_s = bars + 1 + 2 * NS;      // [2] S_b computed
  uint64_t* bar_sfree = bars + 3 + 2 * NS;  // [2] S_b read by every compute warp
  uint64_t* bar_qfree = bars + 5 + 2 * NS;  // the item's last product complete: Q may be reloaded
  uint64_t* bar_never = bars + 6 + 2 * NS;  // nothing arrives (test hook of the bounded waits)
  uint64_t* bar_drain = bars + 7 + 2 * NS;  // the MMA warp's clean-up commit
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 8 + 2 * NS);
  float* xch = reinterpret_cast<float*>(sm + p.sm_rows);  // [6][128]
  const int tid = threadIdx.x, warp = warp_id_uniform();

  if (tid == 0) {
    mbar_init(bar_q, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar_s[b], 1);
      mbar_init(&bar_sfree[b], NCOMP / 32);
    }
    mbar_init(bar_qfree, 1);
    mbar_init(bar_never, 1);
    mbar_init(bar_drain, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_trigger();
  pdl_wait();  // everything below may read what the previous kernel wrote
  const uint32_t tmem = *tslot;
  const bool skip = expire_first_wait(p, bar_never);

  // Work items as in pass 2: (query block, head), longest first, strided over the grid.
  if (skip) {
    // (the test hook's wait ran out before anything was issued)
  } else if (warp == PRODUCER_WARP) {
    int g = 0, n = 0;
    RingPos ld;  // stage of the next K tile loaded
    bool ok = true;
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      if (n > 0 && !mbar_wait_warp(bar_qfree, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) break;
      mbar_arrive_expect_tx(bar_q, parts * tile);
      load_rows_tile(sQ, &maps.q, bar_q, D, 128, 0, qb * 128, bh);
      if (p.x3) load_rows_tile(sQ + tile, &maps.q_lo, bar_q, D, 128, 0, qb * 128, bh);
      for (int kb = 0; kb < nkb; ++kb, ++g, ld.next(NS)) {
        const int s = ld.i;
        if (g >= NS && !mbar_wait_warp(&bar_empty[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        mbar_arrive_expect_tx(&bar_full[s], parts * tile);
        load_rows_tile(dst, &maps.k, &bar_full[s], D, 128, 0, kb * 128, bh);
        if (p.x3) load_rows_tile(dst + tile, &maps.k_lo, &bar_full[s], D, 128, 0, kb * 128, bh);
      }
    }
    // clean-up: the last K tiles and Q tile issued have landed
    drain_ring(bar_full, ld, g, NS, p.wait_ns, p.status);
    if (n > 0) mbar_wait_warp(bar_q, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
  } else if (warp == MMA_WARP) {
    int g = 0, n = 0;
    RingPos cs;  // stage of the current K tile
    bool ok = true;
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, nkb = qb + 1;
      ok = mbar_wait_warp(bar_q, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      for (int kb = 0; kb < nkb && ok; ++kb, cs.next(NS)) {
        const int gk = g + kb, s = cs.i, b = gk & 1;
        // S_b was last read two tiles ago
        if (gk >= 2 && !mbar_wait_warp(&bar_sfree[b], ((gk >> 1) - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) {
          ok = false;
          break;
        }
        if (!mbar_wait_warp(&bar_full[s], cs.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint8_t* sk = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        const uint32_t dcol = tmem + b * 128;
        if (p.x3) {
          mma_smem_smem(dcol, sQ + tile, sk, 128, D, false);  // Q_lo K_hi
          mma_smem_smem(dcol, sQ, sk + tile, 128, D, true);   // Q_hi K_lo
          mma_smem_smem(dcol, sQ, sk, 128, D, true);          // Q_hi K_hi
        } else {
          mma_smem_smem(dcol, sQ, sk, 128, D, false);
        }
        mma_commit(&bar_s[b]);
        mma_commit(&bar_empty[s]);
        if (kb + 1 == nkb) mma_commit(bar_qfree);
      }
      g += nkb;
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else {
    const int row = tid & 127, cg = tid >> 7;
    int g = 0, n = 0;
    bool failed = false;
    for (int item = sched_item(sch, n); item < p.nitems && !failed; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      const int i = qb * 128 + row;
      float M = -FLT_MAX, m = FLT_MAX;
      int amax = 0, amin = 0, nmax = 0, nmin = 0;
      for (int kb = 0; kb < nkb; ++kb) {
        const int gk = g + kb, b = gk & 1;
        if (!mbar_wait(&bar_s[b], (gk >> 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          failed = true;
          break;
        }
        tc_fence_after();
        const bool diag = kb == qb;
#pragma unroll 1
        for (int cc = 0; cc < 2; ++cc) {
          const int c = cg * 2 + cc;
          float v[32];
          tmem_ld32(lane_addr(tmem, b * 128 + c * 32), v);
          tmem_ld_wait();
          const int j0 = kb * 128 + c * 32;
          if (diag)
            stats_chunk<true, MIN, RAW>(v, j0, i, p.scale, M, m, amax, amin, nmax, nmin);
          else
            stats_chunk<false, MIN, RAW>(v, j0, i, p.scale, M, m, amax, amin, nmax, nmin);
        }
        tc_fence_before();
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_sfree[b]);
      }
      g += nkb;
      failed = group_any(BAR_COMPUTE, NCOMP, failed);
      if (failed) break;
      // combine the two column halves of each row
      if (cg == 1) {
        xch[0 * 128 + row] = M;
        xch[1 * 128 + row] = m;
        xch[2 * 128 + row] = __int_as_float(amax);
        xch[3 * 128 + row] = __int_as_float(amin);
        xch[4 * 128 + row] = __int_as_float(nmax);
        xch[5 * 128 + row] = __int_as_float(nmin);
      }
      group_sync(BAR_COMPUTE, NCOMP);
      if (cg == 0 && i < p.T) {
        const float M1 = xch[row], m1 = xch[128 + row];
        const int amax1 = __float_as_int(xch[256 + row]), amin1 = __float_as_int(xch[384 + row]);
        const int nmax1 = __float_as_int(xch[512 + row]), nmin1 = __float_as_int(xch[640 + row]);
        if (M1 > M || (M1 == M && nmax1 > 0 && amax1 < amax)) amax = (M1 > M || nmax == 0) ? amax1 : min(amax, amax1);
        if (M1 > M) {
          nmax = nmax1;
          M = M1;
        } else if (M1 == M) {
          nmax += nmax1;
        }
        if (MIN) {
          if (m1 < m || (m1 == m && nmin1 > 0 && amin1 < amin)) amin = (m1 < m || nmin == 0) ? amin1 : min(amin, amin1);
          if (m1 < m) {
            nmin = nmin1;
            m = m1;
          } else if (m1 == m) {
            nmin += nmin1;
          }
        } else {  // not computed: +inf, index -1, count 0
          m = INFINITY;
          amin = -1;
          nmin = 0;
        }
        if constexpr (RAW) {
          M = __fmul_rn(M, p.scale);
          m = __fmul_rn(m, p.scale);  // (+inf stays +inf when the minimum is not computed)
        }
        const size_t rw = (size_t)bh * p.T + i;
        p.row_max[rw] = M;
        p.row_min[rw] = m;
        p.arg_max[rw] = amax;
        p.arg_min[rw] = amin;
        p.n_max[rw] = nmax;
        p.n_min[rw] = nmin;
      }
      group_sync(BAR_COMPUTE, NCOMP);  // the exchange words are read before the next item writes them
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

cudaError_t launch_fwd_stats(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch) {
  // d = 64: scale 1/8, a power of two (RAW)
  auto kern = p.calib == CAL_MINMAX ? (p.d == 64 ? k_fwd_stats<true, true> : k_fwd_stats<true, false>)
                                    : (p.d == 64 ? k_fwd_stats<false, true> : k_fwd_stats<false, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, launch_grid(p), dim3(NTHR), smem_bytes, s, maps, p, sch);
}

// ---------------------------------------------------------------------------
// Pass 2 element work on one 32-key chunk of one row (App. A): the grid
// position u = acc * k1 + c0, the decisions (r, t, Nearest, FWM tail) and the
// weights w^L = e_r + t (e_{r+1} - e_r), w^N = (t >= 1/2 ? e_{r+1} : e_r), by a
// lookup of the pair (e_r, e_{r+1}) in the row's table and one FMA in place of
// the exponential.  MODE 0: a = forward weight; 1: also w^L for O_lerp; 2: a = w^L.
// ---------------------------------------------------------------------------
template <int CAL, int REC, int MODE, bool DIAG>
__device__ __forceinline__ void fwd_chunk(const float (&v)[32], float (&a1)[32], float (&a2)[32], int j0, int i,
                                          const RowGrid& g, float Kf, uint32_t tab, float sk1, float sc0,
                                          float& wm_sum, float& wl_sum) {
  float wm_acc = 0.f, wl_acc = 0.f;
#pragma unroll
  for (int jj = 0; jj < 32; ++jj) {
    float wm, wl = 0.f;
    if constexpr (CAL == CAL_SOFTMAX) {
      wm = ex2_approx(__fmaf_rn(v[jj], sk1, sc0));  // e^{s - M} (App. A, Softmax)
    } else if constexpr (CAL == CAL_EXP8) {
      wm = e4m3_rn(ex2_approx(__fmaf_rn(v[jj], sk1, sc0)));  // E4M3(e^{s - M})
    } else if constexpr (CAL == CAL_EXPB) {
      float zb;
      wm = bf16_exp_weight(__fadd_rn(__fmul_rn(v[jj], g.k1), g.c0), zb);  // bf16(e^{bf16(s - M)})
    } else if constexpr (CAL == CAL_FWM) {
      // v = 2u = acc * 2k1 + 2c0 (sk1, sc0) clamped to [-1, 2K]; floor(v) = q = 2r + [t >= 1/2]
      // indexes the half-bin table {alpha, beta, w^N, 0} by the float bits of its round-down
      // (entry q at tab + 16 bits), with the tail (u < 0) on the two zero entries below q = 0:
      // w^L = alpha + v beta, w^N = the Nearest endpoint.  Same decisions as decode_u.
      constexpr bool need_wn = REC == REC_NEAREST && MODE != 2;
      constexpr bool need_wl = REC == REC_LERP || MODE != 0;
      const float vc = fminf(fmaxf(__fmaf_rn(v[jj], sk1, sc0), -1.0f), 2.0f * Kf);
      const uint32_t a = tab + (__float_as_uint(__fadd_rd(vc, kMagic)) << 4);
      if constexpr (need_wn && need_wl) {
        const float2 e = lds_f2(a);
        wl = __fmaf_rn(vc, e.y, e.x);
        wm = lds_f32(a + 8u);
      } else if constexpr (need_wn) {
        wm = lds_f32(a + 8u);
      } else {
        const float2 e = lds_f2(a);
        wl = __fmaf_rn(vc, e.y, e.x);
        wm = wl;
      }
    } else {
      const float u = __fmaf_rn(v[jj], g.k1, g.c0);
      float t, rf;
      uint32_t rb;
      decode_u(u, Kf, t, rb, rf);
      // MinMax: this row's table, rows 1024 bytes apart; FWMR: one shared table, entries 8 bytes apart
      float2 e = lds_f2(fwm_like(CAL) ? tab + rb * 8u : tab + rb * 1024u);
      if constexpr (CAL == CAL_FWMR) {
        // below the window: the continued grid (negative r)
        const BelowPair bp = resolved_below(u, g.hl, g.b0l);
        const bool below = u < 0.0f;
        t = below ? bp.t : t;
        e = below ? make_float2(bp.e0, bp.e1) : e;
      }
      wl = __fmaf_rn(t, __fsub_rn(e.y, e.x), e.x);
      float wn = (t >= 0.5f) ? e.y : e.x;
      if constexpr (CAL == CAL_MINMAX) {
        wl = g.nogrid ? 1.f : wl;
        wn = g.nogrid ? 1.f : wn;
      }
      wm = (REC == REC_NEAREST) ? wn : wl;
    }
    if constexpr (DIAG) {
      const bool ok = (j0 + jj) <= i;
      wm = ok ? wm : 0.f;
      wl = ok ? wl : 0.f;
    }
    wm_acc += wm;
    if constexpr (MODE != 0) wl_acc += wl;
    a1[jj] = (MODE == 2) ? wl : wm;
    if constexpr (MODE == 1) a2[jj] = wl;
  }
  wm_sum += wm_acc;
  wl_sum += wl_acc;
}

// Decision codes of one chunk for kint_attn_debug_bins (not on the timed path, but
// inlined into the main loop: the calibration is a template parameter so that each
// instantiation carries only its own branch).
template <int CAL>
__device__ void fwd_debug_codes(const Params& p, const float (&v)[32], int j0, int i, int bh, const RowGrid& g,
                                float sk1, float sc0) {
  if (i >= p.T) return;
  for (int jj = 0; jj < 32; ++jj) {
    const int j = j0 + jj;
    if (j >= p.T) break;
    uint8_t cb = 255, ci = 255;
    if (j <= i) {
      if constexpr (CAL == CAL_EXP8) {
        cb = ci = (uint8_t)e4m3_code(e4m3_rn(ex2_approx(__fmaf_rn(v[jj], sk1, sc0))));
      } else if constexpr (CAL == CAL_EXPB) {
        float zb;
        const float w = bf16_exp_weight(__fadd_rn(__fmul_rn(v[jj], g.k1), g.c0), zb);
        cb = (uint8_t)bf16_low_byte(zb);
        ci = (uint8_t)bf16_low_byte(w);
      } else if (CAL == CAL_SOFTMAX || g.nogrid) {
        cb = ci = 253;
      } else {
        const float u = __fmaf_rn(v[jj], g.k1, g.c0);
        float t, rf;
        uint32_t rb;
        decode_u(u, (float)p.Kint, t, rb, rf);
        if (CAL == CAL_FWM && u < 0.0f) {
          cb = ci = 254;
        } else if constexpr (CAL == CAL_FWMR) {
          // resolved: indices run below zero, stored as index + 128 saturated to [0, 252]
          const int r = u < 0.0f ? (int)floorf(u) : (int)rf;
          const float tt = u < 0.0f ? __fsub_rn(u, floorf(u)) : t;
          const int l = r + (tt >= 0.5f ? 1 : 0);
          ci = (uint8_t)min(max(r + 128, 0), 252);
          cb = (uint8_t)min(max(l + 128, 0), 252);
        } else {
          const int r = (int)rf;
          ci = (uint8_t)r;
          cb = (uint8_t)(r + (t >= 0.5f ? 1 : 0));
        }
      }
    }
    const size_t idx = ((size_t)bh * p.T + i) * p.T + j;
    if (p.bins) p.bins[idx] = cb;
    if (p.ivals) p.ivals[idx] = ci;
  }
}

// ---------------------------------------------------------------------------
// Pass 2: reconstruction, normalization and P V (App. A).
// Work items are (128-row query block, head) pairs, longest blocks first; a CTA
// takes the items sched_item(sch, 0), sched_item(sch, 1), ... (one item per CTA when the
// grid covers them all).  Tile counters run on across items, so the next item's Q
// and first K/V tiles load while the current one finishes.
// TMEM: score buffers S_b at [128 b, 128 b + 128), b < nbuf (the weights
// overwrite their scores as MMA operand A); A2 (w^L for O_lerp, or the tf32 lo
// part of A under 3xTF32) at [128 nbuf, +128); O at cO, O_lerp at cO + d.
// smem: Q (hi[, lo]) at sm_a; stages {K tile, V^T tile} (hi[, lo] each) fed by
// the producer warp; per-row pair tables (e_r, e_{r+1}) [K][128] at sm_table; the
// output staging tile(s) at sm_ostage (also the W exchange words).
// ---------------------------------------------------------------------------
__device__ __forceinline__ const uint8_t* stgl_of(const uint8_t* ostg, int d) { return ostg + 128 * d * 4; }

// MMA warp of k_fwd_main: wait for the K/V stage st (ring position), S_b = Q K^T into
// score buffer b, commit to bar_s[b].
__device__ __forceinline__ bool main_issue_s(const Params& p, RingPos stg, int b, uint64_t* bar_full,
                                             uint64_t* bar_s, const uint8_t* st0, const uint8_t* sQ, uint32_t tmem,
                                             int qtile) {
  const int s = stg.i, D = p.d;
  if (!mbar_wait_warp(&bar_full[s], stg.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) return false;
  tc_fence_after();
  const uint8_t* sk = st0 + s * p.sm_stage_bytes;
  const uint32_t dcol = tmem + b * 128;
  if (p.x3) {
    mma_smem_smem(dcol, sQ + qtile, sk, 128, D, false);  // Q_lo K_hi
    mma_smem_smem(dcol, sQ, sk + qtile, 128, D, true);   // Q_hi K_lo
    mma_smem_smem(dcol, sQ, sk, 128, D, true);           // Q_hi K_hi
  } else {
    mma_smem_smem(dcol, sQ, sk, 128, D, false);
  }
  mma_commit(&bar_s[b]);
  return true;
}

// MODE 1 (Nearest weights for O, LERP weights for O_lerp) in TF32 issues its two P V
// products from two warps on different SM sub-partitions: P V with the S products from
// MMA_WARP, P^L V from MMA2_WARP, which frees the single A2 buffer (w^L) for the next
// tile sooner than one warp issuing 32 MMAs back to back would.
template <int MODE>
constexpr int main_threads() { return MODE == 1 ? NTHR_DQ : NTHR; }

template <int CAL, int REC, int MODE>
__global__ void __launch_bounds__(main_threads<MODE>(), 1) k_fwd_main(const __grid_constant__ Maps maps, const Params p,
                                                                   const __grid_constant__ Sched sch) {
  uint8_t* sm = smem_base();
  const int D = p.d, Kq = p.Kint, parts = p.x3 ? 2 : 1, NS = p.nstage, nbuf = p.nbuf;
  const int qtile = D * 512, vtile = D * 512;
  uint8_t* sQ = sm + p.sm_a;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_q = bars;                     // Q of the item landed
  uint64_t* bar_full = bars + 1;              // [NS]
  uint64_t* bar_empty = bars + 1 + NS;        // [NS]
  uint64_t* bar_s = bars + 1 + 2 * NS;        // [2] S_b computed
  uint64_t* bar_pready = bars + 3 + 2 * NS;   // [2] weights of buffer b stored by every compute warp
  uint64_t* bar_pv = bars + 5 + 2 * NS;       // P V of a tile complete (A2 free again)
  uint64_t* bar_done = bars + 6 + 2 * NS;     // every product of the item complete
  uint64_t* bar_qfree = bars + 7 + 2 * NS;    // the item's last S product complete: Q may be reloaded
  uint64_t* bar_ofree = bars + 8 + 2 * NS;    // O / O_lerp read out of TMEM by every compute warp
  uint64_t* bar_drain = bars + 9 + 2 * NS;    // the MMA warp's clean-up commit
  uint64_t* bar_drain2 = bars + 10 + 2 * NS;  // MMA2_WARP's clean-up commit
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 11 + 2 * NS);
  uint8_t* ostg = sm + p.sm_ostage;
  float* xch = reinterpret_cast<float*>(ostg);  // [4][128], written before the staging tiles each item
  const int tid = threadIdx.x, warp = warp_id_uniform();
  const bool useA2 = (MODE == 1) || p.x3;
  const bool split = MODE == 1 && !p.x3;  // P^L V from MMA2_WARP
  const int cA2 = 128 * nbuf, cO = cA2 + (useA2 ? 128 : 0), cOL = cO + D;

  if (tid == 0) {
    mbar_init(bar_q, 1);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_empty[s], split ? 2 : 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar_s[b], 1);
      mbar_init(&bar_pready[b], NCOMP / 32);
    }
    mbar_init(bar_pv, 1);
    mbar_init(bar_done, split ? 2 : 1);
    mbar_init(bar_qfree, 1);
    mbar_init(bar_ofree, NCOMP / 32);
    mbar_init(bar_drain, 1);
    mbar_init(bar_drain2, 1);
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
    int g = 0, n = 0;
    RingPos ld;  // stage of the next K/V tile loaded
    bool ok = true;
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      // Q of the previous item is an operand until its last S product completes
      if (n > 0 && !mbar_wait_warp(bar_qfree, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) break;
      mbar_arrive_expect_tx(bar_q, parts * qtile);
      load_rows_tile(sQ, &maps.q, bar_q, D, 128, 0, qb * 128, bh);
      if (p.x3) load_rows_tile(sQ + qtile, &maps.q_lo, bar_q, D, 128, 0, qb * 128, bh);
      for (int kb = 0; kb < nkb; ++kb, ++g, ld.next(NS)) {
        const int s = ld.i;
        if (g >= NS && !mbar_wait_warp(&bar_empty[s], ld.ph ^ 1u, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA)) {
          ok = false;
          break;
        }
        uint8_t* dst = sm + p.sm_stage0 + s * p.sm_stage_bytes;
        mbar_arrive_expect_tx(&bar_full[s], parts * (qtile + vtile));
        load_rows_tile(dst, &maps.k, &bar_full[s], D, 128, 0, kb * 128, bh);
        load_rows_tile(dst + parts * qtile, &maps.vt, &bar_full[s], 128, D, kb * 128, 0, bh);
        if (p.x3) {
          load_rows_tile(dst + qtile, &maps.k_lo, &bar_full[s], D, 128, 0, kb * 128, bh);
          load_rows_tile(dst + parts * qtile + vtile, &maps.vt_lo, &bar_full[s], 128, D, kb * 128, 0, bh);
        }
      }
    }
    // clean-up: the last K/V tiles and Q tile issued have landed
    drain_ring(bar_full, ld, g, NS, p.wait_ns, p.status);
    if (n > 0) mbar_wait_warp(bar_q, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
  } else if (warp == MMA_WARP) {
    const uint8_t* st0 = sm + p.sm_stage0;
    int g = 0, n = 0;
    RingPos is, ib, cs, cb;  // stage / buffer of the next S product and of the tile being finished
    bool ok = true;
    for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, nkb = qb + 1;
      ok = mbar_wait_warp(bar_q, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA) &&
           main_issue_s(p, is, ib.i, bar_full, bar_s, st0, sQ, tmem, qtile);
      is.next(NS);
      ib.next(nbuf);
      if (ok && nkb == 1) mma_commit(bar_qfree);
      for (int kb = 0; kb < nkb && ok; ++kb, cs.next(NS), cb.next(nbuf)) {
        const int b = cb.i, s = cs.i;
        // S(kb+1) goes to the other buffer, whose last reader P V(kb-1) precedes it in issue order
        if (nbuf == 2 && kb + 1 < nkb) {
          if (!main_issue_s(p, is, ib.i, bar_full, bar_s, st0, sQ, tmem, qtile)) break;
          is.next(NS);
          ib.next(nbuf);
          if (kb + 2 == nkb) mma_commit(bar_qfree);
        }
        if (!mbar_wait_warp(&bar_pready[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) break;
        // the item's first P V overwrites O: the previous item's epilogue must have read it
        if (kb == 0 && n > 0 && !mbar_wait_warp(bar_ofree, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC))
          break;
        tc_fence_after();
        const uint8_t* vt = st0 + s * p.sm_stage_bytes + parts * qtile;
        const bool acc = kb > 0;
        const uint32_t a = tmem + b * 128;
        if (p.x3) {
          mma_tmem_smem(tmem + cO, tmem + cA2, vt, D, 128, acc);  // A_lo V_hi (frees A2 first)
          mma_tmem_smem(tmem + cO, a, vt + vtile, D, 128, true);   // A_hi V_lo
          mma_tmem_smem(tmem + cO, a, vt, D, 128, true);           // A_hi V_hi
        } else {
          if (MODE == 1 && !split) mma_tmem_smem(tmem + cOL, tmem + cA2, vt, D, 128, acc);  // frees A2 first
          mma_tmem_smem(tmem + cO, a, vt, D, 128, acc);
        }
        if (!split) mma_commit(bar_pv);
        mma_commit(&bar_empty[s]);
        // one buffer: S(kb+1) overwrites the weights P V(kb) reads, in issue order after it
        if (nbuf == 1 && kb + 1 < nkb) {
          if (!main_issue_s(p, is, ib.i, bar_full, bar_s, st0, sQ, tmem, qtile)) break;
          is.next(NS);
          ib.next(nbuf);
          if (kb + 2 == nkb) mma_commit(bar_qfree);
        }
      }
      g += nkb;
      mma_commit(bar_done);
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else if (warp == MMA2_WARP) {
    // P^L V of every tile (split only): O_lerp += w^L V once the tile's weights are stored
    if (split) {
      int n = 0;
      RingPos cs, cb;
      bool ok = true;
      for (int item = sched_item(sch, n); item < p.nitems && ok; item = sched_item(sch, ++n)) {
        const int qb = p.nqb - 1 - item / p.BH, nkb = qb + 1;
        for (int kb = 0; kb < nkb; ++kb, cs.next(NS), cb.next(nbuf)) {
          // the tile's K / V^T stage has landed: its weights, which need S, are stored
          if (!mbar_wait_warp(&bar_pready[cb.i], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC) ||
              (kb == 0 && n > 0 && !mbar_wait_warp(bar_ofree, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint8_t* vt = sm + p.sm_stage0 + cs.i * p.sm_stage_bytes + qtile;
          mma_tmem_smem(tmem + cOL, tmem + cA2, vt, D, 128, kb > 0);
          mma_commit(bar_pv);
          mma_commit(&bar_empty[cs.i]);
        }
        if (!ok) break;
        mma_commit(bar_done);
      }
      drain_mma(bar_drain2, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
    }
  } else {
    const int row = tid & 127, cg = tid >> 7;
    const float Kf = (float)Kq;
    int g = 0, n = 0;
    RingPos cb;  // score buffer of the current tile
    bool failed = false;
    // the row extrema of an item, loaded one item ahead (under the previous item's epilogue)
    auto load_extrema = [&](int n, float& M, float& m) {
      const int item = sched_item(sch, n);
      const int i = (p.nqb - 1 - item / p.BH) * 128 + row;
      const size_t rw = (size_t)(item % p.BH) * p.T + i;
      M = i < p.T ? p.row_max[rw] : 0.0f;
      m = i < p.T ? p.row_min[rw] : 0.0f;
    };
    float nM = 0.f, nm = 0.f;
    if (sched_item(sch, 0) < p.nitems) load_extrema(0, nM, nm);
    for (int item = sched_item(sch, n); item < p.nitems && !failed; item = sched_item(sch, ++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      const int i = qb * 128 + row;
      const bool row_ok = i < p.T;
      const size_t rw = (size_t)bh * p.T + (row_ok ? i : 0);
      const float M = nM, m = nm;
      const RowGrid gr = row_grid(p, M, m);
      // softmax: base-2 exponent coefficients; FWM: the half-bin position v = 2u = acc * 2k1 + 2c0
      // (an exact doubling of u)
      const float sk1 = CAL == CAL_FWM ? 2.0f * gr.k1 : p.scale * 1.4426950408889634f;
      const float sc0 = CAL == CAL_FWM ? 2.0f * gr.c0 : -M * 1.4426950408889634f;
      // Pair tables, entry r = (e_r, e_{r+1}), r = 0..K-1, addressed by the float bits
      // rb = 0x4B000000 + r of the floored position: MinMax keeps one table per row
      // ([K][128], 1024 bytes per r: rb * 1024 wraps to r * 1024); FWMR's grid is the
      // same for every row, so one [K] table serves all (rb * 8 = 0x58000000 + 8 r), and
      // FWM's one half-bin table of line coefficients.
      uint32_t tab;
      if constexpr (CAL == CAL_FWM) {
        // the half-bin table, entry q in [-2, 2K] at sm_table + 16 (q + 2); the float bits
        // 0x4B000000 + q of the rounded-down position times 16 wrap to 0xB0000000 + 16 q
        tab = smem_u32(sm + p.sm_table) + 16u * kHalfTail - 0xB0000000u;
        if (n == 0 && tid < 2 * Kq + 1 + kHalfTail)
          *reinterpret_cast<float4*>(sm + p.sm_table + tid * 16) = fwm_line_entry(p, tid - kHalfTail);
      } else if constexpr (CAL == CAL_FWMR) {
        // entries r = 0 .. K-1 after kFwdTail zero entries
        tab = smem_u32(sm + p.sm_table) + 8u * kFwdTail - 0x58000000u;
        if (n == 0 && tid < Kq)
          *reinterpret_cast<float2*>(sm + p.sm_table + 8 * kFwdTail + tid * 8) =
              make_float2(p.fwm_e[tid], p.fwm_e[tid + 1]);
        if (n == 0 && tid < kFwdTail) *reinterpret_cast<float2*>(sm + p.sm_table + tid * 8) = make_float2(0.f, 0.f);
      } else {
        tab = smem_u32(sm + p.sm_table) + (uint32_t)row * 8u;
        if constexpr (CAL == CAL_MINMAX) {
          for (int r = cg; r < Kq; r += NCG) {
            const float2 e = make_float2(grid_value(p, gr, r), grid_value(p, gr, r + 1));
            *reinterpret_cast<float2*>(sm + p.sm_table + (size_t)r * 1024 + row * 8) = e;
          }
        }
      }
      group_sync(BAR_COMPUTE, NCOMP);

      float Wm = 0.f, Wl = 0.f;
      for (int kb = 0; kb < nkb && !failed; ++kb, cb.next(nbuf)) {
        const int gk = g + kb, b = cb.i;
        if (!mbar_wait(&bar_s[b], cb.ph, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          failed = true;
          break;
        }
        tc_fence_after();
        const bool diag = kb == qb;
#pragma unroll 1
        for (int cc = 0; cc < 2; ++cc) {
          const int c = cg * 2 + cc;
          float v[32], a1[32], a2[32];
          tmem_ld32(lane_addr(tmem, b * 128 + c * 32), v);
          tmem_ld_wait();
          const int j0 = kb * 128 + c * 32;
          if (p.debug) fwd_debug_codes<CAL>(p, v, j0, i, bh, gr, sk1, sc0);
          if (diag)
            fwd_chunk<CAL, REC, MODE, true>(v, a1, a2, j0, i, gr, Kf, tab, sk1, sc0, Wm, Wl);
          else
            fwd_chunk<CAL, REC, MODE, false>(v, a1, a2, j0, i, gr, Kf, tab, sk1, sc0, Wm, Wl);
          if (p.x3) {
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float h = tf32_rna(a1[q]);
              a2[q] = __fsub_rn(a1[q], h);
              a1[q] = h;
            }
          }
          // A2 is still an operand of the previous tile's products until they complete
          if (cc == 0 && useA2 && gk > 0 &&
              !mbar_wait(bar_pv, (gk - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
            failed = true;
            break;
          }
          tmem_st32(lane_addr(tmem, b * 128 + c * 32), a1);
          if (useA2) tmem_st32(lane_addr(tmem, cA2 + c * 32), a2);
        }
        if (failed) break;
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_pready[b]);
      }
      g += nkb;
      if (sched_item(sch, n + 1) < p.nitems) load_extrema(n + 1, nM, nm);
      if (!failed) failed = !mbar_wait(bar_done, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA);
      failed = group_any(BAR_COMPUTE, NCOMP, failed);
      if (failed) break;
      tc_fence_after();
      // the previous item's stores have left the staging area before it is written again
      if (warp < 2) tma_store_wait_read();
      group_sync(BAR_COMPUTE, NCOMP);
      xch[cg * 128 + row] = Wm;
      xch[(2 + cg) * 128 + row] = Wl;
      group_sync(BAR_COMPUTE, NCOMP);
      const float Wmt = xch[row] + xch[128 + row];
      const float Wlt = xch[256 + row] + xch[384 + row];
      group_sync(BAR_COMPUTE, NCOMP);  // the exchange words are read before the tiles overwrite them
      if (!p.debug) {
        // O = (sum_j w_j V_j) / W (and O_lerp): each column group scales half of the d
        // columns into a swizzled tile, one TMA store per tile
        const float Wout = (MODE == 2) ? Wlt : Wmt;
        const float inv = row_ok ? 1.0f / Wout : 0.0f;
        const float invl = row_ok ? 1.0f / Wlt : 0.0f;
        uint8_t* stgl = ostg + 128 * D * 4;
        for (int c = cg * (D / 2); c < (cg + 1) * (D / 2); c += 32) {
          float v[32];
          tmem_ld32(lane_addr(tmem, cO + c), v);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 32; ++q) v[q] *= inv;
          row_to_staged(ostg, row, c / 32, v);
          if constexpr (MODE == 1) {
            tmem_ld32(lane_addr(tmem, cOL + c), v);
            tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < 32; ++q) v[q] *= invl;
            row_to_staged(stgl, row, c / 32, v);
          }
        }
      }
      // the accumulators go back to the MMA warp for the next item
      tc_fence_before();
      __syncwarp();
      if ((tid & 31) == 0) mbar_arrive(bar_ofree);
      if (!p.debug) {
        fence_async_smem();
        group_sync(BAR_COMPUTE, NCOMP);
        if (warp == 0)
          store_rows_tile_boxed(ostg, (MODE == 2) ? &maps.out_lerp : &maps.out, D, 64, qb * 128, bh, false);
        if (MODE == 1 && warp == 1) store_rows_tile_boxed(stgl_of(ostg, D), &maps.out_lerp, D, 64, qb * 128, bh, false);
        if (row_ok && cg == 0) {
          if (MODE != 2) p.W[rw] = Wmt;
          if (MODE != 0 && p.W_lerp) p.W_lerp[rw] = Wlt;
        }
      }
    }
    if (warp < 2) tma_store_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

template <int CAL, int REC, int MODE>
static cudaError_t launch_main_t(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch) {
  auto kern = k_fwd_main<CAL, REC, MODE>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, launch_grid(p), dim3(main_threads<MODE>()), smem_bytes, s, maps, p, sch);
}

cudaError_t launch_fwd_main(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch) {
  const int mode = p.pv_sel;
  if (p.calib == CAL_SOFTMAX) return launch_main_t<CAL_SOFTMAX, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
  if (p.calib == CAL_EXP8) return launch_main_t<CAL_EXP8, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
  if (p.calib == CAL_EXPB) return launch_main_t<CAL_EXPB, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
  if (p.calib == CAL_MINMAX) {
    if (p.recon == REC_LERP) return launch_main_t<CAL_MINMAX, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
    if (mode == PV_MAIN) return launch_main_t<CAL_MINMAX, REC_NEAREST, 0>(maps, p, smem_bytes, s, sch);
    if (mode == PV_MAIN_LERP) return launch_main_t<CAL_MINMAX, REC_NEAREST, 1>(maps, p, smem_bytes, s, sch);
    return launch_main_t<CAL_MINMAX, REC_NEAREST, 2>(maps, p, smem_bytes, s, sch);
  }
  if (p.calib == CAL_FWMR) {
    if (p.recon == REC_LERP) return launch_main_t<CAL_FWMR, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
    if (mode == PV_MAIN) return launch_main_t<CAL_FWMR, REC_NEAREST, 0>(maps, p, smem_bytes, s, sch);
    if (mode == PV_MAIN_LERP) return launch_main_t<CAL_FWMR, REC_NEAREST, 1>(maps, p, smem_bytes, s, sch);
    return launch_main_t<CAL_FWMR, REC_NEAREST, 2>(maps, p, smem_bytes, s, sch);
  }
  if (p.recon == REC_LERP) return launch_main_t<CAL_FWM, REC_LERP, 0>(maps, p, smem_bytes, s, sch);
  if (mode == PV_MAIN) return launch_main_t<CAL_FWM, REC_NEAREST, 0>(maps, p, smem_bytes, s, sch);
  if (mode == PV_MAIN_LERP) return launch_main_t<CAL_FWM, REC_NEAREST, 1>(maps, p, smem_bytes, s, sch);
  return launch_main_t<CAL_FWM, REC_NEAREST, 2>(maps, p, smem_bytes, s, sch);
}

}  // namespace kint
