// Geometry probe of K-interval attention on sm_103a (App. "Geometry probe"): per
// causal row, from the operator's own fp32 scores,
//   span M - m; native width h; softmax entropy H(P^E) = ln Z - sum_j e^{z_j} z_j / Z;
//   share of keys with z < -6; top-bucket mass (softmax mass of the keys in the
//   operator's top level, Nearest l = K, or top interval, LERP r = K - 1); effective
//   buckets exp H(q), q_b the softmax mass of bucket b (the operator's levels, FWM's
//   tail keys as one more bucket, a degenerate MinMax row as one bucket); and the
//   total variation 1/2 sum_j |P_j - P^E_j| between the operator's forward P and
//   softmax P^E.
// The kernel has pass 1's structure (Q tile resident, K tiles through a TMA ring,
// S = Q K^T on tcgen05 into double-buffered TMEM) but runs over each item's key tiles
// twice: the first sweep forms Z = sum e^z, the operator's own W and the bucket
// masses, the second the total variation, which needs both normalizers.
#include <cfloat>
#include "kint_dev.cuh"
#include "kint_launch.h"

namespace kint {

// Per-row accumulators of one column group.
struct ProbeAcc {
  float Z = 0.f, Zz = 0.f, W = 0.f, below = 0.f, top = 0.f, mn = FLT_MAX, tv = 0.f;
};

// One 32-key chunk of row i.  Sweep 0 accumulates everything but the total variation;
// sweep 1 the total variation, with the row's Z and W.
template <int CAL, int REC, bool DIAG>
__device__ __forceinline__ void probe_chunk(const float (&v)[32], int j0, int i, float scale, float M,
                                            const RowGrid& g, int K, int sweep, float invZ, float invW,
                                            float* hist, ProbeAcc& a) {
#pragma unroll 4
  for (int jj = 0; jj < 32; ++jj) {
    if (DIAG && j0 + jj > i) continue;
    const float s = __fmul_rn(v[jj], scale), z = __fsub_rn(s, M);
    const float e = expf(z);
    // the operator's decisions and forward weight (Sec. 3, App. A)
    const float u = __fmaf_rn(v[jj], g.k1, g.c0);
    float t, rf;
    uint32_t rb;
    decode_u(u, (float)K, t, rb, rf);
    const int r = (int)rf, l = r + (t >= 0.5f ? 1 : 0);
    const bool tail = CAL == CAL_FWM && u < 0.0f;
    float w;
    if (g.nogrid) {
      w = 1.0f;
    } else if (tail) {
      w = 0.0f;
    } else if (REC == REC_NEAREST) {
      w = expf(__fmaf_rn((float)l, g.h, g.b0));
    } else {
      const float e0 = expf(__fmaf_rn((float)r, g.h, g.b0)), e1 = expf(__fmaf_rn((float)(r + 1), g.h, g.b0));
      w = __fmaf_rn(t, __fsub_rn(e1, e0), e0);
    }
    if (sweep == 0) {
      a.Z += e;
      a.Zz = __fmaf_rn(e, z, a.Zz);
      a.W += w;
      a.below += z < -6.0f ? 1.0f : 0.0f;
      a.mn = fminf(a.mn, s);
      const int b = g.nogrid ? 0 : (tail ? K + 1 : (REC == REC_NEAREST ? l : r));
      const bool top = g.nogrid || (!tail && (REC == REC_NEAREST ? l == K : r == K - 1));
      hist[b] += e;
      a.top += top ? e : 0.0f;
    } else {
      a.tv += fabsf(__fmaf_rn(w, invW, -e * invZ));
    }
  }
}

template <int CAL, int REC>
__global__ void __launch_bounds__(NTHR, 1) k_fwd_probe(const __grid_constant__ Maps maps, const Params p) {
  uint8_t* sm = smem_base();
  const int D = p.d, tile = D * 512, parts = p.x3 ? 2 : 1, NS = p.nstage, Kq = p.Kint, NB = Kq + 2;
  uint8_t* sQ = sm + p.sm_a;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.sm_bars);
  uint64_t* bar_q = bars;
  uint64_t* bar_full = bars + 1;
  uint64_t* bar_empty = bars + 1 + NS;
  uint64_t* bar_s = bars + 1 + 2 * NS;      // [2] S_b computed
  uint64_t* bar_sfree = bars + 3 + 2 * NS;  // [2] S_b read by every compute warp
  uint64_t* bar_qfree = bars + 5 + 2 * NS;  // the item's last product complete: Q may be reloaded
  uint64_t* bar_drain = bars + 6 + 2 * NS;  // the MMA warp's clean-up commit
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 7 + 2 * NS);
  float* xch = reinterpret_cast<float*>(sm + p.sm_rows);  // [8][128]
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
  pdl_wait();
  const uint32_t tmem = *tslot;

  if (warp == PRODUCER_WARP) {
    int g = 0, n = 0;
    RingPos ld;
    bool ok = true;
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      if (n > 0 && !mbar_wait_warp(bar_qfree, (n - 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC)) break;
      mbar_arrive_expect_tx(bar_q, parts * tile);
      load_rows_tile(sQ, &maps.q, bar_q, D, 128, 0, qb * 128, bh);
      if (p.x3) load_rows_tile(sQ + tile, &maps.q_lo, bar_q, D, 128, 0, qb * 128, bh);
      for (int kt = 0; kt < 2 * nkb; ++kt, ++g, ld.next(NS)) {  // two sweeps over the key blocks
        const int s = ld.i, kb = kt < nkb ? kt : kt - nkb;
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
    RingPos cs;
    bool ok = true;
    for (int item = snake_item(n); item < p.nitems && ok; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH, nt = 2 * (qb + 1);
      ok = mbar_wait_warp(bar_q, n & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_TMA);
      for (int kt = 0; kt < nt && ok; ++kt, cs.next(NS)) {
        const int gk = g + kt, s = cs.i, b = gk & 1;
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
        if (kt + 1 == nt) mma_commit(bar_qfree);
      }
      g += nt;
    }
    drain_mma(bar_drain, p.wait_ns, p.status);  // clean-up: no product still writes TMEM
  } else if (warp < NCOMP / 32) {
    const int row = tid & 127, cg = tid >> 7;
    float* hist = reinterpret_cast<float*>(sm + p.sm_table) + (size_t)(cg * 128 + row) * NB;
    int g = 0, n = 0;
    bool failed = false;
    for (int item = snake_item(n); item < p.nitems && !failed; item = snake_item(++n)) {
      const int qb = p.nqb - 1 - item / p.BH, bh = item % p.BH, nkb = qb + 1;
      const int i = qb * 128 + row;
      const bool row_ok = i < p.T;
      const size_t rw = (size_t)bh * p.T + (row_ok ? i : 0);
      const float M = row_ok ? p.row_max[rw] : 0.f;
      const float m_st = (row_ok && CAL == CAL_MINMAX) ? p.row_min[rw] : 0.f;
      const RowGrid gr = row_grid(p, M, m_st);
      for (int b = 0; b < NB; ++b) hist[b] = 0.f;
      ProbeAcc a;
      float invZ = 0.f, invW = 0.f;
      for (int kt = 0; kt < 2 * nkb; ++kt) {
        const int gk = g + kt, b = gk & 1, sweep = kt < nkb ? 0 : 1, kb = sweep ? kt - nkb : kt;
        if (sweep == 1 && kt == nkb) {
          // the row's Z and W (both column groups) before the second sweep.  Every compute
          // thread passes here once per item, failed or not, so the barrier always completes.
          xch[cg * 128 + row] = a.Z;
          xch[(2 + cg) * 128 + row] = a.W;
          group_sync(BAR_COMPUTE, NCOMP);
          invZ = 1.0f / (xch[row] + xch[128 + row]);
          invW = 1.0f / (xch[256 + row] + xch[384 + row]);
          group_sync(BAR_COMPUTE, NCOMP);
        }
        if (failed) continue;  // (a timed-out wait: no further waits, only the barriers)
        if (!mbar_wait(&bar_s[b], (gk >> 1) & 1, p.wait_ns, p.status, DEV_ERR_TIMEOUT_MMA)) {
          failed = true;
          continue;
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
          if (row_ok) {
            if (diag)
              probe_chunk<CAL, REC, true>(v, j0, i, p.scale, M, gr, Kq, sweep, invZ, invW, hist, a);
            else
              probe_chunk<CAL, REC, false>(v, j0, i, p.scale, M, gr, Kq, sweep, invZ, invW, hist, a);
          }
        }
        tc_fence_before();
        __syncwarp();
        if ((tid & 31) == 0) mbar_arrive(&bar_sfree[b]);
      }
      g += 2 * nkb;
      failed = group_any(BAR_COMPUTE, NCOMP, failed);
      if (failed) break;
      // combine the column groups: group 1 hands its sums (and bucket masses) to group 0
      if (cg == 1) {
        xch[0 * 128 + row] = a.Zz;
        xch[1 * 128 + row] = a.below;
        xch[2 * 128 + row] = a.top;
        xch[3 * 128 + row] = a.mn;
        xch[4 * 128 + row] = a.tv;
        xch[5 * 128 + row] = a.Z;
      }
      group_sync(BAR_COMPUTE, NCOMP);
      if (cg == 0 && row_ok) {
        const float* hist1 = hist + (size_t)128 * NB;
        const float Z = a.Z + xch[5 * 128 + row], Zz = a.Zz + xch[row];
        float Hq = 0.f;
        for (int b = 0; b < NB; ++b) {
          const float q = (hist[b] + hist1[b]) / Z;
          Hq -= q > 0.f ? q * logf(q) : 0.f;
        }
        const float mn = fminf(a.mn, xch[3 * 128 + row]);
        const float m = CAL == CAL_MINMAX ? m_st : mn;
        const size_t plane = (size_t)p.BH * p.T;
        float* out = p.probe + rw;
        out[0 * plane] = gr.nogrid ? 0.f : __fsub_rn(M, m);
        out[1 * plane] = gr.nogrid ? 0.f : gr.h;
        out[2 * plane] = logf(Z) - Zz / Z;
        out[3 * plane] = (a.below + xch[128 + row]) / (float)(i + 1);
        out[4 * plane] = (a.top + xch[2 * 128 + row]) / Z;
        out[5 * plane] = expf(Hq);
        out[6 * plane] = 0.5f * (a.tv + xch[4 * 128 + row]);
      }
      group_sync(BAR_COMPUTE, NCOMP);  // the exchange words and histograms are read before the next item
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

cudaError_t launch_fwd_probe(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  auto kern = p.calib == CAL_MINMAX ? (p.recon == REC_NEAREST ? k_fwd_probe<CAL_MINMAX, REC_NEAREST>
                                                              : k_fwd_probe<CAL_MINMAX, REC_LERP>)
                                    : (p.recon == REC_NEAREST ? k_fwd_probe<CAL_FWM, REC_NEAREST>
                                                              : k_fwd_probe<CAL_FWM, REC_LERP>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3((unsigned)p.ngrid), dim3(NTHR), smem_bytes, s, maps, p);
}

}  // namespace kint
