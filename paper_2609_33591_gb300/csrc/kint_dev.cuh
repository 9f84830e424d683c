// Device building blocks of the K-interval attention kernels: the per-row grid
// (Sec. 3 "Objects and calibration", App. A), the per-key decisions and weights
// (App. A "LERP", "Nearest"), and the tile movement / tensor-core helpers.
#pragma once
#include <cuda_bf16.h>
#include <cstdint>
#include <cuda.h>
#include "kint_params.h"
#include "tc.cuh"

namespace kint {

constexpr float kLog2e = 1.4426950408889634f;  // log2(e)

constexpr int NT = 128;              // threads per CTA; thread t owns TMEM lane t
constexpr int SW = 128;              // bytes of one swizzled panel row (32 fp32)

__device__ __forceinline__ uint8_t* smem_base() {
  extern __shared__ uint8_t smem_raw[];
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
}

// CTA-wide "did anyone fail" barrier.  Every thread reaches it, so a thread that
// timed out in a bounded wait never leaves another one behind.
__device__ __forceinline__ bool cta_any(bool failed) { return __syncthreads_or(failed ? 1 : 0) != 0; }

// Named barrier over the `n` compute threads only (the producer warp never takes
// part), and its "did anyone fail" reduction.
__device__ __forceinline__ void group_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ bool group_any(int id, int n, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// Thread roles of the warp-specialised kernels: NCG column groups of 128
// compute threads (warps [0, 4 NCG); thread t owns TMEM lane t % 128 and the
// column group t / 128 of every score tile), then one MMA warp and one TMA
// producer warp.  The compute warps meet no CTA-wide barrier inside the tile
// loops: tiles change hands through mbarriers only.
constexpr int NCG = 2;
constexpr int NCOMP = 128 * NCG;
constexpr int NTHR = NCOMP + 64;
constexpr int MMA_WARP = NCOMP / 32;
constexpr int PRODUCER_WARP = NCOMP / 32 + 1;
// The dQ kernel issues its two kinds of products from two warps on different SM
// sub-partitions: S, g from MMA_WARP, dQ from MMA2_WARP.
constexpr int MMA2_WARP = NCOMP / 32 + 2;
constexpr int NTHR_DQ = NTHR + 32;
constexpr int BAR_COMPUTE = 1;  // named barrier id of the compute group

// W-column TMEM row access (W = 16 or 32).
template <int W>
__device__ __forceinline__ void tmem_ldw(uint32_t taddr, float (&v)[W]) {
  if constexpr (W == 32) {
    tmem_ld32(taddr, v);
  } else {
    tmem_ld16(taddr, v);
  }
}
template <int W>
__device__ __forceinline__ void tmem_stw(uint32_t taddr, const float (&v)[W]) {
  if constexpr (W == 32) {
    tmem_st32(taddr, v);
  } else {
    tmem_st16(taddr, v);
  }
}

// Per-query-row record written by the dQ kernel for the dK/dV kernel (64 bytes).
struct RowRec {
  float c0, k1, invWf, ga;  // position acc * k1 + c0 (u; 2u for FWM Nearest; log2 e^{s-M} for softmax);
                            // forward 1/W; gamma = g * ga + gb
  float gb, cMn;            // c_M / n_max
  int amax, flags;          // arg-max; flags: 1 no grid, 2 tied maxima, 4 tied minima
  float inv_h, cmn;         // 1/h (MinMax); c_m / n_min
  int amin, pad0;           // arg-min
  float M, m, pad1, pad2;   // extrema
};
constexpr int REC_NOGRID = 1, REC_TIEMAX = 2, REC_TIEMIN = 4;

// Position in a ring of n slots used round robin (pipeline stages, score buffers): the
// slot and the parity of its current use, since the uses of one slot alternate the
// phases of its mbarriers.  Kept as counters, so the per-tile paths divide nothing.
struct RingPos {
  int i = 0;
  uint32_t ph = 0;
  __device__ __forceinline__ void next(int n) {
    if (++i == n) {
      i = 0;
      ph ^= 1u;
    }
  }
};

// Clean-up before a kernel leaves (also after a wait ran out): the last n loads issued
// into a ring of NS stages, `next` being the ring position of the load that would come
// next, have landed, so no copy still writes into shared memory.  Each of those loads was
// the last one into its stage, so waiting on the parity of its phase returns at once when
// it completed long ago.  Bounded like every wait; warp-collective.
__device__ __forceinline__ void drain_ring(uint64_t* bar_full, RingPos next, int n, int NS, uint64_t timeout_ns,
                                           unsigned* status) {
  for (int k = 1; k <= n && k <= NS; ++k) {
    int i = next.i - k;
    uint32_t ph = next.ph;
    if (i < 0) {  // the previous lap of the ring (k <= NS: at most one wrap)
      i += NS;
      ph ^= 1u;
    }
    mbar_wait_warp(&bar_full[i], ph, timeout_ns, status, DEV_ERR_TIMEOUT_TMA);
  }
}
// Clean-up of an MMA-issuing warp: every tcgen05.mma it issued has completed (one commit
// onto `bar`, a barrier used for nothing else, whose first phase counts `arrivals` such
// commits), so the TMEM they write can be released.  Bounded; warp-collective.
__device__ __forceinline__ void drain_mma(uint64_t* bar, uint64_t timeout_ns, unsigned* status) {
  mma_commit(bar);
  mbar_wait_warp(bar, 0, timeout_ns, status, DEV_ERR_TIMEOUT_MMA);
}

// Test hook of the bounded waits (Params::expire_wait): thread 0 waits on `bar`, a
// barrier nothing ever arrives at, until the wait limit runs out and flags the status
// word; the whole CTA learns of it and skips its work (nothing has been issued yet, so
// nothing is in flight).  Returns true when the CTA must skip.
__device__ __forceinline__ bool expire_first_wait(const Params& p, uint64_t* bar) {
  bool ok = true;
  if (p.expire_wait && threadIdx.x == 0) ok = mbar_wait(bar, 0, p.wait_ns, p.status, DEV_ERR_TIMEOUT_SYNC);
  return p.expire_wait ? cta_any(!ok) : false;
}

// A gated launch (Params::gate) on the side of a device-side decision that was not
// taken: the kernel does no work.  Read after pdl_wait, so the writer of the decision
// (an earlier kernel of the stream) has finished.
__device__ __forceinline__ bool gated_off(const Params& p) {
  return p.gate != nullptr && ((*reinterpret_cast<const volatile int*>(p.gate) != 0) != (p.gate_on != 0));
}

// n-th work item of this CTA when the grid loops over items sorted longest first:
// rounds of gridDim.x items taken in alternating directions (CTA 0 takes the longest
// item of even rounds and the shortest of odd ones), which evens out the per-CTA
// totals better than a plain stride.  With one CTA per item it is blockIdx.x.
__device__ __forceinline__ int snake_item(int n) {
  const int G = gridDim.x, c = blockIdx.x;
  return n * G + ((n & 1) ? G - 1 - c : c);
}

// n-th work item of this CTA under a host schedule (Sched), or in snake order without
// one; past the CTA's last item it returns a value above every item index.
__device__ __forceinline__ int sched_item(const Sched& s, int n) {
  if (s.n == 0) return snake_item(n);
  const int k = s.off[blockIdx.x] + n;
  return k < s.off[blockIdx.x + 1] ? (int)s.idx[k] : 0x7fffffff;
}

// ---------------------------------------------------------------------------
// Row grid.  Scores s are fp32 values of acc * scale.  The position of a key in
// grid units is u = s * inv_h + c0:
//   MinMax: u = (s - m) / h, h = (M - m) / K       (App. A "MinMax grid")
//   FWM:    u = (s - M + tau) / h, h = tau / K      (App. A "FWM")
// so u in [0, K] inside the grid; FWM keys with u < 0 are the zero tail.
// Every kernel builds it with this one function, so decisions agree bitwise
// between the passes.
// ---------------------------------------------------------------------------
struct RowGrid {
  float inv_h, c0, h, b0;
  float hl, b0l;  // resolved grid: e_r = 2^(r hl + b0l)
  float k1;     // scale * inv_h: u = acc * k1 + c0 straight from the raw accumulator
  bool nogrid;  // degenerate MinMax row (M - m <= 1e-12) or softmax
};

__device__ __forceinline__ RowGrid row_grid(const Params& p, float M, float m) {
  RowGrid g;
  g.hl = p.fwm_hl;
  g.b0l = p.fwm_b0l;
  if (p.calib == CAL_MINMAX) {
    const float span = __fsub_rn(M, m);
    g.nogrid = !(span > 1e-12f);
    const float sp = g.nogrid ? 1.0f : span;
    g.h = __fdiv_rn(sp, (float)p.Kint);
    g.inv_h = __fdiv_rn((float)p.Kint, sp);
    g.c0 = -__fmul_rn(m, g.inv_h);
    g.b0 = __fsub_rn(m, M);
    g.k1 = __fmul_rn(p.scale, g.inv_h);
  } else if (fwm_like(p.calib)) {
    g.nogrid = false;
    g.h = __fdiv_rn(p.tau, (float)p.Kint);
    g.inv_h = p.fwm_inv_h;
    g.c0 = __fmul_rn(__fsub_rn(p.tau, M), g.inv_h);
    g.b0 = -p.tau;
    g.k1 = __fmul_rn(p.scale, g.inv_h);
  } else {
    // (the FP8 and BF16 exponentials keep the row max's gradient channel)
    g.nogrid = p.calib != CAL_EXP8 && p.calib != CAL_EXPB;
    g.h = 1.0f;
    g.inv_h = 1.0f;
    g.c0 = -M;  // z = acc * scale - M (the BF16 exponential rounds z itself)
    g.b0 = 0.0f;
    g.k1 = p.scale;
  }
  return g;
}

// ---------------------------------------------------------------------------
// Branch-free per-key decisions from the grid position u (App. A):
//   uc = clip(u, 0, K); r = min(floor(uc), K-1); t = uc - r in [0, 1];
//   Nearest takes e_{r+1} when t >= 1/2 (l = r + [t >= 1/2], midpoint up).
// floor uses the float-to-int magic-number method: adding 2^23 with rounding
// toward -inf leaves 2^23 + floor(uc) exactly for 0 <= uc < 2^23, so the float's
// bit pattern is 0x4B000000 + r.  `rb` is that bit pattern; a table whose rows
// are 1024 bytes apart is addressed as base + rb * 1024 (mod 2^32), since
// 0x4B000000 * 1024 = 0 mod 2^32.
// ---------------------------------------------------------------------------
constexpr float kMagic = 8388608.0f;  // 2^23

__device__ __forceinline__ void decode_u(float u, float Kf, float& t, uint32_t& rb, float& rf) {
  const float uc = fminf(fmaxf(u, 0.0f), Kf);
  const float fr = fminf(__fadd_rd(uc, kMagic), kMagic + (Kf - 1.0f));
  rf = __fsub_rn(fr, kMagic);
  t = __fsub_rn(uc, rf);
  rb = __float_as_uint(fr);
}

// Zero entries ahead of r = 0 in the pair table of the resolved policy's forward (FWMR).
constexpr int kFwdTail = 2;

// ---------------------------------------------------------------------------
// FWM half-bin index.  With v = 2u (formed exactly as acc * 2k1 + 2c0) and
// u = r + t, floor(v) = 2r + [t >= 1/2]: one floor gives both the bin r = q >> 1
// and the Nearest endpoint (q + 1) >> 1, with the same decisions as decode_u.
// Clamping v to [-1, 2K] sends u >= K to q = 2K and the tail u < 0 to the two
// patterns just below 2^23 (2^23 - 1 and 2^23 - 1/2 after rounding down), so a
// table of 2K + 3 entries, two tail entries first, is indexed by the float bits:
// entry q sits at base + (bits - 0x4B000000) * size.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t fwm_half_bits(float v, float twoK) {
  return __float_as_uint(__fadd_rd(fminf(fmaxf(v, -1.0f), twoK), kMagic));
}
constexpr int kHalfTail = 2;  // tail entries ahead of q = 0

// Entry q in [-2, 2K] of the half-bin table: (w^N, Delta_r / h) with r = min(q >> 1, K - 1)
// (zeros in the tail); Delta_r / h is rounded as the full decode path rounds it.
__device__ __forceinline__ float2 fwm_half_entry(const Params& p, int q) {
  if (q < 0) return make_float2(0.f, 0.f);
  const int r = min(q >> 1, p.Kint - 1);
  const float dlt = __fmul_rn(__fsub_rn(p.fwm_e[r + 1], p.fwm_e[r]), p.fwm_inv_h);
  return make_float2(p.fwm_e[(q + 1) >> 1], dlt);
}

// Entry q in [-2, 2K] of the forward's FWM half-bin table: {alpha, beta, w^N, 0} with
// r = min(q >> 1, K - 1), beta = (e_{r+1} - e_r) / 2 and alpha = e_r - 2 r beta, so that
// the LERP weight e_r + (u - r)(e_{r+1} - e_r) is the bin's line alpha + v beta at v = 2u
// and w^N = e_{(q+1) >> 1} is the Nearest endpoint; the tail entries (q < 0) are zero, so a
// key below the window reads w^L = w^N = 0 whatever its v.
__device__ __forceinline__ float4 fwm_line_entry(const Params& p, int q) {
  if (q < 0) return make_float4(0.f, 0.f, 0.f, 0.f);
  const int r = min(q >> 1, p.Kint - 1);
  const float beta = 0.5f * __fsub_rn(p.fwm_e[r + 1], p.fwm_e[r]);
  return make_float4(__fmaf_rn(-2.0f * (float)r, beta, p.fwm_e[r]), beta, p.fwm_e[(q + 1) >> 1], 0.f);
}

__device__ __forceinline__ float lds_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ float2 lds_f2(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
  return v;
}
__device__ __forceinline__ float4 lds_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Grid value e^{b_r}, r = 0..K.  MinMax: b_r = b0 + r h from the row's own
// extrema (device expf, K + 1 calls per row).  FWM: host table.
__device__ __forceinline__ float grid_value(const Params& p, const RowGrid& g, int r) {
  if (fwm_like(p.calib)) return p.fwm_e[r];
  return expf(__fmaf_rn((float)r, g.h, g.b0));
}

// BF16 exponential (App. "Reduced-precision exponential baselines"): round to the nearest
// bfloat16, ties to even (the CUDA conversion), and the low byte of its bit pattern (the
// decision code: it tells apart the two bfloat16 neighbours of a value).
__device__ __forceinline__ float bf16_rn(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }
__device__ __forceinline__ int bf16_low_byte(float x) {
  return (int)(__bfloat16_as_ushort(__float2bfloat16_rn(x)) & 0xFFu);
}
// w = bf16(e^{bf16(z)}) from z, and the pair (bf16(z), w) for the decision dump
__device__ __forceinline__ float bf16_exp_weight(float z, float& zb) {
  zb = bf16_rn(z);
  return bf16_rn(ex2_approx(__fmul_rn(zb, 1.4426950408889634f)));
}

// FP8-rounded exponential (App. "Reduced-precision exponential baselines"): 0 <= w <= 1
// to the nearest OCP E4M3 value, ties to even.  Normals (w >= 2^-6) keep 3 mantissa bits:
// adding 2^19 - 1 plus the kept LSB to the bit pattern and clearing the 20 dropped bits
// rounds to nearest even (a mantissa carry moves into the exponent).  Below 2^-6 the
// format's subnormals are the multiples of 2^-9: rint(w 2^9) 2^-9.  Both are exact.
__device__ __forceinline__ float e4m3_rn(float w) {
  uint32_t u = __float_as_uint(w);
  u = (u + 0x7FFFFu + ((u >> 20) & 1u)) & 0xFFF00000u;
  const float wsub = __fmul_rn(rintf(__fmul_rn(w, 512.0f)), 0.001953125f);
  return w < 0.015625f ? wsub : __uint_as_float(u);
}
// The E4M3 byte of an E4M3 value in [0, 1] (for the decision dump).
__device__ __forceinline__ int e4m3_code(float wr) {
  if (wr < 0.015625f) return (int)__fmul_rn(wr, 512.0f);
  const uint32_t u = __float_as_uint(wr);
  return ((int)((u >> 23) & 0xFFu) - 127 + 7) << 3 | (int)((u >> 20) & 7u);
}

// Resolved tail policy (App. "Tail policy in the MinMax -> FWM change"): below the
// window (u < 0) FWM's grid continues with negative indices, r = floor(u), t = u - r
// (exact), and the grid values e^{-tau + r tau/K} = 2^(r hl + b0l) come from the
// exponential unit (far below the window they flush to zero).  Only read where u < 0.
struct BelowPair {
  float t, e0, e1;  // position in the interval, e_r, e_{r+1}
};
__device__ __forceinline__ BelowPair resolved_below(float u, float hl, float b0l) {
  BelowPair b;
  const float rf = floorf(u);
  b.t = __fsub_rn(u, rf);
  b.e0 = ex2_approx(__fmaf_rn(rf, hl, b0l));
  b.e1 = ex2_approx(__fmaf_rn(__fadd_rn(rf, 1.0f), hl, b0l));
  return b;
}

// ---------------------------------------------------------------------------
// Tiles.  Every operand tile in shared memory is stored as 32-column panels of
// 128-byte rows in the 128-byte swizzle that TMA writes and tcgen05 reads:
//   natural tile    X[row0 .. row0+R) x [0, d):  d/32 panels of R*128 bytes
//   transposed tile X^T[0 .. d) x [key0, key0+C): C/32 panels of d*128 bytes
// In both, "rows" are the MMA's M or N index and the 32-wide panels run along K.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void load_rows_tile(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int ncols,
                                               int nrows, int c_first, int r_first, int bh) {
  // ncols/32 panels of nrows x 32 fp32 from coordinates (c_first + 32 p, r_first, bh)
  for (int pnl = 0; pnl < ncols / 32; ++pnl)
    tma_load_3d(dst + pnl * nrows * SW, map, bar, c_first + 32 * pnl, r_first, bh);
}
// A tile of nrows rows fetched as nrows / box row boxes per panel (a map whose box is
// `box` rows); box * 128 bytes is a multiple of the 1024-byte swizzle atom.
__device__ __forceinline__ void load_rows_tile_boxed(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int ncols,
                                                     int nrows, int box, int c_first, int r_first, int bh) {
  for (int pnl = 0; pnl < ncols / 32; ++pnl)
    for (int r = 0; r < nrows; r += box)
      tma_load_3d(dst + pnl * nrows * SW + r * SW, map, bar, c_first + 32 * pnl, r_first + r, bh);
}

// The calling thread's row `row` (values v[0..31], columns [32 pnl, 32 pnl + 32))
// into a 128-row tile in smem laid out like the TMA tiles (128-byte swizzle, panels
// of 32 columns 128 x 128 bytes apart), for a TMA store.
__device__ __forceinline__ void row_to_staged(uint8_t* tile, int row, int pnl, const float (&v)[32]) {
  const uint32_t base = smem_u32(tile) + (uint32_t)pnl * 128u * SW + (uint32_t)row * SW;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const uint32_t a = base + (uint32_t)((c ^ (row & 7)) << 4);
    asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(a), "f"(v[4 * c]), "f"(v[4 * c + 1]),
                 "f"(v[4 * c + 2]), "f"(v[4 * c + 3])
                 : "memory");
  }
}
// A staged 128-row tile (ncols columns) to rows [r_first, r_first + 128) of head bh
// through a map whose box is `box` rows (warp-collective).  With `wait`, returns once
// the tile has been read out of shared memory; otherwise the caller waits later
// (tma_store_wait_read) before it writes the tile again.
__device__ __forceinline__ void store_rows_tile_boxed(const uint8_t* tile, const CUtensorMap* map, int ncols, int box,
                                                      int r_first, int bh, bool wait = true) {
  for (int pnl = 0; pnl < ncols / 32; ++pnl)
    for (int r = 0; r < 128; r += box) tma_store_3d(map, tile + pnl * 128 * SW + r * SW, 32 * pnl, r_first + r, bh);
  tma_store_commit();
  if (wait) tma_store_wait_read();
}

// ---------------------------------------------------------------------------
// Tensor-core products.  The issuing thread's own instruction stream bounds the
// MMA rate (measured on GB300: an M=128, N=128 tf32 MMA every ~33 ns with
// constant descriptors, ~43 ns when each descriptor is rebuilt), so descriptors
// are built once per operand and advanced with one 32-bit add per k-step: the
// start-address field holds (address >> 4) in 14 bits and shared addresses
// stay below 256 KB, so the add never carries out of the field.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t desc_add(uint64_t d, uint32_t off16) {
  uint32_t lo = (uint32_t)d + off16, hi = (uint32_t)(d >> 32);
  return ((uint64_t)hi << 32) | lo;
}

// D[tmem, M=128 x N] (+)= A * B^T over KSTEPS x 8, A and B in smem (panels of
// 32 K-columns, 128 B per row; A panels a_pnl bytes apart, B panels b_pnl).
template <int KSTEPS>
__device__ __forceinline__ void mma_ss_k(uint32_t d_tmem, const uint8_t* a, const uint8_t* b, int a_pnl, int b_pnl,
                                         uint32_t idesc, bool accumulate) {
  const uint64_t a0 = smem_desc_sw128(smem_u32(a), 16, 1024);
  const uint64_t b0 = smem_desc_sw128(smem_u32(b), 16, 1024);
  const uint32_t ap = (uint32_t)a_pnl >> 4, bp = (uint32_t)b_pnl >> 4;
#pragma unroll
  for (int kk = 0; kk < KSTEPS; ++kk) {
    const uint32_t sub = (uint32_t)(kk & 3) * 2u;  // 32 bytes per k-step inside a panel
    mma_tf32_ss(d_tmem, desc_add(a0, (uint32_t)(kk >> 2) * ap + sub), desc_add(b0, (uint32_t)(kk >> 2) * bp + sub),
                idesc, (accumulate || kk > 0) ? 1u : 0u);
  }
}
// D[tmem, M=128 x N] (+)= A * B^T over KSTEPS x 8, A in TMEM columns.
template <int KSTEPS>
__device__ __forceinline__ void mma_ts_k(uint32_t d_tmem, uint32_t a_tmem, const uint8_t* b, int b_pnl,
                                         uint32_t idesc, bool accumulate) {
  const uint64_t b0 = smem_desc_sw128(smem_u32(b), 16, 1024);
  const uint32_t bp = (uint32_t)b_pnl >> 4;
#pragma unroll
  for (int kk = 0; kk < KSTEPS; ++kk)
    mma_tf32_ts(d_tmem, a_tmem + kk * 8, desc_add(b0, (uint32_t)(kk >> 2) * bp + (uint32_t)(kk & 3) * 2u), idesc,
                (accumulate || kk > 0) ? 1u : 0u);
}

// Runtime-K wrappers: K = Ktot columns (a multiple of 64) as a rolled loop over
// blocks of eight unrolled steps, which keeps the issuing code small.
__device__ __forceinline__ void mma_smem_smem(uint32_t d_tmem, const uint8_t* a, const uint8_t* b, int N, int Ktot,
                                              bool accumulate) {
  const uint32_t idesc = idesc_tf32(128, N, 0, 0);
#pragma unroll 1
  for (int k0 = 0; k0 < Ktot; k0 += 64)
    mma_ss_k<8>(d_tmem, a + (k0 / 32) * 128 * SW, b + (k0 / 32) * N * SW, 128 * SW, N * SW, idesc,
                accumulate || k0 > 0);
}
__device__ __forceinline__ void mma_tmem_smem(uint32_t d_tmem, uint32_t a_tmem, const uint8_t* b, int N, int Ktot,
                                              bool accumulate) {
  const uint32_t idesc = idesc_tf32(128, N, 0, 0);
#pragma unroll 1
  for (int k0 = 0; k0 < Ktot; k0 += 64)
    mma_ts_k<8>(d_tmem, a_tmem + k0, b + (k0 / 32) * N * SW, N * SW, idesc, accumulate || k0 > 0);
}

// The calling thread's TMEM lane (its row) at column `col`.  Warp w may only
// touch lane quarter w % 4.
__device__ __forceinline__ uint32_t lane_addr(uint32_t tmem_base, int col) {
  const int warp = threadIdx.x >> 5;
  return tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)col;
}

// Columns [c0, c0 + n) of row `row` of X (d fp32 per row) into the calling
// thread's TMEM lane at columns [col + c0, col + c0 + n); with `split`, the tf32 hi
// part there and the lo part d columns further.  All global loads are issued
// before the first TMEM store.  Rows >= T load zeros.  n is 32 or 64; whole
// warps must call this with the same c0, n.
template <int N>
__device__ __forceinline__ void row_to_tmem_part(uint32_t tmem_base, int col, const float* X, int row, int T, int d,
                                                 int c0, bool split) {
  const bool in = row < T;
  const float4* src = reinterpret_cast<const float4*>(X + (size_t)row * d + c0);
  float hi[N], lo[N];
#pragma unroll
  for (int q = 0; q < N / 4; ++q) {
    const float4 x = in ? __ldg(src + q) : make_float4(0.f, 0.f, 0.f, 0.f);
    hi[4 * q] = x.x;
    hi[4 * q + 1] = x.y;
    hi[4 * q + 2] = x.z;
    hi[4 * q + 3] = x.w;
  }
  if (split) {
#pragma unroll
    for (int q = 0; q < N; ++q) {
      const float h = tf32_rna(hi[q]);
      lo[q] = __fsub_rn(hi[q], h);
      hi[q] = h;
    }
    tmem_stw<N>(lane_addr(tmem_base, col + d + c0), lo);
  }
  tmem_stw<N>(lane_addr(tmem_base, col + c0), hi);
}

// Thread-owned row `row` of X (d fp32) into the thread's TMEM lane at columns
// [col, col+d) (hi/lo with `split`, lo at [col+d, col+2d)), 16 columns at a time:
// the path of the configurations without staged operands, kept small so that it
// does not crowd the registers of the kernels' main loops.
__device__ __forceinline__ void row_to_tmem(uint32_t tmem_base, int col, const float* X, int row, int T, int d,
                                            bool split) {
#pragma unroll 1
  for (int c0 = 0; c0 < d; c0 += 16) row_to_tmem_part<16>(tmem_base, col, X, row, T, d, c0, split);
}

// Row `row` of a 128-row K-major tile staged in smem by TMA (128-byte swizzle,
// 32-column panels 128 x 128 bytes apart) into the calling thread's TMEM lane at
// columns [col, col + d).  Chunk c (16 bytes) of a row sits at chunk c ^ (row % 8).
__device__ __forceinline__ void staged_row_to_tmem(uint32_t tmem_base, int col, const uint8_t* tile, int row, int d) {
  const uint32_t base = smem_u32(tile) + (uint32_t)row * SW;
#pragma unroll 1
  for (int h = 0; h < d / 16; ++h) {  // 16 columns (half a panel) at a time
    const uint32_t pb = base + (uint32_t)(h >> 1) * 128u * SW;
    float v[16];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int chunk = (h & 1) * 4 + c;
      const float4 x = lds_f4(pb + (uint32_t)((chunk ^ (row & 7)) << 4));
      v[4 * c] = x.x;
      v[4 * c + 1] = x.y;
      v[4 * c + 2] = x.z;
      v[4 * c + 3] = x.w;
    }
    tmem_st16(lane_addr(tmem_base, col + 16 * h), v);
  }
}


}  // namespace kint
