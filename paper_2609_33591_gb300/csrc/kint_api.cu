// C ABI of libkint (include/kint_attn.h): argument checks, workspace layout,
// TMA descriptors, shared-memory plans and the launch sequence of each entry
// point.  Nothing here allocates device memory or synchronises, except
// kint_get_status.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <atomic>
#include <memory>
#include <mutex>
#include <vector>

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "../../include/kint_attn.h"
#include "kint_launch.h"
#include "kint_params.h"

namespace kint {

// Device-side fault flags (see tc.cuh); read and cleared by kint_get_status.
__device__ unsigned g_status_word = 0;

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
unsigned* g_status_ptr[kMaxDevices] = {nullptr};
int g_dev_ok[kMaxDevices] = {0};  // 0 unknown, 1 sm_103, -1 other
int g_num_sms[kMaxDevices] = {0};
unsigned long long g_wait_ns = 2000000000ull;
std::atomic<int> g_expire_waits{0};  // test hook: forward calls whose first kernel's first wait runs out
int g_bwd_path = 0;  // 0: single-pass backward where it applies, 1: always the two-pass kernels
constexpr int kSmemLimit = 232448;  // opt-in maximum per CTA on sm_103
constexpr int NCOMP_THREADS = 256;  // compute threads of the warp-specialised kernels (kint_dev.cuh NCOMP)

int round_up(int x, int m) { return (x + m - 1) / m * m; }
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Item schedules of the persistent kernels (Sched), longest processing time first: an
// item costs a + tiles (a = its fixed cost in tiles: operand loads, epilogue, measured
// per CTA), and items in decreasing cost each go to the CTA with the least work so far,
// ties to the lower CTA.  Built once per kernel and shape and kept.
enum SchedKind { SCHED_STATS = 0, SCHED_MAIN = 1, SCHED_FUSED = 2 };

struct SchedEntry {
  int kind, nitems, ngrid, BH, nqb, nqt;
  Sched sch;
};
std::vector<std::unique_ptr<SchedEntry>> g_sched;

const Sched& sched_for(int kind, const Params& p) {
  static const Sched none = [] { Sched z; std::memset(&z, 0, sizeof(z)); return z; }();
  if (p.ngrid >= p.nitems || p.ngrid > SCHED_MAX_CTAS || p.nitems > SCHED_MAX_ITEMS) return none;
  const int nqt = kind == SCHED_FUSED ? p.nqt : 0;
  std::lock_guard<std::mutex> lk(g_mu);
  for (const auto& e : g_sched)
    if (e->kind == kind && e->nitems == p.nitems && e->ngrid == p.ngrid && e->BH == p.BH && e->nqb == p.nqb &&
        e->nqt == nqt)
      return e->sch;
  if (g_sched.size() >= 256) return none;  // entries are never released: bound their number
  // tiles and fixed cost of item i: query blocks (longest first) for the forward passes, key
  // blocks with their 64-row query tiles for the single-pass backward
  const double fixed = kind == SCHED_MAIN ? 2.6 : 2.0;
  std::vector<double> cost(p.nitems);
  for (int i = 0; i < p.nitems; ++i) {
    int tiles;
    if (kind == SCHED_FUSED)
      tiles = p.nqt - (i / p.BH) * 2;
    else
      tiles = p.nqb - i / p.BH;
    cost[i] = fixed + tiles;
  }
  std::vector<int> order(p.nitems);
  for (int i = 0; i < p.nitems; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
  std::vector<double> load(p.ngrid, 0.0);
  std::vector<std::vector<int>> lists(p.ngrid);
  for (int i : order) {
    int best = 0;
    for (int c = 1; c < p.ngrid; ++c)
      if (load[c] < load[best]) best = c;
    load[best] += cost[i];
    lists[best].push_back(i);
  }
  auto e = std::make_unique<SchedEntry>();
  std::memset(&e->sch, 0, sizeof(Sched));
  e->kind = kind;
  e->nitems = p.nitems;
  e->ngrid = p.ngrid;
  e->BH = p.BH;
  e->nqb = p.nqb;
  e->nqt = nqt;
  int k = 0;
  for (int c = 0; c < p.ngrid; ++c) {
    e->sch.off[c] = (uint16_t)k;
    for (int i : lists[c]) e->sch.idx[k++] = (uint16_t)i;
  }
  e->sch.off[p.ngrid] = (uint16_t)k;
  e->sch.n = p.nitems;
  g_sched.push_back(std::move(e));
  return g_sched.back()->sch;
}

// Resolve the device-dependent handles once per device.
int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
  return g_num_sms[dev] > 0 ? g_num_sms[dev] : 1;
}

int device_setup(unsigned** status) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KINT_ERR_NO_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_dev_ok[dev] == 0) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
      return KINT_ERR_NO_DEVICE;
    }
    g_dev_ok[dev] = (major == 10 && minor == 3) ? 1 : -1;
    if (g_dev_ok[dev] == 1) {
      void* ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_status_word) != cudaSuccess) {
        g_dev_ok[dev] = 0;
        return KINT_ERR_NO_DEVICE;
      }
      g_status_ptr[dev] = static_cast<unsigned*>(ptr);
      if (cudaDeviceGetAttribute(&g_num_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
          g_num_sms[dev] < 1) {
        g_dev_ok[dev] = 0;
        return KINT_ERR_NO_DEVICE;
      }
    }
  }
  if (g_dev_ok[dev] != 1) return KINT_ERR_NO_DEVICE;
  if (!g_encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return KINT_ERR_NO_DEVICE;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  *status = g_status_ptr[dev];
  return KINT_OK;
}

// Natural view of X [BH][T][d]: box (32 columns, rows).
bool map_nat(CUtensorMap* m, const float* X, int BH, int T, int d, int rows) {
  cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)T, (cuuint64_t)BH};
  cuuint64_t strides[2] = {(cuuint64_t)d * 4, (cuuint64_t)T * d * 4};
  cuuint32_t box[3] = {32, (cuuint32_t)rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(X), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
// X [BH][T][d] with a box of (cols, rows) and the 64-byte swizzle (cols = 16): the single-pass
// backward's dQ reduce and dV / dK stores, 16 columns per compute warp.
bool map_nat_sw64(CUtensorMap* m, const float* X, int BH, int T, int d, int cols, int rows) {
  cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)T, (cuuint64_t)BH};
  cuuint64_t strides[2] = {(cuuint64_t)d * 4, (cuuint64_t)T * d * 4};
  cuuint32_t box[3] = {(cuuint32_t)cols, (cuuint32_t)rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(X), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
// Transposed view of X^T [BH][d][Tp] (valid columns T): box (32 keys, d rows).
bool map_tr(CUtensorMap* m, const float* XT, int BH, int T, int Tp, int d) {
  cuuint64_t dims[3] = {(cuuint64_t)T, (cuuint64_t)d, (cuuint64_t)BH};
  cuuint64_t strides[2] = {(cuuint64_t)Tp * 4, (cuuint64_t)d * Tp * 4};
  cuuint32_t box[3] = {32, (cuuint32_t)d, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(XT), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Workspace layout (floats), identical for the size query and the launches.
struct Workspace {
  size_t bytes = 0;
  // forward / backward operand copies
  float *qh = nullptr, *ql = nullptr, *kh = nullptr, *kl = nullptr, *vh = nullptr, *vl = nullptr,
        *doh = nullptr, *dol = nullptr;
  float *vth = nullptr, *vtl = nullptr, *kth = nullptr, *ktl = nullptr, *qth = nullptr, *qtl = nullptr,
        *doth = nullptr, *dotl = nullptr;
  void* rec = nullptr;    // [BHT] 64-byte per-row records (dQ kernel -> dK/dV kernel)
  float* rtab = nullptr;  // [BHT][KMAX] (e_r, e_{r+1}) MinMax grid pairs
  float* tie = nullptr;   // [2][BHT][d] sums of tied arg-extremum keys
  int* tileflags = nullptr;  // [BH][ceil(T/64)]
  int* tie_any = nullptr;    // after tileflags (zeroed with them): the ties overflow the tie list
  int *tie_count = nullptr, *tie_total = nullptr;  // (also zeroed with the tile flags)
  int2* tie_list = nullptr;  // [BHT] (row, key) pairs of tied maxima (single-pass backward)
  void* frec = nullptr;      // [BHT] 16-byte rows records of the single-pass backward
  float* rsum = nullptr;     // [BHT] its row sums of gamma Delta
  float* gbar = nullptr;     // [BHT] <g>_{P*} = dO_i . O*_i
};

Workspace plan_workspace(char* base, int BH, int T, int d, bool x3, bool bwd) {
  Workspace w;
  const int Tp = round_up(T, 32);
  const size_t nat = (size_t)BH * T * d * 4, tr = (size_t)BH * d * Tp * 4, rows = (size_t)BH * T * 4;
  size_t off = 0;
  auto take = [&](size_t n) -> float* {
    float* p = base ? reinterpret_cast<float*>(base + off) : nullptr;
    off = align256(off + n);
    return p;
  };
  if (!bwd) {
    if (x3) {
      w.qh = take(nat); w.ql = take(nat); w.kh = take(nat); w.kl = take(nat);
      w.vth = take(tr); w.vtl = take(tr);
    } else {
      w.vth = take(tr);
    }
  } else {
    if (x3) {
      w.qh = take(nat); w.ql = take(nat); w.kh = take(nat); w.kl = take(nat);
      w.vh = take(nat); w.vl = take(nat); w.doh = take(nat); w.dol = take(nat);
      w.kth = take(tr); w.ktl = take(tr); w.qth = take(tr); w.qtl = take(tr); w.doth = take(tr); w.dotl = take(tr);
    } else {
      w.kth = take(tr); w.qth = take(tr); w.doth = take(tr);
    }
    w.rec = take(rows * 16);
    w.rtab = take(rows * 2 * KMAX);
    w.tie = take(2 * nat);
    const size_t ntf = (size_t)BH * ((T + 63) / 64);
    w.tileflags = reinterpret_cast<int*>(take((ntf + 4) * 4));
    if (w.tileflags) {
      w.tie_any = w.tileflags + ntf;
      w.tie_count = w.tileflags + ntf + 1;
      w.tie_total = w.tileflags + ntf + 2;
    }
    w.frec = take(rows * 4);
    w.rsum = take(rows);
    w.tie_list = reinterpret_cast<int2*>(take(rows * 2));  // one (row, key) pair per row
    w.gbar = take(rows);
  }
  w.bytes = off;
  return w;
}

struct Common {
  int B, H, T, d, Kint, calib, recon, ste, grad, prec;
  float tau;
};

int validate(const Common& c, int causal) {
  if (c.B < 1 || c.H < 1 || c.T < 1 || c.d < 1) return KINT_ERR_ARG;
  if (causal != 1) return KINT_ERR_ARG;
  if (c.calib < 0 || c.calib > 5 || c.recon < 0 || c.recon > 1 || c.ste < 0 || c.ste > 1 || c.grad < 0 ||
      c.grad > 4 || c.prec < 0 || c.prec > 1)
    return KINT_ERR_ARG;
  const bool grid = c.calib != KINT_CALIB_SOFTMAX && c.calib != KINT_CALIB_EXP_FP8 && c.calib != KINT_CALIB_EXP_BF16;
  if (grid && (c.Kint < 1 || c.Kint > KMAX)) return KINT_ERR_ARG;
  if ((c.calib == KINT_CALIB_FWM || c.calib == KINT_CALIB_FWM_RESOLVED) && !(c.tau > 0.0f && std::isfinite(c.tau)))
    return KINT_ERR_ARG;
  if (c.d != 64 && c.d != 128) return KINT_ERR_UNSUPPORTED;
  if (c.prec == KINT_PREC_3XTF32 && c.d != 64) return KINT_ERR_UNSUPPORTED;
  // MinMax keeps a (K x 128)-pair grid table per query block in shared memory;
  // above K = 32 it fits only beside the TF32, d = 64 operand tiles.
  if (c.calib == KINT_CALIB_MINMAX && c.Kint > 32 && (c.prec == KINT_PREC_3XTF32 || c.d != 64))
    return KINT_ERR_UNSUPPORTED;
  const long long BH = (long long)c.B * c.H;
  if (BH > 65535 || (long long)c.T * BH > (1ll << 31) - 1 || c.T > (1 << 24)) return KINT_ERR_UNSUPPORTED;
  return KINT_OK;
}

Params base_params(const Common& c, unsigned* status) {
  Params p;
  std::memset(&p, 0, sizeof(p));
  p.B = c.B; p.H = c.H; p.T = c.T; p.d = c.d;
  const bool exp_w = c.calib == KINT_CALIB_SOFTMAX || c.calib == KINT_CALIB_EXP_FP8 ||
                     c.calib == KINT_CALIB_EXP_BF16;  // no grid
  p.Kint = exp_w ? 1 : c.Kint;
  p.calib = c.calib; p.recon = c.recon; p.ste = c.ste; p.grad = c.grad;
  if (exp_w) p.recon = p.ste = 0;  // (neither a reconstruction nor a surrogate placement applies)
  p.x3 = c.prec == KINT_PREC_3XTF32;
  p.BH = c.B * c.H;
  p.nqb = (c.T + 127) / 128;
  p.tau = c.tau;
  p.scale = (float)(1.0 / std::sqrt((double)c.d));
  if (c.calib == KINT_CALIB_FWM || c.calib == KINT_CALIB_FWM_RESOLVED) {
    p.fwm_inv_h = (float)((double)c.Kint / (double)c.tau);
    for (int r = 0; r <= c.Kint; ++r)
      p.fwm_e[r] = (float)std::exp(-(double)c.tau + (double)r * (double)c.tau / (double)c.Kint);
    const double log2e = 1.4426950408889634;
    p.fwm_hl = (float)((double)c.tau / (double)c.Kint * log2e);
    p.fwm_b0l = (float)(-(double)c.tau * log2e);
  }
  p.wait_ns = g_wait_ns;
  p.status = status;
  return p;
}

// Finish a shared-memory plan: barriers (+ TMEM slot) after `off`, + 1 KB for alignment.
int finish_plan(Params& p, int off, int nbars) {
  off = round_up(off, 8);
  p.sm_bars = off;
  off += nbars * 8 + 16;
  return off + 1024;
}
// Kernels that allocate all 512 TMEM columns request more than half of an SM's
// shared memory, so two of their CTAs are never resident on one SM at once.
constexpr int kOneCtaPerSm = 117 * 1024;

int plan_stats(Params& p) {
  const int parts = p.x3 ? 2 : 1, tile = p.d * 512;
  p.nitems = p.nqb * p.BH;
  p.sm_a = 0;
  p.sm_stage0 = parts * tile;
  p.sm_stage_bytes = parts * tile;
  p.nstage = 2;
  p.sm_rows = p.sm_stage0 + p.nstage * p.sm_stage_bytes;  // the 6 x 128 exchange words
  const int total = finish_plan(p, p.sm_rows + 6 * 128 * 4, 8 + 2 * p.nstage);
  // CTAs loop over the items, as many as are resident at once (two per SM when they fit)
  const int per_sm = (2 * total <= 228 * 1024) ? 2 : 1;
  p.ngrid = std::min(p.nitems, per_sm * num_sms());
  return total;
}

// Geometry probe: pass 1's layout, 8 x 128 exchange words and a [2][128][K + 2] float
// bucket-mass array per CTA; one CTA per SM.
int plan_probe(Params& p) {
  const int parts = p.x3 ? 2 : 1, tile = p.d * 512;
  p.nitems = p.nqb * p.BH;
  p.sm_a = 0;
  p.sm_stage0 = parts * tile;
  p.sm_stage_bytes = parts * tile;
  p.nstage = 2;
  p.sm_rows = p.sm_stage0 + p.nstage * p.sm_stage_bytes;
  p.sm_table = p.sm_rows + 8 * 128 * 4;
  const int total = finish_plan(p, p.sm_table + 2 * 128 * (p.Kint + 2) * 4, 7 + 2 * p.nstage);
  p.ngrid = std::min(p.nitems, num_sms());
  return total;
}

// mode: PV_MAIN / PV_MAIN_LERP / PV_LERP.  Picks the TMEM score double-buffering
// and the deepest K/V ring that fit.
int plan_main(Params& p, int mode) {
  const int parts = p.x3 ? 2 : 1, tile = p.d * 512;
  // (e_r, e_{r+1}) pairs: per row for MinMax ([K][128]), one shared [K] for FWMR; FWM's
  // half-bin table of 16-byte entries, q in [-2, 2K]
  const int table = p.calib == KINT_CALIB_MINMAX ? p.Kint * 1024
                    : p.calib == KINT_CALIB_FWM  ? std::max(1024, round_up((2 * p.Kint + 3) * 16, 128))
                    : p.calib == KINT_CALIB_FWM_RESOLVED ? 1024 : 0;
  const bool useA2 = mode == PV_MAIN_LERP || p.x3;
  const int cols1 = 128 + (useA2 ? 128 : 0) + p.d + (mode == PV_MAIN_LERP ? p.d : 0);
  const int ostage = (mode == PV_MAIN_LERP ? 2 : 1) * 128 * p.d * 4;  // O (and O_lerp) staging tiles
  p.nitems = p.nqb * p.BH;
  p.sm_a = 0;
  p.sm_stage0 = parts * tile;
  p.sm_stage_bytes = parts * 2 * tile;
  // One CTA per SM looping over the items needs its own output staging area (the
  // stage ring keeps loading the next item); at least two stages.  Otherwise one item
  // per CTA, staging in the ring, which is idle by the epilogue.
  for (int persist = 1; persist >= 0; --persist) {
    for (p.nstage = 3; p.nstage >= (persist ? 2 : 1); --p.nstage) {
      p.nbuf = (cols1 + 128 <= 512) ? 2 : 1;
      p.sm_table = p.sm_stage0 + p.nstage * p.sm_stage_bytes;
      p.sm_ostage = persist ? round_up(p.sm_table + table, 1024) : p.sm_stage0;
      const int end = persist ? p.sm_ostage + ostage : p.sm_table + table;
      const int total = std::max(finish_plan(p, end, 11 + 2 * p.nstage), kOneCtaPerSm);
      if (total <= kSmemLimit) {
        // Issuing S(kb+1) before P V(kb) needs tile kb+1 in a second stage while
        // tile kb's V^T is still being read; with one stage the two would wait on
        // each other, so a single stage means a single score buffer.
        if (p.nstage == 1) p.nbuf = 1;
        p.ngrid = persist ? std::min(p.nitems, num_sms()) : p.nitems;
        return total;
      }
    }
  }
  return -1;
}

// Backward kernels: compute warps + MMA warp + producer warp.  A second score
// buffer (S/g of tile t+1 computed under the element work of tile t) needs TMEM
// room and at least two stages.
int plan_dq(Params& p) {
  const int parts = p.x3 ? 2 : 1, ktile = 64 * p.d * 4, dp = p.d * parts;
  const int table = p.calib == KINT_CALIB_MINMAX ? p.Kint * 1024 : 1024;
  // TF32 at d = 64: Q and dO arrive as TMA tiles staged in smem (64 KB) and are copied
  // to TMEM from there; otherwise (3xTF32 hi/lo, d = 128) the staging area would not fit
  // next to the K/V stages and the rows are read from global memory.
  p.ops_smem = (!p.x3 && p.d == 64) ? 1 : 0;
  p.nbuf = (2 * dp + 256 + p.d <= 512) ? 2 : 1;
  p.nitems = p.nqb * p.BH;
  p.sm_a = 0;
  p.sm_stage0 = p.ops_smem ? 2 * 128 * p.d * 4 : 0;
  p.sm_stage_bytes = 3 * parts * ktile;
  // One CTA per SM looping over the items (dQ goes straight from TMEM to global memory,
  // so the stage ring keeps loading the next item's tiles under the epilogue).
  for (p.nstage = 4; p.nstage >= 1; --p.nstage) {
    p.sm_table = p.sm_stage0 + p.nstage * p.sm_stage_bytes;
    p.sm_rows = p.sm_table + table;
    p.sm_rstat = p.sm_rows + 8 * 128 * 4;
    p.sm_ostage = 0;
    const int total = std::max(finish_plan(p, p.sm_rstat + 9 * NCOMP_THREADS * 4, 3 * p.nstage + 11), kOneCtaPerSm);
    if (total <= kSmemLimit) {
      if (p.nstage == 1) p.nbuf = 1;
      p.ngrid = std::min(p.nitems, num_sms());
      return total;
    }
  }
  return -1;
}

int plan_dkdv(Params& p, int sel) {
  const int parts = p.x3 ? 2 : 1, qtile = 64 * p.d * 4, dp = p.d * parts;
  const bool doDV = sel != DKV_DK, doDK = sel != DKV_DV;
  // TF32 at d = 64, both products: K and V staged in smem by TMA (see plan_dq)
  p.ops_smem = (!p.x3 && p.d == 64 && doDV && doDK) ? 1 : 0;
  const int base = doDK ? 2 * dp : dp;
  // accumulators, and under 3xTF32 (one product per launch) the cross-term accumulator
  const int acc = (doDV ? p.d : 0) + (doDK ? p.d : 0) + (p.x3 ? p.d : 0);
  if (p.x3 && doDV && doDK) return -1;
  if (base + 128 + acc > 512) return -1;
  p.dkv_sel = sel;
  p.nbuf = (base + 256 + acc <= 512) ? 2 : 1;
  p.sm_a = 0;
  p.sm_stage0 = p.ops_smem ? 2 * 128 * p.d * 4 : 0;
  p.sm_stage_bytes = 4 * parts * qtile + 64 * 64 + (p.calib == KINT_CALIB_MINMAX ? 64 * p.Kp * 8 : 0);
  for (p.nstage = 4; p.nstage >= 1; --p.nstage) {
    p.sm_table = p.sm_stage0 + p.nstage * p.sm_stage_bytes;
    // FWM Nearest: the half-bin table, 2K + 3 entries of 8 bytes
    const int table = (p.calib == KINT_CALIB_FWM || p.calib == KINT_CALIB_FWM_RESOLVED) ? 2048 : 1024;
    const int total = std::max(finish_plan(p, p.sm_table + table, 4 * p.nstage + 9), kOneCtaPerSm);
    if (total <= kSmemLimit) {
      if (p.nstage == 1) p.nbuf = 1;
      // one CTA per SM looping over the (key block, head) items
      p.nitems = p.nqb * p.BH;
      p.ngrid = std::min(p.nitems, num_sms());
      return total;
    }
  }
  return -1;
}

// Single-pass backward (TF32, d = 64): two stages of Q | dO | Q^T | dO^T tiles and their
// 16-byte row records, the item's V and K^T tiles, sixteen 1 KB dQ reduce slices, the FWM
// table; one CTA per SM.
int plan_fused(Params& p) {
  const int qtile = 64 * 64 * 4;
  p.nstage = 2;
  p.nbuf = 2;
  p.ops_smem = 0;
  p.sm_a = 0;
  p.sm_stage0 = 0;
  p.sm_stage_bytes = 4 * qtile + 64 * 16;
  p.sm_v = p.sm_stage0 + p.nstage * p.sm_stage_bytes;
  p.sm_kt = p.sm_v + 128 * 64 * 4;
  p.sm_ostage = p.sm_kt + 128 * 64 * 4;  // the compute warps' 1 KB dQ reduce slices
  p.sm_table = p.sm_ostage + 16 * 1024;
  const int total = std::max(finish_plan(p, p.sm_table + 2048, 5 * p.nstage + 13), kOneCtaPerSm);
  if (total > kSmemLimit) return -1;
  p.nitems = p.nqb * p.BH;
  p.ngrid = std::min(p.nitems, num_sms());
  return total;
}

int launch_rc(cudaError_t e) { return e == cudaSuccess ? KINT_OK : KINT_ERR_LAUNCH; }

kint_launch_cb g_cb = nullptr;
void* g_cb_user = nullptr;

// One kernel launch between the optional tracing callbacks.
template <class F>
cudaError_t traced(const char* name, cudaStream_t s, F&& launch) {
  const kint_launch_cb cb = g_cb;
  if (cb) cb(name, 0, s, g_cb_user);
  const cudaError_t e = launch();
  if (cb) cb(name, 1, s, g_cb_user);
  return e;
}

// The operand copies of one pass, all in one launch.
struct PrepList {
  PrepJobs jobs{};
  void add(const float* X, float* nat_hi, float* nat_lo, float* tr_hi, float* tr_lo, const float* Y = nullptr,
           float* dot = nullptr) {
    jobs.j[jobs.n++] = PrepJob{X, Y, nat_hi, nat_lo, tr_hi, tr_lo, dot};
  }
};
cudaError_t prep(const PrepList& l, int BH, int T, int Tp, int d, bool split, cudaStream_t s) {
  return traced("k_prep", s, [&] { return launch_prep(l.jobs, BH, T, Tp, d, split, num_sms(), s); });
}

// Forward prep + pass 1 (shared by kint_attn_fwd and kint_attn_debug_bins).
int forward_prologue(const float* Q, const float* K, const float* V, const Params& p, const Workspace& w,
                     Maps& maps, cudaStream_t s) {
  const int BH = p.BH, T = p.T, d = p.d, Tp = round_up(T, 32);
  PrepList pl;
  if (p.x3) {
    pl.add(Q, w.qh, w.ql, nullptr, nullptr);
    pl.add(K, w.kh, w.kl, nullptr, nullptr);
    pl.add(V, nullptr, nullptr, w.vth, w.vtl);
  } else {
    pl.add(V, nullptr, nullptr, w.vth, nullptr);
  }
  if (prep(pl, BH, T, Tp, d, p.x3 != 0, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  std::memset(&maps, 0, sizeof(maps));
  bool ok = true;
  if (p.x3) {
    ok = ok && map_nat(&maps.q, w.qh, BH, T, d, 128) && map_nat(&maps.q_lo, w.ql, BH, T, d, 128);
    ok = ok && map_nat(&maps.k, w.kh, BH, T, d, 128) && map_nat(&maps.k_lo, w.kl, BH, T, d, 128);
    ok = ok && map_tr(&maps.vt, w.vth, BH, T, Tp, d) && map_tr(&maps.vt_lo, w.vtl, BH, T, Tp, d);
  } else {
    ok = ok && map_nat(&maps.q, Q, BH, T, d, 128) && map_nat(&maps.k, K, BH, T, d, 128);
    ok = ok && map_tr(&maps.vt, w.vth, BH, T, Tp, d);
  }
  if (!ok) return KINT_ERR_LAUNCH;
  Params ps = p;
  const int smem = plan_stats(ps);
  // test hook of the bounded waits: consume one pending request
  int pending = g_expire_waits.load();
  while (pending > 0 && !g_expire_waits.compare_exchange_weak(pending, pending - 1)) {
  }
  ps.expire_wait = pending > 0 ? 1 : 0;
  return launch_rc(traced("k_fwd_stats", s, [&] { return launch_fwd_stats(maps, ps, smem, s, sched_for(SCHED_STATS, ps)); }));
}

int check_stats(const kint_rowstats* st, bool prob) {
  if (!st || !st->row_max || !st->row_min || !st->arg_max || !st->arg_min || !st->n_max || !st->n_min || !st->W)
    return KINT_ERR_ARG;
  if (prob && (!st->W_lerp || !st->O_lerp)) return KINT_ERR_ARG;
  const void* ptrs[] = {st->row_max, st->row_min, st->arg_max, st->arg_min, st->n_max, st->n_min, st->W};
  for (const void* q : ptrs)
    if (!aligned16(q)) return KINT_ERR_ALIGN;
  if (prob && (!aligned16(st->W_lerp) || !aligned16(st->O_lerp))) return KINT_ERR_ALIGN;
  if ((st->c_M && !aligned16(st->c_M)) || (st->c_m && !aligned16(st->c_m))) return KINT_ERR_ALIGN;
  if ((st->dS_sum && !aligned16(st->dS_sum)) || (st->dS_abs && !aligned16(st->dS_abs))) return KINT_ERR_ALIGN;
  return KINT_OK;
}

// Output maps of pass 2 (O, and O_lerp when the stats carry it) for its TMA stores.
bool map_fwd_outputs(Maps& maps, const Params& p) {
  bool ok = map_nat(&maps.out, p.Out, p.BH, p.T, p.d, 64);
  if (p.O_lerp) ok = ok && map_nat(&maps.out_lerp, p.O_lerp, p.BH, p.T, p.d, 64);
  return ok;
}

void set_stats(Params& p, const kint_rowstats* st) {
  p.row_max = st->row_max; p.row_min = st->row_min;
  p.arg_max = st->arg_max; p.arg_min = st->arg_min;
  p.n_max = st->n_max; p.n_min = st->n_min;
  p.W = st->W; p.W_lerp = st->W_lerp; p.O_lerp = st->O_lerp;
  p.cM_out = st->c_M; p.cm_out = st->c_m;
  p.dsum_out = st->dS_sum; p.dabs_out = st->dS_abs;
}

bool is_prob(const Common& c) {
  return c.calib != KINT_CALIB_SOFTMAX && c.calib != KINT_CALIB_EXP_FP8 && c.calib != KINT_CALIB_EXP_BF16 &&
         c.recon == KINT_RECON_NEAREST && c.ste == KINT_STE_PROB;
}

// The forward's launches once the arguments are checked and the scratch memory is known
// (the caller's workspace, or the library's fixed array): operand prep and pass 1, then
// pass 2 (and, for 3xTF32 Prob-STE, its second launch for O_lerp and W_lerp).
int forward_launches(const float* Q, const float* K, const float* V, float* O, const kint_rowstats* st,
                     const Common& c, unsigned* status, void* scratch, cudaStream_t s) {
  const bool prob = is_prob(c);
  Params p = base_params(c, status);
  set_stats(p, st);
  p.Q = Q; p.K = K; p.V = V; p.Out = O;
  const Workspace w = plan_workspace(static_cast<char*>(scratch), p.BH, c.T, c.d, p.x3 != 0, false);
  Maps maps;
  int rc = forward_prologue(Q, K, V, p, w, maps, s);
  if (rc) return rc;
  if (!map_fwd_outputs(maps, p)) return KINT_ERR_LAUNCH;
  Params pm = p;
  pm.pv_sel = (prob && !p.x3) ? PV_MAIN_LERP : PV_MAIN;
  const int smem = plan_main(pm, pm.pv_sel);
  if (smem < 0 || smem > kSmemLimit) return KINT_ERR_UNSUPPORTED;
  if ((rc = launch_rc(traced("k_fwd_main", s, [&] { return launch_fwd_main(maps, pm, smem, s, sched_for(SCHED_MAIN, pm)); })))) return rc;
  if (prob && p.x3) {
    Params pl = p;
    pl.pv_sel = PV_LERP;
    const int smem2 = plan_main(pl, PV_LERP);
    if (smem2 < 0) return KINT_ERR_UNSUPPORTED;
    if ((rc = launch_rc(traced("k_fwd_main", s, [&] { return launch_fwd_main(maps, pl, smem2, s, sched_for(SCHED_MAIN, pl)); })))) return rc;
  }
  return KINT_OK;
}

}  // namespace
}  // namespace kint

using namespace kint;

extern "C" {

size_t kint_attn_workspace_bytes(int B, int H, int T, int d, kint_prec prec, int is_bwd) {
  if (B < 1 || H < 1 || T < 1 || (d != 64 && d != 128)) return 0;
  if ((long long)B * H * T > (1ll << 31) - 1) return 0;
  return plan_workspace(nullptr, B * H, T, d, prec == KINT_PREC_3XTF32, is_bwd != 0).bytes;
}

int kint_attn_fwd(const float* Q, const float* K, const float* V, float* O, const kint_rowstats* st, int B, int H,
                  int T, int d, int Kint, kint_calib calib, float tau, kint_recon recon, kint_ste ste,
                  kint_grad grad, int causal, kint_prec prec, void* workspace, size_t workspace_bytes,
                  void* stream) {
  const Common c{B, H, T, d, Kint, (int)calib, (int)recon, (int)ste, (int)grad, (int)prec, tau};
  int rc = validate(c, causal);
  if (rc) return rc;
  if (!Q || !K || !V || !O) return KINT_ERR_ARG;
  const bool prob = is_prob(c);
  if ((rc = check_stats(st, prob))) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O)) return KINT_ERR_ALIGN;
  const size_t need = kint_attn_workspace_bytes(B, H, T, d, prec, 0);
  if (!workspace || workspace_bytes < need) return KINT_ERR_WORKSPACE;
  if (!aligned16(workspace)) return KINT_ERR_ALIGN;
  unsigned* status = nullptr;
  if ((rc = device_setup(&status))) return rc;
  return forward_launches(Q, K, V, O, st, c, status, workspace, static_cast<cudaStream_t>(stream));
}

int kint_attn_bwd(const float* Q, const float* K, const float* V, const float* O, const float* dO,
                  const kint_rowstats* st, float* dQ, float* dK, float* dV, int B, int H, int T, int d, int Kint,
                  kint_calib calib, float tau, kint_recon recon, kint_ste ste, kint_grad grad, int causal,
                  kint_prec prec, void* workspace, size_t workspace_bytes, void* stream) {
  const Common c{B, H, T, d, Kint, (int)calib, (int)recon, (int)ste, (int)grad, (int)prec, tau};
  int rc = validate(c, causal);
  if (rc) return rc;
  if (!Q || !K || !V || !O || !dO || !dQ || !dK || !dV) return KINT_ERR_ARG;
  const bool prob = is_prob(c);
  if ((rc = check_stats(st, prob))) return rc;
  const void* ptrs[] = {Q, K, V, O, dO, dQ, dK, dV};
  for (const void* q : ptrs)
    if (!aligned16(q)) return KINT_ERR_ALIGN;
  const size_t need = kint_attn_workspace_bytes(B, H, T, d, prec, 1);
  if (!workspace || workspace_bytes < need) return KINT_ERR_WORKSPACE;
  if (!aligned16(workspace)) return KINT_ERR_ALIGN;
  unsigned* status = nullptr;
  if ((rc = device_setup(&status))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  Params p = base_params(c, status);
  set_stats(p, st);
  p.Q = Q; p.K = K; p.V = V; p.O = O; p.dO = dO;
  p.Ostar = prob ? st->O_lerp : O;
  p.dQ = dQ; p.dK = dK; p.dV = dV;
  const int BH = p.BH, Tp = round_up(T, 32);
  const Workspace w = plan_workspace(static_cast<char*>(workspace), BH, T, d, p.x3 != 0, true);
  p.rec = w.rec; p.rtab = w.rtab; p.tie_acc = w.tie;
  p.Kp = (p.Kint + 1) & ~1;
  p.tileflags = w.tileflags;
  p.gbar = w.gbar;
  p.nqt = (T + 63) / 64;
  if (cudaMemsetAsync(p.tileflags, 0, ((size_t)BH * p.nqt + 3) * 4, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  // the optional per-row dS sums are accumulated by the dK/dV pass
  if (p.dsum_out && cudaMemsetAsync(p.dsum_out, 0, (size_t)BH * T * 4, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  if (p.dabs_out && cudaMemsetAsync(p.dabs_out, 0, (size_t)BH * T * 4, s) != cudaSuccess) return KINT_ERR_LAUNCH;

  // Single-pass backward: TF32 at d = 64 on the FWM grids and the exponentials, without the
  // P1 projection and the row-sum side outputs (those stay on the two-pass kernels).  Tied
  // maxima are found during the pass and listed (one entry per tied key) for k_bwd_ext; when
  // the rows hold more ties than the list has room for (one per row of the call), which the
  // dO prep job finds out, the whole call runs the two-pass kernels instead: both sets are
  // launched, gated on that flag.
  const bool single = g_bwd_path == 0 && !p.x3 && d == 64 && c.calib != KINT_CALIB_MINMAX &&
                      c.grad != KINT_GRAD_DETACH_PROJ && !p.dsum_out && !p.dabs_out;

  // Operand copies: K-major transposes (and 3xTF32 splits); for the single pass, the dO job
  // also writes its row records and zeroes dQ and the row sums.
  PrepList pl;
  if (p.x3) {
    pl.add(Q, w.qh, w.ql, w.qth, w.qtl);
    pl.add(K, w.kh, w.kl, w.kth, w.ktl);
    pl.add(V, w.vh, w.vl, nullptr, nullptr);
    pl.add(dO, w.doh, w.dol, w.doth, w.dotl, p.Ostar, w.gbar);
  } else {
    pl.add(Q, nullptr, nullptr, w.qth, nullptr);
    // the single pass forms its K^T tiles from the K rows it holds in TMEM (k_bwd_ext writes K^T
    // for the two-pass kernels if they run instead)
    if (!single) pl.add(K, nullptr, nullptr, w.kth, nullptr);
    pl.add(dO, nullptr, nullptr, w.doth, nullptr, p.Ostar, w.gbar);
  }
  if (single) {
    RecJob& R = pl.jobs.rec;
    R.frec = reinterpret_cast<float4*>(w.frec);
    R.rsum = w.rsum;
    R.dQ = dQ;
    R.cM_out = p.cM_out;
    R.cm_out = p.cm_out;
    R.row_max = st->row_max;
    R.W = st->W;
    R.Ws = prob ? st->W_lerp : st->W;
    R.n_max = st->n_max;
    R.tileflags = w.tileflags;
    R.tie_total = w.tie_total;
    R.tie_any = w.tie_any;
    R.nqt = p.nqt;
    R.tie_cap = BH * T;
    const bool fwm = c.calib == KINT_CALIB_FWM || c.calib == KINT_CALIB_FWM_RESOLVED;
    R.c0_kind = (c.calib == KINT_CALIB_SOFTMAX || c.calib == KINT_CALIB_EXP_FP8) ? 0 : (fwm ? 1 : 2);
    R.half = fwm && c.recon == KINT_RECON_NEAREST;
    R.softmax = c.calib == KINT_CALIB_SOFTMAX;
    R.tau = p.tau;
    R.inv_h = p.fwm_inv_h;
  }
  if (prep(pl, BH, T, Tp, d, p.x3 != 0, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  Maps maps;
  std::memset(&maps, 0, sizeof(maps));
  bool ok = true;
  if (p.x3) {
    ok = ok && map_nat(&maps.k, w.kh, BH, T, d, 64) && map_nat(&maps.k_lo, w.kl, BH, T, d, 64);
    ok = ok && map_nat(&maps.v, w.vh, BH, T, d, 64) && map_nat(&maps.v_lo, w.vl, BH, T, d, 64);
    ok = ok && map_nat(&maps.q, w.qh, BH, T, d, 64) && map_nat(&maps.q_lo, w.ql, BH, T, d, 64);
    ok = ok && map_nat(&maps.dout, w.doh, BH, T, d, 64) && map_nat(&maps.dout_lo, w.dol, BH, T, d, 64);
    ok = ok && map_tr(&maps.kt, w.kth, BH, T, Tp, d) && map_tr(&maps.kt_lo, w.ktl, BH, T, Tp, d);
    ok = ok && map_tr(&maps.qt, w.qth, BH, T, Tp, d) && map_tr(&maps.qt_lo, w.qtl, BH, T, Tp, d);
    ok = ok && map_tr(&maps.dot, w.doth, BH, T, Tp, d) && map_tr(&maps.dot_lo, w.dotl, BH, T, Tp, d);
  } else {
    ok = ok && map_nat(&maps.k, K, BH, T, d, 64) && map_nat(&maps.v, V, BH, T, d, 64);
    ok = ok && map_nat(&maps.q, Q, BH, T, d, 64) && map_nat(&maps.dout, dO, BH, T, d, 64);
    ok = ok && map_tr(&maps.kt, w.kth, BH, T, Tp, d) && map_tr(&maps.qt, w.qth, BH, T, Tp, d);
    ok = ok && map_tr(&maps.dot, w.doth, BH, T, Tp, d);
  }
  ok = ok && map_nat(&maps.dq, dQ, BH, T, d, 64) && map_nat(&maps.dk, dK, BH, T, d, 64) &&
       map_nat(&maps.dv, dV, BH, T, d, 64);
  if (!ok) return KINT_ERR_LAUNCH;

  if (single) {
    Params pf = p;
    pf.frec = w.frec;
    pf.rsum = w.rsum;
    pf.tie_any = w.tie_any;
    pf.tie_count = w.tie_count;
    pf.tie_total = w.tie_total;
    pf.tie_list = w.tie_list;
    pf.tie_cap = BH * T;
    pf.kt_out = w.kth;
    const bool ext = c.calib != KINT_CALIB_SOFTMAX && c.grad != KINT_GRAD_DETACH;
    if (!map_nat_sw64(&maps.dq16, dQ, BH, T, d, 16, 16) || !map_nat_sw64(&maps.dk32, dK, BH, T, d, 16, 32) ||
        !map_nat_sw64(&maps.dv32, dV, BH, T, d, 16, 32))
      return KINT_ERR_LAUNCH;
    const int smem_f = plan_fused(pf);
    if (smem_f < 0) return KINT_ERR_UNSUPPORTED;
    if (ext) {
      pf.gate = w.tie_any;
      pf.gate_on = 0;
    }
    if ((rc = launch_rc(traced("k_bwd_fused", s, [&] { return launch_bwd_fused(maps, pf, smem_f, s, sched_for(SCHED_FUSED, pf)); })))) return rc;
    if (!ext) return KINT_OK;
    if ((rc = launch_rc(traced("k_bwd_ext", s, [&] { return launch_bwd_ext(pf, s); })))) return rc;
    p.gate = w.tie_any;
    p.gate_on = 1;
  }

  // P1 projection: key prefix sums into the tie-sum buffer (unused by the detached modes)
  if (c.grad == KINT_GRAD_DETACH_PROJ && c.calib != KINT_CALIB_SOFTMAX)
    if ((rc = launch_rc(traced("k_kcum", s, [&] { return launch_kcum(K, w.tie, BH, T, d, s); })))) return rc;
  Params pq = p;
  const int smem_dq = plan_dq(pq);
  if (smem_dq < 0 || smem_dq > kSmemLimit) return KINT_ERR_UNSUPPORTED;
  if ((rc = launch_rc(traced("k_bwd_dq", s, [&] { return launch_bwd_dq(maps, pq, smem_dq, s); })))) return rc;

  Params pk = p;
  int smem_kv = plan_dkdv(pk, DKV_BOTH);
  if (!p.x3 && smem_kv > 0) return launch_rc(traced("k_bwd_dkdv", s, [&] { return launch_bwd_dkdv(maps, pk, smem_kv, s); }));
  // one product per launch (3xTF32 hi/lo operands, or d = 128): dV, then dK
  smem_kv = plan_dkdv(pk, DKV_DV);
  if (smem_kv < 0) return KINT_ERR_UNSUPPORTED;
  if ((rc = launch_rc(traced("k_bwd_dkdv", s, [&] { return launch_bwd_dkdv(maps, pk, smem_kv, s); })))) return rc;
  Params pk2 = p;
  const int smem_kv2 = plan_dkdv(pk2, DKV_DK);
  if (smem_kv2 < 0) return KINT_ERR_UNSUPPORTED;
  return launch_rc(traced("k_bwd_dkdv", s, [&] { return launch_bwd_dkdv(maps, pk2, smem_kv2, s); }));
}

int kint_attn_debug_bins(const float* Q, const float* K, const float* V, const kint_rowstats* st, uint8_t* bins,
                         uint8_t* ivals, int B, int H, int T, int d, int Kint, kint_calib calib, float tau,
                         kint_recon recon, kint_ste ste, int causal, kint_prec prec, void* workspace,
                         size_t workspace_bytes, void* stream) {
  const Common c{B, H, T, d, Kint, (int)calib, (int)recon, (int)ste, 0, (int)prec, tau};
  int rc = validate(c, causal);
  if (rc) return rc;
  if (!Q || !K || !V || (!bins && !ivals)) return KINT_ERR_ARG;
  if ((rc = check_stats(st, false))) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V)) return KINT_ERR_ALIGN;
  if ((bins && !aligned16(bins)) || (ivals && !aligned16(ivals))) return KINT_ERR_ALIGN;
  const size_t need = kint_attn_workspace_bytes(B, H, T, d, prec, 0);
  if (!workspace || workspace_bytes < need) return KINT_ERR_WORKSPACE;
  if (!aligned16(workspace)) return KINT_ERR_ALIGN;
  unsigned* status = nullptr;
  if ((rc = device_setup(&status))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  Params p = base_params(c, status);
  // the decisions need only the extrema; W / W_lerp / O are not written in debug mode
  set_stats(p, st);
  p.Q = Q; p.K = K; p.V = V;
  const size_t n = (size_t)B * H * T * T;
  if (bins && cudaMemsetAsync(bins, 255, n, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  if (ivals && cudaMemsetAsync(ivals, 255, n, s) != cudaSuccess) return KINT_ERR_LAUNCH;
  const Workspace w = plan_workspace(static_cast<char*>(workspace), p.BH, T, d, p.x3 != 0, false);
  Maps maps;
  if ((rc = forward_prologue(Q, K, V, p, w, maps, s))) return rc;
  Params pm = p;
  pm.pv_sel = PV_MAIN;
  const int smem = plan_main(pm, PV_MAIN);
  if (smem < 0 || smem > kSmemLimit) return KINT_ERR_UNSUPPORTED;
  pm.debug = 1;
  pm.bins = bins;
  pm.ivals = ivals;
  return launch_rc(traced("k_fwd_main", s, [&] { return launch_fwd_main(maps, pm, smem, s, sched_for(SCHED_MAIN, pm)); }));
}

int kint_attn_probe(const float* Q, const float* K, const kint_rowstats* st, float* probe, int B, int H, int T,
                    int d, int Kint, kint_calib calib, float tau, kint_recon recon, int causal, kint_prec prec,
                    void* workspace, size_t workspace_bytes, void* stream) {
  const Common c{B, H, T, d, Kint, (int)calib, (int)recon, 0, 0, (int)prec, tau};
  int rc = validate(c, causal);
  if (rc) return rc;
  if (calib != KINT_CALIB_MINMAX && calib != KINT_CALIB_FWM) return KINT_ERR_UNSUPPORTED;
  if (!Q || !K || !probe) return KINT_ERR_ARG;
  if ((rc = check_stats(st, false))) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(probe)) return KINT_ERR_ALIGN;
  const size_t need = kint_attn_workspace_bytes(B, H, T, d, prec, 0);
  if (!workspace || workspace_bytes < need) return KINT_ERR_WORKSPACE;
  if (!aligned16(workspace)) return KINT_ERR_ALIGN;
  unsigned* status = nullptr;
  if ((rc = device_setup(&status))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  Params p = base_params(c, status);
  set_stats(p, st);
  p.Q = Q; p.K = K;
  p.probe = probe;
  const Workspace w = plan_workspace(static_cast<char*>(workspace), p.BH, T, d, p.x3 != 0, false);
  Maps maps;
  std::memset(&maps, 0, sizeof(maps));
  bool ok = true;
  if (p.x3) {
    PrepList pl;
    pl.add(Q, w.qh, w.ql, nullptr, nullptr);
    pl.add(K, w.kh, w.kl, nullptr, nullptr);
    if (prep(pl, p.BH, T, round_up(T, 32), d, true, s) != cudaSuccess) return KINT_ERR_LAUNCH;
    ok = map_nat(&maps.q, w.qh, p.BH, T, d, 128) && map_nat(&maps.q_lo, w.ql, p.BH, T, d, 128) &&
         map_nat(&maps.k, w.kh, p.BH, T, d, 128) && map_nat(&maps.k_lo, w.kl, p.BH, T, d, 128);
  } else {
    ok = map_nat(&maps.q, Q, p.BH, T, d, 128) && map_nat(&maps.k, K, p.BH, T, d, 128);
  }
  if (!ok) return KINT_ERR_LAUNCH;
  // pass 1 (row extrema), then the probe's two sweeps
  Params ps = p;
  const int smem_s = plan_stats(ps);
  if ((rc = launch_rc(traced("k_fwd_stats", s, [&] { return launch_fwd_stats(maps, ps, smem_s, s, sched_for(SCHED_STATS, ps)); })))) return rc;
  Params pp = p;
  const int smem_p = plan_probe(pp);
  if (smem_p < 0 || smem_p > kSmemLimit) return KINT_ERR_UNSUPPORTED;
  return launch_rc(traced("k_fwd_probe", s, [&] { return launch_fwd_probe(maps, pp, smem_p, s); }));
}

int kint_get_status(void* stream, unsigned* detail) {
  unsigned* status = nullptr;
  int rc = device_setup(&status);
  if (rc) return rc;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return KINT_ERR_LAUNCH;
  unsigned v = 0;
  if (cudaMemcpy(&v, status, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return KINT_ERR_LAUNCH;
  if (v && cudaMemset(status, 0, sizeof(unsigned)) != cudaSuccess) return KINT_ERR_LAUNCH;
  if (detail) *detail = v;
  return v ? KINT_ERR_DEVICE : KINT_OK;
}

const char* kint_strerror(int code) {
  switch (code) {
    case KINT_OK: return "ok";
    case KINT_ERR_ARG: return "invalid argument";
    case KINT_ERR_UNSUPPORTED:
      return "unsupported size or mode (d must be 64 or 128; 3xTF32 needs d = 64; MinMax with K > 32 needs TF32 "
             "at d = 64)";
    case KINT_ERR_ALIGN: return "device pointer not 16-byte aligned";
    case KINT_ERR_WORKSPACE: return "workspace missing or too small";
    case KINT_ERR_LAUNCH: return "CUDA launch or tensor-map encoding failed";
    case KINT_ERR_DEVICE: return "a kernel flagged a device-side fault (bounded wait timed out)";
    case KINT_ERR_NO_DEVICE: return "no sm_103 device is current, or the driver lacks tensor maps";
    case KINT_ERR_SCRATCH_LIMIT: return "problem too large for the library's fixed scratch (kint_attn_fwd_noalloc)";
    default: return "unknown error code";
  }
}

void kint_set_wait_timeout_ns(unsigned long long ns) { g_wait_ns = ns < 1000ull ? 1000ull : ns; }

void kint_test_expire_next_wait(int count) { g_expire_waits.store(count > 0 ? count : 0); }

void kint_set_backward_path(int path) { g_bwd_path = path == 1 ? 1 : 0; }

void kint_set_launch_callback(kint_launch_cb cb, void* user) {
  g_cb_user = user;
  g_cb = cb;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Forward with library-owned scratch, for callers that cannot allocate device
// memory or pass a workspace (see kint_attn_fwd_noalloc in kint_attn.h).  The
// scratch is this fixed device array; host code never hands its symbol to a
// kernel, only the device address looked up per device below.
// ---------------------------------------------------------------------------
namespace kint {
namespace {
static __device__ __align__(256) unsigned char g_noalloc_scratch[KINT_NOALLOC_SCRATCH_BYTES];
void* g_noalloc_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device, looked up once per
// device with that device current.
int noalloc_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KINT_ERR_NO_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_noalloc_ptr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return KINT_ERR_NO_DEVICE;
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return KINT_OK;
}
}  // namespace
}  // namespace kint

extern "C" {

int kint_attn_fwd_noalloc(const float* Q, const float* K, const float* V, float* O, const kint_rowstats* st, int B,
                          int H, int T, int d, int Kint, kint_calib calib, float tau, kint_recon recon,
                          kint_ste ste, kint_grad grad, int causal, kint_prec prec, void* stream) {
  const Common c{B, H, T, d, Kint, (int)calib, (int)recon, (int)ste, (int)grad, (int)prec, tau};
  int rc = validate(c, causal);
  if (rc) return rc;
  if (!Q || !K || !V || !O) return KINT_ERR_ARG;
  const bool prob = is_prob(c);
  if ((rc = check_stats(st, prob))) return rc;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O)) return KINT_ERR_ALIGN;
  const size_t need = kint_attn_workspace_bytes(B, H, T, d, prec, 0);
  if (need == 0) return KINT_ERR_UNSUPPORTED;
  if (need > (size_t)KINT_NOALLOC_SCRATCH_BYTES) return KINT_ERR_SCRATCH_LIMIT;
  unsigned* status = nullptr;
  if ((rc = device_setup(&status))) return rc;
  void* scratch = nullptr;
  if ((rc = noalloc_scratch(&scratch))) return rc;
  return forward_launches(Q, K, V, O, st, c, status, scratch, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
