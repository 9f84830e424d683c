"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs, element by element, for every variant of the operator."""
import numpy as np
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity

pytestmark = pytest.mark.gpu

MM, FW, SM, FR = kint.CALIB_MINMAX, kint.CALIB_FWM, kint.CALIB_SOFTMAX, kint.CALIB_FWM_RESOLVED
E8, EB = kint.CALIB_EXP_FP8, kint.CALIB_EXP_BF16
LE, NE = kint.RECON_LERP, kint.RECON_NEAREST
WE, PR = kint.STE_WEIGHT, kint.STE_PROB
FU, DE = kint.GRAD_FULL, kint.GRAD_DETACH
MX, MN = kint.GRAD_MAX_ONLY, kint.GRAD_MIN_ONLY
PJ = kint.GRAD_DETACH_PROJ
X3, TF = kint.PREC_3XTF32, kint.PREC_TF32

COMBOS = [(c, r, s, g) for c in (MM, FW) for r in (LE, NE) for s in (WE, PR) for g in (FU, DE)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    kint.load()


def _cfg(c, r, s, g, K=4, tau=8.0):
    return kint.Config(Kint=K, calib=c, tau=tau, recon=r, ste=s, grad=g)


def test_tiny_config_3xtf32_bit_exact_decisions():
    """B=1, H=2, T=128, d=64, K=4, MinMax, LERP, Weight-STE, full gradient, seed 0."""
    Q, K, V, dO = make_qkvdo(1, 2, 128, 64, seed=0)
    rep = parity.check(Q, K, V, dO, _cfg(MM, LE, WE, FU), X3)
    assert rep["bins_flips"] == 0 and rep["ivals_flips"] == 0
    assert rep["arg_max_flips"] == 0 and rep["arg_min_flips"] == 0


@pytest.mark.parametrize("c,r,s,g", COMBOS)
@pytest.mark.parametrize("Kint", [4, 8, 16])
def test_all_variants_3xtf32_ragged(c, r, s, g, Kint):
    """Every combination at K in {4, 8, 16}; T = 300 spans three 128-row tiles and a ragged tail."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=2)
    parity.check(Q, K, V, dO, _cfg(c, r, s, g, Kint), X3)


@pytest.mark.parametrize("c,r,s,g", COMBOS)
def test_all_variants_tf32(c, r, s, g):
    Q, K, V, dO = make_qkvdo(2, 2, 200, 64, seed=2)
    parity.check(Q, K, V, dO, _cfg(c, r, s, g, 4), TF)


@pytest.mark.parametrize("g", [MX, MN])
@pytest.mark.parametrize("c,r,s", [(MM, LE, WE), (MM, NE, PR), (MM, NE, WE), (FW, NE, WE), (FW, LE, PR)])
@pytest.mark.parametrize("prec", [X3, TF])
def test_single_channel_modes(c, r, s, g, prec):
    """max_only / min_only backward (one extremum term of Eq. full kept); T = 300 is ragged."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=11)
    parity.check(Q, K, V, dO, _cfg(c, r, s, g, 8), prec)


@pytest.mark.parametrize("c,r,s", [(MM, LE, WE), (MM, NE, PR), (FW, NE, WE), (FW, LE, PR)])
@pytest.mark.parametrize("prec", [X3, TF])
def test_zero_sum_projection(c, r, s, prec):
    """P1 control: detached dS minus its causal-row mean (tau = 3 puts FWM keys in the tail);
    T = 300 spans three query blocks and a ragged tail."""
    Q, K, V, dO = make_qkvdo(2, 2, 300, 64, seed=13)
    parity.check(Q, K, V, dO, _cfg(c, r, s, PJ, 8, tau=3.0), prec)


@pytest.mark.parametrize("c,r,s", [(MM, LE, WE), (MM, NE, PR), (FW, NE, PR), (FW, LE, WE)])
def test_full_length_rows_3xtf32(c, r, s):
    """T = 1024 (the GPT-2 context): dK and dV of the first keys sum over every query row, the
    longest accumulation chains of the backward, and must still meet the 3xTF32 tolerance."""
    Q, K, V, dO = make_qkvdo(1, 1, 1024, 64, seed=15)
    parity.check(Q, K, V, dO, _cfg(c, r, s, FU), X3)


@pytest.mark.parametrize("T", [1, 2, 65, 1024])
def test_zero_sum_projection_lengths(T):
    """Short rows (T = 1: the one causal key of row 0 keeps 0) and a full-length head."""
    Q, K, V, dO = make_qkvdo(1, 1, T, 64, seed=14)
    for cfg in (_cfg(MM, NE, WE, PJ), _cfg(FW, NE, PR, PJ)):
        parity.check(Q, K, V, dO, cfg, X3)


@pytest.mark.parametrize("r,s,g", [(r, s, g) for r in (LE, NE) for s in (WE, PR) for g in (FU, DE)] + [(NE, PR, PJ)])
@pytest.mark.parametrize("prec", [X3, TF])
def test_resolved_tail_policy(r, s, g, prec):
    """FWM's grid continued below -tau (App. "Tail policy"): tau = 3 at these score scales puts
    most keys below the window, on negative grid indices; T = 300 is ragged."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=16)
    parity.check(Q, K, V, dO, _cfg(FR, r, s, g, 4, tau=3.0), prec)


@pytest.mark.parametrize("Kint,tau", [(1, 1.0), (16, 8.0), (64, 4.0)])
def test_resolved_tail_policy_grids(Kint, tau):
    """Coarse and fine steps: K = 1 with a 1-nat window, K = 64 (h = 1/16) far below the window."""
    Q, K, V, dO = make_qkvdo(1, 2, 200, 64, seed=17)
    parity.check(Q, K, V, dO, _cfg(FR, NE, PR, FU, Kint, tau=tau), X3 if Kint <= 32 else TF)


@pytest.mark.parametrize("g", [FU, DE, PJ])
@pytest.mark.parametrize("prec", [X3, TF])
def test_fp8_exponential_baseline(g, prec):
    """E4M3(e^z) forward, e^z backward, row max on the gradient path; the E4M3 byte of every weight
    is a decision (compared exactly outside the guard band).  T = 300 is ragged."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=18)
    rep = parity.check(Q, K, V, dO, _cfg(E8, LE, WE, g), prec)
    if prec == X3:  # fp32-accurate scores: a rounding decision flips only within a few ulps
        assert rep["bins_flips"] <= 0.001 * 300 * 301


def test_fp8_exponential_value_set():
    """Scores spread so that every E4M3 level below 1 and the underflow to zero occur: the GPU's
    codes take exactly the format's 56 nonzero values and 0."""
    Q, K, V, dO = make_qkvdo(1, 4, 256, 64, seed=19)
    g = parity.run_gpu(Q * 1.5, K, V, dO, _cfg(E8, LE, WE, FU), X3, want_bwd=False)
    codes = g["bins"][g["bins"] != 255]
    assert codes.max() == 0x38 and codes.min() == 0
    assert len(set(codes[codes > 0].tolist())) == 56


@pytest.mark.parametrize("prec", [X3, TF])
def test_softmax_comparator(prec):
    Q, K, V, dO = make_qkvdo(1, 2, 260, 64, seed=5)
    parity.check(Q, K, V, dO, _cfg(SM, LE, WE, FU), prec)


@pytest.mark.parametrize("c,r,s", [(MM, LE, WE), (FW, NE, WE), (FW, NE, PR), (MM, NE, PR)])
def test_head_dim_128_tf32(c, r, s):
    Q, K, V, dO = make_qkvdo(1, 2, 200, 128, seed=6)
    parity.check(Q, K, V, dO, _cfg(c, r, s, FU, 4), TF)


@pytest.mark.parametrize("T", [1, 2, 63, 64, 65, 127, 129, 257])
def test_lengths(T):
    Q, K, V, dO = make_qkvdo(1, 1, T, 64, seed=7)
    for cfg in (_cfg(MM, NE, WE, FU), _cfg(FW, NE, PR, FU)):
        parity.check(Q, K, V, dO, cfg, X3)


def test_degenerate_and_tied_rows():
    """Q = 0 makes every MinMax row degenerate and every FWM row all-equal; duplicate keys tie."""
    Q, K, V, dO = make_qkvdo(1, 1, 140, 64, seed=8)
    Qz = np.zeros_like(Q)
    for cfg in (_cfg(MM, LE, WE, FU), _cfg(MM, NE, PR, FU), _cfg(FW, NE, WE, FU), _cfg(FW, LE, PR, FU)):
        parity.check(Qz, K, V, dO, cfg, X3)
    Kd = K.copy()
    Kd[0, 0, 5] = Kd[0, 0, 2]
    Kd[0, 0, 130] = Kd[0, 0, 2]
    Kd[0, 0, 77] = Kd[0, 0, 40]
    for cfg in (_cfg(MM, LE, WE, FU), _cfg(MM, NE, WE, FU), _cfg(FW, NE, PR, FU)):
        parity.check(Q * 3, Kd, V, dO, cfg, X3)


@pytest.mark.parametrize("calib", [FW, E8])
def test_single_pass_tied_maxima(calib):
    """TF32 single-pass backward with a few rows whose maximum is tied (three identical
    keys that those rows point at): the pass lists the tied keys and splits c_M over them
    (Eq. full).  Q = 0 makes every row all-equal, more ties than the list holds: the call
    runs the two-pass kernels instead.  Both against the oracle."""
    Q, K, V, dO = make_qkvdo(1, 2, 140, 64, seed=31)
    Kd = K.copy()
    for h in range(2):
        Kd[0, h, 5] = Kd[0, h, 2]
        Kd[0, h, 130] = Kd[0, h, 2]
        u = Kd[0, h, 2] / np.linalg.norm(Kd[0, h, 2])
        for i in (10, 50, 100, 135):
            Q[0, h, i] = (2.5 * 8.0 * u).astype(np.float32)
    cfg = _cfg(calib, NE, PR, FU)
    parity.check(Q, Kd, V, dO, cfg, TF)
    parity.check(np.zeros_like(Q), K, V, dO, cfg, TF)


def test_fwm_far_tail():
    """Scores spread far beyond tau: every key but the maximum falls in the zero tail."""
    Q, K, V, dO = make_qkvdo(1, 1, 150, 64, seed=9)
    for cfg in (_cfg(FW, NE, WE, FU, tau=2.0), _cfg(FW, LE, PR, FU, tau=2.0)):
        parity.check(Q * 20, K, V, dO, cfg, X3)


def test_extreme_K():
    """K = 1 and the largest K each configuration supports (MinMax K = 64 only in TF32 at d = 64)."""
    Q, K, V, dO = make_qkvdo(1, 2, 200, 64, seed=10)
    parity.check(Q, K, V, dO, _cfg(MM, NE, WE, FU, 1), X3)
    parity.check(Q, K, V, dO, _cfg(FW, LE, PR, FU, 1), X3)
    parity.check(Q, K, V, dO, _cfg(MM, NE, WE, FU, 32), X3)
    parity.check(Q, K, V, dO, _cfg(FW, LE, PR, FU, 64), X3)
    parity.check(Q, K, V, dO, _cfg(MM, LE, PR, FU, 64), TF)
    parity.check(Q, K, V, dO, _cfg(FW, NE, PR, DE, 64), TF)


def test_value_ones_rows_sum_to_one():
    """V = 1 gives O = 1 when the rows of P sum to one (App. A, Normalization).  O is the tensor-core sum
    of w_j over the fp32 sum W of the same n <= T weights, so |O - 1| is bounded by the two fp32
    summation errors, about 2 n 2^-24."""
    T = 300
    Q, K, _, dO = make_qkvdo(1, 2, T, 64, seed=11)
    V = np.ones_like(Q)
    for cfg in (_cfg(MM, NE, WE, FU), _cfg(FW, NE, PR, FU), _cfg(SM, LE, WE, FU)):
        g = parity.run_gpu(Q, K, V, dO, cfg, X3, want_bins=False, want_bwd=False)
        assert np.max(np.abs(g["O"] - 1.0)) <= 2 * T * 2.0 ** -24


@pytest.mark.parametrize("c,r,s", [(FW, NE, PR), (MM, LE, WE), (SM, LE, WE)])
def test_many_items_per_cta(c, r, s):
    """More (block, head) items than SMs, so CTAs that loop over items (tile counters
    and barrier phases running on across items) are exercised; ragged T."""
    Q, K, V, dO = make_qkvdo(4, 40, 200, 64, seed=11)
    parity.check(Q, K, V, dO, _cfg(c, r, s, FU, 4), TF)


@pytest.mark.parametrize("prec", [TF, X3])
def test_exact_grid_points(prec):
    """Operands in {-1, 0, 1} make every score a multiple of 1/8, so for FWM (tau = 8, K = 4,
    h = 2) the position u = (s - M + tau) / h is exact and lands on bin edges (t = 0) and
    midpoints (t = 1/2, where Nearest takes e_{r+1}) for many keys: the passes must take
    the oracle's decisions there exactly."""
    rng = np.random.default_rng(12)
    Q = rng.integers(-1, 2, size=(1, 2, 200, 64)).astype(np.float32)
    K = rng.integers(-1, 2, size=(1, 2, 200, 64)).astype(np.float32)
    _, _, V, dO = make_qkvdo(1, 2, 200, 64, seed=12)
    cfgs = (_cfg(FW, NE, PR, FU), _cfg(FW, NE, WE, FU), _cfg(FW, LE, PR, FU), _cfg(FW, NE, PR, DE),
            _cfg(FW, NE, PR, FU, tau=2.0))  # tau = 2: h = 1/2, many keys in the tail and at u = 0
    for cfg in cfgs:
        rep = parity.check(Q, K, V, dO, cfg, prec)
        assert rep["bins_flips"] == 0 and rep["ivals_flips"] == 0
    parity.check(Q, K, V, dO, _cfg(MM, NE, WE, FU), prec)


@pytest.mark.parametrize("c,r", [(MM, LE), (MM, NE), (FW, NE), (FW, LE)])
@pytest.mark.parametrize("prec", [X3, TF])
def test_geometry_probe(c, r, prec):
    """kint_attn_probe against the oracle's probes, decision-aligned (the oracle takes the GPU's
    bins and extrema, as in the parity check); T = 300 is ragged, Q x 2 spreads the rows so that
    keys below z = -6 and FWM tail keys occur."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=20)
    Q = Q * 2.0
    cfg = _cfg(c, r, WE, FU, 4, tau=3.0)
    dev = torch.device("cuda:0")
    q, k, v = (torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in (Q, K, V))
    pr = kint.probe(q, k, cfg, prec)
    O, st = kint.forward(q, k, v, cfg, prec)
    bins, ivals = kint.debug_bins(q, k, v, st, cfg, prec)
    torch.cuda.synchronize()
    kint.check_status()
    amin = st["arg_min"].cpu().numpy() if c == MM else None
    ov = {"bins": bins.cpu().numpy(), "ivals": ivals.cpu().numpy(), "amax": st["arg_max"].cpu().numpy()}
    if amin is not None:
        ov["amin"] = amin
    f = parity.oracle.forward(Q, K, V, parity.to_oracle_cfg(cfg), probes=True, override=ov)
    tol = 2e-5 if prec == X3 else 5e-3
    # "z < -6" is a decision too: a key within the score rounding of -6 may count either way
    S = np.einsum("bhid,bhjd->bhij", Q.astype(np.float64), K.astype(np.float64)) / 8.0
    causal = np.tril(np.ones((300, 300), bool))
    z = np.where(causal, S - np.where(causal, S, -np.inf).max(-1, keepdims=True), 0.0)
    band = parity.BAND_REL[prec] * (np.abs(S).max() + 1.0)
    near = (causal & (np.abs(z + 6.0) <= band)).sum(-1) / np.arange(1, 301)
    for n, ref in zip(parity.oracle.PROBE_NAMES, f["probe"]):
        got = pr[n].cpu().numpy().astype(np.float64)
        err = np.abs(got - ref) / (1.0 + np.abs(ref))
        if n == "frac_below6":
            err = np.maximum(np.abs(got - ref) - near, 0.0)
        assert err.max() <= tol, f"{n}: {err.max():.3g}"


@pytest.mark.parametrize("g", [FU, DE, PJ])
@pytest.mark.parametrize("prec", [X3, TF])
def test_bf16_exponential_baseline(g, prec):
    """bf16(e^{bf16(z)}) forward (both roundings compared as decisions through their bfloat16 low
    bytes), bfloat16 chain-rule backward; T = 300 is ragged."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=22)
    rep = parity.check(Q, K, V, dO, _cfg(EB, LE, WE, g), prec)
    if prec == X3:
        assert rep["errors"]["dV"] <= 1e-5 and rep["errors"]["O"] <= 1e-5
