"""Pins for the fp64 oracle, against what the paper and the mathematics fix.

Each test names the passage it follows.  None of them compares the oracle with
itself: the references are brute-force scans, closed forms, textbook error
bounds of linear interpolation, finite differences, an independent PyTorch
autograd restatement (tests/witness.py), and invariants (row sums, shift
invariance, the zero-sum identity).
"""
import math

import numpy as np
import pytest

import oracle
from oracle import Config, MINMAX, FWM, SOFTMAX, FWM_RESOLVED, EXP_FP8, EXP_BF16, LERP, NEAREST, WEIGHT, PROB, \
    FULL, DETACH, MAX_ONLY, MIN_ONLY, DETACH_PROJ
from tests import witness

ALL_COMBOS = [(c, r, s, g) for c in (MINMAX, FWM) for r in (LERP, NEAREST) for s in (WEIGHT, PROB)
              for g in (FULL, DETACH)]
RES = FWM_RESOLVED
RES_COMBOS = [(RES, r, s, g) for r in (LERP, NEAREST) for s in (WEIGHT, PROB) for g in (FULL, DETACH)]


def rand_inputs(B, H, T, d, seed, scale=1.0, f64=False):
    rng = np.random.default_rng(seed)
    dt = np.float64 if f64 else np.float32
    return [(rng.standard_normal((B, H, T, d)) * (scale if i == 0 else 1.0)).astype(dt) for i in range(4)]


def eye_values(T, d):
    """V = I (T <= d): then O_i = P_i, and g_ij = dO_i[j]."""
    V = np.zeros((1, 1, T, d), np.float32)
    V[0, 0, np.arange(T), np.arange(T)] = 1.0
    return V


def lattice_qk(targets, d=16):
    """Q, K whose every row i sees the scores targets[0..i] exactly:
    Q_i = (2, 0, ...), K_j = (2 t_j, 0, ...), scale 1/sqrt(16) = 1/4."""
    T = len(targets)
    Q = np.zeros((1, 1, T, d), np.float32)
    K = np.zeros((1, 1, T, d), np.float32)
    Q[0, 0, :, 0] = 2.0
    K[0, 0, :, 0] = 2.0 * np.asarray(targets, np.float64)
    return Q, K


def scores_np(Q, K):
    d = Q.shape[-1]
    return np.einsum("bhid,bhjd->bhij", Q.astype(np.float64), K.astype(np.float64)) / math.sqrt(d)


# --- P1: rows sum to one (App. A "Normalization") ------------------------------------------------

@pytest.mark.parametrize("calib,recon,ste,grad", ALL_COMBOS + RES_COMBOS + [(SOFTMAX, LERP, WEIGHT, FULL)])
def test_rows_sum_to_one(calib, recon, ste, grad):
    Q, K, _, _ = rand_inputs(2, 2, 40, 16, 1, scale=2.0)
    V = np.ones_like(Q)
    out = oracle.forward(Q, K, V, Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad))
    assert np.max(np.abs(out["O"] - 1.0)) < 1e-13


# --- two valid keys: both sit on grid points, so every MinMax operator is softmax -----------------

@pytest.mark.parametrize("Kint", [1, 2, 4, 16])
@pytest.mark.parametrize("recon", [LERP, NEAREST])
def test_two_key_rows_equal_softmax(Kint, recon):
    T = 16
    Q, K, _, _ = rand_inputs(1, 1, T, 16, 2)
    out = oracle.forward(Q, K, eye_values(T, 16), Config(Kint=Kint, calib=MINMAX, recon=recon))
    s = scores_np(Q, K)[0, 0, 1, :2]
    ref = np.exp(s - s.max()) / np.exp(s - s.max()).sum()
    assert np.allclose(out["O"][0, 0, 1, :2], ref, rtol=0, atol=1e-15)


# --- P2: brute-force bins on score lattices (Sec. 3 "Reconstruction", App. A, Table "Edge cases") --

def brute_force_row(z, b, tail):
    """Nearest index by scanning all K+1 grid points (ties go up), LERP weight
    by scanning for an interval that contains z."""
    K = len(b) - 1
    ell, r_idx, wl, wn = [], [], [], []
    for zj, tj in zip(z, tail):
        if tj:
            ell.append(254)
            r_idx.append(254)
            wl.append(0.0)
            wn.append(0.0)
            continue
        best, best_l = math.inf, -1
        for l in range(K + 1):
            dist = abs(zj - b[l])
            if dist < best or dist == best:  # equal distance: the larger index wins
                best, best_l = dist, l
        r = max(rr for rr in range(K) if b[rr] <= zj) if zj >= b[0] else 0
        t = min(max((zj - b[r]) / (b[r + 1] - b[r]), 0.0), 1.0)
        ell.append(best_l)
        r_idx.append(r)
        wn.append(math.exp(b[best_l]))
        wl.append((1 - t) * math.exp(b[r]) + t * math.exp(b[r + 1]))
    return np.array(ell), np.array(r_idx), np.array(wl), np.array(wn)


@pytest.mark.parametrize("calib", [MINMAX, FWM])
def test_brute_force_bins_on_lattice(calib):
    rng = np.random.default_rng(3)
    Kint, T, step = 4, 16, 0.125
    for trial in range(60):
        # max key 1.0; for MinMax a min key at 1 - 2 (span 2, h = 0.5); the rest on a 1/8 lattice that
        # hits grid points, Nearest midpoints and (for FWM, tau = 2) the window edge and the tail.
        depth = 16 if calib == MINMAX else 24
        ks = rng.integers(0, depth + 1, size=T)
        ks[rng.integers(0, T)] = 0
        if calib == MINMAX:
            ks[rng.integers(0, T)] = 16
        targets = 1.0 - step * ks
        Q, K = lattice_qk(targets)
        cfg = Config(Kint=Kint, calib=calib, tau=2.0, recon=NEAREST)
        out = oracle.forward(Q, K, eye_values(T, 16), cfg, decisions=True)
        out_l = oracle.forward(Q, K, eye_values(T, 16), Config(Kint=Kint, calib=calib, tau=2.0, recon=LERP))
        z = targets - targets.max()
        if calib == MINMAX:
            b = [z.min() + r * (0 - z.min()) / Kint for r in range(Kint + 1)]
            tail = np.zeros(T, bool)
        else:
            b = [-2.0 + r * 0.5 for r in range(Kint + 1)]
            tail = z < -2.0
        ell, r_idx, wl, wn = brute_force_row(z, b, tail)
        last = T - 1
        assert np.array_equal(out["bins"][0, 0, last], ell), (trial, targets)
        assert np.array_equal(out["ivals"][0, 0, last], r_idx), (trial, targets)
        assert np.allclose(out["O"][0, 0, last, :T], wn / wn.sum(), rtol=0, atol=1e-15)
        assert np.allclose(out_l["O"][0, 0, last, :T], wl / wl.sum(), rtol=0, atol=1e-15)


def test_midpoint_rounds_up_and_window_edge_is_inside():
    # MinMax K=4 over [-1, 1]: h = 0.5, grid z in {-2, -1.5, -1, -0.5, 0}; z = -0.25 sits exactly
    # between b_3 = -0.5 and b_4 = 0 (rounds up to 4); z = -1.5 and z = -1 are grid points 1 and 2.
    targets = [1.0, -1.0, 0.75, -0.5, 0.0]
    Q, K = lattice_qk(targets)
    out = oracle.forward(Q, K, eye_values(5, 16), Config(Kint=4, calib=MINMAX, recon=NEAREST), decisions=True)
    assert list(out["bins"][0, 0, 4, :5]) == [4, 0, 4, 1, 2]
    # FWM tau = 2: z = -2 is in the window (bin 0), z = -2.125 is in the tail.
    targets = [1.0, -1.0, -1.125, 0.0]
    Q, K = lattice_qk(targets)
    out = oracle.forward(Q, K, eye_values(4, 16), Config(Kint=4, calib=FWM, tau=2.0, recon=NEAREST),
                         decisions=True)
    assert list(out["bins"][0, 0, 3, :4]) == [4, 0, 254, 2]


# --- P3: closed form at K = 1 (App. A "LERP") ----------------------------------------------------

def test_lerp_k1_closed_form():
    T = 16
    Q, K, _, _ = rand_inputs(1, 1, T, 16, 4, scale=2.0)
    out = oracle.forward(Q, K, eye_values(T, 16), Config(Kint=1, calib=MINMAX, recon=LERP))
    S = scores_np(Q, K)[0, 0]
    for i in range(1, T):
        s = S[i, : i + 1]
        M, m = s.max(), s.min()
        rho = (s - m) / (M - m)
        w = (1 - rho) * math.exp(m - M) + rho
        assert np.allclose(out["O"][0, 0, i, : i + 1], w / w.sum(), rtol=0, atol=1e-15)


# --- P4: K -> infinity, against textbook interpolation bounds ------------------------------------

@pytest.mark.parametrize("calib", [MINMAX, FWM, FWM_RESOLVED])
def test_convergence_to_softmax(calib):
    T, d = 16, 16
    Q, K, _, _ = rand_inputs(8, 1, T, d, 5, scale=2.5)
    V = np.broadcast_to(eye_values(T, d), (8, 1, T, d)).copy()
    S = scores_np(Q, K)
    span = max(S[b, 0, i, : i + 1].max() - S[b, 0, i, : i + 1].min() for b in range(8) for i in range(T))
    # FWM window covering every row: no tail.  The resolved grid needs no such window: with a
    # 1-nat window most keys sit below it, on the continued grid of the same step.
    tau = 1.0 if calib == FWM_RESOLVED else span + 1.0
    Ks = [2 ** k for k in range(2, 13)]
    errs = {LERP: [], NEAREST: []}
    for Kint in Ks:
        for recon in (LERP, NEAREST):
            out = oracle.forward(Q, K, V, Config(Kint=Kint, calib=calib, tau=tau, recon=recon))
            worst_abs = 0.0
            for b in range(8):
                for i in range(1, T):
                    s = S[b, 0, i, : i + 1]
                    pe = np.exp(s - s.max())
                    pe /= pe.sum()
                    p = out["O"][b, 0, i, : i + 1]
                    worst_abs = max(worst_abs, np.max(np.abs(p - pe)))
                    h = (s.max() - s.min()) / Kint if calib == MINMAX else tau / Kint
                    # chord of a convex function: e^z <= w^L <= e^z (1 + h^2/8 e^h);
                    # nearest grid centre: |b_l - z| <= h/2, so w^N / e^z in [e^-h/2, e^h/2].
                    bound = math.log1p(h * h / 8 * math.exp(h)) if recon == LERP else h / 2
                    assert np.max(np.abs(np.log(p / pe))) <= 2 * bound + 1e-12
            errs[recon].append(worst_abs)
    # convergence order from a log-log fit over K >= 32: 2 for LERP, 1 for Nearest
    sel = [k for k, K_ in enumerate(Ks) if K_ >= 32]
    slope = {r: np.polyfit(np.log([Ks[k] for k in sel]), np.log([errs[r][k] for k in sel]), 1)[0]
             for r in (LERP, NEAREST)}
    assert -2.25 < slope[LERP] < -1.75, slope
    assert -1.3 < slope[NEAREST] < -0.7, slope


# --- P5: finite differences in fp64 (App. B; diagnostics A3/A4 of App. "detach") ------------------

def _loss(Q, K, V, dO, cfg):
    return float(np.sum(oracle.forward(Q, K, V, cfg, f64=True)["O"] * dO))


def _fd_setup(seed, calib, tau):
    # find a seed whose every decision is far from a boundary, so a 1e-6 step flips nothing
    for s in range(seed, seed + 200):
        Q, K, V, dO = rand_inputs(1, 1, 8, 4, s, scale=1.5, f64=True)
        f = oracle.forward(Q, K, V, Config(Kint=4, calib=calib, tau=tau), decisions=True, f64=True)
        if np.min(f["margin"]) > 1e-3 and np.min(f["row_margin"][0, 0, 1:]) > 1e-3:
            return Q, K, V, dO
    raise RuntimeError("no well-separated seed")


@pytest.mark.parametrize("calib", [MINMAX, FWM, SOFTMAX, FWM_RESOLVED])
def test_lerp_full_gradient_matches_finite_differences(calib):
    tau = 2.0
    Q, K, V, dO = _fd_setup(10, calib, tau)
    for recon_ste in ((LERP, WEIGHT), (NEAREST, PROB)) if calib != SOFTMAX else ((LERP, WEIGHT),):
        cfg = Config(Kint=4, calib=calib, tau=tau, recon=recon_ste[0], ste=recon_ste[1])
        g = oracle.backward(Q, K, V, dO, cfg, f64=True)
        # Prob-STE's backward is the Jacobian of normalize(w^L): differentiate the LERP forward
        lcfg = Config(Kint=4, calib=calib, tau=tau, recon=LERP)
        eps = 1e-6
        for name, X, G in (("Q", Q, g["dQ"]), ("K", K, g["dK"]), ("V", V, g["dV"] if recon_ste[0] == LERP else None)):
            if G is None:
                continue
            fd = np.zeros_like(X)
            for idx in np.ndindex(X.shape):
                Xp, Xm = X.copy(), X.copy()
                Xp[idx] += eps
                Xm[idx] -= eps
                args_p = {"Q": Q, "K": K, "V": V}
                args_m = dict(args_p)
                args_p[name], args_m[name] = Xp, Xm
                fd[idx] = (_loss(args_p["Q"], args_p["K"], args_p["V"], dO, lcfg)
                           - _loss(args_m["Q"], args_m["K"], args_m["V"], dO, lcfg)) / (2 * eps)
            assert np.max(np.abs(fd - G)) <= 1e-7 * np.max(np.abs(G)) + 1e-9, (calib, recon_ste, name)


def _dS_probe_inputs(T, seed, scale=1.5):
    """K = 4 I and V = I with d = 16: s_ij = Q_i[j], dQ_i[j] = dL/ds_ij, g_ij = dO_i[j], O_i = P_i."""
    d = 16
    rng = np.random.default_rng(seed)
    Q = np.zeros((1, 1, T, d))
    Q[0, 0, :, :T] = rng.standard_normal((T, T)) * scale
    K = np.zeros((1, 1, T, d))
    K[0, 0, np.arange(T), np.arange(T)] = 4.0
    V = np.zeros((1, 1, T, d))
    V[0, 0, np.arange(T), np.arange(T)] = 1.0
    dO = rng.standard_normal((1, 1, T, d))
    return Q, K, V, dO


@pytest.mark.parametrize("calib", [MINMAX, FWM])
@pytest.mark.parametrize("grad", [FULL, DETACH])
def test_weight_ste_is_lerp_jacobian_at_hard_normalization(calib, grad):
    """Eq. (wste): dL/ds = J_{w^L}(s)^T gamma^W with gamma^W = (g - <g>_{P^N}) / W^N; under detach the
    grid is frozen, so J is diagonal (Delta) -- checked on keys that are not extrema."""
    T, tau, eps = 10, 2.0, 1e-6
    for seed in range(20, 60):
        Q, K, V, dO = _dS_probe_inputs(T, seed)
        f = oracle.forward(Q, K, V, Config(Kint=4, calib=calib, tau=tau), decisions=True, f64=True)
        if np.min(f["margin"]) > 1e-3 and np.min(f["row_margin"][0, 0, 1:]) > 1e-3:
            break
    lerp = Config(Kint=4, calib=calib, tau=tau, recon=LERP)
    near = Config(Kint=4, calib=calib, tau=tau, recon=NEAREST, ste=WEIGHT, grad=grad)
    fn = oracle.forward(Q, K, V, near, f64=True)
    dS = oracle.backward(Q, K, V, dO, near, f64=True)["dQ"][0, 0, :, :T]
    for i in range(1, T):
        n = i + 1
        PN, WN = fn["O"][0, 0, i, :n], fn["W"][0, 0, i]
        g = dO[0, 0, i, :n]
        gammaW = (g - PN @ g) / WN
        J = np.zeros((n, n))  # J[k, j] = d w^L_k / d s_j
        for j in range(n):
            Qp, Qm = Q.copy(), Q.copy()
            Qp[0, 0, i, j] += eps
            Qm[0, 0, i, j] -= eps
            fp = oracle.forward(Qp, K, V, lerp, f64=True)
            fm = oracle.forward(Qm, K, V, lerp, f64=True)
            wp = fp["O"][0, 0, i, :n] * fp["WL"][0, 0, i]
            wm = fm["O"][0, 0, i, :n] * fm["WL"][0, 0, i]
            J[:, j] = (wp - wm) / (2 * eps)
        s = Q[0, 0, i, :n]
        if grad == FULL:
            expect = J.T @ gammaW
            assert np.allclose(dS[i, :n], expect, rtol=0, atol=1e-7 * max(1.0, np.abs(expect).max()))
        else:
            inner = [j for j in range(n) if s[j] != s.max() and s[j] != s.min()]
            if not inner:
                continue
            expect = np.diag(J)[inner] * gammaW[inner]
            assert np.allclose(dS[i, inner], expect, rtol=0, atol=1e-7 * max(1.0, np.abs(expect).max()))


# --- Witness: independent PyTorch autograd restatement -------------------------------------------

@pytest.mark.parametrize("calib,recon,ste,grad", ALL_COMBOS + [(SOFTMAX, LERP, WEIGHT, FULL)])
@pytest.mark.parametrize("Kint", [1, 4, 16])
def test_matches_autograd_witness(calib, recon, ste, grad, Kint):
    Q, K, V, dO = rand_inputs(1, 2, 12, 8, 7, scale=2.0)
    cfg = Config(Kint=Kint, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad)
    f = oracle.forward(Q, K, V, cfg)
    b = oracle.backward(Q, K, V, dO, cfg)
    O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


# --- Single-channel ablations (supplement "Single-channel ablation", "Local gradient decomposition") ---

@pytest.mark.parametrize("calib,recon,ste", [(MINMAX, LERP, WEIGHT), (MINMAX, NEAREST, PROB), (MINMAX, NEAREST, WEIGHT),
                                             (FWM, NEAREST, PROB), (FWM, LERP, WEIGHT)])
@pytest.mark.parametrize("grad", [MAX_ONLY, MIN_ONLY])
def test_single_channel_matches_autograd_witness(calib, recon, ste, grad):
    """max_only keeps the maximum's channel (the witness detaches m only), min_only the minimum's
    (M detached); the forward is unchanged."""
    Q, K, V, dO = rand_inputs(1, 2, 12, 8, 17, scale=2.0)
    cfg = Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad)
    f = oracle.forward(Q, K, V, cfg)
    b = oracle.backward(Q, K, V, dO, cfg)
    O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


@pytest.mark.parametrize("calib,recon,ste", [(MINMAX, LERP, WEIGHT), (MINMAX, NEAREST, PROB), (FWM, NEAREST, PROB)])
def test_gradient_decomposition_identity(calib, recon, ste):
    """g_full = g_self + g_M + g_m with g_max_only = g_self + g_M, g_min_only = g_self + g_m and
    g_detach = g_self, so full + detach = max_only + min_only in every linear image of dS (dQ, dK);
    dV and the calibration sums do not depend on the mode (except detach, which has none).
    For FWM (no minimum channel) max_only is full and min_only is detach."""
    Q, K, V, dO = rand_inputs(1, 2, 16, 8, 19, scale=2.0)
    out = {}
    for g in (FULL, DETACH, MAX_ONLY, MIN_ONLY):
        cfg = Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=g)
        out[g] = oracle.backward(Q, K, V, dO, cfg)
    for n in ("dQ", "dK"):
        lhs = out[FULL][n] + out[DETACH][n]
        rhs = out[MAX_ONLY][n] + out[MIN_ONLY][n]
        assert np.max(np.abs(lhs - rhs)) <= 1e-12 * max(1.0, np.max(np.abs(lhs)))
        assert np.max(np.abs(out[MAX_ONLY][n] - out[FULL][n])) > 0 or calib == FWM
        if calib == FWM:
            assert np.array_equal(out[MAX_ONLY][n], out[FULL][n])
            assert np.array_equal(out[MIN_ONLY][n], out[DETACH][n])
    for g in (DETACH, MAX_ONLY, MIN_ONLY):
        assert np.array_equal(out[g]["dV"], out[FULL]["dV"])
    for g in (MAX_ONLY, MIN_ONLY):
        assert np.array_equal(out[g]["cM"], out[FULL]["cM"]) and np.array_equal(out[g]["cm"], out[FULL]["cm"])
    assert not out[DETACH]["cM"].any()


def test_ties_split_evenly_like_autograd():
    """Duplicate keys give tied extrema; amax/amin split the extremum gradient evenly (Table "Edge cases")."""
    Q, K, V, dO = rand_inputs(1, 1, 12, 8, 8, scale=2.0)
    K[0, 0, 5] = K[0, 0, 2]
    K[0, 0, 9] = K[0, 0, 2]
    K[0, 0, 7] = K[0, 0, 3]
    for calib, recon, ste in ((MINMAX, LERP, WEIGHT), (MINMAX, NEAREST, WEIGHT), (FWM, NEAREST, PROB)):
        cfg = Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=FULL)
        f = oracle.forward(Q, K, V, cfg)
        assert f["nmax"].max() >= 2 or f["nmin"].max() >= 2
        b = oracle.backward(Q, K, V, dO, cfg)
        O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
        for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
            assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


# --- P6 / P8: zero-sum identity, shift invariance, the per-key calibration identity --------------

@pytest.mark.parametrize("calib,recon,ste,grad", ALL_COMBOS + RES_COMBOS)
def test_zero_sum_identity(calib, recon, ste, grad):
    Q, K, V, dO = rand_inputs(1, 2, 48, 16, 9, scale=2.0)
    cfg = Config(Kint=8, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad)
    b = oracle.backward(Q, K, V, dO, cfg)
    live = b["dabs"] > 0
    rho = np.abs(b["dsum"][live]) / b["dabs"][live]
    if grad == FULL:
        assert rho.max() < 1e-13  # Eq. (full): the three per-key terms sum to zero
    else:
        assert np.median(rho) > 1e-3  # detach violates it (App. B "Detach")


@pytest.mark.parametrize("calib,recon,ste,grad", ALL_COMBOS + RES_COMBOS)
def test_key_shift_invariance(calib, recon, ste, grad):
    """K' = K + 1 k0^T adds Q_i.k0/sqrt(d) to every score of row i: F(s + c1) = F(s), so O and dV are
    unchanged; dQ' = dQ + (sum_j dS_ij) k0 / sqrt(d), which is dQ exactly under the full gradient."""
    Q, K, V, dO = rand_inputs(1, 2, 24, 8, 11, scale=2.0, f64=True)
    k0 = np.random.default_rng(12).standard_normal(8) * 0.7
    cfg = Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad)
    f, fs = oracle.forward(Q, K, V, cfg, f64=True), oracle.forward(Q, K + k0, V, cfg, f64=True)
    b, bs = oracle.backward(Q, K, V, dO, cfg, f64=True), oracle.backward(Q, K + k0, V, dO, cfg, f64=True)
    assert np.max(np.abs(f["O"] - fs["O"])) < 1e-12
    assert np.max(np.abs(b["dV"] - bs["dV"])) < 1e-12
    expect = b["dQ"] + b["dsum"][..., None] * k0 / math.sqrt(8)
    assert np.max(np.abs(bs["dQ"] - expect)) < 1e-11
    if grad == FULL:
        assert np.max(np.abs(bs["dQ"] - b["dQ"])) < 1e-11


@pytest.mark.parametrize("calib", [MINMAX, FWM])
@pytest.mark.parametrize("recon,ste", [(LERP, WEIGHT), (NEAREST, WEIGHT), (NEAREST, PROB)])
def test_calibration_sums_cancel_own_terms(calib, recon, ste):
    """Delta_j + dw_j/dM + dw_j/dm = 0 per key (App. B), so c_M + c_m = -sum_j gamma_j Delta_j, which is
    the row sum of the detached gradient; under FWM dw/dM = -Delta."""
    Q, K, V, dO = rand_inputs(2, 2, 32, 16, 13, scale=2.0)
    full = oracle.backward(Q, K, V, dO, Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=FULL))
    det = oracle.backward(Q, K, V, dO, Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=DETACH))
    assert np.max(np.abs(full["cM"] + full["cm"] + det["dsum"])) < 1e-12
    if calib == FWM:
        assert np.max(np.abs(full["cm"])) == 0.0


def test_prob_ste_backward_is_lerp_backward():
    """Eq. (pste): Prob-STE back-propagates the Jacobian of normalize(w^L); only the value path
    (dV, with the hard forward P^N) differs from LERP."""
    Q, K, V, dO = rand_inputs(1, 2, 32, 16, 14, scale=2.0)
    for calib in (MINMAX, FWM):
        a = oracle.backward(Q, K, V, dO, Config(Kint=4, calib=calib, tau=3.0, recon=NEAREST, ste=PROB))
        b = oracle.backward(Q, K, V, dO, Config(Kint=4, calib=calib, tau=3.0, recon=LERP))
        assert np.max(np.abs(a["dQ"] - b["dQ"])) < 1e-13 and np.max(np.abs(a["dK"] - b["dK"])) < 1e-13
        assert np.max(np.abs(a["dV"] - b["dV"])) > 1e-6


# --- P10: edge cases of Table "Edge cases" -------------------------------------------------------

@pytest.mark.parametrize("calib,recon,ste,grad", ALL_COMBOS + [(SOFTMAX, LERP, WEIGHT, FULL)])
def test_single_key(calib, recon, ste, grad):
    Q, K, V, dO = rand_inputs(1, 1, 1, 8, 15)
    cfg = Config(Kint=4, calib=calib, tau=3.0, recon=recon, ste=ste, grad=grad)
    f = oracle.forward(Q, K, V, cfg)
    b = oracle.backward(Q, K, V, dO, cfg)
    assert np.allclose(f["O"], V)
    assert np.all(b["dQ"] == 0) and np.all(b["dK"] == 0)
    assert np.allclose(b["dV"], dO)


def test_degenerate_minmax_rows_are_uniform_with_zero_score_gradient():
    _, K, V, dO = rand_inputs(1, 1, 12, 8, 16)
    Q = np.zeros_like(K)
    for recon in (LERP, NEAREST):
        cfg = Config(Kint=4, calib=MINMAX, recon=recon)
        f = oracle.forward(Q, K, V, cfg)
        b = oracle.backward(Q, K, V, dO, cfg)
        assert np.allclose(f["O"][0, 0], np.cumsum(V[0, 0], 0) / np.arange(1, 13)[:, None])
        assert np.all(b["dQ"] == 0) and np.all(b["dK"] == 0)


def test_fwm_equal_scores_and_far_tail_match_autograd():
    _, K, V, dO = rand_inputs(1, 1, 12, 8, 17)
    cases = [np.zeros_like(K), rand_inputs(1, 1, 12, 8, 18, scale=30.0)[0]]  # all z = 0; all but max in tail
    for Q in cases:
        for recon, ste in ((LERP, WEIGHT), (NEAREST, WEIGHT), (NEAREST, PROB)):
            cfg = Config(Kint=4, calib=FWM, tau=3.0, recon=recon, ste=ste)
            f = oracle.forward(Q, K, V, cfg)
            b = oracle.backward(Q, K, V, dO, cfg)
            O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
            for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
                assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


def test_decision_override_roundtrip():
    Q, K, V, dO = rand_inputs(1, 1, 20, 8, 19, scale=2.0)
    cfg = Config(Kint=4, calib=MINMAX, recon=NEAREST, ste=WEIGHT)
    f = oracle.forward(Q, K, V, cfg, decisions=True)
    ov = {"bins": f["bins"], "ivals": f["ivals"], "amax": f["amax"], "amin": f["amin"]}
    g = oracle.forward(Q, K, V, cfg, override=ov)
    assert np.array_equal(f["O"], g["O"])
    bins = f["bins"].copy()
    i, j = 15, 4
    bins[0, 0, i, j] = bins[0, 0, i, j] + (1 if bins[0, 0, i, j] < 4 else -1)
    h = oracle.forward(Q, K, V, cfg, override={**ov, "bins": bins})
    changed = np.where(np.any(h["O"] != f["O"], axis=-1))
    assert list(changed[2]) == [i]


# --- P1 control: detached gradient projected onto the zero-sum subspace (App. B "Detach (legacy)") ---

@pytest.mark.parametrize("calib,recon,ste,tau", [(MINMAX, LERP, WEIGHT, 3.0), (MINMAX, NEAREST, PROB, 3.0),
                                                 (MINMAX, NEAREST, WEIGHT, 3.0), (FWM, NEAREST, PROB, 1.0),
                                                 (FWM, LERP, WEIGHT, 1.0)])
def test_projection_matches_autograd_witness(calib, recon, ste, tau):
    """The witness detaches M and m and centres the score gradient over each causal row with a
    hook; tau = 1 puts FWM keys in the zero tail, whose centred gradient is -mean."""
    Q, K, V, dO = rand_inputs(1, 2, 14, 8, 23, scale=2.0)
    cfg = Config(Kint=4, calib=calib, tau=tau, recon=recon, ste=ste, grad=DETACH_PROJ)
    b = oracle.backward(Q, K, V, dO, cfg)
    _, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


@pytest.mark.parametrize("calib,recon,ste", [(MINMAX, LERP, WEIGHT), (MINMAX, NEAREST, PROB), (FWM, NEAREST, WEIGHT)])
def test_projection_removes_only_the_common_mode(calib, recon, ste):
    """Every causal row of the projected dS sums to zero; it differs from the detached dS by one
    constant per row (the differences between keys are kept); dV, the forward and the absence of
    calibration sums are those of detach; rows whose detached terms are all zero stay zero."""
    T = 20
    Q, K, V, dO = rand_inputs(1, 2, T, 8, 29, scale=2.0)
    out = {}
    for g in (DETACH, DETACH_PROJ):
        cfg = Config(Kint=4, calib=calib, tau=1.5, recon=recon, ste=ste, grad=g)
        out[g] = oracle.backward(Q, K, V, dO, cfg, want_dS=True)
    dp, dd = out[DETACH_PROJ]["dS"], out[DETACH]["dS"]
    for b in range(1):
        for h in range(2):
            for i in range(T):
                row_p, row_d = dp[b, h, i, :i + 1], dd[b, h, i, :i + 1]
                scale = max(1e-300, np.sum(np.abs(row_d)))
                assert abs(np.sum(row_p)) <= 1e-13 * scale
                shift = row_p - row_d
                assert np.max(np.abs(shift - shift[0])) <= 1e-13 * scale
                assert np.all(dp[b, h, i, i + 1:] == 0)
                if not np.any(row_d):
                    assert not np.any(row_p)
    assert np.array_equal(out[DETACH_PROJ]["dV"], out[DETACH]["dV"])
    assert not out[DETACH_PROJ]["cM"].any() and not out[DETACH_PROJ]["cm"].any()
    # the detached gradient is not zero-sum in general (App. B), so the projection changes dQ, dK
    assert np.max(np.abs(out[DETACH_PROJ]["dK"] - out[DETACH]["dK"])) > 1e-6


# --- Resolved tail policy (App. "Tail policy in the MinMax -> FWM change") --------------------------

@pytest.mark.parametrize("calib,recon,ste,grad", RES_COMBOS + [(RES, NEAREST, PROB, DETACH_PROJ),
                                                               (RES, LERP, WEIGHT, DETACH_PROJ)])
@pytest.mark.parametrize("Kint", [1, 4])
def test_resolved_matches_autograd_witness(calib, recon, ste, grad, Kint):
    """The witness continues FWM's grid below -tau (floor unclipped below, no tail); tau = 1 puts
    most keys of these rows below the window."""
    Q, K, V, dO = rand_inputs(1, 2, 12, 8, 31, scale=2.0)
    cfg = Config(Kint=Kint, calib=calib, tau=1.0, recon=recon, ste=ste, grad=grad)
    f = oracle.forward(Q, K, V, cfg, decisions=True)
    assert np.any(f["ivals"][f["ivals"] != oracle.CODE_MASKED] < oracle.CODE_OFFSET)  # negative indices occur
    b = oracle.backward(Q, K, V, dO, cfg)
    O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


@pytest.mark.parametrize("recon,ste,grad", [(LERP, WEIGHT, FULL), (NEAREST, WEIGHT, FULL), (NEAREST, PROB, FULL),
                                            (NEAREST, PROB, DETACH), (LERP, PROB, DETACH_PROJ)])
def test_resolved_is_fwm_when_no_key_leaves_the_window(recon, ste, grad):
    """Inside the window both policies use the same grid values (the paper: in-window weights
    bit-identical), so with a window wider than every row's span they agree bit for bit."""
    Q, K, V, dO = rand_inputs(1, 2, 20, 8, 33, scale=1.5)
    S = scores_np(Q, K)
    tau = 1.0 + max(S[0, h, i, : i + 1].max() - S[0, h, i, : i + 1].min() for h in range(2) for i in range(20))
    out = {}
    for c in (FWM, RES):
        cfg = Config(Kint=4, calib=c, tau=tau, recon=recon, ste=ste, grad=grad)
        out[c] = (oracle.forward(Q, K, V, cfg, decisions=True), oracle.backward(Q, K, V, dO, cfg))
    for n in ("O", "W"):
        assert np.array_equal(out[FWM][0][n], out[RES][0][n])
    for n in ("dQ", "dK", "dV", "cM"):
        assert np.array_equal(out[FWM][1][n], out[RES][1][n])
    live = out[FWM][0]["bins"] != oracle.CODE_MASKED
    assert np.array_equal(out[FWM][0]["bins"][live].astype(int) + oracle.CODE_OFFSET,
                          out[RES][0]["bins"][live].astype(int))


def test_resolved_brute_force_on_lattice():
    """Nearest index by scanning every grid point b_l = -tau + l h, l = -60..K (ties go up), LERP
    weight from the interval that contains z, on score lattices reaching 11 steps below the
    window; the stored codes are index + 128."""
    rng = np.random.default_rng(35)
    Kint, T, tau = 4, 16, 2.0
    h = tau / Kint
    for trial in range(40):
        ks = rng.integers(0, 61, size=T)
        ks[rng.integers(0, T)] = 0
        targets = 1.0 - 0.125 * ks  # 1/8 lattice: grid points and Nearest midpoints of h = 1/2
        Q, K = lattice_qk(targets)
        cfg = Config(Kint=Kint, calib=RES, tau=tau, recon=NEAREST)
        out = oracle.forward(Q, K, eye_values(T, 16), cfg, decisions=True)
        out_l = oracle.forward(Q, K, eye_values(T, 16), Config(Kint=Kint, calib=RES, tau=tau, recon=LERP))
        z = targets - targets.max()
        grid = {l: -tau + l * h for l in range(-60, Kint + 1)}
        ell, rr, wl, wn = [], [], [], []
        for zj in z:
            best, best_l = math.inf, None
            for l, b in sorted(grid.items()):
                if abs(zj - b) <= best:  # equal distance: the larger index wins
                    best, best_l = abs(zj - b), l
            r = min(max(l for l, b in grid.items() if b <= zj), Kint - 1)
            t = min(max((zj - grid[r]) / h, 0.0), 1.0)
            ell.append(best_l + 128)
            rr.append(r + 128)
            wn.append(math.exp(grid[best_l]))
            wl.append((1 - t) * math.exp(grid[r]) + t * math.exp(grid[r + 1]))
        wl, wn = np.array(wl), np.array(wn)
        last = T - 1
        assert np.array_equal(out["bins"][0, 0, last], ell), (trial, targets)
        assert np.array_equal(out["ivals"][0, 0, last], rr), (trial, targets)
        assert np.allclose(out["O"][0, 0, last, :T], wn / wn.sum(), rtol=0, atol=1e-15)
        assert np.allclose(out_l["O"][0, 0, last, :T], wl / wl.sum(), rtol=0, atol=1e-15)


@pytest.mark.parametrize("recon", [LERP, NEAREST])
def test_resolved_on_grid_scores_is_softmax(recon):
    """Scores on the grid's own points (multiples of h = tau/K from the row max, far below the
    window too) are reconstructed exactly, w = e^z, so the resolved operator is softmax there;
    FWM, which zeroes keys below -tau, is not."""
    T, tau, Kint = 16, 1.0, 4
    rng = np.random.default_rng(37)
    ks = rng.integers(0, 40, size=T)
    ks[3] = 0
    targets = -0.25 * ks  # h = 1/4: every score on a grid point, down to 39 steps below the max
    Q, K = lattice_qk(targets)
    V = eye_values(T, 16)
    z = targets - targets.max()
    pe = np.exp(z) / np.exp(z).sum()
    res = oracle.forward(Q, K, V, Config(Kint=Kint, calib=RES, tau=tau, recon=recon))
    fwm = oracle.forward(Q, K, V, Config(Kint=Kint, calib=FWM, tau=tau, recon=recon))
    assert np.allclose(res["O"][0, 0, T - 1, :T], pe, rtol=1e-13, atol=0)
    assert np.max(np.abs(fwm["O"][0, 0, T - 1, :T] - pe)) > 1e-3


def test_resolved_decision_override_roundtrip():
    Q, K, V, dO = rand_inputs(1, 1, 20, 8, 39, scale=2.0)
    cfg = Config(Kint=4, calib=RES, tau=1.0, recon=NEAREST, ste=PROB)
    f = oracle.forward(Q, K, V, cfg, decisions=True)
    ov = {"bins": f["bins"], "ivals": f["ivals"], "amax": f["amax"], "amin": f["amin"]}
    g = oracle.forward(Q, K, V, cfg, override=ov)
    assert np.array_equal(f["O"], g["O"])
    bins = f["bins"].copy()
    i = 17
    below = [j for j in range(i + 1) if 0 < bins[0, 0, i, j] < oracle.CODE_OFFSET]  # keys below the window
    assert below
    j = below[0]
    bins[0, 0, i, j] += 1
    hh = oracle.forward(Q, K, V, cfg, override={**ov, "bins": bins})
    changed = np.where(np.any(hh["O"] != f["O"], axis=-1))
    assert list(changed[2]) == [i]


# --- FP8-rounded exponential baseline (App. "Reduced-precision exponential baselines") --------------

def _fp8_row_weights(z):
    """Weights of the last causal row for scores (0, z_1, .., z_{T-1}) (max 0): with V = I,
    O_j / O_0 = w_j / w_0 and w_0 = e^0 = 1 is exact in E4M3."""
    z = np.asarray(z, np.float64)
    T, d = len(z) + 1, 64
    assert T <= d
    Q = np.zeros((1, 1, T, d), np.float32)
    K = np.zeros((1, 1, T, d), np.float32)
    Q[0, 0, :, 0] = 8.0  # scale 1/sqrt(64): s_ij = K_j0, exactly
    K[0, 0, :, 0] = np.concatenate([[0.0], z])
    out = oracle.forward(Q, K, eye_values(T, d), Config(Kint=4, calib=EXP_FP8), decisions=True)
    O = out["O"][0, 0, T - 1, :T]
    return O[1:] / O[0], out["bins"][0, 0, T - 1, 1:T], Q, K


def test_fp8_rounding_matches_torch_float8():
    """The oracle's E4M3 rounding (a scan of the format's values) against torch's float8_e4m3fn cast,
    on 3000 scores from 0 down to -8 (every binade of the format's (0, 1] range, its subnormals,
    the underflow to zero)."""
    torch = pytest.importorskip("torch")
    z = -np.linspace(0.0, 8.0, 3001)[1:]
    z = np.round(z * 1024) / 1024  # exact in fp32
    for chunk in np.array_split(z, 60):
        w, codes, Q, K = _fp8_row_weights(chunk)
        we = torch.tensor(np.exp(chunk.astype(np.float32).astype(np.float64)))
        ref = we.to(torch.float8_e4m3fn)
        assert np.allclose(w, ref.to(torch.float64).numpy(), rtol=1e-14, atol=0)
        assert np.array_equal(codes, ref.view(torch.uint8).numpy())


def test_fp8_value_set_and_underflow():
    """E4M3 weights in (0, 1]: 49 normal values (exponents -6..0) and 7 subnormal multiples of 2^-9, so
    56 distinct nonzero weights; z below ln 2^-10 = -6.93 rounds to zero.  (No weight sits exactly on a
    rounding midpoint: e^z is irrational for every rational z != 0, so the tie rule never acts.)"""
    z = -np.round(np.linspace(0.0, 9.0, 4000) * 4096) / 4096
    parts = [_fp8_row_weights(c) for c in np.array_split(z[1:], 80)]
    ws = np.concatenate([p[0] for p in parts])
    codes = np.concatenate([p[1] for p in parts])
    assert len(set(codes[codes > 0].tolist())) == 56
    assert np.array_equal(ws > 0, codes > 0)
    zs = z[1:]
    assert np.all(ws[zs < math.log(2.0 ** -10) - 1e-9] == 0.0)
    assert np.all(ws[zs > math.log(2.0 ** -10) + 1e-9] > 0.0)


@pytest.mark.parametrize("grad", [FULL, DETACH, DETACH_PROJ, MAX_ONLY, MIN_ONLY])
def test_fp8_matches_autograd_witness(grad):
    """The witness rounds with torch's float8 cast and adds (e^z - sg(e^z)); the row max stays on the
    gradient path (torch.amax), detached under detach / min_only (no minimum channel)."""
    Q, K, V, dO = rand_inputs(1, 2, 16, 8, 41, scale=2.0)
    cfg = Config(Kint=4, calib=EXP_FP8, grad=grad)
    f = oracle.forward(Q, K, V, cfg)
    b = oracle.backward(Q, K, V, dO, cfg)
    O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


def test_fp8_zero_sum_and_shift_invariance():
    """With the row max on the gradient path every row of dS sums to zero (the paper's measured
    residual is 2.3e-7 in fp32; exact here up to fp64 rounding), and shifting every key by k0 leaves O,
    dV and (full gradient) dQ unchanged."""
    Q, K, V, dO = rand_inputs(1, 2, 24, 8, 43, scale=2.0, f64=True)
    cfg = Config(Kint=4, calib=EXP_FP8, grad=FULL)
    b = oracle.backward(Q, K, V, dO, cfg, f64=True)
    live = b["dabs"] > 0
    assert np.max(np.abs(b["dsum"][live]) / b["dabs"][live]) < 1e-13
    det = oracle.backward(Q, K, V, dO, Config(Kint=4, calib=EXP_FP8, grad=DETACH), f64=True)
    assert np.median(np.abs(det["dsum"][live]) / det["dabs"][live]) > 1e-3
    k0 = np.random.default_rng(44).standard_normal(8) * 0.7
    f, fs = oracle.forward(Q, K, V, cfg, f64=True), oracle.forward(Q, K + k0, V, cfg, f64=True)
    bs = oracle.backward(Q, K + k0, V, dO, cfg, f64=True)
    assert np.max(np.abs(f["O"] - fs["O"])) < 1e-12
    assert np.max(np.abs(b["dV"] - bs["dV"])) < 1e-12
    assert np.max(np.abs(b["dQ"] - bs["dQ"])) < 1e-11


def test_fp8_rows_sum_to_one_and_decision_override():
    Q, K, _, _ = rand_inputs(2, 2, 40, 16, 45, scale=2.0)
    cfg = Config(Kint=4, calib=EXP_FP8)
    out = oracle.forward(Q, K, np.ones_like(Q), cfg, decisions=True)
    assert np.max(np.abs(out["O"] - 1.0)) < 1e-13
    V = rand_inputs(2, 2, 40, 16, 46)[2]
    f = oracle.forward(Q, K, V, cfg, decisions=True)
    ov = {"bins": f["bins"], "ivals": f["ivals"], "amax": f["amax"], "amin": f["amin"]}
    assert np.array_equal(oracle.forward(Q, K, V, cfg, override=ov)["O"], f["O"])
    bins = f["bins"].copy()
    i, j = 30, 7
    bins[1, 0, i, j] += 1  # one key's weight one E4M3 step up: only that row changes
    g = oracle.forward(Q, K, V, cfg, override={**ov, "bins": bins})
    changed = np.argwhere(np.any(g["O"] != f["O"], axis=-1))
    assert changed.tolist() == [[1, 0, i]]


# --- Geometry probe (App. "Geometry probe") --------------------------------------------------------

def _probe(out, name):
    return out["probe"][oracle.PROBE_NAMES.index(name)]


@pytest.mark.parametrize("calib,recon", [(MINMAX, LERP), (MINMAX, NEAREST), (FWM, NEAREST), (FWM, LERP)])
def test_probe_entropy_tv_span_against_library_routines(calib, recon):
    """Softmax entropy and softmax itself from scipy; the operator's own P from its output with V = I;
    span, width and the share of keys below z = -6 from the scores."""
    scipy_special = pytest.importorskip("scipy.special")
    scipy_stats = pytest.importorskip("scipy.stats")
    T, d, Kint, tau = 16, 16, 4, 3.0
    Q, K, _, _ = rand_inputs(2, 2, T, d, 47, scale=3.0)
    cfg = Config(Kint=Kint, calib=calib, tau=tau, recon=recon)
    out = oracle.forward(Q, K, eye_values(T, d)[None, None].repeat(2, 0).repeat(2, 1), cfg, probes=True)
    S = scores_np(Q, K)
    for b in range(2):
        for h in range(2):
            for i in range(T):
                s = S[b, h, i, : i + 1]
                pe = scipy_special.softmax(s)
                P = out["O"][b, h, i, : i + 1]
                assert abs(_probe(out, "entropy")[b, h, i] - scipy_stats.entropy(pe)) < 1e-12
                assert abs(_probe(out, "tv")[b, h, i] - 0.5 * np.abs(P - pe).sum()) < 1e-12
                span = s.max() - s.min()
                assert abs(_probe(out, "span")[b, h, i] - span) < 1e-12
                assert abs(_probe(out, "h")[b, h, i] - (span / Kint if calib == MINMAX else tau / Kint)) < 1e-12
                assert _probe(out, "frac_below6")[b, h, i] == np.mean(s - s.max() < -6.0)


@pytest.mark.parametrize("calib,recon", [(MINMAX, NEAREST), (MINMAX, LERP), (FWM, NEAREST), (FWM, LERP)])
def test_probe_buckets_brute_force_on_lattice(calib, recon):
    """Top-bucket mass and effective buckets exp H(q) from a brute-force bucket assignment (the
    lattice scan of the bins pin) and numpy softmax masses."""
    rng = np.random.default_rng(48)
    Kint, T, tau = 4, 16, 2.0
    for trial in range(30):
        ks = rng.integers(0, 25, size=T)
        ks[rng.integers(0, T)] = 0
        if calib == MINMAX:
            ks[rng.integers(0, T)] = 16
        targets = 1.0 - 0.125 * ks
        Q, K = lattice_qk(targets)
        out = oracle.forward(Q, K, eye_values(T, 16), Config(Kint=Kint, calib=calib, tau=tau, recon=recon),
                             probes=True)
        z = targets - targets.max()
        if calib == MINMAX:
            b = [z.min() + r * (0 - z.min()) / Kint for r in range(Kint + 1)]
            tail = np.zeros(T, bool)
        else:
            b = [-tau + r * tau / Kint for r in range(Kint + 1)]
            tail = z < -tau
        ell, r_idx, _, _ = brute_force_row(z, b, tail)
        pe = np.exp(z) / np.exp(z).sum()
        bucket = np.where(tail, Kint + 1, ell if recon == NEAREST else r_idx)
        top = (~tail) & ((ell == Kint) if recon == NEAREST else (r_idx == Kint - 1))
        q = np.array([pe[bucket == k].sum() for k in range(Kint + 2)])
        q = q[q > 0]
        assert abs(_probe(out, "top_mass")[0, 0, T - 1] - pe[top].sum()) < 1e-12, trial
        assert abs(_probe(out, "eff_buckets")[0, 0, T - 1] - np.exp(-(q * np.log(q)).sum())) < 1e-12, trial


def test_probe_degenerate_and_single_key_rows():
    """Row 0 (one key) and all-equal MinMax rows: one bucket holding all the mass, no span."""
    T = 12
    Q = np.zeros((1, 1, T, 8), np.float32)
    K = rand_inputs(1, 1, T, 8, 49)[1]
    out = oracle.forward(Q, K, eye_values(T, 8)[:, :8] if T <= 8 else np.zeros((1, 1, T, 8), np.float32),
                         Config(Kint=4, calib=MINMAX, recon=NEAREST), probes=True)
    for n, v in (("span", 0.0), ("h", 0.0), ("top_mass", 1.0), ("eff_buckets", 1.0), ("tv", 0.0), ("frac_below6", 0.0)):
        assert np.allclose(_probe(out, n)[0, 0], v, atol=1e-12), n
    assert np.allclose(_probe(out, "entropy")[0, 0], np.log(np.arange(1, T + 1)), atol=1e-12)


# --- BF16 exponential baseline (App. "Reduced-precision exponential baselines") --------------------

@pytest.mark.parametrize("grad", [FULL, DETACH, DETACH_PROJ, MAX_ONLY, MIN_ONLY])
def test_bf16_matches_autograd_witness(grad):
    """The witness casts z to torch.bfloat16, takes torch.exp in bfloat16 and casts back; autograd
    supplies the bfloat16 chain rule the oracle writes out."""
    Q, K, V, dO = rand_inputs(1, 2, 16, 8, 51, scale=2.0)
    cfg = Config(Kint=4, calib=EXP_BF16, grad=grad)
    f = oracle.forward(Q, K, V, cfg)
    b = oracle.backward(Q, K, V, dO, cfg)
    O, dQ, dK, dV = witness.attention(Q, K, V, dO, cfg)
    for a, w in ((f["O"], O), (b["dQ"], dQ), (b["dK"], dK), (b["dV"], dV)):
        assert np.max(np.abs(a - w)) <= 1e-10 * max(1.0, np.max(np.abs(w)))


def test_bf16_codes_are_torch_bfloat16_bits():
    """The decision codes are the low bytes of torch's bfloat16 bit patterns of z and of e^{bf16(z)}."""
    torch = pytest.importorskip("torch")
    z = -np.round(np.linspace(0.0, 12.0, 63) * 1024) / 1024
    T, d = 64, 64
    Q = np.zeros((1, 1, T, d), np.float32)
    K = np.zeros((1, 1, T, d), np.float32)
    Q[0, 0, :, 0] = 8.0
    K[0, 0, :, 0] = np.concatenate([[0.0], z])
    out = oracle.forward(Q, K, eye_values(T, d), Config(Kint=4, calib=EXP_BF16), decisions=True)
    zb = torch.tensor(np.concatenate([[0.0], z])).to(torch.bfloat16)
    wb = torch.exp(zb)
    lo = lambda t: (t.view(torch.int16).to(torch.int32) & 0xFF).numpy()
    assert np.array_equal(out["bins"][0, 0, T - 1], lo(zb))
    assert np.array_equal(out["ivals"][0, 0, T - 1], lo(wb))
    O = out["O"][0, 0, T - 1]
    assert np.allclose(O / O[0], wb.to(torch.float64).numpy(), rtol=1e-14, atol=0)


def test_bf16_zero_sum_and_override():
    Q, K, V, dO = rand_inputs(1, 2, 24, 8, 53, scale=2.0)
    cfg = Config(Kint=4, calib=EXP_BF16, grad=FULL)
    b = oracle.backward(Q, K, V, dO, cfg)
    live = b["dabs"] > 0
    assert np.max(np.abs(b["dsum"][live]) / b["dabs"][live]) < 1e-13
    f = oracle.forward(Q, K, V, cfg, decisions=True)
    ov = {"bins": f["bins"], "ivals": f["ivals"], "amax": f["amax"], "amin": f["amin"]}
    assert np.array_equal(oracle.forward(Q, K, V, cfg, override=ov)["O"], f["O"])
    iv = f["ivals"].copy()
    i, j = 20, 3
    iv[0, 1, i, j] ^= 1  # the other bfloat16 neighbour of that key's weight
    g = oracle.forward(Q, K, V, cfg, override={**ov, "ivals": iv})
    changed = np.argwhere(np.any(g["O"] != f["O"], axis=-1))
    assert changed.tolist() == [[0, 1, i]]
