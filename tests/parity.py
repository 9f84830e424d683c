"""GPU-vs-oracle parity machinery (test infrastructure).

Decisions (arg-extrema, Nearest bins, interval indices, FWM tail) are compared
exactly wherever the oracle's fp64 distance to the decision boundary exceeds a
guard band set by the GPU's score rounding; inside the band a differing choice
is counted as a flip, and the oracle is re-run taking the GPU's choice there
(both choices are correct readings of a score that sits within rounding of a
boundary).  Tensors are then compared normwise:
    err(x) = max |x_gpu - x_ref| / max |x_ref|.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2609_33591_gb300 import kint

# Normwise tolerances (3xTF32: fp32-level products; TF32: 10-bit mantissa products).
TOL = {kint.PREC_3XTF32: 1e-5, kint.PREC_TF32: 5e-3}
# Guard band on scores, relative to (max |s| + 1): the GPU score error is at most a
# few units of 2^-22 (3xTF32) or 2^-11 (TF32, truncated operands) times the size of
# the terms summed; the factor 16 covers the rounding of u = s / h + c0 as well.
BAND_REL = {kint.PREC_3XTF32: 16 * 2.0 ** -22, kint.PREC_TF32: 16 * 2.0 ** -11}
# The calibration sums c_M, c_m of Eq. (full) add up to T terms gamma_j dw_j of both signs
# (sum_j P*_j gamma_j = 0) that can cancel to zero (an all-equal FWM row, T = 2), so their
# fp32 error is taken against the row's gradient scale sum_j |dS_ij| + |c_M| + |c_m| rather
# than against their own size, and held to four times the output tolerance (one fp32 sum
# over up to T keys, against the tensor-core sums of the outputs).
SUM_TOL_FACTOR = 4.0
# The BF16 exponential baseline computes its score gradient in bfloat16 (dL/dz = bf16(bf16(gamma) w)):
# a gamma within the GPU's rounding of a bfloat16 midpoint rounds to the other neighbour, one
# bfloat16 unit (2^-8 relative) on that key, twice at most; dQ, dK and the calibration sums are
# held to that, 2^-7 normwise.
BF16_GRAD_TOL = 2.0 ** -7


def to_oracle_cfg(cfg: kint.Config) -> oracle.Config:
    return oracle.Config(Kint=cfg.Kint, calib=cfg.calib, tau=cfg.tau, recon=cfg.recon, ste=cfg.ste, grad=cfg.grad)


def run_gpu(Q, K, V, dO, cfg: kint.Config, prec, *, want_bins=True, want_bwd=True):
    dev = torch.device("cuda:0")
    q, k, v, do = (torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in (Q, K, V, dO))
    B, H, T, d = q.shape
    st = kint.alloc_rowstats(B, H, T, d, dev, cfg.prob, calib_sums=want_bwd)
    O, st = kint.forward(q, k, v, cfg, prec, stats=st)
    out = {"O": O}
    if want_bins:
        out["bins"], out["ivals"] = kint.debug_bins(q, k, v, st, cfg, prec)
    if want_bwd:
        out["dQ"], out["dK"], out["dV"] = kint.backward(q, k, v, O, do, st, cfg, prec)
    torch.cuda.synchronize()
    kint.check_status()
    res = {n: t.cpu().numpy() for n, t in out.items()}
    for n, t in st.items():
        if t is not None:
            res[n] = t.cpu().numpy()
    return res


def normwise(a, ref):
    den = float(np.max(np.abs(ref))) if ref.size else 0.0
    num = float(np.max(np.abs(a.astype(np.float64) - ref))) if ref.size else 0.0
    return num / den if den > 0 else num


def check(Q, K, V, dO, cfg: kint.Config, prec, *, want_bwd=True, tol=None, report=None):
    """Run GPU and oracle on the same inputs; assert parity; return a report dict."""
    tol = TOL[prec] if tol is None else tol
    ocfg = to_oracle_cfg(cfg)
    g = run_gpu(Q, K, V, dO, cfg, prec, want_bwd=want_bwd)
    f = oracle.forward(Q, K, V, ocfg, decisions=True, lerp_out=cfg.prob)
    d = Q.shape[-1]
    smax = float(np.max(np.abs(f["M"]))) if f["M"].size else 0.0
    smax = max(smax, float(np.max(np.abs(f["m"]))))
    band = BAND_REL[prec] * (smax + 1.0)
    rep = {"band": band}

    # arg-extrema and tie counts: exact unless the runner-up is within the band
    for name, cnt in (("amax", "n_max"), ("amin", "n_min")):
        gname = "arg_max" if name == "amax" else "arg_min"
        if name == "amin" and cfg.calib != kint.CALIB_MINMAX:
            # the minimum side is computed for MinMax only (the FWM and softmax grids are
            # anchored at M alone); the library marks it as not computed
            assert (g["arg_min"] == -1).all() and (g["n_min"] == 0).all() and np.isposinf(g["row_min"]).all()
            rep["arg_min_flips"] = 0
            continue
        diff = g[gname] != f[name]
        bad = diff & (f["row_margin"] > band)
        assert not bad.any(), f"{gname}: {int(bad.sum())} mismatches outside the guard band"
        rep[f"{gname}_flips"] = int(diff.sum())
        if cfg.calib == kint.CALIB_MINMAX or name == "amax":
            cdiff = (g[cnt] != f[cnt.replace("n_", "n")]) & ~diff & (f["row_margin"] > band)
            assert not cdiff.any(), f"{cnt}: {int(cdiff.sum())} tie-count mismatches"
    # extrema values: the GPU's fp32 scores
    assert np.max(np.abs(g["row_max"] - f["M"])) <= band, "row_max beyond score rounding"
    rep["score_err"] = float(np.max(np.abs(g["row_max"] - f["M"])))

    # per-key decisions
    for name in ("bins", "ivals"):
        diff = g[name] != f[name]
        bad = diff & (f["margin"] > band)
        if bad.any():
            idx = np.argwhere(bad)[:5]
            raise AssertionError(f"{name}: {int(bad.sum())} decisions differ outside the guard band, e.g. "
                                 + ", ".join(f"{tuple(i)} gpu={g[name][tuple(i)]} ref={f[name][tuple(i)]} "
                                             f"margin={f['margin'][tuple(i)]:.3g}" for i in idx))
        rep[f"{name}_flips"] = int(diff.sum())
    valid = f["bins"] != oracle.CODE_MASKED
    rep["flip_fraction"] = rep["bins_flips"] / max(1, int(valid.sum()))

    # decision-aligned oracle (identical to the plain one when nothing flipped)
    aligned = any(rep[k] for k in ("bins_flips", "ivals_flips", "arg_max_flips", "arg_min_flips"))
    ov = None
    if aligned:
        amin = g["arg_min"] if cfg.calib == kint.CALIB_MINMAX else f["amin"]
        ov = {"bins": g["bins"], "ivals": g["ivals"], "amax": g["arg_max"], "amin": amin}
        f = oracle.forward(Q, K, V, ocfg, lerp_out=cfg.prob, override=ov)
    errs = {"O": normwise(g["O"], f["O"]), "W": normwise(g["W"], f["W"])}
    if cfg.prob:
        errs["O_lerp"] = normwise(g["O_lerp"], f["OL"])
        errs["W_lerp"] = normwise(g["W_lerp"], f["WL"])
    if want_bwd:
        b = oracle.backward(Q, K, V, dO, ocfg, override=ov)
        for n in ("dQ", "dK", "dV"):
            errs[n] = normwise(g[n], b[n])
        # the per-row calibration sums of Eq. (full), exactly zero where they are not formed
        scale = float(np.max(b["dabs"] + np.abs(b["cM"]) + np.abs(b["cm"]))) if b["dabs"].size else 0.0
        for n, on in (("c_M", "cM"), ("c_m", "cm")):
            if cfg.grad in (kint.GRAD_DETACH, kint.GRAD_DETACH_PROJ) or cfg.calib == kint.CALIB_SOFTMAX or \
                    (n == "c_m" and cfg.calib != kint.CALIB_MINMAX):
                assert not g[n].any(), f"{n} not zero where the mode forms no calibration sum"
            elif g[n].size:
                num = float(np.max(np.abs(g[n].astype(np.float64) - b[on])))
                errs[n] = num / scale if scale > 0 else num
        live = b["dabs"] > 0
        rep["zero_sum_residual_oracle_median"] = float(np.median(np.abs(b["dsum"][live]) / b["dabs"][live])) \
            if live.any() else 0.0
    rep["errors"] = errs
    for n, e in errs.items():
        t = tol * SUM_TOL_FACTOR if n in ("c_M", "c_m") else tol
        if cfg.calib == kint.CALIB_EXP_BF16 and n in ("dQ", "dK", "c_M", "c_m"):
            t = max(t, BF16_GRAD_TOL)
        assert e <= t, f"{n}: normwise error {e:.3g} > {t:g} ({rep})"
    if report is not None:
        report.update(rep)
    return rep
