"""GPU-vs-oracle parity machinery (test infrastructure).

Decisions (arg-extrema, Nearest bins, interval indices, FWM tail) are compared
exactly wherever the oracle's fp64 distance to the decision boundary exceeds a
guard band set by the GPU's score rounding; inside the band a differing choice
is counted as a flip, and the oracle is re-run taking the GPU's choice there
(both choices are correct readings of a score that sits within rounding of a
boundary).  Tensors are then compared normwise:
    err(x) = max |x_gpu - x_ref| / max |x_ref|,
and the elementwise p99 of |x_gpu - x_ref| / max(|x_ref|, 1e-3 max |x_ref|) is
reported beside it.

Large problems are checked head by head in chunks (every (b, h) head is an
independent problem), so the oracle's per-key decision arrays stay small; the GPU
runs the whole problem at once, in the launch configuration that is timed.

With KINT_PARITY_LOG set, every check appends one JSON line (case, shape,
configuration, flips, errors, zero-sum residuals) to that file.
"""
from __future__ import annotations

import contextlib
import json
import os

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
# over up to T keys, against the tensor-core sums of the outputs).  The per-row dS sums
# (the zero-sum diagnostic) are held to the same bar against the same scale.
SUM_TOL_FACTOR = 4.0
# The BF16 exponential baseline computes its score gradient in bfloat16 (dL/dz = bf16(bf16(gamma) w)).
# Each backward kernel forms gamma from its own recomputed scores and rounds it, so a gamma within the
# fp32 error of a bfloat16 rounding midpoint may round to the other neighbour (one bfloat16 unit,
# 2^-8 of that key's dS) in either kernel, independently; no decision dump can align the oracle with
# both.  In TF32 these flips hide under the 5e-3 bar; in 3xTF32 gamma's error is ~2^-20 relative, so a
# flip needs gamma within ~2^-20 of a midpoint (about one key in 2^11) and moves one term of a dQ or dK
# row by at most 2^-8 of itself: dQ, dK and the row sums are held to 2^-14 there (measured: 2-3e-5 at
# T = 300).
BF16_GRAD_TOL_X3 = 2.0 ** -14
P99_FLOOR = 1e-3  # elementwise relative errors are taken against max(|ref|, P99_FLOOR * max |ref|)


def to_oracle_cfg(cfg: kint.Config) -> oracle.Config:
    return oracle.Config(Kint=cfg.Kint, calib=cfg.calib, tau=cfg.tau, recon=cfg.recon, ste=cfg.ste, grad=cfg.grad)


def single_pass_applies(cfg: kint.Config, prec, d) -> bool:
    """Whether kint_attn_bwd takes its single-pass backward for this configuration (the
    rule stated at kint_attn_bwd in include/kint_attn.h; calls without row-sum outputs,
    and only when no row has tied maxima)."""
    return prec == kint.PREC_TF32 and d == 64 and cfg.calib != kint.CALIB_MINMAX and \
        cfg.grad != kint.GRAD_DETACH_PROJ


@contextlib.contextmanager
def backward_path(path):
    """Run the block with kint_set_backward_path(path), then back to the default."""
    kint.kint_set_backward_path(path)
    try:
        yield
    finally:
        kint.kint_set_backward_path(kint.BWD_AUTO)


def run_gpu(Q, K, V, dO, cfg: kint.Config, prec, *, want_bins=True, want_bwd=True, row_sums=None):
    """Forward, decision dump and backward on cuda:0 through the C ABI.  With
    ``row_sums`` (default: with the backward) the backward runs a second time with the
    per-row dS sums requested, which always runs the two-pass kernels (the diagnostic
    variant of the dK/dV kernel).  Where the plain run took the single-pass backward, its
    dV must equal the two-pass dV bit for bit (the same weights and products) and the
    two-pass dQ, dK come back as dQ_2p, dK_2p for their own comparison with the oracle;
    otherwise all three must equal those of the plain run bit for bit."""
    dev = torch.device("cuda:0")
    q, k, v, do = (torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in (Q, K, V, dO))
    B, H, T, d = q.shape
    row_sums = want_bwd if row_sums is None else (row_sums and want_bwd)
    st = kint.alloc_rowstats(B, H, T, d, dev, cfg.prob, calib_sums=want_bwd)
    O, st = kint.forward(q, k, v, cfg, prec, stats=st)
    out = {"O": O}
    if want_bins:
        out["bins"], out["ivals"] = kint.debug_bins(q, k, v, st, cfg, prec)
    if want_bwd:
        out["dQ"], out["dK"], out["dV"] = kint.backward(q, k, v, O, do, st, cfg, prec)
    if row_sums:
        st2 = dict(st)
        st2["dS_sum"] = torch.empty(B, H, T, device=dev)
        st2["dS_abs"] = torch.empty(B, H, T, device=dev)
        st2["c_M"], st2["c_m"] = None, None
        g2 = kint.backward(q, k, v, O, do, st2, cfg, prec)
        torch.cuda.synchronize()
        single = single_pass_applies(cfg, prec, d)
        for n, t in zip(("dQ", "dK", "dV"), g2):
            if single and n != "dV":
                out[n + "_2p"] = t
            else:
                assert torch.equal(t, out[n]), f"{n}: the row-sum variant of the backward differs from the plain one"
        out["dS_sum"], out["dS_abs"] = st2["dS_sum"], st2["dS_abs"]
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


class _Acc:
    """One tensor's comparison over chunks: running max |x - ref| and max |ref| (the
    normwise error, or the error against a given scale), and the elementwise errors
    for the p99."""

    def __init__(self):
        self.num = 0.0
        self.den = 0.0
        self.diff, self.mag = [], []

    def add(self, a, ref, scale=None):
        if ref.size == 0:
            return
        diff = np.abs(a.astype(np.float64) - ref)
        self.num = max(self.num, float(diff.max()))
        self.den = max(self.den, float(np.abs(ref).max()) if scale is None else float(scale))
        if scale is None:
            self.diff.append(diff.astype(np.float32).ravel())
            self.mag.append(np.abs(ref).astype(np.float32).ravel())

    def err(self):
        return self.num / self.den if self.den > 0 else self.num

    def p99(self):
        if not self.diff:
            return None
        if self.den == 0:  # an all-zero reference: the absolute errors
            return float(np.percentile(np.concatenate(self.diff), 99))
        r = np.concatenate(self.diff) / np.maximum(np.concatenate(self.mag), np.float32(P99_FLOOR * self.den))
        return float(np.percentile(r, 99))


def _compare_chunk(Q, K, V, dO, g, cfg, ocfg, prec, want_bwd, cnt, acc, rho):
    """Decisions, then the decision-aligned tensors, of one chunk of heads ([1, n, ...])."""
    f = oracle.forward(Q, K, V, ocfg, decisions=True, lerp_out=cfg.prob)
    smax = float(np.max(np.abs(f["M"]))) if f["M"].size else 0.0
    smax = max(smax, float(np.max(np.abs(f["m"]))))
    band = BAND_REL[prec] * (smax + 1.0)
    cnt["band"] = max(cnt["band"], band)

    # arg-extrema and tie counts: exact unless the runner-up is within the band
    for name, c in (("amax", "n_max"), ("amin", "n_min")):
        gname = "arg_max" if name == "amax" else "arg_min"
        if name == "amin" and cfg.calib != kint.CALIB_MINMAX:
            # the minimum side is computed for MinMax only (the FWM and softmax grids are
            # anchored at M alone); the library marks it as not computed
            assert (g["arg_min"] == -1).all() and (g["n_min"] == 0).all() and np.isposinf(g["row_min"]).all()
            continue
        diff = g[gname] != f[name]
        bad = diff & (f["row_margin"] > band)
        assert not bad.any(), f"{gname}: {int(bad.sum())} mismatches outside the guard band"
        cnt[f"{gname}_flips"] += int(diff.sum())
        if cfg.calib == kint.CALIB_MINMAX or name == "amax":
            cdiff = (g[c] != f[c.replace("n_", "n")]) & ~diff & (f["row_margin"] > band)
            assert not cdiff.any(), f"{c}: {int(cdiff.sum())} tie-count mismatches"
    # extrema values: the GPU's fp32 scores
    serr = float(np.max(np.abs(g["row_max"] - f["M"]))) if f["M"].size else 0.0
    assert serr <= band, "row_max beyond score rounding"
    cnt["score_err"] = max(cnt["score_err"], serr)

    # per-key decisions
    flipped = False
    for name in ("bins", "ivals"):
        diff = g[name] != f[name]
        bad = diff & (f["margin"] > band)
        if bad.any():
            idx = np.argwhere(bad)[:5]
            raise AssertionError(f"{name}: {int(bad.sum())} decisions differ outside the guard band, e.g. "
                                 + ", ".join(f"{tuple(i)} gpu={g[name][tuple(i)]} ref={f[name][tuple(i)]} "
                                             f"margin={f['margin'][tuple(i)]:.3g}" for i in idx))
        n = int(diff.sum())
        cnt[f"{name}_flips"] += n
        flipped = flipped or n > 0
    cnt["valid"] += int((f["bins"] != oracle.CODE_MASKED).sum())
    flipped = flipped or bool((g["arg_max"] != f["amax"]).any())
    if cfg.calib == kint.CALIB_MINMAX:
        flipped = flipped or bool((g["arg_min"] != f["amin"]).any())

    # decision-aligned oracle (identical to the plain one when nothing flipped)
    ov = None
    if flipped:
        amin = g["arg_min"] if cfg.calib == kint.CALIB_MINMAX else f["amin"]
        ov = {"bins": g["bins"], "ivals": g["ivals"], "amax": g["arg_max"], "amin": amin}
        f = oracle.forward(Q, K, V, ocfg, lerp_out=cfg.prob, override=ov)
    acc["O"].add(g["O"], f["O"])
    acc["W"].add(g["W"], f["W"])
    if cfg.prob:
        acc["O_lerp"].add(g["O_lerp"], f["OL"])
        acc["W_lerp"].add(g["W_lerp"], f["WL"])
    if not want_bwd:
        return
    b = oracle.backward(Q, K, V, dO, ocfg, override=ov)
    for n in ("dQ", "dK", "dV", "dQ_2p", "dK_2p"):
        if n in g:
            acc[n].add(g[n], b[n[:2]])
    # the per-row calibration sums of Eq. (full), exactly zero where they are not formed
    scale = float(np.max(b["dabs"] + np.abs(b["cM"]) + np.abs(b["cm"]))) if b["dabs"].size else 0.0
    for n, on in (("c_M", "cM"), ("c_m", "cm")):
        if cfg.grad in (kint.GRAD_DETACH, kint.GRAD_DETACH_PROJ) or cfg.calib == kint.CALIB_SOFTMAX or \
                (n == "c_m" and cfg.calib != kint.CALIB_MINMAX):
            assert not g[n].any(), f"{n} not zero where the mode forms no calibration sum"
        elif g[n].size:
            acc[n].add(g[n], b[on], scale=scale)
    # the zero-sum identity (Sec. 3 after Eq. full) on the GPU's own score gradient: per-row
    # sums of dS and |dS| against the oracle's, and the residual |sum dS| / sum |dS| on the
    # rows whose gradient is not zero (oracle sum |dS| above 1e-6 of the largest)
    if "dS_sum" in g:
        acc["dS_abs"].add(g["dS_abs"], b["dabs"])
        acc["dS_sum"].add(g["dS_sum"], b["dsum"], scale=scale)
        live = b["dabs"] > 1e-6 * max(float(b["dabs"].max()), 1e-300)
        if live.any():
            rho["gpu"].append(np.abs(g["dS_sum"][live]) / np.maximum(g["dS_abs"][live], 1e-38))
            rho["oracle"].append(np.abs(b["dsum"][live]) / b["dabs"][live])


PREC_NAME = {kint.PREC_TF32: "tf32", kint.PREC_3XTF32: "3xtf32"}


def check(Q, K, V, dO, cfg: kint.Config, prec, *, want_bwd=True, tol=None, report=None, heads_per_chunk=None,
          case=None):
    """Run GPU and oracle on the same inputs; assert parity; return a report dict.

    The GPU runs the whole [B, H, T, d] problem; the oracle compares it in chunks of
    ``heads_per_chunk`` (b, h) heads (default: all at once)."""
    tol = TOL[prec] if tol is None else tol
    ocfg = to_oracle_cfg(cfg)
    g = run_gpu(Q, K, V, dO, cfg, prec, want_bwd=want_bwd)
    B, H, T, d = Q.shape
    BH = B * H
    step = BH if not heads_per_chunk else max(1, int(heads_per_chunk))
    names = ["O", "W"] + (["O_lerp", "W_lerp"] if cfg.prob else []) + \
        (["dQ", "dK", "dV", "dQ_2p", "dK_2p", "c_M", "c_m", "dS_sum", "dS_abs"] if want_bwd else [])
    acc = {n: _Acc() for n in names}
    cnt = dict(band=0.0, score_err=0.0, arg_max_flips=0, arg_min_flips=0, bins_flips=0, ivals_flips=0, valid=0)
    rho = {"gpu": [], "oracle": []}
    for h0 in range(0, BH, step):
        h1 = min(BH, h0 + step)

        def sl(X):
            return np.ascontiguousarray(X.reshape((BH,) + X.shape[2:])[h0:h1][None])

        gc = {n: sl(a) for n, a in g.items()}
        _compare_chunk(sl(Q), sl(K), sl(V), sl(dO), gc, cfg, ocfg, prec, want_bwd, cnt, acc, rho)

    rep = dict(cnt)
    rep["flip_fraction"] = cnt["bins_flips"] / max(1, cnt["valid"])
    errs = {n: a.err() for n, a in acc.items() if a.den > 0 or a.num > 0}
    rep["errors"] = errs
    rep["p99_rel"] = {n: acc[n].p99() for n in names if acc[n].diff}
    for side in ("gpu", "oracle"):
        r = np.concatenate(rho[side]) if rho[side] else np.zeros(0)
        rep[f"zero_sum_{side}"] = {"median": float(np.median(r)) if r.size else None,
                                   "max": float(r.max()) if r.size else None, "rows": int(r.size)}
    rep["zero_sum_residual_oracle_median"] = rep["zero_sum_oracle"]["median"] or 0.0
    log = os.environ.get("KINT_PARITY_LOG")
    if log:
        rec = {"case": case or os.environ.get("PYTEST_CURRENT_TEST", "").split(" (")[0], "shape": [B, H, T, d],
               "cfg": {"Kint": cfg.Kint, "calib": cfg.calib, "tau": cfg.tau, "recon": cfg.recon, "ste": cfg.ste,
                       "grad": cfg.grad}, "prec": PREC_NAME[prec], "tol": tol, **rep}
        with open(log, "a") as fh:
            fh.write(json.dumps(rec) + "\n")
    if report is not None:
        report.update(rep)
    for n, e in errs.items():
        t = tol * SUM_TOL_FACTOR if n in ("c_M", "c_m", "dS_sum") else tol
        if cfg.calib == kint.CALIB_EXP_BF16 and prec == kint.PREC_3XTF32 and \
                n in ("dQ", "dK", "dQ_2p", "dK_2p", "c_M", "c_m", "dS_sum", "dS_abs"):
            t = max(t, BF16_GRAD_TOL_X3)
        assert e <= t, f"{n}: normwise error {e:.3g} > {t:g} ({rep})"
    return rep
