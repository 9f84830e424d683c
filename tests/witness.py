"""Independent witness for the oracle: a plain PyTorch fp64 restatement of the
operator whose backward comes from autograd instead of closed forms.

Written from the paper's definitions (Sec. 3; App. A; Eqs. wste / pste):
the stop-gradient sg(x) is ``x.detach()``, the index (floor, >= 1/2) carries no
gradient, clamps pass gradient inside their range, torch.amax / torch.amin
split the extremum gradient evenly among ties (the convention of the
"Edge cases" table), and the degenerate MinMax branch is a torch.where with a
safe width.  Test code only.
"""
from __future__ import annotations

import math

import numpy as np
import torch

MINMAX, FWM, SOFTMAX, FWM_RESOLVED, EXP_FP8, EXP_BF16 = 0, 1, 2, 3, 4, 5
LERP, NEAREST = 0, 1
WEIGHT, PROB = 0, 1
FULL, DETACH, MAX_ONLY, MIN_ONLY, DETACH_PROJ = 0, 1, 2, 3, 4


def probs(S: torch.Tensor, valid: torch.Tensor, cfg) -> torch.Tensor:
    """Forward probabilities of one batch of score rows S (fp64, autograd)."""
    K = cfg.Kint
    if cfg.calib == SOFTMAX:
        return torch.softmax(S.masked_fill(~valid, -math.inf), dim=-1)
    M = S.masked_fill(~valid, -math.inf).amax(dim=-1, keepdim=True)
    m = S.masked_fill(~valid, math.inf).amin(dim=-1, keepdim=True)
    # detach stops both extremum channels; the single-channel ablations stop one
    if cfg.grad in (DETACH, DETACH_PROJ, MIN_ONLY):
        M = M.detach()
    if cfg.grad in (DETACH, DETACH_PROJ, MAX_ONLY):
        m = m.detach()
    z = S - M
    if cfg.calib == EXP_FP8:
        # E4M3-rounded exponential forward (torch's float8 cast), the exponential's own
        # derivative backward: w = fp8(e^z) + (e^z - sg(e^z))
        we = torch.exp(z.masked_fill(~valid, -math.inf))
        w = we.detach().to(torch.float8_e4m3fn).to(S.dtype) + (we - we.detach())
        w = torch.where(valid, w, torch.zeros_like(w))
        return w / w.sum(-1, keepdim=True)
    if cfg.calib == EXP_BF16:
        # z cast to bfloat16, the exponential evaluated in bfloat16, cast back; autograd then
        # differentiates through the casts in bfloat16 arithmetic
        w = torch.exp(z.masked_fill(~valid, 0.0).to(torch.bfloat16)).to(S.dtype)
        w = torch.where(valid, w, torch.zeros_like(w))
        return w / w.sum(-1, keepdim=True)
    if cfg.calib == MINMAX:
        span = M - m
        degenerate = span <= 1e-12
        h = torch.where(degenerate, torch.ones_like(span), span / K)
        b0 = m - M
        zc = z
        tail = torch.zeros_like(valid)
    elif cfg.calib == FWM:
        h = torch.full_like(M, cfg.tau / K)
        b0 = torch.full_like(M, -cfg.tau)
        tail = z < -cfg.tau
        zc = z.clamp(-cfg.tau, 0.0)
    else:
        # resolved tail policy: FWM's grid, continued below -tau (no tail, no clip)
        h = torch.full_like(M, cfg.tau / K)
        b0 = torch.full_like(M, -cfg.tau)
        tail = torch.zeros_like(valid)
        zc = z
    u = (zc - b0) / h
    r = torch.floor(u.detach()).clamp(max=K - 1)
    if cfg.calib != FWM_RESOLVED:
        r = r.clamp(min=0)
    b_lo = b0 + r * h
    b_hi = b0 + (r + 1) * h
    # With r = clip(floor(u), 0, K-1) the position t lies in [0, 1] up to rounding; its clip only
    # guards rounding, so its derivative is taken as 1 (the own-score slope Delta applies to every
    # in-window key, the arg-max included, as in the detach formula gamma_i Delta_i of App. B).
    t_raw = (zc - b_lo) / h
    t = t_raw + (t_raw.clamp(0.0, 1.0) - t_raw).detach()
    w_lerp = (1 - t) * torch.exp(b_lo) + t * torch.exp(b_hi)
    ell = r + (t.detach() >= 0.5).to(r.dtype)
    w_near = torch.exp(b0 + ell * h)
    zero = torch.zeros_like(S)
    keep = valid & ~tail
    w_lerp = torch.where(keep, w_lerp, zero)
    w_near = torch.where(keep, w_near, zero)
    if cfg.calib == MINMAX:
        one = torch.ones_like(S)
        w_lerp = torch.where(degenerate & valid, one, w_lerp)
        w_near = torch.where(degenerate & valid, one, w_near)
    if cfg.recon == LERP:
        return w_lerp / w_lerp.sum(-1, keepdim=True)
    if cfg.ste == WEIGHT:
        w = w_lerp + (w_near - w_lerp).detach()
        return w / w.sum(-1, keepdim=True)
    p_lerp = w_lerp / w_lerp.sum(-1, keepdim=True)
    p_near = (w_near / w_near.sum(-1, keepdim=True)).detach()
    return p_lerp + (p_near - p_lerp).detach()


def attention(Q, K, V, dO, cfg):
    """O, dQ, dK, dV of causal K-interval attention by autograd (numpy in/out)."""
    Qt = torch.tensor(np.asarray(Q, dtype=np.float64), requires_grad=True)
    Kt = torch.tensor(np.asarray(K, dtype=np.float64), requires_grad=True)
    Vt = torch.tensor(np.asarray(V, dtype=np.float64), requires_grad=True)
    T, d = Qt.shape[-2], Qt.shape[-1]
    S = Qt @ Kt.transpose(-1, -2) / math.sqrt(d)
    valid = torch.ones(T, T, dtype=torch.bool).tril().expand(S.shape)
    if cfg.grad == DETACH_PROJ and cfg.calib != SOFTMAX:
        # P1: the gradient reaching the scores is centred over each causal row
        vf = valid.to(S.dtype)
        S.register_hook(lambda gS: (gS - (gS * vf).sum(-1, keepdim=True) / vf.sum(-1, keepdim=True)) * vf)
    P = probs(S, valid, cfg)
    O = P @ Vt
    (O * torch.tensor(np.asarray(dO, dtype=np.float64))).sum().backward()
    return (O.detach().numpy(), Qt.grad.numpy(), Kt.grad.numpy(), Vt.grad.numpy())
