"""kint_attn_fwd_noalloc: the forward for callers that cannot give the library
device memory (inside CUDA-graph stream capture, allocation-free serving loops,
plug-in hosts that pass only input and output buffers).  It runs the same kernels
as the workspace forward, so its outputs must be the same bits, call after call,
while the library's fixed scratch array keeps the previous call's contents."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo


def test_too_large_problem_is_refused_before_any_work():
    lib = kint.load()
    p = ctypes.c_void_p(256)
    st = kint.kint_rowstats(*([256] * 7 + [None, None]))
    # TF32, d = 64: the forward scratch is B*H*T*d*4 bytes = 8*8*4096*64*4 = 64 MiB, above the 32 MiB array
    assert lib.kint_attn_fwd_noalloc(p, p, p, p, ctypes.byref(st), 8, 8, 4096, 64, 4, 1, 8.0, 1, 0, 0, 1, 0,
                                     None) == -8
    # ragged T: B*H*T = 130800 < 131072, but the scratch holds V^T padded to round_up(T, 32) = 320
    # keys: 436 * 64 * 320 * 4 bytes = 35.7 MB, above the array
    assert kint.kint_attn_workspace_bytes(4, 109, 300, 64, kint.PREC_TF32, 0) > kint.NOALLOC_SCRATCH_BYTES
    assert lib.kint_attn_fwd_noalloc(p, p, p, p, ctypes.byref(st), 4, 109, 300, 64, 4, 1, 8.0, 1, 0, 0, 1, 0,
                                     None) == -8
    assert "scratch" in kint.strerror(-8)


def _noalloc(q, k, v, cfg, prec):
    B, H, T, d = q.shape
    O = torch.full_like(q, float("nan"))
    st = kint.alloc_rowstats(B, H, T, d, q.device, cfg.prob)
    rc = kint.kint_attn_fwd_noalloc(q, k, v, O, st, B, H, T, d, cfg.Kint, cfg.calib, cfg.tau, cfg.recon, cfg.ste,
                                    cfg.grad, 1, prec)
    assert rc == 0, kint.strerror(rc)
    return O, st


@pytest.mark.gpu
def test_noalloc_forward_matches_workspace_forward_on_consecutive_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dev = torch.device("cuda:0")
    cfg = kint.Config(Kint=4, calib=kint.CALIB_FWM, tau=8.0, recon=kint.RECON_NEAREST, ste=kint.STE_PROB,
                      grad=kint.GRAD_FULL)
    # A larger call first, with V = NaN, fills a larger part of the scratch array with NaN
    # (the transposed V): a later, smaller call that read anything it did not write itself
    # would return NaN somewhere.
    Q, K, V, _ = make_qkvdo(2, 8, 1000, 64, seed=20)
    q, k = (torch.from_numpy(x).to(dev) for x in (Q, K))
    v = torch.full_like(q, float("nan"))
    O, _ = _noalloc(q, k, v, cfg, kint.PREC_TF32)
    torch.cuda.synchronize()
    kint.check_status()
    assert torch.isnan(O).any()
    # two checked calls in a row, smaller than the first: TF32, then 3xTF32 Prob-STE (whose
    # second pass-2 launch forms O_lerp and W_lerp from the same scratch)
    for seed, (B, H, T), prec in ((21, (2, 3, 300), kint.PREC_TF32), (22, (1, 4, 517), kint.PREC_3XTF32)):
        Q, K, V, _ = make_qkvdo(B, H, T, 64, seed=seed)
        q, k, v = (torch.from_numpy(x).to(dev) for x in (Q, K, V))
        O_ref, st_ref = kint.forward(q, k, v, cfg, prec)
        O, st = _noalloc(q, k, v, cfg, prec)
        torch.cuda.synchronize()
        kint.check_status()
        assert torch.equal(O, O_ref)
        for name in ("W", "W_lerp", "O_lerp", "row_max", "row_min", "arg_max", "arg_min", "n_max", "n_min"):
            assert torch.equal(st[name], st_ref[name]), name
        assert not torch.isnan(O).any()
