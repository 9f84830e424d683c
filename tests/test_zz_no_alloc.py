"""kint_attn_fwd_noalloc: the forward for callers that cannot give the library
device memory (inside CUDA-graph stream capture, allocation-free serving loops,
plug-in hosts that pass only input and output buffers).  It must give what the
workspace forward gives, call after call, while the library's fixed scratch
array keeps the previous call's contents."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity


def test_too_large_problem_is_refused_before_any_work():
    lib = kint.load()
    p = ctypes.c_void_p(256)
    st = kint.kint_rowstats(*([256] * 7 + [None, None]))
    # TF32, d = 64: the forward scratch is B*H*T*d*4 bytes = 8*8*4096*64*4 = 64 MiB, above the 32 MiB array
    assert lib.kint_attn_fwd_noalloc(p, p, p, p, ctypes.byref(st), 8, 8, 4096, 64, 4, 1, 8.0, 1, 0, 0, 1, 0,
                                     None) == -8
    assert "scratch" in kint.strerror(-8)


@pytest.mark.gpu
def test_noalloc_forward_matches_workspace_forward_on_consecutive_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dev = torch.device("cuda:0")
    cfg = kint.Config(Kint=4, calib=kint.CALIB_FWM, tau=8.0, recon=kint.RECON_NEAREST, ste=kint.STE_PROB,
                      grad=kint.GRAD_FULL)
    prec = kint.PREC_TF32
    tol = parity.TOL[prec]
    for seed, (B, H, T) in ((21, (2, 3, 300)), (22, (1, 4, 517))):  # two calls in a row, different shapes
        Q, K, V, _ = make_qkvdo(B, H, T, 64, seed=seed)
        q, k, v = (torch.from_numpy(x).to(dev) for x in (Q, K, V))
        O_ref, st_ref = kint.forward(q, k, v, cfg, prec)
        O = torch.full_like(q, float("nan"))
        st = kint.alloc_rowstats(B, H, T, 64, dev, cfg.prob)
        rc = kint.kint_attn_fwd_noalloc(q, k, v, O, st, B, H, T, 64, cfg.Kint, cfg.calib, cfg.tau, cfg.recon,
                                        cfg.ste, cfg.grad, 1, prec)
        assert rc == 0, kint.strerror(rc)
        torch.cuda.synchronize()
        kint.check_status()
        assert parity.normwise(O.cpu().numpy(), O_ref.cpu().numpy().astype(np.float64)) <= tol
        for name in ("W", "W_lerp", "O_lerp"):
            assert parity.normwise(st[name].cpu().numpy(), st_ref[name].cpu().numpy().astype(np.float64)) <= tol
        for name in ("row_max", "row_min", "arg_max", "arg_min", "n_max", "n_min"):
            assert torch.equal(st[name], st_ref[name]), name
