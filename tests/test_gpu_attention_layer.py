"""GPU: the autograd wrapper and the GPT-2 attention layer on the C ABI, against the
same layer on the CPU with the fp64 oracle as its attention (test infrastructure)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.attention import KIntSelfAttention, kint_attention
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    kint.load()


class _OracleAttention(torch.autograd.Function):
    """The oracle's forward and closed-form backward as a CPU autograd op (fp64)."""

    @staticmethod
    def forward(ctx, q, k, v, cfg):
        arr = [t.detach().numpy().astype(np.float32) for t in (q, k, v)]
        ctx.arr, ctx.cfg = arr, cfg
        return torch.from_numpy(oracle.forward(*arr, parity.to_oracle_cfg(cfg))["O"])

    @staticmethod
    def backward(ctx, dO):
        b = oracle.backward(*ctx.arr, dO.numpy().astype(np.float32), parity.to_oracle_cfg(ctx.cfg))
        return torch.from_numpy(b["dQ"]), torch.from_numpy(b["dK"]), torch.from_numpy(b["dV"]), None


def _rel(a, ref):
    a, ref = a.detach(), ref.detach()
    return float((a.double() - ref).abs().max() / ref.abs().max())


@pytest.mark.parametrize("calib,recon,ste", [(kint.CALIB_FWM, kint.RECON_NEAREST, kint.STE_PROB),
                                             (kint.CALIB_MINMAX, kint.RECON_LERP, kint.STE_WEIGHT)])
def test_autograd_wrapper_is_the_c_abi(calib, recon, ste):
    """Gradients through the autograd op equal the direct kint_attn_bwd call bit for bit."""
    cfg = kint.Config(Kint=4, calib=calib, tau=8.0, recon=recon, ste=ste)
    Q, K, V, dO = (torch.from_numpy(x).cuda() for x in make_qkvdo(2, 3, 200, 64, seed=21))
    q, k, v = (t.clone().requires_grad_(True) for t in (Q, K, V))
    O = kint_attention(q, k, v, cfg, kint.PREC_3XTF32)
    O.backward(dO)
    O2, st = kint.forward(Q, K, V, cfg, kint.PREC_3XTF32)
    dQ, dK, dV = kint.backward(Q, K, V, O2, dO, st, cfg, kint.PREC_3XTF32)
    torch.cuda.synchronize()
    kint.check_status()
    assert torch.equal(O, O2)
    for a, b in ((q.grad, dQ), (k.grad, dK), (v.grad, dV)):
        assert torch.equal(a, b)


def test_gpt2_attention_layer_matches_oracle_layer():
    """A GPT-2-shaped layer (C = 256, 4 heads of 64, T = 160) on the GPU against the same weights
    on the CPU in fp64 with the oracle as attention: output and every parameter gradient.  The
    layer's own work (projections, head split and merge, the chain rule through the op) does not
    depend on the calibration; the softmax comparator keeps the comparison free of rounding
    decisions, which the two layers' differently rounded projections would flip (the per-variant
    decisions are the parity tests' subject)."""
    torch.manual_seed(0)
    torch.backends.cuda.matmul.allow_tf32 = False  # fp32 projections (the default; stated for the tolerance)
    cfg = kint.Config(Kint=4, calib=kint.CALIB_SOFTMAX)
    layer = KIntSelfAttention(256, 4, cfg, kint.PREC_3XTF32).cuda()
    ref = KIntSelfAttention(256, 4, cfg).double()
    ref.load_state_dict({k: v.double().cpu() for k, v in layer.state_dict().items()})
    x = torch.randn(2, 160, 256)
    dy = torch.randn(2, 160, 256)
    xg = x.cuda().requires_grad_(True)
    y = layer(xg)
    y.backward(dy.cuda())
    torch.cuda.synchronize()
    kint.check_status()

    xr = x.double().requires_grad_(True)
    B, T, C = xr.shape
    qkv = ref.c_attn(xr).split(C, dim=2)
    q, k, v = (t.view(B, T, 4, 64).transpose(1, 2) for t in qkv)
    o = _OracleAttention.apply(q, k, v, cfg)
    yr = ref.c_proj(o.transpose(1, 2).reshape(B, T, C))
    yr.backward(dy.double())

    tol = 1e-4  # the 3xTF32 attention (1e-5) inside fp32 linear layers of width 256
    assert _rel(y.cpu(), yr.detach()) < tol
    assert _rel(xg.grad.cpu(), xr.grad) < tol
    for (n, p), (_, pr) in zip(layer.named_parameters(), ref.named_parameters()):
        assert _rel(p.grad.cpu(), pr.grad) < tol, n
