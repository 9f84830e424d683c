"""End-to-end invariants of the GPU path that the paper fixes independently of any
reference values:

- shift invariance (App. "The detached-gradient record", rows A1/A2): adding one vector
  k0 to every key shifts each row's scores by a constant, which leaves O, dK and dV
  unchanged, leaves dQ unchanged under the full calibration gradient (its per-row score
  gradient sums to zero, Sec. 3 after Eq. full) and moves dQ_i by s (sum_j dS_ij) k0 under
  the detached one;
- the forward does not depend on the backward mode (App. B: detaching changes only the
  backward): full and detached forwards are bitwise equal;
- under LERP the two surrogate placements coincide (Sec. 3: w^N = w^L there), so
  Weight-STE and Prob-STE give bitwise equal forwards and backwards.
"""
import numpy as np
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity

pytestmark = pytest.mark.gpu

MM, FW, SM = kint.CALIB_MINMAX, kint.CALIB_FWM, kint.CALIB_SOFTMAX
LE, NE = kint.RECON_LERP, kint.RECON_NEAREST
WE, PR = kint.STE_WEIGHT, kint.STE_PROB
FU, DE = kint.GRAD_FULL, kint.GRAD_DETACH
X3, TF = kint.PREC_3XTF32, kint.PREC_TF32


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    kint.load()


def _cfg(c, r, s, g, K=4, tau=8.0):
    return kint.Config(Kint=K, calib=c, tau=tau, recon=r, ste=s, grad=g)


def _run(Q, K, V, dO, cfg, prec, row_sums=False):
    dev = torch.device("cuda:0")
    q, k, v, do = (torch.from_numpy(np.ascontiguousarray(x)).to(dev) for x in (Q, K, V, dO))
    B, H, T, d = q.shape
    st = kint.alloc_rowstats(B, H, T, d, dev, cfg.prob, row_sums=row_sums)
    O, st = kint.forward(q, k, v, cfg, prec, stats=st)
    dQ, dK, dV = kint.backward(q, k, v, O, do, st, cfg, prec)
    torch.cuda.synchronize()
    kint.check_status()
    out = {"O": O, "dQ": dQ, "dK": dK, "dV": dV}
    out.update({n: t for n, t in st.items() if t is not None})
    return out


@pytest.mark.parametrize("c,r,s,g", [(MM, LE, WE, FU), (MM, LE, WE, DE), (FW, LE, PR, FU), (FW, LE, PR, DE),
                                     (SM, LE, WE, FU)])
def test_key_shift(c, r, s, g):
    """K' = K + 1 k0^T (3xTF32; LERP, whose weights are continuous in the scores, so the
    score rounding that the shift changes moves no output by more than rounding)."""
    Q, K, V, dO = make_qkvdo(1, 2, 300, 64, seed=23)
    k0 = (0.5 * np.random.default_rng(23).standard_normal(64)).astype(np.float32)
    Ks = (K + k0).astype(np.float32)
    cfg = _cfg(c, r, s, g)
    a = _run(Q, K, V, dO, cfg, X3, row_sums=True)
    b = _run(Q, Ks, V, dO, cfg, X3)
    cpu = lambda t: t.cpu().numpy().astype(np.float64)
    tol = 2e-5
    for n in ("O", "dK", "dV"):
        assert parity.normwise(cpu(b[n]), cpu(a[n])) <= tol, n
    scale = 1.0 / 8.0  # 1 / sqrt(d)
    shift = scale * cpu(a["dS_sum"])[..., None] * k0.astype(np.float64)  # s (sum_j dS_ij) k0
    if g == FU or c == SM:
        # the full gradient sums to zero per row: no shift, and the GPU's row sums say so
        assert parity.normwise(cpu(b["dQ"]), cpu(a["dQ"])) <= tol
        assert np.max(np.abs(shift)) <= tol * np.max(np.abs(cpu(a["dQ"])))
    else:
        # detached: dQ moves by s (sum_j dS_ij) k0, a visible shift
        assert np.max(np.abs(shift)) >= 1e-2 * np.max(np.abs(cpu(a["dQ"])))
        assert parity.normwise(cpu(b["dQ"]), cpu(a["dQ"]) + shift) <= tol


@pytest.mark.parametrize("c,r,s", [(MM, LE, WE), (MM, NE, PR), (FW, NE, PR), (FW, NE, WE)])
@pytest.mark.parametrize("prec", [TF, X3])
def test_detach_forward_is_bitwise_the_full_forward(c, r, s, prec):
    Q, K, V, dO = make_qkvdo(2, 2, 200, 64, seed=24)
    dev = torch.device("cuda:0")
    q, k, v = (torch.from_numpy(x).to(dev) for x in (Q, K, V))
    outs = []
    for g in (FU, DE, kint.GRAD_DETACH_PROJ):
        O, st = kint.forward(q, k, v, _cfg(c, r, s, g), prec)
        outs.append((O, st))
    torch.cuda.synchronize()
    for O, st in outs[1:]:
        assert torch.equal(O, outs[0][0])
        for n, t in st.items():
            if t is not None:
                assert torch.equal(t, outs[0][1][n]), n


@pytest.mark.parametrize("c", [MM, FW])
@pytest.mark.parametrize("g", [FU, DE])
@pytest.mark.parametrize("prec", [TF, X3])
def test_lerp_weight_and_prob_ste_coincide(c, g, prec):
    """Bit for bit on the two-pass backward; on the single-pass one (whose dQ partial sums
    and extremum terms are added in no fixed order) dV and every forward output bit for
    bit, dQ and dK to fp32 summation-order rounding."""
    Q, K, V, dO = make_qkvdo(1, 3, 260, 64, seed=25)
    with parity.backward_path(kint.BWD_TWO_PASS):
        a = _run(Q, K, V, dO, _cfg(c, LE, WE, g), prec)
        b = _run(Q, K, V, dO, _cfg(c, LE, PR, g), prec)
    assert a.keys() == b.keys()
    for n in a:
        assert torch.equal(a[n], b[n]), n
    if parity.single_pass_applies(_cfg(c, LE, WE, g), prec, 64):
        a = _run(Q, K, V, dO, _cfg(c, LE, WE, g), prec)
        b = _run(Q, K, V, dO, _cfg(c, LE, PR, g), prec)
        for n in a:
            if n in ("dQ", "dK"):
                assert parity.normwise(b[n].cpu().numpy(), a[n].cpu().numpy().astype(np.float64)) <= 1e-5, n
            else:
                assert torch.equal(a[n], b[n]), n
