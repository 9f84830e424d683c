"""GPU parity at the benchmark's full sizes, in the launch configuration bench.py times
(persistent CTAs looping over many (block, head) items, 1024-long rows).

- The GPT-2-small attention layer: B=8, H=12, T=1024, d=64; K=4, FWM tau=8, Nearest,
  Prob-STE, full gradients; TF32 (the production mode, 5e-3) and 3xTF32 (1e-5, decisions
  bit-exact outside the rounding guard band).
- The variant sweep: B=4, H=12, T=1024, every combination of {MinMax, FWM tau=8} x {LERP,
  Nearest} x {Weight-STE, Prob-STE} x {full, detached} at K in {4, 8, 16} in TF32, and the
  K=4 slice in 3xTF32, each with the zero-sum residual of its score gradient (the paper's
  gradient-consistency diagnostic, App. "The detached-gradient record"): at the fp32
  rounding level for the full modes, O(1e-2) and above for the detached ones.

The oracle compares the GPU's outputs 12 heads at a time.  Each case's flips, errors and
residuals go to the KINT_PARITY_LOG file when it is set.
"""
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity

pytestmark = pytest.mark.gpu

MM, FW = kint.CALIB_MINMAX, kint.CALIB_FWM
LE, NE = kint.RECON_LERP, kint.RECON_NEAREST
WE, PR = kint.STE_WEIGHT, kint.STE_PROB
FU, DE = kint.GRAD_FULL, kint.GRAD_DETACH
X3, TF = kint.PREC_3XTF32, kint.PREC_TF32
COMBOS = [(c, r, s, g) for c in (MM, FW) for r in (LE, NE) for s in (WE, PR) for g in (FU, DE)]
CHUNK = 12  # heads per oracle chunk

_inputs = {}


def _qkvdo(B, H, T, d, seed):
    key = (B, H, T, d, seed)
    if key not in _inputs:
        _inputs.clear()
        _inputs[key] = make_qkvdo(B, H, T, d, seed=seed)
    return _inputs[key]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    kint.load()


def _zero_sum_bar(rep, g):
    """Full modes: the GPU's score gradient sums to zero per row up to fp32 rounding;
    detached: it does not (the median residual is far above the rounding level)."""
    zs = rep["zero_sum_gpu"]
    assert zs["rows"] > 0
    if g == FU:
        assert zs["median"] <= 1e-5, zs
    else:
        assert zs["median"] >= 1e-3, zs


@pytest.mark.parametrize("prec", [TF, X3])
def test_gpt2_bench_config(prec):
    """The benchmark workload itself (same seed as bench.py)."""
    Q, K, V, dO = _qkvdo(8, 12, 1024, 64, 1)
    cfg = kint.Config(Kint=4, calib=FW, tau=8.0, recon=NE, ste=PR, grad=FU)
    rep = parity.check(Q, K, V, dO, cfg, prec, heads_per_chunk=CHUNK)
    _zero_sum_bar(rep, FU)


@pytest.mark.parametrize("Kint", [4, 8, 16])
@pytest.mark.parametrize("c,r,s,g", COMBOS)
def test_sweep_tf32(c, r, s, g, Kint):
    Q, K, V, dO = _qkvdo(4, 12, 1024, 64, 2)
    rep = parity.check(Q, K, V, dO, kint.Config(Kint=Kint, calib=c, tau=8.0, recon=r, ste=s, grad=g), TF,
                       heads_per_chunk=CHUNK)
    _zero_sum_bar(rep, g)


@pytest.mark.parametrize("c,r,s,g", COMBOS)
def test_sweep_3xtf32_k4(c, r, s, g):
    Q, K, V, dO = _qkvdo(4, 12, 1024, 64, 2)
    rep = parity.check(Q, K, V, dO, kint.Config(Kint=4, calib=c, tau=8.0, recon=r, ste=s, grad=g), X3,
                       heads_per_chunk=CHUNK)
    _zero_sum_bar(rep, g)


@pytest.mark.parametrize("c,r,s", [(FW, NE, WE), (MM, NE, PR)])
def test_head_dim_128_long_peaked_rows(c, r, s):
    """The 1B-scale layer's heads (d = 128, T = 2048) with 5% peaked rows (one key per chosen row
    raised by +12 in score, which pushes the rest of the row toward FWM's tail), two heads, TF32."""
    Q, K, V, dO = make_qkvdo(1, 2, 2048, 128, seed=3, peaked_frac=0.05)
    parity.check(Q, K, V, dO, kint.Config(Kint=4, calib=c, tau=8.0, recon=r, ste=s, grad=FU), TF,
                 heads_per_chunk=1)


def test_long_context_rows():
    """The long-context operator (K = 16, MinMax, LERP, d = 128) on one head of 8192 rows, TF32:
    the longest accumulation chains the oracle checks element by element."""
    Q, K, V, dO = make_qkvdo(1, 1, 8192, 128, seed=4)
    parity.check(Q, K, V, dO, kint.Config(Kint=16, calib=MM, tau=8.0, recon=LE, ste=PR, grad=FU), TF)
