"""The bounded device-side waits: a wait that runs out flags the status word, and the
kernel releases what it holds and leaves, so the context stays usable.  The test makes
the row-statistics kernel's first wait (on a barrier nothing completes, before any copy
or product is issued) run out after a short limit; nothing faults, traps or hangs."""
import numpy as np
import pytest
import torch

from paper_2609_33591_gb300 import kint
from paper_2609_33591_gb300.inputs import make_qkvdo
from tests import parity

pytestmark = pytest.mark.gpu

DEFAULT_WAIT_NS = 2_000_000_000


@pytest.fixture(autouse=True)
def _restore():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    kint.load()
    yield
    kint.kint_test_expire_next_wait(0)
    kint.kint_set_wait_timeout_ns(DEFAULT_WAIT_NS)


def test_expired_wait_is_reported_and_the_next_call_is_correct():
    cfg = kint.Config(Kint=4, calib=kint.CALIB_FWM, tau=8.0, recon=kint.RECON_NEAREST, ste=kint.STE_PROB,
                      grad=kint.GRAD_FULL)
    Q, K, V, dO = make_qkvdo(1, 2, 200, 64, seed=26)
    dev = torch.device("cuda:0")
    q, k, v = (torch.from_numpy(x).to(dev) for x in (Q, K, V))
    assert kint.kint_get_status() == (0, 0)
    st = kint.alloc_rowstats(1, 2, 200, 64, dev, cfg.prob)
    for t in st.values():
        if t is not None:
            t.zero_()
    kint.kint_set_wait_timeout_ns(2_000_000)  # 2 ms
    kint.kint_test_expire_next_wait(1)
    kint.forward(q, k, v, cfg, kint.PREC_TF32, stats=st)
    rc, detail = kint.kint_get_status()
    assert rc == -6 and detail & 4, (rc, detail)  # KINT_ERR_DEVICE, "CTA sync timed out"
    assert kint.kint_get_status() == (0, 0)  # the word was cleared
    kint.kint_set_wait_timeout_ns(DEFAULT_WAIT_NS)
    # the hook was consumed: the same call now runs normally and is correct
    parity.check(Q, K, V, dO, cfg, kint.PREC_TF32)
    assert kint.kint_get_status() == (0, 0)
