"""The oracle against numbers the paper prints (tests/golden/paper_values.json, each with its
citation).  Test infrastructure: CPU only."""
import json
import math
import os

import numpy as np

import oracle
from oracle import Config, FWM, NEAREST
from tests.test_oracle_pins import _fp8_row_weights, rand_inputs

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_values.json")))


def test_e4m3_weight_levels_and_underflow():
    z = -np.round(np.linspace(0.0, 9.0, 4000) * 4096) / 4096
    parts = [_fp8_row_weights(c) for c in np.array_split(z[1:], 80)]
    w = np.concatenate([p[0] for p in parts])
    codes = np.concatenate([p[1] for p in parts])
    nz = codes[codes > 0]
    assert len(set(nz.tolist())) == GOLDEN["e4m3_nonzero_weight_levels"]["value"]
    assert len(set(nz[nz >= 8].tolist())) == GOLDEN["e4m3_normal_weight_levels"]["value"]  # exponent field >= 1
    assert len(set(nz[nz < 8].tolist())) == GOLDEN["e4m3_subnormal_weight_levels"]["value"]
    zs = z[1:]
    last_zero, first_nonzero = zs[w == 0].max(), zs[w > 0].min()  # scores either side of the underflow
    g = GOLDEN["e4m3_underflow_z"]
    assert abs(0.5 * (last_zero + first_nonzero) - g["value"]) <= g["tolerance"]
    assert abs(math.log(2.0 ** -10) - g["value"]) <= g["tolerance"]


def test_fwm_width_printed_for_tau6_k4():
    Q, K, V, _ = rand_inputs(1, 1, 16, 16, 55)
    out = oracle.forward(Q, K, V, Config(Kint=4, calib=FWM, tau=6.0, recon=NEAREST), probes=True)
    h = out["probe"][oracle.PROBE_NAMES.index("h")]
    assert np.all(h == GOLDEN["fwm_width_tau6_k4"]["value"])
