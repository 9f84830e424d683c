"""Host-side checks of the C ABI (no GPU needed): the library builds, loads,
exports every function include/kint_attn.h declares, sizes workspaces, and
rejects bad arguments before touching a device."""
import ctypes
import os
import re

import pytest

from paper_2609_33591_gb300 import kint

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    text = open(os.path.join(ROOT, "include", "kint_attn.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kint_[a-z_]+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    assert declared_functions() == sorted(kint.EXPORTS)


def test_library_loads_and_exports_every_declared_symbol():
    lib = ctypes.CDLL(kint.load().__dict__.get("_name", kint.library_path()))
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_workspace_sizes():
    # forward TF32: one transposed V; backward adds K^T, Q^T, dO^T, row scalars and tie sums
    B, H, T, d = 8, 12, 1024, 64
    fwd = kint.kint_attn_workspace_bytes(B, H, T, d, kint.PREC_TF32, 0)
    assert fwd == B * H * T * d * 4
    bwd = kint.kint_attn_workspace_bytes(B, H, T, d, kint.PREC_TF32, 1)
    assert bwd >= 3 * B * H * T * d * 4 + 3 * B * H * T * 4
    assert kint.kint_attn_workspace_bytes(B, H, T, d, kint.PREC_3XTF32, 0) > fwd
    assert kint.kint_attn_workspace_bytes(B, H, T, 96, kint.PREC_TF32, 0) == 0
    assert kint.kint_attn_workspace_bytes(0, H, T, d, kint.PREC_TF32, 0) == 0


@pytest.mark.parametrize("kw,code", [
    (dict(B=0), -1), (dict(T=0), -1), (dict(Kint=0), -1), (dict(Kint=65), -1),
    (dict(calib=1, tau=0.0), -1), (dict(calib=7), -1), (dict(causal=0), -1), (dict(d=96), -2),
    (dict(d=128, prec=1), -2), (dict(Kint=33, prec=1), -2), (dict(Kint=33, d=128), -2),
    (dict(grad=-1), -1), (dict(grad=5), -1),
])
def test_argument_errors_are_returned_before_any_launch(kw, code):
    args = dict(B=1, H=1, T=8, d=64, Kint=4, calib=0, tau=8.0, recon=0, ste=0, grad=0, causal=1, prec=0)
    args.update(kw)
    st = kint.kint_rowstats()
    fake = ctypes.c_void_p(256)  # never dereferenced: validation fails first
    rc = kint.load().kint_attn_fwd(fake, fake, fake, fake, ctypes.byref(st), args["B"], args["H"], args["T"],
                                   args["d"], args["Kint"], args["calib"], args["tau"], args["recon"], args["ste"],
                                   args["grad"], args["causal"], args["prec"], fake, 1 << 30, None)
    assert rc == code


def test_null_stats_and_alignment_and_workspace():
    lib = kint.load()
    st = kint.kint_rowstats()
    p = ctypes.c_void_p(256)
    args = (1, 1, 8, 64, 4, 0, 8.0, 0, 0, 0, 1, 0)
    assert lib.kint_attn_fwd(p, p, p, p, ctypes.byref(st), *args, p, 1 << 30, None) == -1  # null statistics
    full = kint.kint_rowstats(*([256] * 7 + [None, None]))
    prob = (1, 1, 8, 64, 4, 0, 8.0, 1, 1, 0, 1, 0)  # Nearest + Prob-STE needs W_lerp and O_lerp
    assert lib.kint_attn_fwd(p, p, p, p, ctypes.byref(full), *prob, p, 1 << 30, None) == -1
    odd = ctypes.c_void_p(258)
    assert lib.kint_attn_fwd(odd, p, p, p, ctypes.byref(full), *args, p, 1 << 30, None) == -3
    assert lib.kint_attn_fwd(p, p, p, p, ctypes.byref(full), *args, p, 16, None) == -4
    assert lib.kint_attn_fwd(p, p, p, p, ctypes.byref(full), *args, None, 1 << 30, None) == -4


def test_bwd_side_output_alignment():
    """The optional c_M / c_m outputs of kint_attn_bwd must be 16-byte aligned like every buffer."""
    lib = kint.load()
    p = ctypes.c_void_p(256)
    st = kint.kint_rowstats(*([256] * 7 + [None, None, 260, None]))
    rc = lib.kint_attn_bwd(p, p, p, p, p, ctypes.byref(st), p, p, p, 1, 1, 8, 64, 4, 0, 8.0, 0, 0, 0, 1, 0,
                           p, 1 << 30, None)
    assert rc == -3


def test_strerror_covers_every_code():
    for code in kint.ERRORS:
        assert kint.strerror(code) != "unknown error code"
    assert kint.strerror(12345) == "unknown error code"


def test_torch_entry_points_refuse_host_tensors():
    """The product path has no CPU fallback: the tensor-level API and the autograd layer refuse
    host tensors before any call into the library."""
    import torch
    from paper_2609_33591_gb300.attention import KIntSelfAttention, kint_attention
    q = torch.zeros(1, 1, 8, 64)
    for call in (lambda: kint.forward(q, q, q, kint.Config()), lambda: kint.probe(q, q, kint.Config()),
                 lambda: kint_attention(q, q, q, kint.Config()),
                 lambda: KIntSelfAttention(128, 2)(torch.zeros(1, 8, 128))):
        with pytest.raises(ValueError):
            call()


def test_probe_argument_errors():
    """kint_attn_probe: MinMax and FWM only; arguments are checked before any launch."""
    lib = kint.load()
    p = ctypes.c_void_p(256)
    st = kint.kint_rowstats(*([256] * 7 + [None, None]))
    args = (1, 1, 8, 64, 4)
    assert lib.kint_attn_probe(p, p, ctypes.byref(st), p, *args, kint.CALIB_SOFTMAX, 8.0, 0, 1, 0, p, 1 << 30,
                               None) == -2
    assert lib.kint_attn_probe(p, p, ctypes.byref(st), None, *args, kint.CALIB_FWM, 8.0, 0, 1, 0, p, 1 << 30,
                               None) == -1
    assert lib.kint_attn_probe(p, p, ctypes.byref(st), p, *args, kint.CALIB_FWM, 8.0, 0, 1, 0, p, 16, None) == -4
