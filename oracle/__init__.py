"""fp64 CPU oracle for K-interval attention -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path (the CUDA library and
its binding) never imports, links or runs anything here.

The arithmetic lives in ``kint_oracle.c`` (plain C, fp64, one row at a time);
this module only compiles it with gcc and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kint_oracle.c")
_HDR = os.path.join(_HERE, "kint_oracle.h")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")        # fp32 inputs
_SO64 = os.path.join(_BUILD, "liboracle64.so")    # fp64 inputs, same arithmetic

MINMAX, FWM, SOFTMAX, FWM_RESOLVED, EXP_FP8, EXP_BF16 = 0, 1, 2, 3, 4, 5
LERP, NEAREST = 0, 1
WEIGHT, PROB = 0, 1
FULL, DETACH, MAX_ONLY, MIN_ONLY, DETACH_PROJ = 0, 1, 2, 3, 4
CODE_NOGRID, CODE_TAIL, CODE_MASKED, CODE_OFFSET = 253, 254, 255, 128

_lock = threading.Lock()
_libs = {}


def build(force: bool = False) -> str:
    """Compile the oracle (gcc, -O2) into oracle/_build/liboracle.so (fp32
    inputs) and liboracle64.so (fp64 inputs)."""
    os.makedirs(_BUILD, exist_ok=True)
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    for so, extra in ((_SO, []), (_SO64, ["-DKOR_F64_INPUT"])):
        if force or not os.path.exists(so) or os.path.getmtime(so) < newest:
            tmp = so + f".tmp{os.getpid()}"
            cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", *extra, "-o", tmp, _SRC, "-lm", "-lpthread"]
            subprocess.run(cmd, check=True)
            os.replace(tmp, so)
    return _SO


class _Params(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("H", ctypes.c_int), ("T", ctypes.c_int), ("d", ctypes.c_int),
                ("Kint", ctypes.c_int), ("calib", ctypes.c_int), ("tau", ctypes.c_double),
                ("recon", ctypes.c_int), ("ste", ctypes.c_int), ("grad", ctypes.c_int),
                ("nthreads", ctypes.c_int)]


_P = ctypes.c_void_p


class _FwdOut(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("O", "M", "m", "amax", "amin", "nmax", "nmin", "W", "WL", "OL",
                                  "bins", "ivals", "margin", "row_margin", "probe")]


class _BwdOut(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("dQ", "dK", "dV", "cM", "cm", "dsum", "dabs", "dS")]


class _Override(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("bins", "ivals", "amax", "amin")]


def _load(f64: bool = False):
    with _lock:
        if f64 not in _libs:
            build()
            lib = ctypes.CDLL(_SO64 if f64 else _SO)
            lib.kor_forward.argtypes = [ctypes.POINTER(_Params), _P, _P, _P, ctypes.POINTER(_FwdOut),
                                        ctypes.POINTER(_Override)]
            lib.kor_forward.restype = ctypes.c_int
            lib.kor_backward.argtypes = [ctypes.POINTER(_Params), _P, _P, _P, _P, ctypes.POINTER(_BwdOut),
                                         ctypes.POINTER(_Override)]
            lib.kor_backward.restype = ctypes.c_int
            lib.kor_hardware_threads.restype = ctypes.c_int
            _libs[f64] = lib
    return _libs[f64]


def hardware_threads() -> int:
    return int(_load().kor_hardware_threads())


@dataclass
class Config:
    """Operator choice, mirroring the three design axes plus the backward mode."""
    Kint: int = 4
    calib: int = MINMAX
    tau: float = 8.0
    recon: int = LERP
    ste: int = WEIGHT
    grad: int = FULL


def _in(x, f64):
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64 if f64 else np.float32))


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _params(shape, cfg: Config, nthreads: int):
    B, H, T, d = shape
    return _Params(B, H, T, d, cfg.Kint, cfg.calib, float(cfg.tau), cfg.recon, cfg.ste, cfg.grad,
                   int(nthreads))


def _override(ov):
    if not ov:
        return None, []
    keep = []
    o = _Override()
    for name, dt in (("bins", np.uint8), ("ivals", np.uint8), ("amax", np.int32), ("amin", np.int32)):
        a = ov.get(name)
        if a is not None:
            a = np.ascontiguousarray(np.asarray(a, dtype=dt))
            keep.append(a)
            setattr(o, name, a.ctypes.data)
    return o, keep


PROBE_NAMES = ("span", "h", "entropy", "frac_below6", "top_mass", "eff_buckets", "tv")


def forward(Q, K, V, cfg: Config, *, decisions: bool = False, lerp_out: bool = False, override=None,
            nthreads: int = 0, f64: bool = False, probes: bool = False) -> dict:
    """Forward of K-interval attention in fp64.  Q, K, V: [B, H, T, d], taken
    as fp32 (or as fp64 with ``f64=True``).

    Returns O plus the row statistics; with ``decisions`` also the per-key bin
    and interval codes and their distance to the nearest decision boundary.
    """
    lib = _load(f64)
    Q, K, V = _in(Q, f64), _in(K, f64), _in(V, f64)
    B, H, T, d = Q.shape
    out = {
        "O": np.zeros((B, H, T, d)), "M": np.zeros((B, H, T)), "m": np.zeros((B, H, T)),
        "amax": np.zeros((B, H, T), np.int32), "amin": np.zeros((B, H, T), np.int32),
        "nmax": np.zeros((B, H, T), np.int32), "nmin": np.zeros((B, H, T), np.int32),
        "W": np.zeros((B, H, T)), "WL": np.zeros((B, H, T)), "row_margin": np.zeros((B, H, T)),
    }
    if lerp_out:
        out["OL"] = np.zeros((B, H, T, d))
    if probes:
        out["probe"] = np.zeros((len(PROBE_NAMES), B, H, T))
    if decisions:
        out["bins"] = np.zeros((B, H, T, T), np.uint8)
        out["ivals"] = np.zeros((B, H, T, T), np.uint8)
        out["margin"] = np.zeros((B, H, T, T))
    fo = _FwdOut()
    for name, arr in out.items():
        setattr(fo, name, arr.ctypes.data)
    ov, keep = _override(override)
    p = _params(Q.shape, cfg, nthreads)
    rc = lib.kor_forward(ctypes.byref(p), _ptr(Q), _ptr(K), _ptr(V), ctypes.byref(fo),
                         ctypes.byref(ov) if ov is not None else None)
    del keep
    if rc != 0:
        raise ValueError(f"oracle forward rejected the arguments (rc={rc})")
    return out


def backward(Q, K, V, dO, cfg: Config, *, want_dS: bool = False, override=None, nthreads: int = 0,
             f64: bool = False) -> dict:
    """Backward of K-interval attention in fp64: dQ, dK, dV and per-row sums."""
    lib = _load(f64)
    Q, K, V, dO = _in(Q, f64), _in(K, f64), _in(V, f64), _in(dO, f64)
    B, H, T, d = Q.shape
    out = {"dQ": np.zeros((B, H, T, d)), "dK": np.zeros((B, H, T, d)), "dV": np.zeros((B, H, T, d)),
           "cM": np.zeros((B, H, T)), "cm": np.zeros((B, H, T)), "dsum": np.zeros((B, H, T)),
           "dabs": np.zeros((B, H, T))}
    if want_dS:
        out["dS"] = np.zeros((B, H, T, T))
    bo = _BwdOut()
    for name, arr in out.items():
        setattr(bo, name, arr.ctypes.data)
    ov, keep = _override(override)
    p = _params(Q.shape, cfg, nthreads)
    rc = lib.kor_backward(ctypes.byref(p), _ptr(Q), _ptr(K), _ptr(V), _ptr(dO), ctypes.byref(bo),
                          ctypes.byref(ov) if ov is not None else None)
    del keep
    if rc != 0:
        raise ValueError(f"oracle backward rejected the arguments (rc={rc})")
    return out
