"""Python binding of libkint (include/kint_attn.h): argument marshalling only.

Every step of the operator runs in the CUDA library; PyTorch supplies device
memory and the current stream.  The functions named like the C entry points
take torch tensors and forward their data pointers; ``forward`` / ``backward``
/ ``debug_bins`` additionally allocate outputs, row statistics and workspace
with torch.  If the library cannot be built or loaded this module raises: there
is no other implementation behind it.
"""
from __future__ import annotations

import ctypes
import threading
from dataclasses import dataclass

import torch

from . import build as _build

CALIB_MINMAX, CALIB_FWM, CALIB_SOFTMAX, CALIB_FWM_RESOLVED, CALIB_EXP_FP8, CALIB_EXP_BF16 = 0, 1, 2, 3, 4, 5
RECON_LERP, RECON_NEAREST = 0, 1
STE_WEIGHT, STE_PROB = 0, 1
GRAD_FULL, GRAD_DETACH, GRAD_MAX_ONLY, GRAD_MIN_ONLY, GRAD_DETACH_PROJ = 0, 1, 2, 3, 4
PREC_TF32, PREC_3XTF32 = 0, 1
CODE_NOGRID, CODE_TAIL, CODE_MASKED = 253, 254, 255

ERRORS = {0: "KINT_OK", -1: "KINT_ERR_ARG", -2: "KINT_ERR_UNSUPPORTED", -3: "KINT_ERR_ALIGN",
          -4: "KINT_ERR_WORKSPACE", -5: "KINT_ERR_LAUNCH", -6: "KINT_ERR_DEVICE", -7: "KINT_ERR_NO_DEVICE",
          -8: "KINT_ERR_SCRATCH_LIMIT"}
NOALLOC_SCRATCH_BYTES = 32 << 20

# Every symbol include/kint_attn.h declares.
EXPORTS = ("kint_attn_workspace_bytes", "kint_attn_fwd", "kint_attn_bwd", "kint_attn_debug_bins", "kint_attn_probe",
           "kint_get_status", "kint_strerror", "kint_set_wait_timeout_ns", "kint_set_launch_callback",
           "kint_attn_fwd_noalloc", "kint_test_expire_next_wait", "kint_set_backward_path")

LAUNCH_CB = ctypes.CFUNCTYPE(None, ctypes.c_char_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p)


class KintError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {ERRORS.get(code, code)} ({strerror(code)})")
        self.code = code


class kint_rowstats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("row_max", "row_min", "arg_max", "arg_min", "n_max", "n_min", "W",
                                               "W_lerp", "O_lerp", "c_M", "c_m", "dS_sum", "dS_abs")]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libkint.so (building it first if it is absent or stale)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build() if build_if_missing else _build.LIB
            lib = ctypes.CDLL(path)
            vp, i, f, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
            lib.kint_attn_workspace_bytes.argtypes = [i, i, i, i, i, i]
            lib.kint_attn_workspace_bytes.restype = sz
            lib.kint_attn_fwd.argtypes = [vp, vp, vp, vp, ctypes.POINTER(kint_rowstats), i, i, i, i, i, i, f, i, i,
                                          i, i, i, vp, sz, vp]
            lib.kint_attn_fwd.restype = i
            lib.kint_attn_bwd.argtypes = [vp, vp, vp, vp, vp, ctypes.POINTER(kint_rowstats), vp, vp, vp, i, i, i, i,
                                          i, i, f, i, i, i, i, i, vp, sz, vp]
            lib.kint_attn_bwd.restype = i
            lib.kint_attn_debug_bins.argtypes = [vp, vp, vp, ctypes.POINTER(kint_rowstats), vp, vp, i, i, i, i, i,
                                                 i, f, i, i, i, i, vp, sz, vp]
            lib.kint_attn_debug_bins.restype = i
            lib.kint_attn_probe.argtypes = [vp, vp, ctypes.POINTER(kint_rowstats), vp, i, i, i, i, i, i, f, i, i, i,
                                            vp, sz, vp]
            lib.kint_attn_probe.restype = i
            lib.kint_get_status.argtypes = [vp, ctypes.POINTER(ctypes.c_uint)]
            lib.kint_get_status.restype = i
            lib.kint_strerror.argtypes = [i]
            lib.kint_strerror.restype = ctypes.c_char_p
            lib.kint_set_wait_timeout_ns.argtypes = [ctypes.c_ulonglong]
            lib.kint_set_wait_timeout_ns.restype = None
            lib.kint_set_launch_callback.argtypes = [LAUNCH_CB, ctypes.c_void_p]
            lib.kint_set_launch_callback.restype = None
            lib.kint_attn_fwd_noalloc.argtypes = [vp, vp, vp, vp, ctypes.POINTER(kint_rowstats), i, i, i, i, i, i,
                                                  f, i, i, i, i, i, vp]
            lib.kint_attn_fwd_noalloc.restype = i
            lib.kint_test_expire_next_wait.argtypes = [i]
            lib.kint_test_expire_next_wait.restype = None
            _lib = lib
    return _lib


def strerror(code: int) -> str:
    try:
        return load().kint_strerror(int(code)).decode()
    except Exception:  # the library itself failed to load
        return "unavailable"


@dataclass
class Config:
    """Operator choice: calibration, K, tau, reconstruction, surrogate, backward mode."""
    Kint: int = 4
    calib: int = CALIB_MINMAX
    tau: float = 8.0
    recon: int = RECON_LERP
    ste: int = STE_WEIGHT
    grad: int = GRAD_FULL

    @property
    def prob(self) -> bool:
        return self.calib not in (CALIB_SOFTMAX, CALIB_EXP_FP8, CALIB_EXP_BF16) and self.recon == RECON_NEAREST and \
            self.ste == STE_PROB


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(rc: int, what: str):
    if rc != 0:
        raise KintError(rc, what)


def _stats_struct(st: dict) -> kint_rowstats:
    return kint_rowstats(*[(st[n].data_ptr() if st.get(n) is not None else None) for n, _ in kint_rowstats._fields_])


# ---- the C entry points, tensor in / status out ---------------------------------------------

def kint_attn_workspace_bytes(B, H, T, d, prec=PREC_TF32, is_bwd=0) -> int:
    return int(load().kint_attn_workspace_bytes(B, H, T, d, prec, is_bwd))


def kint_attn_fwd(Q, K, V, O, st: dict, B, H, T, d, Kint, calib, tau, recon, ste, grad, causal, prec, workspace,
                  stream=None) -> int:
    s = _stats_struct(st)
    return load().kint_attn_fwd(_p(Q), _p(K), _p(V), _p(O), ctypes.byref(s), B, H, T, d, Kint, calib, float(tau),
                                recon, ste, grad, causal, prec, _p(workspace),
                                0 if workspace is None else workspace.numel() * workspace.element_size(),
                                _stream(stream))


def kint_attn_bwd(Q, K, V, O, dO, st: dict, dQ, dK, dV, B, H, T, d, Kint, calib, tau, recon, ste, grad, causal,
                  prec, workspace, stream=None) -> int:
    s = _stats_struct(st)
    return load().kint_attn_bwd(_p(Q), _p(K), _p(V), _p(O), _p(dO), ctypes.byref(s), _p(dQ), _p(dK), _p(dV), B, H,
                                T, d, Kint, calib, float(tau), recon, ste, grad, causal, prec, _p(workspace),
                                0 if workspace is None else workspace.numel() * workspace.element_size(),
                                _stream(stream))


def kint_attn_fwd_noalloc(Q, K, V, O, st: dict, B, H, T, d, Kint, calib, tau, recon, ste, grad, causal, prec,
                          stream=None) -> int:
    """Forward with the library's fixed device scratch instead of a workspace: for callers
    that cannot allocate device memory (e.g. inside stream capture)."""
    s = _stats_struct(st)
    return load().kint_attn_fwd_noalloc(_p(Q), _p(K), _p(V), _p(O), ctypes.byref(s), B, H, T, d, Kint, calib,
                                        float(tau), recon, ste, grad, causal, prec, _stream(stream))


def kint_attn_probe(Q, K, st: dict, probe, B, H, T, d, Kint, calib, tau, recon, causal, prec, workspace,
                    stream=None) -> int:
    s = _stats_struct(st)
    return load().kint_attn_probe(_p(Q), _p(K), ctypes.byref(s), _p(probe), B, H, T, d, Kint, calib, float(tau), recon,
                                  causal, prec, _p(workspace),
                                  0 if workspace is None else workspace.numel() * workspace.element_size(),
                                  _stream(stream))


def kint_attn_debug_bins(Q, K, V, st: dict, bins, ivals, B, H, T, d, Kint, calib, tau, recon, ste, causal, prec,
                         workspace, stream=None) -> int:
    s = _stats_struct(st)
    return load().kint_attn_debug_bins(_p(Q), _p(K), _p(V), ctypes.byref(s), _p(bins), _p(ivals), B, H, T, d, Kint,
                                       calib, float(tau), recon, ste, causal, prec, _p(workspace),
                                       0 if workspace is None else workspace.numel() * workspace.element_size(),
                                       _stream(stream))


def kint_get_status(stream=None) -> tuple[int, int]:
    detail = ctypes.c_uint(0)
    rc = load().kint_get_status(_stream(stream), ctypes.byref(detail))
    return int(rc), int(detail.value)


def kint_set_wait_timeout_ns(ns: int) -> None:
    load().kint_set_wait_timeout_ns(int(ns))


def kint_test_expire_next_wait(count: int) -> None:
    load().kint_test_expire_next_wait(int(count))


BWD_AUTO, BWD_TWO_PASS = 0, 1


def kint_set_backward_path(path: int) -> None:
    load().kint_set_backward_path(int(path))


_cb_keep = None


def kint_set_launch_callback(fn) -> None:
    """fn(kernel_name: str, phase: int, stream_handle: int) or None.  The C callback
    object is kept alive here until replaced."""
    global _cb_keep
    if fn is None:
        _cb_keep = None
        load().kint_set_launch_callback(ctypes.cast(None, LAUNCH_CB), None)
        return

    def _tramp(name, phase, stream, user):
        fn(name.decode(), int(phase), stream)

    _cb_keep = LAUNCH_CB(_tramp)
    load().kint_set_launch_callback(_cb_keep, None)


# ---- conveniences that allocate with torch ---------------------------------------------------

def alloc_rowstats(B, H, T, d, device, prob: bool, calib_sums: bool = False, row_sums: bool = False) -> dict:
    """Row statistics for one forward/backward pair.  ``calib_sums`` adds the backward's
    optional per-row outputs c_M and c_m, ``row_sums`` its per-row sums of dS and |dS|."""
    f = dict(device=device, dtype=torch.float32)
    i = dict(device=device, dtype=torch.int32)
    st = {"row_max": torch.empty(B, H, T, **f), "row_min": torch.empty(B, H, T, **f),
          "arg_max": torch.empty(B, H, T, **i), "arg_min": torch.empty(B, H, T, **i),
          "n_max": torch.empty(B, H, T, **i), "n_min": torch.empty(B, H, T, **i), "W": torch.empty(B, H, T, **f),
          "W_lerp": None, "O_lerp": None, "c_M": None, "c_m": None, "dS_sum": None, "dS_abs": None}
    if prob:
        st["W_lerp"] = torch.empty(B, H, T, **f)
        st["O_lerp"] = torch.empty(B, H, T, d, **f)
    if calib_sums:
        st["c_M"] = torch.empty(B, H, T, **f)
        st["c_m"] = torch.empty(B, H, T, **f)
    if row_sums:
        st["dS_sum"] = torch.empty(B, H, T, **f)
        st["dS_abs"] = torch.empty(B, H, T, **f)
    return st


def workspace(B, H, T, d, prec, is_bwd, device) -> torch.Tensor:
    n = kint_attn_workspace_bytes(B, H, T, d, prec, is_bwd)
    return torch.empty(max(n, 16), dtype=torch.uint8, device=device)


def _shape(Q):
    if Q.dim() != 4 or Q.dtype != torch.float32 or not Q.is_cuda or not Q.is_contiguous():
        raise ValueError("expected a contiguous fp32 CUDA tensor [B, H, T, d]")
    return tuple(Q.shape)


def forward(Q, K, V, cfg: Config, prec=PREC_TF32, *, O=None, stats=None, ws=None, stream=None):
    """O, row statistics.  Allocates what is not given."""
    B, H, T, d = _shape(Q)
    O = torch.empty_like(Q) if O is None else O
    stats = alloc_rowstats(B, H, T, d, Q.device, cfg.prob) if stats is None else stats
    ws = workspace(B, H, T, d, prec, 0, Q.device) if ws is None else ws
    _check(kint_attn_fwd(Q, K, V, O, stats, B, H, T, d, cfg.Kint, cfg.calib, cfg.tau, cfg.recon, cfg.ste, cfg.grad,
                         1, prec, ws, stream), "kint_attn_fwd")
    return O, stats


def backward(Q, K, V, O, dO, stats, cfg: Config, prec=PREC_TF32, *, grads=None, ws=None, stream=None):
    """dQ, dK, dV."""
    B, H, T, d = _shape(Q)
    dQ, dK, dV = grads if grads is not None else (torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V))
    ws = workspace(B, H, T, d, prec, 1, Q.device) if ws is None else ws
    _check(kint_attn_bwd(Q, K, V, O, dO, stats, dQ, dK, dV, B, H, T, d, cfg.Kint, cfg.calib, cfg.tau, cfg.recon,
                         cfg.ste, cfg.grad, 1, prec, ws, stream), "kint_attn_bwd")
    return dQ, dK, dV


PROBE_NAMES = ("span", "h", "entropy", "frac_below6", "top_mass", "eff_buckets", "tv")


def probe(Q, K, cfg: Config, prec=PREC_TF32, *, stats=None, ws=None, stream=None) -> dict:
    """Per-row geometry probe [B, H, T] for each of PROBE_NAMES (MinMax and FWM)."""
    B, H, T, d = _shape(Q)
    out = torch.empty(len(PROBE_NAMES), B, H, T, dtype=torch.float32, device=Q.device)
    stats = alloc_rowstats(B, H, T, d, Q.device, False) if stats is None else stats
    ws = workspace(B, H, T, d, prec, 0, Q.device) if ws is None else ws
    _check(kint_attn_probe(Q, K, stats, out, B, H, T, d, cfg.Kint, cfg.calib, cfg.tau, cfg.recon, 1, prec, ws,
                           stream), "kint_attn_probe")
    return dict(zip(PROBE_NAMES, out.unbind(0)))


def debug_bins(Q, K, V, stats, cfg: Config, prec=PREC_TF32, *, ws=None, stream=None):
    """Per-key Nearest index and interval index codes, uint8 [B, H, T, T] each."""
    B, H, T, d = _shape(Q)
    bins = torch.empty(B, H, T, T, dtype=torch.uint8, device=Q.device)
    ivals = torch.empty_like(bins)
    ws = workspace(B, H, T, d, prec, 0, Q.device) if ws is None else ws
    _check(kint_attn_debug_bins(Q, K, V, stats, bins, ivals, B, H, T, d, cfg.Kint, cfg.calib, cfg.tau, cfg.recon,
                                cfg.ste, 1, prec, ws, stream), "kint_attn_debug_bins")
    return bins, ivals


def check_status(stream=None):
    rc, detail = kint_get_status(stream)
    if rc != 0:
        raise KintError(rc, f"device status (flags {detail:#x})")
