"""Efficient-Adam's two-way quantized error-feedback round on GB300 (sm_103a).

A thin ctypes binding of the C ABI in ``include/ea.h`` (libea.so, built in-tree by
``paper_2205_14473_gb300.build``).  The functions keep the C names and only marshal arguments;
every step of the round runs in the library's CUDA kernels.  PyTorch provides the device memory
(the workspace, gradients, x) and the stream.  There is no CPU fallback: if libea.so is missing
or cannot be loaded, the first call raises.

    rnd = EARound(cfg)                 # cfg: EAConfig; allocates the workspace with torch
    for t in range(T):
        for i in range(cfg.n): rnd.worker_compress(i, g[i])
        rnd.server_step()
        rnd.apply(x)
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import threading

from .workloads import (ADAM_AT_SERVER, ADAM_AT_WORKER, Q_IDENTITY, Q_POW2, Q_SIGN_L1,  # noqa: F401
                        Q_UNIFORM_MAX, QuantSpec, Workload)

EA_OK, EA_E_INVAL, EA_E_ALIGN, EA_E_WORKSPACE, EA_E_ORDER = 0, -1, -2, -3, -4
EA_E_CUDA, EA_E_TIMEOUT, EA_E_DEVICE_CHECK, EA_E_UNSUPPORTED = -5, -6, -7, -8
(EA_VIEW_M, EA_VIEW_V, EA_VIEW_E_WORKER, EA_VIEW_E_SERVER, EA_VIEW_M_SERVER, EA_VIEW_V_SERVER,
 EA_VIEW_CODES_WORKER, EA_VIEW_SCALES_WORKER, EA_VIEW_CODES_SERVER, EA_VIEW_SCALES_SERVER) = range(10)

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libea.so")
EXPORTED = ["ea_workspace_bytes", "ea_init", "ea_worker_compress", "ea_server_step", "ea_worker_apply",
            "ea_bits_sent", "ea_round_index", "ea_round_launches", "ea_get_view", "ea_sync_status", "ea_last_error", "ea_destroy",
            "ea_worker_compress_noalloc", "ea_set_hparams", "ea_selftest_bounded_wait"]


class EAError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"status {status}: {msg}")
        self.status = status


class ea_quantizer(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("bits", ctypes.c_int32), ("stochastic", ctypes.c_int32),
                ("pow2_k", ctypes.c_int32), ("pow2_K", ctypes.c_int32), ("n_seg", ctypes.c_int32),
                ("group", ctypes.c_int64), ("seg_lengths", ctypes.POINTER(ctypes.c_int64))]


class ea_config(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int64), ("n", ctypes.c_int32), ("placement", ctypes.c_int32),
                ("qw", ea_quantizer), ("qs", ea_quantizer), ("alpha", ctypes.c_float),
                ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
                ("error_feedback", ctypes.c_int32), ("adam_form", ctypes.c_int32), ("seed", ctypes.c_uint64)]


_lock = threading.Lock()
_lib = None
_P = ctypes.c_void_p


def lib() -> ctypes.CDLL:
    """Load libea.so (raises if it has not been built: there is no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise ImportError(f"{LIB_PATH} is missing: run `python -m paper_2205_14473_gb300.build`")
            L = ctypes.CDLL(LIB_PATH)
            C = ctypes.POINTER(ea_config)
            L.ea_workspace_bytes.argtypes = [C, ctypes.POINTER(ctypes.c_size_t)]
            L.ea_init.argtypes = [C, _P, ctypes.c_size_t, _P, ctypes.POINTER(_P)]
            L.ea_worker_compress.argtypes = [_P, ctypes.c_int32, _P]
            L.ea_server_step.argtypes = [_P]
            L.ea_worker_apply.argtypes = [_P, _P]
            L.ea_bits_sent.argtypes = [_P, ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(ctypes.c_uint64)]
            L.ea_round_index.argtypes = [_P, ctypes.POINTER(ctypes.c_int64)]
            L.ea_round_launches.argtypes = [_P, ctypes.POINTER(ctypes.c_int32)]
            L.ea_get_view.argtypes = [_P, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_P),
                                      ctypes.POINTER(ctypes.c_size_t)]
            L.ea_sync_status.argtypes = [_P]
            L.ea_last_error.argtypes = [_P]
            L.ea_last_error.restype = ctypes.c_char_p
            L.ea_destroy.argtypes = [_P]
            L.ea_set_hparams.argtypes = [_P, ctypes.c_float, ctypes.c_float, ctypes.c_float]
            L.ea_worker_compress_noalloc.argtypes = [C, ctypes.c_int32, ctypes.c_int64, _P, _P, _P, _P, _P, _P, _P]
            L.ea_selftest_bounded_wait.argtypes = [ctypes.c_int64, ctypes.c_int32, _P, ctypes.POINTER(ctypes.c_int32)]
            _lib = L
    return _lib


def _check(status: int, h=None) -> None:
    if status != EA_OK:
        raise EAError(status, lib().ea_last_error(h).decode(errors="replace"))


# ------------------------------------------------------------------ the C functions, same names

def ea_workspace_bytes(cfg: ea_config) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().ea_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)))
    return n.value


def ea_init(cfg: ea_config, workspace_ptr: int, workspace_bytes: int, stream_ptr: int) -> int:
    h = _P()
    _check(lib().ea_init(ctypes.byref(cfg), workspace_ptr, workspace_bytes, stream_ptr, ctypes.byref(h)))
    return h.value


def ea_worker_compress(h: int, worker: int, g_ptr: int) -> None:
    _check(lib().ea_worker_compress(h, worker, g_ptr), h)


def ea_server_step(h: int) -> None:
    _check(lib().ea_server_step(h), h)


def ea_worker_apply(h: int, x_ptr: int) -> None:
    _check(lib().ea_worker_apply(h, x_ptr), h)


def ea_set_hparams(h: int, alpha: float, beta1: float, beta2: float) -> None:
    _check(lib().ea_set_hparams(h, alpha, beta1, beta2), h)


def ea_bits_sent(h: int) -> tuple[int, int]:
    up, down = ctypes.c_uint64(0), ctypes.c_uint64(0)
    _check(lib().ea_bits_sent(h, ctypes.byref(up), ctypes.byref(down)), h)
    return up.value, down.value


def ea_round_index(h: int) -> int:
    t = ctypes.c_int64(0)
    _check(lib().ea_round_index(h, ctypes.byref(t)), h)
    return t.value


def ea_round_launches(h: int) -> int:
    n = ctypes.c_int32(0)
    _check(lib().ea_round_launches(h, ctypes.byref(n)), h)
    return n.value


def ea_get_view(h: int, which: int, index: int = 0) -> tuple[int, int]:
    p, n = _P(), ctypes.c_size_t(0)
    _check(lib().ea_get_view(h, which, index, ctypes.byref(p), ctypes.byref(n)), h)
    return (p.value or 0), n.value


def ea_sync_status(h: int) -> None:
    _check(lib().ea_sync_status(h), h)


def ea_destroy(h: int) -> None:
    lib().ea_destroy(h)


def ea_worker_compress_noalloc(cfg: ea_config, worker: int, round_index: int, g_ptr: int, m_ptr: int, v_ptr: int,
                               e_ptr: int, codes_ptr: int, scales_ptr: int, stream_ptr: int) -> None:
    """Worker compress for callers that cannot allocate (see include/ea.h): no handle, no workspace."""
    _check(lib().ea_worker_compress_noalloc(ctypes.byref(cfg), worker, round_index, g_ptr, m_ptr, v_ptr, e_ptr,
                                            codes_ptr, scales_ptr, stream_ptr))


def ea_selftest_bounded_wait(limit_cycles: int, arrive: int, stream_ptr: int) -> bool:
    """The server's bounded mbarrier wait on its own (see include/ea.h): True if it timed out."""
    t = ctypes.c_int32(-1)
    _check(lib().ea_selftest_bounded_wait(limit_cycles, arrive, stream_ptr, ctypes.byref(t)))
    return t.value == 1


# --------------------------------------------------------------------------- config marshalling

@dataclasses.dataclass
class EAConfig:
    d: int
    n: int
    qw: QuantSpec
    qs: QuantSpec
    alpha: float
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8
    placement: int = ADAM_AT_WORKER
    error_feedback: bool = True
    seed: int = 0
    adam_form: int = 0          # 0: the paper's Adam; 1: the textbook (bias-corrected) form

    @classmethod
    def from_workload(cls, w: Workload, **kw) -> "EAConfig":
        base = dict(d=w.d, n=w.n, qw=w.qw, qs=w.qs, alpha=w.alpha, beta1=w.beta1, beta2=w.beta2, eps=w.eps,
                    seed=w.seed)
        base.update(kw)
        return cls(**base)

    def to_c(self) -> tuple[ea_config, list]:
        keep = []

        def q(spec: QuantSpec) -> ea_quantizer:
            seg = None
            if spec.group < 0:
                arr = (ctypes.c_int64 * len(spec.segments))(*spec.segments)
                keep.append(arr)
                seg = ctypes.cast(arr, ctypes.POINTER(ctypes.c_int64))
            return ea_quantizer(spec.kind, spec.bits, int(spec.stochastic), spec.pow2_k, spec.pow2_K,
                                len(spec.segments) if spec.group < 0 else 0, spec.group, seg)

        c = ea_config(self.d, self.n, self.placement, q(self.qw), q(self.qs), self.alpha, self.beta1, self.beta2,
                      self.eps, int(self.error_feedback), int(self.adam_form), self.seed)
        return c, keep


class EARound:
    """One simulated parameter-server (n workers + server) on the current CUDA device.

    Owns a torch workspace and the library handle; all calls are asynchronous on `stream`
    (default: torch's current stream)."""

    def __init__(self, cfg: EAConfig, stream=None, device=None):
        import torch

        self.cfg = cfg
        self.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        c, keep = cfg.to_c()
        self._c, self._keep = c, keep
        nbytes = ea_workspace_bytes(c)
        self.workspace = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=self.device)
        self.workspace_bytes = nbytes
        self.h = ea_init(c, self.workspace.data_ptr(), nbytes, self.stream.cuda_stream)

    def __del__(self):
        h = getattr(self, "h", None)
        if h:
            ea_destroy(h)
            self.h = None

    # the round
    def worker_compress(self, i: int, g) -> None:
        assert g.dtype.is_floating_point and g.is_contiguous() and g.numel() >= self.cfg.d
        ea_worker_compress(self.h, i, g.data_ptr())

    def server_step(self) -> None:
        ea_server_step(self.h)

    def apply(self, x) -> None:
        assert x.is_contiguous() and x.numel() >= self.cfg.d
        ea_worker_apply(self.h, x.data_ptr())

    def step(self, grads, x) -> None:
        """One full round: every worker compresses its gradient, the server broadcasts, x moves."""
        for i in range(self.cfg.n):
            self.worker_compress(i, grads[i])
        self.server_step()
        self.apply(x)

    # inspection
    def set_hparams(self, alpha: float, beta1: float, beta2: float) -> None:
        ea_set_hparams(self.h, alpha, beta1, beta2)

    def bits_sent(self) -> tuple[int, int]:
        return ea_bits_sent(self.h)

    @property
    def t(self) -> int:
        return ea_round_index(self.h)

    @property
    def launches_per_round(self) -> int:
        return ea_round_launches(self.h)

    def sync(self) -> None:
        ea_sync_status(self.h)

    def view(self, which: int, index: int = 0):
        """A torch view (no copy) of a workspace buffer: float32 for state/scales, int32 for codes."""
        import torch

        ptr, n = ea_get_view(self.h, which, index)
        if n == 0:
            return torch.empty(0, dtype=torch.float32, device=self.device)
        off = ptr - self.workspace.data_ptr()
        dt = torch.int32 if which in (EA_VIEW_CODES_WORKER, EA_VIEW_CODES_SERVER) else torch.float32
        return self.workspace[off:off + n].view(dt)
