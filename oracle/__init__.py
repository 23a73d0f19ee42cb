"""CPU oracle of one Efficient-Adam round (Algorithms 1 and 2 of arxiv 2205.14473).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg and reference arm (``--impl reference``) may import this package.  It shares no code with the CUDA library
(``paper_2205_14473_gb300``); the two agree only through the message format and the op order that
the header of ``ea_oracle.c`` states.

The C file holds all of the method's arithmetic.  This module is argument marshalling plus the round
bookkeeping of the simulation (state arrays, round counter, bits ledger), in the same shape as the
C-ABI of the CUDA library so that tests can drive both in lockstep.
"""
from __future__ import annotations

import concurrent.futures as _futures
import ctypes
import os
import subprocess
import threading

import numpy as np

Q_IDENTITY, Q_SIGN_L1, Q_UNIFORM_MAX, Q_POW2 = 0, 1, 2, 3
ADAM_AT_WORKER, ADAM_AT_SERVER = 0, 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ea_oracle.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libea_oracle.so")
# binary32 per operation in the written order: no contraction into FMA, no fast math
CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
          "-fno-associative-math", "-frounding-math"]

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ea_oracle.c into oracle/_lib/libea_oracle.so with gcc (idempotent)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", *CFLAGS, _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


class _Quant(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("bits", ctypes.c_int32), ("stochastic", ctypes.c_int32),
                ("pow2_k", ctypes.c_int32), ("pow2_K", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("n_groups", ctypes.c_int64), ("offsets", ctypes.POINTER(ctypes.c_int64))]


class _Config(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int64), ("n", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("error_feedback", ctypes.c_int32), ("adam_form", ctypes.c_int32),
                ("alpha", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("seed", ctypes.c_uint64)]


_P = ctypes.c_void_p


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            L.ora_philox4x32_10.argtypes = [_P, _P, _P]
            L.ora_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64]
            L.ora_uniform.restype = ctypes.c_float
            L.ora_code_words.argtypes = [ctypes.c_int64, ctypes.c_int]
            L.ora_code_words.restype = ctypes.c_int64
            L.ora_message_bits.argtypes = [ctypes.POINTER(_Quant), ctypes.c_int64]
            L.ora_message_bits.restype = ctypes.c_uint64
            L.ora_has_scales.argtypes = [ctypes.POINTER(_Quant)]
            L.ora_quantize.argtypes = [ctypes.POINTER(_Quant), ctypes.c_int64, _P, _P, ctypes.c_uint64,
                                       ctypes.c_uint32, ctypes.c_uint32, _P, _P, _P]
            L.ora_decode.argtypes = [ctypes.POINTER(_Quant), ctypes.c_int64, _P, _P, _P]
            L.ora_worker_step.argtypes = [ctypes.POINTER(_Config), ctypes.POINTER(_Quant), _P,
                                          ctypes.c_int32, ctypes.c_uint32, _P, _P, _P, _P, _P, _P, _P, _P]
            L.ora_server_step.argtypes = [ctypes.POINTER(_Config), ctypes.POINTER(_Quant),
                                          ctypes.POINTER(_Quant), _P, ctypes.c_uint32, _P, _P, _P, _P,
                                          _P, _P, _P, _P, _P, _P]
            L.ora_apply.argtypes = [ctypes.POINTER(_Quant), ctypes.c_int64, _P, _P, _P, _P]
            L.ora_bias_correction.argtypes = [ctypes.c_float, ctypes.c_uint32]
            L.ora_bias_correction.restype = ctypes.c_float
            _lib = L
    return _lib


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


# ------------------------------------------------------------------------------------ quantizers

def group_offsets(d: int, group: int, segments=None) -> np.ndarray:
    """Scale groups as offsets: group == 0 whole vector, > 0 fixed blocks (ragged last block),
    < 0 an explicit list of segment lengths."""
    if group == 0:
        return np.array([0, d], dtype=np.int64)
    if group > 0:
        starts = np.arange(0, d, group, dtype=np.int64)
        return np.concatenate([starts, np.array([d], dtype=np.int64)]) if d > 0 else np.array([0], np.int64)
    lens = np.asarray(segments, dtype=np.int64)
    assert lens.sum() == d
    return np.concatenate([np.zeros(1, np.int64), np.cumsum(lens)])


class Quantizer:
    """One quantization mapping Q with its scale groups (see ea_oracle.c for the formats)."""

    def __init__(self, kind: int, bits: int, offsets: np.ndarray, stochastic: bool = False,
                 pow2_k: int = 0, pow2_K: int = 0):
        self.kind, self.bits, self.stochastic = kind, bits, bool(stochastic)
        self.pow2_k, self.pow2_K = pow2_k, pow2_K
        self.offsets = np.ascontiguousarray(offsets, dtype=np.int64)
        self.n_groups = len(self.offsets) - 1
        self._c = _Quant(kind, bits, int(stochastic), pow2_k, pow2_K, 0, self.n_groups,
                         self.offsets.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)))

    @property
    def has_scales(self) -> bool:
        return self.kind in (Q_SIGN_L1, Q_UNIFORM_MAX)

    def n_words(self, d: int) -> int:
        return (d * self.bits + 31) // 32

    def message_bits(self, d: int) -> int:
        return int(lib().ora_message_bits(ctypes.byref(self._c), d))

    def quantize(self, u: np.ndarray, seed: int = 0, qid: int = 0, t: int = 0, gidx=None):
        """Return (words, scales, dec) of Q(u)."""
        u = np.ascontiguousarray(u, dtype=np.float32)
        d = u.shape[0]
        words = np.zeros(max(self.n_words(d), 1), dtype=np.uint32)
        scales = np.zeros(max(self.n_groups, 1), dtype=np.float32)
        dec = np.zeros(d, dtype=np.float32)
        gi = None if gidx is None else np.ascontiguousarray(gidx, dtype=np.int64)
        lib().ora_quantize(ctypes.byref(self._c), d, _ptr(u), _ptr(gi), seed, qid, t, _ptr(words),
                           _ptr(scales), _ptr(dec))
        return words, scales[: self.n_groups], dec

    def decode(self, words: np.ndarray, scales: np.ndarray, d: int) -> np.ndarray:
        words = np.ascontiguousarray(words, dtype=np.uint32)
        scales = np.ascontiguousarray(scales if len(scales) else np.zeros(1), dtype=np.float32)
        dec = np.zeros(d, dtype=np.float32)
        lib().ora_decode(ctypes.byref(self._c), d, _ptr(words), _ptr(scales), _ptr(dec))
        return dec


def philox4x32_10(ctr, key):
    c = np.asarray(ctr, dtype=np.uint32).copy()
    k = np.asarray(key, dtype=np.uint32).copy()
    out = np.zeros(4, dtype=np.uint32)
    lib().ora_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def uniform(seed: int, qid: int, t: int, j: int) -> float:
    return float(lib().ora_uniform(seed, qid, t, j))


# --------------------------------------------------------------------------------- round driver

class OracleRound:
    """The n workers and the server of Algorithms 1-2 as host arrays, stepped like the C-ABI:
    ``worker_compress(i, g)`` for every i, then ``server_step()``, then ``apply(x)``."""

    def __init__(self, d: int, n: int, qw: Quantizer, qs: Quantizer, alpha: float, beta1: float,
                 beta2: float, eps: float, seed: int = 0, mode: int = ADAM_AT_WORKER,
                 error_feedback: bool = True, gidx=None, threads: int = 1, adam_form: int = 0):
        self.d, self.n, self.qw, self.qs, self.mode = d, n, qw, qs, mode
        self.cfg = _Config(d, n, mode, int(error_feedback), int(adam_form), np.float32(alpha), np.float32(beta1),
                           np.float32(beta2), np.float32(eps), seed)
        v0 = np.float32(eps) if adam_form == 0 else np.float32(0.0)  # the textbook form starts v at 0
        f32 = np.float32
        self.e = np.zeros((n, d), f32)
        self.es = np.zeros(d, f32)
        if mode == ADAM_AT_WORKER:  # Algorithm 2: m_0 = 0, v_0 = eps on every worker
            self.m = np.zeros((n, d), f32)
            self.v = np.full((n, d), v0, f32)
            self.ms = self.vs = np.zeros(1, f32)
        else:
            self.m = self.v = np.zeros((n, 1), f32)
            self.ms = np.zeros(d, f32)
            self.vs = np.full(d, v0, f32)
        self.wwords = np.zeros((n, max(qw.n_words(d), 1)), np.uint32)
        self.wscales = np.zeros((n, max(qw.n_groups, 1)), f32)
        self.swords = np.zeros(max(qs.n_words(d), 1), np.uint32)
        self.sscales = np.zeros(max(qs.n_groups, 1), f32)
        self.gidx = None if gidx is None else np.ascontiguousarray(gidx, dtype=np.int64)
        self.t = 0
        self.up_bits = 0
        self.down_bits = 0
        self.threads = max(1, int(threads))
        self._scratch = [(np.zeros(d, f32), np.zeros(d, f32)) for _ in range(n)]
        self._sscratch = (np.zeros(d, f32), np.zeros(d, f32), np.zeros(d, f32))
        self._chunks = self._make_chunks() if self.threads > 1 else []
        self._pool = _futures.ThreadPoolExecutor(self.threads) if self.threads > 1 else None

    # ------------------------------------------------------------------------ chunked execution
    # The round is separable by scale group: every coordinate's arithmetic depends only on its own
    # values and on its groups' scales.  With threads > 1, the vector is cut into chunks at offsets
    # that are group boundaries of both quantizers and start whole code words of both messages, and
    # the C steps run on the chunks concurrently (the same functions, on sub-arrays; global indices
    # key the Philox counters).  Whole-vector groups cannot be cut: they run as one chunk.

    def _make_chunks(self):
        d, qw, qs = self.d, self.qw, self.qs
        cand = None
        for q in (qw, qs):
            if q.has_scales:
                offs = set(int(o) for o in q.offsets[1:-1])
                cand = offs if cand is None else cand & offs
        if cand is None:
            cand = set(range(1024, d, 1024))
        cand = sorted(o for o in cand if (o * qw.bits) % 32 == 0 and (o * qs.bits) % 32 == 0)
        k = min(4 * self.threads, 64)
        cuts = [0]
        for j in range(1, k):
            target = d * j // k
            i = int(np.searchsorted(cand, target))
            near = [cand[i2] for i2 in (i - 1, i) if 0 <= i2 < len(cand)]
            best = min(near, key=lambda c: abs(c - target), default=None)
            if best is not None and best > cuts[-1]:
                cuts.append(best)
        cuts.append(d)
        if len(cuts) <= 2:
            return []
        gidx = self.gidx if self.gidx is not None else (
            np.arange(d, dtype=np.int64) if (qw.stochastic or qs.stochastic) else None)
        chunks = []
        for lo, hi in zip(cuts[:-1], cuts[1:]):
            def sub(q):
                if not q.has_scales:
                    return Quantizer(q.kind, q.bits, np.array([0, hi - lo], np.int64), q.stochastic, q.pow2_k,
                                     q.pow2_K), 0
                g0 = int(np.searchsorted(q.offsets, lo))
                g1 = int(np.searchsorted(q.offsets, hi))
                return Quantizer(q.kind, q.bits, q.offsets[g0:g1 + 1] - lo, q.stochastic, q.pow2_k, q.pow2_K), g0
            (qwc, gw), (qsc, gs) = sub(qw), sub(qs)
            gi = None if gidx is None else np.ascontiguousarray(gidx[lo:hi])
            chunks.append((lo, hi, qwc, gw, qsc, gs, gi))
        return chunks

    def _cfg_for(self, d: int):
        c = self.cfg
        return _Config(d, c.n, c.mode, c.error_feedback, c.adam_form, c.alpha, c.beta1, c.beta2, c.eps, c.seed)

    @staticmethod
    def _at(a: np.ndarray, off: int):
        """Pointer to element `off` of a C-contiguous 1-D array."""
        return ctypes.c_void_p(a.ctypes.data + off * a.itemsize)

    def _worker_chunk(self, i: int, g: np.ndarray, ch) -> None:
        lo, hi, qwc, gw, _, _, gi = ch
        u, dec = self._scratch[i]
        W = self.mode == ADAM_AT_WORKER
        cfg = self._cfg_for(hi - lo)
        lib().ora_worker_step(ctypes.byref(cfg), ctypes.byref(qwc._c), _ptr(gi), i, self.t, self._at(g, lo),
                              self._at(self.m[i], lo) if W else None, self._at(self.v[i], lo) if W else None,
                              self._at(self.e[i], lo), self._at(u, lo), self._at(dec, lo),
                              self._at(self.wwords[i], lo * self.qw.bits // 32), self._at(self.wscales[i], gw))

    def _server_chunk(self, ch) -> None:
        lo, hi, qwc, gw, qsc, gs, gi = ch
        bw = self.qw.bits
        ww = (ctypes.c_void_p * self.n)(*[self.wwords[i].ctypes.data + (lo * bw // 32) * 4 for i in range(self.n)])
        ws = (ctypes.c_void_p * self.n)(*[self.wscales[i].ctypes.data + gw * 4 for i in range(self.n)])
        acc, w, dec = self._sscratch
        S = self.mode == ADAM_AT_SERVER
        cfg = self._cfg_for(hi - lo)
        lib().ora_server_step(ctypes.byref(cfg), ctypes.byref(qwc._c), ctypes.byref(qsc._c), _ptr(gi), self.t,
                              ctypes.cast(ww, _P), ctypes.cast(ws, _P), self._at(self.es, lo),
                              self._at(self.ms, lo) if S else None, self._at(self.vs, lo) if S else None,
                              self._at(acc, lo), self._at(w, lo), self._at(dec, lo),
                              self._at(self.swords, lo * self.qs.bits // 32), self._at(self.sscales, gs))

    def _apply_chunk(self, x: np.ndarray, ch) -> None:
        lo, hi, _, _, qsc, gs, _ = ch
        lib().ora_apply(ctypes.byref(qsc._c), hi - lo, self._at(self.swords, lo * self.qs.bits // 32),
                        self._at(self.sscales, gs), self._at(x, lo), self._at(self._sscratch[2], lo))

    def set_hparams(self, alpha: float, beta1: float, beta2: float) -> None:
        """alpha_t, beta and theta_t for the following rounds (schedules such as Assumption 2's)."""
        self.cfg.alpha, self.cfg.beta1, self.cfg.beta2 = np.float32(alpha), np.float32(beta1), np.float32(beta2)

    def worker_compress(self, i: int, g: np.ndarray) -> None:
        g = np.ascontiguousarray(g, dtype=np.float32)
        assert g.shape == (self.d,)
        u, dec = self._scratch[i]
        W = self.mode == ADAM_AT_WORKER
        lib().ora_worker_step(ctypes.byref(self.cfg), ctypes.byref(self.qw._c), _ptr(self.gidx), i,
                              self.t, _ptr(g), _ptr(self.m[i]) if W else None,
                              _ptr(self.v[i]) if W else None, _ptr(self.e[i]), _ptr(u), _ptr(dec),
                              _ptr(self.wwords[i]), _ptr(self.wscales[i]))

    def compress_all(self, gs) -> None:
        """All n workers; with threads > 1 the workers (and chunks of whole scale groups of each
        worker's vector, where the groups allow it) run concurrently on host threads."""
        if self.threads == 1:
            for i in range(self.n):
                self.worker_compress(i, gs[i])
            return
        if not self._chunks:
            list(self._pool.map(lambda i: self.worker_compress(i, gs[i]), range(self.n)))
            return
        gs = [np.ascontiguousarray(g, dtype=np.float32) for g in gs]
        assert all(g.shape == (self.d,) for g in gs)
        tasks = [(i, ch) for i in range(self.n) for ch in self._chunks]
        list(self._pool.map(lambda a: self._worker_chunk(a[0], gs[a[0]], a[1]), tasks))

    def server_step(self) -> None:
        if self._chunks:
            list(self._pool.map(self._server_chunk, self._chunks))
            self.up_bits += self.n * self.qw.message_bits(self.d)
            self.down_bits += self.n * self.qs.message_bits(self.d)
            self.t += 1
            return
        ww = (ctypes.c_void_p * self.n)(*[self.wwords[i].ctypes.data for i in range(self.n)])
        ws = (ctypes.c_void_p * self.n)(*[self.wscales[i].ctypes.data for i in range(self.n)])
        acc, w, dec = self._sscratch
        S = self.mode == ADAM_AT_SERVER
        lib().ora_server_step(ctypes.byref(self.cfg), ctypes.byref(self.qw._c), ctypes.byref(self.qs._c),
                              _ptr(self.gidx), self.t, ctypes.cast(ww, _P), ctypes.cast(ws, _P),
                              _ptr(self.es), _ptr(self.ms) if S else None, _ptr(self.vs) if S else None,
                              _ptr(acc), _ptr(w), _ptr(dec), _ptr(self.swords), _ptr(self.sscales))
        # Corollary 1's accounting: every worker uploads one message and receives one broadcast
        self.up_bits += self.n * self.qw.message_bits(self.d)
        self.down_bits += self.n * self.qs.message_bits(self.d)
        self.t += 1

    def apply(self, x: np.ndarray) -> None:
        assert x.dtype == np.float32 and x.flags["C_CONTIGUOUS"] and x.shape == (self.d,)
        if self._chunks:
            list(self._pool.map(lambda ch: self._apply_chunk(x, ch), self._chunks))
            return
        dec = self._sscratch[2]
        lib().ora_apply(ctypes.byref(self.qs._c), self.d, _ptr(self.swords), _ptr(self.sscales),
                        _ptr(x), _ptr(dec))

    def last_input(self, i: int) -> np.ndarray:
        """Worker i's residual-corrected input u of the last compress (scratch; copy it)."""
        return self._scratch[i][0]

    def last_server_input(self) -> np.ndarray:
        """The server's w = avg (+ Adam step) + e_s of the last server step (scratch; copy it)."""
        return self._sscratch[1]

    def server_decoded(self) -> np.ndarray:
        return self.qs.decode(self.swords, self.sscales[: self.qs.n_groups], self.d)

    def worker_decoded(self, i: int) -> np.ndarray:
        return self.qw.decode(self.wwords[i], self.wscales[i][: self.qw.n_groups], self.d)
