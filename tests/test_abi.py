"""The C-ABI boundary without a GPU: the library loads, exports every entry point include/ea.h
declares, sizes workspaces and rejects invalid configurations before any CUDA call."""
import ctypes
import os
import re

import pytest

import paper_2205_14473_gb300 as ea
from paper_2205_14473_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            src = open(os.path.join(ROOT, "include", h)).read()
            names += re.findall(r"^(?:int|const char \*|size_t)\s*\*?\s*(ea_\w+)\s*\(", src, re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(ea_lib):
    names = _declared()
    assert len(names) >= 11
    for n in names:
        assert hasattr(ea_lib, n), n
    assert set(ea.EXPORTED) <= set(names)


def _cfg(**kw):
    base = dict(d=10_000, n=2, qw=W.sign_q(4096), qs=W.sign_q(4096), alpha=1e-3)
    base.update(kw)
    return ea.EAConfig(**base)


def test_workspace_bytes_covers_state(ea_lib):
    for name, w in W.WORKLOADS.items():
        for placement in (ea.ADAM_AT_WORKER, ea.ADAM_AT_SERVER):
            cfg = ea.EAConfig.from_workload(w, placement=placement)
            c, keep = cfg.to_c()
            nbytes = ea.ea_workspace_bytes(c)
            vecs = (3 * w.n + 1) if placement == ea.ADAM_AT_WORKER else (w.n + 3)
            # scaled-sign worker groups that span tiles: one more vector, where residual views are formed
            vecs += int(w.qw.kind == W.Q_SIGN_L1 and w.qw.group <= 0 and w.d > 4096)
            code_bytes = (w.n * w.d * w.qw.bits + w.d * w.qs.bits) / 8
            assert nbytes >= vecs * w.d * 4 + code_bytes
            assert nbytes <= (vecs * w.d * 4 + code_bytes) * 1.01 + 2**22, name
    # the largest workload fits the 288 GB part in both placements
    c5 = W.WORKLOADS["c5"]
    c, keep = ea.EAConfig.from_workload(c5).to_c()
    assert ea.ea_workspace_bytes(c) < 170e9


@pytest.mark.parametrize("bad,status", [
    (dict(d=0), ea.EA_E_INVAL),
    (dict(n=0), ea.EA_E_INVAL),
    (dict(n=2000), ea.EA_E_INVAL),
    (dict(beta1=1.0), ea.EA_E_INVAL),
    (dict(beta2=-0.1), ea.EA_E_INVAL),
    (dict(eps=0.0), ea.EA_E_INVAL),
    (dict(alpha=float("nan")), ea.EA_E_INVAL),
    (dict(placement=7), ea.EA_E_INVAL),
    (dict(qw=W.QuantSpec(W.Q_SIGN_L1, 2, 4096)), ea.EA_E_INVAL),
    (dict(qw=W.QuantSpec(W.Q_UNIFORM_MAX, 3, 4096)), ea.EA_E_UNSUPPORTED),
    (dict(qw=W.QuantSpec(W.Q_SIGN_L1, 1, 4096, stochastic=True)), ea.EA_E_INVAL),
    (dict(qs=W.QuantSpec(W.Q_SIGN_L1, 1, -1, (5000, 4999))), ea.EA_E_INVAL),
    (dict(qs=W.QuantSpec(W.Q_SIGN_L1, 1, -1, (10_000, 0))), ea.EA_E_INVAL),
    (dict(qw=W.pow2_q(-17, -9, 4)), ea.EA_E_INVAL),
    (dict(qw=W.QuantSpec(W.Q_POW2, 4, 0, (), False, -130, -125)), ea.EA_E_INVAL),
    (dict(qw=W.QuantSpec(W.Q_IDENTITY, 16)), ea.EA_E_INVAL),
    (dict(qw=W.QuantSpec(9, 1)), ea.EA_E_INVAL),
])
def test_invalid_configs_rejected(ea_lib, bad, status):
    c, keep = _cfg(**bad).to_c()
    with pytest.raises(ea.EAError) as ex:
        ea.ea_workspace_bytes(c)
    assert ex.value.status == status
    assert str(ex.value)
    # ea_init checks the same before touching the device
    h = ctypes.c_void_p()
    assert ea_lib.ea_init(ctypes.byref(c), 256, 1 << 30, None, ctypes.byref(h)) == status
    assert not h.value


def test_workspace_checks_before_device(ea_lib):
    c, keep = _cfg().to_c()
    need = ea.ea_workspace_bytes(c)
    h = ctypes.c_void_p()
    assert ea_lib.ea_init(ctypes.byref(c), None, need, None, ctypes.byref(h)) == ea.EA_E_WORKSPACE
    assert ea_lib.ea_init(ctypes.byref(c), 4096 + 16, need, None, ctypes.byref(h)) == ea.EA_E_WORKSPACE
    assert ea_lib.ea_init(ctypes.byref(c), 4096, need - 1, None, ctypes.byref(h)) == ea.EA_E_WORKSPACE
    assert b"256-byte" in ea_lib.ea_last_error(None) or b"needs" in ea_lib.ea_last_error(None)


def test_null_handle_calls(ea_lib):
    assert ea_lib.ea_worker_compress(None, 0, 4096) == ea.EA_E_INVAL
    assert ea_lib.ea_server_step(None) == ea.EA_E_INVAL
    assert ea_lib.ea_worker_apply(None, 4096) == ea.EA_E_INVAL
    assert ea_lib.ea_sync_status(None) == ea.EA_E_INVAL
    up = ctypes.c_uint64()
    assert ea_lib.ea_bits_sent(None, ctypes.byref(up), ctypes.byref(up)) == ea.EA_E_INVAL
    assert ea_lib.ea_destroy(None) == 0


def test_product_path_has_no_fallback(monkeypatch, tmp_path):
    """Without libea.so the binding raises instead of computing anything elsewhere."""
    import importlib

    monkeypatch.setattr(ea, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(ea, "_lib", None)
    with pytest.raises(ImportError):
        ea.lib()
    importlib.reload(ea)
