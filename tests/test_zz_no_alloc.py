"""ea_worker_compress_noalloc, the worker compress for callers that cannot allocate device memory
(no handle, no workspace; its scratch is a fixed array compiled into the library), against the
handle-based ea_worker_compress on the same inputs, two rounds in a row.  Collected last, and
independent of every other test: it builds what it needs and runs alone or after the others."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2205_14473_gb300 as ea
from paper_2205_14473_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ATOL, RTOL = 1e-7, 1e-5  # the tolerance of the other parity tests


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2205_14473_gb300 import build as B

    B.build()
    torch.cuda.set_device(0)
    yield
    torch.cuda.synchronize()


def _close(a: torch.Tensor, b: torch.Tensor) -> bool:
    a, b = a.double(), b.double()
    return bool(((a - b).abs() <= ATOL + RTOL * b.abs()).all())


@pytest.mark.parametrize("qw,placement", [
    (W.sign_q(0), ea.ADAM_AT_WORKER),
    (W.uniform_q(4, 0, True), ea.ADAM_AT_WORKER),
    (W.sign_q(0), ea.ADAM_AT_SERVER),
])
@pytest.mark.parametrize("d", [3000, 100_003])
def test_noalloc_matches_handle_path(qw, placement, d):
    dev = torch.device("cuda", 0)
    cfg = ea.EAConfig(d=d, n=1, qw=qw, qs=W.sign_q(0), alpha=1e-3, placement=placement, seed=77)
    c, keep = cfg.to_c()
    ref = ea.EARound(cfg)                       # the existing entry point, through its handle
    stream = torch.cuda.current_stream(dev)
    # the caller's own state and message buffers for the allocation-free call
    m = torch.zeros(d, device=dev)
    v = torch.full((d,), cfg.eps, device=dev)
    e = torch.zeros(d, device=dev)
    n_words = 4 * (-(-d * qw.bits // 128))
    codes = torch.zeros(n_words, dtype=torch.int32, device=dev)
    scales = torch.zeros(4, device=dev)
    gen = torch.Generator(device=dev).manual_seed(5)
    x = torch.zeros(d, device=dev)
    for t in range(2):
        g = torch.randn(d, generator=gen, device=dev) * 10 ** (t - 1)
        ref.worker_compress(0, g)
        ea.ea_worker_compress_noalloc(c, 0, t, g.data_ptr(), m.data_ptr(), v.data_ptr(), e.data_ptr(),
                                      codes.data_ptr(), scales.data_ptr(), stream.cuda_stream)
        torch.cuda.synchronize()
        nw = -(-d * qw.bits // 32)
        assert torch.equal(codes[:nw], ref.view(ea.EA_VIEW_CODES_WORKER, 0)[:nw]), f"round {t}: codes differ"
        assert _close(scales[:1], ref.view(ea.EA_VIEW_SCALES_WORKER, 0)[:1]), f"round {t}: scale differs"
        assert _close(e, ref.view(ea.EA_VIEW_E_WORKER, 0)), f"round {t}: residual differs"
        if placement == ea.ADAM_AT_WORKER:
            assert _close(m, ref.view(ea.EA_VIEW_M, 0)) and _close(v, ref.view(ea.EA_VIEW_V, 0))
        ref.server_step()                       # advance the handle's round
        ref.apply(x)
    ref.sync()


def test_noalloc_rejects_what_it_cannot_do():
    dev = torch.device("cuda", 0)
    buf = torch.zeros(1024, device=dev)
    p = buf.data_ptr()
    s = torch.cuda.current_stream(dev).cuda_stream
    big = ea.EAConfig(d=16384 * 4096 + 1, n=1, qw=W.sign_q(0), qs=W.sign_q(0), alpha=1e-3)
    c, keep = big.to_c()
    with pytest.raises(ea.EAError) as ex:
        ea.ea_worker_compress_noalloc(c, 0, 0, p, p, p, p, p, p, s)
    assert ex.value.status == ea.EA_E_INVAL and "limit" in str(ex.value)
    blk = ea.EAConfig(d=1000, n=1, qw=W.sign_q(4096), qs=W.sign_q(0), alpha=1e-3)
    c, keep = blk.to_c()
    with pytest.raises(ea.EAError) as ex:
        ea.ea_worker_compress_noalloc(c, 0, 0, p, p, p, p, p, p, s)
    assert ex.value.status == ea.EA_E_UNSUPPORTED
