"""Failure detection without a GPU fault: the staged server's waits on its stages are bounded and
report EA_E_TIMEOUT through a status word.  ea_selftest_bounded_wait runs that wait on an mbarrier
that nothing arrives on, so it runs out after a short limit; the control completes first.  The
context stays usable afterwards (a round after the timeout matches the oracle)."""
import numpy as np
import pytest
import torch

import paper_2205_14473_gb300 as ea
from paper_2205_14473_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)


def test_wait_with_no_arrival_times_out_and_the_control_does_not():
    s = torch.cuda.current_stream().cuda_stream
    assert ea.ea_selftest_bounded_wait(2_000_000, 0, s) is True    # ~1 ms at 2 GHz, nothing arrives
    assert ea.ea_selftest_bounded_wait(2_000_000, 1, s) is False   # the barrier completes first
    assert ea.ea_selftest_bounded_wait(1, 1, s) is False


def test_argument_checks():
    s = torch.cuda.current_stream().cuda_stream
    for limit, arrive in ((0, 0), (4_000_000_001, 0), (1000, 2)):
        with pytest.raises(ea.EAError) as ex:
            ea.ea_selftest_bounded_wait(limit, arrive, s)
        assert ex.value.status == ea.EA_E_INVAL


def test_context_usable_after_a_timeout():
    from parity import Lockstep

    s = torch.cuda.current_stream().cuda_stream
    assert ea.ea_selftest_bounded_wait(1_000_000, 0, s) is True
    cfg = ea.EAConfig(d=20_000, n=2, qw=W.sign_q(4096), qs=W.sign_q(4096), alpha=1e-3, seed=3)
    L = Lockstep(cfg)
    rng = np.random.default_rng(5)
    x_host = np.zeros(cfg.d, np.float32)
    x_dev = torch.zeros(cfg.d, device="cuda")
    for _ in range(2):
        gs = [rng.standard_normal(cfg.d).astype(np.float32) for _ in range(cfg.n)]
        L.round([torch.from_numpy(g).cuda() for g in gs], gs, x_dev, x_host)
    L.gpu.sync()
