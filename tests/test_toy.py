"""Section 5.1's convex toy, min E||Ax - (x* + xi)||^2 with a 500 x 500 Gaussian A and 10 workers,
run through the oracle: the qualitative claims of Figures 2-3 and the bit counts of the text.
CPU only."""
import numpy as np
import pytest

import oracle as O
from paper_2205_14473_gb300 import workloads as W


def _quant(spec):
    return O.Quantizer(spec.kind, spec.bits, O.group_offsets(W.TOY_D, 0), stochastic=spec.stochastic,
                       pow2_k=spec.pow2_k, pow2_K=spec.pow2_K)


def _run(name, ef, case, T, alpha=1e-4):
    A, xs = W.toy_case(case)
    q = _quant(W.TOY_QUANTIZERS[name])
    orc = O.OracleRound(W.TOY_D, W.TOY_N, q, q, alpha, 0.9, 0.99, 1e-8, error_feedback=ef)
    x = np.zeros(W.TOY_D, np.float32)
    norms = []
    for t in range(T):
        gs = [W.toy_gradient(A, x, xs, W.toy_noise(case, i, t)) for i in range(W.TOY_N)]
        orc.compress_all(gs)
        orc.server_step()
        orc.apply(x)
        if (t + 1) % (T // 4) == 0:
            norms.append(W.toy_full_gradient_norm(A, x, xs))
    return np.array(norms), orc


def test_toy_bits_per_coordinate():
    """Example 1 with k = 1 sends 2 bits a coordinate (plus one scale), Example 2 with k = -17,
    K = -11 sends 4 ("twice more bits")."""
    d = W.TOY_D
    assert _quant(W.TOY_QUANTIZERS["com1"]).message_bits(d) == 2 * d + 32
    assert _quant(W.TOY_QUANTIZERS["com2"]).message_bits(d) == 4 * d
    assert _quant(W.TOY_QUANTIZERS["full"]).message_bits(d) == 32 * d


@pytest.mark.parametrize("case", [0, 1])
def test_toy_error_feedback_claims(case):
    """Error feedback helps the coarse Example 1 quantizer a lot and Example 2 little; with it both
    track the full-precision run; the gradient norm falls."""
    T = 1200
    full, _ = _run("full", True, case, T)
    c1, _ = _run("com1", True, case, T)
    c1_noef, _ = _run("com1", False, case, T)
    c2, _ = _run("com2", True, case, T)
    c2_noef, _ = _run("com2", False, case, T)
    assert np.all(np.diff(full) < 0) and np.all(np.diff(c1) < 0)
    assert c1[-1] < 0.8 * c1_noef[-1]                      # EF helps com1
    assert abs(c2[-1] - c2_noef[-1]) < 0.1 * c2[-1]        # and matters little for com2
    assert c1[-1] < 1.05 * full[-1] and c2[-1] < 1.05 * full[-1]
