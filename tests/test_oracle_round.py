"""Pins of the oracle's round (Algorithms 1 and 2) against what the paper and mathematics fix.

  * the unrolled moment sums of Lemma 1's proof, m_t = sum_k beta^(t-k) (1-beta) g_k and
    v_t = theta^t eps + sum_k theta^(t-k) (1-theta) g_k^2, with the 32-bit identity quantizer
    ("Ours_full" of Table 2), where the method reduces to the paper's form of Adam;
  * Lemma 1: m_t^2 <= v_t / ((1-gamma)(1-theta)), gamma = beta/theta, every coordinate and round;
  * the error-feedback bookkeeping of both algorithms: Q(u) + e_new = u up to one rounding;
  * the virtual iterates of Notation 1: x~ = x - e_s moves by -avg, x^ = x~ - mean_i e_i moves by
    the mean Adam step -(1/N) sum_i alpha m_i / sqrt(v_i);
  * convergence on the quadratic toy (Section 5.1's problem with A = I);
  * the bits ledger of Corollary 1 (b bits per coordinate plus the scale words).
CPU only.
"""
import numpy as np
import pytest

import oracle as O
from paper_2205_14473_gb300 import workloads as W


def _round(d, n, qw_kind=O.Q_SIGN_L1, qs_kind=O.Q_SIGN_L1, bits_w=1, bits_s=1, group=0,
           mode=O.ADAM_AT_WORKER, alpha=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, **kw):
    qw = O.Quantizer(qw_kind, bits_w, O.group_offsets(d, group))
    qs = O.Quantizer(qs_kind, bits_s, O.group_offsets(d, group))
    return O.OracleRound(d, n, qw, qs, alpha, beta1, beta2, eps, mode=mode, **kw)


def _f(x):
    return float(np.float32(x))


@pytest.mark.parametrize("mode", [O.ADAM_AT_WORKER, O.ADAM_AT_SERVER])
def test_identity_quantizer_is_paper_adam_closed_form(mode):
    """With Q_w = Q_s = identity every residual stays 0 and x follows the paper's Adam exactly:
    no bias correction, eps only as v_0, denominator sqrt(v_t).  Compared, in binary64, with the
    unrolled sums of Lemma 1's proof (relative error bounded by the binary32 roundings)."""
    d, n, T = 257, 3, 60
    alpha, b1, b2, eps = 1e-2, 0.9, 0.99, 1e-8
    orc = _round(d, n, O.Q_IDENTITY, O.Q_IDENTITY, 32, 32, mode=mode, alpha=alpha, beta1=b1,
                 beta2=b2, eps=eps)
    A, B1, B2, E = _f(alpha), _f(b1), _f(b2), _f(eps)
    rng = np.random.default_rng(11)
    # W-mode needs identical worker gradients for x to be one Adam trajectory; S-mode averages
    same = mode == O.ADAM_AT_WORKER
    x = np.zeros(d, np.float32)
    xr = np.zeros(d)
    hist = []
    for t in range(1, T + 1):
        base = (rng.standard_normal(d) * 10 ** rng.uniform(-3, 1)).astype(np.float32)
        gs = [base if same else (base + rng.standard_normal(d).astype(np.float32)) for _ in range(n)]
        gavg = np.mean(np.stack(gs).astype(np.float64), axis=0)
        hist.append(gavg if not same else base.astype(np.float64))
        orc.compress_all(gs)
        orc.server_step()
        orc.apply(x)
        H = np.stack(hist)
        k = np.arange(1, t + 1)[:, None]
        m = ((B1 ** (t - k)) * (1 - B1) * H).sum(0)
        v = B2 ** t * E + ((B2 ** (t - k)) * (1 - B2) * H * H).sum(0)
        xr = xr - A * m / np.sqrt(v)
        if same:
            mo, vo = orc.m[0].astype(np.float64), orc.v[0].astype(np.float64)
        else:
            mo, vo = orc.ms.astype(np.float64), orc.vs.astype(np.float64)
        tol = 4e-7 * t + 1e-6
        assert np.all(np.abs(mo - m) <= tol * np.abs(H).max(0).clip(1e-30) + 1e-30)
        np.testing.assert_allclose(vo, v, rtol=tol)
        np.testing.assert_allclose(x, xr, rtol=tol * 10, atol=A * tol * t)
        assert np.all(orc.e == 0) and np.all(orc.es == 0)
    # with identity the message is 32 bits per coordinate and no scale words
    assert orc.up_bits == T * n * d * 32 and orc.down_bits == T * n * d * 32


def test_lemma1_moment_bound_every_round():
    """Lemma 1: (m_t)^2 <= v_t / ((1 - gamma)(1 - theta)) with gamma = beta / theta < 1."""
    d, n, T = 4096, 2, 40
    b1, b2 = 0.9, 0.999
    orc = _round(d, n, alpha=1e-3, beta1=b1, beta2=b2, group=512)
    rng = np.random.default_rng(2)
    gamma = _f(b1) / _f(b2)
    for t in range(T):
        scale = 10 ** rng.uniform(-4, 2)
        orc.compress_all([(rng.standard_t(3, d) * scale).astype(np.float32) for _ in range(n)])
        orc.server_step()
        m, v = orc.m.astype(np.float64), orc.v.astype(np.float64)
        assert np.all(m * m <= v / ((1 - gamma) * (1 - _f(b2))) * (1 + 1e-5))


@pytest.mark.parametrize("kind,bits,stoch", [(O.Q_SIGN_L1, 1, False), (O.Q_UNIFORM_MAX, 4, True),
                                             (O.Q_UNIFORM_MAX, 8, False), (O.Q_POW2, 4, False)])
@pytest.mark.parametrize("mode", [O.ADAM_AT_WORKER, O.ADAM_AT_SERVER])
def test_error_feedback_invariant(kind, bits, stoch, mode):
    """Algorithm 2's e_{t+1} = u - Q_w(u) and Algorithm 1's e_{t+1} = w - Q_s(w): the decoded
    message plus the new residual reproduces the quantized input within half an ulp of e."""
    d, n = 3000, 3
    offs = O.group_offsets(d, 1024)
    kw = dict(pow2_k=-17, pow2_K=-11) if kind == O.Q_POW2 else {}
    qw = O.Quantizer(kind, bits, offs, stochastic=stoch, **kw)
    qs = O.Quantizer(kind, bits, offs, **kw)
    orc = O.OracleRound(d, n, qw, qs, 1e-4, 0.9, 0.999, 1e-8, seed=5, mode=mode)
    rng = np.random.default_rng(4)
    for t in range(6):
        gs = [(rng.standard_normal(d) * 1e-3).astype(np.float32) for _ in range(n)]
        for i in range(n):
            orc.worker_compress(i, gs[i])
            u = orc.last_input(i).astype(np.float64)
            dec = orc.worker_decoded(i).astype(np.float64)
            e = orc.e[i].astype(np.float64)
            ulp = np.spacing(np.abs(orc.e[i])).astype(np.float64)
            assert np.all(np.abs(dec + e - u) <= 0.5 * ulp)
        orc.server_step()
        w = orc.last_server_input().astype(np.float64)
        dec = orc.server_decoded().astype(np.float64)
        ulp = np.spacing(np.abs(orc.es)).astype(np.float64)
        assert np.all(np.abs(dec + orc.es.astype(np.float64) - w) <= 0.5 * ulp)


def test_virtual_iterates_notation1():
    """x~_t = x_t - e_t moves by minus the averaged (decoded) worker messages, and
    x^_t = x~_t - (1/N) sum_i e_t^(i) moves by minus the mean Adam step (1/N) sum_i alpha m/sqrt(v):
    the quantization errors cancel exactly in the virtual iterates (up to binary32 rounding)."""
    d, n, T = 5000, 4, 30
    orc = _round(d, n, alpha=1e-3, group=1000)
    rng = np.random.default_rng(9)
    x = rng.standard_normal(d).astype(np.float32)
    xt_prev = x.astype(np.float64) - orc.es
    xh_prev = xt_prev - orc.e.astype(np.float64).mean(0)
    for t in range(T):
        gs = [rng.standard_normal(d).astype(np.float32) for _ in range(n)]
        e_old = orc.e.astype(np.float64).copy()
        steps, decs = [], []
        for i in range(n):
            orc.worker_compress(i, gs[i])
            # the Adam step alpha m / sqrt(v), from the moments (pinned by the closed-form test)
            m, v = orc.m[i].astype(np.float64), orc.v[i].astype(np.float64)
            steps.append(_f(1e-3) * m / np.sqrt(v))
            decs.append(orc.worker_decoded(i).astype(np.float64))
        orc.server_step()
        orc.apply(x)
        xt = x.astype(np.float64) - orc.es
        xh = xt - orc.e.astype(np.float64).mean(0)
        mag = 2e-6 * (np.abs(x).astype(np.float64) + 1e-3)
        np.testing.assert_allclose(xt, xt_prev - np.mean(decs, 0), rtol=0, atol=mag.max())
        np.testing.assert_allclose(xh, xh_prev - np.mean(steps, 0), rtol=0, atol=mag.max())
        xt_prev, xh_prev = xt, xh


def test_quadratic_toy_converges():
    """Section 5.1's toy with A = I (the c2 recipe at a smaller dimension): ||x - x*|| falls
    steadily and ends far below its start."""
    w = W.WORKLOADS["c2"]
    d, T = 20_000, 600
    orc = _round(d, w.n, alpha=w.alpha, threads=1)
    xs = W.xstar_host(w, d)
    x = np.zeros(d, np.float32)
    dist = [np.linalg.norm(x - xs)]
    for t in range(T):
        gs = [W.quadratic_gradient(x, xs, W.gradient_host(w, i, t, d)) for i in range(w.n)]
        orc.compress_all(gs)
        orc.server_step()
        orc.apply(x)
        dist.append(np.linalg.norm(x - xs))
    dist = np.array(dist)
    assert dist[-1] < 0.1 * dist[0]
    assert np.all(dist[50:301:50] < dist[0:251:50])  # decreasing in 50-round windows


def test_bits_ledger_closed_form():
    """Corollary 1's accounting: per round every worker sends d*b_w bits plus 32 per scale word and
    receives the broadcast of d*b_s bits plus its scale words."""
    d, n = 10_001, 3
    qw = O.Quantizer(O.Q_UNIFORM_MAX, 4, O.group_offsets(d, 4096), stochastic=True)
    qs = O.Quantizer(O.Q_SIGN_L1, 1, O.group_offsets(d, 0))
    orc = O.OracleRound(d, n, qw, qs, 1e-3, 0.9, 0.999, 1e-8)
    rng = np.random.default_rng(0)
    T = 3
    for t in range(T):
        orc.compress_all([rng.standard_normal(d).astype(np.float32) for _ in range(n)])
        orc.server_step()
    assert orc.up_bits == T * n * (d * 4 + 32 * 3)
    assert orc.down_bits == T * n * (d * 1 + 32 * 1)


def test_no_error_feedback_ablation_keeps_residuals_zero():
    """The "_err" rows of Table 2: without error feedback the residuals stay 0 and each message is
    the quantized fresh step."""
    d, n = 2048, 2
    orc = _round(d, n, group=512, error_feedback=False)
    rng = np.random.default_rng(1)
    for t in range(3):
        orc.compress_all([rng.standard_normal(d).astype(np.float32) for _ in range(n)])
        orc.server_step()
        assert np.all(orc.e == 0) and np.all(orc.es == 0)


def test_textbook_form_reduces_to_torch_adam():
    """adam_form = 1 (bias correction, eps in the denominator, v_0 = 0) with the 32-bit identity
    quantizer is plain Adam: x follows torch.optim.Adam, a library implementation, within binary32
    rounding (the two evaluate the same expression in different operation orders)."""
    torch = pytest.importorskip("torch")
    d, T = 300, 60
    a, b1, b2, eps = _f(3e-3), _f(0.9), _f(0.99), _f(1e-3)  # eps comparable to sqrt(v^): it matters
    orc = _round(d, 1, O.Q_IDENTITY, O.Q_IDENTITY, 32, 32, alpha=a, beta1=b1, beta2=b2, eps=eps, adam_form=1)
    rng = np.random.default_rng(21)
    x0 = rng.standard_normal(d).astype(np.float32)
    x = x0.copy()
    p = torch.nn.Parameter(torch.from_numpy(x0.copy()))
    opt = torch.optim.Adam([p], lr=a, betas=(b1, b2), eps=eps, foreach=False)
    for t in range(T):
        g = (rng.standard_normal(d) * 10 ** rng.uniform(-4, 0)).astype(np.float32)
        orc.compress_all([g])
        orc.server_step()
        orc.apply(x)
        p.grad = torch.from_numpy(g.copy())
        opt.step()
        np.testing.assert_allclose(x, p.detach().numpy(), rtol=2e-6, atol=a * 2e-5 * (t + 1))
    assert np.abs(x - x0).max() > 10 * a  # it moved


def test_schedules_follow_the_product_form():
    """alpha_t, beta and theta_t changed every round (Assumption 2 fixes them from T; the experiments
    decay alpha in steps).  With the identity quantizer the paper's moments are the product-form
    sums  v_t = (prod_{j<=t} theta_j) eps + sum_{k<=t} (prod_{k<j<=t} theta_j) (1 - theta_k) g_k^2
    and   m_t = sum_{k<=t} (prod_{k<j<=t} beta_j) (1 - beta_k) g_k,  and x moves by alpha_t m_t/sqrt(v_t)."""
    d, T = 200, 40
    eps = _f(1e-8)
    orc = _round(d, 1, O.Q_IDENTITY, O.Q_IDENTITY, 32, 32, alpha=1e-2, beta1=0.9, beta2=0.99, eps=eps)
    rng = np.random.default_rng(8)
    x = np.zeros(d, np.float32)
    xr = np.zeros(d)
    al, be, th, G = [], [], [], []
    for t in range(1, T + 1):
        al.append(_f(1e-2 / np.sqrt(t)))
        be.append(_f(0.9 - 0.3 * (t % 3 == 0)))
        th.append(_f(1 - 0.5 / (t + 1)))
        orc.set_hparams(al[-1], be[-1], th[-1])
        g = rng.standard_normal(d).astype(np.float32)
        G.append(g.astype(np.float64))
        orc.compress_all([g])
        orc.server_step()
        orc.apply(x)
        v = np.prod(th) * eps + sum(np.prod(th[k + 1:]) * (1 - th[k]) * G[k] ** 2 for k in range(t))
        m = sum(np.prod(be[k + 1:]) * (1 - be[k]) * G[k] for k in range(t))
        xr = xr - al[-1] * m / np.sqrt(v)
        np.testing.assert_allclose(orc.v[0], v, rtol=4e-7 * t + 1e-6)
        assert np.all(np.abs(orc.m[0] - m) <= (4e-7 * t + 1e-6) * np.max(np.abs(G[: t]), axis=0))
        np.testing.assert_allclose(x, xr, rtol=1e-5, atol=1e-7 * t)


@pytest.mark.parametrize("qw,qs", [
    (W.uniform_q(4, 4096, True), W.uniform_q(8, 4096, False)),
    (W.sign_q(-1, (9408, 64, 64, 36864, 64, 4096, 5120, 1000)), W.sign_q(-1, (9408, 64, 64, 36864, 64, 4096, 5120,
                                                                               1000))),
    (W.pow2_q(-17, -11, 4), W.sign_q(4096)),
    (W.identity_q(), W.uniform_q(4, 4096, True)),
])
@pytest.mark.parametrize("mode", [O.ADAM_AT_WORKER, O.ADAM_AT_SERVER])
def test_threaded_chunks_equal_one_thread(qw, qs, mode):
    """The oracle's multi-threaded driver (workers and chunks of whole scale groups on host threads)
    gives the single-threaded results bit for bit: the chunking only splits separable work."""
    d = 56_680 if qw.group < 0 else 41_000
    runs = []
    for threads in (1, 6):
        def q(s):
            offs = O.group_offsets(d, s.group, s.segments if s.group < 0 else None) if s.kind in (1, 2) else \
                O.group_offsets(d, 0)
            return O.Quantizer(s.kind, s.bits, offs, s.stochastic, s.pow2_k, s.pow2_K)
        orc = O.OracleRound(d, 3, q(qw), q(qs), 1e-3, 0.9, 0.999, 1e-8, seed=9, mode=mode, threads=threads)
        rng = np.random.default_rng(4)
        x = rng.standard_normal(d).astype(np.float32)
        for _ in range(3):
            orc.compress_all([rng.standard_normal(d).astype(np.float32) for _ in range(3)])
            orc.server_step()
            orc.apply(x)
        runs.append((orc, x))
    (a, xa), (b, xb) = runs
    assert len(b._chunks) > 1
    for k in ("e", "m", "v", "es", "ms", "vs", "wwords", "wscales", "swords", "sscales"):
        assert np.array_equal(getattr(a, k), getattr(b, k)), k
    assert np.array_equal(xa, xb)
    assert (a.up_bits, a.down_bits, a.t) == (b.up_bits, b.down_bits, b.t)
