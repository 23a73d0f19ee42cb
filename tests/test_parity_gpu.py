"""GPU parity: the CUDA library, called through its C-ABI binding, against the oracle on the same
seeded inputs, every round (see tests/parity.py for the tolerances)."""
import numpy as np
import pytest
import torch

import paper_2205_14473_gb300 as ea
from paper_2205_14473_gb300 import workloads as W

from parity import Lockstep, expected_bits

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _run_host(cfg: ea.EAConfig, rounds: int, seed: int = 0, grad_scale: float = 1.0, x_scale: float = 1.0):
    L = Lockstep(cfg)
    rng = np.random.default_rng(seed)
    x_host = (rng.standard_normal(cfg.d) * x_scale).astype(np.float32)
    x_dev = torch.from_numpy(x_host.copy()).cuda()
    for t in range(rounds):
        scale = grad_scale * (10 ** rng.uniform(-1, 1))
        gs = [(rng.standard_normal(cfg.d) * scale).astype(np.float32) for _ in range(cfg.n)]
        L.round([torch.from_numpy(g).cuda() for g in gs], gs, x_dev, x_host)
    assert L.gpu.bits_sent() == expected_bits(cfg, rounds)
    return L


# ----------------------------------------------------------------------- sizes and edge cases

@pytest.mark.parametrize("d", [1, 3, 31, 32, 33, 4095, 4096, 4097, 12289, 20_000])
@pytest.mark.parametrize("group", [4096, 0])
def test_ragged_sizes(d, group):
    cfg = ea.EAConfig(d=d, n=3, qw=W.sign_q(group), qs=W.sign_q(group), alpha=1e-3, seed=d)
    _run_host(cfg, 3, seed=d)


@pytest.mark.parametrize("n", [1, 2, 5, 8, 9, 16, 33])
@pytest.mark.parametrize("group", [4096, 0])
def test_worker_counts(n, group):
    """Worker counts around the server's 8-worker sign table, with tile and whole-vector scales
    (33 one-bit workers no longer fit the lazy broadcast's shared-memory staging)."""
    cfg = ea.EAConfig(d=9000, n=n, qw=W.sign_q(group), qs=W.sign_q(group), alpha=1e-2)
    _run_host(cfg, 4, seed=n)


@pytest.mark.parametrize("placement", [ea.ADAM_AT_WORKER, ea.ADAM_AT_SERVER])
@pytest.mark.parametrize("ef", [True, False])
@pytest.mark.parametrize("group", [4096, 0, 1000])
def test_placement_and_error_feedback(placement, ef, group):
    cfg = ea.EAConfig(d=15_000, n=3, qw=W.sign_q(group), qs=W.sign_q(group), alpha=1e-3, placement=placement,
                      error_feedback=ef, seed=11)
    _run_host(cfg, 4, seed=3)


_SEGS = (7, 1, 4096, 64, 5000, 3, 8192, 100, 11)


@pytest.mark.parametrize("qw,qs,gs", [
    (W.uniform_q(4, 4096, True), W.uniform_q(8, 4096, False), 1e-3),      # the c4 pair
    (W.uniform_q(2, 0, False), W.uniform_q(2, 0, True), 1.0),             # Example 1 with k = 1
    (W.uniform_q(16, 1000, True), W.uniform_q(16, 4096, False), 1.0),
    (W.QuantSpec(W.Q_UNIFORM_MAX, 8, -1, _SEGS), W.sign_q(-1, _SEGS), 1.0),
    (W.pow2_q(-17, -11, 4), W.pow2_q(-17, -11, 4), 1e-4),                 # Example 2, the paper's k, K
    (W.pow2_q(-20, -5, 8), W.sign_q(4096), 1e-3),
    (W.identity_q(), W.identity_q(), 1.0),                                # "Ours_full"
    (W.sign_q(4096), W.uniform_q(4, 0, True), 1.0),
    (W.identity_q(), W.sign_q(8192), 1.0),
    (W.uniform_q(4, 6000, True), W.sign_q(6000), 1e-3),                 # blocks longer than a tile, not 2^k
])
@pytest.mark.parametrize("placement", [ea.ADAM_AT_WORKER, ea.ADAM_AT_SERVER])
def test_quantizer_kinds(qw, qs, gs, placement):
    d = sum(_SEGS)
    cfg = ea.EAConfig(d=d, n=3, qw=qw, qs=qs, alpha=1e-3, placement=placement, seed=5)
    _run_host(cfg, 4, seed=9, grad_scale=gs)


@pytest.mark.parametrize("case,placement", [
    ("grid_points", ea.ADAM_AT_WORKER), ("grid_points", ea.ADAM_AT_SERVER),
    ("tiny", ea.ADAM_AT_WORKER), ("tiny", ea.ADAM_AT_SERVER),
    ("huge", ea.ADAM_AT_WORKER), ("huge", ea.ADAM_AT_SERVER),
])
def test_uniform_grid_boundaries_and_scale_range(case, placement):
    """Example 1's encode away from its common case: inputs on the grid and exact zeros, where
    y = z L falls on an integer (the stochastic rule's boundary), and group scales below 2^-125
    (subnormal inputs) or above 2^125, outside the range of the division-free index."""
    d, n = 10_000, (2 if case == "huge" else 3)
    alpha = {"grid_points": 1e-3, "tiny": 1e-41, "huge": 1.5e37 if placement == ea.ADAM_AT_WORKER else 1e-3}[case]
    cfg = ea.EAConfig(d=d, n=n, qw=W.uniform_q(4, 4096, True), qs=W.uniform_q(8, 1000, False), alpha=alpha,
                      placement=placement, seed=21)
    L = Lockstep(cfg)
    rng = np.random.default_rng(23)
    x_host = np.zeros(d, np.float32)
    x_dev = torch.zeros(d, device="cuda")
    for t in range(3):
        gs = []
        for _ in range(n):
            if case == "grid_points":
                g = (rng.integers(-7, 8, d) / 7.0 * (rng.random(d) < 0.5)).astype(np.float32)
            elif placement == ea.ADAM_AT_WORKER:  # the step alpha m / sqrt(v) carries alpha's scale
                g = rng.standard_normal(d).astype(np.float32)
            else:                                 # the workers quantize g + e itself
                g = (rng.standard_normal(d) * (1e-41 if case == "tiny" else 2e37)).astype(np.float32)
            gs.append(g)
        rep = L.round([torch.from_numpy(g).cuda() for g in gs], gs, x_dev, x_host)
        assert rep.code_mismatches == 0, f"round {t}: {rep.code_mismatches} codes differ"
    scales = L.gpu.view(ea.EA_VIEW_SCALES_WORKER, 0)[:3].double().abs()
    if case == "tiny":
        assert bool((scales < 2.0 ** -125).all()) and bool((scales > 0).all())
    elif case == "huge":
        assert bool((scales > 2.0 ** 125).all()) and bool(torch.isfinite(scales).all())


@pytest.mark.parametrize("qw,qs,placement", [
    (W.uniform_q(4, 4096, True), W.pow2_q(-20, -5, 8), ea.ADAM_AT_WORKER),
    (W.sign_q(4096), W.identity_q(), ea.ADAM_AT_WORKER),
    (W.uniform_q(4, 4096, True), W.uniform_q(8, 4096, False), ea.ADAM_AT_SERVER),
])
def test_staged_server_several_tiles_per_cta(qw, qs, placement):
    """d large enough that every persistent server CTA runs several tiles through its ring of
    stages (the per-tile decode tables are rebuilt between tiles), with a ragged last tile."""
    d = 4096 * 152 * 3 * 2 + 777
    cfg = ea.EAConfig(d=d, n=3, qw=qw, qs=qs, alpha=1e-3, placement=placement, seed=31)
    _run_host(cfg, 2, seed=37, grad_scale=1e-3)


def test_two_pass_scale_beyond_the_grouped_capacity():
    """A whole-vector scale over 12.3 million coordinates: more tiles than the one-pass grouped
    kernels hold in shared memory at once (about 1,800 on a GB300).  The uniform-grid broadcast
    takes the two-pass scale (stash, finalize, encode: three launches); the scaled-sign worker
    messages take the lazy pass (codes with the partial norms: one launch each, and one finalize
    for all of them)."""
    d = 3000 * 4096 + 3
    cfg = ea.EAConfig(d=d, n=2, qw=W.sign_q(0), qs=W.uniform_q(8, 0, False), alpha=1e-3, seed=41)
    L = _run_host(cfg, 3, seed=43)
    assert L.gpu.launches_per_round == 2 + 1 + 3 + 1


@pytest.mark.parametrize("qw,qs,launches", [(W.sign_q(0), W.sign_q(0), 3 + 1 + 2 + 1),
                                           (W.uniform_q(4, 0, True), W.uniform_q(8, 1000, False), 3 * 1 + 1 + 1)])
def test_grouped_scales_one_launch_per_message(qw, qs, launches):
    """Scale groups that span tiles (74 tiles): uniform-grid messages take the one-pass grouped
    kernels (one tile per worker CTA, one launch each); scaled-sign messages take the lazy pass (the
    signs with the partial norms; one finalize forms the scales of all worker messages, another
    the broadcast's)."""
    cfg = ea.EAConfig(d=300_001, n=3, qw=qw, qs=qs, alpha=1e-3, seed=45)
    L = _run_host(cfg, 3, seed=47)
    assert L.gpu.launches_per_round == launches


@pytest.mark.parametrize("qw,qs,placement,launches", [
    (W.sign_q(0), W.sign_q(0), ea.ADAM_AT_WORKER, 3 + 1 + 2 + 1),
    (W.uniform_q(4, 0, True), W.uniform_q(8, 0, False), ea.ADAM_AT_SERVER, 3 * 3 + 1 + 1),
    (W.uniform_q(4, 0, True), W.uniform_q(8, 0, False), ea.ADAM_AT_WORKER, 3 * 3 + 1 + 1),
    (W.sign_q(-1, (1_500_007, 64, 2_000_000, 128, 900_001)), W.sign_q(-1, (1_500_007, 64, 2_000_000, 128, 900_001)),
     ea.ADAM_AT_WORKER, 3 + 1 + 2 + 1),
    (W.sign_q(-1, (1_500_007, 64, 2_000_000, 128, 900_001)), W.sign_q(-1, (1_500_007, 64, 2_000_000, 128, 900_001)),
     ea.ADAM_AT_SERVER, 3 + 1 + 2 + 1),
])
def test_grouped_broadcast_with_several_tiles_per_cta(qw, qs, placement, launches):
    """4.4 million coordinates (1,075 tiles).  A uniform-grid broadcast takes the grouped kernel,
    whose CTAs each hold several tiles of one wave, and the worker messages the two-pass scale; a
    scaled-sign broadcast and scaled-sign worker messages take the lazy pass (whole vector, and
    segments with tiles that hold several groups)."""
    d = 4_400_200
    cfg = ea.EAConfig(d=d, n=3, qw=qw, qs=qs, alpha=1e-3, placement=placement, seed=49)
    L = _run_host(cfg, 3, seed=51)
    assert L.gpu.launches_per_round == launches


@pytest.mark.parametrize("group", [0, -1])
def test_lazy_views_mid_round_change_nothing(group):
    """Lazy scaled-sign messages: viewing a worker's scales and residual between its compress and the
    server step forms them early (the view matches the values after the round), and the state of a
    handle viewed that way stays bit-identical to that of one never viewed."""
    d = 50_003
    segs = (20_000, 64, 29_939) if group < 0 else ()
    q = W.sign_q(group, segs) if group < 0 else W.sign_q(0)
    cfg = ea.EAConfig(d=d, n=3, qw=q, qs=q, alpha=1e-3, seed=5)
    a, b = ea.EARound(cfg), ea.EARound(cfg)
    gen = torch.Generator(device="cuda").manual_seed(7)
    xa, xb = torch.zeros(d, device="cuda"), torch.zeros(d, device="cuda")
    for t in range(4):
        g = [torch.randn(d, device="cuda", generator=gen) for _ in range(cfg.n)]
        for i in range(cfg.n):
            a.worker_compress(i, g[i])
            b.worker_compress(i, g[i])
        mid = [(a.view(ea.EA_VIEW_SCALES_WORKER, i).clone(), a.view(ea.EA_VIEW_E_WORKER, i)[:d].clone())
               for i in range(cfg.n)]
        for r, x in ((a, xa), (b, xb)):
            r.server_step()
            r.apply(x)
        torch.cuda.synchronize()
        for i in range(cfg.n):
            assert torch.equal(a.view(ea.EA_VIEW_SCALES_WORKER, i), mid[i][0])
            assert torch.equal(a.view(ea.EA_VIEW_E_WORKER, i)[:d], mid[i][1])
            for v in (ea.EA_VIEW_CODES_WORKER, ea.EA_VIEW_SCALES_WORKER, ea.EA_VIEW_E_WORKER):
                assert torch.equal(a.view(v, i), b.view(v, i))
        for v in (ea.EA_VIEW_CODES_SERVER, ea.EA_VIEW_SCALES_SERVER, ea.EA_VIEW_E_SERVER):
            assert torch.equal(a.view(v), b.view(v))
        assert torch.equal(xa, xb)
    assert a.launches_per_round == cfg.n + 1 + 2 + 1


def test_replicas_are_identical_and_protocol():
    cfg = ea.EAConfig(d=10_000, n=2, qw=W.sign_q(4096), qs=W.sign_q(4096), alpha=1e-3)
    rnd = ea.EARound(cfg)
    g = torch.randn(10_000, device="cuda")
    x1 = torch.randn(10_000, device="cuda")
    x2 = x1.clone()
    with pytest.raises(ea.EAError) as ex:
        rnd.apply(x1)
    assert ex.value.status == ea.EA_E_ORDER
    rnd.worker_compress(0, g)
    with pytest.raises(ea.EAError) as ex:
        rnd.worker_compress(0, g)
    assert ex.value.status == ea.EA_E_ORDER
    with pytest.raises(ea.EAError) as ex:
        rnd.server_step()
    assert ex.value.status == ea.EA_E_ORDER
    gbuf = torch.empty(10_004, device="cuda")
    with pytest.raises(ea.EAError) as ex:
        ea.ea_worker_compress(rnd.h, 1, gbuf.data_ptr() + 4)
    assert ex.value.status == ea.EA_E_ALIGN
    with pytest.raises(ea.EAError):
        rnd.worker_compress(2, g)
    rnd.worker_compress(1, g)
    rnd.server_step()
    rnd.apply(x1)
    rnd.apply(x2)
    rnd.sync()
    assert torch.equal(x1, x2)
    assert rnd.t == 1


# ------------------------------------------------------------------------- the five workloads

def _dev_grads(w: W.Workload, t: int, bufs):
    for i, b in enumerate(bufs):
        W.gradient_device(w, i, t, b)
    return bufs


def test_c1_full():
    w = W.WORKLOADS["c1"]
    cfg = ea.EAConfig.from_workload(w)
    L = Lockstep(cfg)
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(w.d, np.float32)
    bufs = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    for t in range(w.rounds):
        _dev_grads(w, t, bufs)
        L.round(bufs, [L.host(b) for b in bufs], x_dev, x_host)
    assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (2_622_720, 2_622_720)
    assert L.gpu.launches_per_round == w.n + 1 + 2 + 1  # scaled-sign messages: the lazy pass + finalize


def test_c2_quadratic_toy_full():
    """The quadratic toy at d = 1e6, n = 8, all 1,000 rounds; both sides form g = (x - x*) + 0.1 xi
    from their own x; ||x - x*|| decreases."""
    w = W.WORKLOADS["c2"]
    cfg = ea.EAConfig.from_workload(w)
    L = Lockstep(cfg)
    xs_host = W.xstar_host(w)
    xs_dev = torch.from_numpy(xs_host).cuda()
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(w.d, np.float32)
    noise = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    dist = [float(np.linalg.norm(x_host - xs_host))]
    for t in range(w.rounds):
        _dev_grads(w, t, noise)
        g_dev = [W.quadratic_gradient(x_dev, xs_dev, nz) for nz in noise]
        g_host = [W.quadratic_gradient(x_host, xs_host, L.host(nz)) for nz in noise]
        L.round(g_dev, g_host, x_dev, x_host)
        if (t + 1) % 50 == 0:
            dist.append(float(torch.linalg.vector_norm(x_dev - xs_dev)))
    assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (8_000_256_000, 8_000_256_000)
    assert dist[-1] < 0.1 * dist[0]
    assert all(b < a for a, b in zip(dist[:6], dist[1:7]))


@pytest.mark.parametrize("placement,rounds", [(ea.ADAM_AT_WORKER, 100), (ea.ADAM_AT_SERVER, 10)])
def test_c3_resnet18_all_tensors(placement, rounds):
    """All 62 ResNet-18 tensors (per-tensor scales, d = 11,689,512, n = 16) against the full oracle:
    all 100 rounds in the paper's placement, the first 10 with Adam at the server."""
    w = W.WORKLOADS["c3"]
    cfg = ea.EAConfig.from_workload(w, placement=placement)
    L = Lockstep(cfg)
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(w.d, np.float32)
    bufs = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    for t in range(rounds):
        _dev_grads(w, t, bufs)
        L.round(bufs, [L.host(b) for b in bufs], x_dev, x_host)
    assert L.total_mismatch == 0
    # per-tensor scales: every message in the lazy pass (codes and partial norms), one finalize for
    # the worker messages' scales and one for the broadcast's
    assert L.gpu.launches_per_round == w.n + 1 + 2 + 1
    if rounds == w.rounds:
        assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (18_706_393_600, 18_706_393_600)


def test_c4_full_oracle_all_rounds():
    """c4 (d = 1.1e8, n = 8, 4-bit stochastic / 8-bit grid, 4096-block scales) in the paper's
    placement against the full oracle: every coordinate of every message and state, all 50 rounds."""
    w = W.WORKLOADS["c4"]
    cfg = ea.EAConfig.from_workload(w, placement=ea.ADAM_AT_WORKER)
    L = Lockstep(cfg)
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(w.d, np.float32)
    bufs = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    for t in range(w.rounds):
        _dev_grads(w, t, bufs)
        L.round(bufs, [L.host(b) for b in bufs], x_dev, x_host)
    assert L.total_mismatch == 0
    assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (176_343_756_800, 352_343_756_800)
    del L, bufs, x_dev
    torch.cuda.empty_cache()


def test_c4_server_placement_sampled_blocks_all_rounds():
    """c4 with Adam at the server, all 50 rounds at full size; the oracle follows 1,024 of the
    26,856 blocks (the round is separable by 4096-block), including the first and the ragged last."""
    w = W.WORKLOADS["c4"]
    cfg = ea.EAConfig.from_workload(w, placement=ea.ADAM_AT_SERVER)
    L = Lockstep(cfg, sample_groups=W.sample_blocks(w, 1024))
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(L.d_o, np.float32)
    bufs = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    for t in range(w.rounds):
        _dev_grads(w, t, bufs)
        L.round(bufs, [L.host(b) for b in bufs], x_dev, x_host)
    assert L.total_mismatch == 0
    assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (176_343_756_800, 352_343_756_800)
    del L, bufs, x_dev
    torch.cuda.empty_cache()


@pytest.mark.parametrize("placement", [ea.ADAM_AT_WORKER, ea.ADAM_AT_SERVER])
def test_c5_sampled_blocks_all_rounds(placement):
    """d = 1.558e9, n = 8 on one GPU (W: ~213 GB resident, S: ~126 GB), all 10 rounds; the oracle
    follows 1,024 of the 380,372 blocks, including the first and the ragged last one."""
    w = W.WORKLOADS["c5"]
    cfg = ea.EAConfig.from_workload(w, placement=placement)
    L = Lockstep(cfg, sample_groups=W.sample_blocks(w, 1024))
    x_dev = torch.zeros(w.d, device="cuda")
    x_host = np.zeros(L.d_o, np.float32)
    bufs = [torch.empty(w.d, device="cuda") for _ in range(w.n)]
    for t in range(w.rounds):
        _dev_grads(w, t, bufs)
        L.round(bufs, [L.host(b) for b in bufs], x_dev, x_host)
    assert L.total_mismatch == 0
    assert L.gpu.bits_sent() == expected_bits(cfg, w.rounds) == (125_613_752_320, 125_613_752_320)
    del L, bufs, x_dev
    torch.cuda.empty_cache()


@pytest.mark.parametrize("placement", [ea.ADAM_AT_WORKER, ea.ADAM_AT_SERVER])
@pytest.mark.parametrize("form", [0, 1])
@pytest.mark.parametrize("group", [4096, 0])
def test_schedules_and_adam_forms(placement, form, group):
    """alpha_t, beta and theta_t changed every round through ea_set_hparams (Assumption 2's
    alpha/sqrt(T), 1 - theta/T and a step decay), in the paper's and the textbook Adam form."""
    d = 13_000
    cfg = ea.EAConfig(d=d, n=3, qw=W.sign_q(group), qs=W.uniform_q(8, group if group else 0, False), alpha=1e-2,
                      placement=placement, adam_form=form, eps=1e-6, seed=3)
    L = Lockstep(cfg)
    rng = np.random.default_rng(17)
    x_host = rng.standard_normal(d).astype(np.float32)
    x_dev = torch.from_numpy(x_host.copy()).cuda()
    T = 6
    for t in range(1, T + 1):
        L.set_hparams(1e-2 / np.sqrt(t) * (0.2 if t > 4 else 1.0), 0.9 - 0.2 * (t % 2), 1 - 0.1 / t)
        gs = [(rng.standard_normal(d) * 10 ** rng.uniform(-3, 0)).astype(np.float32) for _ in range(cfg.n)]
        L.round([torch.from_numpy(g).cuda() for g in gs], gs, x_dev, x_host)
    with pytest.raises(ea.EAError) as ex:
        L.gpu.set_hparams(1e-2, 1.0, 0.9)
    assert ex.value.status == ea.EA_E_INVAL


@pytest.mark.parametrize("name", ["full", "com1", "com2"])
@pytest.mark.parametrize("ef", [True, False])
def test_toy_section51_lockstep(name, ef):
    """Section 5.1's toy (500 x 500 Gaussian A, 10 workers, beta 0.9, theta 0.99) with its three
    quantizer settings; each side forms 2 A^T (A x - x* - xi) from its own x."""
    A, xs = W.toy_case(0)
    spec = W.TOY_QUANTIZERS[name]
    cfg = ea.EAConfig(d=W.TOY_D, n=W.TOY_N, qw=spec, qs=spec, alpha=1e-4, beta1=0.9, beta2=0.99,
                      error_feedback=ef)
    L = Lockstep(cfg)
    x_dev = torch.zeros(W.TOY_D, device="cuda")
    x_host = np.zeros(W.TOY_D, np.float32)
    for t in range(40):
        xi = [W.toy_noise(0, i, t) for i in range(W.TOY_N)]
        xg = x_dev.cpu().numpy()
        g_dev = [torch.from_numpy(W.toy_gradient(A, xg, xs, xi[i])).cuda() for i in range(W.TOY_N)]
        g_host = [W.toy_gradient(A, x_host, xs, xi[i]) for i in range(W.TOY_N)]
        L.round(g_dev, g_host, x_dev, x_host)
    assert W.toy_full_gradient_norm(A, x_host, xs) < W.toy_full_gradient_norm(A, np.zeros_like(x_host), xs)
