"""Lockstep parity harness: the CUDA library (through its C-ABI binding) and the oracle run the same
rounds on the same seeded inputs, each from its own state; after every round every output is
compared.  Nothing computed by the CUDA path is ever fed to the oracle.

Tolerances:
  * codes: the contract allows a code to differ only where the quantizer's input lies within 2 ulp
    of a decision threshold (the input margin 2 ulp(max(|step|, |e_old|)), carried to the decision
    variable: for Example 1's grid that is y = u L / s, so the window is margin * L / s, and nothing
    more), at no more than 1e-6 of the positions.  The tests hold the stronger claim that no code
    differs at all: with `strict` (the default) any code mismatch fails the test, and its message
    says whether the position was inside that window.  Without `strict`, a mismatch inside the
    window is counted and its coordinate is excluded from later comparisons; a later scale that
    differs is then accepted only for a group that holds such a coordinate (and that group is then
    excluded too);
  * scales: within 1e-6 relative;
  * x, m, v and residuals: |gpu - oracle| <= 1e-7 + 1e-5 |oracle| elementwise;
  * bits sent: exactly equal.

Every Lockstep records what it compared (rounds, code positions, state values, mismatches) in
RUNS; tests/conftest.py prints the totals at the end of the session.

Large workloads whose scale groups are blocks or tensors are separable by group: there the oracle
may run on a fixed sample of whole groups (global coordinates kept for the Philox counters).
"""
from __future__ import annotations

import dataclasses
import os

import numpy as np
import torch

import oracle as O
import paper_2205_14473_gb300 as ea
from paper_2205_14473_gb300 import workloads as W

ATOL, RTOL, SCALE_RTOL = 1e-7, 1e-5, 1e-6

RUNS: list[dict] = []  # one record per Lockstep, for the session summary


def host_threads() -> int:
    """Host cores this process may use (the oracle's thread count)."""
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def _agree(g: torch.Tensor, w: torch.Tensor, rtol: float, atol: float) -> torch.Tensor:
    """Within atol + rtol |w|, or equal (infinities of one sign), or NaN on both sides; a NaN or an
    infinity on one side only disagrees."""
    return ((g - w).abs() <= atol + rtol * w.abs()) | (g == w) | (g.isnan() & w.isnan())


def _offsets(d, spec: W.QuantSpec):
    if spec.kind in (W.Q_IDENTITY, W.Q_POW2):
        return O.group_offsets(d, 0)
    return O.group_offsets(d, spec.group, spec.segments if spec.group < 0 else None)


def _oracle_quant(spec: W.QuantSpec, offsets):
    return O.Quantizer(spec.kind, spec.bits, offsets, stochastic=spec.stochastic, pow2_k=spec.pow2_k,
                       pow2_K=spec.pow2_K)


def unpack_codes(words: torch.Tensor, idx: torch.Tensor, bits: int) -> torch.Tensor:
    """Per-coordinate codes at global coordinates idx from an int32 word stream (on words' device)."""
    pos = idx * bits
    w = words.index_select(0, pos >> 5).to(torch.int64) & 0xFFFFFFFF
    if bits == 32:
        return w
    return (w >> (pos & 31)) & ((1 << bits) - 1)


@dataclasses.dataclass
class RoundReport:
    t: int
    code_mismatches: int = 0
    flagged: int = 0
    max_rel: dict = dataclasses.field(default_factory=dict)


class Lockstep:
    def __init__(self, cfg: ea.EAConfig, sample_groups=None, threads: int | None = None, strict: bool = True):
        threads = host_threads() if threads is None else threads
        self.cfg = cfg
        self.strict = strict
        self.dev = torch.device("cuda", torch.cuda.current_device())
        self.gpu = ea.EARound(cfg)
        d = cfg.d
        off_w, off_s = _offsets(d, cfg.qw), _offsets(d, cfg.qs)
        self.sampled = sample_groups is not None
        if self.sampled:
            assert np.array_equal(off_w, off_s) or cfg.qw.kind in (W.Q_IDENTITY, W.Q_POW2) or \
                cfg.qs.kind in (W.Q_IDENTITY, W.Q_POW2)
            offs = off_w if cfg.qw.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX) else off_s
            groups = np.asarray(sample_groups, dtype=np.int64)
            idx = np.concatenate([np.arange(offs[g], offs[g + 1], dtype=np.int64) for g in groups])
            lens = offs[groups + 1] - offs[groups]
            local = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
            self.groups = groups
            self.idx = idx
            qw_o = _oracle_quant(cfg.qw, local if cfg.qw.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX) else
                                 O.group_offsets(len(idx), 0))
            qs_o = _oracle_quant(cfg.qs, local if cfg.qs.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX) else
                                 O.group_offsets(len(idx), 0))
            gidx = idx
        else:
            self.groups = None
            self.idx = np.arange(d, dtype=np.int64)
            qw_o, qs_o = _oracle_quant(cfg.qw, off_w), _oracle_quant(cfg.qs, off_s)
            gidx = None
        self.off_w, self.off_s = off_w, off_s
        self.d_o = len(self.idx)
        self.idx_dev = torch.from_numpy(self.idx).to(self.dev)
        self.orc = O.OracleRound(self.d_o, cfg.n, qw_o, qs_o, cfg.alpha, cfg.beta1, cfg.beta2, cfg.eps,
                                 seed=cfg.seed, mode=cfg.placement, error_feedback=cfg.error_feedback,
                                 gidx=gidx, threads=threads, adam_form=cfg.adam_form)
        self.tainted = torch.zeros(self.d_o, dtype=torch.bool, device=self.dev)
        self.total_mismatch = 0
        self.reports: list[RoundReport] = []
        self.record = {"test": os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0], "d": cfg.d, "n": cfg.n,
                       "d_oracle": self.d_o, "rounds": 0, "code_positions": 0, "values": 0, "scales": 0,
                       "mismatches": 0, "flagged": 0}
        RUNS.append(self.record)

    def set_hparams(self, alpha: float, beta1: float, beta2: float) -> None:
        self.gpu.set_hparams(alpha, beta1, beta2)
        self.orc.set_hparams(alpha, beta1, beta2)

    # ------------------------------------------------------------------------------------ inputs
    def host(self, t_dev: torch.Tensor) -> np.ndarray:
        """Oracle-side copy of a device input (the sampled coordinates only when sampling)."""
        v = t_dev[: self.cfg.d]
        if self.sampled:
            v = v.index_select(0, self.idx_dev)
        return np.ascontiguousarray(v.detach().cpu().numpy().astype(np.float32))

    # ------------------------------------------------------------------------------------- round
    def round(self, grads_dev, grads_host, x_dev: torch.Tensor, x_host: np.ndarray) -> RoundReport:
        n = self.cfg.n
        e_old = self.orc.e.copy() if self.cfg.error_feedback else np.zeros_like(self.orc.e)
        es_old = self.orc.es.copy()
        for i in range(n):
            self.gpu.worker_compress(i, grads_dev[i])
        self.orc.compress_all(grads_host)
        self.gpu.server_step()
        self.orc.server_step()
        self.gpu.apply(x_dev)
        self.orc.apply(x_host)
        rep = RoundReport(self.orc.t)
        self._compare(rep, e_old, es_old, x_dev, x_host)
        self.reports.append(rep)
        self.record["rounds"] += 1
        return rep

    # ------------------------------------------------------------------------------- comparisons
    def _dev(self, a: np.ndarray) -> torch.Tensor:
        return torch.from_numpy(np.ascontiguousarray(a)).to(self.dev)

    def _gather(self, view: torch.Tensor) -> torch.Tensor:
        return view.index_select(0, self.idx_dev) if self.sampled else view[: self.cfg.d]

    def _close(self, name, got: torch.Tensor, want: np.ndarray, rep: RoundReport):
        w = self._dev(want).double()
        g = got.double()
        err = (g - w).abs()
        bad = ~_agree(g, w, RTOL, ATOL) & ~self.tainted
        self.record["values"] += int(w.numel())
        nbad = int(bad.sum())
        rel = torch.nan_to_num(err / (w.abs() + 1e-30), nan=0.0).masked_fill(self.tainted, 0)
        rep.max_rel[name] = float(rel.max()) if rel.numel() else 0.0
        if nbad:
            j = int(torch.nonzero(bad)[0])
            raise AssertionError(f"round {rep.t}: {name} differs at {nbad} coordinates, e.g. local {j}: "
                                 f"gpu {float(g[j])!r} oracle {float(w[j])!r}")

    def _group_ids(self, offs):
        """Local group index of every oracle coordinate."""
        return np.searchsorted(offs, self.idx, side="right") - 1

    def _taint(self, local_js):
        """Exclude these coordinates from later comparisons (their codes differed)."""
        if len(local_js):
            m = np.zeros(self.d_o, bool)
            m[np.asarray(local_js)] = True
            self.tainted |= self._dev(m)

    def _flagged(self, spec, js, u, step, e_old, scale_of, qid, t):
        """Which of the mismatched local coordinates js lie within 2 ulp of a decision threshold."""
        out = []
        for j in js:
            uj = float(u[j])
            margin = 2.0 * float(np.spacing(np.float32(max(abs(float(step[j])), abs(float(e_old[j]))))))
            if spec.kind == W.Q_SIGN_L1:
                out.append(abs(uj) <= margin)
            elif spec.kind == W.Q_UNIFORM_MAX:
                s = float(scale_of(j))
                L = 2 ** (spec.bits - 1) - 1
                y = uj / s * L
                my = margin * L / s  # the input margin carried to y = u L / s
                if spec.stochastic:
                    U = O.uniform(self.cfg.seed, qid, t, int(self.idx[j]))
                    fr = y - np.floor(y)
                    out.append(abs(fr - U) <= my or min(fr, 1 - fr) <= my)
                else:
                    out.append(abs((y - np.floor(y)) - 0.5) <= my)
            elif spec.kind == W.Q_POW2:
                a = abs(uj)
                th = [0.0] + [1.5 * 2.0 ** j2 for j2 in range(spec.pow2_k, spec.pow2_K)]
                out.append(min(abs(a - x) for x in th) <= margin)
            else:
                out.append(False)
        return np.array(out, dtype=bool)

    def _compare_codes(self, name, spec, words_view, orc_words, u, step, e_old, scales_orc, offs_local, qid,
                       rep):
        self.record["code_positions"] += self.d_o
        if not self.sampled and not bool(self.tainted.any()):
            # the whole stream at once (padding bits are 0 on both sides); unpacked only if it differs
            nw = (self.cfg.d * spec.bits + 31) // 32
            if torch.equal(words_view[:nw], self._dev(orc_words[:nw].view(np.int32))):
                return
        got = unpack_codes(words_view, self.idx_dev, spec.bits)
        want = unpack_codes(self._dev(orc_words.view(np.int32)), torch.arange(self.d_o, device=self.dev), spec.bits)
        bad = (got != want) & ~self.tainted
        js = torch.nonzero(bad).flatten().cpu().numpy()
        if len(js):
            gid = np.searchsorted(offs_local, np.arange(self.d_o), side="right") - 1 if len(offs_local) > 1 else None
            flags = self._flagged(spec, js, u, step, e_old,
                                  (lambda j: scales_orc[gid[j]]) if gid is not None else (lambda j: 0.0),
                                  qid, rep.t - 1)
            rep.code_mismatches += len(js)
            rep.flagged += int(flags.sum())
            self.total_mismatch += len(js)
            self.record["mismatches"] += len(js)
            self.record["flagged"] += int(flags.sum())
            if self.strict or not flags.all():
                j = int(js[~flags][0]) if not flags.all() else int(js[0])
                where = "inside" if flags.all() else "outside"
                raise AssertionError(f"round {rep.t}: {name}: {len(js)} codes differ ({int(flags.sum())} within 2 ulp "
                                     f"of a threshold); e.g. local {j} (global {int(self.idx[j])}), {where} the "
                                     f"window: gpu {int(got[j])} oracle {int(want[j])}, u = {float(u[j])!r}")
            self._taint(js)

    def _compare_scales(self, name, got_view, want, offs_full, rep):
        if not len(want):
            return
        if self.sampled:
            g = got_view.index_select(0, torch.from_numpy(self.groups).to(self.dev))
        else:
            g = got_view[: len(want)]
        self.record["scales"] += len(want)
        w = self._dev(want).double()
        err = ~_agree(g.double(), w, SCALE_RTOL, 0.0)
        if bool(err.any()):
            bad = torch.nonzero(err).flatten().cpu().numpy()
            # a group whose scale differs is accepted only if it holds a coordinate whose code
            # differed earlier (its l1 / l_inf input then differs); the group is excluded from then on
            gid = self._group_ids(offs_full)
            tainted = self.tainted.cpu().numpy()
            sampled_groups = self.groups if self.sampled else np.arange(len(want))
            for k in bad:
                members = gid == sampled_groups[k]
                if not tainted[members].any():
                    raise AssertionError(f"round {rep.t}: {name} scale {k}: gpu {float(g[k])!r} "
                                         f"oracle {float(want[k])!r}")
                self._taint(np.nonzero(members)[0])

    def _compare(self, rep, e_old, es_old, x_dev, x_host):
        cfg, orc, gpu = self.cfg, self.orc, self.gpu
        torch.cuda.synchronize()
        has_w = cfg.qw.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX)
        has_s = cfg.qs.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX)
        loc_w, loc_s = orc.qw.offsets, orc.qs.offsets
        for i in range(cfg.n):
            u = orc.last_input(i)
            step = u.astype(np.float64) - e_old[i]
            self._compare_codes(f"worker {i}", cfg.qw, gpu.view(ea.EA_VIEW_CODES_WORKER, i), orc.wwords[i], u, step,
                                e_old[i], orc.wscales[i], loc_w, i, rep)
            if has_w:
                self._compare_scales(f"worker {i}", gpu.view(ea.EA_VIEW_SCALES_WORKER, i),
                                     orc.wscales[i][: orc.qw.n_groups], self.off_w, rep)
            self._close(f"e[{i}]", self._gather(gpu.view(ea.EA_VIEW_E_WORKER, i)), orc.e[i], rep)
            if cfg.placement == ea.ADAM_AT_WORKER:
                self._close(f"m[{i}]", self._gather(gpu.view(ea.EA_VIEW_M, i)), orc.m[i], rep)
                self._close(f"v[{i}]", self._gather(gpu.view(ea.EA_VIEW_V, i)), orc.v[i], rep)
        w = orc.last_server_input()
        step = w.astype(np.float64) - es_old
        self._compare_codes("server", cfg.qs, gpu.view(ea.EA_VIEW_CODES_SERVER), orc.swords, w, step, es_old,
                            orc.sscales, loc_s, cfg.n, rep)
        if has_s:
            self._compare_scales("server", gpu.view(ea.EA_VIEW_SCALES_SERVER), orc.sscales[: orc.qs.n_groups],
                                 self.off_s, rep)
        self._close("e_s", self._gather(gpu.view(ea.EA_VIEW_E_SERVER)), orc.es, rep)
        if cfg.placement == ea.ADAM_AT_SERVER:
            self._close("m_s", self._gather(gpu.view(ea.EA_VIEW_M_SERVER)), orc.ms, rep)
            self._close("v_s", self._gather(gpu.view(ea.EA_VIEW_V_SERVER)), orc.vs, rep)
        self._close("x", self._gather(x_dev), x_host, rep)
        assert gpu.bits_sent() == (orc.up_bits, orc.down_bits) or self.sampled
        limit = int(1e-6 * self.d_o * (cfg.n + 1) * rep.t)
        assert self.total_mismatch <= limit, \
            f"{self.total_mismatch} code mismatches exceed 1e-6 of the {self.d_o * (cfg.n + 1) * rep.t} positions"


def expected_bits(cfg: ea.EAConfig, rounds: int) -> tuple[int, int]:
    """Corollary 1's count, from the message format: b bits per coordinate + 32 per scale word."""
    def msg(spec):
        if spec.kind in (W.Q_IDENTITY, W.Q_POW2):
            return cfg.d * spec.bits
        groups = 1 if spec.group == 0 else (-(-cfg.d // spec.group) if spec.group > 0 else len(spec.segments))
        return cfg.d * spec.bits + 32 * groups
    return rounds * cfg.n * msg(cfg.qw), rounds * cfg.n * msg(cfg.qs)
