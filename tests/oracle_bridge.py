"""Builds oracle problems from synthetic trajectories and runs the oracle's
version of one CommitKV step.  Test infrastructure: inputs come from the
seeded generator only, never from the CUDA path."""
from __future__ import annotations

import math

import numpy as np

from oracle import core
from paper_2608_07855_gb300 import synth


def problems(tr: synth.Trajectory, layers=None, layer_mask=None):
    """(pre, post) oracle problems; `layers` restricts to a sub-list of layers."""
    cfg = tr.cfg
    K = tr.K if layers is None else tr.K[layers]
    V = tr.V if layers is None else tr.V[layers]
    Qm = tr.Q_pre if layers is None else tr.Q_pre[layers]
    Qp = tr.Q_post if layers is None else tr.Q_post[layers]
    K = synth.values_f64(K, cfg.dtype)
    V = synth.values_f64(V, cfg.dtype)
    Qm = synth.values_f64(Qm, cfg.dtype)
    Qp = synth.values_f64(Qp, cfg.dtype)
    L = tr.L_pre
    pre = core.Problem(K[:, :, :L], V[:, :, :L], tr.pos[:L], Qm, tr.qpos_pre, tr.page_start[:tr.P_pre],
                       tr.page_len[:tr.P_pre], layer_mask=layer_mask)
    post = core.Problem(K, V, tr.pos, Qp, tr.qpos_post, tr.page_start, tr.page_len, layer_mask=layer_mask)
    return pre, post


class OracleStep:
    """The oracle's outputs for one step of one trajectory."""

    def __init__(self, tr: synth.Trajectory, mode="explicit", layer_mask=None):
        cfg = tr.cfg
        self.tr = tr
        pre, post = problems(tr, layer_mask=layer_mask)
        self.pre, self.post = pre, post
        Rm, self.H_pre = core.page_effects(pre, mode)
        self.R_post, self.H_post = core.page_effects(post, mode)
        self.R_pre = np.zeros(tr.P_post)
        self.R_pre[:tr.P_pre] = Rm
        self.stats = core.row_stats(post)
        # later stages take fp32 effects, as the library's interface does
        self.R_pre32 = self.R_pre.astype(np.float32)
        self.R_post32 = self.R_post.astype(np.float32)
        self.state, self.cand = core.classify(self.R_pre32, self.R_post32, tr.eligible)
        self.accepted, self.step_R = core.greedy(post, self.cand, cfg.tau_joint,
                                                 "closed", stats=self.stats)
        self.I = core.select_indices(tr.S_post, tr.page_start, tr.page_len, self.accepted,
                                     tr.pending, self.R_post32[tr.pending], tr.fill_score, cfg.B,
                                     cfg.B_N, cfg.pending_cap)


def rel_close(got, want, rtol):
    """Elementwise |got - want| <= rtol * |want| with infinities matching."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    inf_w, inf_g = np.isinf(want), np.isinf(got)
    ok = inf_w == inf_g
    fin = ~inf_w & ~inf_g
    ok[fin] = np.abs(got[fin] - want[fin]) <= rtol * np.abs(want[fin]) + 1e-30
    return ok


def safe_threshold_mask(R, tau, tol):
    """Decisions of a threshold test that are safe at relative tolerance tol."""
    R = np.asarray(R, np.float64)
    return np.abs(R - tau) > tol * tau


def percentile_safe(R, idx, tol):
    """Pages of E_c whose percentile rank cannot move across any threshold
    when the effects move by a relative tol (the margin rule for ranks)."""
    Rc = np.asarray(R, np.float64)[idx]
    n = len(idx)
    lo = np.array([np.count_nonzero(Rc < x * (1 - 2 * tol)) for x in Rc]) / n
    hi = np.array([np.count_nonzero(Rc < x * (1 + 2 * tol)) for x in Rc]) / n
    safe = np.ones(n, bool)
    for rho in (0.75, 0.25):
        safe &= (lo >= rho) == (hi >= rho)
        safe &= (lo <= rho) == (hi <= rho)
    return safe


def gapped_positions(tr: synth.Trajectory, seed=0):
    """Strictly increasing positions with gaps (a cache after an earlier
    compaction); the probe-query positions follow their tokens."""
    rng = np.random.default_rng(seed)
    S = tr.S_post
    newpos = np.cumsum(rng.integers(1, 4, size=S)).astype(np.int32)
    tr.pos = newpos
    return tr


def isclose_tol(dtype):
    return 1e-4 if dtype == "f32" else 2e-2


def finite_max(x):
    x = np.asarray(x, np.float64)
    x = x[np.isfinite(x)]
    return float(x.max()) if x.size else 0.0


def fmt(x):
    return "inf" if math.isinf(x) else f"{x:.6g}"
