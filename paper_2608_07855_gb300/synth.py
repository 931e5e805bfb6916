"""Seeded synthetic agent-shaped KV caches for CommitKV.

Shared by the tests (which hand the same inputs to the CPU oracle and to the
CUDA library) and by bench.py.  This module holds none of the scoring
method's arithmetic: it draws numbers, lays out events and pages, and plants
pages whose keys are aligned with the pre-commit probe queries and turned
away from the post-commit ones.

Trajectory model (Section 3.1, Eq. 1-5)
  pre-commit cache y_t  = events q, z_1, a_1, o_1, ..., z_t, a_t (L_pre tokens);
                          reasoning / tool-call / observation lengths are
                          uniform in [32, 256] and the current tool call a_t
                          ends exactly at L_pre.
  post-commit cache     = y_t || o_t (L_obs tokens) || W decoded tokens.
  Q-  = the last W positions of y_t;  Q+ = the W decoded positions.
  pages                 = tool-call and observation events cut from their
                          first token into G-token pages (the last page of
                          an event takes the remainder).
  E_c (eligible)        = pages of events completed by the commit, a_t
                          included; o_t's pages exist in the post cache but
                          are not eligible.
  positions             = 0, 1, 2, ... (contiguous before any compaction).

Values: Q, K, V ~ N(0,1) from a counter-based generator (synth_normal.c),
rounded to bf16 for the Qwen-shaped workloads; the Qwen shapes scale 4 key
channels per (layer, KV head) by 8.  Planted pages (see _plant_*) replace
the keys of a seeded subset of eligible pages in every (layer, KV head).
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth_normal.c")
_SO = os.path.join(_HERE, "_build", "libsynth.so")
_MASK = (1 << 64) - 1


def build(force: bool = False) -> str:
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC,
                               "-lm", "-lpthread"])
        os.replace(tmp, _SO)
    return _SO


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.synth_normal_fill.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                          ctypes.c_int64, ctypes.c_int, ctypes.c_void_p,
                                          ctypes.c_void_p, ctypes.c_int64, ctypes.c_int]
        lib.synth_normal_fill.restype = ctypes.c_int
        _lib = lib
    return _lib


def normal(seed: int, stream: int, shape, bf16: bool = False, chan_scale=None, out=None):
    """N(0,1) array of `shape` (float32, or bf16 bits as uint16)."""
    n = int(np.prod(shape))
    dt = np.uint16 if bf16 else np.float32
    if out is None:
        out = np.empty(shape, dt)
    assert out.dtype == dt and out.flags.c_contiguous and out.size == n
    cs = None
    if chan_scale is not None:
        cs = np.ascontiguousarray(chan_scale, np.float32)
    rc = _load().synth_normal_fill(seed & _MASK, stream & _MASK, 0, n, 1 if bf16 else 0,
                                   out.ctypes.data, cs.ctypes.data if cs is not None else None,
                                   0 if cs is None else cs.size, os.cpu_count() or 1)
    assert rc == 0
    return out


def _mix64(x: int) -> int:
    x = (x + 0x9E3779B97F4A7C15) & _MASK
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & _MASK
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & _MASK
    return x ^ (x >> 31)


class Draws:
    """Small integer / uniform draws from splitmix64(seed, stream, counter)."""

    def __init__(self, seed: int, stream: int):
        self.key = _mix64((seed * 0x9E3779B97F4A7C15 + stream) & _MASK)
        self.i = 0

    def u64(self) -> int:
        self.i += 1
        return _mix64((self.key + self.i) & _MASK)

    def uniform(self) -> float:
        return ((self.u64() >> 11) + 0.5) / float(1 << 53)

    def randint(self, lo: int, hi: int) -> int:
        """Uniform integer in [lo, hi] (inclusive)."""
        return lo + self.u64() % (hi - lo + 1)

    def sample(self, n: int, k: int):
        """k distinct integers from range(n), in draw order (partial shuffle)."""
        idx = list(range(n))
        for j in range(min(k, n)):
            t = j + self.u64() % (n - j)
            idx[j], idx[t] = idx[t], idx[j]
        return idx[:k]


def uniform_array(seed: int, stream: int, n: int) -> np.ndarray:
    """float32 U(0,1) array, vectorised splitmix64 on a counter."""
    key = np.uint64(_mix64((seed * 0x9E3779B97F4A7C15 + stream) & _MASK))
    x = key + np.arange(1, n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        x = x + np.uint64(0x9E3779B97F4A7C15)
        x = (x ^ (x >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        x = (x ^ (x >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        x = x ^ (x >> np.uint64(31))
    return (((x >> np.uint64(40)).astype(np.float64) + 0.5) / float(1 << 24)).astype(np.float32)


# ----------------------------------------------------------------------------
# bf16 helpers (bit conversions only)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(x, np.float32).view(np.uint32)
    with np.errstate(over="ignore"):
        r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ----------------------------------------------------------------------------
# workloads


@dataclass
class Config:
    name: str
    M: int
    H: int
    Hq: int
    d: int
    dtype: str  # "f32" | "bf16"
    L_pre: int
    L_obs: int
    W: int
    G: int
    B: int
    tau_joint: float = 0.05
    pending_cap: int = 16
    eta: float = 0.125
    n_planted: int = 0
    planted_frac: float = 0.0
    outlier_channels: int = 0
    outlier_scale: float = 8.0
    event_len: tuple = (32, 256)
    plant: str = "orthogonal"  # "orthogonal" (g*W < d) | "shared" (window direction)
    # planting strengths (see _plant_*)
    alpha: float = 0.0
    beta: tuple = (0.0, 0.0)
    gamma: float = 0.0
    sigma: float = 0.25
    nu: float = 0.0  # shared value direction of planted tokens
    # ragged batch
    n_traj: int = 1
    ctx_range: tuple = ()
    obs_range: tuple = ()
    turns_range: tuple = ()

    @property
    def g(self):
        return self.Hq // self.H

    @property
    def B_N(self):
        return int(math.floor(self.eta * self.B))


CONFIGS = {
    # 1. Tiny (fp32 oracle reference)
    "tiny": Config("tiny", M=1, H=2, Hq=4, d=64, dtype="f32", L_pre=2048, L_obs=256, W=16, G=16,
                   B=1024, tau_joint=0.05, pending_cap=8, n_planted=8, plant="orthogonal",
                   alpha=9.0, beta=(2.7, 3.3), nu=6.0),
    # 2. Qwen3-8B shape, 16K + 2K
    "qwen3_8b_16k": Config("qwen3_8b_16k", M=36, H=8, Hq=32, d=128, dtype="bf16", L_pre=16384,
                           L_obs=2048, W=32, G=32, B=4096, pending_cap=16, planted_frac=0.2,
                           outlier_channels=4, plant="shared", alpha=12.0, beta=(8.0, 12.0),
                           gamma=8.0, nu=6.0),
    # 3. Qwen3-8B shape, 32K + 4K (headline)
    "qwen3_8b_32k": Config("qwen3_8b_32k", M=36, H=8, Hq=32, d=128, dtype="bf16", L_pre=32768,
                           L_obs=4096, W=32, G=32, B=8192, pending_cap=32, planted_frac=0.2,
                           outlier_channels=4, plant="shared", alpha=12.0, beta=(8.0, 12.0),
                           gamma=8.0, nu=6.0),
    # 4. 16 ragged trajectories, Qwen3-8B shape
    "ragged16": Config("ragged16", M=36, H=8, Hq=32, d=128, dtype="bf16", L_pre=0, L_obs=0, W=32,
                       G=32, B=8192, pending_cap=16, planted_frac=0.2, outlier_channels=4,
                       plant="shared", alpha=12.0, beta=(8.0, 12.0), gamma=8.0, nu=6.0, n_traj=16,
                       ctx_range=(4096, 32768), obs_range=(256, 4096), turns_range=(4, 24)),
    # 5. Qwen3-32B shape, 128K + 8K
    "qwen3_32b_128k": Config("qwen3_32b_128k", M=64, H=8, Hq=64, d=128, dtype="bf16",
                             L_pre=131072, L_obs=8192, W=64, G=64, B=16384, pending_cap=16,
                             planted_frac=0.05, outlier_channels=4, plant="shared", alpha=12.0,
                             beta=(8.0, 12.0), gamma=8.0, nu=6.0),
}


def small_config(name="small_bf16", **kw) -> Config:
    """Reduced shapes for oracle-speed parity tests (several 128-token tiles
    plus a ragged tail)."""
    base = dict(M=2, H=2, Hq=8, d=128, dtype="bf16", L_pre=700, L_obs=90, W=16, G=32, B=320,
                tau_joint=0.05, pending_cap=4, planted_frac=0.2, outlier_channels=4,
                plant="orthogonal", alpha=9.0, beta=(2.7, 3.3), nu=6.0)
    base.update(kw)
    return Config(name, **base)


# ----------------------------------------------------------------------------


@dataclass
class Trajectory:
    cfg: Config
    seed: int
    index: int
    L_pre: int
    L_obs: int
    events: list  # (kind, start, length); kinds: query/reason/call/obs/decode
    page_start: np.ndarray  # [P_post] int32
    page_len: np.ndarray
    page_event: np.ndarray  # event index of each page
    P_pre: int  # pages resident in the pre cache (a prefix of the page list)
    eligible: np.ndarray  # [P_post] uint8 (E_c)
    planted: np.ndarray  # page ids
    K: np.ndarray = None  # [M][H][S_post][d] float32 or bf16 bits
    V: np.ndarray = None
    Q_pre: np.ndarray = None  # [M][Hq][W][d]
    Q_post: np.ndarray = None
    pos: np.ndarray = None  # [S_post] int32
    fill_score: np.ndarray = None  # [S_post] float32
    pending: np.ndarray = None  # page ids of o_t
    meta: dict = field(default_factory=dict)

    @property
    def S_pre(self):
        return self.L_pre

    @property
    def S_post(self):
        return self.L_pre + self.L_obs + self.cfg.W

    @property
    def qpos_pre(self):
        """Q-c: the positions of the last W tokens of y_t (Eq. 5)."""
        return np.ascontiguousarray(self.pos[self.L_pre - self.cfg.W: self.L_pre], np.int32)

    @property
    def qpos_post(self):
        """Q+c: the positions of the first W decoded tokens after o_t (Eq. 5)."""
        b = self.L_pre + self.L_obs
        return np.ascontiguousarray(self.pos[b: b + self.cfg.W], np.int32)

    @property
    def P_post(self):
        return int(self.page_start.shape[0])


_T_K, _T_V, _T_QPRE, _T_QPOST, _T_DIR, _T_FILL, _T_EVENTS, _T_PLANT, _T_OUTL, _T_PNOISE, _T_RAGGED, _T_VDIR, \
    _T_ROWS = range(13)


def _stream(traj: int, tensor: int, layer: int = 0, head: int = 0) -> int:
    return (((traj * 16 + tensor) * 4096 + layer) * 4096 + head) & _MASK


def _events(cfg: Config, seed: int, traj: int, L_pre: int, turns: int = 0):
    dr = Draws(seed, _stream(traj, _T_EVENTS))
    lo, hi = cfg.event_len
    ev = []
    if turns:
        # 3*turns - 1 events (q/z_1, a_1, o_1, ..., z_T, a_T) cut at seeded points
        n_ev = 3 * turns - 1
        min_len = 8
        cuts = sorted(dr.sample(L_pre - n_ev * min_len, n_ev - 1))
        bounds = [0] + [c + (j + 1) * min_len for j, c in enumerate(cuts)] + [L_pre]
        kinds = ["reason", "call", "obs"]
        for j in range(n_ev):
            kind = "query" if j == 0 else kinds[j % 3]
            ev.append((kind, bounds[j], bounds[j + 1] - bounds[j]))
        return ev
    a_len = dr.randint(lo, hi)
    body = L_pre - a_len
    t, j = 0, 0
    kinds = ["reason", "call", "obs"]
    while t < body:
        n = min(dr.randint(lo, hi), body - t)
        kind = "query" if j == 0 else kinds[j % 3]
        ev.append((kind, t, n))
        t += n
        j += 1
    # the turn's reasoning z_t ends the body; the tool call a_t ends at L_pre
    ev.append(("call", body, a_len))
    return ev


def _pages(cfg: Config, events):
    ps, pl, pe = [], [], []
    for j, (kind, b, n) in enumerate(events):
        if kind not in ("call", "obs"):
            continue
        for s in range(b, b + n, cfg.G):
            ps.append(s)
            pl.append(min(cfg.G, b + n - s))
            pe.append(j)
    return np.asarray(ps, np.int32), np.asarray(pl, np.int32), np.asarray(pe, np.int32)


def _unit(v):
    return v / max(np.linalg.norm(v), 1e-30)


def make_trajectory(cfg: Config, seed: int = 0, traj: int = 0, values: bool = True) -> Trajectory:
    if cfg.n_traj > 1 and cfg.ctx_range:
        dr = Draws(seed, _stream(traj, _T_RAGGED))
        L_pre = dr.randint(*cfg.ctx_range)
        L_obs = dr.randint(*cfg.obs_range)
        turns = dr.randint(*cfg.turns_range)
    else:
        L_pre, L_obs, turns = cfg.L_pre, cfg.L_obs, 0
    ev = _events(cfg, seed, traj, L_pre, turns)
    ev.append(("obs", L_pre, L_obs))  # o_t, appended after the commit
    ev.append(("decode", L_pre + L_obs, cfg.W))  # first W decoded tokens of turn t+1
    ps, pl, pe = _pages(cfg, ev)
    P_pre = int(np.count_nonzero(ps < L_pre))
    eligible = np.zeros(len(ps), np.uint8)
    eligible[:P_pre] = 1
    # planted pages: eligible pages outside the current tool call a_t (whose
    # tail lies inside the pre-commit window)
    a_t = len(ev) - 3
    pool = [E for E in range(P_pre) if pe[E] != a_t]
    n_pl = cfg.n_planted if cfg.n_planted else int(round(cfg.planted_frac * P_pre))
    dr = Draws(seed, _stream(traj, _T_PLANT))
    planted = np.asarray(sorted(dr.sample(len(pool), min(n_pl, len(pool)))), np.int64)
    planted = np.asarray([pool[i] for i in planted], np.int32)
    tr = Trajectory(cfg, seed, traj, L_pre, L_obs, ev, ps, pl, pe, P_pre, eligible, planted)
    tr.pending = np.asarray([E for E in range(len(ps)) if pe[E] == len(ev) - 2], np.int32)
    tr.pos = np.arange(tr.S_post, dtype=np.int32)
    if values:
        _fill_values(tr)
    return tr


def _fill_values(tr: Trajectory):
    cfg, seed, t = tr.cfg, tr.seed, tr.index
    M, H, Hq, d, W, g = cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.W, cfg.g
    S = tr.S_post
    bf = cfg.dtype == "bf16"
    dt = np.uint16 if bf else np.float32
    tr.K = np.empty((M, H, S, d), dt)
    tr.V = np.empty((M, H, S, d), dt)
    Qpre = np.empty((M, Hq, W, d), np.float32)
    Qpost = np.empty((M, Hq, W, d), np.float32)
    tr.fill_score = uniform_array(seed, _stream(t, _T_FILL), S)
    plant_tok = np.concatenate([np.arange(tr.page_start[E], tr.page_start[E] + tr.page_len[E])
                                for E in tr.planted]) if len(tr.planted) else np.zeros(0, np.int64)
    plant_page = np.concatenate([np.full(tr.page_len[E], j) for j, E in enumerate(tr.planted)]) \
        if len(tr.planted) else np.zeros(0, np.int64)
    bl, bh = cfg.beta
    dr = Draws(seed, _stream(t, _T_PLANT, 1))
    beta_page = np.asarray([bl + (bh - bl) * dr.uniform() for _ in tr.planted], np.float64)
    # each planted page is aligned with one pre-window query of its group
    row_page = np.asarray([dr.randint(0, g * W - 1) for _ in tr.planted], np.int64)
    for l in range(M):
        for kvh in range(H):
            cs = None
            if cfg.outlier_channels:
                dro = Draws(seed, _stream(t, _T_OUTL, l, kvh))
                cs = np.ones(d, np.float32)
                cs[dro.sample(d, cfg.outlier_channels)] = cfg.outlier_scale
            normal(seed, _stream(t, _T_K, l, kvh), (S, d), bf, cs, out=tr.K[l, kvh])
            normal(seed, _stream(t, _T_V, l, kvh), (S, d), bf, None, out=tr.V[l, kvh])
            for h in range(kvh * g, (kvh + 1) * g):
                normal(seed, _stream(t, _T_QPRE, l, h), (W, d), False, None, out=Qpre[l, h])
                normal(seed, _stream(t, _T_QPOST, l, h), (W, d), False, None, out=Qpost[l, h])
            if len(plant_tok) and cfg.nu:
                _plant_values(tr, l, kvh, plant_tok)
            if cfg.plant == "shared":
                _plant_shared(tr, l, kvh, Qpre, Qpost, plant_tok, plant_page, beta_page, row_page)
            elif len(plant_tok):
                _plant_orthogonal(tr, l, kvh, Qpre, Qpost, plant_tok, plant_page, beta_page, row_page)
    if bf:
        tr.Q_pre = f32_to_bf16_bits(Qpre)
        tr.Q_post = f32_to_bf16_bits(Qpost)
    else:
        tr.Q_pre, tr.Q_post = Qpre, Qpost
    tr.meta["beta_page"] = beta_page
    tr.meta["row_page"] = row_page


def _store_keys(tr, l, kvh, tok, kf32):
    if tr.cfg.dtype == "bf16":
        tr.K[l, kvh, tok] = f32_to_bf16_bits(kf32)
    else:
        tr.K[l, kvh, tok] = kf32.astype(np.float32)


def _plant_values(tr, l, kvh, tok):
    """Planted tokens' values share one direction per (layer, KV head):
    v = n + nu * c_v, so that deleting several planted pages moves the
    output coherently (their joint effect grows with the number deleted)."""
    cfg = tr.cfg
    cv = _unit(normal(tr.seed, _stream(tr.index, _T_VDIR, l, kvh), (cfg.d,)).astype(np.float64))
    if cfg.dtype == "bf16":
        v = bf16_bits_to_f32(tr.V[l, kvh, tok]).astype(np.float64)
        tr.V[l, kvh, tok] = f32_to_bf16_bits((v + cfg.nu * cv[None, :]).astype(np.float32))
    else:
        tr.V[l, kvh, tok] = (tr.V[l, kvh, tok] + cfg.nu * cv[None, :]).astype(np.float32)


def _plant_orthogonal(tr, l, kvh, Qpre, Qpost, tok, page_of_tok, beta_page, row_page):
    """Planted keys for g*W < d (literal reading of the Tiny workload).

    Page j's keys are k = alpha * u_j + sigma * (noise projected off span(Q+))
    - beta_j * sqrt(d) * k1, where u_j is the unit projection off span(Q+)
    of the pre-window query row_page[j] of the group, and k1 is the
    least-norm vector with <q+, k1> = 1 for every post-window query of the
    group.  The scaled post-window score of every planted key is then
    exactly -beta_j for every post query: beta = 0 is "orthogonal to the
    post-commit queries", beta > 0 also pushes the page to the bottom of the
    post-commit ranking.  alpha sets how strongly the chosen pre-window
    query attends to the page."""
    cfg = tr.cfg
    g, W, d = cfg.g, cfg.W, cfg.d
    qp = Qpost[l, kvh * g:(kvh + 1) * g].reshape(g * W, d).astype(np.float64)
    qm = Qpre[l, kvh * g:(kvh + 1) * g].reshape(g * W, d).astype(np.float64)
    gram = qp @ qp.T
    proj = np.eye(d) - qp.T @ np.linalg.solve(gram, qp)
    u = proj @ qm.T  # [d][g*W]
    u = (u / np.maximum(np.linalg.norm(u, axis=0), 1e-30)).T[row_page]  # [pages][d]
    k1 = qp.T @ np.linalg.solve(gram, np.ones(g * W))
    noise = normal(tr.seed, _stream(tr.index, _T_PNOISE, l, kvh), (len(tok), d)).astype(np.float64)
    k = cfg.alpha * u[page_of_tok] + cfg.sigma * (noise @ proj.T) \
        - (beta_page[page_of_tok] * math.sqrt(d))[:, None] * k1[None, :]
    _store_keys(tr, l, kvh, tok, k.astype(np.float32))


def _plant_shared(tr, l, kvh, Qpre, Qpost, tok, page_of_tok, beta_page, row_page):
    """Shared-direction model for g*W >= d, where no key can be orthogonal to
    every post-window query.  The group's queries get a common direction per
    window, q = n + gamma * c (c- for Q-, c+ for Q+, c+ orthogonal to c-);
    page j's keys are k = alpha * u_j - beta_j * c+ + sigma * n, with u_j the
    unit pre-window query of a seeded row of the group (drawn per slice) with
    its c+ and c- components removed.  The page then dominates the attention of its own
    pre-window row (score about alpha) and of no other (without the c-
    removal every planted page would score alpha * gamma / |q| against every
    pre-window query, the planted pages would share the pre-window mass and
    each one's own effect would stay small).  Post-window scores are about
    -gamma * beta_j / sqrt(d)."""
    cfg = tr.cfg
    g, W, d = cfg.g, cfg.W, cfg.d
    dirs = normal(tr.seed, _stream(tr.index, _T_DIR, l, kvh), (2, d)).astype(np.float64)
    cm = _unit(dirs[0])
    cp = _unit(dirs[1] - (dirs[1] @ cm) * cm)
    Qpre[l, kvh * g:(kvh + 1) * g] += np.float32(cfg.gamma) * cm.astype(np.float32)
    Qpost[l, kvh * g:(kvh + 1) * g] += np.float32(cfg.gamma) * cp.astype(np.float32)
    if len(tok) == 0:
        return
    # the aligned pre-window row of each page is drawn anew for every
    # (layer, KV head): pages that share a row in one slice split its mass,
    # but each page has slices where it is alone in its row
    drr = Draws(tr.seed, _stream(tr.index, _T_ROWS, l, kvh))
    row_page = np.asarray([drr.randint(0, g * W - 1) for _ in beta_page], np.int64)
    qm = Qpre[l, kvh * g:(kvh + 1) * g].reshape(g * W, d).astype(np.float64)[row_page]
    u = qm - (qm @ cp)[:, None] * cp[None, :] - (qm @ cm)[:, None] * cm[None, :]
    u = u / np.maximum(np.linalg.norm(u, axis=1, keepdims=True), 1e-30)
    noise = normal(tr.seed, _stream(tr.index, _T_PNOISE, l, kvh), (len(tok), d)).astype(np.float64)
    k = cfg.alpha * u[page_of_tok] - beta_page[page_of_tok][:, None] * cp[None, :] + cfg.sigma * noise
    _store_keys(tr, l, kvh, tok, k.astype(np.float32))


def values_f64(arr: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 view of stored inputs (bf16 bits or float32)."""
    if dtype == "bf16":
        return bf16_bits_to_f32(arr).astype(np.float64)
    return np.asarray(arr, np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# multi-turn timelines (Algorithm 1's outer loop)

_T_TIMELINE = 32  # stream tags of the timeline draws (disjoint from the tags above)


@dataclass
class Timeline:
    """A multi-turn agent trajectory q, z_1, a_1, o_1, ..., z_T, a_T, o_T,
    z_{T+1} with one commit per tool call a_t.

    events[j] = (kind, first token, length) in timeline order; commit t
    (0-based) ends at commit_end[t] (the end of a_t); its pre-commit window
    is the last W positions before commit_end[t] and its post-commit window
    the first W tokens of the next reasoning event, which start at
    post_start[t] (after the observation o_t).  Positions are the timeline
    indices.  K, V [M][H][S][d], Q_pre / Q_post [T][M][Hq][W][d] (bf16 bits
    or float32), fill [S] (a per-token score for the budget's fill)."""
    cfg: Config
    seed: int
    turns: int
    events: list
    commit_end: np.ndarray
    post_start: np.ndarray
    K: np.ndarray = None
    V: np.ndarray = None
    Q_pre: np.ndarray = None
    Q_post: np.ndarray = None
    fill: np.ndarray = None
    Q_tok: np.ndarray = None  # [S][M][Hq][d]: the query each position decodes with (decode-cadence windows)

    @property
    def S(self):
        kind, b, n = self.events[-1]
        return b + n

    def qpos_pre(self, t):
        return np.arange(self.commit_end[t] - self.cfg.W, self.commit_end[t], dtype=np.int32)

    def qpos_post(self, t):
        return np.arange(self.post_start[t], self.post_start[t] + self.cfg.W, dtype=np.int32)

    def decoded(self, a, b):
        """Decoded tokens in positions [a, b): the model writes the reasoning
        and tool-call events; the query and the observations are prefilled."""
        n = 0
        for kind, s, m in self.events:
            if kind in ("reason", "call"):
                n += max(0, min(b, s + m) - max(a, s))
        return n

    def window(self, end):
        """The probe window of a decode-cadence checkpoint taken when
        position end - 1 has just been decoded: the queries of the last W
        positions, as ([M][Hq][W][d], positions [W])."""
        W = self.cfg.W
        q = np.ascontiguousarray(np.transpose(self.Q_tok[end - W:end], (1, 2, 0, 3)))
        return q, np.arange(end - W, end, dtype=np.int32)


def make_timeline(cfg: Config, seed: int = 0, turns: int = 3, values: bool = True) -> Timeline:
    """Event lengths uniform in cfg.event_len (reasoning events at least W
    long, so that a post-commit window lies inside the next reasoning event);
    Q, K, V ~ N(0, 1) from the counter-based generator; fill uniform."""
    dr = Draws(seed, _stream(0, _T_TIMELINE))
    lo, hi = cfg.event_len
    ev, t = [], 0

    def add(kind, n):
        nonlocal t
        ev.append((kind, t, n))
        t += n

    add("query", dr.randint(lo, hi))
    commit_end, post_start = [], []
    for k in range(turns):
        add("reason", dr.randint(max(lo, cfg.W), max(hi, cfg.W)))
        add("call", dr.randint(lo, hi))
        commit_end.append(t)
        add("obs", dr.randint(lo, hi))
        post_start.append(t)
    add("reason", dr.randint(max(lo, cfg.W), max(hi, cfg.W)))
    tl = Timeline(cfg, seed, turns, ev, np.asarray(commit_end, np.int32), np.asarray(post_start, np.int32))
    if values:
        bf = cfg.dtype == "bf16"
        S, M, H, Hq, W, d = tl.S, cfg.M, cfg.H, cfg.Hq, cfg.W, cfg.d
        tl.K = normal(seed, _stream(0, _T_TIMELINE + 1), (M, H, S, d), bf16=bf)
        tl.V = normal(seed, _stream(0, _T_TIMELINE + 2), (M, H, S, d), bf16=bf)
        tl.Q_pre = normal(seed, _stream(0, _T_TIMELINE + 3), (turns, M, Hq, W, d), bf16=bf)
        tl.Q_post = normal(seed, _stream(0, _T_TIMELINE + 4), (turns, M, Hq, W, d), bf16=bf)
        tl.fill = uniform_array(seed, _stream(0, _T_TIMELINE + 5), S)
        tl.Q_tok = normal(seed, _stream(0, _T_TIMELINE + 6), (S, M, Hq, d), bf16=bf)
    return tl


def timeline_steps(tl: Timeline, decode_every: int = 0):
    """The order in which a timeline is fed to a lifecycle session:
    ("append", a, b) the tokens [a, b); ("pre", t) commit t's pre-commit
    measurement; ("checkpoint",) a compression checkpoint (taken when the
    resident tokens exceed the budget); ("post", t) commit t's post-commit
    measurement and decisions.  With decode_every > 0, appends are also cut
    at the end of the first reasoning or tool-call event after every
    decode_every decoded tokens (Timeline.decoded), and ("decode_checkpoint",
    end) follows each such cut: the compression cadence of the paper's
    setting (every 128 decoded tokens), taken at event boundaries so that a
    cut never splits an event's pages, its fill scored by the window of the
    last W positions before end."""
    steps, t0 = [], 0
    count, due = 0, decode_every

    def append(a, b):
        nonlocal count, due
        if not decode_every:
            steps.append(("append", a, b))
            return
        p = a
        ends = sorted(s + n for kind, s, n in tl.events if kind in ("reason", "call") and a < s + n <= b)
        for e in ends:
            if count + tl.decoded(p, e) >= due and e >= tl.cfg.W:
                count += tl.decoded(p, e)
                steps.append(("append", p, e))
                steps.append(("decode_checkpoint", e))
                while due <= count:
                    due += decode_every
                p = e
        if p < b:
            count += tl.decoded(p, b)
            steps.append(("append", p, b))

    for k in range(tl.turns):
        append(t0, int(tl.commit_end[k]))
        t0 = int(tl.commit_end[k])
        steps.append(("pre", k))
        steps.append(("checkpoint",))
        end = int(tl.post_start[k]) + tl.cfg.W
        append(t0, end)
        t0 = end
        steps.append(("post", k))
    return steps


def timeline_events(tl: Timeline, a: int, b: int):
    """The paged events (tool calls, observations) that lie in [a, b)."""
    return [(k, s, n) for k, s, n in tl.events if k in ("call", "obs") and a <= s and s + n <= b]
