"""CommitKV CPU oracle — TEST INFRASTRUCTURE ONLY (see package docstring).

fp64 throughout.  Deletion effects come from ``commitkv_oracle.c`` (plain
C, pthreads over (layer, query head) units); lifecycle classification,
pending protection, index selection and the gather are written here in
numpy, one step of the paper at a time.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "commitkv_oracle.c")
_SO = os.path.join(_HERE, "_build", "liboracle.so")

# lifecycle states of Eq. 10 (0 = page outside E_c, i.e. not measurable in
# both windows)
STATE_NONE = 0
STATE_CANDIDATE = 1
STATE_DORMANT = 2
STATE_NEWLY_ACTIVE = 3
STATE_STILL_ACTIVE = 4
STATE_UNCERTAIN = 5


def build(force: bool = False) -> str:
    """Compile the C part of the oracle with gcc (no GPU, no CUDA)."""
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
             "-o", tmp, _SRC, "-lm", "-lpthread"])
        os.replace(tmp, _SO)
    return _SO


class _Prob(ctypes.Structure):
    _fields_ = [
        ("M", ctypes.c_int32), ("H", ctypes.c_int32), ("Hq", ctypes.c_int32),
        ("d", ctypes.c_int32), ("S", ctypes.c_int32), ("W", ctypes.c_int32),
        ("P", ctypes.c_int32),
        ("K", ctypes.c_void_p), ("V", ctypes.c_void_p), ("pos", ctypes.c_void_p),
        ("Q", ctypes.c_void_p), ("qpos", ctypes.c_void_p),
        ("page_start", ctypes.c_void_p), ("page_len", ctypes.c_void_p),
        ("layer_mask", ctypes.c_void_p), ("scale", ctypes.c_double),
    ]


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.POINTER(_Prob)
        vp, ci, cd = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
        lib.okv_effects_explicit.argtypes = [P, vp, ci]
        lib.okv_effects_closed.argtypes = [P, vp, ci]
        lib.okv_row_stats.argtypes = [P, vp, vp, vp, vp, ci]
        lib.okv_set_effect_explicit.argtypes = [P, vp, vp, ci]
        lib.okv_set_effect_explicit.restype = cd
        lib.okv_greedy_explicit.argtypes = [P, vp, ci, cd, vp, vp, ci]
        lib.okv_greedy_closed.argtypes = [P, vp, vp, vp, vp, vp, ci, cd, vp, vp, ci]
        _lib = lib
    return _lib


def _ptr(a):
    return a.ctypes.data if a is not None and a.size else None


class Problem:
    """One cache and one probe window, fp64.

    K, V : [M][H][S][d]   keys and values of the resident tokens
    pos  : [S]            absolute positions (p_i in Eq. 6)
    Q    : [M][Hq][W][d]  probe queries (already position-encoded)
    qpos : [W]            absolute positions of the probe queries (p in Eq. 6)
    page_start, page_len : [P] pages as resident-index spans
    layer_mask : [M] or None — layers that take part in the max
    scale : softmax scale (default 1/sqrt(d))
    """

    def __init__(self, K, V, pos, Q, qpos, page_start, page_len, layer_mask=None, scale=None):
        self.K = np.ascontiguousarray(K, dtype=np.float64)
        self.V = np.ascontiguousarray(V, dtype=np.float64)
        self.Q = np.ascontiguousarray(Q, dtype=np.float64)
        self.pos = np.ascontiguousarray(pos, dtype=np.int32)
        self.qpos = np.ascontiguousarray(qpos, dtype=np.int32)
        self.page_start = np.ascontiguousarray(page_start, dtype=np.int32)
        self.page_len = np.ascontiguousarray(page_len, dtype=np.int32)
        M, H, S, d = self.K.shape
        Mq, Hq, W, dq = self.Q.shape
        assert self.V.shape == self.K.shape and Mq == M and dq == d and Hq % H == 0
        assert self.pos.shape == (S,) and self.qpos.shape == (W,)
        assert self.page_start.shape == self.page_len.shape
        self.M, self.H, self.Hq, self.d, self.S, self.W = M, H, Hq, d, S, W
        self.P = int(self.page_start.shape[0])
        self.layer_mask = None if layer_mask is None else np.ascontiguousarray(layer_mask, dtype=np.uint8)
        self.scale = float(1.0 / np.sqrt(d) if scale is None else scale)
        self._s = _Prob(M, H, Hq, d, S, W, self.P, _ptr(self.K), _ptr(self.V), _ptr(self.pos),
                        _ptr(self.Q), _ptr(self.qpos), _ptr(self.page_start), _ptr(self.page_len),
                        _ptr(self.layer_mask), self.scale)

    @property
    def rows(self):
        return self.M * self.Hq * self.W

    def layers_on(self):
        return np.ones(self.M, bool) if self.layer_mask is None else self.layer_mask.astype(bool)


def _threads(n):
    return int(n) if n else (os.cpu_count() or 1)


def effects(pb: Problem, mode: str = "explicit", nthreads=None) -> np.ndarray:
    """R_h(E; Q) of Eq. 7 for every (layer, query head, page): [M][Hq][P]."""
    lib = _load()
    out = np.zeros((pb.M, pb.Hq, pb.P), np.float64)
    fn = {"explicit": lib.okv_effects_explicit, "closed": lib.okv_effects_closed}[mode]
    if fn(ctypes.byref(pb._s), _ptr(out), _threads(nthreads)) != 0:
        raise ValueError("oracle: invalid problem")
    return out


def page_effects(pb: Problem, mode: str = "explicit", nthreads=None):
    """R(E; Q) = max over query heads (Eq. 7) and over the selected layers.

    Returns (R [P], R_head [M][Hq][P])."""
    R_head = effects(pb, mode, nthreads)
    on = pb.layers_on()
    if pb.P == 0:
        return np.zeros(0), R_head
    R = R_head[on].reshape(-1, pb.P).max(axis=0) if on.any() else np.zeros(pb.P)
    return R, R_head


def row_stats(pb: Problem, nthreads=None):
    """Per-row (layer, query head, window position) softmax statistics:
    m = max scaled score, l = sum exp(s - m), o = normalised output,
    n = number of visible tokens."""
    lib = _load()
    rows = pb.rows
    m = np.zeros(rows); l = np.zeros(rows)
    o = np.zeros((rows, pb.d)); n = np.zeros(rows, np.int32)
    if lib.okv_row_stats(ctypes.byref(pb._s), _ptr(m), _ptr(l), _ptr(o), _ptr(n), _threads(nthreads)):
        raise ValueError("oracle: invalid problem")
    return m, l, o, n


def token_scores(pb: Problem) -> np.ndarray:
    """Per-token fill score (the reading taken for the budget fill of Eq. 13,
    which the paper leaves open; a window-attention score in the spirit of
    SnapKV, which the paper cites for its probe windows): token i scores
    the largest attention weight a_{p,i} = exp(s_{p,i} - m_p) / l_p it gets
    from any window position p of any query head of a selected layer, and 0
    when no query sees it.  Written from the softmax row by row in numpy.
    Parity unpinned against the paper, which defines no fill score; pinned
    against the mathematics (uniform attention, invariants, the C row
    statistics)."""
    score = np.zeros(pb.S)
    g = pb.Hq // pb.H
    on = pb.layers_on()
    for li in range(pb.M):
        if not on[li]:
            continue
        for h in range(pb.Hq):
            Kh = pb.K[li, h // g]
            for w in range(pb.W):
                vis = pb.pos <= pb.qpos[w]
                if not vis.any():
                    continue
                s_ = pb.scale * (Kh[vis] @ pb.Q[li, h, w])
                e = np.exp(s_ - s_.max())
                idx = np.flatnonzero(vis)
                score[idx] = np.maximum(score[idx], e / e.sum())
    return score


def _drop_mask(pb: Problem, pages) -> np.ndarray:
    drop = np.zeros(pb.S, np.uint8)
    for E in pages:
        drop[pb.page_start[E]: pb.page_start[E] + pb.page_len[E]] = 1
    return drop


def set_effect(pb: Problem, pages, nthreads=None):
    """R(A; Q) with every token of the page set A deleted at once (the
    quantity tested in Eq. 11), by explicit deletion.  Returns
    (R, R_unit [M][Hq])."""
    lib = _load()
    drop = _drop_mask(pb, pages)
    R_unit = np.zeros((pb.M, pb.Hq))
    R = lib.okv_set_effect_explicit(ctypes.byref(pb._s), _ptr(drop), _ptr(R_unit), _threads(nthreads))
    if R < 0:
        raise ValueError("oracle: invalid problem")
    return R, R_unit


def greedy(pb: Problem, cand, tau: float, mode: str = "explicit", stats=None, nthreads=None):
    """Greedy joint test (Eq. 11; inner loop of Algorithm 1).

    Candidates are examined in the given order; E is accepted iff
    R(D u {E}) <= tau, and a rejection does not stop the scan.
    Returns (accepted [P] uint8, step_R [len(cand)]) where step_R[j] is
    R(D u {cand[j]}) for the D accepted before step j."""
    lib = _load()
    cand = np.ascontiguousarray(cand, dtype=np.int32)
    acc = np.zeros(pb.P, np.uint8)
    step = np.zeros(len(cand))
    if mode == "explicit":
        rc = lib.okv_greedy_explicit(ctypes.byref(pb._s), _ptr(cand), len(cand), float(tau),
                                     _ptr(acc), _ptr(step), _threads(nthreads))
    else:
        m, l, o, n = row_stats(pb, nthreads) if stats is None else stats
        m = np.ascontiguousarray(m, np.float64); l = np.ascontiguousarray(l, np.float64)
        o = np.ascontiguousarray(o, np.float64); n = np.ascontiguousarray(n, np.int32)
        rc = lib.okv_greedy_closed(ctypes.byref(pb._s), _ptr(m), _ptr(l), _ptr(o), _ptr(n),
                                   _ptr(cand), len(cand), float(tau), _ptr(acc), _ptr(step),
                                   _threads(nthreads))
    if rc != 0:
        raise ValueError("oracle: invalid problem or candidate")
    return acc, step


# --------------------------------------------------------------------------
# lifecycle classification, Eq. 9-10


def _f32(x) -> float:
    """Thresholds travel as fp32 through the library's C struct; the oracle
    compares against the same rounded values."""
    return float(np.float32(x))


def percentile_ranks(R, idx) -> np.ndarray:
    """P(E) for E in E_c (= idx): the fraction of pages of E_c whose effect
    is strictly smaller than R(E).  Ties share the lower rank."""
    Rc = np.asarray(R, np.float64)[idx]
    n = len(idx)
    k = np.array([int(np.count_nonzero(Rc < x)) for x in Rc], dtype=np.int64)
    return k / float(n) if n else np.zeros(0)


def classify(R_pre, R_post, eligible, tau_use=0.05, tau_dead=0.01, rho_use=0.75, rho_dead=0.25,
             no_precommit=False, no_percentile=False):
    """Lifecycle states of Eq. 10 and the ordered completion candidates.

    eligible marks E_c, the pages measurable in both windows.  States:
    STATE_NONE outside E_c, else candidate / dormant / newly active /
    still active / uncertain.  Candidates are ordered by increasing R+,
    then decreasing R-, then increasing page index.

    The ablations of Section 4.4: no_percentile drops the percentile
    conditions from H and L (absolute thresholds only); no_precommit takes
    as candidates every page with L+ instead of H- and L+ (the states are
    unchanged)."""
    R_pre = np.asarray(R_pre, np.float64)
    R_post = np.asarray(R_post, np.float64)
    P = R_pre.shape[0]
    assert R_post.shape == (P,)
    if np.isnan(R_pre).any() or np.isnan(R_post).any():
        raise ValueError("NaN effect")
    t_use, t_dead, r_use, r_dead = _f32(tau_use), _f32(tau_dead), _f32(rho_use), _f32(rho_dead)
    if not (t_dead < t_use and r_dead < r_use):
        raise ValueError("thresholds must satisfy tau_dead < tau_use and rho_dead < rho_use")
    idx = np.flatnonzero(np.asarray(eligible, bool))
    state = np.zeros(P, np.uint8)
    if len(idx) == 0:
        return state, np.zeros(0, np.int32)
    Pm = percentile_ranks(R_pre, idx)
    Pp = percentile_ranks(R_post, idx)
    Rm, Rp = R_pre[idx], R_post[idx]
    if no_percentile:
        Pm = np.full(len(idx), 0.5)  # inside every percentile condition below
        Pp = np.full(len(idx), 0.5)
        r_use, r_dead = 0.0, 1.0
    Hm = (Rm >= t_use) & (Pm >= r_use)
    Lm = (Rm <= t_dead) & (Pm <= r_dead)
    Hp = (Rp >= t_use) & (Pp >= r_use)
    Lp = (Rp <= t_dead) & (Pp <= r_dead)
    st = np.full(len(idx), STATE_UNCERTAIN, np.uint8)
    st[Hm & Lp] = STATE_CANDIDATE
    st[Lm & Lp] = STATE_DORMANT
    st[Lm & Hp] = STATE_NEWLY_ACTIVE
    st[Hm & Hp] = STATE_STILL_ACTIVE
    state[idx] = st
    cand = idx[Lp] if no_precommit else idx[st == STATE_CANDIDATE]
    order = sorted(cand.tolist(), key=lambda E: (R_post[E], -R_pre[E], E))
    return state, np.asarray(order, np.int32)


# --------------------------------------------------------------------------
# pending protection (Eq. 12), retained indices (Eq. 13), gather (Eq. 4)


def protect_pending(page_start, page_len, retired, pending, priority, B_N, cap_pages):
    """N_j: pending pages ordered by decreasing pre-commit effect (then page
    index), after dropping retired ones; the longest prefix whose page count
    is <= cap_pages and whose token total is <= B_N.  Returns the page list."""
    pending = [int(E) for E in pending]
    priority = [float(x) for x in priority]
    assert len(pending) == len(priority) and len(set(pending)) == len(pending)
    if any(np.isnan(priority)):
        raise ValueError("NaN priority")
    live = [(E, p) for E, p in zip(pending, priority) if not retired[E]]
    live.sort(key=lambda t: (-t[1], t[0]))
    out, tokens = [], 0
    for E, _ in live:
        if len(out) + 1 > cap_pages or tokens + int(page_len[E]) > B_N:
            break
        out.append(E)
        tokens += int(page_len[E])
    return out


def select_indices(S, page_start, page_len, retired, pending, priority, fill_score, B, B_N, cap_pages):
    """I_j of Eq. 13 (ascending int32).

    Tokens of retired pages are excluded; the protected pending tokens N_j
    are kept; the remaining budget B - |N_j| is filled with the other
    tokens of highest fill score (ties: higher index first); if they all
    fit, all are kept."""
    assert 0 <= B_N <= B and cap_pages >= 0
    page_start = np.asarray(page_start, np.int64)
    page_len = np.asarray(page_len, np.int64)
    retired = np.asarray(retired, bool)
    fill_score = np.asarray(fill_score, np.float32)
    if np.isnan(fill_score).any():
        raise ValueError("NaN fill score")
    tok_retired = np.zeros(S, bool)
    for E in np.flatnonzero(retired):
        tok_retired[page_start[E]: page_start[E] + page_len[E]] = True
    protected_pages = protect_pending(page_start, page_len, retired, pending, priority, B_N, cap_pages)
    tok_protected = np.zeros(S, bool)
    for E in protected_pages:
        tok_protected[page_start[E]: page_start[E] + page_len[E]] = True
    rest = np.flatnonzero(~tok_retired & ~tok_protected)
    room = B - int(tok_protected.sum())
    if len(rest) > room:
        ranked = sorted(rest.tolist(), key=lambda i: (-float(fill_score[i]), -i))
        rest = np.asarray(ranked[:room], np.int64)
    keep = np.zeros(S, bool)
    keep[tok_protected] = True
    keep[rest] = True
    return np.flatnonzero(keep).astype(np.int32)


def gather(K, V, pos, I):
    """Eq. 4: the same index set applied to keys, values and positions."""
    I = np.asarray(I, np.int64)
    return K[:, :, I, :], V[:, :, I, :], np.asarray(pos)[I]
