"""The oracle's multi-commit driver (Algorithm 1's outer loop) against the
invariants of Eq. 4 and Eq. 12-13 over a seeded multi-turn timeline (CPU)."""
import numpy as np

from oracle.lifecycle import OracleSession
from paper_2608_07855_gb300 import synth

TH = dict(tau_use=1.0, tau_dead=0.6, rho_use=0.75, rho_dead=0.5)


def test_oracle_lifecycle_invariants():
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16, M=1, H=1, Hq=4)
    tl = synth.make_timeline(cfg, 3, 4)
    B = 200
    o = OracleSession(cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.G, B, 0.25, protect_cap=4, thresholds=TH,
                      no_precommit=True, tau_joint=0.6)
    K = synth.values_f64(tl.K, cfg.dtype)
    V = synth.values_f64(tl.V, cfg.dtype)
    first_pos = {}  # page id -> its positions when it was cut
    gone = set()
    n_ck = n_acc = 0
    for step in synth.timeline_steps(tl):
        if step[0] == "append":
            a, b = step[1], step[2]
            n0 = len(o.pages)
            o.append(K[:, :, a:b], V[:, :, a:b], np.arange(a, b), synth.timeline_events(tl, a, b))
            for pid, s, n in o.pages[n0:]:
                first_pos[pid] = set(o.pos[s:s + n].tolist())
        elif step[0] == "pre":
            o.pre_commit(synth.values_f64(tl.Q_pre[step[1]], cfg.dtype), tl.qpos_pre(step[1]))
        elif step[0] == "checkpoint":
            if o.pos.shape[0] <= B:
                continue
            waiting = [pid for pid in o.measured if pid not in o.retired]
            retired = set(o.retired)
            before = {pid: set(o.pos[s:s + n].tolist()) for pid, s, n in o.pages}
            I = o.checkpoint(tl.fill)
            n_ck += 1
            assert len(I) <= B and np.all(np.diff(I) > 0)
            assert np.all(np.diff(o.pos) > 0)
            # every resident row holds the timeline's K and V at its position
            assert np.array_equal(o.K, K[:, :, o.pos]) and np.array_equal(o.V, V[:, :, o.pos])
            ids = o.page_ids()
            assert not (set(ids) & retired), "retired pages are dropped"
            gone |= retired
            for pid, s, n in o.pages:
                pos = o.pos[s:s + n]
                # a page's retained tokens are contiguous in resident order (its
                # span); their positions are a subset of the page's own
                assert np.all(np.diff(pos) > 0)
                assert set(pos.tolist()) <= first_pos[pid]
            # the protected pages (a prefix of the waiting ones by R-) are kept whole
            order = sorted(waiting, key=lambda pid: (-np.float32(o.R_pre[pid]), pid))
            kept_tok = 0
            for k, pid in enumerate(order):
                n = len(before[pid])
                if k >= o.protect_cap or kept_tok + n > o.B_N:
                    break
                kept_tok += n
                span = {q[0]: q for q in o.pages}[pid]
                assert set(o.pos[span[1]:span[1] + span[2]].tolist()) == before[pid], "protected page kept whole"
        else:
            out = o.post_commit(synth.values_f64(tl.Q_post[step[1]], cfg.dtype), tl.qpos_post(step[1]))
            assert set(out["accepted"]) <= set(out["cand"])
            assert len(out["cand"]) <= o.scan_cap
            assert not (set(out["cand"]) & gone)
            n_acc += len(out["accepted"])
    assert n_ck >= 2 and n_acc >= 1, (n_ck, n_acc)


def _hand():
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "lifecycle_hand.json")) as f:
        return json.load(f)


def _val(expr):
    """A hand-derived closed form of the golden file: '0' or 'sqrt(a/b)'."""
    from fractions import Fraction
    if expr == "0":
        return 0.0
    assert expr.startswith("sqrt(") and expr.endswith(")")
    return float(np.sqrt(float(Fraction(expr[5:-1]))))


def _run_hand(g, scan_cap=None):
    """Drives an OracleSession through the golden timeline; yields
    (step, session, output) after every step."""
    s = g["setup"]
    o = OracleSession(s["M"], s["H"], s["Hq"], s["d"], s["G"], s["B"], s["eta"],
                      scan_cap=s["scan_cap"] if scan_cap is None else scan_cap,
                      protect_cap=s["protect_cap"], thresholds=s["thresholds"], tau_joint=s["tau_joint"])
    vals = np.asarray(s["values"], np.float64)
    events = [tuple(e) for e in s["events"]]
    Q = np.ones((s["M"], s["Hq"], s["W"], s["d"]))  # K = 0: every score is 0 whatever Q is
    for step in s["steps"]:
        if step[0] == "append":
            a, b = step[1], step[2]
            n = b - a
            K = np.zeros((s["M"], s["H"], n, s["d"]))
            V = np.broadcast_to(vals[a:b], (s["M"], s["H"], n, s["d"])).copy()
            o.append(K, V, np.arange(a, b), [e for e in events if e[0] in ("call", "obs") and a <= e[1]
                                              and e[1] + e[2] <= b])
            continue
        if step[0] == "pre":
            out = o.pre_commit(Q, [step[1]])
        elif step[0] == "checkpoint":
            out = o.checkpoint(s["fill"]) if o.pos.shape[0] > s["B"] else None
        else:
            out = o.post_commit(Q, [step[1]])
        yield step[0], o, out


def test_hand_worked_timeline():
    """Two commits on a five-page cache whose effects are exact closed forms
    (tests/golden/lifecycle_hand.json): E_c at each post-commit (measured at
    the latest pre-commit, not retired, the new observation excluded), the
    pending set and its protection, the page spans after a checkpoint that
    keeps part of a page, D_c growing at an acceptance and shrinking when
    its page is compacted away, and a joint-test rejection."""
    g = _hand()
    exp = iter(g["expected"])
    for kind, o, out in _run_hand(g):
        e = next(exp)
        assert e["step"] == kind
        if kind == "pre":
            assert o.page_ids() == e["page_ids"]
            np.testing.assert_allclose(out, [_val(x) for x in e["R"]], rtol=1e-12, atol=1e-14)
            assert sorted(o.measured) == e["measured"]
        elif kind == "checkpoint":
            assert (out is not None) == e["taken"]
            if e["taken"]:
                assert out.tolist() == e["I"]
                assert o.pos.tolist() == e["pos"]
                assert o.pages == e["pages"]
                assert sorted(o.retired) == e["retired"]
        else:
            assert o.page_ids() == e["page_ids"]
            np.testing.assert_allclose(out["R_post"], [_val(x) for x in e["R_post"]], rtol=1e-12, atol=1e-14)
            assert out["eligible"] == e["eligible"]
            assert out["state"].tolist() == e["state"]
            assert out["cand"] == e["cand"] and out["accepted"] == e["accepted"]
            np.testing.assert_allclose(out["step_R"], [_val(x) for x in e["step_R"]], rtol=1e-12, atol=1e-14)
            assert sorted(o.retired) == e["retired"]
    assert next(exp, None) is None


def test_hand_worked_timeline_scan_cap():
    """The ordered candidate list is cut to scan_cap pages (the paper scans
    at most 64 per commit): with a cap of 0 commit 1 accepts nothing."""
    g = _hand()
    want = g["scan_cap_zero"]
    posts = 0
    for kind, o, out in _run_hand(g, scan_cap=0):
        if kind == "post":
            posts += 1
            if posts == want["commit"]:
                assert out["cand"] == want["cand"] and out["accepted"] == want["accepted"]
                assert not o.retired
                return
    raise AssertionError("no post-commit step")


def test_decode_cadence_steps():
    """timeline_steps with a decode cadence: the same appends (cut further),
    commits and checkpoints in the same order; a decode checkpoint after
    each cut at the end of a reasoning or tool-call event once another
    decode_every decoded tokens are in."""
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16, M=1, H=1, Hq=4)
    tl = synth.make_timeline(cfg, 3, 4, values=False)
    plain = synth.timeline_steps(tl)
    steps = synth.timeline_steps(tl, 40)
    assert [x for x in steps if x[0] not in ("append", "decode_checkpoint")] == \
        [x for x in plain if x[0] != "append"]
    ends = {s + n for k, s, n in tl.events if k in ("reason", "call")}
    pos, last = 0, 0
    n_dc = 0
    for x in steps:
        if x[0] == "append":
            assert x[1] == pos
            pos = x[2]
        elif x[0] == "decode_checkpoint":
            assert x[1] == pos and x[1] in ends
            assert tl.decoded(last, x[1]) >= 40 or last == 0
            last = x[1]
            n_dc += 1
    assert n_dc >= 3
    assert pos == [x for x in plain if x[0] == "append"][-1][2]


def test_oracle_decode_checkpoint_keeps_the_most_attended_tokens():
    """A decode checkpoint fills the budget by the window's attention: among
    the tokens that are neither retired nor protected, every kept token
    scores at least as high as every dropped one (ties by index)."""
    from oracle import core
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16, M=1, H=1, Hq=4)
    tl = synth.make_timeline(cfg, 4, 3)
    K64, V64 = synth.values_f64(tl.K, cfg.dtype), synth.values_f64(tl.V, cfg.dtype)
    o = OracleSession(cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.G, 160, 0.125, protect_cap=0, thresholds=TH)
    end = int(tl.commit_end[1])
    o.append(K64[:, :, :end], V64[:, :, :end], np.arange(end), synth.timeline_events(tl, 0, end))
    q, qp = tl.window(end)
    fill = o.fill_scores(synth.values_f64(q, cfg.dtype), qp)
    assert fill.shape == (end,) and (fill > 0).all() and (fill <= 1).all()
    pb = o._problem(synth.values_f64(q, cfg.dtype), qp)
    assert np.array_equal(fill, core.token_scores(pb))
    I = o.decode_checkpoint(synth.values_f64(q, cfg.dtype), qp)
    assert len(I) == 160
    kept = np.zeros(end, bool)
    kept[I] = True
    f32 = fill.astype(np.float32)
    assert f32[kept].min() >= f32[~kept].max()


def test_decode_checkpoint_after_a_commit_protects_nothing():
    """Once a commit's post-commit decisions are taken no page awaits its
    measurement, so a decode checkpoint has no pending set to protect (Eq. 12's
    N_j is empty) even with a protection cap: among the tokens that are not
    retired, the budget goes to the highest fill scores alone."""
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16, M=1, H=1, Hq=4)
    tl = synth.make_timeline(cfg, 4, 3)
    K64, V64 = synth.values_f64(tl.K, cfg.dtype), synth.values_f64(tl.V, cfg.dtype)
    B = 160
    o = OracleSession(cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.G, B, 0.25, protect_cap=4, thresholds=TH, tau_joint=0.6)
    end, posted = 0, False
    for step in synth.timeline_steps(tl):
        if step[0] == "append":
            a, b = step[1], step[2]
            o.append(K64[:, :, a:b], V64[:, :, a:b], np.arange(a, b), synth.timeline_events(tl, a, b))
            end = b
            if posted:
                break  # the tokens decoded after the first commit's decisions
        elif step[0] == "pre":
            o.pre_commit(synth.values_f64(tl.Q_pre[step[1]], cfg.dtype), tl.qpos_pre(step[1]))
        elif step[0] == "post":
            o.post_commit(synth.values_f64(tl.Q_post[step[1]], cfg.dtype), tl.qpos_post(step[1]))
            posted = True
    assert posted and o.measured == []
    q, qp = tl.window(end)
    q64 = synth.values_f64(q, cfg.dtype)
    fill = o.fill_scores(q64, qp).astype(np.float32)
    retired_tok = np.zeros(o.pos.shape[0], bool)
    for pid, s, n in o.pages:
        if pid in o.retired:
            retired_tok[s:s + n] = True
    live = ~retired_tok
    assert live.sum() > B
    I = o.decode_checkpoint(q64, qp)
    assert len(I) == B
    kept = np.zeros(fill.shape[0], bool)
    kept[I] = True
    assert not kept[retired_tok].any()
    assert fill[kept & live].min() >= fill[~kept & live].max()
