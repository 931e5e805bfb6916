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
