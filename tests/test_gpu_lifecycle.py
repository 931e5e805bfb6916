"""Multi-commit lifecycle driver (Algorithm 1's outer loop) against the
oracle's driver, over seeded multi-turn timelines.

Both sessions get the same appends, windows and checkpoints
(synth.timeline_steps).  Compared at every step: page effects (tolerance of
bf16 inputs), candidate lists and accepted pages (exact), retained indices,
positions and page tables after each checkpoint (exact).  A decision of the
oracle inside the tolerance margin (a classification threshold or
percentile, or a joint-test threshold) may go either way on the GPU, after
which the two sessions may legitimately differ; the comparison stops at the
first such commit and must have covered at least two commits.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle.lifecycle import OracleSession  # noqa: E402
from paper_2608_07855_gb300 import commitkv as ck  # noqa: E402
from paper_2608_07855_gb300 import synth  # noqa: E402
from paper_2608_07855_gb300.lifecycle import Session  # noqa: E402
from paper_2608_07855_gb300.workload import shape_of  # noqa: E402

from oracle_bridge import rel_close, safe_threshold_mask  # noqa: E402

pytestmark = pytest.mark.gpu
TOL = 2e-2
# Random values give effects of a few tenths; the ablations of Section 4.4
# 'w/o pre-commit state' and 'w/o percentile calibration' make the
# candidates the pages with R+ <= tau_dead, with tau_joint below it so that
# the scan both accepts and rejects; 'w/o transition protection' (cap 0)
# keeps the checkpoints free of near-ties in R- (protection has its own
# parity tests).


def _np(t):
    return t.detach().cpu().numpy()


def _dev(a, bf16):
    t = torch.from_numpy(np.ascontiguousarray(a))
    return (t.view(torch.bfloat16) if bf16 else t).cuda()


def _decisions_safe(o_out, tau_dead, tau_joint):
    """Whether every decision of the oracle's post-commit step clears the
    tolerance margin: the L+ threshold of every measured page and the joint
    test's threshold at every scanned candidate."""
    Rp, el = o_out["R_post"], o_out["eligible"]
    idx = np.flatnonzero(el)
    if len(idx) and not safe_threshold_mask(Rp[idx], tau_dead, TOL).all():
        return False
    return bool(safe_threshold_mask(o_out["step_R"], tau_joint, TOL).all())


def _protection_safe(orc):
    """Whether the oracle's protected prefix (waiting pages by decreasing
    R-, within B_N tokens and the page cap) has a margin at its cut: the
    last page inside and the first page outside differ by more than twice
    the tolerance."""
    wait = set(orc.measured)
    cand = [(orc.R_pre[pid], n) for pid, s, n in orc.pages if pid in wait and pid not in orc.retired]
    cand.sort(key=lambda x: -x[0])
    k, tok = 0, 0
    while k < len(cand) and k < orc.protect_cap and tok + cand[k][1] <= orc.B_N:
        tok += cand[k][1]
        k += 1
    if 0 < k < len(cand):
        a, b = cand[k - 1][0], cand[k][0]
        return abs(a - b) > 2 * TOL * max(abs(a), abs(b))
    return True


@pytest.mark.parametrize("seed,tau_dead,tau_joint", [(0, 0.45, 0.3), (7, 0.5, 0.35), (9, 0.45, 0.3)])
def test_lifecycle_against_oracle(seed, tau_dead, tau_joint):
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16)
    tl = synth.make_timeline(cfg, seed, 5)
    bf = cfg.dtype == "bf16"
    B, eta, cap = 256, 0.125, tl.S
    TH = dict(tau_use=1.0, tau_dead=tau_dead, rho_use=0.75, rho_dead=0.5)
    variant = ck.COMMITKV_CLASSIFY_NO_PRECOMMIT | ck.COMMITKV_CLASSIFY_NO_PERCENTILE
    gpu = Session(shape_of(cfg), cfg.G, B, eta, capacity=cap, protect_cap=0, thresholds=ck.Thresholds(**TH),
                  variant=variant, tau_joint=tau_joint)
    orc = OracleSession(cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.G, B, eta, protect_cap=0, thresholds=TH,
                        no_precommit=True, no_percentile=True, tau_joint=tau_joint)
    K64, V64 = synth.values_f64(tl.K, cfg.dtype), synth.values_f64(tl.V, cfg.dtype)
    Kd, Vd = _dev(tl.K, bf), _dev(tl.V, bf)
    fill_d = torch.from_numpy(tl.fill).cuda()
    commits, checkpoints, n_acc, n_rej = 0, 0, 0, 0
    for step in synth.timeline_steps(tl):
        if step[0] == "append":
            a, b = step[1], step[2]
            ev = synth.timeline_events(tl, a, b)
            pos = np.arange(a, b, dtype=np.int32)
            gpu.append(Kd[:, :, a:b], Vd[:, :, a:b], torch.from_numpy(pos).cuda(), ev)
            orc.append(K64[:, :, a:b], V64[:, :, a:b], pos, ev)
        elif step[0] == "pre":
            t = step[1]
            Rg = gpu.pre_commit(_dev(tl.Q_pre[t], bf), torch.from_numpy(tl.qpos_pre(t)).cuda())
            Ro = orc.pre_commit(synth.values_f64(tl.Q_pre[t], cfg.dtype), tl.qpos_pre(t))
            assert gpu.page_ids() == orc.page_ids()
            assert rel_close(_np(Rg), Ro, TOL).all(), f"R- at commit {t}"
        elif step[0] == "checkpoint":
            assert gpu.S == orc.pos.shape[0]
            if gpu.S <= B:
                continue
            if not _protection_safe(orc):
                break  # the protected sets may differ from here on
            Ig = gpu.checkpoint(fill_d[gpu.pos[:gpu.S].long()])
            Io = orc.checkpoint(tl.fill)
            assert np.array_equal(_np(Ig), Io)
            assert np.array_equal(_np(gpu.pos[:gpu.S]), orc.pos)
            assert gpu.pages == orc.pages
            checkpoints += 1
        else:
            t = step[1]
            og = gpu.post_commit(_dev(tl.Q_post[t], bf), torch.from_numpy(tl.qpos_post(t)).cuda())
            el_o = np.asarray([pid in set(orc.measured) and pid not in orc.retired for pid in orc.page_ids()])
            oo = orc.post_commit(synth.values_f64(tl.Q_post[t], cfg.dtype), tl.qpos_post(t))
            oo["eligible"] = el_o
            assert rel_close(_np(og["R_post"]), oo["R_post"], TOL).all(), f"R+ at commit {t}"
            if not _decisions_safe(oo, tau_dead, tau_joint):
                break  # the two sessions may part from here on
            assert og["cand"] == oo["cand"], f"candidates at commit {t}"
            assert og["accepted"] == oo["accepted"], f"accepted at commit {t}"
            assert rel_close(np.asarray(og["step_R"]), oo["step_R"], TOL).all()
            commits += 1
            n_acc += len(oo["accepted"])
            n_rej += len(oo["cand"]) - len(oo["accepted"])
    assert commits >= 3 and checkpoints >= 1 and n_acc >= 1 and n_rej >= 1, (commits, checkpoints, n_acc, n_rej)


@pytest.mark.parametrize("seed", [0, 7])
def test_lifecycle_decode_cadence(seed):
    """The same timelines with a checkpoint after every 48 decoded tokens
    (at event ends), the budget filled by each resident token's largest
    attention weight from the latest window: the GPU's fill scores (row
    stats, then commitkv_token_scores) against the oracle's softmax within
    the bf16 tolerance at every decode checkpoint, and the oracle's
    selection, fed the GPU's scores, gives the GPU's retained indices, page
    table and positions exactly; the commits in between as in the test
    above."""
    tau_dead, tau_joint = 0.45, 0.3
    cfg = synth.small_config("timeline", event_len=(24, 80), G=16)
    tl = synth.make_timeline(cfg, seed, 5)
    bf = cfg.dtype == "bf16"
    B, eta, cap = 256, 0.125, tl.S
    TH = dict(tau_use=1.0, tau_dead=tau_dead, rho_use=0.75, rho_dead=0.5)
    variant = ck.COMMITKV_CLASSIFY_NO_PRECOMMIT | ck.COMMITKV_CLASSIFY_NO_PERCENTILE
    gpu = Session(shape_of(cfg), cfg.G, B, eta, capacity=cap, protect_cap=0, thresholds=ck.Thresholds(**TH),
                  variant=variant, tau_joint=tau_joint, checkpoint_every=48)
    orc = OracleSession(cfg.M, cfg.H, cfg.Hq, cfg.d, cfg.G, B, eta, protect_cap=0, thresholds=TH,
                        no_precommit=True, no_percentile=True, tau_joint=tau_joint)
    K64, V64 = synth.values_f64(tl.K, cfg.dtype), synth.values_f64(tl.V, cfg.dtype)
    Kd, Vd = _dev(tl.K, bf), _dev(tl.V, bf)
    fill_d = torch.from_numpy(tl.fill).cuda()
    commits, decode_ckpts = 0, 0
    for step in synth.timeline_steps(tl, 48):
        if step[0] == "append":
            a, b = step[1], step[2]
            ev = synth.timeline_events(tl, a, b)
            pos = np.arange(a, b, dtype=np.int32)
            gpu.append(Kd[:, :, a:b], Vd[:, :, a:b], torch.from_numpy(pos).cuda(), ev, decoded=tl.decoded(a, b))
            orc.append(K64[:, :, a:b], V64[:, :, a:b], pos, ev)
        elif step[0] == "decode_checkpoint":
            assert gpu.decoded_since > 0
            if gpu.S <= B:
                continue
            q, qp = tl.window(step[1])
            fg = gpu.fill_scores(_dev(q, bf), torch.from_numpy(qp).cuda())
            fo = orc.fill_scores(synth.values_f64(q, cfg.dtype), qp)
            assert rel_close(_np(fg), fo, TOL).all(), f"fill scores at {step[1]}"
            Ig = gpu.checkpoint(fg)
            Io = orc.checkpoint_resident(_np(fg))
            assert np.array_equal(_np(Ig), Io)
            assert np.array_equal(_np(gpu.pos[:gpu.S]), orc.pos)
            assert gpu.pages == orc.pages
            assert gpu.decoded_since == 0
            decode_ckpts += 1
        elif step[0] == "pre":
            t = step[1]
            Rg = gpu.pre_commit(_dev(tl.Q_pre[t], bf), torch.from_numpy(tl.qpos_pre(t)).cuda())
            Ro = orc.pre_commit(synth.values_f64(tl.Q_pre[t], cfg.dtype), tl.qpos_pre(t))
            assert rel_close(_np(Rg), Ro, TOL).all(), f"R- at commit {t}"
        elif step[0] == "checkpoint":
            if gpu.S <= B:
                continue
            Ig = gpu.checkpoint(fill_d[gpu.pos[:gpu.S].long()])
            Io = orc.checkpoint(tl.fill)
            assert np.array_equal(_np(Ig), Io)
            assert gpu.pages == orc.pages
        else:
            t = step[1]
            og = gpu.post_commit(_dev(tl.Q_post[t], bf), torch.from_numpy(tl.qpos_post(t)).cuda())
            el_o = np.asarray([pid in set(orc.measured) and pid not in orc.retired for pid in orc.page_ids()])
            oo = orc.post_commit(synth.values_f64(tl.Q_post[t], cfg.dtype), tl.qpos_post(t))
            oo["eligible"] = el_o
            assert rel_close(_np(og["R_post"]), oo["R_post"], TOL).all(), f"R+ at commit {t}"
            if not _decisions_safe(oo, tau_dead, tau_joint):
                break
            assert og["cand"] == oo["cand"] and og["accepted"] == oo["accepted"], f"commit {t}"
            commits += 1
    assert decode_ckpts >= 2 and commits >= 2, (decode_ckpts, commits)
