"""GPU parity of the CommitKV library against the CPU oracle.

Every test calls the CUDA path through the C ABI (the Python binding only
marshals pointers) on seeded synthetic inputs and compares element by
element with the oracle on the same inputs:
  effects R-, R+ and per-(layer, head) maxima: 1e-4 relative for fp32 inputs,
  2e-2 relative for bf16 inputs (fp32 accumulation), infinities and zeros
  exact;
  classification and ordering: bit-exact on the same fp32 effects;
  joint test: step effects within the effect tolerance, and the accepted
  set identical up to the first step whose decision margin |R - tau| / tau
  is within that tolerance;
  selection, gather and positions: bit-exact.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import core  # noqa: E402
from paper_2608_07855_gb300 import commitkv as ck  # noqa: E402
from paper_2608_07855_gb300 import synth  # noqa: E402
from paper_2608_07855_gb300.workload import DeviceTrajectory, StepBuffers  # noqa: E402

from oracle_bridge import (OracleStep, gapped_positions, isclose_tol, rel_close,  # noqa: E402
                           safe_threshold_mask)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    ck.load_library()


def _cfg(name):
    if name == "tiny":
        return synth.CONFIGS["tiny"]
    if name == "small":
        return synth.small_config()
    if name == "small_w40_g16":  # 160 rows per (layer, KV head): ragged row blocks; G = 16
        return synth.small_config("small_w40_g16", W=40, G=16, L_pre=600, L_obs=70, B=256)
    if name == "small_f32":
        return synth.small_config("small_f32", dtype="f32", d=64, H=2, Hq=4, M=1, W=16, G=16,
                                  L_pre=500, L_obs=60, B=200, outlier_channels=0)
    if name == "small_long_pages":  # pages longer than one 64-token tile
        return synth.small_config("small_long_pages", G=100, L_pre=900, L_obs=80, B=400)
    raise KeyError(name)


CASES = [("tiny", 0), ("tiny", 1), ("small", 0), ("small", 1), ("small_w40_g16", 2),
         ("small_f32", 3), ("small_long_pages", 4)]


class Run:
    """GPU step and oracle step on the same trajectory."""

    def __init__(self, name, seed, gapped=False):
        cfg = _cfg(name)
        tr = synth.make_trajectory(cfg, seed)
        if gapped:
            gapped_positions(tr, seed)
        self.cfg, self.tr = cfg, tr
        self.dev = DeviceTrajectory.upload(tr)
        self.buf = StepBuffers(cfg, [self.dev])
        self.orc = OracleStep(tr, "explicit")
        self.tol = isclose_tol(cfg.dtype)


_runs = {}


def get_run(name, seed, gapped=False):
    key = (name, seed, gapped)
    if key not in _runs:
        _runs[key] = Run(name, seed, gapped)
    return _runs[key]


def _np(t):
    return t.detach().cpu().numpy()


def _assert_close(got, want, tol, what):
    ok = rel_close(got, want, tol)
    if not ok.all():
        bad = np.flatnonzero(~ok.ravel())[:8]
        g, w = np.ravel(got), np.ravel(want)
        raise AssertionError(f"{what}: {int((~ok).sum())} of {ok.size} outside {tol}: "
                             + ", ".join(f"[{i}] gpu {g[i]:.6g} oracle {w[i]:.6g}" for i in bad))


@pytest.mark.parametrize("name,seed", CASES)
def test_page_effects(name, seed):
    r = get_run(name, seed)
    cfg, b, dev = r.cfg, r.buf, r.dev
    headR_pre = torch.zeros(cfg.M, cfg.Hq, dev.P_pre, device="cuda")
    headR_post = torch.zeros(cfg.M, cfg.Hq, dev.P_post, device="cuda")
    R_pre = torch.zeros(dev.P_pre, device="cuda")
    ck.commitkv_page_effects(b.shape, [dev.pre()], [R_pre], head_R_out=[headR_pre], workspace=b.ws)
    ck.commitkv_page_effects(b.shape, [dev.post()], b.R_post, head_R_out=[headR_post],
                             stats_out=b.stats, workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    o = r.orc
    _assert_close(_np(R_pre), o.R_pre[:dev.P_pre], r.tol, "R-")
    _assert_close(_np(b.R_post[0]), o.R_post, r.tol, "R+")
    _assert_close(_np(headR_pre), o.H_pre, r.tol, "R- per head")
    _assert_close(_np(headR_post), o.H_post, r.tol, "R+ per head")
    # stats: m, l, n, o of every post-commit probe row
    m, l, o_vec, n = o.stats
    st = _np(b.stats[0]).reshape(-1, cfg.d + 4)
    assert np.array_equal(st[:, 2].astype(np.int64), n)
    _assert_close(st[:, 0], m, 1e-5, "row max")
    _assert_close(st[:, 1], l, 1e-4, "row sum")
    err = np.linalg.norm(st[:, 4:] - o_vec, axis=1) / np.maximum(np.linalg.norm(o_vec, axis=1), 1e-30)
    assert err.max() <= 1e-4, err.max()


@pytest.mark.parametrize("name,seed", CASES)
def test_classify_isolated(name, seed):
    """Oracle effects (rounded to fp32) into the GPU classifier: states and
    candidate order must equal the oracle's classification of the same fp32
    values, bit for bit."""
    r = get_run(name, seed)
    b, dev, o = r.buf, r.dev, r.orc
    Rm = torch.from_numpy(o.R_pre32).cuda()
    Rp = torch.from_numpy(o.R_post32).cuda()
    ck.commitkv_classify([dev.P_post], [Rm], [Rp], [dev.eligible], b.state, b.cand, b.n_cand, b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    assert np.array_equal(_np(b.state[0]), o.state)
    nc = int(b.n_cand[0])
    assert nc == len(o.cand)
    assert np.array_equal(_np(b.cand[0])[:nc], o.cand)


@pytest.mark.parametrize("variant", [1, 2, 3])
@pytest.mark.parametrize("name,seed", [("tiny", 0), ("small", 1), ("small_w40_g16", 2), ("hand", 0)])
def test_classify_variants(name, seed, variant):
    """The ablations of Section 4.4 (w/o pre-commit state, w/o percentile
    calibration, both): states and candidate order bit for bit against the
    oracle on the same fp32 effects."""
    import json
    import os
    np_ = ck.COMMITKV_CLASSIFY_NO_PRECOMMIT & variant != 0
    npc = ck.COMMITKV_CLASSIFY_NO_PERCENTILE & variant != 0
    if name == "hand":
        with open(os.path.join(os.path.dirname(__file__), "golden", "classify_variants_hand.json")) as f:
            g = json.load(f)
        Rm32 = np.asarray(g["R_pre"], np.float32)
        Rp32 = np.asarray(g["R_post"], np.float32)
        el = torch.tensor(g["eligible"], dtype=torch.uint8, device="cuda")
        ws = get_run("small", 0).buf.ws  # sized for far more than 8 pages
    else:
        r = get_run(name, seed)
        Rm32, Rp32 = r.orc.R_pre32, r.orc.R_post32
        el = r.dev.eligible
        ws = r.buf.ws
    P = len(Rm32)
    st_o, cand_o = core.classify(Rm32, Rp32, _np(el), no_precommit=np_, no_percentile=npc)
    state = torch.zeros(max(P, 1), dtype=torch.uint8, device="cuda")
    cand = torch.full((max(P, 1),), -1, dtype=torch.int32, device="cuda")
    n_cand = torch.zeros(1, dtype=torch.int32, device="cuda")
    ck.commitkv_classify_variant([P], [torch.from_numpy(Rm32).cuda()], [torch.from_numpy(Rp32).cuda()], [el],
                                 variant, [state], [cand], n_cand, ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    assert np.array_equal(_np(state)[:P], st_o)
    nc = int(n_cand[0])
    assert nc == len(cand_o)
    assert np.array_equal(_np(cand)[:nc], cand_o)


@pytest.mark.parametrize("name,seed", CASES)
def test_joint_isolated(name, seed):
    """The oracle's candidate list into the GPU joint test (with the GPU's
    own post-commit stats); compare each step's joint effect and the
    accepted set up to the first decision inside the tolerance."""
    r = get_run(name, seed)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    b.score_post()
    cand = torch.zeros(max(dev.P_post, 1), dtype=torch.int32, device="cuda")
    cand[:len(o.cand)] = torch.from_numpy(o.cand.astype(np.int32)).cuda()
    n_cand = torch.tensor([len(o.cand)], dtype=torch.int32, device="cuda")
    ck.commitkv_joint_test(b.shape, [dev.post()], b.stats, [cand], n_cand, cfg.tau_joint, b.accepted,
                           b.step_R, workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    nc = len(o.cand)
    step = _np(b.step_R[0])[:nc]
    acc = _np(b.accepted[0])[:dev.P_post]
    # compare up to (and including) the first unsafe decision
    safe = safe_threshold_mask(o.step_R, cfg.tau_joint, r.tol)
    upto = nc if safe.all() else int(np.argmin(safe))
    _assert_close(step[:upto], o.step_R[:upto], r.tol, "joint step R")
    for j in range(upto):
        E = o.cand[j]
        assert acc[E] == o.accepted[E], (j, E, step[j], o.step_R[j])
    # decisions agree with the reported effects everywhere
    for j in range(nc):
        assert acc[o.cand[j]] == (step[j] <= cfg.tau_joint)
    # only candidates can be accepted
    others = np.setdiff1d(np.arange(dev.P_post), o.cand)
    assert not acc[others].any()


@pytest.mark.parametrize("name,seed,q", [("small", 0, 0.5), ("small", 1, 0.3), ("small_w40_g16", 2, 0.6),
                                         ("small_long_pages", 4, 0.5)])
def test_joint_rounds_with_rejections(name, seed, q):
    """Up to 23 candidates (several rounds of the joint kernel and a ragged
    last one) with tau at a quantile of their single-page effects, so that
    the scan accepts and rejects, also in the middle of a round; every step
    against the oracle's greedy scan, up to the first decision inside the
    tolerance."""
    r = get_run(name, seed)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    Rp = o.R_post
    pages = [E for E in np.argsort(Rp, kind="stable") if np.isfinite(Rp[E]) and Rp[E] > 0][:23]
    rng = np.random.default_rng(seed)
    cand_np = np.array(pages, np.int64)[rng.permutation(len(pages))]
    tau = float(np.float32(np.quantile(Rp[cand_np], q)))
    acc_o, step_o = core.greedy(o.post, cand_np, tau, "closed", stats=o.stats)
    nc = len(cand_np)
    assert 2 <= int(acc_o[cand_np].sum()) <= nc - 2, "the scan should both accept and reject"
    b.score_post()
    cand = torch.zeros(max(dev.P_post, 1), dtype=torch.int32, device="cuda")
    cand[:nc] = torch.from_numpy(cand_np.astype(np.int32)).cuda()
    n_cand = torch.tensor([nc], dtype=torch.int32, device="cuda")
    ck.commitkv_joint_test(b.shape, [dev.post()], b.stats, [cand], n_cand, tau, b.accepted, b.step_R,
                           workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    step = _np(b.step_R[0])[:nc]
    acc = _np(b.accepted[0])[:dev.P_post]
    safe = safe_threshold_mask(step_o, tau, r.tol)
    upto = nc if safe.all() else int(np.argmin(safe))
    _assert_close(step[:upto], step_o[:upto], r.tol, "joint step R")
    for j in range(upto):
        assert acc[cand_np[j]] == acc_o[cand_np[j]], (j, step[j], step_o[j])
    for j in range(nc):
        assert acc[cand_np[j]] == (step[j] <= tau)
    others = np.setdiff1d(np.arange(dev.P_post), cand_np)
    assert not acc[others].any()


def test_joint_without_validation_accepts_every_candidate():
    """'w/o joint validation' (Section 4.4) is the joint test with tau_joint =
    +inf: every candidate is retired; the step values are those of the scan
    that accepts them all, against the oracle."""
    r = get_run("small", 0)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    Rp = o.R_post
    cand_np = np.array([E for E in np.argsort(Rp, kind="stable") if np.isfinite(Rp[E]) and Rp[E] > 0][:10], np.int64)
    nc = len(cand_np)
    acc_o, step_o = core.greedy(o.post, cand_np, float("inf"), "closed", stats=o.stats)
    assert acc_o[cand_np].all()
    b.score_post()
    cand = torch.zeros(max(dev.P_post, 1), dtype=torch.int32, device="cuda")
    cand[:nc] = torch.from_numpy(cand_np.astype(np.int32)).cuda()
    n_cand = torch.tensor([nc], dtype=torch.int32, device="cuda")
    ck.commitkv_joint_test(b.shape, [dev.post()], b.stats, [cand], n_cand, float("inf"), b.accepted, b.step_R,
                           workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    acc = _np(b.accepted[0])[:dev.P_post]
    assert acc[cand_np].all() and acc.sum() == nc
    fin = np.isfinite(step_o)
    _assert_close(_np(b.step_R[0])[:nc][fin], step_o[fin], r.tol, "step R with every candidate accepted")


@pytest.mark.parametrize("name,seed", CASES)
def test_compact_isolated(name, seed):
    """Same retired set, pending pages, priorities and fill scores into the
    GPU checkpoint: I_j, K~, V~, p~ bit-exact."""
    r = get_run(name, seed)
    cfg, b, dev, o, tr = r.cfg, r.buf, r.dev, r.orc, r.tr
    retired = torch.from_numpy(o.accepted.astype(np.uint8)).cuda()
    prio = torch.from_numpy(o.R_post32).cuda()
    ck.commitkv_compact(b.shape, [dev.post()], [retired], [dev.pending], [prio], [dev.fill], cfg.B,
                        cfg.B_N, cfg.pending_cap, b.idx, b.n_idx, b.k_out, b.v_out, b.pos_out,
                        workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    n = int(b.n_idx[0])
    assert n == len(o.I)
    I = _np(b.idx[0])[:n]
    assert np.array_equal(I, o.I)
    Kw, Vw, pw = core.gather(tr.K, tr.V, tr.pos, o.I)
    kg = b.k_out[0][:, :, :n]
    vg = b.v_out[0][:, :, :n]
    if cfg.dtype == "bf16":
        kg, vg = kg.view(torch.uint16), vg.view(torch.uint16)
    assert np.array_equal(_np(kg), Kw) and np.array_equal(_np(vg), Vw)
    assert np.array_equal(_np(b.pos_out[0])[:n], pw)


@pytest.mark.parametrize("layout", ["capacity", "odd_offset"])
@pytest.mark.parametrize("name,seed", CASES)
def test_compact_in_place(name, seed, layout):
    """commitkv_compact_in_place on a copy of the cache kept inside a larger
    buffer: I_j as the oracle's, and rows / positions [0, |I_j|) of the cache
    itself bit-exact against the oracle's gathered K~, V~, p~; memory
    outside the cache's view untouched.  'capacity': the cache is the first
    S tokens of a buffer with room for more (16-byte vector path);
    'odd_offset': every row starts one element into a row of d + 1 (the
    unaligned path)."""
    r = get_run(name, seed)
    cfg, b, dev, o, tr = r.cfg, r.buf, r.dev, r.orc, r.tr
    retired = torch.from_numpy(o.accepted.astype(np.uint8)).cuda()
    prio = torch.from_numpy(o.R_post32).cuda()
    M, H, S, d = dev.K.shape
    if layout == "capacity":
        Kb = torch.zeros(M, H, S + 37, d, dtype=dev.K.dtype, device="cuda")
        Vb = torch.zeros_like(Kb)
        K, V = Kb[:, :, :S], Vb[:, :, :S]
    else:
        Kb = torch.zeros(M, H, S, d + 1, dtype=dev.K.dtype, device="cuda")
        Vb = torch.zeros_like(Kb)
        K, V = Kb[..., 1:], Vb[..., 1:]
    K.copy_(dev.K)
    V.copy_(dev.V)
    pos = dev.pos.clone()
    cache = ck.TrajTensors(K, V, pos, dev.Q_post, dev.qpos_post, dev.page_start, dev.page_len)
    idx = torch.full_like(b.idx[0], -1)
    n_idx = torch.zeros_like(b.n_idx)
    ck.commitkv_compact_in_place(b.shape, [cache], [retired], [dev.pending], [prio], [dev.fill], cfg.B, cfg.B_N,
                                 cfg.pending_cap, [idx], n_idx, workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    n = int(n_idx[0])
    assert n == len(o.I)
    assert np.array_equal(_np(idx)[:n], o.I)
    Kw, Vw, pw = core.gather(tr.K, tr.V, tr.pos, o.I)
    kg, vg = K[:, :, :n], V[:, :, :n]
    if cfg.dtype == "bf16":
        kg, vg = kg.view(torch.uint16), vg.view(torch.uint16)
    assert np.array_equal(_np(kg), Kw) and np.array_equal(_np(vg), Vw)
    assert np.array_equal(_np(pos)[:n], pw)
    if layout == "capacity":
        assert not Kb[:, :, S:].any() and not Vb[:, :, S:].any()
    else:
        assert not Kb[..., 0].any() and not Vb[..., 0].any()


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("small", 1), ("small_f32", 3)])
def test_full_step(name, seed):
    """The whole launch sequence of one step: every decision of the GPU
    pipeline whose margin is safe matches the oracle pipeline."""
    r = get_run(name, seed)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    b.step()
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    _assert_close(_np(b.R_pre[0]), o.R_pre, r.tol, "R-")
    _assert_close(_np(b.R_post[0]), o.R_post, r.tol, "R+")
    st = _np(b.state[0])
    # classification agrees on pages whose thresholds are not within tolerance
    from oracle_bridge import percentile_safe
    idx = np.flatnonzero(dev.tr.eligible)
    safe = percentile_safe(o.R_pre, idx, r.tol) & percentile_safe(o.R_post, idx, r.tol)
    for th in (0.05, 0.01):
        safe &= safe_threshold_mask(o.R_pre[idx], th, r.tol) & safe_threshold_mask(o.R_post[idx], th, r.tol)
    assert np.array_equal(st[idx][safe], o.state[idx][safe])
    assert safe.any()
    nc = int(b.n_cand[0])
    gpu_cand = _np(b.cand[0])[:nc]
    # the GPU's candidates are the oracle classifier's on the GPU's own effects
    g_state, g_cand = core.classify(_np(b.R_pre[0]).astype(np.float64), _np(b.R_post[0]).astype(np.float64),
                                    dev.tr.eligible)
    assert np.array_equal(st, g_state)
    assert np.array_equal(gpu_cand, g_cand)
    # joint test on that candidate list against the oracle's scan of the same
    # list, up to the first step whose margin is within the tolerance
    acc_o, step_o = core.greedy(o.post, gpu_cand, cfg.tau_joint, "closed", stats=o.stats)
    stepR = _np(b.step_R[0])[:nc]
    safe_s = safe_threshold_mask(step_o, cfg.tau_joint, r.tol)
    upto = nc if safe_s.all() else int(np.argmin(safe_s))
    _assert_close(stepR[:upto], step_o[:upto], r.tol, "step R")
    acc = _np(b.accepted[0])[:dev.P_post]
    for j in range(upto):
        assert acc[gpu_cand[j]] == acc_o[gpu_cand[j]], j
    for j in range(nc):
        assert acc[gpu_cand[j]] == (stepR[j] <= cfg.tau_joint), j  # each decision follows its step value
    assert not acc[np.setdiff1d(np.arange(dev.P_post), gpu_cand)].any()
    # selection on the GPU's own decisions and priorities: bit-exact
    n = int(b.n_idx[0])
    R_post32 = _np(b.R_post[0])
    I_g = core.select_indices(dev.tr.S_post, dev.tr.page_start, dev.tr.page_len, acc, dev.tr.pending,
                              R_post32[dev.tr.pending].astype(np.float64), dev.tr.fill_score, cfg.B, cfg.B_N,
                              cfg.pending_cap)
    assert np.array_equal(_np(b.idx[0])[:n], I_g)
    # and the oracle's own chain, where the GPU took the oracle's decisions
    # and the pending priorities order alike
    if np.array_equal(gpu_cand, o.cand) and np.array_equal(acc, o.accepted):
        pr = o.R_post[dev.tr.pending]
        srt = np.sort(pr)
        if len(srt) < 2 or np.all(np.diff(srt) > 2 * r.tol * srt[1:]):
            assert np.array_equal(_np(b.idx[0])[:n], o.I)


def test_gapped_positions():
    """Non-contiguous absolute positions (a cache compacted earlier)."""
    r = get_run("small", 5, gapped=True)
    b, dev, o = r.buf, r.dev, r.orc
    b.score_pre()
    b.score_post()
    torch.cuda.synchronize()
    _assert_close(_np(b.R_pre[0])[:dev.P_pre], o.R_pre[:dev.P_pre], r.tol, "R-")
    _assert_close(_np(b.R_post[0]), o.R_post, r.tol, "R+")


def test_layer_mask():
    r = get_run("small", 0)
    cfg, b, dev = r.cfg, r.buf, r.dev
    mask = [0, 1]
    pre, post = None, None
    from oracle_bridge import problems
    pre, post = problems(r.tr, layer_mask=np.array(mask, np.uint8))
    Rw, Hw = core.page_effects(post, "explicit")
    R = torch.zeros(dev.P_post, device="cuda")
    H = torch.full((cfg.M, cfg.Hq, dev.P_post), 7.0, device="cuda")
    ck.commitkv_page_effects(b.shape, [dev.post()], [R], head_R_out=[H], layer_mask=mask, workspace=b.ws)
    torch.cuda.synchronize()
    _assert_close(_np(R), Rw, r.tol, "masked R")
    _assert_close(_np(H), Hw, r.tol, "masked per-head R (unselected layers = 0)")


def test_batched_trajectories_match_single():
    """Three trajectories of different lengths in one launch sequence give
    the same effects as the oracle for each."""
    cfgs = [synth.small_config("b0", L_pre=300, L_obs=40), synth.small_config("b1", L_pre=700, L_obs=90),
            synth.small_config("b2", L_pre=450, L_obs=64)]
    trs = [synth.make_trajectory(c, 10 + i, traj=i) for i, c in enumerate(cfgs)]
    devs = [DeviceTrajectory.upload(t) for t in trs]
    buf = StepBuffers(cfgs[1], devs)
    buf.score_pre()
    buf.score_post()
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK
    for t, d, Rm, Rp in zip(trs, devs, buf.R_pre, buf.R_post):
        o = OracleStep(t, "explicit")
        _assert_close(_np(Rm)[:d.P_pre], o.R_pre[:d.P_pre], 2e-2, "batched R-")
        _assert_close(_np(Rp), o.R_post, 2e-2, "batched R+")


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("small", 0), ("small_w40_g16", 2), ("small_long_pages", 4),
                                       ("small_f32", 3)])
def test_from_stats_matches_full_call(name, seed):
    """The page pass alone, fed the stats the full call wrote, gives the
    same effects bit for bit (both paths: the CUDA-core one for fp32 and
    head width 64, the tensor-core one for bf16)."""
    r = get_run(name, seed)
    cfg, b, dev = r.cfg, r.buf, r.dev
    R = torch.zeros(dev.P_post, device="cuda")
    H = torch.zeros(cfg.M, cfg.Hq, dev.P_post, device="cuda")
    st = torch.zeros_like(b.stats[0])
    ck.commitkv_page_effects(b.shape, [dev.post()], [R], head_R_out=[H], stats_out=[st], workspace=b.ws)
    R2 = torch.full_like(R, 7.0)
    H2 = torch.full_like(H, 7.0)
    ck.commitkv_page_effects_from_stats(b.shape, [dev.post()], [st], [R2], head_R_out=[H2], workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    assert torch.equal(R.view(torch.int32), R2.view(torch.int32))
    assert torch.equal(H.view(torch.int32), H2.view(torch.int32))


def _oracle_stats(cfg, o, lse_form):
    m, l, o_vec, n = o.stats
    st = np.zeros((cfg.M * cfg.Hq * o.tr.cfg.W, cfg.d + 4))
    if lse_form:  # an engine's log-sum-exp: m = L, l = 1
        st[:, 0] = np.where(np.isfinite(m), m + np.log(np.where(l > 0, l, 1.0)), m)
        st[:, 1] = np.where(np.isfinite(m), 1.0, 0.0)
    else:
        st[:, 0], st[:, 1] = m, l
    st[:, 4:] = o_vec
    return torch.from_numpy(st.astype(np.float32).reshape(cfg.M, cfg.Hq, o.tr.cfg.W, cfg.d + 4)).cuda()


@pytest.mark.parametrize("name,seed", [("tiny", 1), ("small", 1), ("small_long_pages", 4)])
@pytest.mark.parametrize("lse_form", [False, True])
def test_from_stats_with_oracle_stats(name, seed, lse_form):
    """The oracle's fp64 row stats (rounded to fp32), as (max, sum) or as a
    log-sum-exp with sum 1, into the page pass: effects against the oracle."""
    r = get_run(name, seed)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    st = _oracle_stats(cfg, o, lse_form)
    R = torch.zeros(dev.P_post, device="cuda")
    H = torch.zeros(cfg.M, cfg.Hq, dev.P_post, device="cuda")
    ck.commitkv_page_effects_from_stats(b.shape, [dev.post()], [st], [R], head_R_out=[H], workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    _assert_close(_np(R), o.R_post, r.tol, "R+ from oracle stats")
    _assert_close(_np(H), o.H_post, r.tol, "R+ per head from oracle stats")


def test_pre_and_post_in_one_call():
    """The pre- and post-commit caches of three trajectories scored in one
    call (six caches in one launch sequence): effects match the oracle and
    the separate calls, the post-commit stats match the separate call."""
    cfgs = [synth.small_config("b0", L_pre=300, L_obs=40), synth.small_config("b1", L_pre=700, L_obs=90),
            synth.small_config("b2", L_pre=450, L_obs=64)]
    trs = [synth.make_trajectory(c, 20 + i, traj=i) for i, c in enumerate(cfgs)]
    devs = [DeviceTrajectory.upload(t) for t in trs]
    buf = StepBuffers(cfgs[1], devs)
    buf.score()
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK
    one = ([_np(r).copy() for r in buf.R_pre], [_np(r).copy() for r in buf.R_post],
           [_np(s).copy() for s in buf.stats])
    buf.score_pre()
    buf.score_post()
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK
    for i, (t, d) in enumerate(zip(trs, devs)):
        o = OracleStep(t, "explicit")
        _assert_close(one[0][i][:d.P_pre], o.R_pre[:d.P_pre], 2e-2, "one-call R-")
        _assert_close(one[1][i], o.R_post, 2e-2, "one-call R+")
        _assert_close(one[0][i][:d.P_pre], _np(buf.R_pre[i])[:d.P_pre], 1e-3, "one-call R- vs separate")
        _assert_close(one[1][i], _np(buf.R_post[i]), 1e-3, "one-call R+ vs separate")
        a, b = one[2][i].reshape(-1, t.cfg.d + 4), _np(buf.stats[i]).reshape(-1, t.cfg.d + 4)
        assert np.array_equal(a[:, 2], b[:, 2])
        _assert_close(a[:, 1], b[:, 1], 1e-5, "one-call row sum vs separate")


def test_edge_cases():
    """Empty page list, zero-length pages, a probe row that sees nothing, a
    cache shorter than one tile."""
    cfg = synth.small_config("edge", L_pre=40, L_obs=8, W=4, G=8, B=16, planted_frac=0.0,
                             event_len=(4, 12))
    tr = synth.make_trajectory(cfg, 0)
    # a zero-length page and a probe row before every resident token
    tr.page_len = tr.page_len.copy()
    tr.page_len[0] = 0
    dev = DeviceTrajectory.upload(tr)
    qpos = dev.qpos_post.clone()
    qpos[0] = -1
    dev.qpos_post = qpos
    buf = StepBuffers(cfg, [dev])
    buf.score_post()
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK
    post = core.Problem(synth.values_f64(tr.K, "bf16"), synth.values_f64(tr.V, "bf16"), tr.pos,
                        synth.values_f64(tr.Q_post, "bf16"), _np(qpos), tr.page_start, tr.page_len)
    Rw, _ = core.page_effects(post, "explicit")
    _assert_close(_np(buf.R_post[0]), Rw, 2e-2, "edge R+")
    assert float(buf.R_post[0][0]) == 0.0
    # no pages at all
    empty = ck.TrajTensors(dev.K, dev.V, dev.pos, dev.Q_post, dev.qpos_post,
                           dev.page_start[:0], dev.page_len[:0])
    R0 = torch.zeros(0, device="cuda")
    ck.commitkv_page_effects(buf.shape, [empty], [R0], workspace=buf.ws)
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK


def test_device_input_errors_are_reported():
    """Inputs only the device can check: overlapping pages, a candidate id
    out of range, a NaN fill score.  Each is reported in the workspace status
    and the context stays usable."""
    r = get_run("small", 0)
    cfg, b, dev = r.cfg, r.buf, r.dev
    bad_len = dev.page_len.clone()
    bad_len[1] = bad_len[1] + 40  # overlaps page 2
    t = ck.TrajTensors(dev.K, dev.V, dev.pos, dev.Q_post, dev.qpos_post, dev.page_start, bad_len)
    ck.commitkv_page_effects(b.shape, [t], b.R_post, workspace=b.ws)
    assert b.status() == ck.COMMITKV_ERR_DEVICE_INPUT
    b.score_post()
    cand = torch.tensor([dev.P_post + 5], dtype=torch.int32, device="cuda")
    n_cand = torch.tensor([1], dtype=torch.int32, device="cuda")
    ck.commitkv_joint_test(b.shape, [dev.post()], b.stats, [cand], n_cand, cfg.tau_joint, b.accepted,
                           workspace=b.ws)
    assert b.status() == ck.COMMITKV_ERR_DEVICE_INPUT
    fill = dev.fill.clone()
    fill[3] = float("nan")
    ck.commitkv_compact(b.shape, [dev.post()], b.accepted, [dev.pending], b.R_post, [fill], cfg.B, cfg.B_N,
                        cfg.pending_cap, b.idx, b.n_idx, workspace=b.ws)
    assert b.status() == ck.COMMITKV_ERR_DEVICE_INPUT
    # the context is still usable
    b.score_post()
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK


def test_compact_pending_span_out_of_range():
    """A pending page whose span starts just past the cache (S + 1, inside
    the 256-byte padding of the trajectory's token-class bytes in the
    workspace) is reported as a device input error with |I| = 0, and the
    selection writes no class byte outside [0, S): the padding byte keeps
    the value it had before the call."""
    r = get_run("small", 0)
    cfg, b, dev = r.cfg, r.buf, r.dev
    S = dev.tr.S_post
    assert S % 256 != 0 and S + 1 < (S + 255) // 256 * 256  # the span's start lies in the padding
    p = int(dev.tr.pending[0])
    ps, pl = dev.page_start.clone(), dev.page_len.clone()
    ps[p], pl[p] = S + 1, 1
    t = ck.TrajTensors(dev.K, dev.V, dev.pos, dev.Q_post, dev.qpos_post, ps, pl)
    retired = torch.zeros(dev.P_post, dtype=torch.uint8, device="cuda")
    # token classes of the first trajectory start 256 bytes into the workspace
    sentinel = 0x77
    b.ws[256 + S + 1] = sentinel
    b.n_idx.fill_(-1)
    ck.commitkv_compact(b.shape, [t], [retired], [dev.pending], b.R_post, [dev.fill], cfg.B, cfg.B_N,
                        cfg.pending_cap, b.idx, b.n_idx, workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_ERR_DEVICE_INPUT
    assert int(b.n_idx[0]) == 0
    assert int(b.ws[256 + S + 1]) == sentinel
    # the context is still usable
    b.score_post()
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK


def test_bounded_wait_times_out():
    """A grid barrier that can never fill ends by its time limit with
    COMMITKV_ERR_TIMEOUT, and the context stays usable."""
    r = get_run("small", 0)
    b = r.buf
    ck.commitkv_test_barrier_timeout(b.ws, 2)
    assert b.status() == ck.COMMITKV_ERR_TIMEOUT
    b.score_post()
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK


@pytest.mark.parametrize("name,seed", [("small", 0), ("small_w40_g16", 2), ("small_long_pages", 4)])
def test_scoring_paths_agree(name, seed, monkeypatch):
    """The tensor-core scoring path (bf16, head_dim 128) and the CUDA-core
    path give the same effects and stats within the bf16 tolerance."""
    r = get_run(name, seed)
    b, dev = r.buf, r.dev
    out = {}
    for path in ("tc", "simt"):
        monkeypatch.setenv("COMMITKV_SCORING", path)
        R = torch.zeros(dev.P_post, device="cuda")
        st = torch.zeros_like(b.stats[0])
        ck.commitkv_page_effects(b.shape, [dev.post()], [R], stats_out=[st], workspace=b.ws)
        torch.cuda.synchronize()
        assert b.status() == ck.COMMITKV_OK
        out[path] = (_np(R), _np(st))
    _assert_close(out["tc"][0], out["simt"][0], 2e-2, "R+ tc vs simt")
    a, s_ = out["tc"][1].reshape(-1, r.cfg.d + 4), out["simt"][1].reshape(-1, r.cfg.d + 4)
    assert np.array_equal(a[:, 2], s_[:, 2])
    _assert_close(a[:, 0], s_[:, 0], 1e-5, "row max")


@pytest.mark.parametrize("name,seed", [("small", 0), ("small_w40_g16", 2), ("small_long_pages", 4)])
def test_fused_and_two_launch_scoring_agree(name, seed, monkeypatch):
    """The tensor-core scoring as one cooperative launch of both passes (the
    default) and as separate flash, merge and page launches: effects within
    the bf16 tolerance, visible counts and row maxima alike, and both
    against the oracle."""
    r = get_run(name, seed)
    b, dev, o = r.buf, r.dev, r.orc
    out = {}
    for fused in ("1", "0"):
        monkeypatch.setenv("COMMITKV_FUSED", fused)
        R = torch.zeros(dev.P_post, device="cuda")
        st = torch.zeros_like(b.stats[0])
        ck.commitkv_page_effects(b.shape, [dev.post()], [R], stats_out=[st], workspace=b.ws)
        torch.cuda.synchronize()
        assert b.status() == ck.COMMITKV_OK
        out[fused] = (_np(R), _np(st).reshape(-1, r.cfg.d + 4))
        _assert_close(out[fused][0], o.R_post, r.tol, f"R+ (fused={fused}) against the oracle")
    _assert_close(out["1"][0], out["0"][0], 2e-2, "R+ fused vs two launches")
    a, c = out["1"][1], out["0"][1]
    assert np.array_equal(a[:, 2], c[:, 2])
    _assert_close(a[:, 0], c[:, 0], 1e-6, "row max")
    _assert_close(a[:, 1], c[:, 1], 1e-5, "row sum")


def test_many_zero_length_pages():
    """Zero-length pages take no slot: an item may hold more pages than its
    slots.  Their effect is 0; the other pages are unaffected."""
    cfg = synth.small_config("zeros", L_pre=500, L_obs=40)
    tr = synth.make_trajectory(cfg, 7)
    ps, pl = [], []
    for s_, l_ in zip(tr.page_start.tolist(), tr.page_len.tolist()):
        for _ in range(12):  # zero-length pages at the page's start
            ps.append(s_)
            pl.append(0)
        ps.append(s_)
        pl.append(l_)
    tr.page_start = np.asarray(ps, np.int32)
    tr.page_len = np.asarray(pl, np.int32)
    tr.eligible = np.ones(len(ps), np.uint8)
    dev = DeviceTrajectory.upload(tr)
    buf = StepBuffers(cfg, [dev])
    buf.score_post()
    torch.cuda.synchronize()
    assert buf.status() == ck.COMMITKV_OK
    post = core.Problem(synth.values_f64(tr.K, "bf16"), synth.values_f64(tr.V, "bf16"), tr.pos,
                        synth.values_f64(tr.Q_post, "bf16"), tr.qpos_post, tr.page_start, tr.page_len)
    Rw, _ = core.page_effects(post, "explicit")
    _assert_close(_np(buf.R_post[0]), Rw, 2e-2, "R+ with zero-length pages")
    assert (_np(buf.R_post[0])[np.asarray(pl) == 0] == 0).all()


def test_qwen_shape_plain_normal_inputs():
    """The Qwen3-8B shape (32 query / 8 KV heads, head_dim 128, bf16) with
    Q, K, V ~ N(0, 1) as drawn (four key channels per (layer, KV head)
    scaled by 8, no shared window direction, nothing planted), two layers of
    a 4K + 512 cache: R-, R+ of every page and head, and the post-commit row
    statistics, against the oracle's closed form (Eq. 6) over every slice."""
    cfg = synth.small_config("qwen_n01", M=2, H=8, Hq=32, d=128, W=32, G=32, L_pre=4096, L_obs=512, B=1024,
                             pending_cap=16, planted_frac=0.0, outlier_channels=4, plant="shared", gamma=0.0,
                             alpha=0.0, beta=(0.0, 0.0), nu=0.0)
    tr = synth.make_trajectory(cfg, 9)
    assert len(tr.planted) == 0
    dev = DeviceTrajectory.upload(tr)
    b = StepBuffers(cfg, [dev])
    headR_pre = torch.zeros(cfg.M, cfg.Hq, dev.P_pre, device="cuda")
    headR_post = torch.zeros(cfg.M, cfg.Hq, dev.P_post, device="cuda")
    R_pre = torch.zeros(dev.P_pre, device="cuda")
    ck.commitkv_page_effects(b.shape, [dev.pre()], [R_pre], head_R_out=[headR_pre], workspace=b.ws)
    ck.commitkv_page_effects(b.shape, [dev.post()], b.R_post, head_R_out=[headR_post], stats_out=b.stats,
                             workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    from oracle_bridge import problems
    pre, post = problems(tr)
    Rm, Hm = core.page_effects(pre, "closed")
    Rp, Hp = core.page_effects(post, "closed")
    _assert_close(_np(R_pre), Rm, 2e-2, "R- (N(0,1) inputs)")
    _assert_close(_np(b.R_post[0]), Rp, 2e-2, "R+ (N(0,1) inputs)")
    _assert_close(_np(headR_pre), Hm, 2e-2, "R- per head (N(0,1) inputs)")
    _assert_close(_np(headR_post), Hp, 2e-2, "R+ per head (N(0,1) inputs)")
    m, l, o_vec, n = core.row_stats(post)
    st = _np(b.stats[0]).reshape(-1, cfg.d + 4)
    assert np.array_equal(st[:, 2].astype(np.int64), n)
    _assert_close(st[:, 0], m, 1e-5, "row max")
    _assert_close(st[:, 1], l, 1e-4, "row sum")
    err = np.linalg.norm(st[:, 4:] - o_vec, axis=1) / np.maximum(np.linalg.norm(o_vec, axis=1), 1e-30)
    assert err.max() <= 1e-4, err.max()


def _token_scores_close(got, want, tol, what):
    """Token scores against the oracle: relative tol, exact zeros (tokens no
    probe query sees); scores below 1e-30 (fp32 exponent range) count as 0."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert np.array_equal(got == 0, want < 1e-30), what + ": zeros differ"
    ok = (np.abs(got - want) <= tol * np.abs(want)) | (want < 1e-30)
    assert ok.all(), f"{what}: {int((~ok).sum())} of {ok.size} outside {tol}"


@pytest.mark.parametrize("name,seed", [("tiny", 0), ("small", 0), ("small_w40_g16", 2), ("small_long_pages", 4),
                                       ("small_f32", 3)])
@pytest.mark.parametrize("window", ["pre", "post"])
def test_token_scores(name, seed, window):
    """Per-token fill scores (window attention, Eq. 13's fill) from the
    GPU's own row stats of the same cache and window, against the oracle's
    softmax written out row by row: every token, within the effect
    tolerance; tokens no probe query sees score exactly 0."""
    r = get_run(name, seed)
    cfg, b, dev, o = r.cfg, r.buf, r.dev, r.orc
    t = dev.pre() if window == "pre" else dev.post()
    S = dev.tr.L_pre if window == "pre" else dev.tr.S_post
    stats = torch.zeros_like(b.stats[0])
    R = torch.zeros(max(dev.P_post, 1), device="cuda")
    P = dev.P_pre if window == "pre" else dev.P_post
    ck.commitkv_page_effects(b.shape, [t], [R[:P]], stats_out=[stats], workspace=b.ws)
    scores = torch.full((S,), -1.0, device="cuda")
    ck.commitkv_token_scores(b.shape, [t], [stats], [scores], workspace=b.ws)
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    want = core.token_scores(o.pre if window == "pre" else o.post)
    _token_scores_close(_np(scores), want, r.tol, f"token scores ({window})")


def test_token_scores_layer_mask_and_paths(monkeypatch):
    """One selected layer, and the CUDA-core kernel forced for bf16: both
    against the oracle and against each other."""
    r = get_run("small_w40_g16", 2)
    cfg, b, dev = r.cfg, r.buf, r.dev
    mask = np.zeros(cfg.M, np.uint8)
    mask[1] = 1
    stats = torch.zeros_like(b.stats[0])
    ck.commitkv_page_effects(b.shape, [dev.post()], b.R_post, stats_out=[stats], layer_mask=mask, workspace=b.ws)
    out = {}
    for path in ("tc", "simt"):
        monkeypatch.setenv("COMMITKV_SCORING", path)
        sc = torch.zeros(dev.tr.S_post, device="cuda")
        ck.commitkv_token_scores(b.shape, [dev.post()], [stats], [sc], layer_mask=mask, workspace=b.ws)
        torch.cuda.synchronize()
        assert b.status() == ck.COMMITKV_OK
        out[path] = _np(sc)
    from oracle_bridge import problems
    _, post = problems(dev.tr, layer_mask=mask)
    want = core.token_scores(post)
    for path in out:
        _token_scores_close(out[path], want, 2e-2, f"token scores, layer 1 only ({path})")
    _token_scores_close(out["tc"], out["simt"].astype(np.float64), 2e-2, "tc vs simt")
