"""Parity at the full sizes of the four large workloads, in the launch
configuration the benchmark times: the Qwen3-8B shape (36 layers, 32 query /
8 KV heads, head_dim 128, bf16) at 16K + 2K and 32K + 4K tokens, a batch of
16 ragged Qwen3-8B-shaped trajectories in one launch sequence, and the
Qwen3-32B shape (64 layers, 64 query / 8 KV heads) at 128K + 8K tokens.

The whole cache goes through the library.  The oracle checks what it can
compute one (layer, KV head) slice at a time, and properties that hold at
any size, on sampled trajectories of a batch:
  * per-(layer, query head) effects R_h of sampled slices, pre- and
    post-commit, and the (m, l, n, o) of the sampled slices' probe rows;
  * R equals the maximum of R_h over layers and heads (both come from the
    same fp32 values, so exactly);
  * classification and candidate order on seeded effect arrays of the full
    page counts, bit-exact;
  * the joint test restricted to one or two layers (the layer mask),
    against the oracle's greedy scan of the same layers over the full cache;
  * the per-token fill scores of one or two layers, every token of the
    sampled trajectories;
  * selection (seeded retired set, pending pages, seeded priorities) and
    the gather, bit-exact; the gather is checked on the sampled slices.
Tolerances are the bf16 ones of the other parity tests (2e-2 relative for
effects; decisions compared wherever the oracle's margin exceeds it).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import core  # noqa: E402
from paper_2608_07855_gb300 import commitkv as ck  # noqa: E402
from paper_2608_07855_gb300 import synth  # noqa: E402
from paper_2608_07855_gb300.workload import DeviceTrajectory, shape_of  # noqa: E402

from oracle_bridge import rel_close, safe_threshold_mask  # noqa: E402

pytestmark = pytest.mark.gpu

TOL = 2e-2
SLICES = [(0, 0), (17, 5), (35, 7)]  # (layer, KV head)
# the 64-layer Qwen3-32B shape: one slice in every 8 layers, each KV head once
SLICES_BY_CONFIG = {"qwen3_32b_128k": [(8 * i, i) for i in range(8)]}


def slices_of(cfg):
    return SLICES_BY_CONFIG.get(cfg.name, SLICES)
JOINT_LAYERS = {"qwen3_32b_128k": (3,)}  # the oracle's scan cost grows with rows x tokens
FULL_CONFIGS = ["qwen3_8b_16k", "qwen3_8b_32k", "ragged16", "qwen3_32b_128k"]


def _np(t):
    return t.detach().cpu().numpy()


def _check_close(got, want, tol, what):
    ok = rel_close(got, want, tol)
    if not ok.all():
        bad = np.flatnonzero(~ok.ravel())[:6]
        g, w = np.ravel(got), np.ravel(want)
        raise AssertionError(f"{what}: {int((~ok).sum())} of {ok.size} outside {tol}: "
                             + ", ".join(f"[{i}] gpu {g[i]:.6g} oracle {w[i]:.6g}" for i in bad))


def _slice_problem(tr, l, kvh, post, layers=None):
    """Oracle problem of one (layer, KV head) slice (or of whole layers)."""
    cfg = tr.cfg
    g = cfg.g
    S = tr.S_post if post else tr.L_pre
    P = tr.P_post if post else tr.P_pre
    Qall = tr.Q_post if post else tr.Q_pre
    if layers is None:
        K = tr.K[l:l + 1, kvh:kvh + 1, :S]
        V = tr.V[l:l + 1, kvh:kvh + 1, :S]
        Q = Qall[l:l + 1, kvh * g:(kvh + 1) * g]
    else:
        K, V, Q = tr.K[list(layers), :, :S], tr.V[list(layers), :, :S], Qall[list(layers)]
    return core.Problem(synth.values_f64(K, cfg.dtype), synth.values_f64(V, cfg.dtype), tr.pos[:S],
                        synth.values_f64(Q, cfg.dtype), tr.qpos_post if post else tr.qpos_pre,
                        tr.page_start[:P], tr.page_len[:P])


@pytest.fixture(scope="module", params=FULL_CONFIGS)
def full(request):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    ck.load_library()
    cfg = synth.CONFIGS[request.param]
    trs = [synth.make_trajectory(cfg, 0, traj=t) for t in range(cfg.n_traj)]
    devs = [DeviceTrajectory.upload(tr) for tr in trs]
    shape = shape_of(cfg)
    ws = ck.alloc_workspace(shape, [d.post() for d in devs])
    f32 = dict(dtype=torch.float32, device="cuda")
    n = len(trs)
    out = {"cfg": cfg, "trs": trs, "devs": devs, "shape": shape, "ws": ws,
           "sample": sorted({0, n // 2, n - 1})}
    out["R_pre"] = [torch.zeros(tr.P_pre, **f32) for tr in trs]
    out["R_post"] = [torch.zeros(tr.P_post, **f32) for tr in trs]
    out["H_pre"] = [torch.zeros(cfg.M, cfg.Hq, tr.P_pre, **f32) for tr in trs]
    out["H_post"] = [torch.zeros(cfg.M, cfg.Hq, tr.P_post, **f32) for tr in trs]
    out["stats"] = [torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, **f32) for tr in trs]
    ck.commitkv_page_effects(shape, [d.pre() for d in devs], out["R_pre"], head_R_out=out["H_pre"],
                             workspace=ws)
    ck.commitkv_page_effects(shape, [d.post() for d in devs], out["R_post"], head_R_out=out["H_post"],
                             stats_out=out["stats"], workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    yield out
    del out, devs, ws
    torch.cuda.empty_cache()


def test_sampled_slice_effects(full):
    cfg = full["cfg"]
    g = cfg.g
    for l, kvh in slices_of(cfg):
        for t in full["sample"]:
            tr = full["trs"][t]
            for post, key in ((False, "H_pre"), (True, "H_post")):
                _, H = core.page_effects(_slice_problem(tr, l, kvh, post), "closed")
                got = _np(full[key][t][l, kvh * g:(kvh + 1) * g])
                _check_close(got, H[0], TOL, f"{key} trajectory {t} slice ({l}, {kvh})")


def test_sampled_slice_row_stats(full):
    cfg = full["cfg"]
    g = cfg.g
    for (l, kvh), t in ((s, t) for s in slices_of(cfg) for t in full["sample"]):
        m, lsum, o_vec, n = core.row_stats(_slice_problem(full["trs"][t], l, kvh, True))
        st = _np(full["stats"][t][l, kvh * g:(kvh + 1) * g]).reshape(-1, cfg.d + 4)
        assert np.array_equal(st[:, 2].astype(np.int64), n)
        _check_close(st[:, 0], m, 1e-5, "row max")
        _check_close(st[:, 1], lsum, 1e-4, "row sum")
        err = np.linalg.norm(st[:, 4:] - o_vec, axis=1) / np.maximum(np.linalg.norm(o_vec, axis=1), 1e-30)
        assert err.max() <= 1e-4, (t, err.max())


def test_effect_is_max_over_heads(full):
    for t in range(len(full["trs"])):
        for R, H in (("R_pre", "H_pre"), ("R_post", "H_post")):
            r = _np(full[R][t])
            h = _np(full[H][t]).reshape(-1, r.shape[0]).max(axis=0)
            assert np.array_equal(r, h), (t, R)


def test_classify_fullsize(full):
    """Seeded effects over the full page counts (log-uniform between 1e-4 and
    1, so every lifecycle state occurs) through the GPU classifier (the
    whole batch in one launch) and the oracle's, bit-exact."""
    trs, ws = full["trs"], full["ws"]
    rng = np.random.default_rng(11)
    Rm = [(10.0 ** rng.uniform(-4, 0, tr.P_post)).astype(np.float32) for tr in trs]
    Rp = [(10.0 ** rng.uniform(-4, 0, tr.P_post)).astype(np.float32) for tr in trs]
    state = [torch.zeros(tr.P_post, dtype=torch.uint8, device="cuda") for tr in trs]
    cand = [torch.zeros(tr.P_post, dtype=torch.int32, device="cuda") for tr in trs]
    n_cand = torch.zeros(len(trs), dtype=torch.int32, device="cuda")
    ck.commitkv_classify([tr.P_post for tr in trs], [torch.from_numpy(x).cuda() for x in Rm],
                         [torch.from_numpy(x).cuda() for x in Rp], [d.eligible for d in full["devs"]], state,
                         cand, n_cand, ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    for t, tr in enumerate(trs):
        o_state, o_cand = core.classify(Rm[t].astype(np.float64), Rp[t].astype(np.float64), tr.eligible)
        assert np.array_equal(_np(state[t]), o_state), t
        nc = int(n_cand[t])
        assert nc == len(o_cand) and nc > 0, t
        assert np.array_equal(_np(cand[t])[:nc], o_cand), t


def test_joint_selected_layers(full):
    """The joint test over the full caches of the batch with one or two layers
    selected: the GPU's own post-commit statistics of those layers, seeded
    candidate lists (the planted pages, then other eligible pages), and the
    oracle's greedy scan of the same layers for the sampled trajectories."""
    trs, cfg, devs, shape, ws = full["trs"], full["cfg"], full["devs"], full["shape"], full["ws"]
    layers = JOINT_LAYERS.get(cfg.name, (3, 30))
    mask = np.zeros(cfg.M, np.uint8)
    mask[list(layers)] = 1
    f32 = dict(dtype=torch.float32, device="cuda")
    stats = [torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, **f32) for tr in trs]
    R = [torch.zeros(tr.P_post, **f32) for tr in trs]
    ck.commitkv_page_effects(shape, [d.post() for d in devs], R, stats_out=stats, layer_mask=mask, workspace=ws)
    rng = np.random.default_rng(5)
    cands = []
    for tr in trs:
        others = np.setdiff1d(np.flatnonzero(tr.eligible), tr.planted)
        extra = rng.choice(others, min(16, len(others)), replace=False)
        cands.append(np.concatenate([tr.planted[:32], extra]).astype(np.int32))
    cand = [torch.zeros(tr.P_post, dtype=torch.int32, device="cuda") for tr in trs]
    for c, x in zip(cand, cands):
        c[:len(x)] = torch.from_numpy(x).cuda()
    n_cand = torch.tensor([len(x) for x in cands], dtype=torch.int32, device="cuda")
    acc = [torch.zeros(tr.P_post, dtype=torch.uint8, device="cuda") for tr in trs]
    step = [torch.zeros(tr.P_post, **f32) for tr in trs]
    ck.commitkv_joint_test(shape, [d.post() for d in devs], stats, cand, n_cand, cfg.tau_joint, acc, step,
                           layer_mask=mask, workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    for t in full["sample"]:
        tr, cand_np = trs[t], cands[t]
        o_acc, o_step = core.greedy(_slice_problem(tr, 0, 0, True, layers=layers), cand_np, cfg.tau_joint,
                                    "closed")
        nc = len(cand_np)
        got_step = _np(step[t])[:nc]
        got_acc = _np(acc[t])
        safe = safe_threshold_mask(o_step, cfg.tau_joint, TOL)
        upto = nc if safe.all() else int(np.argmin(safe))
        assert upto > 0, t
        _check_close(got_step[:upto], o_step[:upto], TOL, f"joint step R, trajectory {t}")
        for j in range(upto):
            assert got_acc[cand_np[j]] == o_acc[cand_np[j]], (t, j)
        for j in range(nc):
            assert got_acc[cand_np[j]] == (got_step[j] <= cfg.tau_joint), (t, j)


def test_compact_fullsize(full):
    """Seeded retired pages, the observation's pages pending with seeded
    priorities, the trajectories' fill scores, the whole batch in one launch:
    I_j bit-exact against the oracle's selection, and K, V, positions
    gathered bit-exactly on the sampled slices of the sampled trajectories."""
    trs, cfg, devs, shape, ws = full["trs"], full["cfg"], full["devs"], full["shape"], full["ws"]
    rng = np.random.default_rng(3)
    retired = [(rng.uniform(size=tr.P_post) < 0.3).astype(np.uint8) for tr in trs]
    prio = [rng.uniform(size=tr.P_post).astype(np.float32) for tr in trs]
    B, B_N, cap = cfg.B, cfg.B_N, cfg.pending_cap
    idx = [torch.zeros(B, dtype=torch.int32, device="cuda") for tr in trs]
    n_idx = torch.zeros(len(trs), dtype=torch.int32, device="cuda")
    k_out = [torch.empty(cfg.M, cfg.H, B, cfg.d, dtype=torch.bfloat16, device="cuda") for tr in trs]
    v_out = [torch.empty_like(k) for k in k_out]
    pos_out = [torch.empty(B, dtype=torch.int32, device="cuda") for tr in trs]
    ck.commitkv_compact(shape, [d.post() for d in devs], [torch.from_numpy(x).cuda() for x in retired],
                        [d.pending for d in devs], [torch.from_numpy(x).cuda() for x in prio],
                        [d.fill for d in devs], B, B_N, cap, idx, n_idx, k_out, v_out, pos_out, workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    for t, tr in enumerate(trs):
        I = core.select_indices(tr.S_post, tr.page_start, tr.page_len, retired[t], tr.pending,
                                prio[t][tr.pending].astype(np.float64), tr.fill_score, B, B_N, cap)
        n = int(n_idx[t])
        assert n == len(I), t
        assert np.array_equal(_np(idx[t])[:n], I), t
        assert np.array_equal(_np(pos_out[t])[:n], tr.pos[I]), t
        if t in full["sample"]:
            for l, kvh in slices_of(cfg):
                assert np.array_equal(_np(k_out[t][l, kvh, :n].view(torch.uint16)), tr.K[l, kvh, I]), t
                assert np.array_equal(_np(v_out[t][l, kvh, :n].view(torch.uint16)), tr.V[l, kvh, I]), t
    del k_out, v_out


def test_token_scores_selected_layers(full):
    """Per-token fill scores (commitkv_token_scores, the self-contained fill)
    over the full post-commit caches of the batch with one or two layers
    selected, from the GPU's own row statistics of those layers: every token
    of the sampled trajectories against the oracle's softmax written out row
    by row over the same layers (relative tolerance; tokens no probe query
    sees score exactly 0), and every score of the batch a softmax weight."""
    trs, cfg, devs, shape, ws = full["trs"], full["cfg"], full["devs"], full["shape"], full["ws"]
    layers = JOINT_LAYERS.get(cfg.name, (3, 30))
    mask = np.zeros(cfg.M, np.uint8)
    mask[list(layers)] = 1
    f32 = dict(dtype=torch.float32, device="cuda")
    stats = [torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, **f32) for tr in trs]
    R = [torch.zeros(tr.P_post, **f32) for tr in trs]
    ck.commitkv_page_effects(shape, [d.post() for d in devs], R, stats_out=stats, layer_mask=mask, workspace=ws)
    scores = [torch.full((tr.S_post,), -1.0, **f32) for tr in trs]
    ck.commitkv_token_scores(shape, [d.post() for d in devs], stats, scores, layer_mask=mask, workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    for t, sc in enumerate(scores):
        assert float(sc.min()) >= 0.0 and float(sc.max()) <= 1.0, t
    for t in full["sample"]:
        want = core.token_scores(_slice_problem(trs[t], 0, 0, True, layers=layers))
        got = _np(scores[t]).astype(np.float64)
        assert np.array_equal(got == 0, want < 1e-30), f"trajectory {t}: zeros differ"
        ok = (np.abs(got - want) <= TOL * np.abs(want)) | (want < 1e-30)
        assert ok.all(), f"trajectory {t}: {int((~ok).sum())} of {ok.size} token scores outside {TOL}"
