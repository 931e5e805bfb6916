"""Parity at the full sizes of the Qwen3-8B-shaped workloads (36 layers, 32
query / 8 KV heads, head_dim 128, bf16; 16K + 2K and 32K + 4K tokens), in
the launch configuration the benchmark times.

The whole cache goes through the library.  The oracle checks what it can
compute one (layer, KV head) slice at a time, and properties that hold at
any size:
  * per-(layer, query head) effects R_h of sampled slices, pre- and
    post-commit, and the (m, l, n, o) of the sampled slices' probe rows;
  * R equals the maximum of R_h over layers and heads (both come from the
    same fp32 values, so exactly);
  * classification and candidate order on seeded effect arrays of the full
    page count, bit-exact;
  * the joint test restricted to two layers (the layer mask), against the
    oracle's greedy scan of the same two layers over the full cache;
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
JOINT_LAYERS = (3, 30)


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


@pytest.fixture(scope="module", params=["qwen3_8b_16k", "qwen3_8b_32k"])
def full(request):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    ck.load_library()
    cfg = synth.CONFIGS[request.param]
    tr = synth.make_trajectory(cfg, 0)
    dev = DeviceTrajectory.upload(tr)
    shape = shape_of(cfg)
    ws = ck.alloc_workspace(shape, [dev.post()])
    f32 = dict(dtype=torch.float32, device="cuda")
    out = {"cfg": cfg, "tr": tr, "dev": dev, "shape": shape, "ws": ws}
    out["R_pre"] = torch.zeros(tr.P_pre, **f32)
    out["R_post"] = torch.zeros(tr.P_post, **f32)
    out["H_pre"] = torch.zeros(cfg.M, cfg.Hq, tr.P_pre, **f32)
    out["H_post"] = torch.zeros(cfg.M, cfg.Hq, tr.P_post, **f32)
    out["stats"] = torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, **f32)
    ck.commitkv_page_effects(shape, [dev.pre()], [out["R_pre"]], head_R_out=[out["H_pre"]], workspace=ws)
    ck.commitkv_page_effects(shape, [dev.post()], [out["R_post"]], head_R_out=[out["H_post"]],
                             stats_out=[out["stats"]], workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    yield out
    del out, dev, ws
    torch.cuda.empty_cache()


@pytest.mark.parametrize("l,kvh", SLICES)
def test_sampled_slice_effects(full, l, kvh):
    tr, cfg = full["tr"], full["cfg"]
    g = cfg.g
    for post, key in ((False, "H_pre"), (True, "H_post")):
        _, H = core.page_effects(_slice_problem(tr, l, kvh, post), "closed")
        got = _np(full[key][l, kvh * g:(kvh + 1) * g])
        _check_close(got, H[0], TOL, f"{key} slice ({l}, {kvh})")


@pytest.mark.parametrize("l,kvh", SLICES)
def test_sampled_slice_row_stats(full, l, kvh):
    tr, cfg = full["tr"], full["cfg"]
    g = cfg.g
    m, lsum, o_vec, n = core.row_stats(_slice_problem(tr, l, kvh, True))
    st = _np(full["stats"][l, kvh * g:(kvh + 1) * g]).reshape(-1, cfg.d + 4)
    assert np.array_equal(st[:, 2].astype(np.int64), n)
    _check_close(st[:, 0], m, 1e-5, "row max")
    _check_close(st[:, 1], lsum, 1e-4, "row sum")
    err = np.linalg.norm(st[:, 4:] - o_vec, axis=1) / np.maximum(np.linalg.norm(o_vec, axis=1), 1e-30)
    assert err.max() <= 1e-4, err.max()


def test_effect_is_max_over_heads(full):
    for R, H in (("R_pre", "H_pre"), ("R_post", "H_post")):
        r = _np(full[R])
        h = _np(full[H]).reshape(-1, r.shape[0]).max(axis=0)
        assert np.array_equal(r, h), R


def test_classify_fullsize(full):
    """Seeded effects over the full page count (log-uniform between 1e-4 and
    1, so every lifecycle state occurs) through the GPU classifier and the
    oracle's, bit-exact."""
    tr, ws = full["tr"], full["ws"]
    P = tr.P_post
    rng = np.random.default_rng(11)
    Rm = (10.0 ** rng.uniform(-4, 0, P)).astype(np.float32)
    Rp = (10.0 ** rng.uniform(-4, 0, P)).astype(np.float32)
    state = torch.zeros(P, dtype=torch.uint8, device="cuda")
    cand = torch.zeros(P, dtype=torch.int32, device="cuda")
    n_cand = torch.zeros(1, dtype=torch.int32, device="cuda")
    ck.commitkv_classify([P], [torch.from_numpy(Rm).cuda()], [torch.from_numpy(Rp).cuda()],
                         [full["dev"].eligible], [state], [cand], n_cand, ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    o_state, o_cand = core.classify(Rm.astype(np.float64), Rp.astype(np.float64), tr.eligible)
    assert np.array_equal(_np(state), o_state)
    nc = int(n_cand[0])
    assert nc == len(o_cand) and nc > 0
    assert np.array_equal(_np(cand)[:nc], o_cand)


def test_joint_two_layers(full):
    """The joint test over the full cache with two layers selected: the
    GPU's own post-commit statistics of those layers, a seeded candidate
    list (the planted pages, then other eligible pages), and the oracle's
    greedy scan of the same two-layer problem."""
    tr, cfg, dev, shape, ws = full["tr"], full["cfg"], full["dev"], full["shape"], full["ws"]
    mask = np.zeros(cfg.M, np.uint8)
    mask[list(JOINT_LAYERS)] = 1
    stats = torch.zeros(cfg.M, cfg.Hq, cfg.W, cfg.d + 4, dtype=torch.float32, device="cuda")
    R = torch.zeros(tr.P_post, dtype=torch.float32, device="cuda")
    ck.commitkv_page_effects(shape, [dev.post()], [R], stats_out=[stats], layer_mask=mask, workspace=ws)
    rng = np.random.default_rng(5)
    others = np.setdiff1d(np.flatnonzero(tr.eligible), tr.planted)
    cand_np = np.concatenate([tr.planted, rng.choice(others, 16, replace=False)]).astype(np.int32)
    P = tr.P_post
    cand = torch.zeros(P, dtype=torch.int32, device="cuda")
    cand[:len(cand_np)] = torch.from_numpy(cand_np).cuda()
    n_cand = torch.tensor([len(cand_np)], dtype=torch.int32, device="cuda")
    acc = torch.zeros(P, dtype=torch.uint8, device="cuda")
    step = torch.zeros(P, dtype=torch.float32, device="cuda")
    ck.commitkv_joint_test(shape, [dev.post()], [stats], [cand], n_cand, cfg.tau_joint, [acc], [step],
                           layer_mask=mask, workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    o_acc, o_step = core.greedy(_slice_problem(tr, 0, 0, True, layers=JOINT_LAYERS), cand_np,
                                cfg.tau_joint, "closed")
    nc = len(cand_np)
    got_step = _np(step)[:nc]
    got_acc = _np(acc)
    safe = safe_threshold_mask(o_step, cfg.tau_joint, TOL)
    upto = nc if safe.all() else int(np.argmin(safe))
    assert upto > 0
    _check_close(got_step[:upto], o_step[:upto], TOL, "joint step R")
    for j in range(upto):
        assert got_acc[cand_np[j]] == o_acc[cand_np[j]], j
    for j in range(nc):
        assert got_acc[cand_np[j]] == (got_step[j] <= cfg.tau_joint)


def test_compact_fullsize(full):
    """Seeded retired pages, the observation's pages pending with seeded
    priorities, the trajectory's fill scores: I_j bit-exact against the
    oracle's selection, and K, V, positions gathered bit-exactly on the
    sampled slices."""
    tr, cfg, dev, shape, ws = full["tr"], full["cfg"], full["dev"], full["shape"], full["ws"]
    P, S = tr.P_post, tr.S_post
    rng = np.random.default_rng(3)
    retired = (rng.uniform(size=P) < 0.3).astype(np.uint8)
    prio = rng.uniform(size=P).astype(np.float32)
    B, B_N, cap = cfg.B, cfg.B_N, cfg.pending_cap
    idx = torch.zeros(B, dtype=torch.int32, device="cuda")
    n_idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    k_out = torch.empty(cfg.M, cfg.H, B, cfg.d, dtype=torch.bfloat16, device="cuda")
    v_out = torch.empty_like(k_out)
    pos_out = torch.empty(B, dtype=torch.int32, device="cuda")
    ck.commitkv_compact(shape, [dev.post()], [torch.from_numpy(retired).cuda()], [dev.pending],
                        [torch.from_numpy(prio).cuda()], [dev.fill], B, B_N, cap, [idx], n_idx, [k_out],
                        [v_out], [pos_out], workspace=ws)
    torch.cuda.synchronize()
    assert ck.commitkv_workspace_status(ws) == ck.COMMITKV_OK
    I = core.select_indices(S, tr.page_start, tr.page_len, retired, tr.pending,
                            prio[tr.pending].astype(np.float64), tr.fill_score, B, B_N, cap)
    n = int(n_idx[0])
    assert n == len(I)
    assert np.array_equal(_np(idx)[:n], I)
    assert np.array_equal(_np(pos_out)[:n], tr.pos[I])
    for l, kvh in SLICES:
        assert np.array_equal(_np(k_out[l, kvh, :n].view(torch.uint16)), tr.K[l, kvh, I])
        assert np.array_equal(_np(v_out[l, kvh, :n].view(torch.uint16)), tr.V[l, kvh, I])
