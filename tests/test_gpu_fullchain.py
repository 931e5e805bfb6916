"""Whole-chain parity of one step of the Qwen3-8B-shaped workloads (36
layers, 32 query / 8 KV heads, head_dim 128, bf16): 32K + 4K, 16K + 2K, and
one trajectory of the 16 of the ragged batch, which runs with the other 15
in the same launches.  The launch configuration is the one the benchmark
times (StepBuffers.step: one scoring call over both caches of the batch,
classify, joint test, compaction); against the oracle:

  * R- and R+ of every page over all 288 (layer, KV head) slices of each
    cache (Eq. 6-8), within the bf16 tolerance (2e-2 relative);
  * the classification (Eq. 9-10) of the GPU's own effects equals the
    oracle classifier's on the same fp32 values, bit for bit, and the
    oracle's own classification wherever its margin is safe;
  * the joint test (Eq. 11) over all 36 layers on the GPU's candidate list
    against the oracle's greedy scan of that list, step values and decisions
    up to the first step whose margin is within the tolerance;
  * the selection (Eq. 12-13) on the GPU's decisions and priorities,
    bit-exact, and the gather (Eq. 4) on sampled slices, bit-exact.

The oracle's effects are computed one layer at a time (the maximum over
layers of the per-layer effects is the effect over all layers, Eq. 7); the
joint scan needs every layer at once.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import core  # noqa: E402
from paper_2608_07855_gb300 import commitkv as ck  # noqa: E402
from paper_2608_07855_gb300 import synth  # noqa: E402
from paper_2608_07855_gb300.workload import DeviceTrajectory, StepBuffers  # noqa: E402

from oracle_bridge import percentile_safe, rel_close, safe_threshold_mask  # noqa: E402

pytestmark = pytest.mark.gpu

TOL = 2e-2


def _np(t):
    return t.detach().cpu().numpy()


def _check(got, want, what):
    ok = rel_close(got, want, TOL)
    if not ok.all():
        bad = np.flatnonzero(~ok)[:6]
        raise AssertionError(f"{what}: {int((~ok).sum())} of {ok.size} outside {TOL}: "
                             + ", ".join(f"[{i}] gpu {got[i]:.6g} oracle {want[i]:.6g}" for i in bad))


# (workload, trajectory checked, least number of candidates the planted pages give)
CHAINS = [("qwen3_8b_32k", 0, 100), ("qwen3_8b_16k", 0, 40), ("ragged16", 0, 20)]


@pytest.mark.parametrize("name,t,min_cand", CHAINS)
def test_full_chain(name, t, min_cand):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    ck.load_library()
    cfg = synth.CONFIGS[name]
    trs = [synth.make_trajectory(cfg, 0, traj=i) for i in range(cfg.n_traj)]
    devs = [DeviceTrajectory.upload(x) for x in trs]
    b = StepBuffers(cfg, devs)
    b.step()
    torch.cuda.synchronize()
    assert b.status() == ck.COMMITKV_OK
    tr = trs[t]
    Rm_g = _np(b.R_pre[t]).astype(np.float64)  # [P_post]; the observation's pages stay 0
    Rp_g = _np(b.R_post[t]).astype(np.float64)
    state_g = _np(b.state[t])
    nc = int(b.n_cand[t])
    cand_g = _np(b.cand[t])[:nc].astype(np.int64)
    acc_g = _np(b.accepted[t])[:tr.P_post]
    step_g = _np(b.step_R[t])[:nc]
    n_idx = int(b.n_idx[t])
    idx_g = _np(b.idx[t])[:n_idx]
    k_out, v_out, pos_out = b.k_out[t], b.v_out[t], _np(b.pos_out[t])[:n_idx]

    # 1. effects of every page over every slice, one layer at a time
    f64 = lambda a: synth.values_f64(a, cfg.dtype)  # noqa: E731
    L = tr.L_pre
    Rm_o = np.zeros(tr.P_pre)
    Rp_o = np.zeros(tr.P_post)
    for l in range(cfg.M):
        K, V = f64(tr.K[l:l + 1]), f64(tr.V[l:l + 1])
        pre = core.Problem(K[:, :, :L], V[:, :, :L], tr.pos[:L], f64(tr.Q_pre[l:l + 1]), tr.qpos_pre,
                           tr.page_start[:tr.P_pre], tr.page_len[:tr.P_pre])
        post = core.Problem(K, V, tr.pos, f64(tr.Q_post[l:l + 1]), tr.qpos_post, tr.page_start, tr.page_len)
        Rm_o = np.maximum(Rm_o, core.page_effects(pre, "closed")[0])
        Rp_o = np.maximum(Rp_o, core.page_effects(post, "closed")[0])
    _check(Rm_g[:tr.P_pre], Rm_o, "R- (every page, all layers and heads)")
    _check(Rp_g, Rp_o, "R+ (every page, all layers and heads)")

    # 2. classification: the GPU's candidates are the oracle classifier's on the
    # GPU's own fp32 effects; states equal the oracle chain's where safe
    s_g, c_g = core.classify(Rm_g, Rp_g, tr.eligible)
    assert np.array_equal(state_g, s_g)
    assert np.array_equal(cand_g, c_g)
    Rm_o_full = np.zeros(tr.P_post)
    Rm_o_full[:tr.P_pre] = Rm_o
    s_o, c_o = core.classify(Rm_o_full.astype(np.float32), Rp_o.astype(np.float32), tr.eligible)
    idx = np.flatnonzero(tr.eligible)
    safe = percentile_safe(Rm_o_full, idx, TOL) & percentile_safe(Rp_o, idx, TOL)
    for th in (0.05, 0.01):
        safe &= safe_threshold_mask(Rm_o_full[idx], th, TOL) & safe_threshold_mask(Rp_o[idx], th, TOL)
    assert safe.any()
    assert np.array_equal(state_g[idx][safe], s_o[idx][safe])
    # the workload plants completion candidates: a realistic count of them
    assert nc >= min_cand, nc

    # 3. joint test over all 36 layers on the GPU's candidate list
    del K, V, pre, post
    post = core.Problem(f64(tr.K), f64(tr.V), tr.pos, f64(tr.Q_post), tr.qpos_post, tr.page_start, tr.page_len)
    acc_o, step_o = core.greedy(post, cand_g, cfg.tau_joint, "closed")
    del post
    safe_s = safe_threshold_mask(step_o, cfg.tau_joint, TOL)
    upto = nc if safe_s.all() else int(np.argmin(safe_s))
    assert upto >= min(nc, 20), (upto, nc)
    _check(step_g[:upto].astype(np.float64), step_o[:upto], "joint step R")
    for j in range(upto):
        assert acc_g[cand_g[j]] == acc_o[cand_g[j]], j
    for j in range(nc):
        assert acc_g[cand_g[j]] == (step_g[j] <= cfg.tau_joint), j
    assert not acc_g[np.setdiff1d(np.arange(tr.P_post), cand_g)].any()
    assert 0 < int(acc_g.sum()) < nc  # acceptances and rejections both occur

    # 4. selection on the GPU's decisions and priorities (R+ of the pending
    # pages), bit-exact; the gather on sampled slices
    I = core.select_indices(tr.S_post, tr.page_start, tr.page_len, acc_g, tr.pending,
                            Rp_g[tr.pending], tr.fill_score, cfg.B, cfg.B_N, cfg.pending_cap)
    assert n_idx == len(I)
    assert np.array_equal(idx_g, I)
    assert np.array_equal(pos_out, tr.pos[I])
    for l, kvh in ((0, 0), (17, 5), (35, 7)):
        assert np.array_equal(_np(k_out[l, kvh, :n_idx].view(torch.uint16)), tr.K[l, kvh, I])
        assert np.array_equal(_np(v_out[l, kvh, :n_idx].view(torch.uint16)), tr.V[l, kvh, I])
