"""Host arithmetic of bench.py (CPU): the roofline terms per step, the
launch count per step, and the peak it divides by."""
import json
import os
import types

import bench
from paper_2608_07855_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_algorithmic_terms_of_the_qwen3_8b_32k_step():
    """K and V of both caches read once: M H 2 d bytes of bf16 per token;
    Q K^T and P V once: 4 g W d flops per token and KV head."""
    cfg = synth.CONFIGS["qwen3_8b_32k"]
    bpt, fpt = bench.algorithmic(cfg)
    assert bpt == 36 * 8 * 2 * 128 * 2
    assert fpt == 36 * 8 * 4 * 4 * 32 * 128
    tokens = 32768 + (32768 + 4096 + 32)  # pre-commit cache + post-commit cache (window included)
    assert bpt * tokens == 10_272_374_784
    assert cfg.g == 4


def test_launches_per_step():
    """Tensor-core path: prep, flash pass, combine, page pass (one scoring
    call over both caches of up to 8 trajectories), two classify kernels,
    the joint test, select and gather."""
    for n, cfg in ((1, synth.CONFIGS["qwen3_8b_32k"]), (16, synth.CONFIGS["ragged16"])):
        buf = types.SimpleNamespace(cfg=cfg, trajs=[None] * n)
        groups = (2 * n + 15) // 16
        assert bench.buf_launches(buf) == 4 * groups + 2 + 1 + 2
    tiny = types.SimpleNamespace(cfg=synth.CONFIGS["tiny"], trajs=[None])
    assert bench.buf_launches(tiny) == 3 + 2 + 1 + 2


def test_peaks_are_the_measured_ones():
    """The denominators are the measured peaks when the measurement file is
    there, else the documented fallback."""
    peaks, kind = bench.load_peaks()
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if not os.path.exists(path):
        assert kind == "fallback" and peaks == bench.PEAKS_FALLBACK
        return
    with open(path) as f:
        m = json.load(f)
    assert kind == "measured"
    assert peaks["hbm_gbs"] == m["hbm_gbs"] and peaks["bf16_tflops_sustained"] == m["bf16_tflops_sustained"]


def test_reference_arm_reports_the_same_config_keys():
    """The reference arm's line describes the workload with the same keys
    and values as ours, and its CPU baseline names the host CPU model."""
    args = types.SimpleNamespace(config="tiny", layers=0, seed=0, steps=1, warmup=0,
                                 cpu_sample_seconds=0.5)
    res = bench.run_reference(args, 0, 1)
    cfg = synth.CONFIGS["tiny"]
    trs = [synth.make_trajectory(cfg, 0, traj=0, values=False)]
    assert res["config"] == bench.config_dict(cfg, trs, 1)
    assert res["impl"] == "reference" and res["cpu_baseline"]["cpu_model"]
    assert isinstance(res["config"]["L_pre"], list) and "budget" in res["config"]


def test_joint_report_counts():
    """Candidates, acceptances, rounds of four and time per candidate of
    the joint test, summed over the trajectories of a step."""
    import numpy as np

    class T:
        def __init__(self, n):
            self.n = n

        def cpu(self):
            return self

        def tolist(self):
            return self.n

    acc = [np.array([1, 0, 1, 1, 0], np.uint8), np.array([0, 1, 0], np.uint8)]
    buf = types.SimpleNamespace(n_cand=T([5, 2]), accepted=[a for a in acc],
                                trajs=[types.SimpleNamespace(P_post=5), types.SimpleNamespace(P_post=3)])
    r = bench.joint_report(buf, 0.7)
    assert r["n_cand"] == 7 and r["accepted"] == 4 and r["rejected"] == 3
    assert r["rounds"] == 2 and abs(r["us_per_candidate"] - 100.0) < 1e-9


def test_recorded_traffic_belongs_to_the_current_kernels():
    """The DRAM bytes bench.py reports as roofline.traffic were captured with
    the scoring sources as they are now (their sha256 prefix), and lie
    between once and three times the algorithmic bytes of the step."""
    cfg = synth.CONFIGS["qwen3_8b_32k"]
    traffic, sha = bench.MEASURED_TRAFFIC[cfg.name]
    assert sha == bench.scoring_sources_sha()
    bpt, _ = bench.algorithmic(cfg)
    algo = bpt * (32768 + (32768 + 4096 + 32))
    assert algo <= traffic <= 3 * algo
