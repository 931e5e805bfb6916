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
