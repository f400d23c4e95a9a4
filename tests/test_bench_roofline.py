"""bench.py's roofline arithmetic on CPU: the algorithmic work per kernel, the
choice of roofline by arithmetic intensity, the achieved fraction, and the
committed ncu traffic lookup."""
import pytest

import bench
from paper_2508_06024_gb300 import synth as S

PEAKS = {"hbm_gbs": 6689.1, "bf16_tflops": 1923.1}


def test_switch_up_projection_work():
    cfg = S.preset("switch_bf16")
    flops, byts = bench.kernel_work(cfg, "expert_up")
    n, d, ff, allowed = 4096, 768, 3072, 12
    assert flops == 2.0 * n * d * ff
    # the allowed experts' W1 once, the rows in and the hidden rows out, bf16
    assert byts == 2 * (allowed * ff * d + n * d + n * ff) == 88080384


def test_touched_experts_replace_the_allowed_count():
    cfg = S.preset("decode_bf16", T=1)
    _, all_allowed = bench.kernel_work(cfg, "expert_up")
    _, two = bench.kernel_work(cfg, "expert_up", touched=2)
    w = 2 * 2 * cfg.d_ff * cfg.d  # SwiGLU: W1 and W3, bf16
    assert all_allowed - two == (cfg.n_allowed - 2) * w


def test_roofline_follows_arithmetic_intensity():
    sw = bench.roofline_for(S.preset("switch_bf16"), "expert_up", 0.0325, PEAKS, "measured", None)
    assert sw["bound"] == "hbm"  # ~219 flop/B, below the ridge of ~287
    assert sw["achieved"] == pytest.approx(88080384 / 0.0325e-3 / 1e9, rel=1e-3)
    assert sw["frac"] == pytest.approx(sw["achieved"] / PEAKS["hbm_gbs"], rel=1e-3)
    mx = bench.roofline_for(S.preset("mixtral_bf16"), "expert_up", 2.1, PEAKS, "measured", None)
    assert mx["bound"] == "tensor"
    cfg = S.preset("mixtral_bf16")
    n = cfg.T * cfg.k
    assert mx["achieved"] == pytest.approx(2.0 * n * cfg.d * cfg.d_ff * 2 / 2.1e-3 / 1e12, rel=1e-3)


def test_reduce_kernels_carry_no_layer_flops():
    cfg = S.preset("decode_bf16", T=64)
    for name in ("gate_decide", "lr_reduce"):
        flops, byts = bench.kernel_work(cfg, name)
        assert flops == 0.0 and byts > 0
        assert bench.roofline_for(cfg, name, 0.01, PEAKS, "measured", None)["bound"] == "hbm"


def test_committed_traffic_lookup():
    sw = S.preset("switch_bf16")
    up = bench.committed_traffic(sw, "expert_up")
    assert up is not None and 0.5 < up / bench.kernel_work(sw, "expert_up")[1] < 1.5
    assert bench.committed_traffic(sw, "no_such_kernel") is None
    # a bare preset name holds for the preset's own token count only
    assert bench.committed_traffic(sw.replace(T=2048), "expert_up") is None
    dec = S.preset("decode_bf16", T=1)
    assert bench.committed_traffic(dec, "expert_up") is not None
    assert bench.committed_traffic(S.preset("decode_bf16", T=2), "expert_up") is None
