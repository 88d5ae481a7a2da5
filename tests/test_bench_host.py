"""Host-side arithmetic of the benchmark: the algorithmic FLOP counts and the
per-kernel rooflines built from per-launch event times (no GPU needed)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_29809_gb300 import synth  # noqa: E402


@pytest.mark.parametrize("folded", [True, False])
def test_flops_per_token_block_sum_to_the_method_count(folded):
    """Folding the cross-query projection into the text keys moves its 2 h^2
    from the GEMMs to the cross-attention; the total stays 28 h^2 (linear
    layers at F = 4 h) + 4 N h (self-attention) + 4 M h (cross-attention)."""
    d = synth.PIXART_1024
    h, N, M = d.hidden, d.tokens, d.text_len
    total = (bench.linear_flops_per_token_block(d, folded) +
             bench.attn_flops_per_token_block(d, folded))
    assert d.mlp == 4 * h
    assert total == 28 * h * h + 4 * N * h + 4 * M * h
    assert total == pytest.approx(56.59e6, rel=1e-4)


@pytest.mark.parametrize("per_block", [5, 6])
def test_kernel_rooflines_from_event_times(per_block):
    d = synth.PIXART_1024
    D, steps, peak = 831, 3, 1726.6
    gemm_us = {5: [18.0, 18.0, 14.0, 21.0, 22.0], 6: [18.0, 18.0, 13.0, 14.0, 21.0, 22.0]}[per_block]
    att_us = [49.0, 16.0]
    gemm_each = [u / 1e3 for u in gemm_us] * (d.layers * steps)
    att_each = [u / 1e3 for u in att_us] * (d.layers * steps)
    roof, roof_att = bench.kernel_rooflines(d, D, gemm_each, att_each, peak)
    folded = per_block == 5
    assert roof["cross_query_folded_into_attention"] is folded
    assert roof["launches"] == per_block * d.layers * steps
    names = list(roof["per_gemm"])
    assert names == (["qkv", "out", "cross_out", "fc1", "fc2"] if folded else
                     ["qkv", "out", "cross_q", "cross_out", "fc1", "fc2"])
    for name, us in zip(names, gemm_us):
        g = roof["per_gemm"][name]
        assert g["avg_us"] == pytest.approx(us)
        n, k = g["shape"][1], g["shape"][2]
        assert g["tflops"] == pytest.approx(2 * D * n * k / (us * 1e-6) / 1e12, abs=0.06)
    lin = bench.linear_flops_per_token_block(d, folded) * D * d.layers * steps
    want = lin / (sum(gemm_each) / 1e3) / 1e12
    assert roof["achieved"] == pytest.approx(want, abs=0.006)
    assert roof["frac"] == pytest.approx(want / peak, abs=1e-4)
    att = bench.attn_flops_per_token_block(d, folded) * D * d.layers * steps
    assert roof_att["achieved"] == pytest.approx(att / (sum(att_each) / 1e3) / 1e12, abs=0.006)
    assert roof_att["per_launch"]["self"]["keys"] == d.tokens
    assert roof_att["per_launch"]["cross"]["keys"] == d.text_len


def test_nearest_rank_percentiles():
    xs = [5.0, 1.0, 4.0, 2.0, 3.0]
    assert bench.pct(xs, 50) == 3.0
    assert bench.pct(xs, 99) == 5.0
    assert bench.pct(xs, 1) == 1.0
    assert bench.pct(list(range(1, 101)), 99) == 99
