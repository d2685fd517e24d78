"""The benchmark's algorithmic work per step (bench.algorithmic), against the
byte counts written out by hand for two workloads.

The HBM fraction in the bench line divides these bytes by the step time, and
the tensor roofline divides these flops by the dominant pass's time, so a
wrong count would misstate both. Bytes per step: K read once (T x Hkv x d x
2 bytes per layer) plus the gathered K and V rows read and written (4 x kept
rows x Hkv x d x 2 bytes per layer). Flops per softmax pass: 2 d per (proxy
row, key, KV head, layer), with N r proxy rows plus the r anchor rows per KV
head.
"""
import numpy as np

import bench
from paper_2607_22586_gb300 import synth as S

PAPER = dict(n_proxies=512)


def test_32k_stack_bytes_and_flops():
    wl = S.WORKLOADS["qwen7b-28l-32k"]
    total, k_read, flops = bench.algorithmic(wl, PAPER)
    # 28 layers x 32768 keys x 4 KV heads x 128 dims x 2 bytes: 33.55 MB a layer
    assert k_read == 28 * 33_554_432
    # 2048 kept rows per head: 8.39 MB a layer of gather traffic
    assert total - k_read == 28 * 8_388_608
    assert total == 1_174_405_120
    # (512 x 7 + 7) proxy rows per KV head
    assert flops == 2.0 * 128 * 3591 * 32768 * 4 * 28


def test_72b_ragged_bytes():
    wl = S.WORKLOADS["72b-80l-ragged"]
    total, k_read, _ = bench.algorithmic(wl, PAPER)
    tokens = 2048 + 3000 + 4096 + 6000 + 8192 + 12000 + 16384 + 24576        # 76,296
    kept = 192 + 320 + 384 + 576 + 832 + 1216 + 1664 + 2432                  # 10% rounded to 64
    assert k_read == 80 * tokens * 8 * 128 * 2                              # 156.3 MB a layer
    assert total - k_read == 80 * 4 * kept * 8 * 128 * 2                    # 62.4 MB a layer


def test_head_budgets_count_each_heads_kept_rows():
    wl = S.WORKLOADS["qwen7b-1layer"]
    T = wl.seq_lens[0]
    hb = np.array([[[1, 2, T + 5, 7]]], dtype=np.int32)      # [L][B][Hkv]; one budget above T
    total, k_read, _ = bench.algorithmic(wl, PAPER, hb)
    assert total - k_read == 4 * (1 + 2 + T + 7) * wl.head_dim * 2


def test_pyramid_budgets_average_the_uniform_budget():
    wl = S.WORKLOADS["qwen7b-28l-32k"]
    hb = bench.pyramid_budgets(wl)
    C = wl.budgets[0]
    assert hb.shape == (28, 1, 4) and hb.dtype == np.int32
    assert hb[0, 0, 0] == round(1.5 * C) and hb[-1, 0, 0] == round(0.5 * C)
    assert np.all(np.diff(hb[:, 0, 0]) <= 0)                      # shrinking with depth
    assert abs(hb.mean() - C) <= 1.0                               # C on average
    assert np.all(hb == hb[:, :, :1])                              # equal across heads


PEAKS = {"hbm_gbs": 6783.5, "bf16_tflops": 1910.3, "bf16_tflops_sustained": 1704.3,
         "sm_max_mhz": 2070.0, "clocks_under_load": {"sm_mhz_median": 1447.0}}


def test_tensor_peak_follows_the_clock_seen():
    """A timed region at the maximum SM clock is held to the burst GEMM peak;
    one whose median clock sat near the sustained run's clock to the
    sustained peak; with no clock record, the higher (burst) peak."""
    peak, kind = bench.tensor_peak(PEAKS, {"sm_mhz": 2070.0}, "measured")
    assert peak == 1910.3 and "burst" in kind
    peak, kind = bench.tensor_peak(PEAKS, {"sm_mhz": 1500.0}, "measured")
    assert peak == 1704.3 and "sustained" in kind
    peak, kind = bench.tensor_peak(PEAKS, None, "measured")
    assert peak == 1910.3 and "no clock record" in kind


def test_score_roofline_recomputes_from_stage_times():
    """The reported fraction is the pass's algorithmic flops over its event
    time over the chosen peak: recomputable from stage_ms and the formula."""
    wl = S.WORKLOADS["qwen7b-28l-32k"]
    stage = {"softmax_pass": 3.2, "mass_pass": 3.416}
    roof = bench.score_roofline(wl, PAPER, stage, True, PEAKS, "measured", {"sm_mhz": 2070.0})
    flops = 2.0 * 128 * (512 * 7 + 7) * 32768 * 4 * 28
    assert roof["kernel"] == "mass_pass"
    assert abs(roof["achieved"] - flops / 3.416e-3 / 1e12) < 1e-6
    assert abs(roof["frac"] - roof["achieved"] / 1910.3) < 1e-12
    assert abs(roof["frac"] - 0.517) < 0.002
    assert abs(roof["hbm"]["bytes_per_launch"] - 28 * 33_554_432) < 1
