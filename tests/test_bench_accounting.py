"""The benchmark's roofline accounting against values worked out by hand.

Every reported fraction divides by these numbers, so they are pinned here
from the definitions, independently of bench.py's code:
  eviction bytes = e Hkv d (N + 4 R) + q_win bytes
      (K read once to score; retained K and V rows read and written),
  decode bytes   = 2 e Hkv d len + B Hq d (e + 4)
      (K and V of the compacted cache; the query and the fp32 output),
  scoring flops  = 2 Hq W d N (the method's one Q K^T over the N keys),
      executed as 2 Hq W d (N + (N - W)) by the two-pass kernel
      (N keys for the row statistics, then the N - W prefix keys),
with R = k + W and k = ceil((1 - alpha) N) prefix rows (Eq. 8 reading).
"""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2512_21859_gb300 import inputs  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2512_21859_gb300 import binding, build
    build.build()
    binding.load()


def test_32k_alpha_half():
    wl = inputs.WORKLOADS["32k"]            # 28q / 4kv, d 128, bf16, W 32
    n, a = np.array([32768]), np.array([0.5])
    # k = 16384, R = 16416; decode length R + 1 (the step's own row)
    ab = bench.alg_bytes(wl, n, a, [16417])
    assert ab["R"] == [16416]
    q_win = 28 * 32 * 128 * 2                            # 229,376
    assert ab["evict"] == 2 * 4 * 128 * (32768 + 4 * 16416) + q_win == 101_023_744
    assert ab["decode_attn"] == 2 * 2 * 4 * 128 * 16417 + 28 * 128 * (2 + 4) == 33_643_520
    assert ab["step"] == ab["evict"] + ab["decode_attn"]
    assert ab["gather_kv"] == 4 * 2 * 128 * 4 * 16416    # retained K, V rows read and written
    assert ab["window_scores"] == 2 * 128 * 4 * 32768 + q_win


def test_128k_alpha_point_nine():
    wl = inputs.WORKLOADS["128k"]           # 32q / 8kv, d 128, bf16, W 64
    n, a = np.array([131072]), np.array([0.9])
    # (1 - 0.9) * 131072 = 13107.2 -> k = 13108, R = 13172
    ab = bench.alg_bytes(wl, n, a, [13173])
    assert ab["R"] == [13172]
    q_win = 32 * 64 * 128 * 2                            # 524,288
    assert ab["evict"] == 2 * 8 * 128 * (131072 + 4 * 13172) + q_win == 376_864_768
    assert ab["decode_attn"] == 2 * 2 * 8 * 128 * 13173 + 32 * 128 * (2 + 4) == 53_981_184
    peaks = {"hbm_gbs": 6790.3, "bf16_tflops": 1904.5, "bf16_tflops_sustained": 1717.4}
    roof = bench.stage_rooflines(wl, n, ab, {"window_scores": 0.1, "decode_attn": 0.01}, peaks)
    method = 2 * 32 * 64 * 128 * 131072
    executed = 2 * 32 * 64 * 128 * (131072 + (131072 - 64))
    t = roof["window_scores"]["tensor"]
    assert t["flops"] == method == 68_719_476_736
    assert t["executed_flops"] == executed == 137_405_399_040
    # 0.1 ms per launch: 687.19 TFLOP/s of the method's flops against the burst 1904.5
    assert t["frac"] == pytest.approx(687.19476736 / 1904.5, abs=1e-4)
    assert t["executed_frac"] == pytest.approx(1374.0539904 / 1904.5, abs=1e-4)
    # the headline roofline is HBM: 268,959,744 bytes (K once + q_win) in 0.1 ms
    assert ab["window_scores"] == 2 * 8 * 128 * 131072 + q_win == 268_959_744
    assert roof["window_scores"]["frac"] == pytest.approx(2689.59744 / 6790.3, abs=1e-4)
    assert roof["decode_attn"]["achieved_gbs"] == pytest.approx(53_981_184 / 1e-5 / 1e9, rel=1e-3)


def test_ragged_batch_sums_per_request():
    wl = inputs.WORKLOADS["ragged"]         # 28q / 4kv, d 128, bf16, W 32
    n = np.array([1024, 5000, 16384])
    a = np.array([0.1, 0.5, 0.9])
    # k_b = ceil((1 - a_b) n_b): 922, 2500, 1639 (16384 * 0.1 = 1638.4)
    R = [922 + 32, 2500 + 32, 1639 + 32]
    ab = bench.alg_bytes(wl, n, a, [r + 1 for r in R])
    assert ab["R"] == R
    q_win = 3 * 28 * 32 * 128 * 2
    assert ab["evict"] == 2 * 4 * 128 * (int(n.sum()) + 4 * sum(R)) + q_win
    assert ab["decode_attn"] == 2 * 2 * 4 * 128 * sum(r + 1 for r in R) + 3 * 28 * 128 * 6
