"""bench.py's own arithmetic, without a GPU: the roofline units against the oracle's counts
(Sec. 3.3), and the parsing of the nvidia-smi samples that go beside every timed number."""
import os
import sys

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

SHAPES = [(4096, 4096, 2048), (11008, 4096, 2048), (4096, 11008, 2048), (8192, 8192, 4096), (28672, 8192, 4096),
          (256, 256, 128), (300, 200, 77)]


@pytest.mark.parametrize("m,n,r", SHAPES)
@pytest.mark.parametrize("T", [1, 8, 16, 2048])
def test_roofline_units_match_the_paper_counts(m, n, r, T):
    """Decode bytes = every stored weight once in bf16 (the oracle's storage count, Sec. 3.3), X
    read and Y written in bf16, both int32 index arrays; prefill FLOPs = the oracle's count."""
    assert bench.decode_bytes(T, m, n, r) == 2 * oracle.storage_count(m, n, r) + 2 * T * (n + m) + 4 * m
    assert bench.pifa_flops(T, m, n, r) == oracle.flop_count(T, m, n, r)


def test_attn7b_decode_bytes_value():
    """The main line's unit: 25.31 MB per call at 4096 x 4096, r = 2048, T = 8."""
    assert bench.decode_bytes(8, 4096, 4096, 2048) == 25_313_280


def _sampler(lines):
    c = bench.ClockSampler(0)
    c.lines = lines
    return c.summary()


def test_clock_summary_with_memory_clock_and_temperatures():
    s = _sampler(["2070, 2070, 300.1, Active, Not Active, Not Active, Not Active, Not Active, 3996, 55, 61",
                  "2070, 2070, 310.0, Active, Not Active, Not Active, Not Active, Active, 3996, 57, 63",
                  "1900, 2070, 320.0, Active, Not Active, Not Active, Not Active, Not Active, 3996, 58, 64"])
    assert s["sm_mhz"] == 2070 and s["sm_max_mhz"] == 2070 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    assert s["mem_mhz"] == 3996 and s["gpu_temp_c"] == [55, 58] and s["hbm_temp_c"] == [61, 64]


def test_clock_summary_without_the_extra_fields_or_with_na():
    s = _sampler(["2070, 2070, 300.1, Active, Not Active, Active, Not Active, Not Active",
                  "2070, 2070, 300.1, Active, Not Active, Not Active, Not Active, Not Active, 3996, 50, [N/A]",
                  "garbage line", ""])
    assert s["samples"] == 2 and s["reasons"] == ["hw_thermal_slowdown"]
    assert s["gpu_temp_c"] == [50, 50] and "hbm_temp_c" not in s


def test_clock_summary_empty():
    assert _sampler([]) == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}


@pytest.mark.parametrize("m,n,r", SHAPES + [(40000, 520, 264), (30000, 520, 264), (19456 + 4096, 8192, 4096)])
def test_bench_decode_rule_is_the_library_selector(m, n, r):
    """bench.py names a workload decode (HBM roofline, L2-defeating weight copies) exactly when the
    library's selector runs the decode variant."""
    from paper_2501_19090_gb300 import pifa as P
    for T in (1, 16, 64, 65, 96, 128, 129, 2048):
        assert (P.pifa_select_variant(T, m, n, r) == P.PIFA_VARIANT_DECODE) == bench.is_decode(T, m, r), T
