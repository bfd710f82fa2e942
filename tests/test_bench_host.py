"""Host-side logic of bench.py without a GPU: the verification pass's
integer ceiling (the splitmix64 operation count split over the two integer
pipes), the reference arm's line (the CPU oracle over a bounded sample,
reporting exactly what it ran), and the digest sum over ranks."""
import io
import json
import os
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def rates(alu, fma):
    return {"alu": {"lane_ops_per_clk_per_sm": alu}, "fma": {"lane_ops_per_clk_per_sm": fma}}


def test_term_operation_counts():
    """20 operations per term as defined, whatever the word width: the
    16-bit identity turns a funnel shift into a one-pipe-or-the-other
    multiply-add, it does not remove it."""
    for t in bench.TERM_OPS.values():
        assert t["alu_only"] + t["mul_only"] + t["flex"] + t["funnel"] == 20
        assert t["alu_only"] == 6 and t["mul_only"] == 6


def test_integer_ceiling_closed_forms():
    words = {"f32": 3, "bf16": 1}
    # equal pipes: the flexible work balances them, and issue (80 ops at 128
    # lanes per clock) binds: 1.6 elements per clock per SM
    assert bench.integer_ceiling(words, rates(64, 64)) == pytest.approx(128 / 80, rel=1e-3)
    # a half-width multiply pipe: balance (56 - x) / 64 = (24 + x) / 32 at
    # x = 8/3 moved operations, 53.33 ALU operations per element
    assert bench.integer_ceiling(words, rates(64, 32)) == pytest.approx(64 / (56 - 8 / 3), rel=1e-3)
    # no room on the multiply pipe beyond its own multiplies: everything
    # else on the ALU (56 of the 80 operations)
    assert bench.integer_ceiling(words, rates(64, 1e-9 + 24 * 64 / 56)) == pytest.approx(64 / 56, rel=2e-2)
    # an ALU far faster than issue: issue binds at 80 operations
    assert bench.integer_ceiling(words, rates(1e6, 1e6)) == pytest.approx(128 / 80, rel=1e-6)
    # 64-bit multiplies measured at full rate change nothing
    full = dict(rates(64, 64), mul64={"lane_ops_per_clk_per_sm": 64})
    assert bench.integer_ceiling(words, full) == pytest.approx(128 / 80, rel=1e-3)
    # at half rate the 24 multiply-adds take 0.75 clocks; balance
    # (56 - x) / 64 = 0.75 + x / 64 at x = 4 gives 52 / 64 clocks per element
    half = dict(rates(64, 64), mul64={"lane_ops_per_clk_per_sm": 32})
    assert bench.integer_ceiling(words, half) == pytest.approx(64 / 52, rel=1e-3)
    # of two measured forms, the faster one counts
    assert bench.integer_ceiling(words, dict(half, mul64x={"lane_ops_per_clk_per_sm": 64})) == \
        pytest.approx(128 / 80, rel=1e-3)


def test_reference_arm_reports_what_it_ran():
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.main(["--impl", "reference", "--steps", "2", "--warmup", "1", "--ref-elements", str(1 << 16)])
    line = json.loads(buf.getvalue().strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["config"]["elements"] == 1 << 16
    assert line["value"] == pytest.approx((1 << 16) / (line["ms_per_step"] * 1e-3), rel=1e-9)
    assert line["verify_matches_commit"] is True
    assert line["cpu_baseline"]["value"] == line["value"] and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["higher_is_better"] is True and line["unit"] == "elements/s"


def test_sum_over_ranks_single_process_wraps():
    d = [(1 << 64) - 1, 5, 1 << 63, 0]
    assert bench.sum_over_ranks(None, d) == d
