"""The integer-pipe probe behind the verification roofline: its measured
lane rates must be physical (at most the 128 issue lanes per clock per SM,
each pipe at most its 64 lanes), and the pipes must be distinct (the mix of
both runs near their sum), or the roofline's denominator would be wrong."""
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # the probe is a GPU kernel
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2609_18178_gb300 import peak  # noqa: E402


def test_probe_rates_are_physical():
    r = peak.int_rates(iters=2048, reps=3, kinds=("alu", "fma", "both", "mulhi", "mulwide", "mul64", "mul64x"))
    alu, fma, both = (r[k]["lane_ops_per_clk_per_sm"] for k in ("alu", "fma", "both"))
    assert 40 <= alu <= 64.5 and 40 <= fma <= 64.5
    assert 1.6 * min(alu, fma) <= both <= 128.5
    # a high multiply-add takes more of the multiply pipe than a plain one
    assert r["mulhi"]["lane_ops_per_clk_per_sm"] < 0.8 * fma
    assert r["mulwide"]["lane_ops_per_clk_per_sm"] > 0.8 * fma
    # a 64-bit multiply is three multiply-adds, one of them widening: at most
    # the plain rate, and not far below it
    for k in ("mul64", "mul64x"):
        assert 0.4 * fma <= r[k]["lane_ops_per_clk_per_sm"] <= 1.01 * fma
    for k in ("alu", "fma", "both"):
        assert r[k]["lane_ops_per_s"] > 0
