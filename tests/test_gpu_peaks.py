"""The measurement helper gaus_measure_peak on the device: plausible FP32 FMA and SFU
exp2 throughputs (the nominal FP32 rate is SMs x 128 lanes x 2 flop x clock)."""
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def g():
    import paper_2602_20427_gb300 as g
    g.build()
    g.lib()
    return g


def test_fp32_and_ex2_throughput_are_plausible(g):
    props = torch.cuda.get_device_properties(0)
    nominal = props.multi_processor_count * 128 * 2 * 2.2e9   # above any boost clock
    fp32 = g.measure_peak(g.PEAK_FP32)
    ex2 = g.measure_peak(g.PEAK_EX2)
    assert 0.2 * nominal < fp32 < 1.05 * nominal, (fp32, nominal)
    # the SFU is slower than the FMA pipe, but it is not a software loop
    assert 1e11 < ex2 < fp32, (ex2, fp32)
