"""The FP32 FMA-rate probe behind the FP32 roofline denominator runs through the C ABI,
reports the FLOPs of its launch and stores every chain's result."""
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_fma_probe_flops_and_outputs():
    from paper_2607_05272_gb300 import build as B
    B.build()
    from paper_2607_05272_gb300 import simx
    n = simx.fma_probe_sink_floats()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert n == sms * 4 * 256
    sink = torch.full((n,), float("nan"), device="cuda")
    flops = simx.fma_probe(10, sink)
    torch.cuda.synchronize()
    assert flops == 2.0 * 16 * 10 * n
    assert bool(torch.isfinite(sink).all())
    with pytest.raises(simx.SimxError):
        simx.fma_probe(0, sink)
