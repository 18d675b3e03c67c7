"""GPU checks of the roofline probes (auv_probe_*): the cuBLAS GEMM probe
computes the product (against torch's fp32 product within the tf32 / bf16
operand tolerance), the FFMA probe reaches a plausible fraction of the FP32
pipe's unit-count peak and no more, and bad arguments are rejected."""
import numpy as np
import pytest

from parity_util import need_gpu, to_np

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("precision,tol", [("tf32", 2e-3), ("bf16", 1e-2)])
def test_gemm_probe_computes_the_product(precision, tol):
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n = 256
    g = torch.Generator(device="cuda").manual_seed(1)
    a = torch.randn(n, n, device="cuda", generator=g)
    b = torch.randn(n, n, device="cuda", generator=g)
    c = torch.empty(n, n, device="cuda")
    aa, bb = (a, b) if precision == "tf32" else (a.to(torch.bfloat16), b.to(torch.bfloat16))
    flop = auvenv.probe_gemm(precision, aa, bb, c)
    assert flop == 2 * n ** 3
    torch.cuda.synchronize()
    # read column-major, the row-major tensors a and b hold A = a^T and B = b^T,
    # and the row-major c holds (A B)^T = b a
    ref = b.double() @ a.double()
    got = to_np(c).astype(np.float64)
    scale = np.abs(to_np(ref)).max()
    assert np.abs(got - to_np(ref)).max() <= tol * scale


def test_ffma_probe_rate_is_plausible():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    blocks, threads = sms * 8, 256
    sink = torch.zeros(blocks * threads, device="cuda")
    auvenv.probe_ffma(blocks, threads, 1000, sink)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    flop = auvenv.probe_ffma(blocks, threads, 20000, sink)
    e1.record()
    torch.cuda.synchronize()
    rate = flop / (e0.elapsed_time(e1) * 1e-3)
    peak_at_max = 2 * 128 * sms * 2.07e9     # no GB300 SM clock exceeds 2,070 MHz
    print(f"[probe] FFMA {rate / 1e12:.1f} TFLOP/s, {rate / peak_at_max:.3f} of the peak at 2,070 MHz")
    assert 0.3 * peak_at_max <= rate <= 1.02 * peak_at_max


def test_probes_reject_bad_arguments():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    sink = torch.zeros(1024, device="cuda")
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_ffma(0, 256, 10, sink)
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_tanh(4, 100, 10, sink)          # not a multiple of 32
    a = torch.zeros(24, 24, device="cuda")
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_gemm("tf32", a, a, a)           # n not a multiple of 16


def test_mma_probe_costs_grow_with_n():
    """The tcgen05 probe completes (no bounded wait gives up) and a wider
    MMA never costs fewer cycles than a narrower one."""
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    cyc = torch.zeros(4, dtype=torch.int64, device="cuda")
    for tf32 in (False, True):
        per = {}
        for n in (16, 64, 256):
            for a_tmem in (False, True):
                auvenv.probe_mma(n, a_tmem, 256, cyc, tf32=tf32)
                torch.cuda.synchronize()
                c = cyc.cpu()
                assert int((c == 0).sum()) == 0
                per[(n, a_tmem)] = float(c.double().median()) / 256
        print("[probe] cycles per MMA", "tf32" if tf32 else "bf16", per)
        for a_tmem in (False, True):
            assert per[(16, a_tmem)] <= per[(64, a_tmem)] * 1.05 <= per[(256, a_tmem)] * 1.05
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_mma(48, False, 16, cyc)            # not a supported N
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_mma(64, False, 0, cyc)             # no MMA
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_mma(64, False, 16, torch.zeros(4, dtype=torch.int64))   # host memory


def test_ex2_probe_runs():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    sink = torch.zeros(4 * 256, device="cuda")
    assert auvenv.probe_ex2(4, 256, 10, sink) == 8 * 4 * 256 * 10
    torch.cuda.synchronize()
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_ex2(4, 100, 10, sink)
    with pytest.raises(auvenv.AuvError):
        auvenv.probe_ex2(4, 256, 10, torch.zeros(4 * 256))               # host memory
