"""Failure detection on the GPU without a fault: a bounded wait that nothing
completes gives up, the kernel records the timeout in the device error word
and returns, fc_get_error reports FC_ERR_TIMEOUT (and clears it), and the
context keeps working; the same wait with the arrival made succeeds."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_17139_gb300 import build
    build.build()
    import paper_2502_17139_gb300.fastcoder as fcm
    return fcm


def test_bounded_wait_times_out_and_recovers(fc):
    assert fc.fc_get_error() == "FC_OK"
    fc.fc_selftest_wait(arrive=True)
    assert fc.fc_get_error() == "FC_OK"
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    fc.fc_selftest_wait(arrive=False, limit_cycles=2_000_000)  # ~1 ms at 2 GHz
    ev1.record()
    assert fc.fc_get_error() == "FC_ERR_TIMEOUT"
    assert ev0.elapsed_time(ev1) < 100.0  # gave up promptly
    assert fc.fc_get_error() == "FC_OK"   # read and cleared
    # the context is intact: ordinary work still runs and checks clean
    x = torch.arange(1 << 20, device="cuda", dtype=torch.float32)
    assert float(x.sum().item()) == float((1 << 20) * ((1 << 20) - 1) / 2)
    fc.fc_selftest_wait(arrive=True)
    assert fc.fc_get_error() == "FC_OK"


def test_selftest_rejects_bad_limits(fc):
    with pytest.raises(fc.FastCoderError):
        fc.fc_selftest_wait(arrive=False, limit_cycles=0)
