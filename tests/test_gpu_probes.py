"""Measurement probes on the GPU: the integer-datapath peaks and the latency floor of the
batch-of-few recurrence return plausible values and leave the status word clean."""
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qnn():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1607_04683_gb300 import build, qnn as q
    build.build()
    q.lib()
    torch.cuda.set_device(0)
    return q


@pytest.mark.parametrize("cs", [1, 4, 16])
def test_exchange_floor_is_plausible(qnn, cs):
    us = qnn.measure_exchange_floor(cs, 2000)
    assert 0.05 < us < 50.0
    assert qnn.device_status() == qnn.QNN_OK


def test_exchange_floor_grows_with_the_cluster(qnn):
    # more peers per exchange cannot make a round cheaper by much
    assert qnn.measure_exchange_floor(16, 4000) > 0.8 * qnn.measure_exchange_floor(2, 4000)


def test_exchange_floor_rejects_bad_sizes(qnn):
    for cs, rounds in ((0, 10), (17, 10), (4, 0)):
        with pytest.raises(qnn.QnnError):
            qnn.measure_exchange_floor(cs, rounds)


def test_datapath_peaks_are_plausible(qnn):
    assert 20.0 < qnn.measure_peak(0) < 2000.0  # mma.sync u8
    assert 20.0 < qnn.measure_peak(1) < 2000.0  # dp4a
