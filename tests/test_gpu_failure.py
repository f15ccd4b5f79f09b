"""Failure detection on the GPU without a fault: a bounded wait that nothing ends gives up, records
QNN_ERR_TIMEOUT in the device status word, and leaves the context usable."""
import time

import numpy as np
import pytest

import oracle

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
    assert q.device_status() == q.QNN_OK
    return q


def test_bounded_wait_gives_up_and_reports(qnn):
    t0 = time.perf_counter()
    qnn.selftest_wait_timeout(5_000_000)  # 5 ms
    elapsed = time.perf_counter() - t0
    assert elapsed < 2.0
    assert qnn.device_status() == qnn.QNN_ERR_TIMEOUT
    assert qnn.device_status() == qnn.QNN_OK  # reading clears it


def test_context_usable_after_a_timeout(qnn):
    qnn.selftest_wait_timeout(1_000_000)
    assert qnn.device_status() == qnn.QNN_ERR_TIMEOUT
    g = np.random.Generator(np.random.PCG64(1))
    A = g.normal(0, 1, (130, 96)).astype(np.float32)
    W = g.uniform(-0.1, 0.1, (64, 96)).astype(np.float32)
    ca, pa, ra = oracle.quantize(A, oracle.PER_ROW)
    cw, pw, cs = oracle.quantize(W, oracle.PER_MATRIX)
    ref = oracle.qmatmul(ca, pa, 1, cw, pw)
    gpu = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    Y, acc = qnn.qnn_qmatmul(gpu(ca), qnn.params_tensor(pa), 1, gpu(ra), gpu(cw), qnn.params_tensor(pw), gpu(cs),
                             want_acc=True)
    assert qnn.device_status() == qnn.QNN_OK
    assert np.array_equal(acc.cpu().numpy(), ref["acc"]) and np.array_equal(Y.cpu().numpy(), ref["y"])


def test_limit_out_of_range_is_rejected(qnn):
    for bad in (0, 999, 2_000_000_000):
        with pytest.raises(qnn.QnnError):
            qnn.selftest_wait_timeout(bad)
