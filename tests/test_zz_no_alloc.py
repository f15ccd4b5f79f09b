"""The allocation-free per-matrix quantizer (qnn_quantize_matrix_static) against qnn_quantize.

Some callers cannot let a library allocate device memory: they run with a fixed, pre-reserved
memory budget, own all device memory through their own allocator, or cannot afford the
device-wide synchronization of cudaMalloc/cudaFree in a latency-critical stream. This entry
point quantizes a whole matrix as one unit using only a static device array inside the library.
The test calls it through the C ABI twice in a row (the shared scratch keeps the previous call's
contents) and checks codes, parameters and code sums bit-exact against the allocating entry
point. It lives in its own file, collected last, and passes alone or after the other tests.
"""
import ctypes as C

import numpy as np
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


def _static_quantize(qnn, x):
    rows, cols = x.shape
    codes = torch.empty((rows, cols), dtype=torch.uint8, device="cuda")
    params = torch.zeros((1, 4), dtype=torch.int32, device="cuda")
    sums = torch.empty(rows, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = qnn.lib().qnn_quantize_matrix_static(C.c_void_p(x.data_ptr()), rows, cols, x.stride(0),
                                              C.c_void_p(codes.data_ptr()), cols, C.c_void_p(params.data_ptr()),
                                              C.c_void_p(sums.data_ptr()), C.c_void_p(status.data_ptr()),
                                              C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == qnn.QNN_OK
    torch.cuda.synchronize()
    return codes, params, sums, int(status.item())


@pytest.mark.parametrize("rows,cols", [(1, 1), (37, 500), (4096, 512), (20000, 40)])
def test_static_matches_allocating_quantizer_twice(qnn, rows, cols):
    for call in range(2):
        g = np.random.Generator(np.random.PCG64(1000 * rows + cols + call))
        x = (g.normal(0.1 * (call + 1), 1.0 + call, (rows, cols))).astype(np.float32)
        xg = torch.from_numpy(x).cuda()
        codes, params, sums, status = _static_quantize(qnn, xg)
        assert status == 0
        c_ref, p_ref, s_ref = qnn.qnn_quantize(xg, qnn.PER_MATRIX)
        assert torch.equal(codes, c_ref)
        assert torch.equal(params, p_ref)
        assert torch.equal(sums, s_ref)


def test_static_rejects_too_many_rows_and_flags_nonfinite(qnn):
    big = torch.zeros((524289, 1), dtype=torch.float32, device="cuda")
    st = qnn.lib().qnn_quantize_matrix_static(C.c_void_p(big.data_ptr()), big.shape[0], 1, 1, None, 1, None, None,
                                              None, None)
    assert st == qnn.QNN_ERR_INVALID_ARG
    x = torch.ones((8, 16), dtype=torch.float32, device="cuda")
    x[3, 5] = float("nan")
    _, _, _, status = _static_quantize(qnn, x)
    assert status == qnn.QNN_ERR_NONFINITE
