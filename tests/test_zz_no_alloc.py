"""The allocation-free per-matrix quantizer (qnn_quantize_matrix_static) against the oracle and
against qnn_quantize.

Some callers cannot let a library allocate device memory: they run with a fixed, pre-reserved
memory budget, own all device memory through their own allocator, or cannot afford the
device-wide synchronization of cudaMalloc/cudaFree in a latency-critical stream. This entry
point quantizes a whole matrix as one unit using only a static device array inside the library.
The test calls it through the C ABI twice in a row (the shared scratch keeps the previous call's
contents) and checks codes, parameters and code sums bit-exact against the CPU oracle and against
the allocating entry point; it also checks that a call leaves the device's free memory unchanged
and that host pointers are refused before anything runs. It lives in its own file, collected last,
and passes alone or after the other tests.
"""
import ctypes as C

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
    return q


def _call(qnn, x, codes, params, sums, status):
    rows, cols = x.shape
    return qnn.lib().qnn_quantize_matrix_static(C.c_void_p(x.data_ptr()), rows, cols, x.stride(0),
                                                C.c_void_p(codes.data_ptr()), codes.stride(0),
                                                C.c_void_p(params.data_ptr()),
                                                None if sums is None else C.c_void_p(sums.data_ptr()),
                                                None if status is None else C.c_void_p(status.data_ptr()),
                                                C.c_void_p(torch.cuda.current_stream().cuda_stream))


def _static_quantize(qnn, x):
    rows, cols = x.shape
    codes = torch.empty((rows, cols), dtype=torch.uint8, device="cuda")
    params = torch.zeros((1, 4), dtype=torch.int32, device="cuda")
    sums = torch.empty(rows, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert _call(qnn, x, codes, params, sums, status) == qnn.QNN_OK
    torch.cuda.synchronize()
    return codes, params, sums, int(status.item())


@pytest.mark.parametrize("rows,cols", [(1, 1), (37, 500), (4096, 512), (20000, 40)])
def test_static_matches_oracle_and_allocating_quantizer_twice(qnn, rows, cols):
    for call in range(2):
        g = np.random.Generator(np.random.PCG64(1000 * rows + cols + call))
        x = (g.normal(0.1 * (call + 1), 1.0 + call, (rows, cols))).astype(np.float32)
        xg = torch.from_numpy(x).cuda()
        codes, params, sums, status = _static_quantize(qnn, xg)
        assert status == 0
        c_ref, p_ref, s_ref = oracle.quantize(x, oracle.PER_MATRIX)
        assert np.array_equal(codes.cpu().numpy(), c_ref)
        assert np.array_equal(params.cpu().numpy().view(oracle.QPARAMS_DTYPE).reshape(-1), p_ref)
        assert np.array_equal(sums.cpu().numpy(), s_ref)
        c_a, p_a, s_a = qnn.qnn_quantize(xg, qnn.PER_MATRIX)
        assert torch.equal(codes, c_a) and torch.equal(params, p_a) and torch.equal(sums, s_a)


def test_static_call_allocates_no_device_memory(qnn):
    x = torch.randn((3000, 700), device="cuda")
    codes = torch.empty((3000, 700), dtype=torch.uint8, device="cuda")
    params = torch.zeros((1, 4), dtype=torch.int32, device="cuda")
    sums = torch.empty(3000, dtype=torch.int32, device="cuda")
    assert _call(qnn, x, codes, params, sums, None) == qnn.QNN_OK  # first call on the device: set-up
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        assert _call(qnn, x, codes, params, sums, None) == qnn.QNN_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_static_rejects_too_many_rows_host_pointers_and_flags_nonfinite(qnn):
    big = torch.zeros((524289, 1), dtype=torch.float32, device="cuda")
    st = qnn.lib().qnn_quantize_matrix_static(C.c_void_p(big.data_ptr()), big.shape[0], 1, 1, None, 1, None, None,
                                              None, None)
    assert st == qnn.QNN_ERR_INVALID_ARG
    xd = torch.ones((4, 8), dtype=torch.float32, device="cuda")
    cd = torch.empty((4, 8), dtype=torch.uint8, device="cuda")
    pd = torch.zeros((1, 4), dtype=torch.int32, device="cuda")
    sd = torch.empty(4, dtype=torch.int32, device="cuda")
    xh, ch, ph = xd.cpu(), cd.cpu(), pd.cpu()
    sh, sth = sd.cpu(), torch.zeros(1, dtype=torch.int32)
    stp = torch.zeros(1, dtype=torch.int32).pin_memory()
    for args in ((xh, cd, pd, sd, None), (xd, ch, pd, sd, None), (xd, cd, ph, sd, None), (xd, cd, pd, sh, None),
                 (xd, cd, pd, sd, sth), (xd, cd, pd, sd, stp)):
        assert _call(qnn, *args) == qnn.QNN_ERR_INVALID_ARG
    x = torch.ones((8, 16), dtype=torch.float32, device="cuda")
    x[3, 5] = float("nan")
    _, _, _, status = _static_quantize(qnn, x)
    assert status == qnn.QNN_ERR_NONFINITE
