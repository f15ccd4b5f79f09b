"""CPU-side checks of the boundary: the library builds for sm_103a, loads without a GPU and exports
every symbol include/qnn.h declares; host-side argument checks that never reach a kernel."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def qlib():
    from paper_1607_04683_gb300 import build, qnn
    build.build()
    return qnn.lib()


def declared_functions():
    hdr = open(os.path.join(ROOT, "include", "qnn.h")).read()
    hdr = re.sub(r"/\*.*?\*/", "", hdr, flags=re.S)
    return sorted(set(re.findall(r"\b(qnn_[a-z0-9_]+)\s*\(", hdr)))


def test_every_declared_symbol_is_exported(qlib):
    from paper_1607_04683_gb300 import qnn
    names = declared_functions()
    assert names, "no declarations found"
    for n in names:
        assert hasattr(qlib, n), n
    assert sorted(qnn.EXPORTS) == names


def test_status_strings(qlib):
    for s in range(8):
        assert qlib.qnn_status_string(s).decode().startswith("QNN_")


def test_param_count_matches_oracle_layout(qlib):
    import oracle
    from paper_1607_04683_gb300 import inputs, qnn
    for wl in inputs.LSTM_WORKLOADS.values():
        d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
        od = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
        assert qnn.qnn_lstm_param_count(d) == oracle.lstm_param_count(od) == wl.param_count()
    # frame stacking: the first layer takes input_dim * stack features
    d = qnn.lstm_desc(2, 40, 64, 16, 10, stack=8, stack_stride=3)
    assert qnn.qnn_lstm_param_count(d) == oracle.lstm_param_count(oracle.desc(2, 320, 64, 16, 10))
    assert qnn.qnn_lstm_param_count(qnn.lstm_desc(1, 40, 8, stack=-1)) == -1
    bad = qnn.lstm_desc(0, 4, 4)
    assert qnn.qnn_lstm_param_count(bad) == -1
    bad = qnn.LstmDesc(1, 4, 4, 0, 5, qnn.OUT_NONE)  # classes without an output layer mode
    assert qnn.qnn_lstm_param_count(bad) == -1


def test_argument_errors_need_no_gpu(qlib):
    from paper_1607_04683_gb300 import qnn
    # invalid sizes are rejected before any pointer or device is touched
    assert qlib.qnn_quantize(None, 4, 0, 4, 0, None, 4, None, None, None) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_quantize(None, 4, 8, 4, 0, None, 8, None, None, None) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_quantize(None, 4, 8, 8, 7, None, 8, None, None, None) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_qmatmul(None, 40000, None, 0, None, 1, 40000, None, 40000, None, 1, None, 1, None, None, 1, None,
                            None) == qnn.QNN_ERR_K_TOO_LARGE
    assert qlib.qnn_qmatmul(None, 8, None, 0, None, 1, 8, None, 8, None, 3, None, 4, None, None, 4, None,
                            None) == qnn.QNN_ERR_INVALID_ARG
    h = C.c_void_p()
    assert qlib.qnn_lstm_model_create(C.byref(qnn.lstm_desc(0, 1, 1)), None, C.byref(h)) == qnn.QNN_ERR_INVALID_ARG
    for args in ((-1, 3, 4, 8, 3), (1, 0, 4, 8, 3), (1, 3, 0, 8, 3), (1, 3, 4, 0, 3), (1, 3, 4, 8, 0)):
        assert qlib.qnn_stack_frames(None, *args, None, None) == qnn.QNN_ERR_INVALID_ARG
    # streaming session calls: null handles and out-of-range sizes
    s = C.c_void_p()
    assert qlib.qnn_lstm_stream_open(None, 1, 8, 1.0, C.byref(s)) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_lstm_stream_push(None, None, 1) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_lstm_stream_pull(None, None, 1, 1.0) == qnn.QNN_ERR_INVALID_ARG
    assert qlib.qnn_lstm_stream_close(None) == qnn.QNN_ERR_INVALID_ARG
