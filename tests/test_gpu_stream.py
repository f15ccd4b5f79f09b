"""Streaming server mode (qnn_lstm_stream_*): frames pushed a few at a time to a resident kernel
give what the oracle gives on the whole sequence — the recurrence bit for bit, the posteriors
within 1e-4 absolute and 1e-5 relative (tests/parity.py) — across launch (chunk) boundaries and for 1 to 4 sequences. A stream
left without input gives up after its idle limit with QNN_ERR_TIMEOUT, flags no frame it could
not compute, and leaves the GPU usable."""
import time

import numpy as np
import pytest

import oracle
import parity
from paper_1607_04683_gb300 import inputs

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


def _wl(L, I, H, C, B, T, seed=11, w=0.5, wo=0.0):
    return inputs.LstmWorkload("stream", seed=seed, num_layers=L, input_dim=I, hidden=H, proj=0, num_classes=C,
                               batch=B, frames=T, w_range=w, forget_bias=1.0, seq_mean_range=0.3,
                               output_mode=1 if C > 0 else 0, out_w_range=wo)


def _model(qnn, wl, params):
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, 0, wl.num_classes, wl.output_mode)
    return qnn.LstmModel(d, torch.from_numpy(params).cuda())


def _run_stream(qnn, model, x, chunk, seed):
    """Pushes x [B, T, I] in random slices (at most `chunk` frames ahead of the pulls), pulling
    random amounts in between; returns the pulled outputs [B, T, out]."""
    B, T, _ = x.shape
    r = np.random.Generator(np.random.PCG64(seed))
    s = qnn.LstmStream(model, B, chunk=chunk, idle_seconds=5.0)
    out, pushed, pulled = [], 0, 0
    while pulled < T:
        room = chunk - (pushed - pulled)
        if pushed < T and room > 0:
            n = min(int(r.integers(1, 7)), T - pushed, room)
            s.push(x[:, pushed:pushed + n])
            pushed += n
        k = int(r.integers(0, pushed - pulled + 1))
        if k:
            out.append(s.pull(k))
            pulled += k
    assert s.close() == qnn.QNN_OK
    return np.concatenate(out, 1)


STREAM_CASES = [
    dict(L=2, I=7, H=9, C=11, B=1, T=37),
    dict(L=3, I=40, H=64, C=300, B=3, T=21),            # three output blocks exchange their partials
    dict(L=2, I=5, H=16, C=0, B=2, T=19),               # no output layer: the top layer's outputs
    dict(L=1, I=40, H=500, C=2000, B=1, T=14, w=0.08),  # one full cluster of 16 output blocks
    dict(L=2, I=40, H=100, C=4500, B=4, T=9, w=0.1),    # 36 output blocks: two gathering rounds
    dict(L=2, I=40, H=64, C=2000, B=2, T=11, w=0.3, wo=1.0),  # logits spread over several units
]


@pytest.mark.parametrize("cfg", STREAM_CASES)
@pytest.mark.parametrize("chunk", [8, 64])
def test_stream_matches_oracle(qnn, cfg, chunk):
    wl = _wl(**cfg)
    params, x = wl.make()
    model = _model(qnn, wl, params)
    y = _run_stream(qnn, model, x, chunk, seed=chunk + wl.frames)
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, 0, wl.num_classes, wl.output_mode)
    ref = oracle.lstm_forward(d, params, x)
    if wl.num_classes > 0:
        parity.check_posteriors(y, ref["y"])
        np.testing.assert_allclose(y.sum(-1), 1.0, atol=1e-5)
        # the same recurrence as the batch call: posteriors agree to a few ulp of the softmax
        y_fwd = model.forward(torch.from_numpy(x).cuda()).cpu().numpy()
        assert np.max(np.abs(y - y_fwd)) <= 1e-6
        assert np.array_equal(np.argmax(y, -1), np.argmax(y_fwd, -1))
    else:
        assert np.array_equal(y, ref["y"])
    assert qnn.device_status() == qnn.QNN_OK


def test_stream_benchmarked_model_frame_by_frame(qnn):
    # the 5 x 500 x 2000-class model, one frame per push and per pull, across two launches
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make()
    x = x[:, :40]
    model = _model(qnn, wl, params)
    s = qnn.LstmStream(model, 1, chunk=32, idle_seconds=5.0)
    ys = []
    for t in range(x.shape[1]):
        s.push(x[:, t:t + 1])
        ys.append(s.pull(1))
    assert s.close() == qnn.QNN_OK
    y = np.concatenate(ys, 1)
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, 0, wl.num_classes, wl.output_mode)
    ref = oracle.lstm_forward(d, params, x)
    parity.check_posteriors(y, ref["y"])


def test_stream_push_and_pull_limits(qnn):
    wl = _wl(L=1, I=4, H=8, C=3, B=2, T=10)
    params, x = wl.make()
    model = _model(qnn, wl, params)
    s = qnn.LstmStream(model, 2, chunk=4, idle_seconds=5.0)
    with pytest.raises(qnn.QnnError):
        s.push(x[:, :5])  # more than one chunk ahead of the pulls
    s.push(x[:, :3])
    with pytest.raises(qnn.QnnError):
        s.pull(4)  # more than was pushed
    assert s.pull(3).shape == (2, 3, 3)
    assert s.close() == qnn.QNN_OK
    with pytest.raises(qnn.QnnError):
        qnn.LstmStream(model, 5, chunk=4)  # more sequences than the resident kernel takes


def test_stream_idle_limit_gives_up_and_gpu_stays_usable(qnn):
    wl = _wl(L=2, I=7, H=9, C=11, B=1, T=4)
    params, x = wl.make()
    model = _model(qnn, wl, params)
    s = qnn.LstmStream(model, 1, chunk=16, idle_seconds=0.2)
    s.push(x[:, :2])
    y01 = s.pull(2)
    time.sleep(1.0)  # longer than the idle limit: the kernel's wait for frame 2 gives up
    s.push(x[:, 2:3])
    with pytest.raises(qnn.QnnError) as e:
        s.pull(1, timeout=10.0)
    assert e.value.status == qnn.QNN_ERR_TIMEOUT
    assert s.close() == qnn.QNN_ERR_TIMEOUT
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, 0, wl.num_classes, wl.output_mode)
    ref = oracle.lstm_forward(d, params, x)
    parity.check_posteriors(y01, ref["y"][:, :2])  # frames before the stall were good
    # the context is intact: a new stream and a batch call both still match the oracle
    y = _run_stream(qnn, model, x, 8, seed=3)
    parity.check_posteriors(y, ref["y"])
    assert qnn.device_status() == qnn.QNN_OK
