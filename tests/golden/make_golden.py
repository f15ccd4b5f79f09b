"""Writes tests/golden/*.json from the oracle alone (no CUDA path is imported).

Run: python tests/golden/make_golden.py
The fixtures freeze the oracle's outputs on two tiny seeded cases so that any later change to
the oracle's arithmetic shows up as a test failure and has to be justified by the passage of the
paper it follows.
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_1607_04683_gb300 import inputs  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))


def tiny_lstm_case():
    wl = inputs.LstmWorkload("golden_lstm_2x6_c5", seed=99, num_layers=2, input_dim=4, hidden=6, proj=0,
                             num_classes=5, batch=2, frames=3, w_range=0.5, forget_bias=1.0)
    params, x = wl.make()
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
    res = oracle.lstm_forward(d, params, x)
    return {
        "cite": "Sec. 3.1 and Fig. 1 layer scheme; eq. (1)-(3); LSTM cell reading R4",
        "workload": wl.name, "seed": wl.seed, "num_layers": wl.num_layers, "input_dim": wl.input_dim,
        "hidden": wl.hidden, "num_classes": wl.num_classes, "batch": wl.batch, "frames": wl.frames,
        "w_range": wl.w_range, "forget_bias": wl.forget_bias,
        "y_hex": [float(v).hex() for v in res["y"].ravel()],
        "h_hex": [float(v).hex() for v in res["h"].ravel()],
    }


def quantizer_case():
    rng = np.random.Generator(np.random.PCG64(98))
    x = rng.normal(0.2, 1.3, (3, 11)).astype(np.float32)
    codes, p, sums = oracle.quantize(x, oracle.PER_ROW)
    return {
        "cite": "Sec. 3 Quantizing; eq. (2); readings R1-R2",
        "x_hex": [float(v).hex() for v in x.ravel()], "rows": 3, "cols": 11,
        "codes": codes.ravel().tolist(), "Q_hex": [float(v).hex() for v in p["Q"]],
        "z": p["z"].tolist(), "sums": sums.tolist(),
    }


if __name__ == "__main__":
    with open(os.path.join(HERE, "oracle_lstm_tiny.json"), "w") as f:
        json.dump(tiny_lstm_case(), f, indent=1)
    with open(os.path.join(HERE, "oracle_quantizer_rows.json"), "w") as f:
        json.dump(quantizer_case(), f, indent=1)
    print("wrote golden fixtures")
