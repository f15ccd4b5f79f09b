// lstm_model.h — the device-side representation of a quantized LSTM model (internal).
#pragma once

#include <cstdint>
#include <vector>

#include "qnn_host.h"

namespace qnn {

struct QUnitDev {  // one quantized weight matrix (or the four gate matrices of one kind)
    uint8_t *codes = nullptr;       // [rows][ld] u8 codes, zero padded to ld (a multiple of 64)
    int32_t *sums = nullptr;        // [rows] row code sums
    qnn_qparams *params = nullptr;  // [n_units]: rows split into n_units equal blocks
    int64_t rows = 0, cols = 0, ld = 0;
    int n_units = 0;
};

struct LayerDev {
    QUnitDev wx, wh, wp;    // wx/wh: 4 gate blocks of H rows (row g*H + j); wp: P x H
    float *bias = nullptr;  // [4H]
    int64_t kin = 0;
};

}  // namespace qnn

struct qnn_lstm_model {
    qnn_lstm_desc d{};
    int64_t L = 0, I = 0, H = 0, P = 0, C = 0, R = 0;
    int device = 0;
    void *weights = nullptr;
    std::vector<qnn::LayerDev> layers;
    qnn::QUnitDev wo;
    float *wo_f = nullptr, *bo = nullptr;
    // forward workspace (layer-by-layer path)
    void *ws = nullptr;
    size_t ws_bytes = 0;
    // workspace of the batch-of-few path: epoch-tagged layer outputs and logits
    void *sws = nullptr;
    size_t sws_bytes = 0;
    uint32_t epoch = 0;
    // host mirror of the unit parameters (filled at creation)
    std::vector<qnn_qparams> host_params;
};

namespace qnn {
// Runs qnn_lstm_forward on the batch-of-few persistent path (lstm_small.cu) if the model and
// batch qualify; *used tells whether it ran (false: the caller takes the layer-by-layer path).
// Arguments as for qnn_lstm_forward.
qnn_status small_path_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *h_state,
                              float *c_state, float *h_all, cudaStream_t st, bool *used);
// Which forward path to take, from the QNN_LSTM_PATH environment variable: "layerwise", "small"
// or unset/"auto" (small when it qualifies).
enum class PathChoice { kAuto, kLayerwise, kSmall };
PathChoice path_choice();
}  // namespace qnn
