// lstm_model.h — the device-side representation of a quantized LSTM model (internal).
#pragma once

#include <cstdint>
#include <functional>
#include <vector>

#include "qnn_host.h"

struct __half;

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

struct TcLayer {  // fp16 centered weight copies for the tensor-core recurrence (lstm_tc.cu)
    __half *wh16 = nullptr;  // [4 * round_up(H, 8)][kh]: gate rows interleaved in 8-cell groups
    __half *wp16 = nullptr;  // [P][kp] (P > 0)
    __half *wx16 = nullptr;  // [4 * round_up(H, 8)][kx], interleaved like wh16 (kx <= 1024)
    void *colc = nullptr;    // with wx16: [12][H] column constants of the gate kernel (bias, Wx and Wh
                             // row code sums, gate-major; see TcLstmInput)
    int64_t kh = 0, kp = 0, kx = 0;
};

// The layer input of a recurrence whose input product is fused into the gate kernel: in [B*T][kin]
// fp32 (row b T + t), and workspace for its centered fp16 codes x16 [T*B][round_up(kin, 64)], row
// units prm [T*B] and code sums rs [T*B], time-major (row t B + b: one step's rows are contiguous).
struct TcFusedInput {
    const float *in = nullptr;
    int64_t kin = 0;
    __half *x16 = nullptr;
    qnn_qparams *prm = nullptr;
    int32_t *rs = nullptr;
};

}  // namespace qnn

struct qnn_lstm_model {
    qnn_lstm_desc d{};
    int64_t L = 0, I = 0, H = 0, P = 0, C = 0, R = 0;  // I: features per network input
    // frame stacking (Sec. 4 frontend): I = frame_dim * stack; one input every stack_stride frames
    int64_t frame_dim = 0, stack = 1, stack_stride = 1;
    int64_t S = 1;  // quantization units per weight matrix (equal row blocks, Sec. 3.1 granularity)
    void *fws = nullptr;  // frontend workspace: staged host frames and the stacked inputs
    size_t fws_bytes = 0;
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
    // fp16 weight copies of the tensor-core recurrence (made on first use)
    void *tcw = nullptr;
    // streams of layers 1 .. L - 1 and events of the layer wavefront (made on first use)
    std::vector<cudaStream_t> wave_st;
    std::vector<cudaEvent_t> wave_ev;
    // the output layer's stream, the stream of its copies to the host and their events when it runs
    // beside the recurrence (made on first use): [0] a chunk of the top layer done, [1] output stream
    // joined, [2, 3] posteriors staged in buffer 0 / 1, [4, 5] buffer 0 / 1 copied out, [6] copy
    // stream joined
    cudaStream_t out_st = nullptr, cp_st = nullptr;
    cudaEvent_t out_ev[7] = {};
    // the 8-bit output layer's Wo as centered fp16 [C][round_up(R, 64)] (in tcw)
    __half *wo16 = nullptr;
    std::vector<qnn::TcLayer> tc_layers;
    // host mirror of the unit parameters (filled at creation)
    std::vector<qnn_qparams> host_params;
};

namespace qnn {
// Runs qnn_lstm_forward on the batch-of-few persistent path (lstm_small.cu) if the model and
// batch qualify; *used tells whether it ran (false: the caller takes the layer-by-layer path).
// Arguments as for qnn_lstm_forward_logits (logits nullable).
qnn_status small_path_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *logits,
                              float *h_state, float *c_state, float *h_all, cudaStream_t st, bool *used);
// Streaming with the batch-of-few kernel (stream.cu): one launch serves T frames that the host
// supplies while it runs. Buffers: xs [B][T][I] tagged input rows (host-mapped), out [B][T][C]
// posteriors (or [B][T][R] top-layer outputs without an output layer; host-mapped), done
// [T][writer blocks] frame flags (host-mapped), hx [L][B][T][R] and smx [B][T][nout][2] tagged
// device words (zeroed once; tags are launch epochs, never 0), state in h0/c0, out to h_fin/c_fin.
struct SmallStreamArgs {
    const unsigned long long *xs = nullptr;
    float *out = nullptr;
    unsigned *done = nullptr;
    unsigned long long *hx = nullptr, *smx = nullptr;
    const float *h0 = nullptr, *c0 = nullptr;
    float *h_fin = nullptr, *c_fin = nullptr;
    int *status = nullptr, *abort_flag = nullptr;
    unsigned epoch = 0;
    int64_t B = 0, T = 0;
    unsigned long long wait_ns = 0;
};
// Whether model m streams at batch B on that kernel (QNN_ERR_INVALID_ARG: shape not supported;
// QNN_ERR_NO_COOP: its clusters cannot all be resident), the number of blocks that flag each frame,
// and the number of output blocks.
qnn_status small_stream_plan(const qnn_lstm_model *m, int64_t B, int *writer_blocks, int *nout);
qnn_status small_stream_launch(const qnn_lstm_model *m, const SmallStreamArgs &s, cudaStream_t st);

// Which forward path to take, from the QNN_LSTM_PATH environment variable: "layerwise" (the
// persistent integer-MMA recurrence), "tc" (the tensor-core recurrence), "small" or unset/"auto"
// (small when it qualifies, else tc for batches of at least kTcMinBatch, else layerwise).
enum class PathChoice { kAuto, kLayerwise, kTc, kSmall };
PathChoice path_choice();
constexpr int64_t kTcMinBatch = 64;

// Tensor-core recurrence (lstm_tc.cu). Supported when H is a multiple of 4 and the recurrent input
// (R values) fits one exact accumulation chunk (round_up(R, 64) <= 1024).
bool tc_recurrence_supported(const qnn_lstm_model *m);
// Makes the fp16 weight copies (once per model).
qnn_status tc_prepare(qnn_lstm_model *m);
// Device workspace bytes tc_layer_recurrence needs for a batch of B.
size_t tc_work_bytes(const qnn_lstm_model *m, int64_t B);
// The T recurrent steps of layer l: px [B*T][4H] (row b*T + t) recovered input products plus bias,
// h0 [B][R], cbuf [B][H] cell state in/out, out [B][T][R] layer outputs, mbuf [B][H] (P > 0).
// With fx the step's input product is computed in the gate kernel from fx->in (px unused);
// otherwise px holds it.
qnn_status tc_layer_recurrence(const qnn_lstm_model *m, int64_t l, const float *px, const float *h0, float *cbuf,
                               float *out, float *mbuf, int64_t B, int64_t T, void *work, cudaStream_t st,
                               const TcFusedInput *fx = nullptr);
// The tensor-core recurrences of all layers as a wavefront across layers (fused input product, two
// or more layers; QNN_TC_WAVE=0 turns it off): layer l runs on streams[l], its step t after step t
// of layer l - 1 (edges[l - 1], recorded on streams[l - 1]); the kernel that quantizes a step's
// outputs for the layer's next step (the projection's finishing kernel, else the row quantizer)
// also writes them as the next layer's input codes of that step (fx.x16 / prm / rs of layer l + 1,
// time-major [B T][round_up(R, 64)]), so consecutive layers overlap. Layer 0's input is quantized at its start from fx.in. Per layer: h0 [B][R], cell state
// cbuf [B][H] in/out, mbuf [B][H], workspace of tc_work_bytes, outputs: row b of step t at
// out + t out_t + b out_b. The streams must already follow everything the buffers depend on.
struct TcStackLayer {
    const float *h0 = nullptr;
    float *cbuf = nullptr, *mbuf = nullptr;
    void *work = nullptr;
    float *out = nullptr;
    int64_t out_t = 0, out_b = 0;
    TcFusedInput fx;
};
// With top_codes the top layer's step kernel also writes its outputs' codes there (the output
// layer's input, time-major like fx.x16); after_top_step(t) is called once the top layer's step t
// is queued on its stream (streams[L - 1]).
bool tc_stack_supported(const qnn_lstm_model *m);
qnn_status tc_stack_recurrence(const qnn_lstm_model *m, const TcStackLayer *layers, int64_t B, int64_t T,
                               const cudaStream_t *streams, const cudaEvent_t *edges,
                               const TcFusedInput *top_codes = nullptr,
                               const std::function<qnn_status(int64_t)> &after_top_step = nullptr);
// Whether every layer's input product can be fused into its gate kernel (input width <= 1024; the
// environment variable QNN_TC_FUSE_X=0 turns it off), and the workspace for the layer input's codes.
bool tc_input_fused(const qnn_lstm_model *m);
size_t tc_xwork_bytes(const qnn_lstm_model *m, int64_t rows);
}  // namespace qnn
