/*
 * qnn.h — C ABI of libqnn: 8-bit quantized LSTM acoustic-model inference on one GB300 (sm_103a).
 *
 * The method is the one of Alvarez, Prabhavalkar and Bakhtin, "On the efficient representation
 * and execution of deep acoustic models" (INTERSPEECH 2016):
 *   - a uniform linear quantizer to 8 bits, S = 255, Q = S / (Vmax - Vmin), with the offset
 *     rounded consistently: V' = round(Q V) - round(Q Vmin)          (Sec. 3, eq. 2);
 *   - products of independently quantized matrices in 8-bit integers with 32-bit accumulators,
 *     recovered as (V_a'' V_b'') / (Q_a Q_b), V'' = V' + round(Q Vmin)  (Sec. 3.1, eq. 1, eq. 3);
 *   - layers that take fp32 in and give fp32 out: inputs quantized on the fly, weights offline,
 *     recovered products plus bias through the activation function (Sec. 3.1, Fig. 1);
 *   - one quantization unit per weight matrix, e.g. per LSTM gate (Sec. 3.1, last paragraph).
 *
 * Conventions for every call:
 *   - Matrices are row-major with an explicit leading dimension in elements.
 *   - Unless a call says otherwise, pointers are DEVICE pointers on the current CUDA device, and
 *     the caller owns them. A host pointer where a device pointer is required is rejected with
 *     QNN_ERR_INVALID_ARG.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream). Calls are asynchronous on it:
 *     argument errors are returned at once; errors found by the GPU (non-finite inputs, a
 *     persistent-kernel wait that timed out) are recorded in a device status word and returned
 *     by qnn_device_status().
 *   - There is no CPU fallback: without a usable CUDA device every compute call returns
 *     QNN_ERR_CUDA.
 */
#ifndef QNN_H
#define QNN_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    QNN_OK = 0,
    QNN_ERR_INVALID_ARG = 1,  /* bad size, stride, pointer kind or enum value */
    QNN_ERR_NONFINITE = 2,    /* a quantization unit held NaN or +-Inf (no range exists, Sec. 3) */
    QNN_ERR_K_TOO_LARGE = 3,  /* K > 33025: K * 255^2 would overflow the 32-bit accumulator */
    QNN_ERR_CUDA = 4,         /* a CUDA runtime call failed, or no device */
    QNN_ERR_TIMEOUT = 5,      /* a grid-wide wait in a persistent kernel gave up (bounded spin) */
    QNN_ERR_NO_COOP = 6,      /* the persistent grid cannot be co-resident on this device */
    QNN_ERR_NO_MEMORY = 7,    /* device allocation failed */
} qnn_status;

typedef enum { QNN_PER_MATRIX = 0, QNN_PER_ROW = 1 } qnn_granularity;

/* Output layer of an LSTM model: none (the top layer's outputs are returned), 8-bit
 * ("quant-all" of Sec. 5), or float ("quant" of Sec. 5: all layers but the softmax quantized). */
typedef enum { QNN_OUT_NONE = 0, QNN_OUT_QUANT = 1, QNN_OUT_FLOAT = 2 } qnn_output_mode;

/* Largest reduction length for which 8-bit codes cannot overflow a 32-bit accumulator:
 * K * 255 * 255 <= 2^31 - 1. */
#define QNN_K_MAX 33025

/* Quantization parameters of one unit (16 bytes). vmin/vmax: the exact fp32 range of the unit;
 * Q: the fp32 scale S / (vmax - vmin), S = 255 (Sec. 3); z: round(Q vmin), the rounded offset of
 * eq. (2). Code of v: clamp(round(Q v) - z, 0, 255). Recovery (eq. 3): (code + z) / Q.
 * Readings where the paper is silent: Q is raised by single ulps until the range maximum reaches
 * code 255; codes are clamped to [0, 255]; a unit with vmax == vmin, or with |Q vmin| or
 * |Q vmax| >= 2^22, uses Q = 255 / max(|vmin|, |vmax|) (Q = 1 if all values are 0). That rule
 * takes the place of a range error: no call fails on a unit without a usable range (an all-zero
 * initial state, a constant row); only non-finite values are errors (QNN_ERR_NONFINITE). */
typedef struct {
    float vmin;
    float vmax;
    float Q;
    int32_t z;
} qnn_qparams;

/* Human-readable name of a status code (static string). */
const char *qnn_status_string(qnn_status s);

/* Waits for `stream`, then returns and clears the device status word of the current device:
 * QNN_OK, QNN_ERR_NONFINITE or QNN_ERR_TIMEOUT (the first error recorded since the last call), or
 * QNN_ERR_CUDA if the stream itself failed. */
qnn_status qnn_device_status(void *stream);

/*
 * qnn_quantize — Sec. 3 "Quantizing" and eq. (2): fp32 -> 8-bit codes, on the fly.
 *   x          [rows x cols] fp32, leading dimension ldx >= cols.
 *   granularity QNN_PER_MATRIX: one unit for the whole matrix (one params entry);
 *              QNN_PER_ROW: one unit per row (rows params entries).
 *   codes      [rows x cols] uint8 out, leading dimension ldc >= cols.
 *   params     out: 1 or `rows` entries.
 *   code_sums  out, nullable: [rows] int32, sum of each row's codes (used by the offset terms of
 *              eq. 1).
 * Non-finite values: the unit's codes are unspecified and QNN_ERR_NONFINITE is recorded.
 * Per-matrix quantization allocates a small library-owned scratch buffer on first use.
 */
qnn_status qnn_quantize(const float *x, int64_t rows, int64_t cols, int64_t ldx, int granularity,
                        uint8_t *codes, int64_t ldc, qnn_qparams *params, int32_t *code_sums, void *stream);

/*
 * qnn_qmatmul — eq. (1) with eq. (2)'s offsets, recovered to fp32 (Fig. 1: y = R(Mult(Q(X), W')) + B).
 *   A     [M x K] uint8 activation codes (lda >= K); pa: 1 (ga = QNN_PER_MATRIX) or M
 *         (ga = QNN_PER_ROW) params; rsA [M] int32 row code sums of A.
 *   W     [N x K] uint8 weight codes (ldw >= K): the rows split into n_blocks equal blocks
 *         (N % n_blocks == 0), block b quantized with pw[b] (e.g. one block per LSTM gate);
 *         csW [N] int32 row code sums of W.
 *   bias  [N] fp32, nullable.
 *   Y     [M x N] fp32 out (ldy >= N): Y[m,n] = S / (Qa Qw) + bias[n], with the exact integer
 *         S = sum_k (A[m,k] + za)(W[n,k] + zw) = acc + zw*rsA[m] + za*csW[n] + K*za*zw and
 *         the fp32 operations (float)S, Qa*Qw, divide, add, each rounded once.
 *   acc_out [M x N] int32 out, nullable: acc[m,n] = sum_k A[m,k] W[n,k] (the 32-bit accumulator).
 * 1 <= K <= QNN_K_MAX.
 */
qnn_status qnn_qmatmul(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA,
                       int64_t M, int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw,
                       int64_t n_blocks, const int32_t *csW, int64_t N, const float *bias, float *Y,
                       int64_t ldy, int32_t *acc_out, void *stream);

/* ---------------------------------------------------------------------------------------------
 * Quantized LSTM / LSTMP stack (Sec. 4 model family) with an optional softmax output layer.
 * ------------------------------------------------------------------------------------------- */

typedef struct {
    int32_t num_layers;  /* L >= 1 */
    int32_t input_dim;   /* I, features per frame */
    int32_t hidden;      /* H, LSTM cells per layer */
    int32_t proj;        /* P, recurrent projection units after each layer; 0 = none */
    int32_t num_classes; /* C, softmax outputs; 0 = no output layer */
    int32_t output_mode; /* qnn_output_mode; must be QNN_OUT_NONE iff num_classes == 0 */
    int32_t stack;        /* Sec. 4 frontend: frames stacked into one network input (the frame and
                             stack - 1 frames of right context; the paper uses 8); 0 or 1 = none.
                             The first layer then takes I * stack features. */
    int32_t stack_stride; /* only every stack_stride-th stacked frame is presented (the paper: 3);
                             0 or 1 = every frame */
    int32_t weight_blocks; /* Sec. 3.1 granularity: every weight matrix (each gate's Wx and Wh, Wp,
                              Wo) is quantized as this many equal blocks of rows (sub-matrices), each
                              its own unit; 0 or 1 = one unit per matrix, the paper's setting. H, P
                              and (quantized output layer) C must be multiples of it. */
} qnn_lstm_desc;

typedef struct qnn_lstm_model qnn_lstm_model;

/* Number of fp32 values in the packed parameter buffer. Layout, layer by layer, with
 * Ik = I * max(stack, 1) for the first layer and R = (P > 0 ? P : H) otherwise, gates in the order
 * [i, f, g, o]:
 *   Wx[4][H][Ik], Wh[4][H][R], b[4][H], then Wp[P][H] if P > 0;
 * after the last layer, if C > 0: Wo[C][R], bo[C]. Returns -1 on an invalid descriptor. */
int64_t qnn_lstm_param_count(const qnn_lstm_desc *d);

/* Quantizes the weights offline (Sec. 3.1: one unit per gate matrix, per projection and per
 * output matrix, or weight_blocks units per matrix) and keeps device copies in the model. `params` (host or device) is read during
 * the call only. The call is synchronous. *out receives the model (destroy with
 * qnn_lstm_model_destroy). */
qnn_status qnn_lstm_model_create(const qnn_lstm_desc *d, const float *params, qnn_lstm_model **out);

void qnn_lstm_model_destroy(qnn_lstm_model *m);

/* Copies the model's weight codes (host buffer, qnn_lstm_param_count bytes; the packed layout
 * with every bias slot zero) and the parameters of each unit in order (4 Wx, 4 Wh, Wp per layer,
 * then Wo, each matrix's blocks in row order; host buffer of at least S (9 L + 1) entries,
 * S = max(weight_blocks, 1)) and their count. Synchronous. */
qnn_status qnn_lstm_model_weights(const qnn_lstm_model *m, uint8_t *codes_host, qnn_qparams *params_host,
                                  int64_t *n_units);

/*
 * qnn_lstm_forward — inference over B independent sequences of T frames.
 *   x        [B][T][I] fp32 frames. With frame stacking (desc.stack, desc.stack_stride) the
 *            network runs on T' = ceil(T / stride) stacked inputs, formed as qnn_stack_frames does
 *            within this call (frames past the end of x repeat its last frame); every output
 *            below then has T' frames instead of T.
 *   y        [B][T][C] softmax outputs if the model has an output layer, else [B][T][R] top-layer
 *            outputs.
 *   h_state  [L][B][R], c_state [L][B][H], nullable: initial state in, final state out (a
 *            stream can therefore be processed in chunks); NULL means a zero initial state and
 *            the final state is not returned.
 *   h_all    [L][B][T][R], nullable: every layer's output at every frame (diagnostics).
 * x, y, h_state, c_state and h_all may each be host or device memory: host buffers are copied
 * to or from device memory on `stream` inside the call (pinned host memory keeps the copies
 * asynchronous). Posteriors (num_classes > 0) for a y in pinned host memory are written there
 * by the softmax kernel itself, or, when the output layer runs beside the recurrence (below),
 * staged chunk by chunk in two device buffers of the workspace and copied by the copy engines.
 * With any host buffer the results are complete once `stream` has been synchronized.
 * Activations are quantized per row (one frame of one sequence), weights per gate matrix.
 * Large batches of a multi-layer model run their layers as a wavefront: the call may place its
 * work on streams and events the model owns (one stream per layer, one for the output layer and
 * one for its copies to the host), which start after everything queued on `stream` before the
 * call, and `stream` waits for all of them before anything queued after it, so the call stays
 * ordered on `stream` as a single launch would be. The model keeps a device workspace sized for
 * the largest B*T seen; calls on one model must not overlap in time.
 */
qnn_status qnn_lstm_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *h_state,
                            float *c_state, float *h_all, void *stream);

/*
 * qnn_lstm_forward_logits — qnn_lstm_forward that also returns the output layer's values before
 * the softmax (Sec. 5: "quant-all" takes the softmax layer's product in 8 bits, "quant" in float).
 *   logits   [B][T][C] fp32, host or device memory, caller-owned, nullable (NULL: the call is
 *            qnn_lstm_forward). logits[b][t][c] is exactly the value the softmax receives: with
 *            QNN_OUT_QUANT the recovered product of the top layer's quantized outputs with the
 *            output weights, eq. (1) and eq. (3), plus the output bias (Fig. 1); with QNN_OUT_FLOAT
 *            the fp32 product plus the bias. With frame stacking T is the stacked length T'.
 * Other arguments and behaviour as for qnn_lstm_forward. QNN_ERR_INVALID_ARG if logits is given
 * for a model without an output layer (num_classes == 0). The copy is made on `stream` after the
 * output product; a host buffer is complete once the stream has been synchronized.
 */
qnn_status qnn_lstm_forward_logits(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *logits,
                                   float *h_state, float *c_state, float *h_all, void *stream);

/*
 * Streaming server mode — frame-at-a-time inference with a resident kernel (the embedded,
 * frame-by-frame setting of Sec. 1 and Sec. 3.1, where inputs are quantized on the fly as they
 * arrive). One launch of the batch-of-few dataflow kernel stays resident for `chunk` frames and
 * takes each frame as soon as the host has written it into host-mapped memory; the output blocks
 * finish the softmax in the kernel and write each frame's posteriors straight to host-mapped
 * memory, flagging the frame when it is complete. The next chunk's launch is queued when its
 * first frame is pushed, with the state (h, c) carried from the previous launch on the device,
 * so the results equal qnn_lstm_forward on the whole sequence (the recurrence bit for bit; the
 * posteriors to within the rounding of the softmax's sum order).
 *
 * qnn_lstm_stream_open — B sequences (1 <= B <= 4) of model m (no projection, H <= 512, R and I
 *   <= 512, output layer absent or quantized; the model's frame stacking is not applied: push
 *   network input rows of m's input width). chunk: frames per launch (1 .. 65536). idle_seconds
 *   (0.001 .. 3600): every wait of the kernel gives up after this long, so a stream left without
 *   input for longer ends with QNN_ERR_TIMEOUT (reopen it to continue). Allocates pinned
 *   host-mapped buffers of 2 chunk B (8 I + 4 out) bytes and device buffers on the current
 *   device, and creates its own CUDA stream. Errors: QNN_ERR_INVALID_ARG (a size or the model out
 *   of range), QNN_ERR_NO_COOP (the kernel's clusters cannot all be resident), QNN_ERR_CUDA.
 *   The model must outlive the session.
 * qnn_lstm_stream_push — appends n frames of every sequence: x is host memory [B][n][I]
 *   (sequence-major, as for qnn_lstm_forward), read during the call only. At most `chunk` frames
 *   may be pushed ahead of those pulled (QNN_ERR_INVALID_ARG otherwise, nothing pushed). Returns
 *   without waiting for the GPU.
 * qnn_lstm_stream_pull — waits (at most timeout_seconds) for the next n frames and copies them
 *   into y, host memory [B][n][C] posteriors (or [B][n][R] top-layer outputs without an output
 *   layer). n must not exceed the frames pushed and not yet pulled (QNN_ERR_INVALID_ARG).
 *   QNN_ERR_TIMEOUT if the frames are not ready in time or the kernel gave up (see idle_seconds);
 *   the session is then unusable except for qnn_lstm_stream_close.
 * qnn_lstm_stream_close — completes the current launch with zero frames (their outputs are
 *   dropped), waits for it, frees the session and returns the first error the kernel recorded
 *   (QNN_ERR_NONFINITE for a non-finite input, QNN_ERR_TIMEOUT) or QNN_OK.
 * A session's calls must not overlap in time (one host thread at a time).
 */
typedef struct qnn_lstm_stream qnn_lstm_stream;
qnn_status qnn_lstm_stream_open(qnn_lstm_model *m, int64_t B, int64_t chunk, double idle_seconds,
                                qnn_lstm_stream **out);
qnn_status qnn_lstm_stream_push(qnn_lstm_stream *s, const float *x, int64_t n);
qnn_status qnn_lstm_stream_pull(qnn_lstm_stream *s, float *y, int64_t n, double timeout_seconds);
qnn_status qnn_lstm_stream_close(qnn_lstm_stream *s);

/*
 * qnn_stack_frames — the frontend of Sec. 4: features of n consecutive frames are stacked (the frame
 * and n - 1 frames of right context) and only every stride-th stacked frame is kept.
 *   x   [B][T][I] fp32, device memory, caller-owned.
 *   out [B][T'][n I] fp32, T' = ceil(T / stride), device memory, caller-owned: out[b][t'] is frames
 *       stride t' .. stride t' + n - 1 of sequence b, concatenated; a frame past the end of the
 *       sequence is replaced by its last frame (the paper does not say).
 * QNN_ERR_INVALID_ARG for B < 0, T < 1, I < 1, n < 1, stride < 1 or non-device pointers (B > 0).
 * Asynchronous on `stream`.
 */
qnn_status qnn_stack_frames(const float *x, int64_t B, int64_t T, int64_t I, int32_t n, int32_t stride, float *out,
                            void *stream);

/*
 * qnn_quantize_matrix_static — qnn_quantize with QNN_PER_MATRIX, allocating nothing.
 * The paper has no counterpart: this is an interface for callers that cannot allocate device
 * memory inside a library call (a fixed pre-reserved memory budget, device memory owned by the
 * caller's own allocator or pool, or a latency-critical stream where the device-wide
 * synchronization of cudaMalloc/cudaFree is not acceptable). Same results as qnn_quantize with
 * QNN_PER_MATRIX (codes, params[0], code_sums) for finite inputs.
 *   x, codes, params, code_sums: as for qnn_quantize (device memory, caller-owned); params has
 *     one entry.
 *   status   device int, nullable, caller-owned: QNN_ERR_NONFINITE is written into it (if it is
 *     still 0) when the matrix holds NaN or +-Inf; the codes are then unspecified.
 *   A pointer that is not device memory of the current device (x, codes, params, and code_sums or
 *   status when given) returns QNN_ERR_INVALID_ARG before anything runs.
 * Limits: rows <= 524288 (its scratch holds one partial range per 32 rows); larger inputs return
 * QNN_ERR_INVALID_ARG before anything runs.
 * Scratch: a 128 KiB + 256 B static device array inside the library, held on every GPU that loads
 * the library until the process exits and shared by all calls. Calls that overlap in time on the
 * GPU (unordered streams) race on it; ordered calls are safe (each call clears the completion
 * counter on its stream before its kernels run). The first call on each device resolves the
 * array's device address (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture. Calls no cudaMalloc or cudaFree.
 */
qnn_status qnn_quantize_matrix_static(const float *x, int64_t rows, int64_t cols, int64_t ldx, uint8_t *codes,
                                      int64_t ldc, qnn_qparams *params, int32_t *code_sums, int *status,
                                      void *stream);

/* ---------------------------------------------------------------------------------------------
 * Kernel timing (diagnostics and benchmarks; no counterpart in the paper).
 * ------------------------------------------------------------------------------------------- */

/* While enabled, every kernel launch the library makes is bracketed by two CUDA events on the
 * launching stream (process-wide switch, off by default). */
qnn_status qnn_profile_enable(int on);

/* Waits for the recorded events, then returns per kernel name (static strings) the number of
 * launches and their summed device time in milliseconds since the last read, and resets the
 * totals. Up to `capacity` entries are written to the (nullable) host arrays; *count receives
 * the number of distinct kernels. */
qnn_status qnn_profile_read(int capacity, const char **names, double *total_ms, int64_t *launches, int *count);

/* Measures the peak rate of an integer datapath on the current device, in tera-operations per
 * second (a multiply-add counts as two operations): kind 0 = the warp-level integer tensor-core
 * MMA (mma.sync m16n8k32 u8 x u8 -> s32) the products use, kind 1 = dp4a on the CUDA cores.
 * Register-only loops on every SM; synchronous; the best of three timed runs. */
qnn_status qnn_measure_peak(int kind, double *tops);

/* Measures the latency floor of the batch-of-few recurrence (no counterpart in the paper): the
 * time per round, in microseconds, of that kernel's per-frame synchronisation skeleton with all
 * arithmetic removed, on one cluster of cluster_size (1 .. 16) blocks: product warps wait for the
 * cluster-wide exchange of the previous frame's outputs (distributed shared memory stores completing
 * on a transaction-count barrier) and hand over to the epilogue warps, which send their values to
 * every block of the cluster. A layer of that kernel cannot take less per frame. rounds: 1 ..
 * 10^6 rounds per launch; synchronous; best of three launches; QNN_ERR_NO_COOP if the cluster
 * cannot be launched, QNN_ERR_TIMEOUT if a (bounded) wait gave up. */
qnn_status qnn_measure_exchange_floor(int32_t cluster_size, int32_t rounds, double *us_per_round);

/* Diagnostic (no counterpart in the paper): out[i] = in[i] rounded to the nearest fp32 value, ties
 * to even, by the conversion the recovery of eq. (3) uses on the device for the exact int64 sums
 * S of eq. (1). in [n] int64 and out [n] float are device buffers owned by the caller; errors:
 * QNN_ERR_INVALID_ARG for n < 0 or null/host pointers with n > 0. Asynchronous on `stream`. */
qnn_status qnn_selftest_s64_to_f32(const int64_t *in, float *out, int64_t n, void *stream);

/* Diagnostic (no counterpart in the paper): the tensor-core gate kernel evaluates the pinned E,
 * sigma, tanh, the cell update and the recovery's quotient on two cells at once with paired fp32
 * instructions; this runs them and their one-value forms on the pairs (in[2i], in[2i+1]) and
 * writes into *mismatches (device, caller-owned) the number of pairs where any result differs in
 * any bit (0 is required for bit-exact parity). in [2 npairs] fp32, device memory. Errors:
 * QNN_ERR_INVALID_ARG for npairs < 0 or null/host pointers. Asynchronous on `stream`. */
qnn_status qnn_selftest_pair_functions(const float *in, int64_t npairs, unsigned long long *mismatches, void *stream);

/* Diagnostic (no counterpart in the paper): runs one warp that waits, through the bounded wait of
 * the tensor-core kernels, on a barrier nothing completes, for limit_ns (1 us .. 1 s). The wait
 * gives up and records QNN_ERR_TIMEOUT in the device status word (read it with qnn_device_status);
 * the context stays usable. Synchronous on `stream`. Returns QNN_OK when the wait gave up as
 * designed, QNN_ERR_INVALID_ARG for a limit out of range. */
qnn_status qnn_selftest_wait_timeout(int64_t limit_ns, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* QNN_H */
