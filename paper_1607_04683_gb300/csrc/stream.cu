// stream.cu — streaming server mode (qnn_lstm_stream_* in qnn.h): frame-at-a-time inference with
// a resident batch-of-few launch fed through host-mapped memory.
//
// Each launch serves `chunk` frames. The host writes a frame's input row as 64-bit words (value in
// the low half, the launch's epoch in the high half) into a host-mapped buffer; the first layer's
// loader polls until every word of the row carries the epoch, so no separate doorbell or ordering
// between the host's stores is needed. The output blocks finish the softmax in the kernel, write
// the posteriors into host-mapped memory and set one flag per block and frame to the epoch; the
// host reads a frame once all flags of the frame carry it. Buffers alternate between two sets by
// launch parity: launch k + 1 is queued (behind launch k on the session's stream) when its first
// frame is pushed, and reads the state launch k leaves in the other state buffer.
#include <atomic>
#include <chrono>
#include <cstring>

#include "lstm_model.h"
#include "qnn_host.h"

using namespace qnn;

struct qnn_lstm_stream {
    qnn_lstm_model *m = nullptr;
    int64_t B = 0, T = 0, I = 0, out_dim = 0;
    int writers = 0, nout = 0;
    unsigned long long wait_ns = 0;
    cudaStream_t st = nullptr;
    // host-mapped, by launch parity: tagged inputs [B][T][I], outputs [B][T][out_dim], flags [T][writers]
    unsigned long long *xin[2] = {nullptr, nullptr};
    float *yout[2] = {nullptr, nullptr};
    unsigned *done[2] = {nullptr, nullptr};
    int *status_h = nullptr;  // copy of the device status word after each launch
    void *host_block = nullptr;
    // device: tagged layer outputs, softmax partials, state by parity, status, abort flag
    void *dev_block = nullptr;
    unsigned long long *hx = nullptr, *smx = nullptr;
    float *h[2] = {nullptr, nullptr}, *c[2] = {nullptr, nullptr};
    int *status = nullptr, *abort_flag = nullptr;
    unsigned epoch[2] = {0, 0};
    unsigned next_epoch = 0;
    int64_t pushed = 0, pulled = 0, launched = 0;
    qnn_status failed = QNN_OK;
};

namespace {

size_t align256(size_t n) { return (n + 255) / 256 * 256; }

template <typename T>
T *device_alias(T *host) {
    void *d = nullptr;
    if (cudaHostGetDevicePointer(&d, host, 0) != cudaSuccess) return nullptr;
    return static_cast<T *>(d);
}

void release(qnn_lstm_stream *s) {
    if (s->host_block) cudaFreeHost(s->host_block);
    if (s->dev_block) cudaFree(s->dev_block);
    if (s->st) cudaStreamDestroy(s->st);
    delete s;
}

// Queues launch k (frames k T .. k T + T - 1).
qnn_status launch_chunk(qnn_lstm_stream *s) {
    const int par = (int)(s->launched & 1);
    if (s->next_epoch == 0xFFFFFFFFu) return QNN_ERR_INVALID_ARG;  // tag space of the session used up
    s->epoch[par] = ++s->next_epoch;
    QNN_CUDA_TRY(cudaMemsetAsync(s->abort_flag, 0, sizeof(int), s->st));
    SmallStreamArgs a;
    a.xs = device_alias(s->xin[par]);
    a.out = device_alias(s->yout[par]);
    a.done = device_alias(s->done[par]);
    if (!a.xs || !a.out || !a.done) return QNN_ERR_CUDA;
    a.hx = s->hx, a.smx = s->smx;
    a.h0 = s->h[par], a.c0 = s->c[par], a.h_fin = s->h[par ^ 1], a.c_fin = s->c[par ^ 1];
    a.status = s->status, a.abort_flag = s->abort_flag;
    a.epoch = s->epoch[par];
    a.B = s->B, a.T = s->T;
    a.wait_ns = s->wait_ns;
    QNN_TRY(small_stream_launch(s->m, a, s->st));
    QNN_CUDA_TRY(cudaMemcpyAsync(s->status_h, s->status, sizeof(int), cudaMemcpyDeviceToHost, s->st));
    ++s->launched;
    return QNN_OK;
}

// Writes frame g (global index) of every sequence: rows[b] points at its I values (null: zeros).
qnn_status write_frame(qnn_lstm_stream *s, int64_t g, const float *x, int64_t n, int64_t f) {
    const int64_t t = g % s->T;
    if (t == 0) QNN_TRY(launch_chunk(s));
    const int par = (int)((g / s->T) & 1);
    const unsigned long long tag = (unsigned long long)s->epoch[par] << 32;
    for (int64_t b = 0; b < s->B; ++b) {
        unsigned long long *dst = s->xin[par] + (b * s->T + t) * s->I;
        const float *src = x ? x + (b * n + f) * s->I : nullptr;
        for (int64_t i = 0; i < s->I; ++i) {
            uint32_t bits = 0;
            if (src) std::memcpy(&bits, src + i, sizeof(bits));
            __atomic_store_n(dst + i, tag | bits, __ATOMIC_RELAXED);
        }
    }
    return QNN_OK;
}

bool frame_ready(const qnn_lstm_stream *s, int par, int64_t t) {
    const unsigned *f = s->done[par] + t * s->writers;
    for (int w = 0; w < s->writers; ++w)
        if (__atomic_load_n(f + w, __ATOMIC_ACQUIRE) != s->epoch[par]) return false;
    return true;
}

}  // namespace

extern "C" qnn_status qnn_lstm_stream_open(qnn_lstm_model *m, int64_t B, int64_t chunk, double idle_seconds,
                                           qnn_lstm_stream **out) {
    if (!m || !out || B < 1 || chunk < 1 || chunk > 65536 || !(idle_seconds >= 0.001 && idle_seconds <= 3600.0))
        return QNN_ERR_INVALID_ARG;
    *out = nullptr;
    int writers = 0, nout = 0;
    QNN_TRY(small_stream_plan(m, B, &writers, &nout));
    auto *s = new qnn_lstm_stream;
    s->m = m, s->B = B, s->T = chunk, s->I = m->I;
    s->out_dim = m->C > 0 ? m->C : m->R;
    s->writers = writers, s->nout = nout;
    s->wait_ns = (unsigned long long)(idle_seconds * 1e9);
    auto fail = [&](qnn_status e) {
        release(s);
        return e;
    };
    if (cudaStreamCreateWithFlags(&s->st, cudaStreamNonBlocking) != cudaSuccess) return fail(QNN_ERR_CUDA);
    const int64_t T = chunk, L = m->L;
    const size_t bx = align256(sizeof(unsigned long long) * B * T * s->I);
    const size_t by = align256(sizeof(float) * B * T * s->out_dim);
    const size_t bd = align256(sizeof(unsigned) * T * writers);
    const size_t host_bytes = 2 * (bx + by + bd) + 256;
    if (cudaHostAlloc(&s->host_block, host_bytes, cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess) {
        cudaGetLastError();
        return fail(QNN_ERR_NO_MEMORY);
    }
    std::memset(s->host_block, 0, host_bytes);  // tags and flags 0: no epoch (epochs start at 1)
    char *hp = static_cast<char *>(s->host_block);
    for (int p = 0; p < 2; ++p) {
        s->xin[p] = reinterpret_cast<unsigned long long *>(hp), hp += bx;
        s->yout[p] = reinterpret_cast<float *>(hp), hp += by;
        s->done[p] = reinterpret_cast<unsigned *>(hp), hp += bd;
    }
    s->status_h = reinterpret_cast<int *>(hp);
    const size_t dhx = align256(sizeof(unsigned long long) * L * B * T * m->R);
    const size_t dsm = align256(sizeof(unsigned long long) * B * T * (size_t)nout * 2);
    const size_t dh = align256(sizeof(float) * L * B * m->R), dc = align256(sizeof(float) * L * B * m->H);
    const size_t dev_bytes = dhx + dsm + 2 * (dh + dc) + 512;
    if (cudaMalloc(&s->dev_block, dev_bytes) != cudaSuccess) {
        cudaGetLastError();
        return fail(QNN_ERR_NO_MEMORY);
    }
    if (cudaMemset(s->dev_block, 0, dev_bytes) != cudaSuccess) return fail(QNN_ERR_CUDA);  // zero state, no tags
    char *dp = static_cast<char *>(s->dev_block);
    s->hx = reinterpret_cast<unsigned long long *>(dp), dp += dhx;
    s->smx = reinterpret_cast<unsigned long long *>(dp), dp += dsm;
    for (int p = 0; p < 2; ++p) {
        s->h[p] = reinterpret_cast<float *>(dp), dp += dh;
        s->c[p] = reinterpret_cast<float *>(dp), dp += dc;
    }
    s->status = reinterpret_cast<int *>(dp);
    s->abort_flag = reinterpret_cast<int *>(dp + 256);
    *out = s;
    return QNN_OK;
}

extern "C" qnn_status qnn_lstm_stream_push(qnn_lstm_stream *s, const float *x, int64_t n) {
    if (!s || n < 0 || (n > 0 && (!x || is_device_ptr(x)))) return QNN_ERR_INVALID_ARG;
    if (s->failed != QNN_OK) return s->failed;
    if (s->pushed + n - s->pulled > s->T) return QNN_ERR_INVALID_ARG;
    for (int64_t f = 0; f < n; ++f) {
        const qnn_status e = write_frame(s, s->pushed + f, x, n, f);
        if (e != QNN_OK) {
            s->pushed += f;
            s->failed = e;
            return e;
        }
    }
    s->pushed += n;
    std::atomic_thread_fence(std::memory_order_release);
    return QNN_OK;
}

extern "C" qnn_status qnn_lstm_stream_pull(qnn_lstm_stream *s, float *y, int64_t n, double timeout_seconds) {
    if (!s || n < 0 || (n > 0 && (!y || is_device_ptr(y))) || !(timeout_seconds >= 0.0)) return QNN_ERR_INVALID_ARG;
    if (s->failed != QNN_OK) return s->failed;
    if (s->pulled + n > s->pushed) return QNN_ERR_INVALID_ARG;
    using clk = std::chrono::steady_clock;
    const auto deadline = clk::now() + std::chrono::duration_cast<clk::duration>(
                                           std::chrono::duration<double>(timeout_seconds));
    for (int64_t f = 0; f < n; ++f) {
        const int64_t g = s->pulled + f, t = g % s->T;
        const int par = (int)((g / s->T) & 1);
        for (int spins = 0; !frame_ready(s, par, t); ++spins) {
            if ((spins & 1023) != 1023) continue;
            const cudaError_t q = cudaStreamQuery(s->st);
            if (q == cudaSuccess) {  // every queued launch has ended
                if (frame_ready(s, par, t)) break;
                const int st = __atomic_load_n(s->status_h, __ATOMIC_ACQUIRE);
                s->failed = st != QNN_OK ? (qnn_status)st : QNN_ERR_TIMEOUT;
                return s->failed;
            }
            if (q != cudaErrorNotReady) {
                cudaGetLastError();
                s->failed = QNN_ERR_CUDA;
                return s->failed;
            }
            if (clk::now() > deadline) {
                s->failed = QNN_ERR_TIMEOUT;
                return s->failed;
            }
        }
        for (int64_t b = 0; b < s->B; ++b)
            std::memcpy(y + (b * n + f) * s->out_dim, s->yout[par] + (b * s->T + t) * s->out_dim,
                        sizeof(float) * s->out_dim);
    }
    s->pulled += n;
    return QNN_OK;
}

extern "C" qnn_status qnn_lstm_stream_close(qnn_lstm_stream *s) {
    if (!s) return QNN_ERR_INVALID_ARG;
    qnn_status result = s->failed;
    // complete the current launch with zero frames so that it ends
    while (s->launched > 0 && s->pushed < s->launched * s->T) {
        if (write_frame(s, s->pushed, nullptr, 1, 0) != QNN_OK) break;
        ++s->pushed;
    }
    std::atomic_thread_fence(std::memory_order_release);
    if (cudaStreamSynchronize(s->st) != cudaSuccess) {
        cudaGetLastError();
        result = QNN_ERR_CUDA;
    } else if (s->launched > 0 && result == QNN_OK) {
        result = (qnn_status)*s->status_h;
    }
    release(s);
    return result;
}
