// api.cu — host-side plumbing of libqnn: pointer-kind checks, the per-device status word and
// scratch buffers, and the status calls of the C ABI.
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "qnn_host.h"

namespace qnn {

namespace {

constexpr int kMaxDevices = 64;

struct DeviceState {
    void *scratch[kScratchCount] = {};
    size_t scratch_bytes[kScratchCount] = {};
    int *status = nullptr;
    int sms = 0;
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];

qnn_status current(int *dev) {
    QNN_CUDA_TRY(cudaGetDevice(dev));
    if (*dev < 0 || *dev >= kMaxDevices) return QNN_ERR_CUDA;
    return QNN_OK;
}

}  // namespace

bool is_device_ptr(const void *p) {
    if (!p) return false;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

void *host_mapped_ptr(void *p) {
    if (!p) return nullptr;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

qnn_status scratch(ScratchSlot slot, size_t bytes, void **out) {
    int dev = 0;
    QNN_TRY(current(&dev));
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceState &d = g_dev[dev];
    if (d.scratch_bytes[slot] < bytes) {
        if (d.scratch[slot]) {
            QNN_CUDA_TRY(cudaDeviceSynchronize());
            QNN_CUDA_TRY(cudaFree(d.scratch[slot]));
            d.scratch[slot] = nullptr;
            d.scratch_bytes[slot] = 0;
        }
        QNN_CUDA_TRY(cudaMalloc(&d.scratch[slot], bytes));
        QNN_CUDA_TRY(cudaMemset(d.scratch[slot], 0, bytes));
        d.scratch_bytes[slot] = bytes;
    }
    *out = d.scratch[slot];
    return QNN_OK;
}

qnn_status status_word(int **out) {
    int dev = 0;
    QNN_TRY(current(&dev));
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceState &d = g_dev[dev];
    if (!d.status) {
        QNN_CUDA_TRY(cudaMalloc(&d.status, sizeof(int)));
        QNN_CUDA_TRY(cudaMemset(d.status, 0, sizeof(int)));
    }
    *out = d.status;
    return QNN_OK;
}

int sm_count() {
    int dev = 0;
    if (current(&dev) != QNN_OK) return 1;
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceState &d = g_dev[dev];
    if (!d.sms) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) v = 1;
        d.sms = v;
    }
    return d.sms;
}

}  // namespace qnn

using namespace qnn;

extern "C" const char *qnn_status_string(qnn_status s) {
    switch (s) {
        case QNN_OK: return "QNN_OK";
        case QNN_ERR_INVALID_ARG: return "QNN_ERR_INVALID_ARG: invalid argument";
        case QNN_ERR_NONFINITE: return "QNN_ERR_NONFINITE: a quantization unit held NaN or Inf";
        case QNN_ERR_K_TOO_LARGE: return "QNN_ERR_K_TOO_LARGE: K exceeds 33025 (int32 accumulator limit)";
        case QNN_ERR_CUDA: return "QNN_ERR_CUDA: CUDA runtime error or no device";
        case QNN_ERR_TIMEOUT: return "QNN_ERR_TIMEOUT: a persistent-kernel grid wait timed out";
        case QNN_ERR_NO_COOP: return "QNN_ERR_NO_COOP: persistent grid cannot be co-resident";
        case QNN_ERR_NO_MEMORY: return "QNN_ERR_NO_MEMORY: device allocation failed";
    }
    return "unknown qnn_status";
}

extern "C" qnn_status qnn_device_status(void *stream) {
    int *w = nullptr;
    QNN_TRY(status_word(&w));
    QNN_CUDA_TRY(cudaStreamSynchronize(as_stream(stream)));
    int v = 0;
    QNN_CUDA_TRY(cudaMemcpy(&v, w, sizeof(int), cudaMemcpyDeviceToHost));
    if (v) QNN_CUDA_TRY(cudaMemset(w, 0, sizeof(int)));
    return static_cast<qnn_status>(v);
}

// ------------------------------------------------------------------------------------------------
// Kernel timing (diagnostics): CUDA events around every launch while enabled.
// ------------------------------------------------------------------------------------------------

namespace qnn {
namespace {

struct ProfPending {
    const char *name;
    cudaEvent_t a, b;
};
struct ProfAgg {
    const char *name;
    double ms;
    int64_t n;
};
std::mutex g_pmu;
bool g_prof_on = false;
std::vector<ProfPending> g_pending;
std::vector<cudaEvent_t> g_pool;
std::vector<ProfAgg> g_agg;

cudaEvent_t take_event() {
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

}  // namespace

ProfScope::ProfScope(const char *name, cudaStream_t st) : st_(st), idx_(-1) {
    std::lock_guard<std::mutex> lk(g_pmu);
    if (!g_prof_on) return;
    ProfPending p{name, take_event(), take_event()};
    if (!p.a || !p.b) return;
    cudaEventRecord(p.a, st);
    g_pending.push_back(p);
    idx_ = (int)g_pending.size() - 1;
}

ProfScope::~ProfScope() {
    if (idx_ < 0) return;
    std::lock_guard<std::mutex> lk(g_pmu);
    if (idx_ < (int)g_pending.size()) cudaEventRecord(g_pending[idx_].b, st_);
}

}  // namespace qnn

extern "C" qnn_status qnn_profile_enable(int on) {
    std::lock_guard<std::mutex> lk(g_pmu);
    g_prof_on = on != 0;
    return QNN_OK;
}

extern "C" qnn_status qnn_profile_read(int capacity, const char **names, double *total_ms, int64_t *launches,
                                       int *count) {
    std::lock_guard<std::mutex> lk(g_pmu);
    for (ProfPending &p : g_pending) {
        float ms = 0.0f;
        QNN_CUDA_TRY(cudaEventSynchronize(p.b));
        QNN_CUDA_TRY(cudaEventElapsedTime(&ms, p.a, p.b));
        bool found = false;
        for (ProfAgg &g : g_agg)
            if (g.name == p.name || std::strcmp(g.name, p.name) == 0) {
                g.ms += ms;
                g.n += 1;
                found = true;
                break;
            }
        if (!found) g_agg.push_back({p.name, (double)ms, 1});
        g_pool.push_back(p.a);
        g_pool.push_back(p.b);
    }
    g_pending.clear();
    int n = (int)g_agg.size();
    for (int i = 0; i < n && i < capacity; ++i) {
        if (names) names[i] = g_agg[i].name;
        if (total_ms) total_ms[i] = g_agg[i].ms;
        if (launches) launches[i] = g_agg[i].n;
    }
    if (count) *count = n;
    g_agg.clear();
    return QNN_OK;
}
