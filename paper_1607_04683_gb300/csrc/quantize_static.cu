// quantize_static.cu — an allocation-free variant of the per-matrix quantizer.
//
// Who needs it: callers that must not allocate device memory from inside a library call — code
// that runs with a fixed, pre-reserved memory budget (embedded and real-time audio front ends),
// processes whose device memory is owned by their own allocator or memory pool, and code paths
// that may not trigger cudaMalloc/cudaFree (which synchronize the device) in the middle of a
// latency-critical stream. qnn_quantize with QNN_PER_MATRIX allocates a small reduction scratch
// and the library status word on first use; this entry point never does.
//
// Its scratch is a file-scope static device array of fixed size: one (min, max) partial per block
// of 32 rows plus a completion counter. Every GPU that loads the library holds it until the
// process exits. All calls share it, so calls that overlap in time on the GPU (different streams
// without ordering between them) race and give wrong results; calls on one stream, or otherwise
// ordered, are fine. The counter is cleared by each call before its kernels run.
#include <cfloat>
#include <mutex>

#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int kStaticWarps = 8;
constexpr int kStaticRowsPerWarp = 4;
constexpr int kStaticRowsPerBlock = kStaticWarps * kStaticRowsPerWarp;  // 32
constexpr int kStaticMaxBlocks = 16384;
constexpr int64_t kStaticMaxRows = (int64_t)kStaticMaxBlocks * kStaticRowsPerBlock;  // 524288
constexpr size_t kStaticHeader = 256;                                                // counter
constexpr size_t kStaticBytes = kStaticHeader + sizeof(float) * 2 * kStaticMaxBlocks;  // 128 KiB + 256 B

static __device__ __align__(256) unsigned char g_quant_scratch[kStaticBytes];

// Address of g_quant_scratch on each device, resolved once per device with that device current.
constexpr int kMaxDev = 64;
std::mutex g_static_mu;
void *g_static_ptr[kMaxDev] = {};

__global__ void __launch_bounds__(kStaticWarps * 32) static_range_kernel(const float *__restrict__ x, int64_t rows,
                                                                        int cols, int64_t ldx, unsigned char *scratch,
                                                                        qnn_qparams *__restrict__ params,
                                                                        int *status) {
    __shared__ float s_mn[kStaticWarps], s_mx[kStaticWarps];
    __shared__ int s_bad;
    __shared__ bool s_last;
    unsigned *counter = reinterpret_cast<unsigned *>(scratch);
    float *partials = reinterpret_cast<float *>(scratch + kStaticHeader);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) s_bad = 0;
    __syncthreads();
    float mn = FLT_MAX, mx = -FLT_MAX;
    bool bad = false;
    const int64_t r0 = (int64_t)blockIdx.x * kStaticRowsPerBlock + warp * kStaticRowsPerWarp;
    for (int64_t row = r0; row < r0 + kStaticRowsPerWarp && row < rows; ++row) {
        const float *xr = x + row * ldx;
        for (int k = lane; k < cols; k += 32) {
            float v = xr[k];
            bad |= !isfinite(v);
            if (isfinite(v)) {
                mn = fminf(mn, v);
                mx = fmaxf(mx, v);
            }
        }
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    if (__any_sync(0xffffffffu, bad) && lane == 0) s_bad = 1;
    if (lane == 0) {
        s_mn[warp] = mn;
        s_mx[warp] = mx;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < kStaticWarps; ++w) {
            mn = fminf(mn, s_mn[w]);
            mx = fmaxf(mx, s_mx[w]);
        }
        if (s_bad && status) atomicCAS(status, 0, (int)QNN_ERR_NONFINITE);
        partials[2 * blockIdx.x] = mn;
        partials[2 * blockIdx.x + 1] = mx;
        __threadfence();
        s_last = atomicAdd(counter, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (warp == 0) {
        mn = FLT_MAX;
        mx = -FLT_MAX;
        for (unsigned b = lane; b < gridDim.x; b += 32) {
            mn = fminf(mn, __ldcg(partials + 2 * b));
            mx = fmaxf(mx, __ldcg(partials + 2 * b + 1));
        }
        mn = warp_min(mn);
        mx = warp_max(mx);
        if (mn > mx) {  // no finite value at all
            mn = 0.0f;
            mx = 0.0f;
        }
        if (lane == 0) params[0] = params_from_range(mn, mx);
    }
}

__global__ void __launch_bounds__(kStaticWarps * 32) static_codes_kernel(const float *__restrict__ x, int64_t rows,
                                                                        int cols, int64_t ldx,
                                                                        uint8_t *__restrict__ codes, int64_t ldc,
                                                                        const qnn_qparams *__restrict__ params,
                                                                        int32_t *__restrict__ sums) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float Q = params[0].Q;
    const int z = params[0].z;
    const int64_t r0 = (int64_t)blockIdx.x * kStaticRowsPerBlock + warp * kStaticRowsPerWarp;
    for (int64_t row = r0; row < r0 + kStaticRowsPerWarp && row < rows; ++row) {
        const float *xr = x + row * ldx;
        uint8_t *cr = codes + row * ldc;
        int s = 0;
        for (int k = lane; k < cols; k += 32) {
            uint32_t c = quant_code(xr[k], Q, z);
            cr[k] = (uint8_t)c;
            s += (int)c;
        }
        s = warp_sum(s);
        if (lane == 0 && sums) sums[row] = s;
    }
}

// Once per device: the device address of the static scratch (the host-side symbol is only a
// stand-in and must never be passed to a kernel).
qnn_status static_scratch_address(void **out) {
    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDev) return QNN_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_static_mu);
    if (!g_static_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_quant_scratch);
        if (e != cudaSuccess || !p) return QNN_ERR_CUDA;
        g_static_ptr[dev] = p;
    }
    *out = g_static_ptr[dev];
    return QNN_OK;
}

}  // namespace
}  // namespace qnn

using namespace qnn;

extern "C" qnn_status qnn_quantize_matrix_static(const float *x, int64_t rows, int64_t cols, int64_t ldx,
                                                 uint8_t *codes, int64_t ldc, qnn_qparams *params,
                                                 int32_t *code_sums, int *status, void *stream) {
    if (rows <= 0 || cols <= 0 || ldx < cols || ldc < cols || cols > INT32_MAX) return QNN_ERR_INVALID_ARG;
    if (rows > kStaticMaxRows) return QNN_ERR_INVALID_ARG;  // the static scratch holds 16384 block partials
    if (!x || !codes || !params) return QNN_ERR_INVALID_ARG;
    // every pointer must be device memory of the current device: a host pointer is rejected here
    // rather than faulting in a kernel
    if (!is_device_ptr(x) || !is_device_ptr(codes) || !is_device_ptr(params) ||
        (code_sums && !is_device_ptr(code_sums)) || (status && !is_device_ptr(status)))
        return QNN_ERR_INVALID_ARG;
    void *scratch = nullptr;
    QNN_TRY(static_scratch_address(&scratch));
    cudaStream_t st = as_stream(stream);
    const unsigned blocks = (unsigned)((rows + kStaticRowsPerBlock - 1) / kStaticRowsPerBlock);
    QNN_CUDA_TRY(cudaMemsetAsync(scratch, 0, sizeof(unsigned), st));  // completion counter starts at zero
    static_range_kernel<<<blocks, kStaticWarps * 32, 0, st>>>(x, rows, (int)cols, ldx,
                                                              reinterpret_cast<unsigned char *>(scratch), params,
                                                              status);
    QNN_CUDA_TRY(cudaGetLastError());
    static_codes_kernel<<<blocks, kStaticWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params,
                                                              code_sums);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}
