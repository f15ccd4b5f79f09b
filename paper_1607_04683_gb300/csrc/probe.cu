// probe.cu — peak-rate microbenchmarks of the integer datapaths the library uses, so that
// throughput can be reported against the measured rate of this GPU rather than a datasheet.
//
//   kind 0: mma.sync m16n8k32 u8 x u8 -> s32 (warp-level integer tensor-core MMA)
//   kind 1: dp4a (four 8-bit products summed into a 32-bit integer, on the CUDA cores)
//
// Every warp runs eight independent accumulator chains from registers (no memory traffic in the
// loop); the result is written once so the work cannot be removed by the compiler.
#include <algorithm>

#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int kChains = 8;

__global__ void __launch_bounds__(256) mma_u8_peak_kernel(int iters, int *sink) {
    uint32_t a[4] = {0x01020304u ^ threadIdx.x, 0x05060708u, 0x090a0b0cu, 0x0d0e0f10u};
    uint32_t b0 = 0x11121314u ^ blockIdx.x, b1 = 0x15161718u;
    int acc[kChains][4] = {};
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c)
            asm volatile(
                "mma.sync.aligned.m16n8k32.row.col.s32.u8.u8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                "{%0,%1,%2,%3};\n"
                : "+r"(acc[c][0]), "+r"(acc[c][1]), "+r"(acc[c][2]), "+r"(acc[c][3])
                : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
    }
    int s = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) s += acc[c][0] + acc[c][1] + acc[c][2] + acc[c][3];
    if (s == 0x7fffffff) sink[0] = s;
}

__global__ void __launch_bounds__(256) dp4a_peak_kernel(int iters, int *sink) {
    int acc[kChains];
    const int a = 0x01020304 ^ threadIdx.x, b = 0x05060708 ^ blockIdx.x;
#pragma unroll
    for (int c = 0; c < kChains; ++c) acc[c] = c;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) acc[c] = __dp4a((unsigned)a, (unsigned)b, (unsigned)acc[c]);
    }
    int s = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) s += acc[c];
    if (s == 0x7fffffff) sink[0] = s;
}

// A wait nothing ends: one warp waits on an mbarrier that no thread arrives at, through the same
// bounded wait the tensor-core kernels use, with a short limit.
__global__ void wait_timeout_kernel(int *status, unsigned long long limit_ns, int *result) {
    __shared__ __align__(8) unsigned long long bar;
    const uint32_t b = static_cast<uint32_t>(__cvta_generic_to_shared(&bar));
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(b) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    const bool completed = mbar_wait_bounded(b, 0, status, limit_ns);
    if (threadIdx.x == 0) *result = completed ? 1 : 2;
}
}  // namespace
}  // namespace qnn

using namespace qnn;

// Measures the peak rate of an integer datapath in tera-operations per second (one multiply-add
// counts as two operations). Synchronous; allocates a 4-byte sink. kind: 0 = mma.sync u8, 1 = dp4a.
extern "C" qnn_status qnn_measure_peak(int kind, double *tops) {
    if (!tops || kind < 0 || kind > 1) return QNN_ERR_INVALID_ARG;
    int *sink = nullptr;
    QNN_CUDA_TRY(cudaMalloc(&sink, sizeof(int)));
    const int blocks = sm_count() * 4;
    const int iters = kind == 0 ? 4096 : 16384;
    cudaEvent_t e0, e1;
    QNN_CUDA_TRY(cudaEventCreate(&e0));
    QNN_CUDA_TRY(cudaEventCreate(&e1));
    double best = 0.0;
    for (int rep = 0; rep < 4; ++rep) {
        QNN_CUDA_TRY(cudaEventRecord(e0));
        if (kind == 0)
            mma_u8_peak_kernel<<<blocks, 256>>>(iters, sink);
        else
            dp4a_peak_kernel<<<blocks, 256>>>(iters, sink);
        QNN_CUDA_TRY(cudaEventRecord(e1));
        QNN_CUDA_TRY(cudaEventSynchronize(e1));
        float ms = 0.0f;
        QNN_CUDA_TRY(cudaEventElapsedTime(&ms, e0, e1));
        const double warps = (double)blocks * 8.0;
        const double ops = kind == 0 ? warps * iters * kChains * (2.0 * 16 * 8 * 32)
                                     : (double)blocks * 256.0 * iters * kChains * 8.0;
        const double r = ops / (ms * 1e-3) / 1e12;
        if (rep > 0 && r > best) best = r;
    }
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    cudaFree(sink);
    *tops = best;
    return QNN_OK;
}

namespace qnn {
namespace {
__global__ void s64_to_f32_kernel(const int64_t *__restrict__ in, float *__restrict__ out, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = s64_to_f32_rn(in[i]);
}

__device__ __forceinline__ bool bits_differ(float a, float b) { return __float_as_uint(a) != __float_as_uint(b); }

// Pairs (in[2i], in[2i+1]) through the paired-instruction functions and the scalar ones: counts
// the pairs where any of E, sigma, tanh, the cell update and the reciprocal-based quotient differ.
__global__ void pair_functions_kernel(const float *__restrict__ in, int64_t npairs, unsigned long long *mismatches) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < npairs; i += (int64_t)gridDim.x * blockDim.x) {
        const float2 x = make_float2(in[2 * i], in[2 * i + 1]);
        bool bad = false;
        const float2 e = pexp2(x), sg = psigmoid2(x), th = ptanh2(x);
        bad |= bits_differ(e.x, pexp(x.x)) || bits_differ(e.y, pexp(x.y));
        bad |= bits_differ(sg.x, psigmoid(x.x)) || bits_differ(sg.y, psigmoid(x.y));
        bad |= bits_differ(th.x, ptanh(x.x)) || bits_differ(th.y, ptanh(x.y));
        // a cell with gates built from both values, and its scalar twins
        const float qx = __fmul_rn(0.25f, x.x), qy = __fmul_rn(0.5f, x.y);
        float c0 = __fmul_rn(x.x, 0.37f), c1 = __fmul_rn(x.y, -0.51f);
        float2 c = make_float2(c0, c1);
        const float2 m = lstm_cell2(x, make_float2(x.y, x.x), make_float2(-x.x, qy), make_float2(qx, x.y), c);
        float m0, m1;
        lstm_cell(x.x, x.y, -x.x, qx, c0, m0);
        lstm_cell(x.y, x.x, qy, x.y, c1, m1);
        bad |= bits_differ(m.x, m0) || bits_differ(m.y, m1) || bits_differ(c.x, c0) || bits_differ(c.y, c1);
        // the recovery's quotient: integer numerators (converted from int, as the kernel's exact sums
        // are, so never -0) over a divisor from its correctly rounded reciprocal
        const float d = __fadd_rn(__fmul_rn(fabsf(x.x), 977.0f), 0.75f);
        const float2 v = make_float2(__int2float_rn(__float2int_rn(__fmul_rn(x.y, 1.0e6f))),
                                     __int2float_rn(__float2int_rn(__fmul_rn(x.x, 3.0e5f))));
        const float2 q = div_by_recip2(v, d, __frcp_rn(d));
        bad |= bits_differ(q.x, __fdiv_rn(v.x, d)) || bits_differ(q.y, __fdiv_rn(v.y, d));
        if (bad) atomicAdd(mismatches, 1ull);
    }
}
}  // namespace
}  // namespace qnn

extern "C" qnn_status qnn_selftest_s64_to_f32(const int64_t *in, float *out, int64_t n, void *stream) {
    if (n < 0) return QNN_ERR_INVALID_ARG;
    if (n == 0) return QNN_OK;
    if (!in || !out || !qnn::is_device_ptr(in) || !qnn::is_device_ptr(out)) return QNN_ERR_INVALID_ARG;
    const unsigned blocks = (unsigned)std::min<int64_t>((n + 255) / 256, 4096);
    qnn::s64_to_f32_kernel<<<blocks, 256, 0, qnn::as_stream(stream)>>>(in, out, n);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

extern "C" qnn_status qnn_selftest_pair_functions(const float *in, int64_t npairs, unsigned long long *mismatches,
                                                   void *stream) {
    if (npairs < 0 || !mismatches || !qnn::is_device_ptr(mismatches)) return QNN_ERR_INVALID_ARG;
    cudaStream_t st = qnn::as_stream(stream);
    QNN_CUDA_TRY(cudaMemsetAsync(mismatches, 0, sizeof(unsigned long long), st));
    if (npairs == 0) return QNN_OK;
    if (!in || !qnn::is_device_ptr(in)) return QNN_ERR_INVALID_ARG;
    const unsigned blocks = (unsigned)std::min<int64_t>((npairs + 255) / 256, 4096);
    qnn::pair_functions_kernel<<<blocks, 256, 0, st>>>(in, npairs, mismatches);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

extern "C" qnn_status qnn_selftest_wait_timeout(int64_t limit_ns, void *stream) {
    if (limit_ns < 1000 || limit_ns > 1000000000) return QNN_ERR_INVALID_ARG;
    int *status = nullptr, *result = nullptr;
    QNN_TRY(qnn::status_word(&status));
    void *scratch = nullptr;
    QNN_TRY(qnn::scratch(qnn::kScratchReduce, 256, &scratch));
    result = reinterpret_cast<int *>(scratch);
    cudaStream_t st = qnn::as_stream(stream);
    qnn::wait_timeout_kernel<<<1, 32, 0, st>>>(status, (unsigned long long)limit_ns, result);
    QNN_CUDA_TRY(cudaGetLastError());
    int r = 0;
    QNN_CUDA_TRY(cudaMemcpyAsync(&r, result, sizeof(int), cudaMemcpyDeviceToHost, st));
    QNN_CUDA_TRY(cudaStreamSynchronize(st));
    return r == 2 ? QNN_OK : QNN_ERR_CUDA;  // 2: the wait gave up, as it must
}
