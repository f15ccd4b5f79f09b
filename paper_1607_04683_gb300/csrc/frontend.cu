// frontend.cu — the frame stacking of Sec. 4: features of n consecutive frames (the frame and n - 1
// frames of right context) form one network input, and only every stride-th stacked frame is
// presented. A pure gather: each output element is one input element (frames past the end of the
// sequence repeat its last frame).
#include <algorithm>

#include "qnn_host.h"

namespace qnn {
namespace {

// out [B][Tp][n I] from x [B][T][I]; `vec` = 4 floats per thread (I % 4 == 0, 16-byte aligned).
template <int VEC>
__global__ void stack_frames_kernel(const float *__restrict__ x, int64_t B, int64_t T, int64_t I, int n, int stride,
                                    int64_t Tp, float *__restrict__ out) {
    const int64_t row = (int64_t)n * I;                  // floats per stacked input
    const int64_t total = B * Tp * row / VEC;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t o = e * VEC;
        const int64_t r = o / row, w = o % row;          // stacked input (b, t') and position in it
        const int64_t b = r / Tp, tp = r % Tp;
        const int64_t k = w / I, i = w % I;              // which stacked frame, which feature
        const int64_t t = tp * stride + k < T - 1 ? tp * stride + k : T - 1;
        const float *src = x + (b * T + t) * I + i;
        if (VEC == 4)
            *reinterpret_cast<float4 *>(out + o) = *reinterpret_cast<const float4 *>(src);
        else
            out[o] = *src;
    }
}

}  // namespace

qnn_status launch_stack_frames(const float *x, int64_t B, int64_t T, int64_t I, int n, int stride, float *out,
                               cudaStream_t st) {
    if (B == 0) return QNN_OK;
    const int64_t Tp = (T + stride - 1) / stride;
    const bool vec = I % 4 == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(out) & 15) == 0;
    const int64_t total = B * Tp * n * I / (vec ? 4 : 1);
    const unsigned blocks = (unsigned)std::min<int64_t>((total + 255) / 256, 8 * (int64_t)sm_count());
    ProfScope prof("stack_frames", st);
    if (vec)
        stack_frames_kernel<4><<<blocks, 256, 0, st>>>(x, B, T, I, n, stride, Tp, out);
    else
        stack_frames_kernel<1><<<blocks, 256, 0, st>>>(x, B, T, I, n, stride, Tp, out);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

}  // namespace qnn

extern "C" qnn_status qnn_stack_frames(const float *x, int64_t B, int64_t T, int64_t I, int32_t n, int32_t stride,
                                       float *out, void *stream) {
    if (B < 0 || T < 1 || I < 1 || n < 1 || stride < 1) return QNN_ERR_INVALID_ARG;
    if (B == 0) return QNN_OK;
    if (!x || !out || !qnn::is_device_ptr(x) || !qnn::is_device_ptr(out)) return QNN_ERR_INVALID_ARG;
    return qnn::launch_stack_frames(x, B, T, I, n, stride, out, qnn::as_stream(stream));
}
