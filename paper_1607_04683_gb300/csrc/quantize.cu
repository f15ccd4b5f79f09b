// quantize.cu — the on-the-fly activation quantizer (Sec. 3 "Quantizing", eq. 2) on sm_103a.
//
// Two passes over each unit: a range pass (exact fp32 min/max, warp shuffles; non-finite values
// flagged) and a code pass (eq. 2 with the unit's Q and z, four codes per 32-bit store, row code
// sums). Per-row units (one frame of one sequence) take one warp per row; rows of up to 1024
// values stay in the warp's registers between the passes (read once), longer ones are re-read
// from L1/L2. A per-matrix unit first reduces block partials into a small scratch array;
// the last block to finish folds them into the unit's parameters, then a second launch writes codes.
#include <cfloat>
#include <cstdlib>

#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {

namespace {

constexpr int kRowWarps = 8;  // warps (rows) per block in the per-row kernels

// Range of one row held by one warp; returns false if a value is not finite.
template <bool kVec>
__device__ __forceinline__ bool warp_row_range(const float *__restrict__ xr, int cols, float &mn, float &mx) {
    const int lane = threadIdx.x & 31;
    mn = FLT_MAX;
    mx = -FLT_MAX;
    bool bad = false;
    if (kVec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(xr);
        const int n4 = cols >> 2;
        for (int i = lane; i < n4; i += 32) {
            float4 v = __ldg(x4 + i);
            bad |= !isfinite(v.x) | !isfinite(v.y) | !isfinite(v.z) | !isfinite(v.w);
            mn = fminf(fminf(mn, v.x), fminf(v.y, fminf(v.z, v.w)));
            mx = fmaxf(fmaxf(mx, v.x), fmaxf(v.y, fmaxf(v.z, v.w)));
        }
        for (int i = (n4 << 2) + lane; i < cols; i += 32) {
            float v = __ldg(xr + i);
            bad |= !isfinite(v);
            mn = fminf(mn, v);
            mx = fmaxf(mx, v);
        }
    } else {
        for (int i = lane; i < cols; i += 32) {
            float v = __ldg(xr + i);
            bad |= !isfinite(v);
            mn = fminf(mn, v);
            mx = fmaxf(mx, v);
        }
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    return !__any_sync(0xffffffffu, bad);
}

// Codes of one row (eq. 2) and their sum, one warp.
template <bool kVec>
__device__ __forceinline__ int warp_row_codes(const float *__restrict__ xr, int cols, float Q, int z,
                                              uint8_t *__restrict__ cr) {
    const int lane = threadIdx.x & 31;
    int s = 0;
    if (kVec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(xr);
        uint32_t *c4 = reinterpret_cast<uint32_t *>(cr);
        const int n4 = cols >> 2;
        for (int i = lane; i < n4; i += 32) {
            float4 v = __ldg(x4 + i);
            uint32_t a = quant_code(v.x, Q, z), b = quant_code(v.y, Q, z), c = quant_code(v.z, Q, z),
                     d = quant_code(v.w, Q, z);
            s += (int)(a + b + c + d);
            c4[i] = a | (b << 8) | (c << 16) | (d << 24);
        }
        for (int i = (n4 << 2) + lane; i < cols; i += 32) {
            uint32_t a = quant_code(__ldg(xr + i), Q, z);
            s += (int)a;
            cr[i] = (uint8_t)a;
        }
    } else {
        for (int i = lane; i < cols; i += 32) {
            uint32_t a = quant_code(__ldg(xr + i), Q, z);
            s += (int)a;
            cr[i] = (uint8_t)a;
        }
    }
    return warp_sum(s);
}

template <bool kVec>
__global__ void __launch_bounds__(kRowWarps * 32) quantize_rows_kernel(const float *__restrict__ x, int64_t rows,
                                                                      int cols, int64_t ldx, uint8_t *__restrict__ codes,
                                                                      int64_t ldc, qnn_qparams *__restrict__ params,
                                                                      int32_t *__restrict__ sums, int *status) {
    const int64_t row = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (row >= rows) return;
    const float *xr = x + row * ldx;
    float mn, mx;
    bool ok = warp_row_range<kVec>(xr, cols, mn, mx);
    if (!ok) {
        if ((threadIdx.x & 31) == 0) record_status(status, QNN_ERR_NONFINITE);
        mn = 0.0f;
        mx = 0.0f;
    }
    qnn_qparams p = params_from_range(mn, mx);
    int s = warp_row_codes<kVec>(xr, cols, p.Q, p.z, codes + row * ldc);
    if ((threadIdx.x & 31) == 0) {
        params[row] = p;
        if (sums) sums[row] = s;
    }
}

// Per-row units of at most 1024 values (16-byte aligned input rows): the warp holds its row in
// registers, NV float4 per lane, all loads issued before any is used, so the row is read once and
// the code pass needs no second read.
template <int NV>
__global__ void __launch_bounds__(kRowWarps * 32) quantize_rows_reg_kernel(const float *__restrict__ x, int64_t rows,
                                                                          int cols, int64_t ldx,
                                                                          uint8_t *__restrict__ codes, int64_t ldc,
                                                                          qnn_qparams *__restrict__ params,
                                                                          int32_t *__restrict__ sums, int *status,
                                                                          bool pack) {
    const int64_t row = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (row >= rows) return;
    const int lane = threadIdx.x & 31;
    const float *xr = x + row * ldx;
    float4 v[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int k = 4 * (lane + 32 * i);
        if (k + 4 <= cols) {
            v[i] = __ldg(reinterpret_cast<const float4 *>(xr + k));
        } else {  // ragged end of the row
            v[i].x = k < cols ? __ldg(xr + k) : 0.0f;
            v[i].y = k + 1 < cols ? __ldg(xr + k + 1) : 0.0f;
            v[i].z = k + 2 < cols ? __ldg(xr + k + 2) : 0.0f;
            v[i].w = k + 3 < cols ? __ldg(xr + k + 3) : 0.0f;
        }
    }
    float mn = FLT_MAX, mx = -FLT_MAX;
    bool bad = false;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int k = 4 * (lane + 32 * i);
        const float e[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (k + j < cols) {
                bad |= !isfinite(e[j]);
                mn = fminf(mn, e[j]);
                mx = fmaxf(mx, e[j]);
            }
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    if (__any_sync(0xffffffffu, bad)) {
        if (lane == 0) record_status(status, QNN_ERR_NONFINITE);
        mn = 0.0f;
        mx = 0.0f;
    }
    const qnn_qparams p = params_from_range(mn, mx);
    uint8_t *cr = codes + row * ldc;
    int s = 0;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        const int k = 4 * (lane + 32 * i);
        if (k >= cols) continue;
        const uint32_t a = quant_code(v[i].x, p.Q, p.z), b = quant_code(v[i].y, p.Q, p.z),
                       c = quant_code(v[i].z, p.Q, p.z), d = quant_code(v[i].w, p.Q, p.z);
        if (pack && k + 4 <= cols) {  // 4-byte aligned code rows: one store for four codes
            s += (int)(a + b + c + d);
            *reinterpret_cast<uint32_t *>(cr + k) = a | (b << 8) | (c << 16) | (d << 24);
        } else {
            const uint32_t q4[4] = {a, b, c, d};
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (k + j < cols) {
                    s += (int)q4[j];
                    cr[k + j] = (uint8_t)q4[j];
                }
        }
    }
    s = warp_sum(s);
    if (lane == 0) {
        params[row] = p;
        if (sums) sums[row] = s;
    }
}

// Per-matrix pass 1: block partial ranges; the last block folds them into params[0].
template <bool kVec>
__global__ void __launch_bounds__(kRowWarps * 32) matrix_range_kernel(const float *__restrict__ x, int64_t rows,
                                                                     int cols, int64_t ldx, float *__restrict__ partials,
                                                                     unsigned *__restrict__ counter,
                                                                     qnn_qparams *__restrict__ params, int *status) {
    __shared__ float s_mn[kRowWarps], s_mx[kRowWarps];
    __shared__ int s_bad;
    __shared__ bool s_last;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) s_bad = 0;
    __syncthreads();
    float mn = FLT_MAX, mx = -FLT_MAX;
    for (int64_t row = (int64_t)blockIdx.x * kRowWarps + warp; row < rows; row += (int64_t)gridDim.x * kRowWarps) {
        float a, b;
        if (!warp_row_range<kVec>(x + row * ldx, cols, a, b)) {
            if (lane == 0) s_bad = 1;
        } else {
            mn = fminf(mn, a);
            mx = fmaxf(mx, b);
        }
    }
    if (lane == 0) {
        s_mn[warp] = mn;
        s_mx[warp] = mx;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < kRowWarps; ++w) {
            mn = fminf(mn, s_mn[w]);
            mx = fmaxf(mx, s_mx[w]);
        }
        if (s_bad) record_status(status, QNN_ERR_NONFINITE);
        partials[2 * blockIdx.x] = mn;
        partials[2 * blockIdx.x + 1] = mx;
        __threadfence();
        unsigned done = atomicAdd(counter, 1u);
        s_last = (done == gridDim.x - 1);
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
        if (mn > mx) {  // every value was non-finite
            mn = 0.0f;
            mx = 0.0f;
        }
        if (lane == 0) {
            params[0] = params_from_range(mn, mx);
            *counter = 0u;  // ready for the next call on this scratch
        }
    }
}

// Per-matrix pass 2: codes and row sums with the single unit's parameters.
template <bool kVec>
__global__ void __launch_bounds__(kRowWarps * 32) matrix_codes_kernel(const float *__restrict__ x, int64_t rows,
                                                                     int cols, int64_t ldx, uint8_t *__restrict__ codes,
                                                                     int64_t ldc, const qnn_qparams *__restrict__ params,
                                                                     int32_t *__restrict__ sums) {
    const int64_t row = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (row >= rows) return;
    const float Q = params[0].Q;
    const int z = params[0].z;
    int s = warp_row_codes<kVec>(x + row * ldx, cols, Q, z, codes + row * ldc);
    if ((threadIdx.x & 31) == 0 && sums) sums[row] = s;
}

inline bool vec_ok(const float *x, int64_t ldx, const uint8_t *codes, int64_t ldc) {
    return ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && (ldx % 4 == 0) &&
           ((reinterpret_cast<uintptr_t>(codes) & 3) == 0) && (ldc % 4 == 0);
}

}  // namespace

qnn_status launch_quantize_rows(const float *x, int64_t rows, int64_t cols, int64_t ldx, uint8_t *codes, int64_t ldc,
                                qnn_qparams *params, int32_t *sums, cudaStream_t st) {
    if (rows == 0) return QNN_OK;
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    dim3 grid((unsigned)((rows + kRowWarps - 1) / kRowWarps));
    ProfScope prof("quantize_rows", st);
    const int nv = (int)((cols + 127) / 128);  // float4 per lane for a register-resident row
    const bool x_ok = ((reinterpret_cast<uintptr_t>(x) & 15) == 0) && (ldx % 4 == 0);
    if (x_ok && nv <= 8) {
        const bool pack = ((reinterpret_cast<uintptr_t>(codes) & 3) == 0) && (ldc % 4 == 0);
        const int r = nv <= 1 ? 1 : nv <= 2 ? 2 : nv <= 4 ? 4 : 8;
        switch (r) {
            case 1: quantize_rows_reg_kernel<1><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status, pack); break;
            case 2: quantize_rows_reg_kernel<2><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status, pack); break;
            case 4: quantize_rows_reg_kernel<4><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status, pack); break;
            default: quantize_rows_reg_kernel<8><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status, pack); break;
        }
    } else if (vec_ok(x, ldx, codes, ldc))
        quantize_rows_kernel<true><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status);
    else
        quantize_rows_kernel<false><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums, status);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

qnn_status launch_quantize_matrix(const float *x, int64_t rows, int64_t cols, int64_t ldx, uint8_t *codes, int64_t ldc,
                                  qnn_qparams *params, int32_t *sums, float *partials, unsigned *counter,
                                  int max_blocks, cudaStream_t st) {
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    int64_t want = (rows + kRowWarps - 1) / kRowWarps;
    unsigned nb = (unsigned)(want < max_blocks ? want : max_blocks);
    const bool v = vec_ok(x, ldx, codes, ldc);
    {
    ProfScope prof("quantize_matrix_range", st);
    if (v)
        matrix_range_kernel<true><<<nb, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, partials, counter, params, status);
    else
        matrix_range_kernel<false><<<nb, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, partials, counter, params, status);
    QNN_CUDA_TRY(cudaGetLastError());
    }
    ProfScope prof("quantize_matrix_codes", st);
    dim3 grid((unsigned)want);
    if (v)
        matrix_codes_kernel<true><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums);
    else
        matrix_codes_kernel<false><<<grid, kRowWarps * 32, 0, st>>>(x, rows, (int)cols, ldx, codes, ldc, params, sums);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

}  // namespace qnn

using namespace qnn;

extern "C" qnn_status qnn_quantize(const float *x, int64_t rows, int64_t cols, int64_t ldx, int granularity,
                                   uint8_t *codes, int64_t ldc, qnn_qparams *params, int32_t *code_sums,
                                   void *stream) {
    if (rows < 0 || cols <= 0 || ldx < cols || ldc < cols || cols > INT32_MAX) return QNN_ERR_INVALID_ARG;
    if (granularity != QNN_PER_MATRIX && granularity != QNN_PER_ROW) return QNN_ERR_INVALID_ARG;
    if (rows == 0) return granularity == QNN_PER_MATRIX ? QNN_ERR_INVALID_ARG : QNN_OK;
    if (!is_device_ptr(x) || !is_device_ptr(codes) || !is_device_ptr(params) ||
        (code_sums && !is_device_ptr(code_sums)))
        return QNN_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    if (granularity == QNN_PER_ROW) return launch_quantize_rows(x, rows, cols, ldx, codes, ldc, params, code_sums, st);
    const int max_blocks = 4 * sm_count();
    void *ws = nullptr;
    QNN_TRY(scratch(kScratchReduce, 256 + sizeof(float) * 2 * (size_t)max_blocks, &ws));
    unsigned *counter = reinterpret_cast<unsigned *>(ws);
    float *partials = reinterpret_cast<float *>(reinterpret_cast<char *>(ws) + 256);
    return launch_quantize_matrix(x, rows, cols, ldx, codes, ldc, params, code_sums, partials, counter, max_blocks, st);
}
