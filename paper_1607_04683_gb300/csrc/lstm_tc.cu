// lstm_tc.cu — the recurrence of an LSTM / LSTMP layer for large batches, each step's products on
// the sm_103a tcgen05 tensor cores (exact fp16 datapath of qgemm_tc.cu).
//
// Per step t of a layer (Sec. 3.1 applied to every gate matrix, Fig. 1):
//   1. quantize_rows_f16_kernel: every row (sequence) of the layer output h_{t-1} is one unit
//      (eq. 2); its codes are written centered (c - 128) in fp16, with the unit parameters and the
//      row code sum;
//   2. the gate product with Wh' (four gate matrices interleaved in 16-cell groups, so that one
//      tile holds all four gates of its cells) runs on the tensor cores; its epilogue applies
//      eq. (1)'s offsets and eq. (3)'s recovery, adds the batched input product px, and applies
//      the gate nonlinearities and the cell update;
//   3. with a projection, m_t is quantized the same way and multiplied with Wp' (eq. 1, eq. 3):
//      r_t is the layer output and the next step's recurrent input.
// Every step is a few kernel launches in stream order; the stream orders the steps.
#include <cfloat>
#include <cstdlib>
#include <cstring>

#include "lstm_model.h"
#include "qnn_device.cuh"
#include "tc_gemm.h"

namespace qnn {
namespace {

__host__ __device__ inline int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

constexpr int kQuantRowsPerBlock = 8;  // warp-per-row kernel

// Rows of fp32 values (row r at src + r*ld, len values) -> centered fp16 codes [rows][kp] (zero
// past len), unit parameters and code sums; one warp per row, eq. (2). Used when kp > 2048.
__global__ void __launch_bounds__(32 * kQuantRowsPerBlock)
    quantize_rows_f16_warp_kernel(const float *__restrict__ src, int64_t ld, int rows, int len, int kp,
                                  __half *__restrict__ dst, qnn_qparams *__restrict__ prm,
                                  int32_t *__restrict__ rsum, int *status) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * kQuantRowsPerBlock + (threadIdx.x >> 5);
    if (r >= rows) return;
    const float *xr = src + (int64_t)r * ld;
    float mn = FLT_MAX, mx = -FLT_MAX;
    bool bad = false;
    for (int k = lane; k < len; k += 32) {
        const float v = xr[k];
        bad |= !isfinite(v);
        mn = fminf(mn, v);
        mx = fmaxf(mx, v);
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    if (__any_sync(0xffffffffu, bad)) {
        if (lane == 0) record_status(status, QNN_ERR_NONFINITE);
        mn = 0.0f;
        mx = 0.0f;
    }
    const qnn_qparams p = params_from_range(mn, mx);
    __half *dr = dst + (int64_t)r * kp;
    int s = 0;
    for (int k8 = lane * 8; k8 < kp; k8 += 256) {
        __align__(16) __half v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int k = k8 + e;
            int c = 128;  // centered zero past len
            if (k < len) {
                c = (int)quant_code(xr[k], p.Q, p.z);
                s += c;
            }
            v[e] = __int2half_rn(c - 128);
        }
        *reinterpret_cast<uint4 *>(dr + k8) = *reinterpret_cast<const uint4 *>(v);
    }
    s = warp_sum(s);
    if (lane == 0) {
        prm[r] = p;
        rsum[r] = s;
    }
}

// The same for kp <= 2048 with more parallelism per row: a group of G threads (a power of two,
// 8 G >= kp) per row, each holding 8 consecutive values in registers, so the row is read once.
template <int G>
__global__ void __launch_bounds__(256)
    quantize_rows_f16_kernel(const float *__restrict__ src, int64_t ld, int rows, int len, int kp,
                             __half *__restrict__ dst, qnn_qparams *__restrict__ prm, int32_t *__restrict__ rsum,
                             int *status) {
    constexpr int RPB = 256 / G;                 // rows per block
    constexpr int W = G > 32 ? G / 32 : 1;       // warps per row
    __shared__ float s_mn[8], s_mx[8];
    __shared__ int s_n[8];
    grid_dependency_wait();
    grid_dependents_launch();
    const int t = threadIdx.x % G, rl = threadIdx.x / G, w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x * RPB + rl;
    const bool rv = r < rows;
    const int k0 = 8 * t;
    const float *xr = src + (int64_t)(rv ? r : 0) * ld;
    float v[8];
    float mn = FLT_MAX, mx = -FLT_MAX;
    int bad = 0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const int k = k0 + e;
        const bool in = rv && k < len;
        v[e] = in ? xr[k] : 0.0f;
        if (in) {
            bad |= !isfinite(v[e]);
            mn = fminf(mn, v[e]);
            mx = fmaxf(mx, v[e]);
        }
    }
#pragma unroll
    for (int o = (G < 32 ? G : 32) / 2; o > 0; o >>= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    if constexpr (W > 1) {
        if (lane == 0) {
            s_mn[w] = mn;
            s_mx[w] = mx;
            s_n[w] = bad;
        }
        __syncthreads();
        mn = s_mn[rl * W], mx = s_mx[rl * W], bad = s_n[rl * W];
#pragma unroll
        for (int i = 1; i < W; ++i) {
            mn = fminf(mn, s_mn[rl * W + i]);
            mx = fmaxf(mx, s_mx[rl * W + i]);
            bad |= s_n[rl * W + i];
        }
        __syncthreads();  // s_n is reused for the sums
    }
    if (bad) {
        if (t == 0 && rv) record_status(status, QNN_ERR_NONFINITE);
        mn = 0.0f;
        mx = 0.0f;
    }
    const qnn_qparams p = params_from_range(mn, mx);
    int sum = 0;
    __align__(16) __half h[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        int c = 128;  // centered zero past len
        if (k0 + e < len) {
            c = (int)quant_code(v[e], p.Q, p.z);
            sum += c;
        }
        h[e] = __int2half_rn(c - 128);
    }
    if (rv && k0 < kp) *reinterpret_cast<uint4 *>(dst + (int64_t)r * kp + k0) = *reinterpret_cast<const uint4 *>(h);
#pragma unroll
    for (int o = (G < 32 ? G : 32) / 2; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if constexpr (W > 1) {
        if (lane == 0) s_n[w] = sum;
        __syncthreads();
        sum = s_n[rl * W];
#pragma unroll
        for (int i = 1; i < W; ++i) sum += s_n[rl * W + i];
    }
    if (t == 0 && rv) {
        prm[r] = p;
        rsum[r] = sum;
    }
}

// The four Wh gate matrices (u8 codes, row g*H + j, ld bytes) -> centered fp16 rows in 8-cell
// groups: row 32*G + 8*g + jj holds gate g of cell 8*G + jj; rows of cells >= H are zero.
__global__ void interleave_gates_kernel(const uint8_t *__restrict__ codes, int64_t ld, int H, int K, int kp,
                                        __half *__restrict__ out) {
    const int64_t rows = 4 * round_up(H, 8);
    const int64_t total = rows * (kp / 8);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t n = i / (kp / 8);
        const int k0 = (int)(i % (kp / 8)) * 8;
        const int G = (int)(n / 32), g = (int)((n % 32) / 8), jj = (int)(n % 8);
        const int j = 8 * G + jj;
        __align__(16) __half v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int k = k0 + e;
            v[e] = (j < H && k < K) ? __int2half_rn((int)codes[((int64_t)g * H + j) * ld + k] - 128) : __int2half_rn(0);
        }
        *reinterpret_cast<uint4 *>(out + n * kp + k0) = *reinterpret_cast<const uint4 *>(v);
    }
}

// Launches one of the two row quantizers; with `pdl` as a programmatic dependent launch.
qnn_status launch_quantize_rows_f16(const float *src, int64_t ld, int64_t rows, int64_t len, int64_t kp, __half *dst,
                                    qnn_qparams *prm, int32_t *rsum, int *status, bool pdl, cudaStream_t st) {
    ProfScope prof("quantize_rows_f16", st);
    int g = 8;
    while (g * 8 < kp) g *= 2;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const int ir = (int)rows, il = (int)len, ik = (int)kp;
    auto grid_for = [&](int rpb) { return dim3((unsigned)((rows + rpb - 1) / rpb)); };
    cudaError_t e;
    switch (g) {
        case 8: cfg.gridDim = grid_for(32); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<8>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        case 16: cfg.gridDim = grid_for(16); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<16>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        case 32: cfg.gridDim = grid_for(8); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<32>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        case 64: cfg.gridDim = grid_for(4); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<64>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        case 128: cfg.gridDim = grid_for(2); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<128>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        case 256: cfg.gridDim = grid_for(1); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<256>, src, ld, ir, il, ik, dst, prm, rsum, status); break;
        default:
            cfg.gridDim = grid_for(kQuantRowsPerBlock);
            e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_warp_kernel, src, ld, ir, il, ik, dst, prm, rsum, status);
    }
    QNN_CUDA_TRY(e);
    return QNN_OK;
}

// Programmatic dependent launches between the recurrence's kernels (QNN_PDL=0 turns them off).
bool pdl_enabled() {
    const char *e = std::getenv("QNN_PDL");
    return !(e && std::strcmp(e, "0") == 0);
}

}  // namespace

bool tc_recurrence_supported(const qnn_lstm_model *m) {
    return m->H % 4 == 0 && (m->H / m->S) % 4 == 0 && round_up(m->R, 64) <= 1024;
}

qnn_status tc_prepare(qnn_lstm_model *m) {
    if (m->tcw) return QNN_OK;
    const int64_t H = m->H, R = m->R, P = m->P, H8 = round_up(H, 8);
    const int64_t kh = round_up(R, 64), kpj = round_up(H, 64);
    size_t bytes = 0;
    for (int64_t l = 0; l < m->L; ++l) {
        bytes += (size_t)round_up(4 * H8 * kh * 2, 256);
        if (P > 0) bytes += (size_t)round_up(P * kpj * 2, 256);
    }
    void *buf = nullptr;
    QNN_CUDA_TRY(cudaMalloc(&buf, bytes));
    char *p = reinterpret_cast<char *>(buf);
    m->tc_layers.assign(m->L, TcLayer{});
    for (int64_t l = 0; l < m->L; ++l) {
        const LayerDev &ly = m->layers[l];
        TcLayer &tl = m->tc_layers[l];
        tl.kh = kh;
        tl.wh16 = reinterpret_cast<__half *>(p);
        p += round_up(4 * H8 * kh * 2, 256);
        const int64_t tot = 4 * H8 * (kh / 8);
        interleave_gates_kernel<<<(unsigned)((tot + 255) / 256), 256>>>(ly.wh.codes, ly.wh.ld, (int)H, (int)R,
                                                                        (int)kh, tl.wh16);
        if (cudaGetLastError() != cudaSuccess) {
            cudaFree(buf);
            return QNN_ERR_CUDA;
        }
        if (P > 0) {
            tl.kp = kpj;
            tl.wp16 = reinterpret_cast<__half *>(p);
            p += round_up(P * kpj * 2, 256);
            qnn_status s = launch_center_fp16(ly.wp.codes, P, H, ly.wp.ld, tl.wp16, kpj, nullptr);
            if (s != QNN_OK) {
                cudaFree(buf);
                return s;
            }
        }
    }
    if (cudaDeviceSynchronize() != cudaSuccess) {
        cudaFree(buf);
        return QNN_ERR_CUDA;
    }
    m->tcw = buf;
    return QNN_OK;
}

size_t tc_work_bytes(const qnn_lstm_model *m, int64_t B) {
    const int64_t kh = round_up(m->R, 64), kpj = m->P > 0 ? round_up(m->H, 64) : 0;
    return (size_t)round_up(B * kh * 2, 256) + (size_t)round_up(B * kpj * 2, 256) +
           2 * (size_t)round_up(B * (int64_t)sizeof(qnn_qparams), 256) + 2 * (size_t)round_up(B * 4, 256);
}

qnn_status tc_layer_recurrence(const qnn_lstm_model *m, int64_t l, const float *px, const float *h0, float *cbuf,
                               float *out, float *mbuf, int64_t B, int64_t T, void *work, cudaStream_t st) {
    const LayerDev &ly = m->layers[l];
    const TcLayer &tl = m->tc_layers[l];
    const int64_t H = m->H, R = m->R, P = m->P, H8 = round_up(H, 8);
    const int64_t kh = tl.kh, kpj = tl.kp;
    char *w = reinterpret_cast<char *>(work);
    __half *a16 = reinterpret_cast<__half *>(w);
    w += round_up(B * kh * 2, 256);
    __half *m16 = reinterpret_cast<__half *>(w);
    w += round_up(B * kpj * 2, 256);
    qnn_qparams *prm = reinterpret_cast<qnn_qparams *>(w);
    w += round_up(B * (int64_t)sizeof(qnn_qparams), 256);
    qnn_qparams *prm_m = reinterpret_cast<qnn_qparams *>(w);
    w += round_up(B * (int64_t)sizeof(qnn_qparams), 256);
    int32_t *rs = reinterpret_cast<int32_t *>(w);
    w += round_up(B * 4, 256);
    int32_t *rs_m = reinterpret_cast<int32_t *>(w);

    int *status = nullptr;
    QNN_TRY(status_word(&status));
    TcOperands gates, proj;
    static const int gate_bn[] = {128, 64, 32};
    QNN_TRY(tc_operands(&gates, a16, B, tl.wh16, 4 * H8, kh, tc_choose_bn(B, 4 * H8, gate_bn, 3)));
    if (P > 0) QNN_TRY(tc_operands(&proj, m16, B, tl.wp16, P, kpj, tc_pick_bn(B, P, kpj)));
    // the steps' kernels chain by programmatic dependent launches (see tc_gemm.h); the first one of
    // the layer follows ordinary stream order
    gates.pdl = proj.pdl = pdl_enabled();
    for (int64_t t = 0; t < T; ++t) {
        const float *src = t == 0 ? h0 : out + (t - 1) * R;
        const int64_t ld = t == 0 ? R : T * R;
        QNN_TRY(launch_quantize_rows_f16(src, ld, B, R, kh, a16, prm, rs, status, t > 0 && gates.pdl, st));
        TcLstmOut o{px + t * 4 * H, T * 4 * H, cbuf, P > 0 ? mbuf : out + t * R, P > 0 ? H : T * R, (int)H,
                    (int)m->S, (int)(H / m->S)};
        QNN_TRY(tc_lstm_gates(gates, prm, rs, R, ly.wh.params, ly.wh.sums, o, st));
        if (P > 0) {
            QNN_TRY(launch_quantize_rows_f16(mbuf, H, B, H, kpj, m16, prm_m, rs_m, status, gates.pdl, st));
            QNN_TRY(tc_linear(proj, prm_m, 1, rs_m, H, ly.wp.params, P / m->S, ly.wp.sums, nullptr, out + t * R,
                              T * R, nullptr, st));
        }
    }
    return QNN_OK;
}

}  // namespace qnn
