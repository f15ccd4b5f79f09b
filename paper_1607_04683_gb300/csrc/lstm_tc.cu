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
#include <algorithm>
#include <cfloat>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <vector>

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
                                  int32_t *__restrict__ rsum, int *status, int tm_T, int tm_B) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * kQuantRowsPerBlock + (threadIdx.x >> 5);
    if (r >= rows) return;
    const float *xr = src + (int64_t)r * ld;
    const int ro = tm_T > 0 ? (r % tm_T) * tm_B + r / tm_T : r;  // output row (see launch_quantize_rows_f16)
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
    __half *dr = dst + (int64_t)ro * kp;
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
        prm[ro] = p;
        rsum[ro] = s;
    }
}

// Row-group quantizer shared by the kernels below: a group of G threads (a power of two) holds a
// row of len values, V (8 or 16) consecutive values per thread (v, starting at k0 = V t); writes the
// centered fp16 codes [kp] (zero past len), the unit parameters and the code sum of the row (eq. 2),
// and the same again to dst2, prm2, rsum2 (row r2) when dst2 is given.
template <int G, int V = 8>
__device__ __forceinline__ void quantize_row_group(const float (&v)[V], int len, int kp, int t, int rl, bool rv, int r,
                                                   __half *__restrict__ dst, qnn_qparams *__restrict__ prm,
                                                   int32_t *__restrict__ rsum, int *status, float *s_mn, float *s_mx,
                                                   int *s_n, __half *dst2 = nullptr, qnn_qparams *prm2 = nullptr,
                                                   int32_t *rsum2 = nullptr, int r2 = 0) {
    constexpr int W = G > 32 ? G / 32 : 1;  // warps per row
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k0 = V * t;
    float mn = FLT_MAX, mx = -FLT_MAX;
    int bad = 0;
#pragma unroll
    for (int e = 0; e < V; ++e) {
        if (rv && k0 + e < len) {
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
    __align__(16) __half h[V];
#pragma unroll
    for (int e = 0; e < V; ++e) {
        int c = 128;  // centered zero past len
        if (k0 + e < len) {
            c = (int)quant_code(v[e], p.Q, p.z);
            sum += c;
        }
        h[e] = __int2half_rn(c - 128);
    }
#pragma unroll
    for (int e8 = 0; e8 < V; e8 += 8)
        if (rv && k0 + e8 < kp) {
            *reinterpret_cast<uint4 *>(dst + (int64_t)r * kp + k0 + e8) = *reinterpret_cast<const uint4 *>(h + e8);
            if (dst2)
                *reinterpret_cast<uint4 *>(dst2 + (int64_t)r2 * kp + k0 + e8) = *reinterpret_cast<const uint4 *>(h + e8);
        }
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
        if (dst2) {
            prm2[r2] = p;
            rsum2[r2] = sum;
        }
    }
}

// A second destination of a row quantizer's codes, unit params and code sums (nullable dst).
struct RowCodes {
    __half *dst;
    qnn_qparams *prm;
    int32_t *rsum;
};

// Rows of fp32 values (row r at src + r*ld) -> centered fp16 codes for kp <= 2048: a group of G
// threads (V G >= kp) per row, each holding V consecutive values, so the row is read once; the same
// results also to d2 when d2.dst is given.
template <int G, int V = 8>
__global__ void __launch_bounds__(256)
    quantize_rows_f16_kernel(const float *__restrict__ src, int64_t ld, int rows, int len, int kp,
                             __half *__restrict__ dst, qnn_qparams *__restrict__ prm, int32_t *__restrict__ rsum,
                             int *status, int tm_T, int tm_B, const RowCodes d2) {
    constexpr int RPB = 256 / G;  // rows per block
    __shared__ float s_mn[8], s_mx[8];
    __shared__ int s_n[8];
    grid_dependency_wait();
    grid_dependents_launch();
    const int t = threadIdx.x % G, rl = threadIdx.x / G;
    const int r = blockIdx.x * RPB + rl;
    const bool rv = r < rows;
    const int k0 = V * t;
    const float *xr = src + (int64_t)(rv ? r : 0) * ld;
    float v[V];
    if (rv && k0 + V <= len && (ld % 4) == 0 && (reinterpret_cast<uintptr_t>(src) & 15) == 0) {
#pragma unroll
        for (int e4 = 0; e4 < V; e4 += 4) {
            const float4 a = *reinterpret_cast<const float4 *>(xr + k0 + e4);
            v[e4] = a.x, v[e4 + 1] = a.y, v[e4 + 2] = a.z, v[e4 + 3] = a.w;
        }
    } else {
#pragma unroll
        for (int e = 0; e < V; ++e) v[e] = (rv && k0 + e < len) ? xr[k0 + e] : 0.0f;
    }
    const int ro = tm_T > 0 ? (r % tm_T) * tm_B + r / tm_T : r;  // output row (see launch_quantize_rows_f16)
    quantize_row_group<G, V>(v, len, kp, t, rl, rv, ro, dst, prm, rsum, status, s_mn, s_mx, s_n, d2.dst, d2.prm,
                             d2.rsum, ro);
}

// Arguments of the projection's finishing kernel (one recurrent step of an LSTMP layer).
struct FinishArgs {
    const int32_t *part;       // [splits][B][ldpart] split-K partial sums of the centered product
    int splits;
    int64_t ldpart;
    const qnn_qparams *prm_m;  // [B] units of the m_t rows (the product's activations)
    const int32_t *rs_m;       // [B] their code sums
    const qnn_qparams *wp_p;   // Wp units, rows_per_unit rows each
    const int32_t *wp_sum;     // [P] Wp row code sums
    int rows_per_unit;
    int K;                     // H, the product's true reduction length
    float *out;                // r_t: row b at out + b * ldo
    int64_t ldo;
    int rows, P;
    int quantize;              // also quantize r_t for the next step
    int kp;                    // round_up(P, 64)
    __half *dst;               // next step's codes [B][kp], params and sums
    qnn_qparams *prm;
    int32_t *rsum;
    int *status;
    // nullable: the same codes, params and sums again as the next layer's input of this step
    // ([B][kp] rows of the next layer's time-major input codes)
    __half *dst2;
    qnn_qparams *prm2;
    int32_t *rsum2;
};

// Adds the split-K slices, applies eq. (1)'s offsets and eq. (3)'s recovery (the same integer
// and the same two roundings as the product kernels' epilogues) to give r_t, writes it as the
// layer output, and quantizes it as the next step's recurrent input.
template <int G>
__global__ void __launch_bounds__(256) proj_finish_kernel(const FinishArgs a) {
    constexpr int RPB = 256 / G;
    __shared__ float s_mn[8], s_mx[8];
    __shared__ int s_n[8];
    grid_dependency_wait();
    grid_dependents_launch();
    const int t = threadIdx.x % G, rl = threadIdx.x / G;
    const int r = blockIdx.x * RPB + rl;
    const bool rv = r < a.rows;
    const int k0 = 8 * t;
    float v[8];
    int za = 0, ra = 0;
    float Qa = 1.0f;
    if (rv) {
        const qnn_qparams pm = a.prm_m[r];
        za = pm.z, Qa = pm.Q, ra = a.rs_m[r];
    }
    // the exact centered sums of this thread's 8 outputs: slices added in int32 (16-byte loads when
    // the row of 8 lies inside P and the slices are 16-byte aligned)
    int Psum[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (rv && k0 + 8 <= a.P && a.ldpart % 4 == 0) {
        for (int s = 0; s < a.splits; ++s) {
            const int4 *src = reinterpret_cast<const int4 *>(a.part + ((int64_t)s * a.rows + r) * a.ldpart + k0);
            const int4 u = src[0], w = src[1];
            Psum[0] += u.x, Psum[1] += u.y, Psum[2] += u.z, Psum[3] += u.w;
            Psum[4] += w.x, Psum[5] += w.y, Psum[6] += w.z, Psum[7] += w.w;
        }
    } else if (rv) {
        for (int s = 0; s < a.splits; ++s)
#pragma unroll
            for (int e = 0; e < 8; ++e)
                if (k0 + e < a.P) Psum[e] += a.part[((int64_t)s * a.rows + r) * a.ldpart + k0 + e];
    }
    // The usual case: the 8 columns lie in one weight unit and the sums S of eq. (1) fit in 32 bits
    // (K max|a' + za| max|w' + zw| < 2^31: wrapping 32-bit arithmetic gives them exactly), so S =
    // Psum + rt + (128 + za) cs, and S / (Qa Qw) is taken from the divisor's correctly rounded
    // reciprocal (div_by_recip: the IEEE quotient while the divisor stays within 2^-60 .. 2^60).
    // Otherwise each output the general way (64-bit S, IEEE divide).
    const int u0 = k0 / a.rows_per_unit;
    bool fast = rv && k0 + 8 <= a.P && (k0 + 7) / a.rows_per_unit == u0 && (reinterpret_cast<uintptr_t>(a.wp_sum) & 15) == 0;
    qnn_qparams qw0{};
    float d = 1.0f;
    if (fast) {
        qw0 = a.wp_p[u0];
        d = __fmul_rn(Qa, qw0.Q);
        fast = (long long)a.K * max(abs(za), abs(za + 255)) * (long long)max(abs(qw0.z), abs(qw0.z + 255)) < (1LL << 31) &&
               d >= 0x1p-60f && d <= 0x1p60f;
    }
    if (fast) {
        const float rcp = __frcp_rn(d);
        const uint32_t rt = (uint32_t)(128 + qw0.z) * (uint32_t)ra + (uint32_t)a.K * (uint32_t)(za * qw0.z - 16384);
        const int4 c0 = *reinterpret_cast<const int4 *>(a.wp_sum + k0), c1 = *reinterpret_cast<const int4 *>(a.wp_sum + k0 + 4);
        const int cs[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int S = (int)((uint32_t)Psum[e] + rt + (uint32_t)(128 + za) * (uint32_t)cs[e]);
            v[e] = div_by_recip(__int2float_rn(S), d, rcp);
        }
        float *o = a.out + (int64_t)r * a.ldo + k0;
        if ((reinterpret_cast<uintptr_t>(o) & 15) == 0) {
            *reinterpret_cast<float4 *>(o) = make_float4(v[0], v[1], v[2], v[3]);
            *reinterpret_cast<float4 *>(o + 4) = make_float4(v[4], v[5], v[6], v[7]);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) o[e] = v[e];
        }
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int n = k0 + e;
            v[e] = 0.0f;
            if (rv && n < a.P) {
                const int cs = a.wp_sum[n];
                const qnn_qparams qw = a.wp_p[n / a.rows_per_unit];
                const int acc = Psum[e] + 128 * (ra + cs) - 16384 * a.K;  // raw code product
                v[e] = recover_product(offset_product(acc, za, qw.z, ra, cs, a.K), Qa, qw.Q);
                a.out[(int64_t)r * a.ldo + n] = v[e];
            }
        }
    }
    if (!a.quantize) return;
    quantize_row_group<G>(v, a.P, a.kp, t, rl, rv, r, a.dst, a.prm, a.rsum, a.status, s_mn, s_mx, s_n, a.dst2, a.prm2,
                          a.rsum2, r);
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

// Row code sums (integers below 2^24) as exact fp32 values.
__global__ void sums_to_f32_kernel(const int32_t *__restrict__ in, float *__restrict__ out, int64_t n) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = (float)in[i];
}

// Launches one of the two row quantizers; with `pdl` as a programmatic dependent launch. With
// tm_T > 0 the source rows are b tm_T + t (sequence-major, tm_B sequences) and row b tm_T + t is
// written to output row t tm_B + b (time-major), so that one step's rows of all sequences are
// contiguous for the tensor-core kernel's loads. With d2.dst the same results go there too (kp <=
// 2048).
qnn_status launch_quantize_rows_f16(const float *src, int64_t ld, int64_t rows, int64_t len, int64_t kp, __half *dst,
                                    qnn_qparams *prm, int32_t *rsum, int *status, bool pdl, cudaStream_t st,
                                    int64_t tm_T = 0, int64_t tm_B = 0, RowCodes d2 = RowCodes{nullptr, nullptr, nullptr}) {
    ProfScope prof("quantize_rows_f16", st);
    int g = 8;
    while (g * 8 < kp) g *= 2;
    if (d2.dst && g > 256) return QNN_ERR_INVALID_ARG;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const int ir = (int)rows, il = (int)len, ik = (int)kp, tmT = (int)tm_T, tmB = (int)tm_B;
    auto grid_for = [&](int rpb) { return dim3((unsigned)((rows + rpb - 1) / rpb)); };
    cudaError_t e;
    switch (g) {
        case 8: cfg.gridDim = grid_for(32); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<8>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB, d2); break;
        case 16: cfg.gridDim = grid_for(16); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<16>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB, d2); break;
        case 32: cfg.gridDim = grid_for(8); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<32>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB, d2); break;
        case 64: cfg.gridDim = grid_for(4); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<64>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB, d2); break;
        case 128: cfg.gridDim = grid_for(2); e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<128>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB, d2); break;
        case 256:  // 128 threads x 16 values a row: two rows a block
            cfg.gridDim = grid_for(2);
            e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_kernel<128, 16>, src, ld, ir, il, ik, dst, prm, rsum, status, tmT, tmB,
                                   d2);
            break;
        default:
            cfg.gridDim = grid_for(kQuantRowsPerBlock);
            e = cudaLaunchKernelEx(&cfg, quantize_rows_f16_warp_kernel, src, ld, ir, il, ik, dst, prm, rsum, status, tmT,
                                   tmB);
    }
    QNN_CUDA_TRY(e);
    return QNN_OK;
}

// Launches the projection's finishing kernel (P <= 2048 values per row); with `pdl` as a
// programmatic dependent launch.
qnn_status launch_proj_finish(const FinishArgs &fa, bool pdl, cudaStream_t st) {
    ProfScope prof("proj_finish", st);
    int g = 8;
    while (g * 8 < fa.P) g *= 2;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    auto grid_for = [&](int rpb) { return dim3((unsigned)((fa.rows + rpb - 1) / rpb)); };
    cudaError_t e;
    switch (g) {
        case 8: cfg.gridDim = grid_for(32); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<8>, fa); break;
        case 16: cfg.gridDim = grid_for(16); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<16>, fa); break;
        case 32: cfg.gridDim = grid_for(8); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<32>, fa); break;
        case 64: cfg.gridDim = grid_for(4); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<64>, fa); break;
        case 128: cfg.gridDim = grid_for(2); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<128>, fa); break;
        case 256: cfg.gridDim = grid_for(1); e = cudaLaunchKernelEx(&cfg, proj_finish_kernel<256>, fa); break;
        default: return QNN_ERR_INVALID_ARG;
    }
    QNN_CUDA_TRY(e);
    return QNN_OK;
}

// Split-K slices of the projection (see tc_partial): at most this many, so the workspace is bounded.
int64_t max_proj_splits(const qnn_lstm_model *m) {
    const int64_t kb = round_up(m->H, 64) / 64;
    return std::max<int64_t>((kb + 15) / 16, 8);
}

// The projection of a step after the m_t quantizer: by default split-K partial sums and a finishing
// row kernel (P <= 2048); with QNN_TC_PROJ=linear, and for P > 2048, one tensor-core product over
// the whole K whose epilogue writes r_t, the next step's quantizer then reading r_t.
bool split_proj_enabled(int64_t P) {
    const char *e = std::getenv("QNN_TC_PROJ");
    return P <= 2048 && !(e && std::strcmp(e, "linear") == 0);
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
        const int64_t kx = round_up(m->layers[l].kin, 64);
        if (kx <= 1024) {  // Wx for the fused input product, and the gate kernel's column constants
            bytes += (size_t)round_up(4 * H8 * kx * 2, 256);
            bytes += (size_t)round_up(12 * H * 4, 256);
        }
    }
    // the 8-bit output layer's Wo as centered fp16 [C][kh], for its product on the top layer's codes
    const bool wo16 = m->C > 0 && m->d.output_mode == QNN_OUT_QUANT;
    if (wo16) bytes += (size_t)round_up(m->C * kh * 2, 256);
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
            return QNN_FAIL(QNN_ERR_CUDA);
        }
        const int64_t kx = round_up(ly.kin, 64);
        if (kx <= 1024) {
            tl.kx = kx;
            tl.wx16 = reinterpret_cast<__half *>(p);
            p += round_up(4 * H8 * kx * 2, 256);
            const int64_t totx = 4 * H8 * (kx / 8);
            interleave_gates_kernel<<<(unsigned)((totx + 255) / 256), 256>>>(ly.wx.codes, ly.wx.ld, (int)H, (int)ly.kin,
                                                                             (int)kx, tl.wx16);
            if (cudaGetLastError() != cudaSuccess) {
                cudaFree(buf);
                return QNN_FAIL(QNN_ERR_CUDA);
            }
            // [12][H] fp32: bias [4][H], Wx row code sums [4][H], Wh row code sums [4][H] (all
            // gate-major; the sums, at most 255 K < 2^24, exact)
            tl.colc = p;
            p += round_up(12 * H * 4, 256);
            float *cc = reinterpret_cast<float *>(tl.colc);
            if (cudaMemcpy(cc, ly.bias, 4 * H * 4, cudaMemcpyDeviceToDevice) != cudaSuccess) {
                cudaFree(buf);
                return QNN_FAIL(QNN_ERR_CUDA);
            }
            sums_to_f32_kernel<<<(unsigned)((4 * H + 255) / 256), 256>>>(ly.wx.sums, cc + 4 * H, 4 * H);
            sums_to_f32_kernel<<<(unsigned)((4 * H + 255) / 256), 256>>>(ly.wh.sums, cc + 8 * H, 4 * H);
            if (cudaGetLastError() != cudaSuccess) {
                cudaFree(buf);
                return QNN_FAIL(QNN_ERR_CUDA);
            }
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
    if (wo16) {
        m->wo16 = reinterpret_cast<__half *>(p);
        p += round_up(m->C * kh * 2, 256);
        qnn_status s = launch_center_fp16(m->wo.codes, m->C, R, m->wo.ld, m->wo16, kh, nullptr);
        if (s != QNN_OK) {
            cudaFree(buf);
            return s;
        }
    }
    if (cudaDeviceSynchronize() != cudaSuccess) {
        cudaFree(buf);
        return QNN_FAIL(QNN_ERR_CUDA);
    }
    m->tcw = buf;
    return QNN_OK;
}

size_t tc_work_bytes(const qnn_lstm_model *m, int64_t B) {
    const int64_t kh = round_up(m->R, 64), kpj = m->P > 0 ? round_up(m->H, 64) : 0;
    const int64_t part = m->P > 0 ? max_proj_splits(m) * B * m->P * 4 : 0;
    return (size_t)round_up(B * kh * 2, 256) + (size_t)round_up(B * kpj * 2, 256) +
           2 * (size_t)round_up(B * (int64_t)sizeof(qnn_qparams), 256) + 2 * (size_t)round_up(B * 4, 256) +
           (size_t)round_up(part, 256);
}

bool tc_input_fused(const qnn_lstm_model *m) {
    const char *v = std::getenv("QNN_TC_FUSE_X");
    if (v && std::strcmp(v, "0") == 0) return false;
    for (int64_t l = 0; l < m->L; ++l)
        if (round_up(m->layers[l].kin, 64) > 1024) return false;
    return true;
}

size_t tc_xwork_bytes(const qnn_lstm_model *m, int64_t rows) {
    int64_t kx = 0;
    for (int64_t l = 0; l < m->L; ++l) kx = std::max(kx, round_up(m->layers[l].kin, 64));
    return (size_t)round_up(rows * kx * 2, 256);
}

namespace {
// One layer's tensor-core recurrence, launched a step at a time: tc_layer_begin, then tc_layer_step
// for t = 0 .. T - 1 in order, all on the run's stream.
struct TcLayerRun {
    const qnn_lstm_model *m = nullptr;
    int64_t l = 0, B = 0, T = 0;
    const float *px = nullptr;  // batched input products (unfused input), row b T + t
    float *cbuf = nullptr, *mbuf = nullptr;
    float *out = nullptr;       // row b of step t's output at out + t * out_t + b * out_b
    int64_t out_t = 0, out_b = 0;
    // nullable: the next layer's time-major input codes, unit params and code sums, which the
    // finishing kernel writes for each step (split projection only)
    __half *nx16 = nullptr;
    qnn_qparams *nprm = nullptr;
    int32_t *nrs = nullptr;
    cudaStream_t st = nullptr;
    bool wave = false;  // one layer of a wavefront (other layers' kernels run beside this one's)
    // set by tc_layer_begin
    TcOperands gates, proj;
    bool split_proj = false, fused = false;
    int splits = 0;
    TcLstmInput xin;
    const __half *x16 = nullptr;
    const qnn_qparams *xprm = nullptr;
    const int32_t *xrs = nullptr;
    __half *a16 = nullptr, *m16 = nullptr;
    qnn_qparams *prm = nullptr, *prm_m = nullptr;
    int32_t *rs = nullptr, *rs_m = nullptr, *part = nullptr;
    int *status = nullptr;
};
}  // namespace

qnn_status tc_layer_begin(TcLayerRun &s, const float *h0, void *work, const TcFusedInput *fx, bool quantize_input) {
    const qnn_lstm_model *m = s.m;
    const LayerDev &ly = m->layers[s.l];
    const TcLayer &tl = m->tc_layers[s.l];
    const int64_t B = s.B, T = s.T, H = m->H, R = m->R, P = m->P, H8 = round_up(H, 8);
    const int64_t kh = tl.kh, kpj = tl.kp;
    char *w = reinterpret_cast<char *>(work);
    s.a16 = reinterpret_cast<__half *>(w);
    w += round_up(B * kh * 2, 256);
    s.m16 = reinterpret_cast<__half *>(w);
    w += round_up(B * kpj * 2, 256);
    s.prm = reinterpret_cast<qnn_qparams *>(w);
    w += round_up(B * (int64_t)sizeof(qnn_qparams), 256);
    s.prm_m = reinterpret_cast<qnn_qparams *>(w);
    w += round_up(B * (int64_t)sizeof(qnn_qparams), 256);
    s.rs = reinterpret_cast<int32_t *>(w);
    w += round_up(B * 4, 256);
    s.rs_m = reinterpret_cast<int32_t *>(w);
    w += round_up(B * 4, 256);
    s.part = reinterpret_cast<int32_t *>(w);

    QNN_TRY(status_word(&s.status));
    // tile widths, widest first; the fused kernel's 96-column tile (24 warps at 72 registers) spills
    // with the second recovery and measured slower than 64 columns, so it is left out there
    static const int gate_bn[] = {128, 96, 64, 32}, gate_bn_fused[] = {128, 64, 32};
    // The fused kernel's operand stream (A re-read for every tile of a block) is bounded by the rate at
    // which a block's TMA ring turns over, so with at least a full wave of tiles the widest tile wins
    // (LSTMP 5x2048p512 B=1024: 128 columns 49.6 us per step against 52.0 for 64); with less than a
    // wave the tile count that fills the SMs best decides, except in a wavefront, where the other
    // layers' kernels fill the SMs a narrow grid leaves: there the widest tile always wins (5 x 500
    // B = 256: 32 blocks of 128 columns 8.9M frames/s, 64 of 64 columns 8.5M, 126 of 32 columns 6.0M).
    int bn_gates = fx ? tc_choose_bn(B, 4 * H8, gate_bn_fused, 3) : tc_choose_bn(B, 4 * H8, gate_bn, 4);
    if (fx && !std::getenv("QNN_TC_BN") &&
        (s.wave || ((B + 127) / 128) * ((4 * H8 + 127) / 128) >= sm_count()))
        bn_gates = 128;
    QNN_TRY(tc_operands(&s.gates, s.a16, B, tl.wh16, 4 * H8, kh, bn_gates));
    // the projection after the m_t quantizer: split-K partial sums finished (offsets, recovery, next
    // step's quantization) by one row kernel; or one tcgen05 product with its own epilogue per step
    s.split_proj = P > 0 && split_proj_enabled(P);
    s.splits = 0;
    if (P > 0) {
        QNN_TRY(tc_operands(&s.proj, s.m16, B, tl.wp16, P, kpj, s.split_proj ? 128 : tc_pick_bn(B, P, kpj)));
        if (s.split_proj) s.splits = tc_partial_splits(s.proj, (int)max_proj_splits(m));
    }
    // the steps' kernels chain by programmatic dependent launches (see tc_gemm.h); the first one of
    // the layer follows ordinary stream order
    s.gates.pdl = s.proj.pdl = pdl_enabled();
    // fused input product: the layer input as centered fp16 codes, time-major (row t B + b), so a
    // step's x_t rows of all sequences are one contiguous block; quantized here at once, or written
    // step by step by the previous layer (quantize_input false)
    s.fused = fx != nullptr;
    if (fx) {
        if (!tl.wx16 || tl.kx != round_up(fx->kin, 64)) return QNN_ERR_INVALID_ARG;
        if (quantize_input)
            QNN_TRY(launch_quantize_rows_f16(fx->in, fx->kin, B * T, (int)fx->kin, (int)tl.kx, fx->x16, fx->prm,
                                             fx->rs, s.status, false, s.st, T, B));
        s.x16 = fx->x16, s.xprm = fx->prm, s.xrs = fx->rs;
        s.xin.x_pitch = tl.kx, s.xin.kx = tl.kx, s.xin.K_x = (int)fx->kin, s.xin.stride = 1;
        s.xin.wx16 = tl.wx16, s.xin.pw4 = ly.wx.params, s.xin.cs = ly.wx.sums, s.xin.bias = ly.bias;
        s.xin.colc = tl.colc;
    }
    QNN_TRY(launch_quantize_rows_f16(h0, R, B, R, kh, s.a16, s.prm, s.rs, s.status, false, s.st));
    return QNN_OK;
}

qnn_status tc_layer_step(TcLayerRun &s, int64_t t) {
    const qnn_lstm_model *m = s.m;
    const LayerDev &ly = m->layers[s.l];
    const TcLayer &tl = m->tc_layers[s.l];
    const int64_t B = s.B, T = s.T, H = m->H, R = m->R, P = m->P;
    const int64_t kh = tl.kh, kpj = tl.kp;
    cudaStream_t st = s.st;
    float *out_t = s.out + t * s.out_t;  // row b of this step's output at out_t + b * out_b
    // the next layer's input codes of this step (wavefront), written with this step's own codes
    const RowCodes next{s.nx16 ? s.nx16 + t * B * kh : nullptr, s.nx16 ? s.nprm + t * B : nullptr,
                        s.nx16 ? s.nrs + t * B : nullptr};
    TcLstmOut o{s.fused ? nullptr : s.px + t * 4 * H, T * 4 * H, s.cbuf, P > 0 ? s.mbuf : out_t, P > 0 ? H : s.out_b,
                (int)H, (int)m->S, (int)(H / m->S)};
    if (s.fused) {
        TcLstmInput xin = s.xin;
        xin.x16 = s.x16 + t * B * tl.kx, xin.pa = s.xprm + t * B, xin.rs = s.xrs + t * B;
        QNN_TRY(tc_lstm_gates_x(s.gates, s.prm, s.rs, R, ly.wh.params, ly.wh.sums, o, xin, st));
    } else {
        QNN_TRY(tc_lstm_gates(s.gates, s.prm, s.rs, R, ly.wh.params, ly.wh.sums, o, st));
    }
    if (P > 0) {
        QNN_TRY(launch_quantize_rows_f16(s.mbuf, H, B, H, kpj, s.m16, s.prm_m, s.rs_m, s.status, s.gates.pdl, st));
        if (s.split_proj) {
            QNN_TRY(tc_partial(s.proj, s.splits, s.part, P, st));
            FinishArgs fa{s.part, s.splits, P, s.prm_m, s.rs_m, ly.wp.params, ly.wp.sums, (int)(P / m->S), (int)H,
                          out_t, s.out_b, (int)B, (int)P, t + 1 < T || s.nx16 != nullptr, (int)kh, s.a16, s.prm,
                          s.rs, s.status, next.dst, next.prm, next.rsum};
            QNN_TRY(launch_proj_finish(fa, s.gates.pdl, st));
        } else {
            QNN_TRY(tc_linear(s.proj, s.prm_m, 1, s.rs_m, H, ly.wp.params, P / m->S, ly.wp.sums, nullptr, out_t, s.out_b,
                              nullptr, st));
        }
    }
    // without the finishing kernel: this step's outputs quantized as the next step's recurrent input
    // (and the next layer's input)
    if (!s.split_proj && (t + 1 < T || s.nx16))
        QNN_TRY(launch_quantize_rows_f16(out_t, s.out_b, B, R, kh, s.a16, s.prm, s.rs, s.status, s.gates.pdl, st, 0, 0,
                                         next));
    return QNN_OK;
}

qnn_status tc_layer_recurrence(const qnn_lstm_model *m, int64_t l, const float *px, const float *h0, float *cbuf,
                               float *out, float *mbuf, int64_t B, int64_t T, void *work, cudaStream_t st,
                               const TcFusedInput *fx) {
    TcLayerRun s;
    s.m = m, s.l = l, s.B = B, s.T = T, s.px = px, s.cbuf = cbuf, s.mbuf = mbuf;
    s.out = out, s.out_t = m->R, s.out_b = T * m->R, s.st = st;
    QNN_TRY(tc_layer_begin(s, h0, work, fx, true));
    for (int64_t t = 0; t < T; ++t) QNN_TRY(tc_layer_step(s, t));
    return QNN_OK;
}

bool tc_stack_supported(const qnn_lstm_model *m) {
    const char *e = std::getenv("QNN_TC_WAVE");
    if (e && std::strcmp(e, "0") == 0) return false;
    return m->L >= 2 && tc_input_fused(m);
}

qnn_status tc_stack_recurrence(const qnn_lstm_model *m, const TcStackLayer *layers, int64_t B, int64_t T,
                               const cudaStream_t *streams, const cudaEvent_t *edges, const TcFusedInput *top_codes,
                               const std::function<qnn_status(int64_t)> &after_top_step) {
    if (!tc_stack_supported(m)) return QNN_ERR_INVALID_ARG;
    const int64_t L = m->L;
    std::vector<TcLayerRun> runs((size_t)L);
    for (int64_t l = 0; l < L; ++l) {
        TcLayerRun &r = runs[(size_t)l];
        const TcStackLayer &sl = layers[l];
        r.m = m, r.l = l, r.B = B, r.T = T, r.cbuf = sl.cbuf, r.mbuf = sl.mbuf;
        r.out = sl.out, r.out_t = sl.out_t, r.out_b = sl.out_b, r.st = streams[l];
        if (l + 1 < L)
            r.nx16 = layers[l + 1].fx.x16, r.nprm = layers[l + 1].fx.prm, r.nrs = layers[l + 1].fx.rs;
        else if (top_codes)  // the output layer's input codes
            r.nx16 = top_codes->x16, r.nprm = top_codes->prm, r.nrs = top_codes->rs;
        r.wave = true;
        QNN_TRY(tc_layer_begin(r, sl.h0, sl.work, &sl.fx, l == 0));
        // whole tiles in the last, partial wave: the blocks that finish early free their SMs for
        // the other layers' kernels, which gains more than halving those tiles to even out the
        // wave (LSTMP 5 x 2048p512 B = 1024: 3.94M against 3.82M frames/s); and a gate grid of 90%
        // of the SMs, so that the projection kernels of the other layers always find some
        // (4.15M against 4.07M frames/s with every SM; 128 and 144 of 152 blocks: 4.11M)
        r.gates.half_items = false;
        r.gates.max_blocks = sm_count() * 9 / 10;
        // the projection's split-K product in as few K ranges as its exact chunks allow: fewer,
        // longer work items hold fewer SMs beside the other layers' gate kernels (4.38M against
        // 4.09-4.13M frames/s with 2 ranges of 1024 instead of 4 of 512)
        if (r.split_proj) r.splits = tc_partial_splits(r.proj, (int)max_proj_splits(m), false);
    }
    // step t of layer l after step t of layer l - 1 (its input codes); each layer's own steps follow
    // its stream order
    for (int64_t t = 0; t < T; ++t)
        for (int64_t l = 0; l < L; ++l) {
            if (l > 0) QNN_CUDA_TRY(cudaStreamWaitEvent(streams[l], edges[l - 1], 0));
            QNN_TRY(tc_layer_step(runs[(size_t)l], t));
            if (l + 1 < L) QNN_CUDA_TRY(cudaEventRecord(edges[l], streams[l]));
            else if (after_top_step) QNN_TRY(after_top_step(t));
        }
    return QNN_OK;
}

}  // namespace qnn
