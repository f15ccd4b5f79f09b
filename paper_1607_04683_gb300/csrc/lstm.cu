// lstm.cu — the quantized LSTM / LSTMP stack (Sec. 3.1 layer scheme applied to every gate matrix,
// Sec. 4 model family) and its softmax output layer.
//
// Per layer:
//   1. quantize every input frame on the fly (one unit per row, eq. 2);
//   2. one batched integer product over all B*T frames with the four Wx gate matrices, recovered
//      and biased in the epilogue: px = R(Q(x) Wx') + b  (eq. 1, eq. 3, Fig. 1);
//   3. a persistent kernel runs the T recurrent steps: each step quantizes h_{t-1} in-kernel,
//      multiplies it with the shared-memory-resident Wh' slice of the block on the integer tensor
//      cores, recovers, adds px and applies the gates and the cell update; with a projection it
//      then quantizes m_t and multiplies with Wp'. Steps are separated by a grid-wide barrier
//      whose waits are bounded in time.
// Output layer: quantize the top layer's outputs, integer product with Wo', recovery + bias, then
// softmax with the pinned exponential.
#include <algorithm>
#include <cfloat>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <vector>

#include "lstm_model.h"
#include "qnn_device.cuh"
#include "qnn_host.h"
#include "tc_gemm.h"

namespace qnn {
namespace {

constexpr int kRecThreads = 256;
constexpr int kRecWarps = kRecThreads / 32;
constexpr int kPad = 16;  // extra bytes per shared-memory code row (bank spread for ldmatrix)
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s per grid-wide wait
constexpr int kDistQuantMinBatch = 8;  // batch from which rows are quantized once per step, grid-wide

inline int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma_u8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.u8.u8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ unsigned ld_acquire(const unsigned *p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;\n" : "=l"(t));
    return t;
}

struct RecArgs {
    const uint8_t *wh;        // [4H][ldh] codes, row g*H + j, zero padded
    const int32_t *wh_sum;    // [4H] row code sums
    const qnn_qparams *wh_p;  // [4] one unit per gate matrix
    const float *px;          // [B*T][4H] recovered input product + bias, row b*T + t
    const float *h0;          // [B][R] outputs before the first frame
    float *cbuf;              // [B][H] cell state (in/out)
    float *out;               // [B][T][R] layer outputs
    const uint8_t *wp;        // [P][ldp] projection codes (P > 0)
    const int32_t *wp_sum;    // [P]
    const qnn_qparams *wp_p;  // [1]
    float *mbuf;              // [B][H] cell outputs before the projection (P > 0)
    unsigned *bar;            // grid barrier counter, zero at launch
    int *abort_flag;          // set when any wait gave up, zero at launch
    int *status;
    // shared quantization (large batches): each row is quantized once per step by one warp of
    // the grid into these buffers, then every block copies the rows it needs
    uint8_t *qcodes;          // [B][ldq]
    qnn_qparams *qprm;        // [B]
    int *qsum;                // [B]
    int ldq, distq;
    int B, T, H, R, P, ldh, ldp, nc, np, bc;
    int ups, cpu, ppu;        // weight units per gate matrix; cells (Wh rows) and Wp rows per unit
};

// Grid-wide barrier with a bounded wait: returns false if this or another block gave up, in
// which case QNN_ERR_TIMEOUT has been recorded and every block leaves its loop.
__device__ __forceinline__ bool grid_sync(const RecArgs &a, unsigned &epoch, int *s_flag) {
    __syncthreads();
    if (threadIdx.x == 0) {
        epoch += 1;
        const unsigned target = epoch * gridDim.x;
        __threadfence();
        atomicAdd(a.bar, 1u);
        const unsigned long long t0 = global_ns();
        int ok = 1;
        while (ld_acquire(a.bar) < target) {
            if (*(volatile int *)a.abort_flag) {
                ok = 0;
                break;
            }
            if (global_ns() - t0 > kWaitLimitNs) {
                record_status(a.status, QNN_ERR_TIMEOUT);
                atomicExch(a.abort_flag, 1);
                ok = 0;
                break;
            }
            __nanosleep(20);
        }
        *s_flag = ok;
    }
    __syncthreads();
    return *s_flag != 0;
}

// Quantizes `nb` rows of `len` fp32 values (row r at src + r*ld) into shared-memory codes
// (row stride srow, zero past len up to kdim) plus per-row offset, scale and code sum. Rows
// nb..rows_total-1 become zero rows. One warp per row.
__device__ __forceinline__ void quantize_rows_smem(const float *src, int64_t ld, int nb, int rows_total, int len,
                                                   int kdim, uint8_t *sact, int srow, int *sza, float *sQa, int *srs,
                                                   int *status) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int r = warp; r < rows_total; r += kRecWarps) {
        uint8_t *dst = sact + r * srow;
        if (r >= nb) {
            for (int k = lane * 4; k < kdim; k += 128) *reinterpret_cast<uint32_t *>(dst + k) = 0u;
            if (lane == 0) {
                sza[r] = 0;
                sQa[r] = 1.0f;
                srs[r] = 0;
            }
            continue;
        }
        const float *xr = src + r * ld;
        float mn = FLT_MAX, mx = -FLT_MAX;
        bool bad = false;
        for (int k = lane; k < len; k += 32) {
            float v = xr[k];
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
        int s = 0;
        for (int k4 = lane * 4; k4 < kdim; k4 += 128) {
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int k = k4 + e;
                if (k < len) {
                    uint32_t c = quant_code(xr[k], p.Q, p.z);
                    s += (int)c;
                    w |= c << (8 * e);
                }
            }
            *reinterpret_cast<uint32_t *>(dst + k4) = w;
        }
        s = warp_sum(s);
        if (lane == 0) {
            sza[r] = p.z;
            sQa[r] = p.Q;
            srs[r] = s;
        }
    }
}

// Quantizes `rows` rows of `len` fp32 values (row r at src + r*ld) into the shared global buffers,
// one warp per row, the rows spread over every warp of the grid.
__device__ __forceinline__ void quantize_rows_global(const float *src, int64_t ld, int rows, int len, int kdim,
                                                     const RecArgs &a) {
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * kRecWarps + (threadIdx.x >> 5), nw = gridDim.x * kRecWarps;
    for (int r = gw; r < rows; r += nw) {
        const float *xr = src + r * ld;
        float mn = FLT_MAX, mx = -FLT_MAX;
        bool bad = false;
        for (int k = lane; k < len; k += 32) {
            float v = __ldcg(xr + k);
            bad |= !isfinite(v);
            mn = fminf(mn, v);
            mx = fmaxf(mx, v);
        }
        mn = warp_min(mn);
        mx = warp_max(mx);
        if (__any_sync(0xffffffffu, bad)) {
            if (lane == 0) record_status(a.status, QNN_ERR_NONFINITE);
            mn = 0.0f;
            mx = 0.0f;
        }
        const qnn_qparams p = params_from_range(mn, mx);
        uint8_t *dst = a.qcodes + (int64_t)r * a.ldq;
        int s = 0;
        for (int k4 = lane * 4; k4 < kdim; k4 += 128) {
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int k = k4 + e;
                if (k < len) {
                    uint32_t c = quant_code(__ldcg(xr + k), p.Q, p.z);
                    s += (int)c;
                    w |= c << (8 * e);
                }
            }
            *reinterpret_cast<uint32_t *>(dst + k4) = w;
        }
        s = warp_sum(s);
        if (lane == 0) {
            a.qprm[r] = p;
            a.qsum[r] = s;
        }
    }
}

// Copies rows b0 .. b0 + nb - 1 of the shared quantized rows (kdim bytes each) into shared memory
// as quantize_rows_smem would have produced them; rows nb .. rows_total - 1 become zero rows.
__device__ __forceinline__ void load_rows_smem(const RecArgs &a, int b0, int nb, int rows_total, int kdim,
                                               uint8_t *sact, int srow, int *sza, float *sQa, int *srs) {
    const int chunks = kdim / 16;
    for (int i = threadIdx.x; i < rows_total * chunks; i += kRecThreads) {
        const int r = i / chunks, ch = i % chunks;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (r < nb) v = __ldcg(reinterpret_cast<const uint4 *>(a.qcodes + (int64_t)(b0 + r) * a.ldq + ch * 16));
        *reinterpret_cast<uint4 *>(sact + r * srow + ch * 16) = v;
    }
    for (int r = threadIdx.x; r < rows_total; r += kRecThreads) {
        if (r < nb) {
            sza[r] = __ldcg(&a.qprm[b0 + r].z);
            sQa[r] = __ldcg(&a.qprm[b0 + r].Q);
            srs[r] = __ldcg(a.qsum + b0 + r);
        } else {
            sza[r] = 0;
            sQa[r] = 1.0f;
            srs[r] = 0;
        }
    }
}

// Integer products of `mrows` shared-memory weight rows with `bc` activation rows over kdim
// (multiple of 32), recovered into sy[row][col] with the expanded offsets of eq. (1).
// `row_info(lr, &zw, &Qw, &csw, &valid)` gives the weight unit of local row lr.
template <typename RowInfo>
__device__ __forceinline__ void product_block(const uint8_t *sw, int wrow, const uint8_t *sact, int arow, int mrows,
                                              int bc, int kdim, int ktrue, const int *sza, const float *sQa,
                                              const int *srs, float *sy, RowInfo row_info) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mfr = mrows / 16, npair = bc / 16;
    const uint32_t w0 = smem_u32(sw), a0 = smem_u32(sact);
    for (int item = warp; item < mfr * npair; item += kRecWarps) {
        const int mi = item / npair, nj = item % npair;
        int acc[2][4] = {{0, 0, 0, 0}, {0, 0, 0, 0}};
        const uint32_t wa = w0 + (mi * 16 + (lane & 15)) * wrow + (lane >> 4) * 16;
        const uint32_t aa = a0 + (nj * 16 + (lane & 7) + ((lane >> 4) << 3)) * arow + ((lane >> 3) & 1) * 16;
        for (int k = 0; k < kdim; k += 32) {
            uint32_t af[4], b0, b1, b2, b3;
            ldmatrix_x4(wa + k, af[0], af[1], af[2], af[3]);
            ldmatrix_x4(aa + k, b0, b1, b2, b3);
            mma_u8(acc[0], af, b0, b1);
            mma_u8(acc[1], af, b2, b3);
        }
        const int g = lane >> 2, tq = lane & 3;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int lr = mi * 16 + g + h * 8;
            int zw, csw;
            float Qw;
            bool valid;
            row_info(lr, zw, Qw, csw, valid);
#pragma unroll
            for (int ni = 0; ni < 2; ++ni)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int col = nj * 16 + ni * 8 + tq * 2 + e;
                    float y = 0.0f;
                    if (valid) {
                        const long long S = offset_product(acc[ni][h * 2 + e], sza[col], zw, srs[col], csw, ktrue);
                        y = recover_product(S, sQa[col], Qw);
                    }
                    sy[lr * bc + col] = y;
                }
        }
    }
}

__global__ void __launch_bounds__(kRecThreads, 1) lstm_recurrent_kernel(RecArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int s_flag;
    const int nc = a.nc, np = a.np, bc = a.bc;
    const int j0 = blockIdx.x * nc;
    const int p0 = blockIdx.x * np;
    const int wrow_h = a.ldh + kPad, wrow_p = a.ldp + kPad;
    const int arow = (a.ldh > a.ldp ? a.ldh : a.ldp) + kPad;
    // shared-memory carve-up
    uint8_t *sw_h = smem;
    uint8_t *sw_p = sw_h + 4 * nc * wrow_h;
    uint8_t *sact = sw_p + (a.P > 0 ? np * wrow_p : 0);
    float *sy = reinterpret_cast<float *>(sact + bc * arow);
    const int ymax = (4 * nc > np ? 4 * nc : np);
    int *sza = reinterpret_cast<int *>(sy + ymax * bc);
    float *sQa = reinterpret_cast<float *>(sza + bc);
    int *srs = reinterpret_cast<int *>(sQa + bc);

    // Resident weight slices: gate rows of this block's cells, local row g*nc + jj.
    for (int idx = threadIdx.x; idx < 4 * nc * (a.ldh / 16); idx += kRecThreads) {
        const int lr = idx / (a.ldh / 16), ch = idx % (a.ldh / 16);
        const int gate = lr / nc, j = j0 + lr % nc;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (j < a.H) v = *reinterpret_cast<const uint4 *>(a.wh + ((int64_t)gate * a.H + j) * a.ldh + ch * 16);
        *reinterpret_cast<uint4 *>(sw_h + lr * wrow_h + ch * 16) = v;
    }
    if (a.P > 0) {
        for (int idx = threadIdx.x; idx < np * (a.ldp / 16); idx += kRecThreads) {
            const int lr = idx / (a.ldp / 16), ch = idx % (a.ldp / 16);
            const int p = p0 + lr;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (p < a.P) v = *reinterpret_cast<const uint4 *>(a.wp + (int64_t)p * a.ldp + ch * 16);
            *reinterpret_cast<uint4 *>(sw_p + lr * wrow_p + ch * 16) = v;
        }
    }
    __syncthreads();

    const int H = a.H, R = a.R, T = a.T;
    const int64_t G4 = 4 * (int64_t)H;
    auto h_row_info = [&](int lr, int &zw, float &Qw, int &csw, bool &valid) {
        const int gate = lr / nc, j = j0 + lr % nc;
        valid = j < H;
        const qnn_qparams q = a.wh_p[gate * a.ups + (valid ? j : 0) / a.cpu];  // the row's unit
        zw = q.z;
        Qw = q.Q;
        csw = valid ? a.wh_sum[gate * H + j] : 0;
    };
    auto p_row_info = [&](int lr, int &zw, float &Qw, int &csw, bool &valid) {
        const int p = p0 + lr;
        valid = p < a.P;
        const qnn_qparams q = a.wp_p[(valid ? p : 0) / a.ppu];
        zw = q.z;
        Qw = q.Q;
        csw = valid ? a.wp_sum[p] : 0;
    };

    unsigned epoch = 0;
    for (int t = 0; t < T; ++t) {
        if (a.distq) {  // every row of h_{t-1} quantized once, by one warp of the grid
            const float *hsrc = (t == 0) ? a.h0 : a.out + (t - 1) * (int64_t)R;
            quantize_rows_global(hsrc, (t == 0) ? R : (int64_t)T * R, a.B, R, a.ldh, a);
            if (!grid_sync(a, epoch, &s_flag)) return;
        }
        for (int b0 = 0; b0 < a.B; b0 += bc) {
            const int nb = min(bc, a.B - b0);
            if (a.distq) {
                load_rows_smem(a, b0, nb, bc, a.ldh, sact, arow, sza, sQa, srs);
            } else {
                const float *hsrc = (t == 0) ? a.h0 + (int64_t)b0 * R : a.out + ((int64_t)b0 * T + (t - 1)) * R;
                const int64_t hld = (t == 0) ? R : (int64_t)T * R;
                quantize_rows_smem(hsrc, hld, nb, bc, R, a.ldh, sact, arow, sza, sQa, srs, a.status);
            }
            __syncthreads();
            product_block(sw_h, wrow_h, sact, arow, 4 * nc, bc, a.ldh, R, sza, sQa, srs, sy, h_row_info);
            __syncthreads();
            for (int idx = threadIdx.x; idx < nb * nc; idx += kRecThreads) {
                const int r = idx / nc, jj = idx % nc;
                const int j = j0 + jj;
                if (j >= H) continue;
                const int64_t b = b0 + r;
                const float *pxr = a.px + (b * T + t) * G4;
                float pre[4];
#pragma unroll
                for (int gte = 0; gte < 4; ++gte) pre[gte] = __fadd_rn(pxr[gte * H + j], sy[(gte * nc + jj) * bc + r]);
                float c = a.cbuf[b * H + j], m;
                lstm_cell(pre[0], pre[1], pre[2], pre[3], c, m);
                a.cbuf[b * H + j] = c;
                if (a.P > 0)
                    a.mbuf[b * H + j] = m;
                else
                    a.out[(b * T + t) * R + j] = m;
            }
            __syncthreads();
        }
        if (a.P > 0) {
            if (!grid_sync(a, epoch, &s_flag)) return;
            if (a.distq) {  // every row of m_t quantized once
                quantize_rows_global(a.mbuf, H, a.B, H, a.ldp, a);
                if (!grid_sync(a, epoch, &s_flag)) return;
            }
            if (p0 < a.P) {
                for (int b0 = 0; b0 < a.B; b0 += bc) {
                    const int nb = min(bc, a.B - b0);
                    if (a.distq)
                        load_rows_smem(a, b0, nb, bc, a.ldp, sact, arow, sza, sQa, srs);
                    else
                        quantize_rows_smem(a.mbuf + (int64_t)b0 * H, H, nb, bc, H, a.ldp, sact, arow, sza, sQa, srs,
                                           a.status);
                    __syncthreads();
                    product_block(sw_p, wrow_p, sact, arow, np, bc, a.ldp, H, sza, sQa, srs, sy, p_row_info);
                    __syncthreads();
                    for (int idx = threadIdx.x; idx < nb * np; idx += kRecThreads) {
                        const int r = idx / np, pp = idx % np;
                        const int p = p0 + pp;
                        if (p >= a.P) continue;
                        a.out[((int64_t)(b0 + r) * T + t) * R + p] = sy[pp * bc + r];
                    }
                    __syncthreads();
                }
            }
        }
        if (!grid_sync(a, epoch, &s_flag)) return;
    }
}

__global__ void __launch_bounds__(256) softmax_rows_kernel(const float *__restrict__ logits, int C,
                                                           float *__restrict__ y, int64_t tm_B, int64_t tm_T,
                                                           int64_t tm_t0) {
    __shared__ float red[8];
    __shared__ float s_bcast;
    const int64_t row = blockIdx.x;
    const float *l = logits + row * C;
    // time-major rows (tm_B > 0): row i is frame tm_t0 + i / tm_B of sequence i % tm_B, whose
    // posteriors go to row (i % tm_B) tm_T + tm_t0 + i / tm_B of y
    const int64_t yrow = tm_B > 0 ? (row % tm_B) * tm_T + tm_t0 + row / tm_B : row;
    float *yr = y + yrow * C;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float mx = -FLT_MAX;
    for (int c = threadIdx.x; c < C; c += 256) mx = fmaxf(mx, l[c]);
    mx = warp_max(mx);
    if (lane == 0) red[warp] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = red[0];
        for (int w = 1; w < 8; ++w) v = fmaxf(v, red[w]);
        s_bcast = v;
    }
    __syncthreads();
    mx = s_bcast;
    float s = 0.0f;
    for (int c = threadIdx.x; c < C; c += 256) s = __fadd_rn(s, pexp(__fsub_rn(l[c], mx)));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xffffffffu, s, o));
    __syncthreads();
    if (lane == 0) red[warp] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = red[0];
        for (int w = 1; w < 8; ++w) v = __fadd_rn(v, red[w]);
        s_bcast = v;
    }
    __syncthreads();
    s = s_bcast;
    // y is written once (it may be host memory): E(l - max) is recomputed, the same value as above;
    // 16-byte stores where the rows allow them (each posterior is computed on its own, so the
    // grouping does not change a value)
    if ((C & 3) == 0 && ((reinterpret_cast<uintptr_t>(l) | reinterpret_cast<uintptr_t>(yr)) & 15) == 0) {
        const float4 *l4 = reinterpret_cast<const float4 *>(l);
        float4 *y4 = reinterpret_cast<float4 *>(yr);
        for (int v = threadIdx.x; v < C / 4; v += 256) {
            const float4 lv = l4[v];
            y4[v] = make_float4(__fdiv_rn(pexp(__fsub_rn(lv.x, mx)), s), __fdiv_rn(pexp(__fsub_rn(lv.y, mx)), s),
                                __fdiv_rn(pexp(__fsub_rn(lv.z, mx)), s), __fdiv_rn(pexp(__fsub_rn(lv.w, mx)), s));
        }
    } else {
        for (int c = threadIdx.x; c < C; c += 256) yr[c] = __fdiv_rn(pexp(__fsub_rn(l[c], mx)), s);
    }
}

// The same softmax with the row held in registers (rows of at most 256 V values, C a multiple of 4,
// 16-byte aligned rows): the logits are read once, each E(l - max) is computed once and kept, and
// the quotients E / sum come from the sum's correctly rounded reciprocal r (q = RN(E r), then
// RN(q + (E - q sum) r), the last step of Markstein's division; equal to the IEEE quotient while
// E >= 2^-100 and 1 <= sum <= 2^24, which a CPU test checks; smaller E divide as IEEE). Thread t
// holds the 4-value groups t, t + 256, ...
template <int V>
__global__ void __launch_bounds__(256) softmax_rows_reg_kernel(const float *__restrict__ logits, int C,
                                                               float *__restrict__ y, int64_t tm_B, int64_t tm_T,
                                                               int64_t tm_t0) {
    __shared__ float red[8];
    __shared__ float s_bcast;
    const int64_t row = blockIdx.x;
    const float4 *l4 = reinterpret_cast<const float4 *>(logits + row * C);
    const int64_t yrow = tm_B > 0 ? (row % tm_B) * tm_T + tm_t0 + row / tm_B : row;
    float4 *y4 = reinterpret_cast<float4 *>(y + yrow * C);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int C4 = C / 4;
    float e[V];
    float mx = -FLT_MAX;
#pragma unroll
    for (int j = 0; j < V / 4; ++j) {
        const int v = (int)threadIdx.x + 256 * j;
        float4 a = make_float4(-FLT_MAX, -FLT_MAX, -FLT_MAX, -FLT_MAX);
        if (v < C4) a = l4[v];
        e[4 * j] = a.x, e[4 * j + 1] = a.y, e[4 * j + 2] = a.z, e[4 * j + 3] = a.w;
        mx = fmaxf(mx, fmaxf(fmaxf(a.x, a.y), fmaxf(a.z, a.w)));
    }
    mx = warp_max(mx);
    if (lane == 0) red[warp] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = red[0];
        for (int w = 1; w < 8; ++w) v = fmaxf(v, red[w]);
        s_bcast = v;
    }
    __syncthreads();
    mx = s_bcast;
    float s = 0.0f;
#pragma unroll
    for (int j = 0; j < V / 4; ++j) {
        if ((int)threadIdx.x + 256 * j >= C4) break;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            e[4 * j + i] = pexp(__fsub_rn(e[4 * j + i], mx));
            s = __fadd_rn(s, e[4 * j + i]);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xffffffffu, s, o));
    __syncthreads();
    if (lane == 0) red[warp] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = red[0];
        for (int w = 1; w < 8; ++w) v = __fadd_rn(v, red[w]);
        s_bcast = v;
    }
    __syncthreads();
    s = s_bcast;
    const float r = __frcp_rn(s);
    auto quot = [&](float x) { return x >= 0x1p-100f ? div_by_recip(x, s, r) : __fdiv_rn(x, s); };
#pragma unroll
    for (int j = 0; j < V / 4; ++j) {
        const int v = (int)threadIdx.x + 256 * j;
        if (v >= C4) break;
        y4[v] = make_float4(quot(e[4 * j]), quot(e[4 * j + 1]), quot(e[4 * j + 2]), quot(e[4 * j + 3]));
    }
}

// fp32 output layer for the "quant" variant: logits[m][c] = sum_k r[m][k] Wo[c][k] + bo[c].
__global__ void __launch_bounds__(256) float_linear_kernel(const float *__restrict__ X, int64_t M, int K,
                                                           const float *__restrict__ Wt, int C,
                                                           const float *__restrict__ bias, float *__restrict__ Y) {
    __shared__ float xs[32][33];
    __shared__ float ws[32][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 8 rows of 32
    const int64_t m0 = (int64_t)blockIdx.y * 32;
    const int c0 = blockIdx.x * 32;
    float acc[4] = {0, 0, 0, 0};
    for (int k0 = 0; k0 < K; k0 += 32) {
        for (int i = ty; i < 32; i += 8) {
            xs[i][tx] = (m0 + i < M && k0 + tx < K) ? X[(m0 + i) * K + k0 + tx] : 0.0f;
            ws[i][tx] = (c0 + i < C && k0 + tx < K) ? Wt[(int64_t)(c0 + i) * K + k0 + tx] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 32; ++k)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[q] = fmaf(xs[ty + 8 * q][k], ws[tx][k], acc[q]);
        __syncthreads();
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int64_t m = m0 + ty + 8 * q;
        const int c = c0 + tx;
        if (m < M && c < C) Y[m * C + c] = acc[q] + bias[c];
    }
}

}  // namespace

qnn_status launch_softmax_rows(const float *logits, int64_t rows, int64_t C, float *y, cudaStream_t st, int64_t tm_B,
                               int64_t tm_T, int64_t tm_t0) {
    if (rows == 0) return QNN_OK;
    ProfScope prof("softmax_rows", st);
    // rows in registers when they fit (1 <= sum <= C <= 8192 keeps the reciprocal quotient exact)
    const bool reg = (C & 3) == 0 && C <= 8192 &&
                     ((reinterpret_cast<uintptr_t>(logits) | reinterpret_cast<uintptr_t>(y)) & 15) == 0;
    if (reg && C <= 2048)
        softmax_rows_reg_kernel<8><<<(unsigned)rows, 256, 0, st>>>(logits, (int)C, y, tm_B, tm_T, tm_t0);
    else if (reg && C <= 4096)
        softmax_rows_reg_kernel<16><<<(unsigned)rows, 256, 0, st>>>(logits, (int)C, y, tm_B, tm_T, tm_t0);
    else if (reg)
        softmax_rows_reg_kernel<32><<<(unsigned)rows, 256, 0, st>>>(logits, (int)C, y, tm_B, tm_T, tm_t0);
    else
        softmax_rows_kernel<<<(unsigned)rows, 256, 0, st>>>(logits, (int)C, y, tm_B, tm_T, tm_t0);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

}  // namespace qnn

// ------------------------------------------------------------------------------------------------
// Model
// ------------------------------------------------------------------------------------------------

using namespace qnn;

namespace {

// Features per network input: the frame features times the frames stacked (Sec. 4 frontend).
int64_t network_input_dim(const qnn_lstm_desc *d) { return (int64_t)d->input_dim * (d->stack > 1 ? d->stack : 1); }

bool valid_desc(const qnn_lstm_desc *d) {
    if (!d || d->num_layers < 1 || d->input_dim < 1 || d->hidden < 1 || d->proj < 0 || d->num_classes < 0) return false;
    if (d->stack < 0 || d->stack_stride < 0 || d->weight_blocks < 0) return false;
    const int S = d->weight_blocks > 1 ? d->weight_blocks : 1;  // units per weight matrix
    if (d->hidden % S || (d->proj > 0 && d->proj % S)) return false;
    if (d->num_classes > 0 && d->output_mode == QNN_OUT_QUANT && d->num_classes % S) return false;
    if ((d->num_classes == 0) != (d->output_mode == QNN_OUT_NONE)) return false;
    if (d->output_mode < QNN_OUT_NONE || d->output_mode > QNN_OUT_FLOAT) return false;
    return true;
}

struct Bump {
    char *base;
    size_t off = 0;
    template <typename T>
    T *take(size_t n) {
        off = (size_t)round_up((int64_t)off, 256);
        T *p = reinterpret_cast<T *>(base + off);
        off += n * sizeof(T);
        return p;
    }
};

// Quantizes n_units row blocks of an fp32 matrix [rows][cols] (block b = rows b*rows/n..), each
// one unit (per-matrix rule), into codes [rows][ld] (zero padded), row sums and params.
qnn_status quantize_units(const float *w, int64_t rows, int64_t cols, int n_units, QUnitDev &u, float *partials,
                          unsigned *counter, int max_blocks, cudaStream_t st) {
    const int64_t per = rows / n_units;
    for (int b = 0; b < n_units; ++b)
        QNN_TRY(launch_quantize_matrix(w + b * per * cols, per, cols, cols, u.codes + b * per * u.ld, u.ld,
                                       u.params + b, u.sums + b * per, partials, counter, max_blocks, st));
    return QNN_OK;
}

}  // namespace

extern "C" int64_t qnn_lstm_param_count(const qnn_lstm_desc *d) {
    if (!valid_desc(d)) return -1;
    const int64_t H = d->hidden, P = d->proj, R = P > 0 ? P : H;
    int64_t n = 0;
    for (int l = 0; l < d->num_layers; ++l) {
        const int64_t Ik = l == 0 ? network_input_dim(d) : R;
        n += 4 * H * Ik + 4 * H * R + 4 * H + (P > 0 ? P * H : 0);
    }
    if (d->num_classes > 0) n += (int64_t)d->num_classes * R + d->num_classes;
    return n;
}

extern "C" void qnn_lstm_model_destroy(qnn_lstm_model *m) {
    if (!m) return;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(m->device);
    cudaDeviceSynchronize();
    cudaFree(m->weights);
    cudaFree(m->ws);
    cudaFree(m->sws);
    cudaFree(m->tcw);
    cudaFree(m->fws);
    for (cudaStream_t w : m->wave_st) cudaStreamDestroy(w);
    for (cudaEvent_t e : m->wave_ev) cudaEventDestroy(e);
    if (m->out_st) cudaStreamDestroy(m->out_st);
    if (m->cp_st) cudaStreamDestroy(m->cp_st);
    for (cudaEvent_t e : m->out_ev)
        if (e) cudaEventDestroy(e);
    cudaSetDevice(prev);
    delete m;
}

extern "C" qnn_status qnn_lstm_model_create(const qnn_lstm_desc *d, const float *params, qnn_lstm_model **out) {
    if (!out || !params || !valid_desc(d)) return QNN_ERR_INVALID_ARG;
    *out = nullptr;
    const int64_t L = d->num_layers, I = network_input_dim(d), H = d->hidden, P = d->proj, C = d->num_classes;
    const int64_t R = P > 0 ? P : H;
    if (I > QNN_K_MAX || H > QNN_K_MAX || R > QNN_K_MAX) return QNN_ERR_K_TOO_LARGE;
    const int64_t n_params = qnn_lstm_param_count(d);

    auto *m = new qnn_lstm_model();
    m->d = *d;
    m->L = L, m->I = I, m->H = H, m->P = P, m->C = C, m->R = R;
    m->frame_dim = d->input_dim;
    m->S = d->weight_blocks > 1 ? d->weight_blocks : 1;
    m->stack = d->stack > 1 ? d->stack : 1;
    m->stack_stride = d->stack_stride > 1 ? d->stack_stride : 1;
    cudaGetDevice(&m->device);
    m->layers.resize(L);

    // sizes
    const int64_t S = m->S;
    size_t bytes = 0;
    auto acct = [&](size_t n) { bytes = (size_t)round_up((int64_t)bytes, 256) + n; };
    for (int64_t l = 0; l < L; ++l) {
        const int64_t kin = l == 0 ? I : R;
        acct(4 * H * round_up(kin, 64)), acct(4 * H * 4), acct(4 * S * sizeof(qnn_qparams));
        acct(4 * H * round_up(R, 64)), acct(4 * H * 4), acct(4 * S * sizeof(qnn_qparams));
        acct(4 * H * 4);
        if (P > 0) acct(P * round_up(H, 64)), acct(P * 4), acct(S * sizeof(qnn_qparams));
    }
    if (C > 0) {
        acct(C * round_up(R, 64)), acct(C * 4), acct(S * sizeof(qnn_qparams)), acct(C * 4);
        if (d->output_mode == QNN_OUT_FLOAT) acct(C * R * 4);
    }
    acct((size_t)n_params * 4);  // device copy of the fp32 parameters (freed region reused later)
    bytes += 256;

    qnn_status st = QNN_OK;
    cudaStream_t s = nullptr;
    float *partials = nullptr;
    unsigned *counter = nullptr;
    const int max_blocks = 4 * sm_count();
    void *red = nullptr;
    if (cudaMalloc(&m->weights, bytes) != cudaSuccess) {
        delete m;
        return QNN_ERR_NO_MEMORY;
    }
    if (cudaMemset(m->weights, 0, bytes) != cudaSuccess) st = QNN_ERR_CUDA;
    Bump bp{reinterpret_cast<char *>(m->weights)};
    for (int64_t l = 0; l < L && st == QNN_OK; ++l) {
        LayerDev &ly = m->layers[l];
        ly.kin = l == 0 ? I : R;
        auto mk = [&](QUnitDev &u, int64_t rows, int64_t cols, int units) {
            u.rows = rows, u.cols = cols, u.ld = round_up(cols, 64), u.n_units = units;
            u.codes = bp.take<uint8_t>(rows * u.ld);
            u.sums = bp.take<int32_t>(rows);
            u.params = bp.take<qnn_qparams>(units);
        };
        mk(ly.wx, 4 * H, ly.kin, 4 * (int)m->S);
        mk(ly.wh, 4 * H, R, 4 * (int)m->S);
        ly.bias = bp.take<float>(4 * H);
        if (P > 0) mk(ly.wp, P, H, (int)m->S);
    }
    if (C > 0) {
        m->wo.rows = C, m->wo.cols = R, m->wo.ld = round_up(R, 64), m->wo.n_units = (int)m->S;
        m->wo.codes = bp.take<uint8_t>(C * m->wo.ld);
        m->wo.sums = bp.take<int32_t>(C);
        m->wo.params = bp.take<qnn_qparams>(m->S);
        m->bo = bp.take<float>(C);
        if (d->output_mode == QNN_OUT_FLOAT) m->wo_f = bp.take<float>(C * R);
    }
    float *pdev = bp.take<float>(n_params);
    if (st == QNN_OK && cudaMemcpy(pdev, params, n_params * 4, cudaMemcpyDefault) != cudaSuccess) st = QNN_ERR_CUDA;
    if (st == QNN_OK) st = scratch(kScratchReduce, 256 + sizeof(float) * 2 * (size_t)max_blocks, &red);
    if (st == QNN_OK) {
        counter = reinterpret_cast<unsigned *>(red);
        partials = reinterpret_cast<float *>(reinterpret_cast<char *>(red) + 256);
    }
    const float *q = pdev;
    for (int64_t l = 0; l < L && st == QNN_OK; ++l) {
        LayerDev &ly = m->layers[l];
        st = quantize_units(q, 4 * H, ly.kin, ly.wx.n_units, ly.wx, partials, counter, max_blocks, s);
        q += 4 * H * ly.kin;
        if (st == QNN_OK) st = quantize_units(q, 4 * H, R, ly.wh.n_units, ly.wh, partials, counter, max_blocks, s);
        q += 4 * H * R;
        if (st == QNN_OK && cudaMemcpy(ly.bias, q, 4 * H * 4, cudaMemcpyDeviceToDevice) != cudaSuccess)
            st = QNN_ERR_CUDA;
        q += 4 * H;
        if (P > 0) {
            if (st == QNN_OK) st = quantize_units(q, P, H, ly.wp.n_units, ly.wp, partials, counter, max_blocks, s);
            q += P * H;
        }
    }
    if (C > 0 && st == QNN_OK) {
        if (d->output_mode == QNN_OUT_QUANT)
            st = quantize_units(q, C, R, m->wo.n_units, m->wo, partials, counter, max_blocks, s);
        else if (cudaMemcpy(m->wo_f, q, C * R * 4, cudaMemcpyDeviceToDevice) != cudaSuccess)
            st = QNN_ERR_CUDA;
        q += C * R;
        if (st == QNN_OK && cudaMemcpy(m->bo, q, C * 4, cudaMemcpyDeviceToDevice) != cudaSuccess) st = QNN_ERR_CUDA;
    }
    if (st == QNN_OK && cudaDeviceSynchronize() != cudaSuccess) st = QNN_ERR_CUDA;
    if (st == QNN_OK) {
        qnn_status ds = qnn_device_status(nullptr);
        if (ds != QNN_OK) st = ds;
    }
    // host mirror of the unit parameters, in the documented order
    if (st == QNN_OK) {
        auto mirror = [&](const QUnitDev &u) {
            std::vector<qnn_qparams> tmp(u.n_units);
            if (cudaMemcpy(tmp.data(), u.params, u.n_units * sizeof(qnn_qparams), cudaMemcpyDeviceToHost) !=
                cudaSuccess)
                st = QNN_ERR_CUDA;
            m->host_params.insert(m->host_params.end(), tmp.begin(), tmp.end());
        };
        for (int64_t l = 0; l < L && st == QNN_OK; ++l) {
            const LayerDev &ly = m->layers[l];
            mirror(ly.wx);
            mirror(ly.wh);
            if (P > 0) mirror(ly.wp);
        }
        if (C > 0 && d->output_mode == QNN_OUT_QUANT && st == QNN_OK) mirror(m->wo);
    }
    if (st != QNN_OK) {
        qnn_lstm_model_destroy(m);
        return st;
    }
    *out = m;
    return QNN_OK;
}

extern "C" qnn_status qnn_lstm_model_weights(const qnn_lstm_model *m, uint8_t *codes_host, qnn_qparams *params_host,
                                             int64_t *n_units) {
    if (!m) return QNN_ERR_INVALID_ARG;
    if (n_units) *n_units = (int64_t)m->host_params.size();
    if (params_host) std::memcpy(params_host, m->host_params.data(), m->host_params.size() * sizeof(qnn_qparams));
    if (!codes_host) return QNN_OK;
    std::memset(codes_host, 0, (size_t)qnn_lstm_param_count(&m->d));
    const int64_t H = m->H, R = m->R, P = m->P, C = m->C;
    int64_t off = 0;
    auto copy_unit = [&](const QUnitDev &u) -> qnn_status {
        QNN_CUDA_TRY(cudaMemcpy2D(codes_host + off, u.cols, u.codes, u.ld, u.cols, u.rows, cudaMemcpyDeviceToHost));
        off += u.rows * u.cols;
        return QNN_OK;
    };
    for (int64_t l = 0; l < m->L; ++l) {
        const LayerDev &ly = m->layers[l];
        QNN_TRY(copy_unit(ly.wx));
        QNN_TRY(copy_unit(ly.wh));
        off += 4 * H;
        if (P > 0) QNN_TRY(copy_unit(ly.wp));
    }
    if (C > 0 && m->d.output_mode == QNN_OUT_QUANT) QNN_TRY(copy_unit(m->wo));
    (void)R;
    return QNN_OK;
}

namespace {

struct FwdPlan {
    int nc, np, bc, grid;
    size_t smem;
};

FwdPlan plan_recurrent(const qnn_lstm_model *m, int64_t B) {
    FwdPlan p{};
    const int sms = sm_count();
    const int64_t H = m->H, P = m->P, R = m->R;
    int nc = (int)round_up((H + sms - 1) / sms, 4);
    if (nc < 4) nc = 4;
    p.nc = nc;
    p.grid = (int)((H + nc - 1) / nc);
    p.np = P > 0 ? (int)round_up((P + p.grid - 1) / p.grid, 16) : 0;
    const int64_t ldh = round_up(R, 64), ldp = P > 0 ? round_up(H, 64) : 0;
    const int64_t arow = (ldh > ldp ? ldh : ldp) + kPad;
    int bc = (int)round_up(B, 16);
    if (bc > 64) bc = 64;
    auto smem_for = [&](int bcv) {
        const int ymax = 4 * nc > p.np ? 4 * nc : p.np;
        size_t s = (size_t)4 * nc * (ldh + kPad) + (P > 0 ? (size_t)p.np * (ldp + kPad) : 0) + (size_t)bcv * arow;
        s = (size_t)round_up((int64_t)s, 16) + (size_t)ymax * bcv * 4 + (size_t)bcv * 12;
        return s;
    };
    while (bc > 16 && smem_for(bc) > 200 * 1024) bc -= 16;
    p.bc = bc;
    p.smem = smem_for(bc);
    return p;
}

}  // namespace

namespace {

// Frame stacking (Sec. 4 frontend) ahead of the first layer: x [B][T][frame_dim] (host or device)
// -> the model's frontend workspace [B][T'][I]; *xs and *Tn receive the network input and T'.
qnn_status stack_input(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, cudaStream_t st, const float **xs,
                       int64_t *Tn) {
    const int64_t Tp = (T + m->stack_stride - 1) / m->stack_stride;
    const bool x_dev = is_device_ptr(x);
    const size_t raw = x_dev ? 0 : (size_t)round_up(B * T * m->frame_dim * 4, 256);
    const size_t need = raw + (size_t)(B * Tp * m->I * 4);
    if (need > m->fws_bytes) {
        if (m->fws) {
            QNN_CUDA_TRY(cudaStreamSynchronize(st));
            QNN_CUDA_TRY(cudaFree(m->fws));
            m->fws = nullptr;
            m->fws_bytes = 0;
        }
        QNN_CUDA_TRY(cudaMalloc(&m->fws, need));
        m->fws_bytes = need;
    }
    char *w = reinterpret_cast<char *>(m->fws);
    const float *src = x;
    if (!x_dev) {
        QNN_CUDA_TRY(cudaMemcpyAsync(w, x, B * T * m->frame_dim * 4, cudaMemcpyHostToDevice, st));
        src = reinterpret_cast<const float *>(w);
    }
    float *out = reinterpret_cast<float *>(w + raw);
    QNN_TRY(launch_stack_frames(src, B, T, m->frame_dim, (int)m->stack, (int)m->stack_stride, out, st));
    *xs = out;
    *Tn = Tp;
    return QNN_OK;
}

}  // namespace

namespace {

// qnn_lstm_forward with an optional copy of the output layer's logits ([B][T'][C], host or device).
qnn_status forward_impl(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *logits,
                        float *h_state, float *c_state, float *h_all, void *stream) {
    if (!m || B < 0 || T < 0) return QNN_ERR_INVALID_ARG;
    if (logits && m->C == 0) return QNN_ERR_INVALID_ARG;
    if (B == 0 || T == 0) return QNN_OK;
    if (!x || !y) return QNN_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    if (m->stack > 1 || m->stack_stride > 1) QNN_TRY(stack_input(m, x, B, T, st, &x, &T));
    const int64_t L = m->L, I = m->I, H = m->H, P = m->P, C = m->C, R = m->R;
    const int64_t rows = B * T;
    const int64_t ld_in = round_up(I > R ? I : R, 64);
    const int64_t ycols = C > 0 ? C : R;
    const bool x_dev = is_device_ptr(x), y_dev = is_device_ptr(y);
    const bool hs_dev = h_state && is_device_ptr(h_state), cs_dev = c_state && is_device_ptr(c_state);
    const bool ha_dev = h_all && is_device_ptr(h_all);
    // posteriors into pinned host memory: the softmax writes them there directly (no staging copy)
    float *const y_map = (!y_dev && C > 0) ? static_cast<float *>(host_mapped_ptr(y)) : nullptr;
    const PathChoice choice = path_choice();
    if (choice == PathChoice::kAuto || choice == PathChoice::kSmall) {
        bool used = false;
        QNN_TRY(small_path_forward(m, x, B, T, y, logits, h_state, c_state, h_all, st, &used));
        if (used) return QNN_OK;
        if (choice == PathChoice::kSmall) return QNN_ERR_INVALID_ARG;
    }
    // recurrence: tensor cores for large batches, else the persistent integer-MMA kernel
    const bool use_tc = tc_recurrence_supported(m) && (!ha_dev || (reinterpret_cast<uintptr_t>(h_all) & 15) == 0) &&
                        (choice == PathChoice::kTc || (choice == PathChoice::kAuto && B >= kTcMinBatch));
    if (choice == PathChoice::kTc && !use_tc) return QNN_ERR_INVALID_ARG;
    if (use_tc) QNN_TRY(tc_prepare(m));
    // the tensor-core recurrence computes each step's input product in its gate kernel (no px)
    const bool fused = use_tc && tc_input_fused(m);
    // layers as a wavefront on one stream each (every layer's recurrence state its own; the layer
    // outputs are kept whole only where they are read: the top layer, and every layer with h_all)
    const bool wave = fused && tc_stack_supported(m) && (!h_all || ha_dev);
    // the 8-bit output layer beside the recurrence (wavefront) when the posteriors go to pinned host
    // memory, so that they cross the host link while the recurrence runs (end to end 2.71M against
    // 2.39-2.49M frames/s at LSTMP 5 x 2048p512 B = 1024); with a device y the output layer runs
    // after the recurrence, where its one large product costs less SM time than the chunks' (4.49M
    // against 4.44M frames/s). QNN_OUT_OVERLAP=1 / 0 forces either way.
    const char *ov_env = std::getenv("QNN_OUT_OVERLAP");
    const bool ov_on = ov_env && std::strcmp(ov_env, "1") == 0, ov_off = ov_env && std::strcmp(ov_env, "0") == 0;
    const bool out_overlap = wave && C > 0 && m->d.output_mode == QNN_OUT_QUANT && m->wo16 && !ov_off &&
                             (ov_on || y_map != nullptr);
    // chunks of about 32768 rows (QNN_OUT_CHUNK sets the frames of a chunk); posteriors for pinned
    // host memory go through two device buffers of a chunk each, so that the copy engines carry
    // them to the host while the SMs go on with the recurrence (QNN_OUT_STAGE=0: the softmax writes
    // them to the host itself)
    const char *ce = std::getenv("QNN_OUT_CHUNK");
    const int64_t tchunk = std::min<int64_t>(
        T, ce && std::atoi(ce) > 0 ? std::atoi(ce) : std::max<int64_t>(1, (32768 + B - 1) / B));
    const char *se = std::getenv("QNN_OUT_STAGE");
    const bool out_stage = out_overlap && y_map && !(se && std::strcmp(se, "0") == 0);
    const FwdPlan plan = plan_recurrent(m, B);

    // workspace layout
    size_t need = 0;
    auto acct = [&](size_t n) {
        size_t at = (size_t)round_up((int64_t)need, 256);
        need = at + n;
        return at;
    };
    const size_t o_bar = acct(256);
    const size_t o_x = x_dev ? 0 : acct(rows * I * 4);
    const size_t o_codes = acct(rows * ld_in);
    const size_t o_prm = acct(rows * sizeof(qnn_qparams));
    const size_t o_rs = acct(rows * 4);
    const size_t o_px = acct(fused ? 0 : rows * 4 * H * 4);
    const size_t o_x16 = acct(fused ? tc_xwork_bytes(m, rows) : 0);
    const size_t o_seq0 = acct(rows * R * 4);
    const size_t o_seq1 = acct(rows * R * 4);
    const size_t o_h0 = acct(B * R * 4 * L);
    const size_t o_c = acct(B * H * 4);
    const size_t o_m = acct(P > 0 ? B * H * 4 : 0);
    const int64_t ldq = round_up(R > H ? R : H, 64);
    const size_t o_qc = acct(B * ldq);
    const size_t o_qp = acct(B * sizeof(qnn_qparams));
    const size_t o_qs = acct(B * 4);
    // logits: every row, or with the output layer beside the recurrence one chunk at a time (the
    // chunks' products, copies and softmaxes run in order on one stream)
    const size_t o_lg = acct(C > 0 ? (out_overlap ? std::min(rows, tchunk * B) : rows) * C * 4 : 0);
    const size_t o_y = (y_dev || y_map) ? 0 : acct(rows * ycols * 4);
    const size_t o_tc = use_tc ? acct(tc_work_bytes(m, B)) : 0;
    // wavefront: for layers 1 .. L - 1 (index l - 1) the input codes the previous layer writes and
    // the recurrence state; for every layer l (index l) the step's output when the layer's outputs
    // are not kept
    const int64_t kxr = round_up(R, 64);
    std::vector<size_t> o_wx16, o_wprm, o_wrs, o_wc, o_wm, o_wtc, o_wout;
    if (wave) {
        for (int64_t l = 1; l < L; ++l) {
            o_wx16.push_back(acct(rows * kxr * 2));
            o_wprm.push_back(acct(rows * sizeof(qnn_qparams)));
            o_wrs.push_back(acct(rows * 4));
            o_wc.push_back(acct(B * H * 4));
            o_wm.push_back(acct(B * H * 4));
            o_wtc.push_back(acct(tc_work_bytes(m, B)));
        }
        for (int64_t l = 0; l < L; ++l) o_wout.push_back(acct(B * R * 4));
    }
    // the output layer's input codes, which the top layer's step kernels write time-major (row
    // t B + b), with their units and code sums; the staged posteriors
    const size_t o_ox16 = out_overlap ? acct(rows * kxr * 2) : 0;
    const size_t o_oprm = out_overlap ? acct(rows * sizeof(qnn_qparams)) : 0;
    const size_t o_ors = out_overlap ? acct(rows * 4) : 0;
    const size_t o_ystage = out_stage ? acct(2 * tchunk * B * C * 4) : 0;
    if (need > m->ws_bytes) {
        if (m->ws) {
            QNN_CUDA_TRY(cudaStreamSynchronize(st));
            QNN_CUDA_TRY(cudaFree(m->ws));
            m->ws = nullptr;
            m->ws_bytes = 0;
        }
        QNN_CUDA_TRY(cudaMalloc(&m->ws, need));
        m->ws_bytes = need;
    }
    char *ws = reinterpret_cast<char *>(m->ws);
    unsigned *bar = reinterpret_cast<unsigned *>(ws + o_bar);
    int *abort_flag = reinterpret_cast<int *>(ws + o_bar + 128);
    const float *xd = x;
    if (!x_dev) {
        QNN_CUDA_TRY(cudaMemcpyAsync(ws + o_x, x, rows * I * 4, cudaMemcpyHostToDevice, st));
        xd = reinterpret_cast<const float *>(ws + o_x);
    }
    uint8_t *codes = reinterpret_cast<uint8_t *>(ws + o_codes);
    qnn_qparams *prm = reinterpret_cast<qnn_qparams *>(ws + o_prm);
    int32_t *rs = reinterpret_cast<int32_t *>(ws + o_rs);
    float *px = reinterpret_cast<float *>(ws + o_px);
    float *seq[2] = {reinterpret_cast<float *>(ws + o_seq0), reinterpret_cast<float *>(ws + o_seq1)};
    float *h0 = reinterpret_cast<float *>(ws + o_h0);
    float *cbuf = reinterpret_cast<float *>(ws + o_c);
    float *mbuf = P > 0 ? reinterpret_cast<float *>(ws + o_m) : nullptr;
    float *lg = C > 0 ? reinterpret_cast<float *>(ws + o_lg) : nullptr;
    float *yd = y_dev ? y : y_map ? y_map : reinterpret_cast<float *>(ws + o_y);

    if (h_state)
        QNN_CUDA_TRY(cudaMemcpyAsync(h0, h_state, L * B * R * 4, cudaMemcpyDefault, st));
    else
        QNN_CUDA_TRY(cudaMemsetAsync(h0, 0, L * B * R * 4, st));

    int *status = nullptr;
    QNN_TRY(status_word(&status));
    static bool configured = false;
    if (!configured) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstm_recurrent_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          200 * 1024 + 4096));
        configured = true;
    }

    const float *in = xd;
    int64_t kin = I;
    if (wave) {
        // one stream per layer (all at the default priority: with the layers above the output
        // layer's stream, the output work waited for the end of the recurrence, and with the output
        // layer above the layers, the recurrence slowed more than the output work gained), and the
        // events: L - 1 layer edges, a fork, L joins
        if ((int64_t)m->wave_st.size() != L) {
            for (cudaStream_t w : m->wave_st) cudaStreamDestroy(w);
            for (cudaEvent_t e : m->wave_ev) cudaEventDestroy(e);
            m->wave_st.assign((size_t)L, nullptr);
            m->wave_ev.assign((size_t)(2 * L), nullptr);
            for (auto &w : m->wave_st) QNN_CUDA_TRY(cudaStreamCreateWithFlags(&w, cudaStreamNonBlocking));
            for (auto &e : m->wave_ev) QNN_CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
        }
        std::vector<cudaStream_t> streams(m->wave_st.begin(), m->wave_st.end());
        const cudaEvent_t *edges = m->wave_ev.data(), fork = m->wave_ev[(size_t)(L - 1)];
        const cudaEvent_t *joins = m->wave_ev.data() + L;  // L of them
        std::vector<TcStackLayer> sl((size_t)L);
        std::vector<const float *> hsrc((size_t)L);
        std::vector<int64_t> hsrc_ld((size_t)L);
        for (int64_t l = 0; l < L; ++l) {
            TcStackLayer &y = sl[(size_t)l];
            const bool keep = ha_dev || l == L - 1;  // outputs kept whole
            y.h0 = h0 + l * B * R;
            y.cbuf = l == 0 ? cbuf : reinterpret_cast<float *>(ws + o_wc[(size_t)(l - 1)]);
            y.mbuf = l == 0 ? mbuf : reinterpret_cast<float *>(ws + o_wm[(size_t)(l - 1)]);
            y.work = l == 0 ? ws + o_tc : ws + o_wtc[(size_t)(l - 1)];
            if (keep) {
                y.out = ha_dev ? h_all + l * rows * R : seq[0];
                y.out_t = R, y.out_b = T * R;
            } else {
                y.out = reinterpret_cast<float *>(ws + o_wout[(size_t)l]);
                y.out_t = 0, y.out_b = R;
            }
            hsrc[(size_t)l] = y.out + (T - 1) * y.out_t;
            hsrc_ld[(size_t)l] = y.out_b;
            if (l == 0) {
                y.fx.in = xd, y.fx.kin = I, y.fx.x16 = reinterpret_cast<__half *>(ws + o_x16), y.fx.prm = prm;
                y.fx.rs = rs;
            } else {
                y.fx.in = nullptr, y.fx.kin = R;
                y.fx.x16 = reinterpret_cast<__half *>(ws + o_wx16[(size_t)(l - 1)]);
                y.fx.prm = reinterpret_cast<qnn_qparams *>(ws + o_wprm[(size_t)(l - 1)]);
                y.fx.rs = reinterpret_cast<int32_t *>(ws + o_wrs[(size_t)(l - 1)]);
            }
            if (c_state)
                QNN_CUDA_TRY(cudaMemcpyAsync(y.cbuf, c_state + l * B * H, B * H * 4, cudaMemcpyDefault, st));
            else
                QNN_CUDA_TRY(cudaMemsetAsync(y.cbuf, 0, B * H * 4, st));
        }
        // the layer streams follow everything queued so far on the caller's stream
        QNN_CUDA_TRY(cudaEventRecord(fork, st));
        for (int64_t l = 0; l < L; ++l) QNN_CUDA_TRY(cudaStreamWaitEvent(streams[(size_t)l], fork, 0));
        // The output layer on chunks of frames as the top layer completes them, on its own stream:
        // the product on the codes the top layer's step kernels write (time-major), logits
        // time-major in lg, then the softmax into y's sequence-major rows.
        TcFusedInput oc;
        std::function<qnn_status(int64_t)> after_top;
        int64_t t0 = 0;
        if (out_overlap) {
            if (!m->out_st) {
                QNN_CUDA_TRY(cudaStreamCreateWithFlags(&m->out_st, cudaStreamNonBlocking));
                QNN_CUDA_TRY(cudaStreamCreateWithFlags(&m->cp_st, cudaStreamNonBlocking));
                for (auto &e : m->out_ev) QNN_CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
            }
            QNN_CUDA_TRY(cudaStreamWaitEvent(m->out_st, fork, 0));
            oc.x16 = reinterpret_cast<__half *>(ws + o_ox16), oc.kin = R;
            oc.prm = reinterpret_cast<qnn_qparams *>(ws + o_oprm), oc.rs = reinterpret_cast<int32_t *>(ws + o_ors);
            const cudaStream_t top = streams[(size_t)(L - 1)], os = m->out_st, cs = m->cp_st;
            float *const ystage = out_stage ? reinterpret_cast<float *>(ws + o_ystage) : nullptr;
            after_top = [&, top, os, cs, ystage](int64_t t) -> qnn_status {
                if (t + 1 - t0 < tchunk && t + 1 < T) return QNN_OK;
                const int64_t t1 = t + 1, rc = (t1 - t0) * B;
                QNN_CUDA_TRY(cudaEventRecord(m->out_ev[0], top));
                QNN_CUDA_TRY(cudaStreamWaitEvent(os, m->out_ev[0], 0));
                TcOperands op;
                QNN_TRY(tc_operands(&op, oc.x16 + t0 * B * kxr, rc, m->wo16, C, kxr, tc_pick_bn(rc, C, kxr)));
                QNN_TRY(tc_linear(op, oc.prm + t0 * B, 1, oc.rs + t0 * B, R, m->wo.params, C / m->S, m->wo.sums, m->bo,
                                  lg, C, nullptr, os));
                if (logits)
                    for (int64_t tt = t0; tt < t1; ++tt)
                        QNN_CUDA_TRY(cudaMemcpy2DAsync(logits + tt * C, T * C * 4, lg + (tt - t0) * B * C, C * 4, C * 4, B,
                                                       cudaMemcpyDefault, os));
                if (ystage) {
                    // softmax into the chunk's buffer (sequence-major within the chunk) once the copy
                    // out of that buffer two chunks ago is done, then the copy into y's rows
                    const int64_t k = t0 / tchunk, n = t1 - t0;
                    float *const sb = ystage + (k & 1) * tchunk * B * C;
                    if (k >= 2) QNN_CUDA_TRY(cudaStreamWaitEvent(os, m->out_ev[4 + (k & 1)], 0));
                    QNN_TRY(launch_softmax_rows(lg, rc, C, sb, os, B, n, 0));
                    QNN_CUDA_TRY(cudaEventRecord(m->out_ev[2 + (k & 1)], os));
                    QNN_CUDA_TRY(cudaStreamWaitEvent(cs, m->out_ev[2 + (k & 1)], 0));
                    QNN_CUDA_TRY(cudaMemcpy2DAsync(y + t0 * C, T * C * 4, sb, n * C * 4, n * C * 4, B,
                                                   cudaMemcpyDeviceToHost, cs));
                    QNN_CUDA_TRY(cudaEventRecord(m->out_ev[4 + (k & 1)], cs));
                } else {
                    QNN_TRY(launch_softmax_rows(lg, rc, C, yd, os, B, T, t0));
                }
                t0 = t1;
                return QNN_OK;
            };
        }
        QNN_TRY(tc_stack_recurrence(m, sl.data(), B, T, streams.data(), edges, out_overlap ? &oc : nullptr,
                                    after_top));
        // ... and the caller's stream follows every layer (and the output layer's stream)
        for (int64_t l = 0; l < L; ++l) {
            QNN_CUDA_TRY(cudaEventRecord(joins[l], streams[(size_t)l]));
            QNN_CUDA_TRY(cudaStreamWaitEvent(st, joins[l], 0));
        }
        if (out_overlap) {
            QNN_CUDA_TRY(cudaEventRecord(m->out_ev[1], m->out_st));
            QNN_CUDA_TRY(cudaStreamWaitEvent(st, m->out_ev[1], 0));
        }
        if (out_stage) {
            QNN_CUDA_TRY(cudaEventRecord(m->out_ev[6], m->cp_st));
            QNN_CUDA_TRY(cudaStreamWaitEvent(st, m->out_ev[6], 0));
        }
        for (int64_t l = 0; l < L; ++l) {
            if (h_state)  // final h of the layer: its output at the last frame
                QNN_CUDA_TRY(cudaMemcpy2DAsync(h_state + l * B * R, R * 4, hsrc[(size_t)l], hsrc_ld[(size_t)l] * 4,
                                               R * 4, B, cudaMemcpyDefault, st));
            if (c_state)
                QNN_CUDA_TRY(cudaMemcpyAsync(c_state + l * B * H, sl[(size_t)l].cbuf, B * H * 4, cudaMemcpyDefault, st));
        }
        in = sl[(size_t)(L - 1)].out;
        kin = R;
    }
    for (int64_t l = 0; l < L && !wave; ++l) {
        const LayerDev &ly = m->layers[l];
        if (!fused) {
            // 1. quantize every frame of the layer input (one unit per row)
            QNN_TRY(launch_quantize_rows(in, rows, kin, kin, codes, ld_in, prm, rs, st));
            // 2. batched input product, recovered, plus bias
            QNN_TRY(launch_qgemm(codes, ld_in, prm, QNN_PER_ROW, rs, rows, kin, ly.wx.codes, ly.wx.ld, ly.wx.params,
                                 H / m->S, ly.wx.sums, 4 * H, ly.bias, px, 4 * H, nullptr, st));
        }
        // 3. recurrence
        float *outl = (ha_dev ? h_all + l * rows * R : seq[l & 1]);
        if (c_state)
            QNN_CUDA_TRY(cudaMemcpyAsync(cbuf, c_state + l * B * H, B * H * 4, cudaMemcpyDefault, st));
        else
            QNN_CUDA_TRY(cudaMemsetAsync(cbuf, 0, B * H * 4, st));
        if (use_tc) {
            TcFusedInput fx;
            fx.in = in, fx.kin = kin, fx.x16 = reinterpret_cast<__half *>(ws + o_x16), fx.prm = prm, fx.rs = rs;
            QNN_TRY(tc_layer_recurrence(m, l, fused ? nullptr : px, h0 + l * B * R, cbuf, outl, mbuf, B, T,
                                        ws + o_tc, st, fused ? &fx : nullptr));
        } else {
            QNN_CUDA_TRY(cudaMemsetAsync(bar, 0, 256, st));
            RecArgs a{};
            a.wh = ly.wh.codes, a.wh_sum = ly.wh.sums, a.wh_p = ly.wh.params;
            a.px = px, a.h0 = h0 + l * B * R, a.cbuf = cbuf, a.out = outl;
            a.wp = P > 0 ? ly.wp.codes : nullptr, a.wp_sum = P > 0 ? ly.wp.sums : nullptr;
            a.wp_p = P > 0 ? ly.wp.params : nullptr, a.mbuf = mbuf;
            a.bar = bar, a.abort_flag = abort_flag, a.status = status;
            a.B = (int)B, a.T = (int)T, a.H = (int)H, a.R = (int)R, a.P = (int)P;
            a.ldh = (int)ly.wh.ld, a.ldp = P > 0 ? (int)ly.wp.ld : 0;
            a.nc = plan.nc, a.np = plan.np, a.bc = plan.bc;
            a.qcodes = reinterpret_cast<uint8_t *>(ws + o_qc);
            a.qprm = reinterpret_cast<qnn_qparams *>(ws + o_qp);
            a.qsum = reinterpret_cast<int *>(ws + o_qs);
            a.ldq = (int)ldq;
            a.distq = B >= kDistQuantMinBatch;  // below this, each block quantizing its rows is cheaper
            a.ups = (int)m->S, a.cpu = (int)(H / m->S), a.ppu = P > 0 ? (int)(P / m->S) : 1;
            void *args[] = {&a};
            ProfScope prof("lstm_recurrent", st);
            cudaError_t e = cudaLaunchCooperativeKernel((const void *)lstm_recurrent_kernel, dim3(plan.grid),
                                                        dim3(kRecThreads), args, plan.smem, st);
            if (e == cudaErrorCooperativeLaunchTooLarge) {
                cudaGetLastError();
                return QNN_ERR_NO_COOP;
            }
            QNN_CUDA_TRY(e);
        }
        if (h_state) {  // final h of this layer = its output at the last frame
            QNN_CUDA_TRY(cudaMemcpy2DAsync(h_state + l * B * R, R * 4, outl + (T - 1) * R, T * R * 4, R * 4, B,
                                           cudaMemcpyDefault, st));
        }
        if (c_state) QNN_CUDA_TRY(cudaMemcpyAsync(c_state + l * B * H, cbuf, B * H * 4, cudaMemcpyDefault, st));
        if (h_all && !ha_dev)
            QNN_CUDA_TRY(cudaMemcpyAsync(h_all + l * rows * R, outl, rows * R * 4, cudaMemcpyDeviceToHost, st));
        in = outl;
        kin = R;
    }
    if (C > 0 && out_overlap) {
        // done beside the recurrence
    } else if (C > 0) {
        if (m->d.output_mode == QNN_OUT_QUANT) {
            QNN_TRY(launch_quantize_rows(in, rows, R, R, codes, ld_in, prm, rs, st));
            QNN_TRY(launch_qgemm(codes, ld_in, prm, QNN_PER_ROW, rs, rows, R, m->wo.codes, m->wo.ld, m->wo.params,
                                 C / m->S, m->wo.sums, C, m->bo, lg, C, nullptr, st));
        } else {
            dim3 grid((unsigned)((C + 31) / 32), (unsigned)((rows + 31) / 32));
            ProfScope prof("float_linear", st);
            float_linear_kernel<<<grid, 256, 0, st>>>(in, rows, (int)R, m->wo_f, (int)C, m->bo, lg);
            QNN_CUDA_TRY(cudaGetLastError());
        }
        if (logits) QNN_CUDA_TRY(cudaMemcpyAsync(logits, lg, rows * C * 4, cudaMemcpyDefault, st));
        QNN_TRY(launch_softmax_rows(lg, rows, C, yd, st));
    } else {
        QNN_CUDA_TRY(cudaMemcpyAsync(yd, in, rows * R * 4, cudaMemcpyDeviceToDevice, st));
    }
    if (!y_dev && !y_map) QNN_CUDA_TRY(cudaMemcpyAsync(y, yd, rows * ycols * 4, cudaMemcpyDeviceToHost, st));
    (void)hs_dev;
    (void)cs_dev;
    return QNN_OK;
}

}  // namespace

extern "C" qnn_status qnn_lstm_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y,
                                       float *h_state, float *c_state, float *h_all, void *stream) {
    return forward_impl(m, x, B, T, y, nullptr, h_state, c_state, h_all, stream);
}

extern "C" qnn_status qnn_lstm_forward_logits(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y,
                                              float *logits, float *h_state, float *c_state, float *h_all,
                                              void *stream) {
    return forward_impl(m, x, B, T, y, logits, h_state, c_state, h_all, stream);
}
