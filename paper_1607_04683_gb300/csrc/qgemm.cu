// qgemm.cu — eq. (1): 8-bit code products with 32-bit accumulators, offset terms and recovery.
//
// Datapath. sm_103a accepts no 8-bit integer tcgen05 MMA, so the exact integer product runs on
// the warp-level integer tensor-core instruction mma.sync m16n8k32 (u8 x u8 -> s32). Tiles of
// 128 x 128 outputs, K in steps of 64 bytes, a four-stage cp.async pipeline into padded shared
// memory rows (80-byte stride: the 16-byte ldmatrix rows of eight consecutive rows hit disjoint
// banks), ldmatrix fragment loads, eight warps of 64 x 32 outputs each.
//
// Epilogue (fused): S = acc + zw*rsA[m] + za[m]*csW[n] + K*za*zw in 64-bit integers (eq. 1 with
// V'' = V' + round(Q Vmin)), then y = S / (Qa Qw) + bias (eq. 3 recovery and Fig. 1's bias), and
// optionally the raw accumulator.
#include <cstdlib>
#include <cstring>

#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4, THREADS = 256;
constexpr int SROW = BK + 16;  // padded shared-memory row (bytes)
constexpr int TILE_BYTES = BM * SROW;  // same for the BN side
constexpr int SMEM_BYTES = STAGES * 2 * TILE_BYTES;

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
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

// Copies a BM x BK byte tile (rows r0.., bytes k0..) of a row-major u8 matrix into shared memory.
// Bytes past `rows` or `K` are zero so they add nothing to the integer sums.
template <bool kAligned>
__device__ __forceinline__ void load_tile(uint32_t sdst, const uint8_t *__restrict__ g, int64_t ld, int64_t rows,
                                          int64_t r0, int64_t K, int64_t k0) {
#pragma unroll
    for (int i = 0; i < (BM * BK / 16) / THREADS; ++i) {
        const int c = threadIdx.x + i * THREADS;
        const int r = c >> 2, ch = c & 3;
        const int64_t gr = r0 + r, gk = k0 + ch * 16;
        int valid = 0;
        if (gr < rows) {
            int64_t rem = K - gk;
            valid = rem <= 0 ? 0 : (rem >= 16 ? 16 : (int)rem);
        }
        const uint32_t d = sdst + r * SROW + ch * 16;
        if (kAligned) {
            const uint8_t *src = valid ? g + gr * ld + gk : g;
            cp_async16(d, src, valid);
        } else {
            uint32_t w[4] = {0, 0, 0, 0};
            const uint8_t *src = g + gr * ld + gk;
            for (int b = 0; b < valid; ++b) w[b >> 2] |= (uint32_t)__ldg(src + b) << ((b & 3) * 8);
            asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(d), "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]));
        }
    }
}

template <bool kAligned>
__global__ void __launch_bounds__(THREADS) qgemm_imma_kernel(
    const uint8_t *__restrict__ A, int64_t lda, const qnn_qparams *__restrict__ pa, int a_per_row,
    const int32_t *__restrict__ rsA, int64_t M, int64_t K, const uint8_t *__restrict__ W, int64_t ldw,
    const qnn_qparams *__restrict__ pw, int64_t rows_per_block, const int32_t *__restrict__ csW, int64_t N,
    const float *__restrict__ bias, float *__restrict__ Y, int64_t ldy, int32_t *__restrict__ acc_out) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wm = warp >> 2, wn = warp & 3;  // 2 x 4 warps, 64 x 32 outputs each
    const uint32_t s0 = smem_u32(smem);
    auto sa = [&](int s) { return s0 + s * 2 * TILE_BYTES; };
    auto sw = [&](int s) { return s0 + s * 2 * TILE_BYTES + TILE_BYTES; };

    const int KT = (int)((K + BK - 1) / BK);
#pragma unroll
    for (int s = 0; s < STAGES - 1; ++s) {
        if (s < KT) {
            load_tile<kAligned>(sa(s), A, lda, M, m0, K, (int64_t)s * BK);
            load_tile<kAligned>(sw(s), W, ldw, N, n0, K, (int64_t)s * BK);
        }
        cp_async_commit();
    }

    int acc[4][4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int k = 0; k < 4; ++k) acc[i][j][k] = 0;

    for (int kt = 0; kt < KT; ++kt) {
        cp_async_wait<STAGES - 2>();
        __syncthreads();
        const int pf = kt + STAGES - 1;
        if (pf < KT) {
            load_tile<kAligned>(sa(pf % STAGES), A, lda, M, m0, K, (int64_t)pf * BK);
            load_tile<kAligned>(sw(pf % STAGES), W, ldw, N, n0, K, (int64_t)pf * BK);
        }
        cp_async_commit();
        const uint32_t ta = sa(kt % STAGES), tw = sw(kt % STAGES);
#pragma unroll
        for (int kk = 0; kk < BK; kk += 32) {
            uint32_t af[4][4], bf[4][2];
#pragma unroll
            for (int mi = 0; mi < 4; ++mi) {
                const int r = wm * 64 + mi * 16 + (lane & 15);
                ldmatrix_x4(ta + r * SROW + kk + (lane >> 4) * 16, af[mi][0], af[mi][1], af[mi][2], af[mi][3]);
            }
#pragma unroll
            for (int nj = 0; nj < 2; ++nj) {
                const int r = wn * 32 + nj * 16 + (lane & 7) + ((lane >> 4) << 3);
                ldmatrix_x4(tw + r * SROW + kk + ((lane >> 3) & 1) * 16, bf[2 * nj][0], bf[2 * nj][1],
                            bf[2 * nj + 1][0], bf[2 * nj + 1][1]);
            }
#pragma unroll
            for (int mi = 0; mi < 4; ++mi)
#pragma unroll
                for (int ni = 0; ni < 4; ++ni) mma_u8(acc[mi][ni], af[mi], bf[ni][0], bf[ni][1]);
        }
    }
    cp_async_wait<0>();

    // Epilogue: offsets, recovery, bias.
    const int g = lane >> 2, tq = lane & 3;
    const int Ki = (int)K;
#pragma unroll
    for (int mi = 0; mi < 4; ++mi) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t m = m0 + wm * 64 + mi * 16 + g + h * 8;
            if (m >= M) continue;
            const qnn_qparams qa = pa[a_per_row ? m : 0];
            const int ra = rsA[m];
#pragma unroll
            for (int ni = 0; ni < 4; ++ni) {
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int64_t n = n0 + wn * 32 + ni * 8 + tq * 2 + e;
                    if (n >= N) continue;
                    const qnn_qparams qw = pw[n / rows_per_block];
                    const int a = acc[mi][ni][h * 2 + e];
                    const long long S = offset_product(a, qa.z, qw.z, ra, csW[n], Ki);
                    float y = recover_product(S, qa.Q, qw.Q);
                    if (bias) y = __fadd_rn(y, bias[n]);
                    if (Y) Y[m * ldy + n] = y;
                    if (acc_out) acc_out[m * N + n] = a;
                }
            }
        }
    }
}

}  // namespace

qnn_status launch_qgemm_imma(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA,
                             int64_t M, int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw,
                             int64_t rows_per_block, const int32_t *csW, int64_t N, const float *bias, float *Y,
                             int64_t ldy, int32_t *acc_out, cudaStream_t st) {
    if (M == 0 || N == 0) return QNN_OK;
    static bool configured[2] = {false, false};
    const bool aligned = ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(W)) & 15) == 0 &&
                         lda % 16 == 0 && ldw % 16 == 0;
    auto kern = aligned ? qgemm_imma_kernel<true> : qgemm_imma_kernel<false>;
    if (!configured[aligned]) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES));
        configured[aligned] = true;
    }
    dim3 grid((unsigned)((N + BN - 1) / BN), (unsigned)((M + BM - 1) / BM));
    ProfScope prof("qgemm_imma", st);
    kern<<<grid, THREADS, SMEM_BYTES, st>>>(A, lda, pa, ga == QNN_PER_ROW, rsA, M, K, W, ldw, pw, rows_per_block, csW,
                                            N, bias, Y, ldy, acc_out);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

// Datapath choice: the tcgen05 path runs whole 128 x 256 tiles at the fp16 tensor rate (after
// centering both operands into fp16 scratch); below one tile of rows the integer MMA path, which
// needs no conversion, is used. QNN_QGEMM=imma or =tc forces one (tests compare the two).
qnn_status launch_qgemm(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA, int64_t M,
                        int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw, int64_t rows_per_block,
                        const int32_t *csW, int64_t N, const float *bias, float *Y, int64_t ldy, int32_t *acc_out,
                        cudaStream_t st) {
    if (M == 0 || N == 0) return QNN_OK;
    const char *force = std::getenv("QNN_QGEMM");
    bool tc = M >= 128;
    if (force && std::strcmp(force, "imma") == 0) tc = false;
    if (force && std::strcmp(force, "tc") == 0) tc = true;
    if (tc) {
        void *ws = nullptr;
        QNN_TRY(scratch(kScratchTc, tc_scratch_bytes(M, N, K), &ws));
        return launch_qgemm_tc(A, lda, pa, ga, rsA, M, K, W, ldw, pw, rows_per_block, csW, N, bias, Y, ldy, acc_out, ws,
                               st);
    }
    return launch_qgemm_imma(A, lda, pa, ga, rsA, M, K, W, ldw, pw, rows_per_block, csW, N, bias, Y, ldy, acc_out, st);
}

}  // namespace qnn

using namespace qnn;

extern "C" qnn_status qnn_qmatmul(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA,
                                  int64_t M, int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw,
                                  int64_t n_blocks, const int32_t *csW, int64_t N, const float *bias, float *Y,
                                  int64_t ldy, int32_t *acc_out, void *stream) {
    if (M < 0 || N <= 0 || K <= 0 || lda < K || ldw < K || n_blocks <= 0 || N % n_blocks) return QNN_ERR_INVALID_ARG;
    if (ga != QNN_PER_MATRIX && ga != QNN_PER_ROW) return QNN_ERR_INVALID_ARG;
    if (K > QNN_K_MAX) return QNN_ERR_K_TOO_LARGE;
    if (Y && ldy < N) return QNN_ERR_INVALID_ARG;
    if (M == 0) return QNN_OK;
    if (!is_device_ptr(A) || !is_device_ptr(pa) || !is_device_ptr(rsA) || !is_device_ptr(W) || !is_device_ptr(pw) ||
        !is_device_ptr(csW) || (bias && !is_device_ptr(bias)) || (Y && !is_device_ptr(Y)) ||
        (acc_out && !is_device_ptr(acc_out)))
        return QNN_ERR_INVALID_ARG;
    return launch_qgemm(A, lda, pa, ga, rsA, M, K, W, ldw, pw, N / n_blocks, csW, N, bias, Y, ldy, acc_out,
                        as_stream(stream));
}
