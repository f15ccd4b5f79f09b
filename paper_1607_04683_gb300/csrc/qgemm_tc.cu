// qgemm_tc.cu — eq. (1) on the sm_103a tcgen05 tensor cores, exactly.
//
// sm_103a has no 8-bit integer tcgen05 MMA, but the integer product can still run on the fp16
// datapath without any rounding: a code c in [0, 255] is stored centered, s = c - 128 in
// [-128, 127], which fp16 represents exactly; every product s_a s_w has |s_a s_w| <= 2^14, also
// exact, and a sum of at most 1024 of them stays within 2^24 in magnitude, where every integer is
// an fp32 value. The fp32 accumulator in tensor memory therefore holds the exact integer
//   P = sum_k s_a s_w   and the raw code product is   acc = P + 128 (rowsum(A) + rowsum(W)) - 128^2 K,
// from which the epilogue applies eq. (1)'s offsets and the eq. (3) recovery as the other paths do.
// K above 1024 is split into chunks of at most 1024; each chunk accumulates into its own tensor
// memory buffer (two, alternating) and is drained into int32 registers as soon as it completes.
//
// Tile: 128 rows of A x 256 rows of W per block, K in steps of 64 fp16 (128-byte rows, TMA with
// 128-byte swizzle into a 4-stage shared-memory ring). Warp 0 issues TMA, warp 1 issues the MMAs
// (tcgen05.mma.cta_group::1.kind::f16, M 128 N 256 K 16) and owns the tensor memory, warps 2-9 are
// the epilogue (each tensor-memory lane quarter is read by two warps, one per column half).
// Every wait is bounded in time; a wait that gives up records QNN_ERR_TIMEOUT and the block skips
// ahead, waits (bounded) for its own copies in flight, frees its tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <cstdlib>
#include <algorithm>
#include <mutex>

#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int TBM = 128, TBN = 256, TBK = 64;     // fp16 elements per k-block (128 bytes)
constexpr int TSTAGES = 3;
constexpr int A_BYTES = TBM * TBK * 2;            // 16 KB
constexpr int B_BYTES = TBN * TBK * 2;            // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TC_THREADS = 10 * 32;
constexpr int KCHUNK = 1024;                      // exact fp32 accumulation bound (see above)
constexpr int TMEM_COLS = 512;                    // two 128 x 256 fp32 accumulators
constexpr unsigned long long TC_WAIT_NS = 2000000000ull;

struct TcArgs {
    const qnn_qparams *pa;
    int a_per_row;
    const int32_t *rsA;
    const qnn_qparams *pw;
    int64_t rows_per_block;
    const int32_t *csW;
    const float *bias;
    float *Y;
    int64_t ldy;
    int32_t *acc_out;
    int64_t M, N;
    int K;      // true K
    int KB;     // k-blocks of 64
    int *status;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }
__device__ __forceinline__ unsigned long long gtime() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mb_init(uint32_t b, unsigned n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(b), "r"(n) : "memory");
}
__device__ __forceinline__ void mb_expect(uint32_t b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mb_try(uint32_t b, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(b), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait; false (and QNN_ERR_TIMEOUT recorded) if the phase did not complete in time.
__device__ __forceinline__ bool mb_wait(uint32_t b, unsigned parity, int *status) {
    if (mb_try(b, parity)) return true;
    const unsigned long long t0 = gtime();
    int spins = 0;
    while (!mb_try(b, parity)) {
        if (++spins >= 256) {
            spins = 0;
            if (gtime() - t0 > TC_WAIT_NS) {
                record_status(status, QNN_ERR_TIMEOUT);
                return false;
            }
        }
    }
    return true;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
            dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
        : "memory");
}

// Shared-memory matrix descriptor of a K-major tile with 128-byte swizzle: rows of 128 bytes,
// 8-row groups 1024 bytes apart (stride byte offset), tcgen05 descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFF) >> 4);        // start address
    d |= (uint64_t)1 << 16;                          // leading byte offset (unused with this swizzle)
    d |= (uint64_t)(1024 >> 4) << 32;                // stride byte offset
    d |= (uint64_t)1 << 46;                          // version
    d |= (uint64_t)2 << 61;                          // 128-byte swizzle
    return d;
}

// Instruction descriptor: fp32 accumulator, fp16 A and B, both K-major, M = 128, N = 256.
constexpr uint32_t IDESC = (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(TBN >> 3) << 17) | ((uint32_t)(TBM >> 4) << 24);

__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(IDESC), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

template <int N>
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[N]);
template <>
__device__ __forceinline__ void tmem_ld32<32>(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
        "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__global__ void __launch_bounds__(TC_THREADS, 1) qgemm_tc_kernel(const __grid_constant__ CUtensorMap mapA,
                                                                 const __grid_constant__ CUtensorMap mapW,
                                                                 const TcArgs args) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte alignment for the swizzled tiles
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    int *stage_out = reinterpret_cast<int *>(smem + TSTAGES * STAGE_BYTES);        // [8 warps][32][33]
    int *row_c = stage_out + 8 * 32 * 33;                                          // [8 warps][3][32]
    uint64_t *bars = reinterpret_cast<uint64_t *>(row_c + 8 * 3 * 32);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * TSTAGES + 4);
    const uint32_t full0 = su32(bars), empty0 = su32(bars + TSTAGES), chunk0 = su32(bars + 2 * TSTAGES),
                   drained0 = su32(bars + 2 * TSTAGES + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int KB = args.KB;
    const int kpc = KCHUNK / TBK;  // k-blocks per chunk (16)
    const int nchunks = (KB + kpc - 1) / kpc;
    const int tiles_n = (int)((args.N + TBN - 1) / TBN);
    const int64_t tiles = (int64_t)((args.M + TBM - 1) / TBM) * tiles_n;
    __shared__ int s_abort;

    if (threadIdx.x == 0) {
        s_abort = 0;
        for (int i = 0; i < TSTAGES; ++i) {
            mb_init(full0 + 8 * i, 1);
            mb_init(empty0 + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mb_init(chunk0 + 8 * i, 1);      // MMA -> epilogue: chunk accumulated in buffer i
            mb_init(drained0 + 8 * i, 8);    // epilogue -> MMA: buffer i read out (8 epilogue warps)
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {  // allocate the two accumulators
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem_base = *tmem_slot;

    // Persistent: block b takes tiles b, b + grid, ... (row-tile major, so neighbouring blocks share
    // the same rows of A through L2). The k-block and chunk counters run across tiles, so the two
    // accumulator buffers alternate and one tile's epilogue overlaps the next tile's MMAs.
    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            int64_t g = 0;  // k-blocks issued by this block
            for (int64_t tile = blockIdx.x; tile < tiles && !s_abort; tile += gridDim.x) {
                const int m0 = (int)(tile / tiles_n) * TBM, n0 = (int)(tile % tiles_n) * TBN;
                for (int kb = 0; kb < KB; ++kb, ++g) {
                    const int s = (int)(g % TSTAGES);
                    if (g >= TSTAGES && !mb_wait(empty0 + 8 * s, (unsigned)((g / TSTAGES) - 1) & 1, args.status)) {
                        s_abort = 1;
                        break;
                    }
                    const uint32_t sa = su32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
                    mb_expect(full0 + 8 * s, STAGE_BYTES);
                    tma_load_2d(sa, &mapA, full0 + 8 * s, kb * TBK, m0);
                    tma_load_2d(sb, &mapW, full0 + 8 * s, kb * TBK, n0);
                }
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            int64_t g = 0, gc = 0;  // k-blocks and chunks consumed by this block
            for (int64_t tile = blockIdx.x; tile < tiles && !s_abort; tile += gridDim.x) {
                for (int kb = 0; kb < KB; ++kb, ++g) {
                    const int s = (int)(g % TSTAGES);
                    const int kc = kb % kpc;
                    const int buf = (int)(gc & 1);
                    if (kc == 0 && gc >= 2 &&
                        !mb_wait(drained0 + 8 * buf, (unsigned)((gc / 2) - 1) & 1, args.status)) {  // buffer free
                        s_abort = 1;
                        break;
                    }
                    if (!mb_wait(full0 + 8 * s, (unsigned)(g / TSTAGES) & 1, args.status)) {
                        s_abort = 1;
                        break;
                    }
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t sa = su32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
                    const uint32_t tmem_d = tmem_base + (uint32_t)(buf * TBN);
#pragma unroll
                    for (int k = 0; k < TBK / 16; ++k) {
                        // advance 16 fp16 = 32 bytes along K inside the swizzled 128-byte rows
                        mma_f16(tmem_d, smem_desc(sa + 32 * k), smem_desc(sb + 32 * k), (kc == 0 && k == 0) ? 0u : 1u);
                    }
                    mma_commit(empty0 + 8 * s);  // frees the stage when these MMAs have read it
                    if (kc == kpc - 1 || kb == KB - 1) {
                        mma_commit(chunk0 + 8 * buf);
                        ++gc;
                    }
                }
                if (s_abort) break;
            }
        }
    } else {
        // ---------------- epilogue (warps 2..9) ----------------
        const int q = warp & 3;                 // tensor-memory lane quarter this warp may read
        const int half = (warp - 2) >> 2;       // column half: 0 -> [0, 128), 1 -> [128, 256)
        const int ew = warp - 2;
        int *stg = stage_out + ew * 32 * 33;
        int *rz = row_c + ew * 96, *rr = rz + 32;
        float *rq = reinterpret_cast<float *>(rz + 64);
        const int K = args.K;
        int64_t gc = 0;
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
            const int64_t m0 = (tile / tiles_n) * TBM, n0 = (tile % tiles_n) * TBN;
            {  // this lane's row constants, shared with the warp for the transposed stores
                const int64_t m = m0 + 32 * q + lane;
                const bool mv = m < args.M;
                const qnn_qparams qa = args.pa[args.a_per_row ? (mv ? m : 0) : 0];
                rz[lane] = qa.z;
                rq[lane] = qa.Q;
                rr[lane] = mv ? args.rsA[m] : 0;
            }
            // 32 x 32 block: P values of rows (this warp's 32 lanes) x columns c0 .. c0 + 31, written
            // row-wise to shared memory and read back column-wise, so that each store instruction
            // writes 32 consecutive outputs of one row.
            auto emit = [&](int c0, const int (&P)[32]) {
#pragma unroll
                for (int i = 0; i < 32; ++i) stg[lane * 33 + i] = P[i];
                __syncwarp();
                const int64_t n = n0 + c0 + lane;
                const bool nv = n < args.N;
                const qnn_qparams qw = args.pw[nv ? n / args.rows_per_block : 0];
                const int cs = nv ? args.csW[n] : 0;
                const float bn = (nv && args.bias) ? args.bias[n] : 0.0f;
                for (int r = 0; r < 32; ++r) {
                    const int64_t m = m0 + 32 * q + r;
                    if (m >= args.M) break;
                    if (nv) {
                        const int ra = rr[r];
                        const int acc = stg[r * 33 + lane] + 128 * (ra + cs) - 16384 * K;  // raw code product
                        const long long S = offset_product(acc, rz[r], qw.z, ra, cs, K);
                        float y = recover_product(S, rq[r], qw.Q);
                        if (args.bias) y = __fadd_rn(y, bn);
                        if (args.Y) args.Y[m * args.ldy + n] = y;
                        if (args.acc_out) args.acc_out[m * args.N + n] = acc;
                    }
                }
                __syncwarp();
            };
            auto taddr_of = [&](int buf, int j) {
                return tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * TBN + half * 128 + 32 * j);
            };
            __syncwarp();
            if (nchunks == 1) {  // K <= 1024: read the accumulator and finish directly
                const int buf = (int)(gc & 1);
                ok = __all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status));
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll 1
                for (int j = 0; j < 4; ++j) {
                    uint32_t r[32];
                    tmem_ld32<32>(taddr_of(buf, j), r);
                    int P[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) P[i] = __float2int_rn(__uint_as_float(r[i]));
                    emit(half * 128 + 32 * j, P);
                }
                // the accumulator is free again: the tile after next may use it
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0)
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(drained0 + 8 * buf) : "memory");
                ++gc;
            } else {  // drain every chunk into int32 running sums
                int run[4][32];
#pragma unroll
                for (int j = 0; j < 4; ++j)
#pragma unroll
                    for (int i = 0; i < 32; ++i) run[j][i] = 0;
                for (int c = 0; c < nchunks; ++c, ++gc) {
                    const int buf = (int)(gc & 1);
                    ok = __all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status));
                    if (!ok) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        uint32_t rr32[32];
                        tmem_ld32<32>(taddr_of(buf, j), rr32);
#pragma unroll
                        for (int i = 0; i < 32; ++i) run[j][i] += __float2int_rn(__uint_as_float(rr32[i]));
                    }
                    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                    __syncwarp();
                    if (lane == 0)
                        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(drained0 + 8 * buf) : "memory");
                }
                if (!ok) break;
#pragma unroll
                for (int j = 0; j < 4; ++j) emit(half * 128 + 32 * j, run[j]);
            }
        }
    }
    __syncwarp();
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (s_abort && warp == 0 && lane == 0) {
        // let copies still in flight land before the block leaves (bounded)
        const unsigned long long t0 = gtime();
        while (gtime() - t0 < 4000000ull) __nanosleep(1000);
    }
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                     : "memory");
    }
}

// u8 codes -> centered fp16 (c - 128), rows padded with zeros to ldo (a multiple of 64).
__global__ void center_fp16_kernel(const uint8_t *__restrict__ in, int64_t rows, int K, int64_t ldi,
                                   __half *__restrict__ out, int ldo) {
    const int64_t total = rows * (int64_t)(ldo / 8);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / (ldo / 8);
        const int k0 = (int)(i % (ldo / 8)) * 8;
        __align__(16) __half v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int k = k0 + e;
            v[e] = k < K ? __int2half_rn((int)in[r * ldi + k] - 128) : __int2half_rn(0);
        }
        *reinterpret_cast<uint4 *>(out + r * ldo + k0) = *reinterpret_cast<const uint4 *>(v);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_encode_mu;

qnn_status get_encode(PFN_cuTensorMapEncodeTiled_v12000 *out) {
    std::lock_guard<std::mutex> lk(g_encode_mu);
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &fn, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn) {
            cudaGetLastError();
            return QNN_ERR_CUDA;
        }
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    *out = g_encode;
    return QNN_OK;
}

// 2-D fp16 tensor [rows][ld] (ld a multiple of 64), boxes of 64 x box_rows, 128-byte swizzle.
qnn_status make_map(CUtensorMap *map, const __half *base, int64_t rows, int64_t ld, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
    QNN_TRY(get_encode(&enc));
    cuuint64_t dims[2] = {(cuuint64_t)ld, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(ld * 2)};
    cuuint32_t box[2] = {(cuuint32_t)TBK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half *>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? QNN_OK : QNN_ERR_CUDA;
}

}  // namespace

size_t tc_scratch_bytes(int64_t M, int64_t N, int64_t K) {
    const int64_t kp = (K + 63) / 64 * 64;
    return (size_t)(M + N) * kp * 2 + 512;
}

// Centers A and W into fp16 scratch and runs the tensor-core product (K <= QNN_K_MAX).
qnn_status launch_qgemm_tc(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA, int64_t M,
                           int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw, int64_t rows_per_block,
                           const int32_t *csW, int64_t N, const float *bias, float *Y, int64_t ldy, int32_t *acc_out,
                           void *scratch_ptr, cudaStream_t st) {
    if (M == 0 || N == 0) return QNN_OK;
    const int kp = (int)((K + 63) / 64 * 64);
    __half *A16 = reinterpret_cast<__half *>(scratch_ptr);
    __half *W16 = A16 + M * kp;
    {
        ProfScope prof("center_fp16", st);
        const int64_t totA = M * (kp / 8), totW = N * (kp / 8);
        center_fp16_kernel<<<(unsigned)std::min<int64_t>((totA + 255) / 256, 65535 * 4), 256, 0, st>>>(A, M, (int)K, lda,
                                                                                                      A16, kp);
        center_fp16_kernel<<<(unsigned)std::min<int64_t>((totW + 255) / 256, 65535 * 4), 256, 0, st>>>(W, N, (int)K, ldw,
                                                                                                      W16, kp);
        QNN_CUDA_TRY(cudaGetLastError());
    }
    CUtensorMap mA, mW;
    QNN_TRY(make_map(&mA, A16, M, kp, TBM));
    QNN_TRY(make_map(&mW, W16, N, kp, TBN));
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    TcArgs a{pa, ga == QNN_PER_ROW, rsA, pw, rows_per_block, csW, bias, Y, ldy, acc_out, M, N, (int)K, kp / TBK, status};
    const size_t smem = (size_t)TSTAGES * STAGE_BYTES + 1024 + (8 * 32 * 33 + 8 * 96) * 4 + 256;
    static int configured = -1;
    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (configured != dev) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(qgemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        configured = dev;
    }
    const int64_t tiles = ((M + TBM - 1) / TBM) * ((N + TBN - 1) / TBN);
    dim3 grid((unsigned)std::min<int64_t>(tiles, sm_count()));  // persistent: at most one block per SM
    ProfScope prof("qgemm_tc", st);
    qgemm_tc_kernel<<<grid, TC_THREADS, smem, st>>>(mA, mW, a);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

}  // namespace qnn
