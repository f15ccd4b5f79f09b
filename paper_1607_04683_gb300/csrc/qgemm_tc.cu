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

#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <algorithm>
#include <mutex>

#include "qnn_device.cuh"
#include "qnn_host.h"
#include "tc_gemm.h"
#include "tc_ptx.cuh"

namespace qnn {
namespace {

constexpr int TBM = 128, TBK = 64;               // rows of A per tile; fp16 elements per k-block (128 bytes)
constexpr int A_BYTES = TBM * TBK * 2;            // 16 KB
constexpr int KCHUNK = 1024;                      // exact fp32 accumulation bound (see above)
constexpr unsigned long long TC_WAIT_NS = 2000000000ull;

// kEpiLinear: recovered product, any K (chunked drains), outputs staged through shared memory.
// kEpiRow: recovered product for K <= 1024, one output row per lane, two blocks per SM.
// kEpiLstm: the LSTM cell update on gate-interleaved columns, K <= 1024. (Issuing its input-product
// and cell-state loads before the accumulator wait was measured slower even for single-tile grids:
// those HBM loads delay the tile's TMA stream.)
// kEpiPartial: split-K, each work item (tile, K range of at most 1024) stores its exact centered
// integer sums P as int32 into its own slice of a partial-sum buffer; a consumer adds the slices.
enum Epilogue { kEpiLinear = 0, kEpiLstm = 1, kEpiRow = 2, kEpiPartial = 4, kEpiLstmX = 5 };

struct ColConst {  // per-output-column constants of kEpiRow, staged in shared memory per tile
    int cs, zw;
    float Qw, bias;
    float csf;  // cs as an exact fp32 value (cs <= 255 K < 2^24)
};
struct ColUnit {  // and the weight unit of each column (-1 past N)
    int unit;
};

// Per tile width BN (rows of W per tile) and epilogue: warps (TMA producer, MMA issuer, then the
// epilogue warps), stage ring depth, tensor-memory columns (two fp32 accumulators of BN columns),
// register cap, the epilogue's shared staging, and the MMA instruction descriptor (fp32
// accumulator, fp16 A and B, both K-major, M = 128, N = BN). A block that allocates tensor memory
// has its SM to itself, so the ALU-bound row and LSTM epilogues run sixteen warps (four per
// tensor-memory lane quarter); eighteen warps fit the register file at 96 registers a thread.
template <int BN, int EPI>
struct Tile {
    static_assert(EPI == kEpiLinear || BN <= 128, "row and LSTM epilogues take tiles of at most 128 columns");
    // a 96-column LSTM tile has six 4-cell slices per lane quarter: 24 epilogue warps, one slice each
    // kEpiLstmX: the LSTM step with the input product fused in (a second operand pair and accumulator)
    static constexpr bool IS_LSTM = EPI == kEpiLstm || EPI == kEpiLstmX;
    static constexpr bool LSTM96 = IS_LSTM && BN == 96;
    static constexpr int EPI_WARPS = EPI == kEpiLinear ? 8 : (LSTM96 ? 24 : 16);
    // LSTM: cells per epilogue slice (a 32-column tile has 8 cells: 2-cell slices keep 4 warps busy)
    static constexpr int CPS = BN == 32 ? 2 : 4;
    static constexpr int THREADS = 32 * (2 + EPI_WARPS);
    static constexpr int B_BYTES = BN * TBK * 2;
    // a pipeline stage carries KPS consecutive k-blocks (A sub-tiles first, then the W sub-tiles):
    // the operand stream advances by stages at a pace that hardly depends on their size, so short
    // reductions (K <= 1024) take several k-blocks a stage: four for narrow LSTM tiles (two stages in
    // flight), two for row tiles, split-K items and the 128-column LSTM tiles with the input product
    // (two 64 KB stages: 38.9 against 41.1 us a step with four of 32 KB); the long-K linear tiles and
    // the other 96- and 128-column LSTM tiles keep more, smaller stages in flight (each choice
    // measured on GB300)
    static constexpr int KPS = IS_LSTM ? (BN <= 32 ? 4 : ((BN == 64 || (BN == 128 && EPI == kEpiLstmX)) ? 2 : 1))
                                               : ((EPI == kEpiPartial || EPI == kEpiRow) ? 2 : 1);
    static constexpr int SUB_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGE_BYTES = KPS * SUB_BYTES;
    static constexpr int BASE_STAGES = EPI == kEpiLinear    ? (BN == 256 ? 4 : 6)
                                       : EPI == kEpiPartial ? 6  // one K range per item: keep it all in flight
                                                            : (BN == 128 ? 4 : 6);
    // LSTM: the tile's input products px (4 gates x 128 rows x BN/4 cells) and cell state c (128 x
    // BN/4), fp32, double-buffered in shared memory after the stages
    static constexpr int PX_BOX = TBM * (BN / 4) * 4;  // one gate's px box, bytes
    // kEpiLstmX: the tile's column constants after the c box: per gate the bias, the Wx and the Wh row
    // code sums of its BN / 4 cells ([12][BN / 4] 32-bit words)
    static constexpr int COL_BYTES = 12 * (BN / 4) * 4;
    static constexpr int LSTM_TX = EPI == kEpiLstmX ? PX_BOX + COL_BYTES : 5 * PX_BOX;  // bytes of one fill
    static constexpr int LSTM_BUF = (LSTM_TX + 1023) / 1024 * 1024;  // [4 px boxes +] the c box [+ constants]
    // kEpiLstmX: per epilogue thread, its row's per-gate constants of eq. (1)/(3), kept in shared
    // memory across the block's tiles: per warp [4 gates][32 lanes] float4 (1/dx, 1/dh, rt_x, rt_h),
    // then [4 gates][32 lanes] float2 (dx, dh)
    static constexpr int RC_BYTES = EPI == kEpiLstmX ? EPI_WARPS * 24 * 32 * 4 : 0;
    static constexpr int EPI_BYTES = IS_LSTM              ? 2 * LSTM_BUF + RC_BYTES
                                     : EPI == kEpiPartial ? 0
                                                          : 2 * BN * (int)(sizeof(ColConst) + sizeof(ColUnit));
    static constexpr int SMEM_CAP = 227 * 1024 - 1024 - 256;  // dynamic shared memory left for stages + EPI_BYTES
    static constexpr int FIT_STAGES = (SMEM_CAP - EPI_BYTES) / STAGE_BYTES;
    static constexpr int WANT_STAGES = BASE_STAGES / KPS < 2 ? 2 : BASE_STAGES / KPS;
    static constexpr int STAGES = WANT_STAGES < FIT_STAGES ? WANT_STAGES : FIT_STAGES;
    static_assert(STAGES >= 2, "at least two pipeline stages must fit");
    static constexpr int ACC_COLS = (EPI == kEpiLstmX ? 2 : 1) * BN;  // one tile buffer's accumulator columns
    static constexpr int TMEM_COLS =
        2 * ACC_COLS <= 32 ? 32
                           : (2 * ACC_COLS <= 64 ? 64 : (2 * ACC_COLS <= 128 ? 128 : (2 * ACC_COLS <= 256 ? 256 : 512)));
    // warps sit on the four SM sub-partitions by index: 18 warps put 5 on one (5 x 32 x 96 <= 16384),
    // 26 warps put 7 on one (7 x 32 x 72 <= 16384)
    static constexpr int MAX_REGS = EPI == kEpiLinear ? 168 : (LSTM96 ? 72 : 96);
    static constexpr uint32_t IDESC = mma_idesc_f16(TBM, BN);
    static constexpr uint32_t IDESC_HALF = mma_idesc_f16(TBM, BN / 2 >= 16 ? BN / 2 : 16);  // half-width items
    static constexpr size_t SMEM = (size_t)STAGES * STAGE_BYTES + 1024 + EPI_BYTES + 256;
};

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
    TcLstmOut lstm;  // kEpiLstm only
    int splits;      // K ranges per tile (kEpiPartial; 1 otherwise)
    int kbs;         // k-blocks per K range
    int32_t *part;   // kEpiPartial: [splits][M][ldpart] int32
    int64_t ldpart;
    int w_static;    // W was written before the previous kernel of the stream started (model weights):
                     // its first tiles may load before the programmatic-launch wait
    // kEpiLstmX: the input product x_t Wx of the step (k-blocks 0 .. KB_x - 1 of the K loop, into a
    // second accumulator; A from the x map, W from the Wx map). Row b of x_t has its unit at
    // pa_x[b * x_stride] and its code sum at rsA_x[b * x_stride]; pw_x, csW_x (gate-major [4][H]) and
    // bias_x ([4H]) as for the recurrent product; K_x the true input width.
    const qnn_qparams *pa_x;
    int64_t x_stride;
    const int32_t *rsA_x;
    const qnn_qparams *pw_x;
    const int32_t *csW_x;
    const float *bias_x;
    int K_x, KB_x;
    // LSTM epilogues: tiles from full_tiles on (the last, partial wave of the persistent grid) run as
    // two half-width items each, so that the blocks of that wave finish together (0: none)
    int64_t full_tiles;
};

__device__ __forceinline__ unsigned long long gtime() { return global_timer_ns(); }
// Bounded wait; false (and QNN_ERR_TIMEOUT recorded) if the phase did not complete in time.
__device__ __forceinline__ bool mb_wait(uint32_t b, unsigned parity, int *status) {
    return mbar_wait_bounded(b, parity, status, TC_WAIT_NS);
}
// Vector loads and stores of 2 or 4 consecutive (8- or 16-byte aligned) values.
__device__ __forceinline__ void ld_vec(const float *p, float (&v)[4]) {
    const float4 a = *reinterpret_cast<const float4 *>(p);
    v[0] = a.x, v[1] = a.y, v[2] = a.z, v[3] = a.w;
}
__device__ __forceinline__ void ld_vec(const float *p, float (&v)[2]) {
    const float2 a = *reinterpret_cast<const float2 *>(p);
    v[0] = a.x, v[1] = a.y;
}
__device__ __forceinline__ void ld_vec(const int *p, int (&v)[4]) {
    const int4 a = *reinterpret_cast<const int4 *>(p);
    v[0] = a.x, v[1] = a.y, v[2] = a.z, v[3] = a.w;
}
__device__ __forceinline__ void ld_vec(const int *p, int (&v)[2]) {
    const int2 a = *reinterpret_cast<const int2 *>(p);
    v[0] = a.x, v[1] = a.y;
}
__device__ __forceinline__ void st_vec(float *p, const float (&v)[4]) {
    *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
__device__ __forceinline__ void st_vec(float *p, const float (&v)[2]) {
    *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
}

// Tile order: groups of kGroupM row tiles, columns outer within a group, so that the tiles one
// wave of blocks works on span a compact block of A and W (both stay in L2 across the wave).
constexpr int kGroupM = 16;
__device__ __forceinline__ void tile_origin(int64_t tile, int64_t tiles_m, int tiles_n, int bn, int64_t &m0,
                                            int64_t &n0) {
    const int64_t per_group = (int64_t)kGroupM * tiles_n;
    const int64_t first = (tile / per_group) * kGroupM;
    const int64_t rows = tiles_m - first < kGroupM ? tiles_m - first : kGroupM;
    const int64_t local = tile % per_group;
    m0 = (first + local % rows) * TBM;
    n0 = (local / rows) * bn;
}

// Recovered outputs of one 16-column block of one row that lies in one weight unit, in fp32: the
// tensor-core sum P is an exact integer and, when |rt| + |za + 128| 255 K < 2^24, so is the offset
// term rt + (za + 128) cs, formed by one fused multiply-add without rounding; the one rounded add
// P + (offset term) then equals the rounded integer sum S of eq. (1), and S / (Qa Qw) comes from the
// divisor's correctly rounded reciprocal (div_by_recip2: the IEEE quotient while the divisor lies
// within 2^-60 .. 2^60). Two columns at a time with paired fp32 instructions; four 16-byte stores.
template <bool BIAS>
__device__ __forceinline__ void row_block_f32(const uint32_t (&r)[16], const ColConst *cc, float rtf, float za128f,
                                              float den, float rden, float *yr) {
#pragma unroll
    for (int v4 = 0; v4 < 4; ++v4) {
        float y[4];
#pragma unroll
        for (int e2 = 0; e2 < 4; e2 += 2) {
            const int i = 4 * v4 + e2;
            const float2 off = ffma2_rn(f2(za128f), make_float2(cc[i].csf, cc[i + 1].csf), f2(rtf));
            const float2 S = fadd2_rn(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), off);
            float2 q = div_by_recip2(S, den, rden);
            if (BIAS) q = fadd2_rn(q, make_float2(cc[i].bias, cc[i + 1].bias));
            y[e2] = q.x, y[e2 + 1] = q.y;
        }
        *reinterpret_cast<float4 *>(yr + 4 * v4) = make_float4(y[0], y[1], y[2], y[3]);
    }
}

// The same block with the integer sum formed in 64 bits and an IEEE divide (rows outside the
// bounds above).
template <bool BIAS>
__device__ __forceinline__ void row_block_fast(const uint32_t (&r)[16], const ColConst *cc, long long rt, int za128,
                                               float den, float *yr) {
#pragma unroll
    for (int v4 = 0; v4 < 4; ++v4) {
        float y[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int i = 4 * v4 + e;
            const long long S = (long long)f32_integer_to_s32(__uint_as_float(r[i])) + rt + (long long)za128 * cc[i].cs;
            const float x = s64_to_f32_rn(S);
            y[e] = __fdiv_rn(x, den);
            if (BIAS) y[e] = __fadd_rn(y[e], cc[i].bias);
        }
        *reinterpret_cast<float4 *>(yr + 4 * v4) = make_float4(y[0], y[1], y[2], y[3]);
    }
}

// Persistent tile loop. Warp 0: TMA producer; warp 1: tensor-memory owner and MMA issuer; warps
// 2.. : epilogue. EPI = kEpiLinear / kEpiRow write the recovered product (plus bias) and
// optionally the raw int32 accumulator; EPI = kEpiLstm treats the columns as gate-interleaved LSTM
// pre-activations (8-cell groups of [i f g o] x 8 rows of W) and applies the cell update (K <= 1024).
// With a programmatic dependent launch the block setup overlaps the previous kernel of the stream.
template <int BN, int EPI>
__global__ void __launch_bounds__((Tile<BN, EPI>::THREADS)) __maxnreg__((Tile<BN, EPI>::MAX_REGS))
    qgemm_tc_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapW,
                    const __grid_constant__ CUtensorMap mapPX, const __grid_constant__ CUtensorMap mapC,
                    const __grid_constant__ CUtensorMap mapAX, const __grid_constant__ CUtensorMap mapWX,
                    const TcArgs args) {
    using TL = Tile<BN, EPI>;
    constexpr int STAGES = TL::STAGES;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte alignment for the swizzled tiles
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + STAGES * TL::STAGE_BYTES + TL::EPI_BYTES);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * STAGES + 8);
    const uint32_t full0 = su32(bars), empty0 = su32(bars + STAGES), chunk0 = su32(bars + 2 * STAGES),
                   drained0 = su32(bars + 2 * STAGES + 2);
    // LSTM only: px/c buffer i loaded (pxfull0 + 8 i) and released by every epilogue warp (pxempty0 + 8 i)
    const uint32_t pxfull0 = su32(bars + 2 * STAGES + 4), pxempty0 = su32(bars + 2 * STAGES + 6);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr bool LX = EPI == kEpiLstmX;
    const int KB = args.KB + (LX ? args.KB_x : 0);  // k-blocks of the K loop (kEpiLstmX: x's, then h's)
    const int kpc = LX ? 64 : KCHUNK / TBK;        // k-blocks per chunk (16; kEpiLstmX: the whole loop, each
                                                   // accumulator summing at most 1024)
    const int nchunks = (KB + kpc - 1) / kpc;
    const int tiles_n = (int)((args.N + BN - 1) / BN);
    const int64_t tiles_m = (args.M + TBM - 1) / TBM;
    const int64_t tiles = tiles_m * tiles_n;
    // work items: (tile, K range); one K range per tile except for split-K. LSTM epilogues may split
    // the tiles of the last wave into half-width items (the first BN / 2 columns of the tile's W box
    // feed an MMA of N = BN / 2; the px, c and constant boxes are loaded whole)
    const int splits = args.splits;
    const int64_t full_tiles =
        (TL::IS_LSTM && args.full_tiles > 0 && args.full_tiles < tiles) ? args.full_tiles : tiles;
    const int64_t work = full_tiles + 2 * (tiles - full_tiles);  // tile items
    const int64_t items = work * splits;
    // origin of tile item w; true for a half-width item
    auto item_origin = [&](int64_t w, int64_t &m0, int64_t &n0) -> bool {
        if (w < full_tiles) {
            tile_origin(w, tiles_m, tiles_n, BN, m0, n0);
            return false;
        }
        const int64_t j = w - full_tiles;
        tile_origin(full_tiles + j / 2, tiles_m, tiles_n, BN, m0, n0);
        n0 += (j & 1) * (BN / 2);
        return true;
    };
    // the A and W tiles of k-block kb (kEpiLstmX: x_t and Wx for kb < KB_x, then h_{t-1} and Wh)
    auto load_a = [&](uint32_t dst, uint32_t bar, int kb, int m0) {
        if (LX && kb < args.KB_x)
            tma_load_2d(dst, &mapAX, bar, kb * TBK, m0);
        else
            tma_load_2d(dst, &mapA, bar, (kb - (LX ? args.KB_x : 0)) * TBK, m0);
    };
    auto load_w = [&](uint32_t dst, uint32_t bar, int kb, int n0) {
        if (LX && kb < args.KB_x)
            tma_load_2d(dst, &mapWX, bar, kb * TBK, n0);
        else
            tma_load_2d(dst, &mapW, bar, (kb - (LX ? args.KB_x : 0)) * TBK, n0);
    };
    __shared__ int s_abort;

    if (threadIdx.x == 0) {
        s_abort = 0;
        for (int i = 0; i < STAGES; ++i) {
            mb_init(full0 + 8 * i, 1);
            mb_init(empty0 + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mb_init(chunk0 + 8 * i, 1);      // MMA -> epilogue: chunk accumulated in buffer i
            mb_init(drained0 + 8 * i, TL::EPI_WARPS);  // epilogue -> MMA: buffer i read out by every epilogue warp
            mb_init(pxfull0 + 8 * i, 1);
            mb_init(pxempty0 + 8 * i, TL::EPI_WARPS);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {  // allocate the two accumulators
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)),
                     "n"(TL::TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem_base = *tmem_slot;
    // Static weights: the producer starts the W tiles of its first stages before the wait below
    // (the A tiles, outputs of the previous kernel, follow after it); their barriers expect both.
    int w_early = 0;
    // kEpiLstmX: the input side (x_t codes, Wx) was written before the step loop began, not by the
    // previous kernel, so leading stages that hold only x's k-blocks are issued whole before the
    // wait (their MMAs then overlap the previous kernel too)
    int full_early = 0;
    if (warp == 0 && lane == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapW)) : "memory");
        if (LX) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapAX)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapWX)) : "memory");
        }
        if (args.w_static && blockIdx.x < items) {
            int64_t m0, n0;
            item_origin(blockIdx.x / splits, m0, n0);
            const int kb0 = (int)(blockIdx.x % splits) * args.kbs, kb1 = min(KB, kb0 + args.kbs);
            if constexpr (TL::KPS == 1) {
                w_early = min(STAGES, kb1 - kb0);
                for (int j = 0; j < w_early; ++j) {
                    const uint32_t sb = su32(smem + j * TL::STAGE_BYTES) + A_BYTES;
                    mb_expect(full0 + 8 * j, TL::STAGE_BYTES);
                    load_w(sb, full0 + 8 * j, kb0 + j, (int)n0);
                    if (LX && full_early == j && kb0 + j < args.KB_x) {
                        load_a(sb - A_BYTES, full0 + 8 * j, kb0 + j, (int)m0);
                        ++full_early;
                    }
                }
            } else {
                w_early = min(STAGES, (kb1 - kb0 + TL::KPS - 1) / TL::KPS);
                for (int j = 0; j < w_early; ++j) {
                    const int kbj = kb0 + j * TL::KPS, nv = min(TL::KPS, kb1 - kbj);
                    const uint32_t sb = su32(smem + j * TL::STAGE_BYTES) + TL::KPS * A_BYTES;
                    mb_expect(full0 + 8 * j, (uint32_t)(nv * TL::SUB_BYTES));
                    for (int v = 0; v < nv; ++v)
                        load_w(sb + v * TL::B_BYTES, full0 + 8 * j, kbj + v, (int)n0);
                    if (LX && full_early == j && kbj + nv <= args.KB_x) {
                        for (int v = 0; v < nv; ++v)
                            load_a(sb - TL::KPS * A_BYTES + v * A_BYTES, full0 + 8 * j, kbj + v, (int)m0);
                        ++full_early;
                    }
                }
            }
        }
    }
    // With a programmatic dependent launch the setup above overlaps the previous kernel of the
    // stream; its outputs (this kernel's operands) are complete and visible after this wait.
    // (kEpiLstmX: the MMA warp reads only shared and tensor memory, so it starts on the early
    // input-side stages at once.)
    if (!(LX && warp == 1)) grid_dependency_wait();
    grid_dependents_launch();

    // Persistent: block b takes tiles b, b + grid, ... in grouped order (tile_origin). The k-block
    // and chunk counters run across tiles, so the two accumulator buffers alternate and one tile's
    // epilogue overlaps the next tile's MMAs.
    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if constexpr (TL::KPS == 1) {
            if (lane == 0) {
                int64_t g = 0;  // k-blocks issued by this block
                for (int64_t item = blockIdx.x; item < items && !s_abort; item += gridDim.x) {
                    int64_t m0, n0;
                    item_origin(item / splits, m0, n0);
                    const int kb0 = (int)(item % splits) * args.kbs, kb1 = min(KB, kb0 + args.kbs);
                    for (int kb = kb0; kb < kb1; ++kb, ++g) {
                        const int s = (int)(g % STAGES);
                        if (g >= STAGES && !mb_wait(empty0 + 8 * s, (unsigned)((g / STAGES) - 1) & 1, args.status)) {
                            s_abort = 1;
                            break;
                        }
                        const uint32_t sa = su32(smem + s * TL::STAGE_BYTES), sb = sa + A_BYTES;
                        if (g < full_early) continue;  // issued whole before the wait
                        if (g < w_early) {  // W already on its way (expect set with it)
                            load_a(sa, full0 + 8 * s, kb, (int)m0);
                            continue;
                        }
                        mb_expect(full0 + 8 * s, TL::STAGE_BYTES);
                        load_a(sa, full0 + 8 * s, kb, (int)m0);
                        load_w(sb, full0 + 8 * s, kb, (int)n0);
                    }
                }
            }
        } else {
            if (lane == 0) {
                // One thread issues every copy; its loop is on the critical path of the operand stream,
                // so the ring position (slot, phase, shared-memory address) advances incrementally in
                // 32-bit registers instead of being derived from a 64-bit counter every stage.
                const uint32_t ring0 = su32(smem);
                int slot = 0, issued = 0;  // ring slot; stages issued (saturating at STAGES)
                unsigned phase = 0;        // parity of the slot's current use
                uint32_t st_addr = ring0, bar_full = full0, bar_empty = empty0;
                for (int64_t item = blockIdx.x; item < items && !s_abort; item += gridDim.x) {
                    int64_t m0l, n0l;
                    item_origin(item / splits, m0l, n0l);
                    const int m0 = (int)m0l, n0 = (int)n0l;
                    const int kb0 = (int)(item % splits) * args.kbs, kb1 = min(KB, kb0 + args.kbs);
                    for (int kb = kb0; kb < kb1; kb += TL::KPS) {
                        if (issued >= STAGES && !mb_wait(bar_empty, phase ^ 1u, args.status)) {
                            s_abort = 1;
                            break;
                        }
                        const int nv = min(TL::KPS, kb1 - kb);  // k-blocks in this stage (the last may be short)
                        const uint32_t sb = st_addr + TL::KPS * A_BYTES;
                        const bool w_sent = issued < w_early;   // W already on its way (expect set with it)
                        if (issued >= full_early) {             // (else issued whole before the wait)
                            if (!w_sent) mb_expect(bar_full, (uint32_t)(nv * TL::SUB_BYTES));
#pragma unroll
                            for (int v = 0; v < TL::KPS; ++v) {
                                if (v >= nv) break;
                                load_a(st_addr + v * A_BYTES, bar_full, kb + v, m0);
                                if (!w_sent) load_w(sb + v * TL::B_BYTES, bar_full, kb + v, n0);
                            }
                        }
                        if (issued < STAGES) ++issued;
                        if (++slot == STAGES) {
                            slot = 0;
                            phase ^= 1u;
                            st_addr = ring0, bar_full = full0, bar_empty = empty0;
                        } else {
                            st_addr += TL::STAGE_BYTES, bar_full += 8, bar_empty += 8;
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if constexpr (TL::KPS == 1) {
            if (lane == 0) {
                int64_t g = 0, gc = 0;  // k-blocks and chunks consumed by this block
                for (int64_t item = blockIdx.x; item < items && !s_abort; item += gridDim.x) {
                    const int kb0 = (int)(item % splits) * args.kbs, kb1 = min(KB, kb0 + args.kbs);
                    const uint32_t idesc = item / splits < full_tiles ? TL::IDESC : TL::IDESC_HALF;
                    for (int kb = kb0; kb < kb1; ++kb, ++g) {
                        const int s = (int)(g % STAGES);
                        const int kc = (kb - kb0) % kpc;
                        const int buf = (int)(gc & 1);
                        if (kc == 0 && gc >= 2 &&
                            !mb_wait(drained0 + 8 * buf, (unsigned)((gc / 2) - 1) & 1, args.status)) {  // buffer free
                            s_abort = 1;
                            break;
                        }
                        if (!mb_wait(full0 + 8 * s, (unsigned)(g / STAGES) & 1, args.status)) {
                            s_abort = 1;
                            break;
                        }
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint32_t sa = su32(smem + s * TL::STAGE_BYTES), sb = sa + A_BYTES;
                        // kEpiLstmX: x's k-blocks into the buffer's first accumulator, h's into the second
                        const bool hpart = LX && kb >= args.KB_x;
                        const uint32_t tmem_d = tmem_base + (uint32_t)(buf * TL::ACC_COLS + (hpart ? BN : 0));
                        const bool fresh = kc == 0 || (LX && kb == args.KB_x);
#pragma unroll
                        for (int k = 0; k < TBK / 16; ++k) {
                            // advance 16 fp16 = 32 bytes along K inside the swizzled 128-byte rows
                            mma_f16(tmem_d, smem_desc(sa + 32 * k), smem_desc(sb + 32 * k), idesc,
                                    (fresh && k == 0) ? 0u : 1u);
                        }
                        mma_commit(empty0 + 8 * s);  // frees the stage when these MMAs have read it
                        if (kc == kpc - 1 || kb == kb1 - 1) {
                            mma_commit(chunk0 + 8 * buf);
                            ++gc;
                        }
                    }
                    if (s_abort) break;
                }
            }
        } else {
            if (lane == 0) {
                // The same incremental ring position as the producer's; the shared-memory descriptors of
                // a stage are its base descriptor plus the byte offset / 16 in the address field (the
                // address stays below 2^18, so the 14-bit field never carries).
                const uint32_t ring0 = su32(smem);
                int slot = 0;
                unsigned phase = 0;
                uint32_t st_addr = ring0, bar_full = full0, bar_empty = empty0;
                int64_t gc = 0;  // chunks accumulated by this block
                for (int64_t item = blockIdx.x; item < items && !s_abort; item += gridDim.x) {
                    const int kb0 = (int)(item % splits) * args.kbs, kb1 = min(KB, kb0 + args.kbs);
                    const uint32_t idesc = item / splits < full_tiles ? TL::IDESC : TL::IDESC_HALF;
                    int kc = 0;  // position of the stage in its K chunk (chunks hold whole stages)
                    for (int kb = kb0; kb < kb1; kb += TL::KPS) {
                        const int nv = min(TL::KPS, kb1 - kb);
                        const int buf = (int)(gc & 1);
                        if (kc == 0 && gc >= 2 &&
                            !mb_wait(drained0 + 8 * buf, (unsigned)((gc / 2) - 1) & 1, args.status)) {  // buffer free
                            s_abort = 1;
                            break;
                        }
                        if (!mb_wait(bar_full, phase, args.status)) {
                            s_abort = 1;
                            break;
                        }
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint64_t da = smem_desc(st_addr), db = smem_desc(st_addr + TL::KPS * A_BYTES);
#pragma unroll
                        for (int v = 0; v < TL::KPS; ++v) {
                            if (v >= nv) break;
                            // kEpiLstmX: x's k-blocks into the buffer's first accumulator, h's into the second
                            const bool hpart = LX && kb + v >= args.KB_x;
                            const uint32_t tmem_d = tmem_base + (uint32_t)(buf * TL::ACC_COLS + (hpart ? BN : 0));
                            const bool fresh = (kc == 0 && v == 0) || (LX && kb + v == args.KB_x);
#pragma unroll
                            for (int k = 0; k < TBK / 16; ++k) {
                                // advance 16 fp16 = 32 bytes along K inside the swizzled 128-byte rows
                                mma_f16(tmem_d, da + (uint64_t)((v * A_BYTES + 32 * k) >> 4),
                                        db + (uint64_t)((v * TL::B_BYTES + 32 * k) >> 4), idesc,
                                        (fresh && k == 0) ? 0u : 1u);
                            }
                        }
                        mma_commit(bar_empty);  // frees the stage when these MMAs have read it
                        kc += nv;
                        if (kc >= kpc || kb + nv >= kb1) {
                            mma_commit(chunk0 + 8 * buf);
                            ++gc;
                            kc = 0;
                        }
                        if (++slot == STAGES) {
                            slot = 0;
                            phase ^= 1u;
                            st_addr = ring0, bar_full = full0, bar_empty = empty0;
                        } else {
                            st_addr += TL::STAGE_BYTES, bar_full += 8, bar_empty += 8;
                        }
                    }
                    if (s_abort) break;
                }
            }
        }
    } else if constexpr (EPI == kEpiLinear) {
        // ---------------- epilogue (warps 2..9): recovered product, any K ----------------
        // Each lane owns one output row and one column half of the tile. Every K chunk is drained
        // from tensor memory into int32 running sums in registers; after the last chunk the sums
        // are recovered (eq. 1 offsets, eq. 3) and stored as 16-byte vectors straight from
        // registers (ragged or unaligned outputs element by element). Column constants are staged
        // in shared memory per tile (double-buffered; one named barrier of the epilogue warps).
        constexpr int NJ = BN / 64;             // 32-column blocks per warp
        ColConst *scol = reinterpret_cast<ColConst *>(smem + STAGES * TL::STAGE_BYTES);
        ColUnit *sunit = reinterpret_cast<ColUnit *>(scol + 2 * BN);
        const int q = warp & 3;                 // tensor-memory lane quarter this warp may read
        const int half = (warp - 2) >> 2;       // column half: [0, BN/2) or [BN/2, BN)
        const int ew = warp - 2;
        const int K = args.K;
        const bool vec = args.Y && (args.ldy % 4 == 0) && ((reinterpret_cast<uintptr_t>(args.Y) & 15) == 0);
        int64_t gc = 0, it = 0;
        bool failed = false;
        for (int64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
            int64_t m0, n0;
            tile_origin(tile, tiles_m, tiles_n, BN, m0, n0);
            ColConst *cc = scol + (it & 1) * BN;
            ColUnit *cu = sunit + (it & 1) * BN;
            for (int c = ew * 32 + lane; c < BN; c += 32 * TL::EPI_WARPS) {
                const int64_t n = n0 + c;
                ColConst v{0, 0, 1.0f, 0.0f, 0.0f};
                int unit = -1;
                if (n < args.N) {
                    unit = (int)(n / args.rows_per_block);
                    const qnn_qparams qw = args.pw[unit];
                    v.cs = args.csW[n];
                    v.csf = (float)v.cs;
                    v.zw = qw.z;
                    v.Qw = qw.Q;
                    v.bias = args.bias ? args.bias[n] : 0.0f;
                }
                cc[c] = v;
                cu[c].unit = unit;
            }
            asm volatile("bar.sync 1, %0;" ::"n"(32 * TL::EPI_WARPS) : "memory");
            int run[NJ][32];
#pragma unroll
            for (int j = 0; j < NJ; ++j)
#pragma unroll
                for (int i = 0; i < 32; ++i) run[j][i] = 0;
            for (int c = 0; c < nchunks; ++c, ++gc) {
                const int buf = (int)(gc & 1);
                if (!failed && *reinterpret_cast<volatile int *>(&s_abort)) failed = true;
                if (!failed) {
                    failed = !__all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status));
                    if (failed) *reinterpret_cast<volatile int *>(&s_abort) = 1;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                if (!failed) {
#pragma unroll
                    for (int j = 0; j < NJ; ++j) {
                        uint32_t r32[32];
                        tmem_ld32(tmem_base + ((uint32_t)(32 * q) << 16) +
                                      (uint32_t)(buf * BN + half * (BN / 2) + 32 * j),
                                  r32);
#pragma unroll
                        for (int i = 0; i < 32; ++i) run[j][i] += f32_integer_to_s32(__uint_as_float(r32[i]));
                    }
                }
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mb_arrive(drained0 + 8 * buf);
            }
            const int64_t m = m0 + 32 * q + lane;
            if (failed || m >= args.M) continue;
            const qnn_qparams qa = args.pa[args.a_per_row ? m : 0];
            const int za = qa.z, ra = args.rsA[m];
            const float Qa = qa.Q;
#pragma unroll
            for (int j = 0; j < NJ; ++j) {
                const int c0 = half * (BN / 2) + 32 * j;
                const int64_t nb = n0 + c0;
                if (nb >= args.N) continue;
                const bool full = vec && nb + 32 <= args.N;
                float *yr = args.Y ? args.Y + m * args.ldy + nb : nullptr;
#pragma unroll
                for (int v4 = 0; v4 < 8; ++v4) {
                    float y[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int i = 4 * v4 + e;
                        const ColConst v = cc[c0 + i];
                        const int acc = run[j][i] + 128 * (ra + v.cs) - 16384 * K;  // raw code product
                        y[e] = recover_product(offset_product(acc, za, v.zw, ra, v.cs, K), Qa, v.Qw);
                        if (args.bias) y[e] = __fadd_rn(y[e], v.bias);
                        if (args.acc_out && nb + i < args.N) args.acc_out[m * args.N + nb + i] = acc;
                    }
                    if (full) {
                        *reinterpret_cast<float4 *>(yr + 4 * v4) = make_float4(y[0], y[1], y[2], y[3]);
                    } else if (yr) {
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (nb + 4 * v4 + e < args.N) yr[4 * v4 + e] = y[e];
                    }
                }
            }
        }
    } else if constexpr (EPI == kEpiRow) {
        // ---------------- epilogue (warps 2..17): recovered product, one row per lane ----------------
        // Each lane owns one output row; the four warps of a lane quarter take its 16-column blocks
        // in turn: eq. (1)'s offsets and eq. (3)'s recovery per element, stored as 16-byte vectors
        // (ragged edges element by element). The column constants of the tile are staged in shared
        // memory (double-buffered by tile parity; one named barrier of the epilogue warps per tile).
        ColConst *scol = reinterpret_cast<ColConst *>(smem + STAGES * TL::STAGE_BYTES);
        ColUnit *sunit = reinterpret_cast<ColUnit *>(scol + 2 * BN);
        const int q = warp & 3;
        const int part = (warp - 2) >> 2;
        const int ew = warp - 2;
        const int K = args.K;
        const bool vec = args.Y && (args.ldy % 4 == 0) && ((reinterpret_cast<uintptr_t>(args.Y) & 15) == 0);
        // Every epilogue warp runs every tile (the named barrier counts on it); after a wait gave
        // up, the remaining tiles are skipped without waiting.
        int64_t gc = 0;
        bool failed = false;
        for (int64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
            int64_t m0, n0;
            tile_origin(tile, tiles_m, tiles_n, BN, m0, n0);
            ColConst *cc = scol + (gc & 1) * BN;
            ColUnit *cu = sunit + (gc & 1) * BN;
            for (int c = ew * 32 + lane; c < BN; c += 32 * TL::EPI_WARPS) {
                const int64_t n = n0 + c;
                ColConst v{0, 0, 1.0f, 0.0f, 0.0f};
                int unit = -1;
                if (n < args.N) {
                    unit = (int)(n / args.rows_per_block);
                    const qnn_qparams qw = args.pw[unit];
                    v.cs = args.csW[n];
                    v.csf = (float)v.cs;
                    v.zw = qw.z;
                    v.Qw = qw.Q;
                    v.bias = args.bias ? args.bias[n] : 0.0f;
                }
                cc[c] = v;
                cu[c].unit = unit;
            }
            asm volatile("bar.sync 1, %0;" ::"n"(32 * TL::EPI_WARPS) : "memory");
            const int64_t m = m0 + 32 * q + lane;
            const bool mv = m < args.M;
            int za = 0, ra = 0;
            float Qa = 1.0f;
            if (mv) {
                const qnn_qparams qa = args.pa[args.a_per_row ? m : 0];
                za = qa.z;
                Qa = qa.Q;
                ra = args.rsA[m];
            }
            const int za128 = 128 + za;
            const int buf = (int)(gc & 1);
            if (!failed && *reinterpret_cast<volatile int *>(&s_abort)) failed = true;
            if (!failed) {
                failed = !__all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status));
                if (failed) *reinterpret_cast<volatile int *>(&s_abort) = 1;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll 1
            for (int j = part; j < BN / 16 && !failed; j += TL::EPI_WARPS / 4) {
                const int c0 = 16 * j;
                uint32_t r[16];
                tmem_ld16(tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * BN + c0), r);
                const int64_t nb = n0 + c0;
                if (!mv || nb >= args.N) continue;
                // one weight unit across the 16 columns (the usual case): row terms hoisted
                const bool one_unit = cu[c0].unit == cu[c0 + 15].unit;  // -1 past N: ragged blocks take the general way
                long long rt = 0;
                float den = 0.0f;
                if (one_unit) {
                    const int zw = cc[c0].zw;
                    rt = (long long)(128 + zw) * ra + (long long)K * ((long long)za * zw - 16384);
                    den = __fmul_rn(Qa, cc[c0].Qw);
                }
                float *yr = args.Y ? args.Y + m * args.ldy + nb : nullptr;
                const bool full = vec && nb + 16 <= args.N;
                if (one_unit && full && !args.acc_out) {  // the usual block: no per-element branches
                    if (den >= 0x1p-60f && den <= 0x1p60f &&
                        llabs(rt) + (long long)abs(za128) * 255 * K < (1LL << 24)) {
                        const float rden = __frcp_rn(den);
                        if (args.bias)
                            row_block_f32<true>(r, cc + c0, (float)rt, (float)za128, den, rden, yr);
                        else
                            row_block_f32<false>(r, cc + c0, (float)rt, (float)za128, den, rden, yr);
                    } else if (args.bias) {
                        row_block_fast<true>(r, cc + c0, rt, za128, den, yr);
                    } else {
                        row_block_fast<false>(r, cc + c0, rt, za128, den, yr);
                    }
                    continue;
                }
#pragma unroll
                for (int v4 = 0; v4 < 4; ++v4) {
                    float y[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int i = 4 * v4 + e;
                        const ColConst v = cc[c0 + i];
                        const int P = f32_integer_to_s32(__uint_as_float(r[i]));
                        long long S;
                        float dn;
                        if (one_unit) {
                            S = (long long)P + rt + (long long)za128 * v.cs;
                            dn = den;
                        } else {
                            S = (long long)P + (long long)(128 + v.zw) * ra + (long long)za128 * v.cs +
                                (long long)K * ((long long)za * v.zw - 16384);
                            dn = __fmul_rn(Qa, v.Qw);
                        }
                        y[e] = __fdiv_rn(s64_to_f32_rn(S), dn);
                        if (args.bias) y[e] = __fadd_rn(y[e], v.bias);
                        if (args.acc_out && nb + i < args.N)
                            args.acc_out[m * args.N + nb + i] = P + 128 * (ra + v.cs) - 16384 * K;  // raw code product
                    }
                    if (full) {
                        *reinterpret_cast<float4 *>(yr + 4 * v4) = make_float4(y[0], y[1], y[2], y[3]);
                    } else if (yr) {
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (nb + 4 * v4 + e < args.N) yr[4 * v4 + e] = y[e];
                    }
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mb_arrive(drained0 + 8 * buf);
            ++gc;
        }
    } else if constexpr (EPI == kEpiPartial) {
        // ---------------- epilogue (warps 2..17): split-K partial sums ----------------
        // The item's K range is at most one accumulation chunk, so its fp32 accumulator holds the
        // exact integer sum of centered products; each lane stores its row's 16-column blocks.
        const int q = warp & 3;
        const int part = (warp - 2) >> 2;
        int64_t gc = 0;
        bool ok = true;
        const bool vec = args.ldpart % 4 == 0;
        for (int64_t item = blockIdx.x; item < items && ok; item += gridDim.x, ++gc) {
            int64_t m0, n0;
            item_origin(item / splits, m0, n0);
            int32_t *dst = args.part + (item % splits) * args.M * args.ldpart;
            const int64_t m = m0 + 32 * q + lane;
            const int buf = (int)(gc & 1);
            ok = __all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status));
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll 1
            for (int j = part; j < BN / 16; j += TL::EPI_WARPS / 4) {
                uint32_t r[16];
                tmem_ld16(tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * BN + 16 * j), r);
                const int64_t nb = n0 + 16 * j;
                if (m >= args.M || nb >= args.N) continue;
                int32_t *o = dst + m * args.ldpart + nb;
                if (vec && nb + 16 <= args.N) {
#pragma unroll
                    for (int v4 = 0; v4 < 4; ++v4)
                        *reinterpret_cast<int4 *>(o + 4 * v4) =
                            make_int4(f32_integer_to_s32(__uint_as_float(r[4 * v4])),
                                      f32_integer_to_s32(__uint_as_float(r[4 * v4 + 1])),
                                      f32_integer_to_s32(__uint_as_float(r[4 * v4 + 2])),
                                      f32_integer_to_s32(__uint_as_float(r[4 * v4 + 3])));
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i)
                        if (nb + i < args.N) o[i] = f32_integer_to_s32(__uint_as_float(r[i]));
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mb_arrive(drained0 + 8 * buf);
        }
    } else {
        // ---------------- epilogue: LSTM cell update ----------------
        // Column n of the tile is gate g = (n % 32) / 8 of cell 8 * (n / 32) + n % 8. Each lane owns
        // one batch row; the warps of a lane quarter take slices of CPS cells in turn, reading the
        // four gates of their cells from tensor memory, so a thread has everything for eq. (1)/(3)
        // and the cell update of CPS cells.
        constexpr int CPS = TL::CPS;
        constexpr int SLICES = BN / (4 * CPS);   // slices per tile
        constexpr int SPG = 8 / CPS;             // slices per 8-cell group
        const int q = warp & 3;
        const int eh = (warp - 2) >> 2;
        const int K = args.K;
        const TcLstmOut &E = args.lstm;
        const int H = E.H;
        // px and c of a tile come into shared memory by TMA, two tiles ahead: buffer i % 2 holds
        // the block's i-th tile; one thread (warp 2, lane 0) refills a buffer once every epilogue
        // warp has released it, so the loads overlap the arithmetic of the tile in between
        constexpr int CW = BN / 4;  // cells per tile
        constexpr int C_OFF = LX ? 0 : 4 * TL::PX_BOX;  // the c box within a buffer (after the px boxes)
        float *const pxs0 = reinterpret_cast<float *>(smem + STAGES * TL::STAGE_BYTES);
        const bool issuer = warp == 2 && lane == 0;
        auto issue_px = [&](int64_t t_issue, int pbuf) {
            int64_t m1, n1;
            item_origin(t_issue, m1, n1);
            const uint32_t bar = pxfull0 + 8 * pbuf;
            const uint32_t dst = su32(pxs0) + (uint32_t)(pbuf * TL::LSTM_BUF);
            mb_expect(bar, (uint32_t)TL::LSTM_TX);
            if constexpr (!LX) {
#pragma unroll
                for (int g = 0; g < 4; ++g)
                    tma_load_2d(dst + g * TL::PX_BOX, &mapPX, bar, g * H + (int)(n1 / 4), (int)m1);
            } else {  // kEpiLstmX computes the input products itself: c and the column constants (mapPX
                      // then maps the [12][H] constant table)
                tma_load_2d(dst + TL::PX_BOX, &mapPX, bar, (int)(n1 / 4), 0);
            }
            tma_load_2d(dst + C_OFF, &mapC, bar, (int)(n1 / 4), (int)m1);
        };
        if (issuer) {
            if (blockIdx.x < work) issue_px(blockIdx.x, 0);
            if (blockIdx.x + gridDim.x < work) issue_px(blockIdx.x + gridDim.x, 1);
        }
        // kEpiLstmX with one weight unit per gate matrix: the correctly rounded reciprocals of the
        // per-row, per-gate divisors Qa Qw of eq. (3) are computed once for the block's row tile and
        // kept (in this thread's shared-memory slots) while it stays on that tile; the other row
        // terms are cheap to re-form
        int64_t cm0 = -1;
        bool fastrow = false;
        float *const rcw = pxs0 + 2 * (TL::LSTM_BUF / 4) + (warp - 2) * 24 * 32;  // this warp's constants
        float4 *const rq = reinterpret_cast<float4 *>(rcw) + lane;                 // rq[32 g]
        float2 *const rd = reinterpret_cast<float2 *>(rcw + 16 * 32) + lane;       // rd[32 g]
        int64_t gc = 0;
        bool ok = true;
        // row b's units and code sums: za, Qa, rs of h_{t-1}; zx, Qx, rsx of x_t (kEpiLstmX)
        int64_t lm0 = -1;
        int za = 0, rs = 0, zx = 0, rsx = 0;
        float Qa = 1.0f, Qx = 1.0f;
        for (int64_t tile = blockIdx.x; tile < work && ok; tile += gridDim.x) {
            int64_t m0, n0;
            const int slices = item_origin(tile, m0, n0) ? SLICES / 2 : SLICES;  // half-width items: half the slices
            const int pbuf = (int)(gc & 1);  // this tile's px/c buffer (gc counts the block's tiles)
            const float *pxb = pxs0 + pbuf * (TL::LSTM_BUF / 4);
            const int rl = 32 * q + lane;    // row within the tile
            const int64_t b = m0 + 32 * q + lane;
            const bool bv = b < args.M;
            if (m0 != lm0) {  // the row's units and code sums (kept while the block stays on this row tile)
                lm0 = m0;
                za = 0, rs = 0, Qa = 1.0f, zx = 0, rsx = 0, Qx = 1.0f;
                if (bv) {
                    const qnn_qparams qa = args.pa[b];
                    za = qa.z;
                    Qa = qa.Q;
                    rs = args.rsA[b];
                }
                if (LX && bv) {
                    const qnn_qparams qa = args.pa_x[b * args.x_stride];
                    zx = qa.z;
                    Qx = qa.Q;
                    rsx = args.rsA_x[b * args.x_stride];
                }
            }
            const int za128 = 128 + za;
            const float za128f = (float)za128;
            const float zx128f = (float)(128 + zx);
            if (LX && E.ups == 1 && m0 != cm0) {
                // The fast path forms S = P + rt_g + (128 + z_row) cs of eq. (1) in fp32: the tensor-core
                // sum P is an exact integer, and when |rt_g| + |128 + z_row| 255 K < 2^24 the offset term
                // rt_g + (128 + z_row) cs is an exact integer too (cs <= 255 K) and one fused multiply-add
                // forms it without rounding, so the single rounded addition P + (offset term) equals the
                // correctly rounded S (S itself stays below 2^31 when K max|a' + za| max|w' + zw| < 2^31).
                // The quotient S / (Qa Qw) is the correctly rounded q + (S - q d) r with r = RN(1/d),
                // q = RN(S r) (Markstein's final step), which needs d and r far from the ends of the fp32
                // range. Rows outside these bounds take the general path below.
                cm0 = m0;
                const long long ax = max(abs(zx), abs(zx + 255)), ah = max(abs(za), abs(za + 255));
                bool f = bv;
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const qnn_qparams qw = args.pw_x[g], qh = args.pw[g];
                    const float dx = __fmul_rn(Qx, qw.Q), dh = __fmul_rn(Qa, qh.Q);
                    const long long rtx = (long long)(128 + qw.z) * rsx + (long long)args.K_x * ((long long)zx * qw.z - 16384);
                    const long long rth = (long long)(128 + qh.z) * rs + (long long)K * ((long long)za * qh.z - 16384);
                    // (rt_x, rt_h exact when the bound below holds)
                    rq[32 * g] = make_float4(__frcp_rn(dx), __frcp_rn(dh), (float)rtx, (float)rth);
                    rd[32 * g] = make_float2(dx, dh);
                    f &= (long long)args.K_x * ax * (long long)max(abs(qw.z), abs(qw.z + 255)) < (1LL << 31) &&
                         (long long)K * ah * (long long)max(abs(qh.z), abs(qh.z + 255)) < (1LL << 31) &&
                         llabs(rtx) + (long long)abs(128 + zx) * 255 * args.K_x < (1LL << 24) &&
                         llabs(rth) + (long long)abs(za128) * 255 * K < (1LL << 24) &&
                         dx >= 0x1p-60f && dx <= 0x1p60f && dh >= 0x1p-60f && dh <= 0x1p60f;
                }
                fastrow = f;
            }
            const int buf = (int)(gc & 1);
            ok = __all_sync(0xffffffffu, mb_wait(chunk0 + 8 * buf, (unsigned)(gc / 2) & 1, args.status) &&
                                             mb_wait(pxfull0 + 8 * pbuf, (unsigned)(gc / 2) & 1, args.status));
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll 1
            for (int s = eh; s < slices; s += TL::EPI_WARPS / 4) {
                const int gi = s / SPG, part = s % SPG;
                const int j0 = (int)(n0 / 4) + gi * 8 + part * CPS;  // H is a multiple of 4: all CPS valid or none
                if constexpr (LX) {
                    // pre = (R(x_t Wx) + b) + R(h_{t-1} Wh): both exact sums recovered as in eq. (1)/(3)
                    // (the input side exactly as the batched product computes px), then the cell
                    const bool valid = bv && j0 < H;
                    const int jt = j0 - (int)(n0 / 4);  // cell within the tile
                    const uint32_t tx = tmem_base + ((uint32_t)(32 * q) << 16) +
                                        (uint32_t)(buf * TL::ACC_COLS + gi * 32 + part * CPS);
                    // column constants of the slice from shared memory: bias, Wx and Wh row code sums (the
                    // sums as exact fp32 integers)
                    const float *colb = pxb + TL::PX_BOX / 4 + jt;
                    // two cells at a time (fewer live registers): the four gates' x and h sums from
                    // tensor memory (warp-wide loads), eq. (1)/(3), then the cell update. Rows whose
                    // constants were cached take reciprocal-based quotients and 32-bit sums; the others
                    // the general way (any weight unit, 64-bit sums when needed, IEEE divides).
                    const int unit = j0 / E.cpu;
                    // the slice's cell state in, and its new state and outputs out, as one vector each
                    float cst[CPS], mst[CPS];
                    if (valid) ld_vec(pxb + C_OFF / 4 + rl * CW + jt, cst);
#pragma unroll
                    for (int c2 = 0; c2 < CPS; c2 += 2) {
                        uint32_t rx[4][2], rh[4][2];
#pragma unroll
                        for (int g = 0; g < 4; ++g) {
                            tmem_ld_nowait(tx + 8 * g + c2, rx[g]);
                            tmem_ld_nowait(tx + BN + 8 * g + c2, rh[g]);
                        }
                        tmem_wait_ld();
                        if (!valid) continue;
                        float pre[4][2];
                        if (fastrow) {
#pragma unroll
                            for (int g = 0; g < 4; ++g) {
                                float bias[2], csx[2], csh[2];
                                ld_vec(colb + g * CW + c2, bias);
                                ld_vec(colb + (4 + g) * CW + c2, csx);
                                ld_vec(colb + (8 + g) * CW + c2, csh);
                                const float4 rr = rq[32 * g];  // 1/dx, 1/dh, rt_x, rt_h
                                const float2 dd = rd[32 * g];  // dx, dh
                                const float dx = dd.x, dh = dd.y, rcx = rr.x, rch = rr.y;
                                // S = P + (rt + (128 + z) cs): the offset term exact, then one rounding
                                const float2 ox = ffma2_rn(f2(zx128f), make_float2(csx[0], csx[1]), f2(rr.z));
                                const float2 oh = ffma2_rn(f2(za128f), make_float2(csh[0], csh[1]), f2(rr.w));
                                const float2 vx = fadd2_rn(make_float2(__uint_as_float(rx[g][0]), __uint_as_float(rx[g][1])), ox);
                                const float2 vh = fadd2_rn(make_float2(__uint_as_float(rh[g][0]), __uint_as_float(rh[g][1])), oh);
                                const float2 yx = fadd2_rn(div_by_recip2(vx, dx, rcx), make_float2(bias[0], bias[1]));
                                const float2 y = fadd2_rn(yx, div_by_recip2(vh, dh, rch));
                                pre[g][0] = y.x;
                                pre[g][1] = y.y;
                            }
                        } else {
                            const long long ax = max(abs(zx), abs(zx + 255)), ah = max(abs(za), abs(za + 255));
#pragma unroll
                            for (int g = 0; g < 4; ++g) {
                                const qnn_qparams qw = args.pw_x[g * E.ups + unit], qh = args.pw[g * E.ups + unit];
                                const long long rtx = (long long)(128 + qw.z) * rsx +
                                                      (long long)args.K_x * ((long long)zx * qw.z - 16384);
                                const long long rth =
                                    (long long)(128 + qh.z) * rs + (long long)K * ((long long)za * qh.z - 16384);
                                const float dx = __fmul_rn(Qx, qw.Q), dh = __fmul_rn(Qa, qh.Q);
                                const bool fits =
                                    (long long)args.K_x * ax * (long long)max(abs(qw.z), abs(qw.z + 255)) < (1LL << 31) &&
                                    (long long)K * ah * (long long)max(abs(qh.z), abs(qh.z + 255)) < (1LL << 31);
                                float bias[2], csxf[2], cshf[2];
                                ld_vec(colb + g * CW + c2, bias);
                                ld_vec(colb + (4 + g) * CW + c2, csxf);
                                ld_vec(colb + (8 + g) * CW + c2, cshf);
                                const int csx[2] = {__float2int_rn(csxf[0]), __float2int_rn(csxf[1])};
                                const int csh[2] = {__float2int_rn(cshf[0]), __float2int_rn(cshf[1])};
#pragma unroll
                                for (int jj = 0; jj < 2; ++jj) {
                                    const int Px = f32_integer_to_s32(__uint_as_float(rx[g][jj]));
                                    const int Ph = f32_integer_to_s32(__uint_as_float(rh[g][jj]));
                                    float vx, vh;
                                    if (fits) {
                                        vx = __int2float_rn((int)((uint32_t)Px + (uint32_t)rtx +
                                                                  (uint32_t)(128 + zx) * (uint32_t)csx[jj]));
                                        vh = __int2float_rn((int)((uint32_t)Ph + (uint32_t)rth +
                                                                  (uint32_t)za128 * (uint32_t)csh[jj]));
                                    } else {
                                        vx = s64_to_f32_rn((long long)Px + rtx + (long long)(128 + zx) * csx[jj]);
                                        vh = s64_to_f32_rn((long long)Ph + rth + (long long)za128 * csh[jj]);
                                    }
                                    const float yx = __fadd_rn(__fdiv_rn(vx, dx), bias[jj]);
                                    pre[g][jj] = __fadd_rn(yx, __fdiv_rn(vh, dh));
                                }
                            }
                        }
                        float2 cv = make_float2(cst[c2], cst[c2 + 1]);
                        const float2 mv = lstm_cell2(make_float2(pre[0][0], pre[0][1]), make_float2(pre[1][0], pre[1][1]),
                                                     make_float2(pre[2][0], pre[2][1]), make_float2(pre[3][0], pre[3][1]),
                                                     cv);
                        cst[c2] = cv.x, cst[c2 + 1] = cv.y;
                        mst[c2] = mv.x, mst[c2 + 1] = mv.y;
                    }
                    if (valid) {
                        st_vec(E.c + b * (int64_t)H + j0, cst);
                        st_vec(E.h + b * E.h_ld + j0, mst);
                    }
                    continue;
                }
                uint32_t r[4][CPS];
                const uint32_t ta = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * BN + gi * 32 + part * CPS);
#pragma unroll
                for (int g = 0; g < 4; ++g) tmem_ld_nowait(ta + 8 * g, r[g]);
                tmem_wait_ld();
                if (bv && j0 < H) {
                    // eq. (1) expanded around the centered product P: S = P + rt[g] + (128 + za) csW,
                    // with the weight unit of the slice's cells (one per gate matrix, or per block)
                    // S sums K products (a' + za)(w' + zw) of magnitude at most amax * wmax, so when
                    // K amax wmax < 2^31 it fits in 32 bits and wrapping 32-bit arithmetic gives it
                    // exactly (the usual case: offsets within [-255, 255]); otherwise 64-bit
                    long long rt[4];
                    float den[4];
                    const int unit = j0 / E.cpu;
                    const long long amax = max(abs(za), abs(za + 255));
                    bool fits = true;
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        const qnn_qparams qw = args.pw[g * E.ups + unit];
                        rt[g] = (long long)(128 + qw.z) * rs + (long long)K * ((long long)za * qw.z - 16384);
                        den[g] = __fmul_rn(Qa, qw.Q);
                        fits &= (long long)K * amax * (long long)max(abs(qw.z), abs(qw.z + 255)) < (1LL << 31);
                    }
                    const int jt = j0 - (int)(n0 / 4);  // cell within the tile
                    const float *pxr = pxb + rl * CW + jt;
                    float *cr = E.c + b * (int64_t)H + j0;
                    float pre[4][CPS];
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        float pv[CPS];
                        int csv[CPS];
                        ld_vec(pxr + g * (TL::PX_BOX / 4), pv);
                        ld_vec(args.csW + g * H + j0, csv);
#pragma unroll
                        for (int jj = 0; jj < CPS; ++jj) {
                            const int P = f32_integer_to_s32(__uint_as_float(r[g][jj]));
                            float x;
                            if (fits) {
                                const uint32_t u = (uint32_t)P + (uint32_t)rt[g] + (uint32_t)za128 * (uint32_t)csv[jj];
                                x = __int2float_rn((int)u);
                            } else {
                                x = s64_to_f32_rn((long long)P + rt[g] + (long long)za128 * csv[jj]);
                            }
                            pre[g][jj] = __fadd_rn(pv[jj], __fdiv_rn(x, den[g]));
                        }
                    }
                    float cv[CPS], mv[CPS];
                    ld_vec(pxb + C_OFF / 4 + rl * CW + jt, cv);
#pragma unroll
                    for (int jj = 0; jj < CPS; ++jj) lstm_cell(pre[0][jj], pre[1][jj], pre[2][jj], pre[3][jj], cv[jj], mv[jj]);
                    st_vec(cr, cv);
                    st_vec(E.h + b * E.h_ld + j0, mv);
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
                mb_arrive(drained0 + 8 * buf);
                mb_arrive(pxempty0 + 8 * pbuf);
            }
            // refill the buffer with the tile two ahead once every epilogue warp has released it
            if (issuer && tile + 2 * (int64_t)gridDim.x < work &&
                mb_wait(pxempty0 + 8 * pbuf, (unsigned)(gc / 2) & 1, args.status))
                issue_px(tile + 2 * (int64_t)gridDim.x, pbuf);
            ++gc;
        }
        if (!ok) s_abort = 1;  // copies may still be in flight: the block waits for them before leaving
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
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "n"(TL::TMEM_COLS)
                     : "memory");
    }
}

// Two codes (bytes lo and hi of w selected by sel) as two centered fp16 values c - 128: the byte
// placed under the exponent pattern 0x64 is the fp16 value 1024 + c (exact), and 1024 + 128 is
// then subtracted (exact: integers below 2048).
__device__ __forceinline__ uint32_t center2(uint32_t w, uint32_t sel) {
    const uint32_t bits = __byte_perm(w, 0x64646464u, sel);
    const __half2 v = __hsub2(*reinterpret_cast<const __half2 *>(&bits), __halves2half2(__ushort_as_half(0x6480),
                                                                                      __ushort_as_half(0x6480)));
    return *reinterpret_cast<const uint32_t *>(&v);
}

// u8 codes -> centered fp16 (c - 128), rows padded with zeros to ldo (a multiple of 64). A thread
// converts 16 codes: one 16-byte load and two 16-byte stores when the row is 16-byte aligned and
// the 16 codes lie inside K, element by element otherwise (ragged tail, padding, unaligned rows).
__global__ void center_fp16_kernel(const uint8_t *__restrict__ in, int64_t rows, int K, int64_t ldi,
                                   __half *__restrict__ out, int ldo) {
    const int per_row = ldo / 16;
    const int64_t total = rows * (int64_t)per_row;
    const bool vec = (reinterpret_cast<uintptr_t>(in) & 15) == 0 && ldi % 16 == 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / per_row;
        const int k0 = (int)(i - r * per_row) * 16;
        uint4 o[2];
        if (vec && k0 + 16 <= K) {
            const uint4 w = *reinterpret_cast<const uint4 *>(in + r * ldi + k0);
            o[0] = make_uint4(center2(w.x, 0x4140u), center2(w.x, 0x4342u), center2(w.y, 0x4140u), center2(w.y, 0x4342u));
            o[1] = make_uint4(center2(w.z, 0x4140u), center2(w.z, 0x4342u), center2(w.w, 0x4140u), center2(w.w, 0x4342u));
        } else {
            __align__(16) __half v[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int k = k0 + e;
                v[e] = k < K ? __int2half_rn((int)in[r * ldi + k] - 128) : __int2half_rn(0);
            }
            o[0] = reinterpret_cast<const uint4 *>(v)[0];
            o[1] = reinterpret_cast<const uint4 *>(v)[1];
        }
        uint4 *dst = reinterpret_cast<uint4 *>(out + r * ldo + k0);
        dst[0] = o[0];
        dst[1] = o[1];
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
            return QNN_FAIL(QNN_ERR_CUDA);
        }
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    *out = g_encode;
    return QNN_OK;
}

// 2-D fp32 tensor: rows of `cols` values, `ld` values apart (ld a multiple of 4, base 16-byte
// aligned), boxes of box_cols x box_rows, no swizzle (rows of the box land box_cols * 4 bytes apart).
qnn_status make_map_f32(CUtensorMap *map, const float *base, int64_t rows, int64_t cols, int64_t ld, int box_cols,
                        int box_rows) {
    if ((reinterpret_cast<uintptr_t>(base) & 15) || ld % 4 || box_cols % 4) return QNN_ERR_INVALID_ARG;
    PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
    QNN_TRY(get_encode(&enc));
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(ld * 4)};
    cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? QNN_OK : QNN_FAIL(QNN_ERR_CUDA);
}

// 2-D fp16 tensor [rows][ld] (ld a multiple of 64), boxes of 64 x box_rows, 128-byte swizzle.
qnn_status make_map(CUtensorMap *map, const __half *base, int64_t rows, int64_t ld, int box_rows,
                    int64_t pitch = 0) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
    QNN_TRY(get_encode(&enc));
    cuuint64_t dims[2] = {(cuuint64_t)ld, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)((pitch > 0 ? pitch : ld) * 2)};  // rows may lie further apart
    cuuint32_t box[2] = {(cuuint32_t)TBK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half *>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? QNN_OK : QNN_FAIL(QNN_ERR_CUDA);
}

}  // namespace

size_t tc_scratch_bytes(int64_t M, int64_t N, int64_t K) {
    const int64_t kp = (K + 63) / 64 * 64;
    return (size_t)(M + N) * kp * 2 + 512;
}

namespace {

template <int BN, int EPI>
qnn_status launch_tc(const TcOperands &op, const TcArgs &a, const char *name, cudaStream_t st,
                     const CUtensorMap *map_px = nullptr, const CUtensorMap *map_c = nullptr,
                     const CUtensorMap *map_ax = nullptr, const CUtensorMap *map_wx = nullptr) {
    using TL = Tile<BN, EPI>;
    static int configured = -1;
    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (configured != dev) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(qgemm_tc_kernel<BN, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)TL::SMEM));
        QNN_CUDA_TRY(cudaFuncSetAttribute(qgemm_tc_kernel<BN, EPI>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                          (int)cudaSharedmemCarveoutMaxShared));
        int n = 0;
        QNN_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, qgemm_tc_kernel<BN, EPI>, TL::THREADS, TL::SMEM));
        if (std::getenv("QNN_DEBUG")) {
            cudaFuncAttributes fa{};
            cudaFuncGetAttributes(&fa, qgemm_tc_kernel<BN, EPI>);
            std::fprintf(stderr, "qnn: qgemm_tc_kernel<%d,%d>: %d threads (at most %d), %d registers, %zu bytes "
                         "static and %zu dynamic shared, %zu local, %d blocks per SM\n", BN, EPI, TL::THREADS,
                         fa.maxThreadsPerBlock, fa.numRegs, fa.sharedSizeBytes, TL::SMEM, fa.localSizeBytes, n);
        }
        if (n < 1) return QNN_FAIL(QNN_ERR_CUDA);
        configured = dev;
    }
    const int64_t items = ((a.M + TBM - 1) / TBM) * ((a.N + BN - 1) / BN) * a.splits;  // (tile, K range) pairs
    // persistent: one block per SM (a block holding tensor memory has its SM to itself)
    const int64_t blocks = op.max_blocks > 0 ? std::min(op.max_blocks, sm_count()) : sm_count();
    const unsigned grid = (unsigned)std::min<int64_t>(items, blocks);
    // LSTM tiles of 64 or 128 columns: when the last wave is partial and its tiles, halved, fit one
    // wave, they run as two half-width items each (the busiest block then does half a tile less;
    // QNN_TC_HALF=0 keeps whole tiles)
    TcArgs args = a;
    args.full_tiles = 0;
    if (TL::IS_LSTM && op.half_items && (BN == 64 || BN == 128) && a.splits == 1 && items > grid) {
        const char *e = std::getenv("QNN_TC_HALF");
        const int64_t r = items % grid;
        if (r > 0 && 2 * r <= grid && !(e && std::strcmp(e, "0") == 0)) args.full_tiles = items - r;
    }
    ProfScope prof(name, st);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(TL::THREADS);
    cfg.dynamicSmemBytes = TL::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = op.pdl ? 1 : 0;
    // the px, c, x and Wx maps are read by the LSTM kernels only (the others get A's map, unused)
    QNN_CUDA_TRY(cudaLaunchKernelEx(&cfg, qgemm_tc_kernel<BN, EPI>, op.a, op.w, map_px ? *map_px : op.a,
                                    map_c ? *map_c : op.a, map_ax ? *map_ax : op.a, map_wx ? *map_wx : op.w, args));
    return QNN_OK;
}

qnn_status dispatch_linear(const TcOperands &op, const TcArgs &a, cudaStream_t st) {
    if (op.row_epilogue) {
        switch (op.bn) {
            case 64: return launch_tc<64, kEpiRow>(op, a, "qgemm_tc", st);
            case 128: return launch_tc<128, kEpiRow>(op, a, "qgemm_tc", st);
            default: return QNN_ERR_INVALID_ARG;
        }
    }
    switch (op.bn) {
        case 64: return launch_tc<64, kEpiLinear>(op, a, "qgemm_tc", st);
        case 128: return launch_tc<128, kEpiLinear>(op, a, "qgemm_tc", st);
        case 256: return launch_tc<256, kEpiLinear>(op, a, "qgemm_tc", st);
        default: return QNN_ERR_INVALID_ARG;
    }
}

qnn_status dispatch_lstm(const TcOperands &op, const TcArgs &a, cudaStream_t st) {
    // the epilogue's px (B rows of 4H, px_ld apart) and c (B x H) tiles, 128 rows x bn / 4 cells
    const TcLstmOut &E = a.lstm;
    CUtensorMap map_px, map_c;
    QNN_TRY(make_map_f32(&map_px, E.px, a.M, 4 * (int64_t)E.H, E.px_ld, op.bn / 4, TBM));
    QNN_TRY(make_map_f32(&map_c, E.c, a.M, E.H, E.H, op.bn / 4, TBM));
    switch (op.bn) {
        case 32: return launch_tc<32, kEpiLstm>(op, a, "lstm_gates_tc", st, &map_px, &map_c);
        case 64: return launch_tc<64, kEpiLstm>(op, a, "lstm_gates_tc", st, &map_px, &map_c);
        case 96: return launch_tc<96, kEpiLstm>(op, a, "lstm_gates_tc", st, &map_px, &map_c);
        case 128: return launch_tc<128, kEpiLstm>(op, a, "lstm_gates_tc", st, &map_px, &map_c);
        default: return QNN_ERR_INVALID_ARG;
    }
}

}  // namespace

int tc_choose_bn(int64_t M, int64_t N, const int *cands, int n) {
    if (const char *e = std::getenv("QNN_TC_BN")) {
        const int v = std::atoi(e);
        for (int i = 0; i < n; ++i)
            if (cands[i] == v) return v;
    }
    const int64_t mt = (M + TBM - 1) / TBM, sms = sm_count();
    double eff[8] = {0};
    double best = 0.0;
    for (int i = 0; i < n; ++i) {
        const int64_t tiles = mt * ((N + cands[i] - 1) / cands[i]);
        const int64_t waves = (tiles + sms - 1) / sms;
        eff[i] = (double)tiles / (double)(waves * sms);
        best = std::max(best, eff[i]);
    }
    for (int i = 0; i < n; ++i)  // candidates widest first
        if (eff[i] >= 0.9 * best) return cands[i];
    return cands[n - 1];
}

int tc_pick_bn(int64_t M, int64_t N, int64_t kp) {
    if (kp > KCHUNK) {  // chunked drains: the widest tile whose tiles fill three quarters of the SMs
        if (const char *e = std::getenv("QNN_TC_BN")) {
            const int v = std::atoi(e);
            if (v == 64 || v == 128 || v == 256) return v;
        }
        const int64_t mt = (M + TBM - 1) / TBM;
        for (int bn : {256, 128})
            if (4 * mt * ((N + bn - 1) / bn) >= 3 * (int64_t)sm_count()) return bn;
        return 64;
    }
    static const int c[] = {128, 64};  // row epilogue
    return tc_choose_bn(M, N, c, 2);
}

qnn_status tc_operands(TcOperands *op, const __half *A16, int64_t M, const __half *W16, int64_t N, int64_t kp, int bn) {
    if (bn != 32 && bn != 64 && bn != 96 && bn != 128 && bn != 256) return QNN_ERR_INVALID_ARG;
    if (kp <= 0 || kp % TBK != 0 || M <= 0 || N <= 0) return QNN_ERR_INVALID_ARG;
    QNN_TRY(make_map(&op->a, A16, M, kp, TBM));
    QNN_TRY(make_map(&op->w, W16, N, kp, bn));
    op->M = M, op->N = N, op->kp = kp, op->bn = bn, op->pdl = false;
    op->row_epilogue = kp <= KCHUNK && (bn == 64 || bn == 128);
    return QNN_OK;
}

qnn_status tc_linear(const TcOperands &op, const qnn_qparams *pa, int per_row, const int32_t *rsA, int64_t K,
                     const qnn_qparams *pw, int64_t rows_per_block, const int32_t *csW, const float *bias, float *Y,
                     int64_t ldy, int32_t *acc_out, cudaStream_t st) {
    if (K <= 0 || K > QNN_K_MAX || K > op.kp) return QNN_ERR_INVALID_ARG;
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    TcArgs a{pa, per_row, rsA, pw, rows_per_block, csW, bias, Y, ldy, acc_out, op.M, op.N, (int)K,
             (int)(op.kp / TBK), status, TcLstmOut{}, 1, (int)(op.kp / TBK), nullptr, 0};
    return dispatch_linear(op, a, st);
}

qnn_status tc_lstm_gates(const TcOperands &op, const qnn_qparams *pa, const int32_t *rsA, int64_t K,
                         const qnn_qparams *pw4, const int32_t *cs, const TcLstmOut &out, cudaStream_t st) {
    if (K <= 0 || op.kp > KCHUNK || K > op.kp || out.H <= 0 || out.H % 4 != 0) return QNN_ERR_INVALID_ARG;
    if (out.ups < 1 || out.cpu < 4 || out.cpu % 4 != 0 || out.cpu * out.ups != out.H) return QNN_ERR_INVALID_ARG;
    if (op.N != 4 * ((out.H + 7) / 8 * 8)) return QNN_ERR_INVALID_ARG;
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    TcArgs a{pa, 1, rsA, pw4, 0, cs, nullptr, nullptr, 0, nullptr, op.M, op.N, (int)K, (int)(op.kp / TBK), status, out,
             1, (int)(op.kp / TBK), nullptr, 0, 1};
    return dispatch_lstm(op, a, st);
}

qnn_status tc_lstm_gates_x(const TcOperands &op, const qnn_qparams *pa, const int32_t *rsA, int64_t K,
                           const qnn_qparams *pw4, const int32_t *cs, const TcLstmOut &out, const TcLstmInput &in,
                           cudaStream_t st) {
    if (K <= 0 || op.kp > KCHUNK || K > op.kp || out.H <= 0 || out.H % 4 != 0) return QNN_ERR_INVALID_ARG;
    if (out.ups < 1 || out.cpu < 4 || out.cpu % 4 != 0 || out.cpu * out.ups != out.H) return QNN_ERR_INVALID_ARG;
    if (op.N != 4 * ((out.H + 7) / 8 * 8)) return QNN_ERR_INVALID_ARG;
    if (in.K_x <= 0 || in.kx % TBK != 0 || in.kx > KCHUNK || in.K_x > in.kx || in.x_pitch < in.kx || in.x_pitch % 8)
        return QNN_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(in.x16) & 15) || (reinterpret_cast<uintptr_t>(in.wx16) & 15) || !in.colc)
        return QNN_ERR_INVALID_ARG;
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    const int kbh = (int)(op.kp / TBK), kbx = (int)(in.kx / TBK);
    TcArgs a{pa, 1, rsA, pw4, 0, cs, nullptr, nullptr, 0, nullptr, op.M, op.N, (int)K, kbh, status, out,
             1, kbh + kbx, nullptr, 0, 1};
    a.pa_x = in.pa, a.x_stride = in.stride, a.rsA_x = in.rs, a.pw_x = in.pw4, a.csW_x = in.cs, a.bias_x = in.bias;
    a.K_x = in.K_x, a.KB_x = kbx;
    CUtensorMap map_c, map_ax, map_wx, map_col;
    QNN_TRY(make_map_f32(&map_c, out.c, op.M, out.H, out.H, op.bn / 4, TBM));
    QNN_TRY(make_map_f32(&map_col, reinterpret_cast<const float *>(in.colc), 12, out.H, out.H, op.bn / 4, 12));
    QNN_TRY(make_map(&map_ax, in.x16, op.M, in.kx, TBM, in.x_pitch));
    QNN_TRY(make_map(&map_wx, in.wx16, op.N, in.kx, op.bn));
    switch (op.bn) {
        case 32: return launch_tc<32, kEpiLstmX>(op, a, "lstm_gates_tc", st, &map_col, &map_c, &map_ax, &map_wx);
        case 64: return launch_tc<64, kEpiLstmX>(op, a, "lstm_gates_tc", st, &map_col, &map_c, &map_ax, &map_wx);
        case 96: return launch_tc<96, kEpiLstmX>(op, a, "lstm_gates_tc", st, &map_col, &map_c, &map_ax, &map_wx);
        case 128: return launch_tc<128, kEpiLstmX>(op, a, "lstm_gates_tc", st, &map_col, &map_c, &map_ax, &map_wx);
        default: return QNN_ERR_INVALID_ARG;
    }
}

int tc_partial_splits(const TcOperands &op, int max_splits, bool fill_sms) {
    const int KB = (int)(op.kp / TBK), kpc = KCHUNK / TBK;
    const int64_t tiles = ((op.M + TBM - 1) / TBM) * ((op.N + op.bn - 1) / op.bn);
    // as many K ranges as keep the work items within one wave (without fill_sms: as few as the
    // exact chunks allow), but at least one exact chunk each
    int splits = (int)std::max<int64_t>((KB + kpc - 1) / kpc, fill_sms ? sm_count() / tiles : 1);
    splits = std::max(1, std::min({splits, KB, std::max(max_splits, (KB + kpc - 1) / kpc)}));
    const int kbs = (KB + splits - 1) / splits;  // equal ranges (the last one shorter)
    return (KB + kbs - 1) / kbs;
}

qnn_status tc_partial(const TcOperands &op, int splits, int32_t *part, int64_t ldpart, cudaStream_t st) {
    const int KB = (int)(op.kp / TBK);
    if (splits < 1 || splits > KB || (op.bn != 64 && op.bn != 128) || ldpart < op.N) return QNN_ERR_INVALID_ARG;
    const int kbs = (KB + splits - 1) / splits;
    if (kbs > KCHUNK / TBK || (KB + kbs - 1) / kbs != splits) return QNN_ERR_INVALID_ARG;  // one exact chunk each
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    TcArgs a{nullptr, 0, nullptr, nullptr, 0, nullptr, nullptr, nullptr, 0, nullptr, op.M, op.N, 0, KB, status,
             TcLstmOut{}, splits, kbs, part, ldpart, 1};
    return op.bn == 64 ? launch_tc<64, kEpiPartial>(op, a, "qgemm_tc_partial", st)
                       : launch_tc<128, kEpiPartial>(op, a, "qgemm_tc_partial", st);
}

qnn_status launch_center_fp16(const uint8_t *in, int64_t rows, int64_t K, int64_t ldi, __half *out, int64_t ldo,
                              cudaStream_t st) {
    if (rows == 0) return QNN_OK;
    const int64_t tot = rows * (ldo / 16);
    center_fp16_kernel<<<(unsigned)std::min<int64_t>((tot + 255) / 256, (int64_t)sm_count() * 16), 256, 0, st>>>(
        in, rows, (int)K, ldi, out, (int)ldo);
    QNN_CUDA_TRY(cudaGetLastError());
    return QNN_OK;
}

// Centers A and W into fp16 scratch and runs the tensor-core product (K <= QNN_K_MAX).
qnn_status launch_qgemm_tc(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA, int64_t M,
                           int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw, int64_t rows_per_block,
                           const int32_t *csW, int64_t N, const float *bias, float *Y, int64_t ldy, int32_t *acc_out,
                           void *scratch_ptr, cudaStream_t st) {
    if (M == 0 || N == 0) return QNN_OK;
    const int64_t kp = (K + 63) / 64 * 64;
    __half *A16 = reinterpret_cast<__half *>(scratch_ptr);
    __half *W16 = A16 + M * kp;
    {
        ProfScope prof("center_fp16", st);
        QNN_TRY(launch_center_fp16(A, M, K, lda, A16, kp, st));
        QNN_TRY(launch_center_fp16(W, N, K, ldw, W16, kp, st));
    }
    TcOperands op;
    QNN_TRY(tc_operands(&op, A16, M, W16, N, kp, tc_pick_bn(M, N, kp)));
    return tc_linear(op, pa, ga == QNN_PER_ROW, rsA, K, pw, rows_per_block, csW, bias, Y, ldy, acc_out, st);
}

}  // namespace qnn
