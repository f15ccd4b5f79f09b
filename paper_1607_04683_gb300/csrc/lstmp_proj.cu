// lstmp_proj.cu — one recurrent step's LSTMP projection r_t = R(Q(m_t) Wp') (Sec. 3.1, eq. 1 and
// eq. 3 applied to the projection matrix of the Sec. 4 LSTMP layer) and the quantization of r_t as
// the next step's recurrent input (eq. 2), in one launch on the sm_103a tensor cores.
//
// A cluster of kCL CTAs owns 128 rows (sequences) of the batch; CTA j of it computes the j-th
// group of P / kCL output columns over the whole reduction:
//   1. the centered fp16 codes of m_t (one unit per row, written by the row quantizer) and the
//      CTA's rows of Wp' stream in by TMA through a shared-memory ring; tcgen05.mma accumulates each
//      chunk of at most 1024 k values (exact in fp32) in its own tensor-memory buffer;
//   2. the epilogue adds the chunks as int32, applies eq. (1)'s offsets and eq. (3)'s recovery (the
//      same integer and the same two roundings as every other epilogue) and writes r_t as the layer
//      output;
//   3. the row range of r_t (all P columns) is gathered across the cluster through distributed
//      shared memory, so each CTA quantizes its own columns as the next step's codes; the row's
//      code sum is added up by one CTA of the cluster, which writes the row's unit and sum.
// Only the small per-row ranges and sums cross the cluster: partial products never leave a CTA
// (a split of the reduction across CTAs would move 224 KB a CTA through distributed shared
// memory, which measured tens of GB/s per SM on this part).
// Every mbarrier wait is bounded in time (a wait that gives up records QNN_ERR_TIMEOUT and the CTA
// skips ahead); every thread passes every cluster barrier on every path, so no CTA waits on one
// that has left.
#include <algorithm>
#include <cfloat>
#include <cuda.h>
#include <cuda_fp16.h>

#include "qnn_device.cuh"
#include "qnn_host.h"
#include "tc_gemm.h"
#include "tc_ptx.cuh"

namespace qnn {
namespace {

constexpr int kCL = 8;                 // CTAs per cluster: the column groups of one row block
constexpr int kRows = 128;             // rows per cluster (the MMA's M)
constexpr int kNcMax = 64;             // columns per CTA (P / kCL)
constexpr int kKps = 2;                // k-blocks (64 values) per pipeline stage
constexpr int kStages = 4;
constexpr int kChunkKb = 16;           // k-blocks per exact accumulation chunk (1024 values)
constexpr int kEpiWarps = 16;          // epilogue warps (warps 2..17): four per tensor-memory lane quarter
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kABytes = kRows * 128;                  // one k-block of A (128 rows x 64 fp16)
constexpr int kWBytes = kNcMax * 128;                 // one k-block of the CTA's Wp' rows (at most)
constexpr int kStageBytes = kKps * (kABytes + kWBytes);
// shared-memory layout (offsets from the 1024-byte-aligned base); a stage is [A sub-tiles][W sub-tiles]
constexpr int OFF_COL = kStages * kStageBytes;        // [kNcMax] column constants
constexpr int OFF_RNG = OFF_COL + kNcMax * 16;        // [4 parts][kRows] (min, max) of r_t: the 4 warps of a row
constexpr int OFF_SUM = OFF_RNG + 4 * kRows * 8;      // [4 parts][kRows] code sums
constexpr int OFF_XRNG = OFF_SUM + 4 * kRows * 4;     // [kCL][kRows] (min, max) of each CTA's columns
constexpr int OFF_XRS = OFF_XRNG + kCL * kRows * 8;   // [kCL][kRows] code sums of each CTA's columns
constexpr int OFF_BAR = OFF_XRS + kCL * kRows * 4;    // full[kStages], empty[kStages], mma_done
constexpr int OFF_TMEM = OFF_BAR + (2 * kStages + 1) * 8;
constexpr int SMEM_BYTES = OFF_TMEM + 16 + 1024;      // + slack for aligning the base
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory");
static_assert(SMEM_BYTES > 114 * 1024, "one CTA per SM: its tensor-memory allocation never waits");
constexpr unsigned long long kWaitNs = 2000000000ull;

struct ColConst {
    int cs, zw;
    float Qw;
    int pad;
};

struct ProjArgs {
    const qnn_qparams *prm_m;  // [B] units of the m_t rows (the product's activations)
    const int32_t *rs_m;       // [B] their code sums
    const qnn_qparams *wp_p;   // Wp units, rows_per_unit rows each
    const int32_t *wp_sum;     // [P] Wp row code sums
    int rows_per_unit;
    float *out;                // r_t: row b at out + b * ldo
    int64_t ldo;
    int B, K, P, KB;           // K: the true reduction length H; KB: k-blocks of 64 in the padded one
    int quantize;              // also quantize r_t for the next step
    int kh;                    // the next step's code pitch (== P)
    __half *dst;               // [B][kh] centered fp16 codes of r_t
    qnn_qparams *prm;          // [B] their units
    int32_t *rsum;             // [B] their code sums
    int *status;
};

__device__ __forceinline__ bool wait_bar(uint32_t bar, unsigned parity, int *status) {
    return mbar_wait_bounded(bar, parity, status, kWaitNs);
}

template <int COLS>
__device__ __forceinline__ void tmem_alloc_cols(uint32_t slot) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot), "n"(COLS) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
template <int COLS>
__device__ __forceinline__ void tmem_free_cols(uint32_t base) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(base), "n"(COLS) : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    lstmp_proj_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapW,
                      const ProjArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sb = su32(smem);
    const uint32_t full0 = sb + OFF_BAR, empty0 = full0 + 8 * kStages, mma_done = empty0 + 8 * kStages;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + OFF_TMEM);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int m0 = blockIdx.y * kRows;
    const int NC = a.P / kCL, n0 = (int)rank * NC;      // this CTA's columns
    const int nst = (a.KB + kKps - 1) / kKps;           // pipeline stages of the reduction
    const int nchunks = (a.KB + kChunkKb - 1) / kChunkKb;
    const int tcols = nchunks * NC <= 32 ? 32 : nchunks * NC <= 64 ? 64 : nchunks * NC <= 128 ? 128 : nchunks * NC <= 256 ? 256 : 512;
    const uint32_t sub_bytes = (uint32_t)(kABytes + NC * 128);
    __shared__ int s_fail;

    if (threadIdx.x == 0) {
        s_fail = 0;
        for (int i = 0; i < kStages; ++i) {
            mb_init(full0 + 8 * i, 1);
            mb_init(empty0 + 8 * i, 1);
        }
        mb_init(mma_done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {  // one fp32 accumulator of NC columns per chunk
        const uint32_t slot = su32(tmem_slot);
        switch (tcols) {
            case 32: tmem_alloc_cols<32>(slot); break;
            case 64: tmem_alloc_cols<64>(slot); break;
            case 128: tmem_alloc_cols<128>(slot); break;
            case 256: tmem_alloc_cols<256>(slot); break;
            default: tmem_alloc_cols<512>(slot); break;
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem_base = *tmem_slot;
    // every CTA of the cluster has started before any writes into another's shared memory (the
    // matching wait comes just before the first such write)
    cluster_arrive();

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapA)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&mapW)) : "memory");
            // Wp' (model weights, written before the step loop) for the first stages before the wait
            // on the previous kernel; the A tiles (its output) after it
            const int early = min(kStages, nst);
            for (int g = 0; g < early; ++g) {
                const int nv = min(kKps, a.KB - g * kKps);
                const uint32_t st = sb + g * kStageBytes;
                mb_expect(full0 + 8 * g, nv * sub_bytes);
                for (int v = 0; v < nv; ++v)
                    tma_load_2d(st + kKps * kABytes + v * kWBytes, &mapW, full0 + 8 * g, (g * kKps + v) * 64, n0);
            }
            grid_dependency_wait();
            for (int g = 0; g < nst; ++g) {
                const int s = g % kStages, nv = min(kKps, a.KB - g * kKps);
                const uint32_t st = sb + s * kStageBytes;
                if (g >= kStages) {
                    if (!wait_bar(empty0 + 8 * s, (unsigned)((g / kStages) - 1) & 1, a.status)) {
                        s_fail = 1;
                        break;
                    }
                    mb_expect(full0 + 8 * s, nv * sub_bytes);
                    for (int v = 0; v < nv; ++v)
                        tma_load_2d(st + kKps * kABytes + v * kWBytes, &mapW, full0 + 8 * s, (g * kKps + v) * 64, n0);
                }
                for (int v = 0; v < nv; ++v)
                    tma_load_2d(st + v * kABytes, &mapA, full0 + 8 * s, (g * kKps + v) * 64, m0);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const uint32_t idesc = mma_idesc_f16(kRows, NC);
            bool ok = true;
            for (int g = 0; g < nst && ok; ++g) {
                const int s = g % kStages, nv = min(kKps, a.KB - g * kKps);
                if (!wait_bar(full0 + 8 * s, (unsigned)(g / kStages) & 1, a.status)) {
                    ok = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t st = sb + s * kStageBytes;
                for (int v = 0; v < nv; ++v) {
                    const int kb = g * kKps + v;
                    const uint32_t d = tmem_base + (uint32_t)((kb / kChunkKb) * NC);
                    const uint64_t da = smem_desc(st + v * kABytes), dw = smem_desc(st + kKps * kABytes + v * kWBytes);
#pragma unroll
                    for (int k = 0; k < 4; ++k)  // 16 fp16 (32 bytes) along K per MMA, inside the swizzled rows
                        mma_f16_rt(d, da + (uint64_t)(2 * k), dw + (uint64_t)(2 * k), idesc,
                                   (kb % kChunkKb == 0 && k == 0) ? 0u : 1u);
                }
                mma_commit(empty0 + 8 * s);  // frees the stage when these MMAs have read it
            }
            if (!ok) s_fail = 1;
            mma_commit(mma_done);
        }
        __syncwarp();
    } else {
        // ---------------- epilogue ----------------
        const int et = threadIdx.x - 64;
        const int q = warp & 3, part = (warp - 2) >> 2;  // tensor-memory lane quarter; column quarter
        const int row = 32 * q + lane, b = m0 + row;
        const int nv = NC / 4, c0 = part * nv;           // this thread's columns: c0 .. c0 + nv - 1
        grid_dependency_wait();  // the m_t units and sums, and this step's outputs, follow the previous kernel
        grid_dependents_launch();
        ColConst *scol = reinterpret_cast<ColConst *>(smem + OFF_COL);
        for (int c = et; c < NC; c += kEpiThreads) {
            const qnn_qparams qw = a.wp_p[(n0 + c) / a.rows_per_unit];
            scol[c] = ColConst{a.wp_sum[n0 + c], qw.z, qw.Q, 0};
        }
        int za = 0, ra = 0;
        float Qa = 1.0f;
        if (b < a.B) {
            const qnn_qparams pm = a.prm_m[b];
            za = pm.z, Qa = pm.Q, ra = a.rs_m[b];
        }
        asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
        bool ok = __all_sync(0xffffffffu, wait_bar(mma_done, 0, a.status));
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // the exact centered sums of this thread's columns: the chunks added in int32
        int run[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) run[e] = 0;
        for (int ch = 0; ch < nchunks && ok; ++ch) {
            uint32_t r4[4][4];
            const uint32_t ta = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(ch * NC + c0);
#pragma unroll
            for (int g4 = 0; g4 < 4; ++g4)
                if (4 * g4 < nv) tmem_ld_nowait(ta + 4 * g4, r4[g4]);
            tmem_wait_ld();
#pragma unroll
            for (int g4 = 0; g4 < 4; ++g4)
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (4 * g4 < nv) run[4 * g4 + e] += f32_integer_to_s32(__uint_as_float(r4[g4][e]));
        }
        // The usual case: the thread's columns share one weight unit and the sums S of eq. (1) fit in
        // 32 bits (K max|a' + za| max|w' + zw| < 2^31: wrapping 32-bit arithmetic gives them exactly),
        // so S = run + rt + (128 + za) cs and S / (Qa Qw) comes from the divisor's correctly rounded
        // reciprocal (div_by_recip: the IEEE quotient while the divisor stays within 2^-60 .. 2^60);
        // otherwise each output the general way (64-bit S, IEEE divide).
        const ColConst cf = scol[c0], cl = scol[c0 + nv - 1];
        const float d = __fmul_rn(Qa, cf.Qw);
        const bool fast = cf.zw == cl.zw && __float_as_uint(cf.Qw) == __float_as_uint(cl.Qw) &&
                          (long long)a.K * max(abs(za), abs(za + 255)) * (long long)max(abs(cf.zw), abs(cf.zw + 255)) <
                              (1LL << 31) &&
                          d >= 0x1p-60f && d <= 0x1p60f;
        const float rcp = fast ? __frcp_rn(d) : 1.0f;
        const uint32_t rt = (uint32_t)(128 + cf.zw) * (uint32_t)ra + (uint32_t)a.K * (uint32_t)(za * cf.zw - 16384);
        float v[16];
        float mn = FLT_MAX, mx = -FLT_MAX;
        bool bad = false;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            v[e] = 0.0f;
            if (e < nv) {
                const ColConst cc = scol[c0 + e];
                if (fast) {
                    const int S = (int)((uint32_t)run[e] + rt + (uint32_t)(128 + za) * (uint32_t)cc.cs);
                    v[e] = div_by_recip(__int2float_rn(S), d, rcp);
                } else {
                    const int acc = run[e] + 128 * (ra + cc.cs) - 16384 * a.K;  // raw code product
                    v[e] = recover_product(offset_product(acc, za, cc.zw, ra, cc.cs, a.K), Qa, cc.Qw);
                }
                bad |= !isfinite(v[e]);
                mn = fminf(mn, v[e]);
                mx = fmaxf(mx, v[e]);
            }
        }
        const bool bv = b < a.B && ok;
        if (bv) {
            float *o = a.out + (int64_t)b * a.ldo + n0 + c0;
            if ((reinterpret_cast<uintptr_t>(o) & 15) == 0) {
#pragma unroll
                for (int g4 = 0; g4 < 4; ++g4)
                    if (4 * g4 < nv)
                        *reinterpret_cast<float4 *>(o + 4 * g4) = make_float4(v[4 * g4], v[4 * g4 + 1], v[4 * g4 + 2], v[4 * g4 + 3]);
            } else {
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (e < nv) o[e] = v[e];
            }
        }
        cluster_wait();  // every CTA of the cluster has started
        if (a.quantize) {
            // the row's range over this CTA's columns (the four column-quarter warps of the row), then
            // to every CTA of the cluster
            float2 *srng = reinterpret_cast<float2 *>(smem + OFF_RNG);
            srng[part * kRows + row] = bad ? make_float2(__int_as_float(0x7FC00000), 0.0f) : make_float2(mn, mx);
            asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
            if (part == 0) {
                float cmn = FLT_MAX, cmx = -FLT_MAX;
                bool cbad = false;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 g = srng[i * kRows + row];
                    if (isnan(g.x)) {
                        cbad = true;
                    } else {
                        cmn = fminf(cmn, g.x);
                        cmx = fmaxf(cmx, g.y);
                    }
                }
                const uint32_t u0 = cbad ? 0x7FC00000u : __float_as_uint(cmn), u1 = __float_as_uint(cmx);
                const uint32_t la = sb + OFF_XRNG + (uint32_t)(rank * kRows + row) * 8u;
#pragma unroll
                for (int j = 0; j < kCL; ++j) st_cluster_v2(cluster_map(la, j), u0, u1);
            }
            cluster_sync();
            mn = FLT_MAX, mx = -FLT_MAX, bad = false;
#pragma unroll
            for (int j = 0; j < kCL; ++j) {
                const float2 g = *reinterpret_cast<const float2 *>(smem + OFF_XRNG + (j * kRows + row) * 8);
                if (isnan(g.x)) {
                    bad = true;
                } else {
                    mn = fminf(mn, g.x);
                    mx = fmaxf(mx, g.y);
                }
            }
            if (bad) {  // as the row quantizer: a non-finite value gives the unit of an all-zero range
                if (part == 0 && rank == 0 && bv) record_status(a.status, QNN_ERR_NONFINITE);
                mn = 0.0f;
                mx = 0.0f;
            }
            const qnn_qparams p = params_from_range(mn, mx);
            int s = 0;
            __align__(16) __half hv[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                int cc = 128;
                if (e < nv) {
                    cc = (int)quant_code(v[e], p.Q, p.z);
                    s += cc;
                }
                hv[e] = __int2half_rn(cc - 128);
            }
            if (bv) {
                __half *d = a.dst + (int64_t)b * a.kh + n0 + c0;
                if (nv % 8 == 0 && (reinterpret_cast<uintptr_t>(d) & 15) == 0) {
#pragma unroll
                    for (int e8 = 0; e8 < 2; ++e8)
                        if (8 * e8 < nv) *reinterpret_cast<uint4 *>(d + 8 * e8) = *reinterpret_cast<const uint4 *>(hv + 8 * e8);
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        if (e < nv) d[e] = hv[e];
                }
            }
            // the row's code sum: the four warps' parts, then the CTAs' parts at the row's owner
            // (CTA row / (kRows / kCL) of the cluster), which writes the row's unit and sum
            int *ssum = reinterpret_cast<int *>(smem + OFF_SUM);
            ssum[part * kRows + row] = s;
            asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
            const uint32_t owner = (uint32_t)(row / (kRows / kCL));
            if (part == 0) {
                const int cs4 = ssum[row] + ssum[kRows + row] + ssum[2 * kRows + row] + ssum[3 * kRows + row];
                st_cluster_u32(cluster_map(sb + OFF_XRS + (uint32_t)(rank * kRows + row) * 4u, owner), (uint32_t)cs4);
            }
            cluster_sync();
            if (part == 0 && rank == owner && bv) {
                int tot = 0;
#pragma unroll
                for (int j = 0; j < kCL; ++j) tot += *reinterpret_cast<const int *>(smem + OFF_XRS + (j * kRows + row) * 4);
                a.rsum[b] = tot;
                a.prm[b] = p;
            }
        }
        if (!ok) s_fail = 1;
    }
    if (warp < 2) {  // the producer and MMA warps pass the epilogue's cluster barriers
        cluster_wait();
        if (a.quantize) {
            cluster_sync();
            cluster_sync();
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (s_fail && threadIdx.x == 0) {
        // let copies still in flight land before the CTA leaves (bounded)
        const unsigned long long t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 4000000ull) __nanosleep(1000);
    }
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        switch (tcols) {
            case 32: tmem_free_cols<32>(tmem_base); break;
            case 64: tmem_free_cols<64>(tmem_base); break;
            case 128: tmem_free_cols<128>(tmem_base); break;
            case 256: tmem_free_cols<256>(tmem_base); break;
            default: tmem_free_cols<512>(tmem_base); break;
        }
    }
}

}  // namespace

bool tc_proj_cluster_supported(int64_t H, int64_t P) {
    const int64_t KB = (H + 63) / 64, nc = P / kCL;
    return P % (16 * kCL) == 0 && nc <= kNcMax && ((KB + kChunkKb - 1) / kChunkKb) * nc <= 512;
}

qnn_status tc_lstmp_projection(const TcProjStep &s, bool pdl, cudaStream_t st) {
    if (!tc_proj_cluster_supported(s.H, s.P) || s.B <= 0 || s.kh != s.P || s.rows_per_unit <= 0 ||
        s.kp != (s.H + 63) / 64 * 64)
        return QNN_ERR_INVALID_ARG;
    static int configured = -1;
    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (configured != dev) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstmp_proj_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES));
        configured = dev;
    }
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    ProjArgs a{s.prm_m, s.rs_m, s.wp_p, s.wp_sum, (int)s.rows_per_unit, s.out, s.ldo, (int)s.B, (int)s.H, (int)s.P,
               (int)(s.kp / 64), s.quantize ? 1 : 0, (int)s.kh, s.dst, s.prm, s.rsum, status};
    ProfScope prof("lstmp_proj_tc", st);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kCL, (unsigned)((s.B + kRows - 1) / kRows));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kCL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    QNN_CUDA_TRY(cudaLaunchKernelEx(&cfg, lstmp_proj_kernel, *s.amap, *s.wmap, a));
    return QNN_OK;
}

}  // namespace qnn
