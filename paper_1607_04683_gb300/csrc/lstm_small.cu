// lstm_small.cu — the whole quantized LSTM stack for a batch of a few sequences in one persistent
// launch, organised as a dataflow pipeline of thread-block clusters (no grid-wide barrier).
//
// Roles. Each LSTM layer is one cluster of CS blocks (CS = ceil(H / 32) <= 16); block r of the
// cluster owns cells [32 r, 32 r + 32): all four gate rows of its cells in Wx and Wh, held in
// registers (warp w: cells 2w, 2w+1, i.e. 8 gate rows; lane l: bytes [16 l, 16 l + 16) of every
// row, so K <= 512). The softmax layer's 8-bit product runs in further clusters, 128 rows of Wo
// per block. Every block has 16 compute warps and one loader warp.
//
// Per frame t, in every layer block:
//   X  the loader warp has put the layer's input row for frame t (x_t, or the previous layer's
//      h_t) into a shared-memory ring; each compute warp quantizes it (one unit per row, eq. 2),
//      multiplies with its Wx rows (dp4a, u8 x u8 -> s32), reduces across the warp and recovers
//      the product plus bias (eq. 1, eq. 3, Fig. 1).
//   H  it waits until all blocks of the cluster have delivered h_{t-1} into its shared memory
//      (distributed shared memory stores + remote mbarrier arrivals), quantizes h_{t-1}, multiplies
//      with its Wh rows, adds, applies the gates and the cell update (c stays in registers) and
//      sends its two new h values to every block of the cluster; it also writes them to global
//      memory tagged with the launch's epoch, where the next layer's loader polls for them.
// Layers therefore run one frame apart, and the recurrence of a layer only waits on its own
// cluster. Every wait is bounded in time (QNN_ERR_TIMEOUT, then every block leaves its loop and
// meets its cluster at the final cluster barrier).
#include <cfloat>
#include <cstdlib>
#include <cstring>

#include "lstm_model.h"
#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int kSW = 16;                     // compute warps per block
constexpr int kSThreads = (kSW + 1) * 32;   // plus one loader warp
constexpr int kRing = 4;                    // input ring depth (frames)
constexpr int kMaxB = 4;                    // batch limit of this path
constexpr int kMaxK = 512;                  // 16 bytes of every weight row per lane
constexpr int kCellsPerBlock = 2 * kSW;     // 32
constexpr int kOutRowsPerBlock = 8 * kSW;   // 128
constexpr int kMaxLayers = 8;
constexpr unsigned long long kWaitNs = 2000000000ull;

struct SmallLayer {
    const uint8_t *wx;
    const int32_t *wx_sum;
    const qnn_qparams *wx_p;
    const uint8_t *wh;
    const int32_t *wh_sum;
    const qnn_qparams *wh_p;
    const float *bias;
    int ldx, ldh, kin;
};

struct SmallArgs {
    SmallLayer layer[kMaxLayers];
    const uint8_t *wo;
    const int32_t *wo_sum;
    const qnn_qparams *wo_p;
    const float *bo;
    int ldo;
    const float *x;           // [B][T][I]
    unsigned long long *hx;   // [L][B][T][R] tagged outputs: low 32 bits value, high 32 bits epoch
    float *h_all;             // [L][B][T][R] or null
    float *ytop;              // [B][T][R] when there is no output layer
    float *logits;            // [B][T][C]
    const float *h0, *c0;     // [L][B][R], [L][B][H]
    float *h_fin, *c_fin;     // nullable
    int *status;
    int *abort_flag;
    unsigned epoch;
    int L, I, H, R, C, B, T, CS;
};

// ---- PTX helpers --------------------------------------------------------------------------------

__device__ __forceinline__ uint32_t saddr(const void *p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

__device__ __forceinline__ unsigned long long now_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_local(uint32_t bar) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_local(uint32_t bar, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ bool mbar_try_cluster(uint32_t bar, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint32_t map_rank(uint32_t local, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}

__device__ __forceinline__ void st_cluster_f32x2(uint32_t raddr, float a, float b) {
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(raddr), "f"(a), "f"(b) : "memory");
}

__device__ __forceinline__ void mbar_arrive_remote(uint32_t raddr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(raddr) : "memory");
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ unsigned long long ld_tag(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_tag(unsigned long long *p, unsigned long long v) {
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Bounded wait helpers: false when the wait gave up (timeout recorded) or another block aborted.
struct Waiter {
    const SmallArgs *a;
    unsigned long long t0;
    __device__ bool expired() {
        if (*(volatile int *)a->abort_flag) return true;
        if (now_ns() - t0 > kWaitNs) {
            record_status(a->status, QNN_ERR_TIMEOUT);
            atomicExch(a->abort_flag, 1);
            return true;
        }
        return false;
    }
};

// Warp-uniform results: every lane of the warp gets the same answer.
__device__ __forceinline__ bool wait_local(const SmallArgs &a, uint32_t bar, unsigned parity) {
    bool ok = true;
    if (!mbar_try_local(bar, parity)) {
        Waiter w{&a, now_ns()};
        while (!mbar_try_local(bar, parity))
            if (w.expired()) {
                ok = false;
                break;
            }
    }
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ bool wait_cluster(const SmallArgs &a, uint32_t bar, unsigned parity) {
    bool ok = true;
    if (!mbar_try_cluster(bar, parity)) {
        Waiter w{&a, now_ns()};
        while (!mbar_try_cluster(bar, parity))
            if (w.expired()) {
                ok = false;
                break;
            }
    }
    return __all_sync(0xffffffffu, ok);
}

// ---- per-warp quantization of one row held in shared memory ------------------------------------

struct RowQ {
    uint32_t code[4];  // codes of bytes [16 lane, 16 lane + 16), zero past len
    int za, rs;
    float Qa;
};

// Row of `len` fp32 values in shared memory; every lane of the warp gets the unit's parameters
// (eq. 2), its 16 codes and the row code sum.
__device__ __forceinline__ RowQ quantize_row_warp(const float *row, int len, const SmallArgs &a) {
    const int lane = threadIdx.x & 31;
    const int k0 = lane * 16;
    float mn = FLT_MAX, mx = -FLT_MAX;
    bool bad = false;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int k = k0 + 4 * q;
        if (k < len) {
            float4 v = *reinterpret_cast<const float4 *>(row + k);
            float e[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (k + i < len) {
                    bad |= !isfinite(e[i]);
                    mn = fminf(mn, e[i]);
                    mx = fmaxf(mx, e[i]);
                }
        }
    }
    mn = warp_min(mn);
    mx = warp_max(mx);
    if (__any_sync(0xffffffffu, bad)) {
        if (lane == 0) record_status(a.status, QNN_ERR_NONFINITE);
        mn = 0.0f;
        mx = 0.0f;
    }
    const qnn_qparams p = params_from_range(mn, mx);
    RowQ r;
    int s = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int k = k0 + 4 * q;
        uint32_t w = 0;
        if (k < len) {
            float4 v = *reinterpret_cast<const float4 *>(row + k);
            float e[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (k + i < len) {
                    uint32_t c = quant_code(e[i], p.Q, p.z);
                    s += (int)c;
                    w |= c << (8 * i);
                }
        }
        r.code[q] = w;
    }
    r.rs = warp_sum(s);
    r.za = p.z;
    r.Qa = p.Q;
    return r;
}

// Eight row partial dot products (8 rows x 16 bytes of this lane), reduced across the warp so that
// lane l ends with the full sum of row ((l >> 2) & 7).
__device__ __forceinline__ int dot8_reduce(const uint32_t (&w)[8][4], const RowQ &q) {
    int v[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        unsigned acc = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) acc = __dp4a(w[r][i], q.code[i], acc);  // u8 x u8 summed into u32
        v[r] = (int)acc;
    }
    const int lane = threadIdx.x & 31;
    const bool b4 = lane & 16, b3 = lane & 8, b2 = lane & 4;
    int u[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int send = b4 ? v[i] : v[i + 4];
        const int keep = b4 ? v[i + 4] : v[i];
        u[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
    int x2[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int send = b3 ? u[i] : u[i + 2];
        const int keep = b3 ? u[i + 2] : u[i];
        x2[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
    const int send = b2 ? x2[0] : x2[1];
    const int keep = b2 ? x2[1] : x2[0];
    int s = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    return s;
}

__device__ __forceinline__ void load_rows(uint32_t (&w)[8][4], const uint8_t *base, int ld, int H, int kind,
                                          int first, int valid_rows, int lane) {
    // kind 0: gate rows of two cells (row r -> gate r & 3 of cell first + (r >> 2)), rows g*H + j
    // kind 1: plain rows first + r
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        int64_t row;
        bool ok;
        if (kind == 0) {
            const int j = first + (r >> 2);
            ok = j < H && (r >> 2) < valid_rows;
            row = (int64_t)(r & 3) * H + j;
        } else {
            ok = r < valid_rows;
            row = first + r;
        }
        uint4 v = make_uint4(0, 0, 0, 0);
        if (ok && lane * 16 < ld) v = *reinterpret_cast<const uint4 *>(base + row * ld + lane * 16);
        w[r][0] = v.x;
        w[r][1] = v.y;
        w[r][2] = v.z;
        w[r][3] = v.w;
    }
}

__global__ void __launch_bounds__(kSThreads, 1) lstm_small_kernel(const __grid_constant__ SmallArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    float *hbuf = reinterpret_cast<float *>(smem);                 // [2][kMaxB][kMaxK]
    float *ring = hbuf + 2 * kMaxB * kMaxK;                        // [kRing][kMaxB][kMaxK]
    uint8_t *swx = reinterpret_cast<uint8_t *>(ring + kRing * kMaxB * kMaxK);  // [8 kSW][kMaxK] Wx rows
    uint64_t *bars = reinterpret_cast<uint64_t *>(swx + 8 * kSW * kMaxK);
    const uint32_t full0 = saddr(bars), empty0 = saddr(bars + kRing), hbar0 = saddr(bars + 2 * kRing);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int CS = a.CS;
    const int cid = blockIdx.x / CS;
    const uint32_t rank = cluster_rank();
    const bool is_layer = cid < a.L;
    const int l = cid;
    const int B = a.B, T = a.T, H = a.H, R = a.R;
    const int kin = is_layer ? a.layer[l].kin : R;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(full0 + 8 * i, 32);
            mbar_init(empty0 + 8 * i, kSW);
        }
        mbar_init(hbar0, CS * kSW);
        mbar_init(hbar0 + 8, CS * kSW);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // initial state h_{-1} of this layer into hbuf[1]
    if (is_layer) {
        for (int i = threadIdx.x; i < B * kMaxK; i += kSThreads) {
            const int b = i / kMaxK, k = i % kMaxK;
            hbuf[(1 * kMaxB + b) * kMaxK + k] = k < R ? a.h0[((int64_t)l * B + b) * R + k] : 0.0f;
        }
    }
    __syncthreads();
    cluster_sync();

    bool ok = true;
    if (warp == kSW) {
        // ---------------- loader warp ----------------
        const float *xin = a.x;
        const unsigned long long *src = nullptr;
        if (!(is_layer && l == 0)) src = a.hx + (int64_t)(is_layer ? l - 1 : a.L - 1) * B * T * R;
        for (int t = 0; t < T && ok; ++t) {
            const int slot = t % kRing;
            if (t >= kRing) ok = wait_local(a, empty0 + 8 * slot, ((t / kRing) - 1) & 1);
            if (!ok) break;
            for (int b = 0; b < B && ok; ++b) {
                float *dst = ring + ((int64_t)slot * kMaxB + b) * kMaxK;
                if (src == nullptr) {
                    const float *xr = xin + ((int64_t)b * T + t) * a.I;
                    for (int k = lane; k < kin; k += 32) dst[k] = xr[k];
                } else {
                    const unsigned long long *hr = src + ((int64_t)b * T + t) * R;
                    unsigned long long v[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int k = lane + 32 * i;
                        v[i] = k < kin ? ld_tag(hr + k) : ((unsigned long long)a.epoch << 32);
                    }
                    Waiter wt{&a, now_ns()};
                    while (true) {
                        bool ready = true;
#pragma unroll
                        for (int i = 0; i < 16; ++i) ready &= (unsigned)(v[i] >> 32) == a.epoch;
                        if (__all_sync(0xffffffffu, ready)) break;
                        if (wt.expired()) {
                            ok = false;
                            break;
                        }
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int k = lane + 32 * i;
                            if (k < kin && (unsigned)(v[i] >> 32) != a.epoch) v[i] = ld_tag(hr + k);
                        }
                    }
                    ok = __all_sync(0xffffffffu, ok);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int k = lane + 32 * i;
                        if (k < kin) dst[k] = __uint_as_float((unsigned)(v[i] & 0xffffffffu));
                    }
                }
            }
            mbar_arrive_local(full0 + 8 * slot);
        }
    } else if (is_layer) {
        // ---------------- LSTM layer compute warp ----------------
        const SmallLayer &ly = a.layer[l];
        const int j0 = (int)rank * kCellsPerBlock;
        const int cell0 = j0 + 2 * warp;  // this warp's cells: cell0, cell0 + 1
        // Wh rows (the recurrent critical path) in registers, Wx rows in shared memory
        uint32_t whr[8][4];
        load_rows(whr, ly.wh, ly.ldh, H, 0, cell0, 2, lane);
        {
            uint32_t tmp[8][4];
            load_rows(tmp, ly.wx, ly.ldx, H, 0, cell0, 2, lane);
            uint8_t *mine = swx + (size_t)warp * 8 * kMaxK;
#pragma unroll
            for (int r = 0; r < 8; ++r)
                *reinterpret_cast<uint4 *>(mine + r * kMaxK + lane * 16) =
                    make_uint4(tmp[r][0], tmp[r][1], tmp[r][2], tmp[r][3]);
            __syncwarp();
        }
        const uint8_t *wx_rows = swx + (size_t)warp * 8 * kMaxK;
        const int e = (lane >> 4) & 1, g = (lane >> 2) & 3;
        const int j = cell0 + e;
        const bool jv = j < H;
        const int64_t n = (int64_t)g * H + (jv ? j : 0);
        const int csx = jv ? ly.wx_sum[n] : 0, csh = jv ? ly.wh_sum[n] : 0;
        const float bias = jv ? ly.bias[n] : 0.0f;
        const qnn_qparams px = ly.wx_p[g], ph = ly.wh_p[g];
        float c[kMaxB], yxb[kMaxB], hlast[kMaxB];
#pragma unroll
        for (int b = 0; b < kMaxB; ++b) {
            c[b] = (b < B && jv) ? a.c0[((int64_t)l * B + b) * H + j] : 0.0f;
            hlast[b] = 0.0f;
            yxb[b] = 0.0f;
        }
        const bool tag_out = (l < a.L - 1) || (a.C > 0);
        const uint32_t my_hbuf = saddr(hbuf);
        for (int t = 0; t < T && ok; ++t) {
            // X: input product of frame t
            const int slot = t % kRing;
            ok = wait_local(a, full0 + 8 * slot, (t / kRing) & 1);
            if (!ok) break;
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const RowQ q = quantize_row_warp(ring + ((int64_t)slot * kMaxB + b) * kMaxK, kin, a);
                uint32_t wx8[8][4];
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                    const uint4 v = *reinterpret_cast<const uint4 *>(wx_rows + r * kMaxK + lane * 16);
                    wx8[r][0] = v.x, wx8[r][1] = v.y, wx8[r][2] = v.z, wx8[r][3] = v.w;
                }
                const int s = dot8_reduce(wx8, q);
                const long long S = offset_product(s, q.za, px.z, q.rs, csx, kin);
                yxb[b] = __fadd_rn(recover_product(S, q.Qa, px.Q), bias);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive_local(empty0 + 8 * slot);
            // H: wait for h_{t-1} from the whole cluster (h_{-1} was preloaded)
            const int pb = (t - 1) & 1;
            if (t > 0) {
                ok = wait_cluster(a, hbar0 + 8 * pb, ((t - 1) >> 1) & 1);
                if (!ok) break;
            }
            float hv[kMaxB];
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                hv[b] = 0.0f;
                if (b >= B) break;
                const RowQ q = quantize_row_warp(hbuf + ((int64_t)pb * kMaxB + b) * kMaxK, R, a);
                const int s = dot8_reduce(whr, q);
                const long long S = offset_product(s, q.za, ph.z, q.rs, csh, R);
                const float pre = __fadd_rn(yxb[b], recover_product(S, q.Qa, ph.Q));
                const int base = lane & 16;
                const float pi = __shfl_sync(0xffffffffu, pre, base + 0);
                const float pf = __shfl_sync(0xffffffffu, pre, base + 4);
                const float pg = __shfl_sync(0xffffffffu, pre, base + 8);
                const float po = __shfl_sync(0xffffffffu, pre, base + 12);
                float m;
                lstm_cell(pi, pf, pg, po, c[b], m);
                hv[b] = jv ? m : 0.0f;
                hlast[b] = hv[b];
            }
            // send h_t: lane d < CS delivers both cells' values to block d of the cluster
            const int cb = t & 1;
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const float v0 = __shfl_sync(0xffffffffu, hv[b], 0);
                const float v1 = __shfl_sync(0xffffffffu, hv[b], 16);
                if (lane < CS && cell0 < H) {
                    const uint32_t raddr =
                        map_rank(my_hbuf + 4u * (uint32_t)(((cb * kMaxB + b) * kMaxK) + cell0), (uint32_t)lane);
                    st_cluster_f32x2(raddr, v0, v1);
                }
                // outputs to global: lanes 0 and 16 own cell0 and cell0 + 1
                if ((lane & 15) == 0 && jv) {
                    const int64_t o = (((int64_t)l * B + b) * T + t) * R + j;
                    if (tag_out)
                        st_tag(a.hx + o, ((unsigned long long)a.epoch << 32) | __float_as_uint(hv[b]));
                    if (a.h_all) a.h_all[o] = hv[b];
                    if (a.ytop && l == a.L - 1) a.ytop[((int64_t)b * T + t) * R + j] = hv[b];
                }
            }
            if (lane < CS) mbar_arrive_remote(map_rank(hbar0 + 8 * cb, (uint32_t)lane));
        }
        if (ok && (lane & 15) == 0 && jv) {
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                if (a.h_fin) a.h_fin[((int64_t)l * B + b) * R + j] = hlast[b];
                if (a.c_fin) a.c_fin[((int64_t)l * B + b) * H + j] = c[b];
            }
        }
    } else {
        // ---------------- output layer compute warp ----------------
        const int ob = (cid - a.L) * CS + (int)rank;
        const int n0 = ob * kOutRowsPerBlock + warp * 8;
        const int nv = a.C - n0 < 8 ? (a.C - n0 < 0 ? 0 : a.C - n0) : 8;
        uint32_t wor[8][4];
        load_rows(wor, a.wo, a.ldo, 0, 1, n0, nv, lane);
        const int r = (lane >> 2) & 7;
        const int n = n0 + r;
        const bool nvld = r < nv;
        const int cso = nvld ? a.wo_sum[n] : 0;
        const float bo = nvld ? a.bo[n] : 0.0f;
        const qnn_qparams po = a.wo_p[0];
        for (int t = 0; t < T && ok; ++t) {
            const int slot = t % kRing;
            ok = wait_local(a, full0 + 8 * slot, (t / kRing) & 1);
            if (!ok) break;
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const RowQ q = quantize_row_warp(ring + ((int64_t)slot * kMaxB + b) * kMaxK, R, a);
                const int s = dot8_reduce(wor, q);
                const long long S = offset_product(s, q.za, po.z, q.rs, cso, R);
                const float y = __fadd_rn(recover_product(S, q.Qa, po.Q), bo);
                if ((lane & 3) == 0 && nvld) a.logits[((int64_t)b * T + t) * a.C + n] = y;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive_local(empty0 + 8 * slot);
        }
    }
    __syncwarp();
    // no block leaves while a cluster peer may still write into its shared memory
    cluster_sync();
}

int g_small_cfg_dev = -1;

}  // namespace

PathChoice path_choice() {
    const char *v = std::getenv("QNN_LSTM_PATH");
    if (!v || !*v || std::strcmp(v, "auto") == 0) return PathChoice::kAuto;
    if (std::strcmp(v, "layerwise") == 0) return PathChoice::kLayerwise;
    if (std::strcmp(v, "small") == 0) return PathChoice::kSmall;
    return PathChoice::kAuto;
}

qnn_status small_path_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *h_state,
                              float *c_state, float *h_all, cudaStream_t st, bool *used) {
    *used = false;
    const int64_t L = m->L, I = m->I, H = m->H, C = m->C, R = m->R;
    if (m->P != 0 || B > kMaxB || L > kMaxLayers || I > kMaxK || R > kMaxK || H > kCellsPerBlock * 16) return QNN_OK;
    if (C > 0 && m->d.output_mode != QNN_OUT_QUANT) return QNN_OK;
    if (T > (int64_t)INT32_MAX / 4) return QNN_OK;
    const int CS = (int)((H + kCellsPerBlock - 1) / kCellsPerBlock);
    const int out_blocks = C > 0 ? (int)((C + kOutRowsPerBlock - 1) / kOutRowsPerBlock) : 0;
    const int out_clusters = (out_blocks + CS - 1) / CS;
    const int clusters = (int)L + out_clusters;
    const size_t smem = sizeof(float) * (2 + kRing) * kMaxB * kMaxK + (size_t)8 * kSW * kMaxK +
                        sizeof(uint64_t) * (2 * kRing + 2);

    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (g_small_cfg_dev != dev) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstm_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstm_small_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
        g_small_cfg_dev = dev;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(clusters * CS));
    cfg.blockDim = dim3(kSThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int max_clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&max_clusters, lstm_small_kernel, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return QNN_OK;
    }
    if (max_clusters < clusters) return QNN_OK;  // cannot be co-resident: layer-by-layer path

    // workspace: staging, tagged layer outputs, logits, zero state
    const bool x_dev = is_device_ptr(x), y_dev = is_device_ptr(y);
    const bool hs_dev = h_state && is_device_ptr(h_state), cs_dev = c_state && is_device_ptr(c_state);
    const bool ha_dev = h_all && is_device_ptr(h_all);
    const int64_t rows = B * T, ycols = C > 0 ? C : R;
    size_t need = 0;
    auto acct = [&](size_t n) {
        size_t at = (need + 255) / 256 * 256;
        need = at + n;
        return at;
    };
    const size_t o_flag = acct(256);
    const size_t o_hx = acct(sizeof(unsigned long long) * L * rows * R);
    const size_t o_lg = acct(C > 0 ? sizeof(float) * rows * C : 0);
    const size_t o_x = x_dev ? 0 : acct(sizeof(float) * rows * I);
    const size_t o_y = y_dev ? 0 : acct(sizeof(float) * rows * ycols);
    const size_t o_h = acct(sizeof(float) * L * B * R);
    const size_t o_c = acct(sizeof(float) * L * B * H);
    const size_t o_ha = (h_all && !ha_dev) ? acct(sizeof(float) * L * rows * R) : 0;
    if (need > m->sws_bytes) {
        if (m->sws) {
            QNN_CUDA_TRY(cudaStreamSynchronize(st));
            QNN_CUDA_TRY(cudaFree(m->sws));
            m->sws = nullptr;
            m->sws_bytes = 0;
        }
        QNN_CUDA_TRY(cudaMalloc(&m->sws, need));
        QNN_CUDA_TRY(cudaMemset(m->sws, 0, need));  // tags 0 never match an epoch (epochs start at 1)
        m->sws_bytes = need;
    }
    if (++m->epoch == 0) {  // tag space wrapped: clear every tag once
        QNN_CUDA_TRY(cudaMemsetAsync(reinterpret_cast<char *>(m->sws) + o_hx, 0,
                                     sizeof(unsigned long long) * L * rows * R, st));
        m->epoch = 1;
    }
    char *ws = reinterpret_cast<char *>(m->sws);
    SmallArgs a{};
    for (int64_t l = 0; l < L; ++l) {
        const LayerDev &ly = m->layers[l];
        a.layer[l] = SmallLayer{ly.wx.codes, ly.wx.sums, ly.wx.params, ly.wh.codes, ly.wh.sums, ly.wh.params,
                                ly.bias, (int)ly.wx.ld, (int)ly.wh.ld, (int)ly.kin};
    }
    if (C > 0) {
        a.wo = m->wo.codes, a.wo_sum = m->wo.sums, a.wo_p = m->wo.params, a.bo = m->bo, a.ldo = (int)m->wo.ld;
    }
    const float *xd = x;
    if (!x_dev) {
        QNN_CUDA_TRY(cudaMemcpyAsync(ws + o_x, x, sizeof(float) * rows * I, cudaMemcpyHostToDevice, st));
        xd = reinterpret_cast<const float *>(ws + o_x);
    }
    float *yd = y_dev ? y : reinterpret_cast<float *>(ws + o_y);
    float *h0 = reinterpret_cast<float *>(ws + o_h), *c0 = reinterpret_cast<float *>(ws + o_c);
    if (h_state)
        QNN_CUDA_TRY(cudaMemcpyAsync(h0, h_state, sizeof(float) * L * B * R, cudaMemcpyDefault, st));
    else
        QNN_CUDA_TRY(cudaMemsetAsync(h0, 0, sizeof(float) * L * B * R, st));
    if (c_state)
        QNN_CUDA_TRY(cudaMemcpyAsync(c0, c_state, sizeof(float) * L * B * H, cudaMemcpyDefault, st));
    else
        QNN_CUDA_TRY(cudaMemsetAsync(c0, 0, sizeof(float) * L * B * H, st));
    int *status = nullptr;
    QNN_TRY(status_word(&status));
    QNN_CUDA_TRY(cudaMemsetAsync(ws + o_flag, 0, 256, st));
    a.x = xd;
    a.hx = reinterpret_cast<unsigned long long *>(ws + o_hx);
    a.h_all = h_all ? (ha_dev ? h_all : reinterpret_cast<float *>(ws + o_ha)) : nullptr;
    a.ytop = C > 0 ? nullptr : yd;
    a.logits = C > 0 ? reinterpret_cast<float *>(ws + o_lg) : nullptr;
    a.h0 = h0, a.c0 = c0;
    a.h_fin = h_state ? (hs_dev ? h_state : h0) : nullptr;  // host state: written back from h0/c0 below
    a.c_fin = c_state ? (cs_dev ? c_state : c0) : nullptr;
    a.status = status;
    a.abort_flag = reinterpret_cast<int *>(ws + o_flag);
    a.epoch = m->epoch;
    a.L = (int)L, a.I = (int)I, a.H = (int)H, a.R = (int)R, a.C = (int)C, a.B = (int)B, a.T = (int)T, a.CS = CS;
    {
        ProfScope prof("lstm_small", st);
        QNN_CUDA_TRY(cudaLaunchKernelEx(&cfg, lstm_small_kernel, a));
    }
    if (C > 0) QNN_TRY(launch_softmax_rows(a.logits, rows, C, yd, st));
    if (!y_dev) QNN_CUDA_TRY(cudaMemcpyAsync(y, yd, sizeof(float) * rows * ycols, cudaMemcpyDeviceToHost, st));
    if (h_all && !ha_dev)
        QNN_CUDA_TRY(cudaMemcpyAsync(h_all, a.h_all, sizeof(float) * L * rows * R, cudaMemcpyDeviceToHost, st));
    if (h_state && !hs_dev)
        QNN_CUDA_TRY(cudaMemcpyAsync(h_state, h0, sizeof(float) * L * B * R, cudaMemcpyDeviceToHost, st));
    if (c_state && !cs_dev)
        QNN_CUDA_TRY(cudaMemcpyAsync(c_state, c0, sizeof(float) * L * B * H, cudaMemcpyDeviceToHost, st));
    *used = true;
    return QNN_OK;
}

}  // namespace qnn
