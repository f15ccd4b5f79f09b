// lstm_small.cu — the whole quantized LSTM stack for a batch of a few sequences in one persistent
// launch, organised as a dataflow pipeline of thread-block clusters (no grid-wide barrier).
//
// Roles. Each LSTM layer is one cluster of CS blocks (CS = ceil(H / 32) <= 16); block r of the
// cluster owns cells [32 r, 32 r + 32): the 128 gate rows (cell c, gate g -> local row 4 c + g)
// of Wx and Wh. The softmax layer's 8-bit product runs in further clusters, 128 rows of Wo per
// block. A block has three kinds of warps:
//   16 product warps  8 local rows each, dp4a (u8 x u8 -> s32) reduced across the warp; Wh (or
//                     Wo) rows in registers, lane l holding bytes [16 l, 16 l + 16) of each row (so
//                     K <= 512), Wx rows in shared memory.
//   4 epilogue warps  one thread per (cell, gate): recovery, bias, gate nonlinearity, and in the
//                     first lane of each quad the cell update (c stays in that register).
//   1 loader warp     brings each frame's input row into a shared-memory ring: x_t for the first
//                     layer, otherwise the previous layer's h_t, polled from global memory where
//                     it is written tagged with the launch's epoch; it also finds the row's range.
// Per frame t of a layer block:
//   X  the product warps quantize the input row cooperatively (one value per thread, eq. 2 with
//      the parameters the loader computed), multiply with Wx and hand the int32 partial sums to
//      the epilogue warps (mbarrier).
//   H  they wait until every epilogue warp of the cluster has delivered its 8 values of h_{t-1}
//      and their range (st.async into distributed shared memory, completing on a transaction-count
//      mbarrier), quantize h_{t-1} cooperatively, multiply with Wh and hand the sums over; then
//      they start the input product of frame t + 1 while the epilogue works on frame t.
//   E  the epilogue warps apply eq. 1's offsets, recover, add the bias, apply
//      the gates and the cell update, send their new h values and range to every block of the
//      cluster, and write them tagged to global memory for the next layer.
// (Streaming launches, whose inputs arrive one at a time, take H before X within each frame: the
// Wh product of frame t is done while x_t is still awaited.)
// A layer's recurrence only waits on its own cluster; consecutive layers run one frame apart. Every
// wait is bounded in time: one that gives up records QNN_ERR_TIMEOUT and raises an abort flag,
// after which all waits return at once, so every block runs its loop to the end (outputs then
// meaningless) and meets its cluster at the final cluster barrier; no block exits while a peer
// may still write into its shared memory.
#include <cfloat>
#include <cstdlib>
#include <cstring>

#include "lstm_model.h"
#include "qnn_device.cuh"
#include "qnn_host.h"

namespace qnn {
namespace {

constexpr int kPW = 16;                       // product warps
constexpr int kEW = 4;                        // epilogue warps
constexpr int kPT = kPW * 32;                 // product threads (512)
constexpr int kET = kEW * 32;                 // epilogue threads (128)
constexpr int kLoaderWarp = kPW + kEW;        // warp 20
constexpr int kSThreads = (kPW + kEW + 1) * 32;  // 672
constexpr int kRowsPW = 8;                    // local rows per product warp
constexpr int kRowShift = 2;                  // after the warp reduction lane l holds row (l >> 2) & 7
constexpr int kRing = 4;                      // input ring depth (frames)
constexpr int kMaxB = 4;                      // batch limit of this path
constexpr int kMaxK = 512;                    // 16 bytes of every weight row per lane
constexpr int kRows = 128;                    // local rows per block
constexpr int kCellsPerBlock = kRows / 4;     // 32
constexpr int kMaxCS = 16;
constexpr int kMaxLayers = 8;
constexpr unsigned long long kWaitNs = 2000000000ull;
constexpr int kSpinCheck = 512;               // polls between checks of the clock and the abort flag
constexpr int kHParts = kMaxCS * kEW;          // range partials per row: one per epilogue warp of the cluster
constexpr int kHBytes = 8 * 4 + 8;             // one epilogue warp's 8 h values of one row and their range
// Whether product warps wait for the epilogue's gate arithmetic before the next frame's input
// product (less contention on the critical path) or start it at once (overlap). Measured on
// GB300 with the 5 x 500 stack: overlapping is faster (2.1 vs 2.8 us per frame).
constexpr bool kXAfterEpilogue = false;

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
    int ups, cpu, opu;  // weight units per matrix; cells per gate unit; output rows per Wo unit
    unsigned long long wait_ns;  // limit of every wait
    // streaming (null otherwise): the first layer polls xs instead of reading x; the output blocks
    // finish the softmax in the kernel and write probs; each writer block flags every frame in done
    const unsigned long long *xs;  // [B][T][I] input rows tagged like hx, in host-mapped memory
    float *probs;                  // [B][T][C] posteriors (host-mapped)
    unsigned long long *smx;       // [B][T][nout][2] tagged (max, sum) softmax partials per output block
    unsigned *done;                // [T][writer blocks]: the launch's epoch once the block's rows of frame t are out
    int nout;                      // output blocks (output clusters x CS)
    int h_first;                   // order of a frame's products: Wh h_{t-1} before Wx x_t (latency, for
                                   // inputs that arrive one at a time) instead of Wx x_{t+1} right after
                                   // Wh h_{t-1} (throughput: it overlaps the cluster exchange)
};

// ---- shared memory layout ---------------------------------------------------------------------

struct RowMeta {  // quantized activation row: offset, scale, code sum
    int za;
    float Qa;
    int rs;
    int pad;
};

struct Smem {
    float hbuf[2][kMaxB][kMaxK];        // h_{t} of the whole layer, by frame parity (cluster writes)
    float2 hmm[2][kMaxB][kHParts];      // per source epilogue warp: range of its 8 values
    float ring[kRing][kMaxB][kMaxK];    // input rows (loader writes)
    qnn_qparams ring_p[kRing][kMaxB];   // their quantization parameters (loader computes them)
    uint8_t codes_x[kMaxB][kMaxK];      // quantized input rows of the current frame
    uint8_t codes_h[kMaxB][kMaxK];      // quantized h_{t-1}
    int acc_x[2][kMaxB][kRows];         // int32 sums [frame parity][seq][row]
    int acc_h[2][kMaxB][kRows];
    RowMeta meta_x[2][kMaxB], meta_h[2][kMaxB];
    float red_m[kPW][kMaxB], red_s[kPW][kMaxB];  // in-kernel softmax: per-warp partials
    float2 sm_fin[kMaxB];                        // (max, sum) of the whole output row
    uint8_t wx[kRows][kMaxK];            // Wx rows of this block (local row order)
    unsigned long long bar_full[kRing], bar_empty[kRing], bar_h[2], bar_ax[2], bar_ah[2], bar_ep[2];
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
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, unsigned parity) {
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
// Asynchronous stores into a peer block's shared memory; each completes `bytes` of the peer's
// mbarrier transaction count when its data has landed (no fence needed by the sender).
__device__ __forceinline__ void st_async_v4(uint32_t raddr, float4 v, uint32_t rbar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                     raddr),
                 "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
                 : "memory");
}
__device__ __forceinline__ void st_async_v2(uint32_t raddr, float a, float b, uint32_t rbar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(raddr),
                 "f"(a), "f"(b), "r"(rbar)
                 : "memory");
}
// Arrive on a local mbarrier and add `bytes` to the transaction count its phase waits for.
__device__ __forceinline__ void mbar_arrive_expect(uint32_t bar, uint32_t bytes) {
    asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}" ::"r"(bar), "r"(bytes)
                 : "memory");
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
// Host-mapped words written by the host (inputs) or read by it (frame flags): system scope.
__device__ __forceinline__ unsigned long long ld_tag_sys(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.relaxed.sys.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_flag_sys(unsigned *p, unsigned v) {
    asm volatile("st.release.sys.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void named_bar(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Bounded waits. A wait that gives up records QNN_ERR_TIMEOUT and raises the abort flag; every
// later wait then returns within kSpinCheck polls. Waits never make a warp leave its loop, so all
// warps keep executing the same sequence of named barriers and the launch always runs to its end.
// (A: any argument block with status, abort_flag and wait_ns.)
template <typename A>
struct DeadlineT {
    const A *a;
    unsigned long long t0;
    int spins;
    __device__ bool expired() {
        if (++spins < kSpinCheck) return false;
        spins = 0;
        if (*(volatile int *)a->abort_flag) return true;
        if (now_ns() - t0 > a->wait_ns) {
            record_status(a->status, QNN_ERR_TIMEOUT);
            atomicExch(a->abort_flag, 1);
            __threadfence();  // the flag is visible before anything computed after the give-up
            return true;
        }
        return false;
    }
};
using Deadline = DeadlineT<SmallArgs>;

// Whether some wait of the launch has given up (after a fence, so that data which depends on a
// give-up is never taken for good).
__device__ __forceinline__ bool aborted(const SmallArgs &a) {
    __threadfence();
    return *(volatile int *)a.abort_flag != 0;
}

template <typename A>
__device__ __forceinline__ void wait_cta(const A &a, uint32_t bar, unsigned parity) {
    if (mbar_try(bar, parity)) return;
    DeadlineT<A> d{&a, now_ns(), 0};
    while (!mbar_try(bar, parity))
        if (d.expired()) return;
}

template <typename A>
__device__ __forceinline__ void wait_cluster(const A &a, uint32_t bar, unsigned parity) {
    if (mbar_try_cluster(bar, parity)) return;
    DeadlineT<A> d{&a, now_ns(), 0};
    while (!mbar_try_cluster(bar, parity))
        if (d.expired()) return;
}

// ---- product warps ------------------------------------------------------------------------------

// Code of one value per product thread (k = tid < len) into `codes` (eq. 2 with the unit's range
// already known). Zero past len.
__device__ __forceinline__ void code_row(const float *row, int len, const qnn_qparams &p, uint8_t *codes, int tid) {
#pragma unroll
    for (int i = 0; i < kMaxK / kPT; ++i) {
        const int k = tid + i * kPT;
        codes[k] = k < len ? (uint8_t)quant_code(row[k], p.Q, p.z) : (uint8_t)0;
    }
}

// Eight row partial dot products of this lane (8 rows x 16 bytes), summed across the warp so that
// lane l ends with the full sum of local row ((l >> 2) & 7). With want_rs it also returns the
// row code sum in rs.
// `row(r)` yields this lane's 16 bytes of local row r (from registers or shared memory; a row is
// fetched only when it is multiplied, so shared-memory rows never occupy registers all at once).
// (dp4a rather than the warp-level integer MMA: on this GPU the two have the same peak rate, and
// with one to four activation rows the MMA's eight columns would be mostly wasted.)
template <typename RowBytes>
__device__ __forceinline__ int dot8(RowBytes row, const uint8_t *codes, bool want_rs, int &rs) {
    const int lane = threadIdx.x & 31;
    const uint4 cv = *reinterpret_cast<const uint4 *>(codes + lane * 16);
    const uint32_t c[4] = {cv.x, cv.y, cv.z, cv.w};
    if (want_rs) {  // warp-uniform
        unsigned bs = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) bs = __dp4a(c[i], 0x01010101u, bs);
        rs = warp_sum((int)bs);
    }
    int v[kRowsPW];
#pragma unroll
    for (int r = 0; r < kRowsPW; ++r) {
        const uint4 w = row(r);
        unsigned acc = __dp4a(w.x, c[0], 0u);
        acc = __dp4a(w.y, c[1], acc);
        acc = __dp4a(w.z, c[2], acc);
        acc = __dp4a(w.w, c[3], acc);
        v[r] = (int)acc;
    }
#pragma unroll
    for (int s = 4; s >= 2; --s) {  // halve the live rows at each exchange: 4, 2, 1
        const int half = kRowsPW >> (5 - s);
        // choose with bit masks, not a conditional: a select between two array elements can be
        // compiled into an indexed access, which would put v[] in local memory
        const int up = -((lane >> s) & 1);
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const int send = (v[i] & up) | (v[i + half] & ~up);
            const int keep = (v[i + half] & up) | (v[i] & ~up);
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 1 << s);
        }
    }
    int s = v[0] + __shfl_xor_sync(0xffffffffu, v[0], 2);
    return s + __shfl_xor_sync(0xffffffffu, s, 1);
}

// Loads a product warp's local rows into registers; local row lr maps to a global row through
// row_of(lr) (negative: absent, zero codes).
template <typename RowOf>
__device__ __forceinline__ void load_rows(uint32_t (&w)[kRowsPW][4], const uint8_t *base, int ld, int first,
                                          RowOf row_of) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int r = 0; r < kRowsPW; ++r) {
        const int64_t row = row_of(first + r);
        uint4 v = make_uint4(0, 0, 0, 0);
        if (row >= 0 && lane * 16 < ld) v = *reinterpret_cast<const uint4 *>(base + row * ld + lane * 16);
        w[r][0] = v.x, w[r][1] = v.y, w[r][2] = v.z, w[r][3] = v.w;
    }
}

__global__ void __launch_bounds__(kSThreads, 1) lstm_small_kernel(const __grid_constant__ SmallArgs a) {
    extern __shared__ __align__(128) uint8_t smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>(smem_raw);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
    const int CS = a.CS;
    const int cid = blockIdx.x / CS;
    const uint32_t rank = cluster_rank();
    const bool is_layer = cid < a.L;
    const int l = cid;
    const int B = a.B, T = a.T, H = a.H, R = a.R;
    const int kin = is_layer ? a.layer[l].kin : R;
    const int j0 = (int)rank * kCellsPerBlock;

    const uint32_t full0 = saddr(&S.bar_full[0]), empty0 = saddr(&S.bar_empty[0]);
    const uint32_t hbar0 = saddr(&S.bar_h[0]), axb0 = saddr(&S.bar_ax[0]), ahb0 = saddr(&S.bar_ah[0]);

    if (tid == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(full0 + 8 * i, 32);
            mbar_init(empty0 + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(hbar0 + 8 * i, 1);  // one local arrival (with the expected bytes) per phase
            mbar_init(axb0 + 8 * i, kPW);
            mbar_init(ahb0 + 8 * i, kPW);
            mbar_init(saddr(&S.bar_ep[i]), kEW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (is_layer) {  // frames 0 and 1: every block of the cluster sends B x (32 values + range)
            mbar_arrive_expect(hbar0, (uint32_t)(CS * kEW * B * kHBytes));
            mbar_arrive_expect(hbar0 + 8, (uint32_t)(CS * kEW * B * kHBytes));
        }
    }
    if (is_layer) {
        // h_{-1} of the whole layer into hbuf[1]; its range into every source slot of hmm[1]
        for (int i = tid; i < B * kMaxK; i += kSThreads) {
            const int b = i / kMaxK, k = i % kMaxK;
            S.hbuf[1][b][k] = k < R ? a.h0[((int64_t)l * B + b) * R + k] : 0.0f;
        }
        __syncthreads();
        if (warp < B) {
            float mn = FLT_MAX, mx = -FLT_MAX;
            for (int k = lane; k < R; k += 32) {
                mn = fminf(mn, S.hbuf[1][warp][k]);
                mx = fmaxf(mx, S.hbuf[1][warp][k]);
            }
            mn = warp_min(mn);
            mx = warp_max(mx);
            for (int i = lane; i < kHParts; i += 32) S.hmm[1][warp][i] = make_float2(mn, mx);
        }
        // Wx rows of this block, local row 4c + g <- global row g H + j0 + c
        const SmallLayer &ly = a.layer[l];
        for (int i = tid; i < kRows * (kMaxK / 16); i += kSThreads) {
            const int lr = i / (kMaxK / 16), ch = i % (kMaxK / 16);
            const int j = j0 + lr / 4, g = lr % 4;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (j < H && ch * 16 < ly.ldx)
                v = *reinterpret_cast<const uint4 *>(ly.wx + ((int64_t)g * H + j) * ly.ldx + ch * 16);
            *reinterpret_cast<uint4 *>(&S.wx[lr][ch * 16]) = v;
        }
    }
    __syncthreads();
    cluster_sync();

    if (warp == kLoaderWarp) {
        // ---------------- loader ----------------
        const unsigned long long *src = nullptr;
        int64_t src_ld = R;
        const bool sys = is_layer && l == 0;  // streamed input rows, written by the host
        if (!(is_layer && l == 0))
            src = a.hx + (int64_t)(is_layer ? l - 1 : a.L - 1) * B * T * R;
        else if (a.xs)
            src = a.xs, src_ld = a.I;
        for (int t = 0; t < T; ++t) {
            const int slot = t % kRing;
            if (t >= kRing) wait_cta(a, empty0 + 8 * slot, ((t / kRing) - 1) & 1);
            for (int b = 0; b < B; ++b) {
                float *dst = S.ring[slot][b];
                float mn = FLT_MAX, mx = -FLT_MAX;
                bool bad = false;
                if (src == nullptr) {
                    const float *xr = a.x + ((int64_t)b * T + t) * a.I;
                    for (int k = lane; k < kin; k += 32) {
                        const float v = xr[k];
                        dst[k] = v;
                        bad |= !isfinite(v);
                        mn = fminf(mn, v);
                        mx = fmaxf(mx, v);
                    }
                } else {
                    const unsigned long long *hr = src + ((int64_t)b * T + t) * src_ld;
                    auto ld = [&](const unsigned long long *p) { return sys ? ld_tag_sys(p) : ld_tag(p); };
                    unsigned long long v[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int k = lane + 32 * i;
                        v[i] = k < kin ? ld(hr + k) : ((unsigned long long)a.epoch << 32);
                    }
                    Deadline d{&a, now_ns(), 0};
                    while (true) {
                        bool ready = true;
#pragma unroll
                        for (int i = 0; i < 16; ++i) ready &= (unsigned)(v[i] >> 32) == a.epoch;
                        if (__all_sync(0xffffffffu, ready)) break;
                        if (__any_sync(0xffffffffu, d.expired())) break;
                        if (sys) __nanosleep(64);  // host-mapped input: fewer polls across the host link
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int k = lane + 32 * i;
                            if (k < kin && (unsigned)(v[i] >> 32) != a.epoch) v[i] = ld(hr + k);
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int k = lane + 32 * i;
                        if (k < kin) {
                            const float f = __uint_as_float((unsigned)(v[i] & 0xffffffffu));
                            dst[k] = f;
                            bad |= !isfinite(f);
                            mn = fminf(mn, f);
                            mx = fmaxf(mx, f);
                        }
                    }
                }
                mn = warp_min(mn);
                mx = warp_max(mx);
                bad = __any_sync(0xffffffffu, bad);
                if (bad) {
                    if (lane == 0) record_status(a.status, QNN_ERR_NONFINITE);
                    mn = 0.0f;
                    mx = 0.0f;
                }
                if (lane == 0) S.ring_p[slot][b] = params_from_range(mn, mx);  // the row's unit (eq. 2)
            }
            mbar_arrive(full0 + 8 * slot);
        }
    } else if (warp < kPW) {
        // ---------------- product warps ----------------
        const int lr0 = warp * kRowsPW;  // local rows lr0 .. lr0 + 7
        const int my_row = lr0 + ((lane >> kRowShift) & (kRowsPW - 1));  // row this lane ends with
        const bool row_writer = (lane & ((1 << kRowShift) - 1)) == 0;
        uint32_t wr[kRowsPW][4];
        if (is_layer) {
            const SmallLayer &ly = a.layer[l];
            load_rows(wr, ly.wh, ly.ldh, lr0, [&](int lr) -> int64_t {
                const int j = j0 + lr / 4;
                return j < H ? (int64_t)(lr % 4) * H + j : -1;
            });
        } else {
            const int nb = ((cid - a.L) * CS + (int)rank) * kRows;
            load_rows(wr, a.wo, a.ldo, lr0, [&](int lr) -> int64_t { return nb + lr < a.C ? nb + lr : -1; });
        }
        // output-layer epilogue constants of my_row
        int o_cs = 0, o_n = -1;
        float o_b = 0.0f;
        if (!is_layer) {
            const int n = ((cid - a.L) * CS + (int)rank) * kRows + my_row;
            if (n < a.C) {
                o_n = n;
                o_cs = a.wo_sum[n];
                o_b = a.bo[n];
            }
        }
        // Streaming: the softmax of frame t over the rows of every output block. Each block reduces
        // its rows to (m_b, s_b) = (max l, sum E(l - m_b)), publishes them as tagged words, gathers
        // every block's pair, and merges them the same way in every block: M = max m_b,
        // sum = sum_b s_b E(m_b - M); a row's posterior is E(l - M) / sum. The block then flags the
        // frame for the host.
        auto softmax_out = [&](int t, const float (&lg)[kMaxB]) {
            const bool mine = row_writer && o_n >= 0;
            const int ob = (cid - a.L) * CS + (int)rank;
            const unsigned long long tag = (unsigned long long)a.epoch << 32;
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const float m = warp_max(mine ? lg[b] : -FLT_MAX);
                if (lane == 0) S.red_m[warp][b] = m;
            }
            named_bar(1, kPT);
            float bm[kMaxB];
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                bm[b] = -FLT_MAX;
                if (b >= B) break;
                for (int w = 0; w < kPW; ++w) bm[b] = fmaxf(bm[b], S.red_m[w][b]);
                const float e = warp_sum_f(mine ? pexp(__fsub_rn(lg[b], bm[b])) : 0.0f);
                if (lane == 0) S.red_s[warp][b] = e;
            }
            named_bar(1, kPT);
            if (warp == 0) {
#pragma unroll
                for (int b = 0; b < kMaxB; ++b) {
                    if (b >= B) break;
                    unsigned long long *row = a.smx + ((int64_t)b * T + t) * a.nout * 2;
                    if (lane == 0) {
                        float sum = 0.0f;
                        for (int w = 0; w < kPW; ++w) sum = __fadd_rn(sum, S.red_s[w][b]);
                        st_tag(row + 2 * ob, tag | __float_as_uint(bm[b]));
                        st_tag(row + 2 * ob + 1, tag | __float_as_uint(sum));
                    }
                    // lane i gathers the pairs of blocks i, i + 32, ...: first wait for them and take
                    // the maximum, then read them again (now present) for the sum
                    const int rounds = (a.nout + 31) / 32;
                    float M = -FLT_MAX;
#pragma unroll 1
                    for (int q = 0; q < rounds; ++q) {
                        const int i = lane + 32 * q;
                        unsigned long long mv = tag, sv = tag;  // absent blocks: never waited for
                        if (i < a.nout) mv = ld_tag(row + 2 * i), sv = ld_tag(row + 2 * i + 1);
                        Deadline d{&a, now_ns(), 0};
                        while (true) {
                            const bool ready = (unsigned)(mv >> 32) == a.epoch && (unsigned)(sv >> 32) == a.epoch;
                            if (__all_sync(0xffffffffu, ready)) break;
                            if (__any_sync(0xffffffffu, d.expired())) break;
                            if (i < a.nout && (unsigned)(mv >> 32) != a.epoch) mv = ld_tag(row + 2 * i);
                            if (i < a.nout && (unsigned)(sv >> 32) != a.epoch) sv = ld_tag(row + 2 * i + 1);
                        }
                        if (i < a.nout) M = fmaxf(M, __uint_as_float((unsigned)mv));
                    }
                    M = warp_max(M);
                    float part = 0.0f;
#pragma unroll 1
                    for (int q = 0; q < rounds; ++q) {
                        const int i = lane + 32 * q;
                        if (i < a.nout) {
                            const float mi = __uint_as_float((unsigned)ld_tag(row + 2 * i));
                            const float si = __uint_as_float((unsigned)ld_tag(row + 2 * i + 1));
                            part = __fadd_rn(part, __fmul_rn(si, pexp(__fsub_rn(mi, M))));
                        }
                    }
                    part = warp_sum_f(part);  // xor butterfly: the same sum in every lane and block
                    if (lane == 0) S.sm_fin[b] = make_float2(M, part);
                }
            }
            named_bar(1, kPT);
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                if (mine) {
                    const float2 f = S.sm_fin[b];
                    a.probs[((int64_t)b * T + t) * a.C + o_n] = __fdiv_rn(pexp(__fsub_rn(lg[b], f.x)), f.y);
                }
            }
            if (mine) __threadfence_system();
            named_bar(1, kPT);
            // a frame computed after some wait gave up is not flagged (its values may be stale)
            if (tid == 0 && !aborted(a)) st_flag_sys(a.done + (int64_t)t * a.nout + ob, a.epoch);
        };
        // X phase of frame t: ring -> codes -> products (layer: Wx sums to the epilogue; output
        // layer: logits).
        auto x_phase = [&](int t) {
            const int slot = t % kRing, par = t & 1;
            wait_cta(a, full0 + 8 * slot, (t / kRing) & 1);
            for (int b = 0; b < B; ++b) {
                const qnn_qparams p = S.ring_p[slot][b];
                code_row(S.ring[slot][b], kin, p, S.codes_x[b], tid);
                if (tid == 0) S.meta_x[par][b] = RowMeta{p.z, p.Q, 0, 0};
            }
            named_bar(1, kPT);
            if (tid == 0) mbar_arrive(empty0 + 8 * slot);
            if (is_layer) {
                for (int b = 0; b < B; ++b) {
                    int rs = 0;
                    const int s =
                        dot8([&](int r) { return *reinterpret_cast<const uint4 *>(&S.wx[lr0 + r][lane * 16]); },
                             S.codes_x[b], warp == 0, rs);
                    if (row_writer) S.acc_x[par][b][my_row] = s;
                    if (tid == 0) S.meta_x[par][b].rs = rs;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(axb0 + 8 * par);
            } else {
                float lg[kMaxB];
#pragma unroll
                for (int b = 0; b < kMaxB; ++b) {
                    lg[b] = 0.0f;
                    if (b >= B) break;
                    int rs = 0;
                    const int s = dot8([&](int r) { return make_uint4(wr[r][0], wr[r][1], wr[r][2], wr[r][3]); },
                                       S.codes_x[b], true, rs);
                    if (row_writer && o_n >= 0) {
                        const RowMeta mt = S.meta_x[par][b];
                        const qnn_qparams po = a.wo_p[o_n / a.opu];
                        const long long Sv = offset_product(s, mt.za, po.z, rs, o_cs, R);
                        lg[b] = __fadd_rn(recover_product(Sv, mt.Qa, po.Q), o_b);
                        if (a.logits) a.logits[((int64_t)b * T + t) * a.C + o_n] = lg[b];
                    }
                }
                if (a.probs) softmax_out(t, lg);
            }
        };
        if (!is_layer) {
            for (int t = 0; t < T; ++t) {
                x_phase(t);
                named_bar(1, kPT);  // codes_x is rewritten next frame
            }
        } else {
            if (T > 0 && !a.h_first) x_phase(0);
            for (int t = 0; t < T; ++t) {
                const int par = t & 1, pb = (t - 1) & 1;
                if (t > 0) {
                    wait_cluster(a, hbar0 + 8 * pb, ((t - 1) >> 1) & 1);
                    // re-arm this buffer's barrier for frame t + 1 (its senders need our frame t first)
                    if (tid == 0 && t + 1 < T)
                        mbar_arrive_expect(hbar0 + 8 * pb, (uint32_t)(CS * kEW * B * kHBytes));
                }
                // H phase: quantize h_{t-1} cooperatively, product with Wh
                for (int b = 0; b < B; ++b) {
                    // range of the row: lane i folds partials i and i + 32, then the warp reduces
                    float mn = FLT_MAX, mx = -FLT_MAX;
#pragma unroll
                    for (int q = 0; q < kHParts / 32; ++q) {
                        const int i = lane + 32 * q;
                        if (i < CS * kEW) {
                            const float2 mm = S.hmm[pb][b][i];
                            mn = fminf(mn, mm.x);
                            mx = fmaxf(mx, mm.y);
                        }
                    }
                    mn = warp_min(mn);
                    mx = warp_max(mx);
                    const qnn_qparams p = params_from_range(mn, mx);
                    code_row(S.hbuf[pb][b], R, p, S.codes_h[b], tid);
                    if (tid == 0) S.meta_h[par][b] = RowMeta{p.z, p.Q, 0, 0};
                }
                named_bar(1, kPT);
                for (int b = 0; b < B; ++b) {
                    int rs = 0;
                    const int s =
                        dot8([&](int r) { return make_uint4(wr[r][0], wr[r][1], wr[r][2], wr[r][3]); },
                             S.codes_h[b], warp == 0, rs);
                    if (row_writer) S.acc_h[par][b][my_row] = s;
                    if (tid == 0) S.meta_h[par][b].rs = rs;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(ahb0 + 8 * par);
                // X phase of the next frame overlaps the cluster exchange of this one
                if (a.h_first) {
                    x_phase(t);  // h_{t-1} was known before x_t arrived: only Wx x_t is left after it
                } else {
                    if (kXAfterEpilogue) wait_cta(a, saddr(&S.bar_ep[par]), (t >> 1) & 1);
                    if (t + 1 < T) x_phase(t + 1);
                }
            }
        }
    } else if (is_layer) {
        // ---------------- epilogue warps ----------------
        const SmallLayer &ly = a.layer[l];
        const int et = tid - kPT;            // 0..127: local row 4c + g
        const int cl = et >> 2, g = et & 3;  // cell within the block, gate
        const int j = j0 + cl;
        const bool jv = j < H;
        const int64_t n = (int64_t)g * H + (jv ? j : 0);
        const int csx = jv ? ly.wx_sum[n] : 0, csh = jv ? ly.wh_sum[n] : 0;
        const float bias = jv ? ly.bias[n] : 0.0f;
        const int unit = g * a.ups + (jv ? j : 0) / a.cpu;  // this (cell, gate) row's weight unit
        const qnn_qparams px = ly.wx_p[unit], ph = ly.wh_p[unit];
        const int ew = warp - kPW;
        const bool tag_out = (l < a.L - 1) || (a.C > 0);
        float c[kMaxB], hl[kMaxB];
#pragma unroll
        for (int b = 0; b < kMaxB; ++b) {
            c[b] = (b < B && jv) ? a.c0[((int64_t)l * B + b) * H + j] : 0.0f;
            hl[b] = 0.0f;
        }
        const uint32_t hbuf_l = saddr(&S.hbuf[0][0][0]), hmm_l = saddr(&S.hmm[0][0][0]);
        for (int t = 0; t < T; ++t) {
            const int par = t & 1;
            wait_cta(a, axb0 + 8 * par, (t >> 1) & 1);
            float yx[kMaxB];
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const RowMeta mt = S.meta_x[par][b];
                const long long Sv = offset_product(S.acc_x[par][b][et], mt.za, px.z, mt.rs, csx, ly.kin);
                yx[b] = __fadd_rn(recover_product(Sv, mt.Qa, px.Q), bias);
            }
            wait_cta(a, ahb0 + 8 * par, (t >> 1) & 1);
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                const RowMeta mt = S.meta_h[par][b];
                const long long Sv = offset_product(S.acc_h[par][b][et], mt.za, ph.z, mt.rs, csh, R);
                const float pre = __fadd_rn(yx[b], recover_product(Sv, mt.Qa, ph.Q));
                // each lane applies its own gate's nonlinearity, then the quad gathers the four
                const float act = gate_activation(pre, g == 2);
                const int q0 = lane & ~3;
                const float ig = __shfl_sync(0xffffffffu, act, q0 + 0);
                const float fg = __shfl_sync(0xffffffffu, act, q0 + 1);
                const float gg = __shfl_sync(0xffffffffu, act, q0 + 2);
                const float og = __shfl_sync(0xffffffffu, act, q0 + 3);
                const float m = lstm_cell_update(ig, fg, gg, og, c[b]);
                const float h = jv ? m : 0.0f;
                hl[b] = h;
                // the warp's 8 values (quad q holds cell 8 ew + q) in every lane, and their range
                float v8[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) v8[q] = __shfl_sync(0xffffffffu, h, 4 * q);
                float mn = FLT_MAX, mx = -FLT_MAX;
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    if (j0 + 8 * ew + q < H) {
                        mn = fminf(mn, v8[q]);
                        mx = fmaxf(mx, v8[q]);
                    }
                // ... sent to every block of the cluster (lane d -> block d); the stores complete on
                // the peer's barrier. The last frame's values are not sent: no block waits for them
                // (nothing is in flight at exit).
                if (lane < CS && t + 1 < T) {
                    const uint32_t rbar = map_rank(hbar0 + 8 * par, lane);
                    const uint32_t dst =
                        map_rank(hbuf_l + 4u * (uint32_t)((par * kMaxB + b) * kMaxK + j0 + 8 * ew), lane);
                    st_async_v4(dst, make_float4(v8[0], v8[1], v8[2], v8[3]), rbar);
                    st_async_v4(dst + 16u, make_float4(v8[4], v8[5], v8[6], v8[7]), rbar);
                    st_async_v2(map_rank(hmm_l + 8u * (uint32_t)((par * kMaxB + b) * kHParts + rank * kEW + ew), lane),
                                mn, mx, rbar);
                }
                if (g == 0 && jv) {
                    const int64_t o = (((int64_t)l * B + b) * T + t) * R + j;
                    if (tag_out) st_tag(a.hx + o, ((unsigned long long)a.epoch << 32) | __float_as_uint(h));
                    if (a.h_all) a.h_all[o] = h;
                    if (a.ytop && l == a.L - 1) a.ytop[((int64_t)b * T + t) * R + j] = h;
                }
            }
            if (a.done && a.C == 0 && l == a.L - 1) {  // streaming without an output layer: h_t is the output
                if (g == 0 && jv) __threadfence_system();
                named_bar(2, kET);
                if (et == 0 && !aborted(a)) st_flag_sys(a.done + (int64_t)t * CS + rank, a.epoch);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(saddr(&S.bar_ep[par]));  // gate arithmetic of frame t done
        }
        if (g == 0 && jv) {
#pragma unroll
            for (int b = 0; b < kMaxB; ++b) {
                if (b >= B) break;
                if (a.h_fin) a.h_fin[((int64_t)l * B + b) * R + j] = hl[b];
                if (a.c_fin) a.c_fin[((int64_t)l * B + b) * H + j] = c[b];
            }
        }
    }
    __syncwarp();
    // After an aborted run some waits returned early; give peer stores still in flight time to
    // land (they take microseconds) before any block of the cluster can leave.
    if (*(volatile int *)a.abort_flag)
        for (int i = 0; i < 100; ++i) __nanosleep(100000);
    // no block leaves while a cluster peer may still write into its shared memory
    cluster_sync();
}

// ---- latency floor probe --------------------------------------------------------------------------
// The per-frame synchronisation skeleton of one layer cluster of lstm_small_kernel with the
// arithmetic taken out: per round, the 16 product warps of every block wait for the cluster
// exchange (transaction-count mbarrier), re-arm it and hand over to the 4 epilogue warps (local
// mbarrier); the epilogue warps send their 40 bytes to every block of the cluster (st.async),
// which completes the next round's exchange. Its time per round is the floor under the time per
// frame of a layer, whatever the products and the gate arithmetic cost.
struct FloorArgs {
    int rounds;
    int *status;
    int *abort_flag;
    unsigned long long wait_ns;
};

__global__ void __launch_bounds__(kSThreads, 1) exchange_floor_kernel(const __grid_constant__ FloorArgs f) {
    __shared__ __align__(16) float hbuf[2][kMaxK];
    __shared__ __align__(16) float2 hmm[2][kHParts];
    __shared__ __align__(8) unsigned long long bar_h[2], bar_a[2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
    uint32_t CS;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(CS));
    const uint32_t rank = cluster_rank();
    const uint32_t hb0 = saddr(&bar_h[0]), ab0 = saddr(&bar_a[0]);
    const uint32_t bytes = CS * kEW * kHBytes;
    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(hb0 + 8 * i, 1);
            mbar_init(ab0 + 8 * i, kPW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        mbar_arrive_expect(hb0, bytes);
        if (f.rounds > 1) mbar_arrive_expect(hb0 + 8, bytes);
    }
    __syncthreads();
    cluster_sync();
    if (warp < kPW) {
        __syncwarp();
        if (lane == 0) mbar_arrive(ab0);  // round 0 may start
        for (int t = 0; t < f.rounds; ++t) {
            const int par = t & 1;
            wait_cluster(f, hb0 + 8 * par, (t >> 1) & 1);
            if (tid == 0 && t + 2 < f.rounds) mbar_arrive_expect(hb0 + 8 * par, bytes);
            __syncwarp();
            if (lane == 0 && t + 1 < f.rounds) mbar_arrive(ab0 + 8 * (par ^ 1));
        }
    } else if (warp < kPW + kEW) {
        const int ew = warp - kPW;
        const uint32_t hbuf_l = saddr(&hbuf[0][0]), hmm_l = saddr(&hmm[0][0]);
        for (int t = 0; t < f.rounds; ++t) {
            const int par = t & 1;
            wait_cta(f, ab0 + 8 * par, (t >> 1) & 1);
            if (lane < (int)CS) {
                const float v = (float)t;
                const uint32_t rbar = map_rank(hb0 + 8 * par, lane);
                const uint32_t dst = map_rank(hbuf_l + 4u * (uint32_t)(par * kMaxK + rank * kCellsPerBlock + 8 * ew), lane);
                st_async_v4(dst, make_float4(v, v, v, v), rbar);
                st_async_v4(dst + 16u, make_float4(v, v, v, v), rbar);
                st_async_v2(map_rank(hmm_l + 8u * (uint32_t)(par * kHParts + rank * kEW + ew), lane), v, v, rbar);
            }
        }
    }
    __syncwarp();
    if (*(volatile int *)f.abort_flag)
        for (int i = 0; i < 100; ++i) __nanosleep(100000);
    cluster_sync();
}

int g_small_cfg_dev = -1;

// Launch geometry of the kernel for model m at batch B; false when the model or batch does not
// fit this path (then nothing is set).
struct SmallGeom {
    int CS = 0, clusters = 0, nout = 0;
};
bool small_geometry(const qnn_lstm_model *m, int64_t B, SmallGeom *g) {
    const int64_t L = m->L, I = m->I, H = m->H, C = m->C, R = m->R;
    if (m->P != 0 || B < 1 || B > kMaxB || L > kMaxLayers || I > kMaxK || R > kMaxK || H > kCellsPerBlock * kMaxCS)
        return false;
    if (C > 0 && m->d.output_mode != QNN_OUT_QUANT) return false;
    g->CS = (int)((H + kCellsPerBlock - 1) / kCellsPerBlock);
    const int out_blocks = C > 0 ? (int)((C + kRows - 1) / kRows) : 0;
    const int out_clusters = (out_blocks + g->CS - 1) / g->CS;
    g->clusters = (int)L + out_clusters;
    g->nout = out_clusters * g->CS;
    return true;
}

// Sets the kernel's attributes (once per device) and fills the cluster launch configuration;
// *fits tells whether all clusters can be resident at once (the dataflow between them needs it).
qnn_status small_config(const SmallGeom &g, cudaStream_t st, cudaLaunchConfig_t *cfg, cudaLaunchAttribute *attr,
                        bool *fits) {
    const size_t smem = sizeof(Smem);
    int dev = 0;
    QNN_CUDA_TRY(cudaGetDevice(&dev));
    if (g_small_cfg_dev != dev) {
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstm_small_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        QNN_CUDA_TRY(cudaFuncSetAttribute(lstm_small_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
        g_small_cfg_dev = dev;
    }
    *cfg = cudaLaunchConfig_t{};
    cfg->gridDim = dim3((unsigned)(g.clusters * g.CS));
    cfg->blockDim = dim3(kSThreads);
    cfg->dynamicSmemBytes = smem;
    cfg->stream = st;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)g.CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg->attrs = attr;
    cfg->numAttrs = 1;
    int max_clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&max_clusters, lstm_small_kernel, cfg) != cudaSuccess) {
        cudaGetLastError();
        *fits = false;
        return QNN_OK;
    }
    *fits = max_clusters >= g.clusters;
    return QNN_OK;
}

// The model's weights, units and shapes into the kernel arguments.
void small_model_args(const qnn_lstm_model *m, const SmallGeom &g, int64_t B, int64_t T, SmallArgs *a) {
    for (int64_t l = 0; l < m->L; ++l) {
        const LayerDev &ly = m->layers[l];
        a->layer[l] = SmallLayer{ly.wx.codes, ly.wx.sums, ly.wx.params, ly.wh.codes, ly.wh.sums, ly.wh.params,
                                 ly.bias, (int)ly.wx.ld, (int)ly.wh.ld, (int)ly.kin};
    }
    if (m->C > 0) {
        a->wo = m->wo.codes, a->wo_sum = m->wo.sums, a->wo_p = m->wo.params, a->bo = m->bo, a->ldo = (int)m->wo.ld;
    }
    a->L = (int)m->L, a->I = (int)m->I, a->H = (int)m->H, a->R = (int)m->R, a->C = (int)m->C;
    a->B = (int)B, a->T = (int)T, a->CS = g.CS, a->nout = g.nout;
    a->ups = (int)m->S, a->cpu = (int)(m->H / m->S), a->opu = m->C > 0 ? (int)(m->C / m->S) : 1;
    a->wait_ns = kWaitNs;
}

}  // namespace

qnn_status small_stream_plan(const qnn_lstm_model *m, int64_t B, int *writer_blocks, int *nout) {
    SmallGeom g;
    if (!small_geometry(m, B, &g)) return QNN_ERR_INVALID_ARG;
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    bool fits = false;
    QNN_TRY(small_config(g, nullptr, &cfg, attr, &fits));
    if (!fits) return QNN_ERR_NO_COOP;
    *nout = g.nout;
    *writer_blocks = m->C > 0 ? g.nout : g.CS;
    return QNN_OK;
}

qnn_status small_stream_launch(const qnn_lstm_model *m, const SmallStreamArgs &s, cudaStream_t st) {
    SmallGeom g;
    if (!small_geometry(m, s.B, &g)) return QNN_ERR_INVALID_ARG;
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    bool fits = false;
    QNN_TRY(small_config(g, st, &cfg, attr, &fits));
    if (!fits) return QNN_ERR_NO_COOP;
    SmallArgs a{};
    small_model_args(m, g, s.B, s.T, &a);
    a.xs = s.xs;
    a.hx = s.hx;
    a.smx = s.smx;
    a.done = s.done;
    if (m->C > 0)
        a.probs = s.out;
    else
        a.ytop = s.out;
    a.h0 = s.h0, a.c0 = s.c0, a.h_fin = s.h_fin, a.c_fin = s.c_fin;
    a.status = s.status;
    a.abort_flag = s.abort_flag;
    a.epoch = s.epoch;
    a.wait_ns = s.wait_ns;
    a.h_first = 1;
    ProfScope prof("lstm_small_stream", st);
    QNN_CUDA_TRY(cudaLaunchKernelEx(&cfg, lstm_small_kernel, a));
    return QNN_OK;
}

PathChoice path_choice() {
    const char *v = std::getenv("QNN_LSTM_PATH");
    if (!v || !*v || std::strcmp(v, "auto") == 0) return PathChoice::kAuto;
    if (std::strcmp(v, "layerwise") == 0) return PathChoice::kLayerwise;
    if (std::strcmp(v, "small") == 0) return PathChoice::kSmall;
    if (std::strcmp(v, "tc") == 0) return PathChoice::kTc;
    return PathChoice::kAuto;
}

qnn_status small_path_forward(qnn_lstm_model *m, const float *x, int64_t B, int64_t T, float *y, float *logits,
                              float *h_state, float *c_state, float *h_all, cudaStream_t st, bool *used) {
    *used = false;
    const int64_t L = m->L, I = m->I, H = m->H, C = m->C, R = m->R;
    SmallGeom geo;
    if (!small_geometry(m, B, &geo) || T > (int64_t)INT32_MAX / 4) return QNN_OK;
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    bool fits = false;
    QNN_TRY(small_config(geo, st, &cfg, attr, &fits));
    if (!fits) return QNN_OK;  // cannot be co-resident: layer-by-layer path

    // workspace: staging, tagged layer outputs, logits, state
    const bool x_dev = is_device_ptr(x), y_dev = is_device_ptr(y);
    const bool hs_dev = h_state && is_device_ptr(h_state), cs_dev = c_state && is_device_ptr(c_state);
    const bool ha_dev = h_all && is_device_ptr(h_all);
    // posteriors into pinned host memory: the softmax writes them there directly (no staging copy)
    float *const y_map = (!y_dev && C > 0) ? static_cast<float *>(host_mapped_ptr(y)) : nullptr;
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
    const size_t o_y = (y_dev || y_map) ? 0 : acct(sizeof(float) * rows * ycols);
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
    small_model_args(m, geo, B, T, &a);
    const float *xd = x;
    if (!x_dev) {
        QNN_CUDA_TRY(cudaMemcpyAsync(ws + o_x, x, sizeof(float) * rows * I, cudaMemcpyHostToDevice, st));
        xd = reinterpret_cast<const float *>(ws + o_x);
    }
    float *yd = y_dev ? y : y_map ? y_map : reinterpret_cast<float *>(ws + o_y);
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
    {
        ProfScope prof("lstm_small", st);
        QNN_CUDA_TRY(cudaLaunchKernelEx(&cfg, lstm_small_kernel, a));
    }
    if (logits) QNN_CUDA_TRY(cudaMemcpyAsync(logits, a.logits, sizeof(float) * rows * C, cudaMemcpyDefault, st));
    if (C > 0) QNN_TRY(launch_softmax_rows(a.logits, rows, C, yd, st));
    if (!y_dev && !y_map)
        QNN_CUDA_TRY(cudaMemcpyAsync(y, yd, sizeof(float) * rows * ycols, cudaMemcpyDeviceToHost, st));
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

// Time per round of the batch-of-few kernel's per-frame synchronisation skeleton on one cluster of
// cluster_size blocks (exchange_floor_kernel). Synchronous; best of three timed launches.
extern "C" qnn_status qnn_measure_exchange_floor(int32_t cluster_size, int32_t rounds, double *us_per_round) {
    using namespace qnn;
    if (!us_per_round || cluster_size < 1 || cluster_size > kMaxCS || rounds < 1 || rounds > 1000000)
        return QNN_ERR_INVALID_ARG;
    QNN_CUDA_TRY(cudaFuncSetAttribute(exchange_floor_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cluster_size);
    cfg.blockDim = dim3(kSThreads);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cluster_size;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int max_clusters = 0;
    QNN_CUDA_TRY(cudaOccupancyMaxActiveClusters(&max_clusters, exchange_floor_kernel, &cfg));
    if (max_clusters < 1) return QNN_ERR_NO_COOP;
    int *words = nullptr;  // status, abort flag
    QNN_CUDA_TRY(cudaMalloc(&words, 2 * sizeof(int)));
    QNN_CUDA_TRY(cudaMemset(words, 0, 2 * sizeof(int)));
    FloorArgs f{rounds, words, words + 1, kWaitNs};
    cudaEvent_t e0, e1;
    QNN_CUDA_TRY(cudaEventCreate(&e0));
    QNN_CUDA_TRY(cudaEventCreate(&e1));
    double best = 1e30;
    qnn_status result = QNN_OK;
    for (int rep = 0; rep < 4 && result == QNN_OK; ++rep) {
        if (cudaEventRecord(e0) != cudaSuccess || cudaLaunchKernelEx(&cfg, exchange_floor_kernel, f) != cudaSuccess ||
            cudaEventRecord(e1) != cudaSuccess || cudaEventSynchronize(e1) != cudaSuccess) {
            result = QNN_ERR_CUDA;
            break;
        }
        float ms = 0.0f;
        cudaEventElapsedTime(&ms, e0, e1);
        if (rep > 0) best = std::min(best, 1e3 * ms / rounds);
    }
    int st = 0;
    if (result == QNN_OK && cudaMemcpy(&st, words, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        result = QNN_ERR_CUDA;
    if (result == QNN_OK && st != 0) result = (qnn_status)st;
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    cudaFree(words);
    if (result == QNN_OK) *us_per_round = best;
    return result;
}
