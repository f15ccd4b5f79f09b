// qnn_device.cuh — device arithmetic shared by the libqnn kernels: the quantizer's parameter
// rule (Sec. 3, eq. 2), code and recovery (eq. 2, eq. 3), the recovered offset-applied product
// (eq. 1), the pinned fp32 exponential and the LSTM gate functions.
//
// Every fp32 operation that can decide a code is written with an explicit round-to-nearest
// intrinsic (__fmul_rn, __fadd_rn, __fdiv_rn, __fmaf_rn) so that the compiler can neither fuse
// nor reorder it: the same inputs give the same bits on every run and every launch shape.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/qnn.h"

namespace qnn {

constexpr float kScale = 255.0f;          // S for 8 bits (Sec. 3)
constexpr float kDegenerateLim = 4194304.0f;  // 2^22: |Q v| beyond this leaves no fractional bit

// Device status word (library-owned, one per device): keeps the first error a kernel finds
// (QNN_ERR_NONFINITE, QNN_ERR_TIMEOUT) until qnn_device_status() reads and clears it.
__device__ __forceinline__ void record_status(int *status, int st) { atomicCAS(status, 0, st); }

// Sec. 3: Q = S / (vmax - vmin); eq. (2): z = round(Q vmin). Q is raised one ulp at a time until
// round(Q vmax) - z reaches S, so the range maximum gets the top code. Degenerate units (no
// range, or a range so narrow that Q v has no fractional bits left) use Q = S / max|v|.
__device__ __forceinline__ qnn_qparams params_from_range(float vmin, float vmax) {
    qnn_qparams p;
    p.vmin = vmin;
    p.vmax = vmax;
    float R = __fsub_rn(vmax, vmin);
    float Q = (R > 0.0f) ? __fdiv_rn(kScale, R) : 0.0f;
    bool degenerate = !(R > 0.0f) || !isfinite(Q) || !(fabsf(__fmul_rn(Q, vmin)) < kDegenerateLim) ||
                      !(fabsf(__fmul_rn(Q, vmax)) < kDegenerateLim);
    if (degenerate) {
        float amax = fmaxf(fabsf(vmin), fabsf(vmax));
        Q = (amax > 0.0f) ? __fdiv_rn(kScale, amax) : 1.0f;
        p.Q = Q;
        p.z = __float2int_rn(__fmul_rn(Q, vmin));
        return p;
    }
    int z = __float2int_rn(__fmul_rn(Q, vmin));
    for (int it = 0; it < 64; ++it) {
        int top = __float2int_rn(__fmul_rn(Q, vmax)) - z;
        if (top >= 255) break;
        Q = __int_as_float(__float_as_int(Q) + 1);
        z = __float2int_rn(__fmul_rn(Q, vmin));
    }
    p.Q = Q;
    p.z = z;
    return p;
}

// Eq. (2): code = clamp(round(Q v) - round(Q vmin), 0, S).
__device__ __forceinline__ uint32_t quant_code(float v, float Q, int z) {
    int c = __float2int_rn(__fmul_rn(Q, v)) - z;
    c = c < 0 ? 0 : c;
    c = c > 255 ? 255 : c;
    return (uint32_t)c;
}

// (float)S rounded to nearest, ties to even, without the 64-bit conversion instruction (which runs
// on this part's narrow fp64 pipe). |S| < 2^31 converts from 32 bits; wider values (rare: large
// offsets z) are rounded to a 24-bit significand by integer arithmetic out of line: the bits below
// the significand decide (above half: up; exactly half: to the even significand).
static __device__ __noinline__ float s64_to_f32_rn_wide(long long S) {
    const unsigned long long u = S < 0 ? 0ULL - (unsigned long long)S : (unsigned long long)S;
    const int top = 63 - __clzll((long long)u);  // position of the leading one, 31..63
    const int sh = top - 23;                     // bits below the significand, >= 8
    unsigned long long m = u >> sh;
    const unsigned long long rem = u & ((1ULL << sh) - 1), half = 1ULL << (sh - 1);
    m += (rem > half || (rem == half && (m & 1ULL))) ? 1ULL : 0ULL;
    int e = top + 127;
    if (m >> 24) {  // rounding carried into a new leading bit
        m >>= 1;
        ++e;
    }
    return __uint_as_float(((unsigned)e << 23) | ((unsigned)m & 0x7FFFFFu) | (S < 0 ? 0x80000000u : 0u));
}
__device__ __forceinline__ float s64_to_f32_rn(long long S) {
    const int lo = (int)S;
    if ((long long)lo == S) return __int2float_rn(lo);
    return s64_to_f32_rn_wide(S);
}

// An integer-valued float (an exact tensor-core sum) as int.
__device__ __forceinline__ int f32_integer_to_s32(float v) { return __float2int_rn(v); }

// x / d correctly rounded, from r = RN(1/d) (the correctly rounded reciprocal, computed once per
// divisor): q = RN(x r), the remainder x - q d exactly by a fused multiply-add, then RN(q + (x - q d) r)
// (the final step of Markstein's division). This equals the IEEE quotient while d and r stay well
// inside the normal range and x q does not overflow (the caller checks d against 2^-60 .. 2^60 and
// passes |x| < 2^63); a CPU test checks the identity over every 24-bit numerator significand
// against thousands of divisors.
__device__ __forceinline__ float div_by_recip(float x, float d, float r) {
    const float q = __fmul_rn(x, r);
    const float e = __fmaf_rn(-q, d, x);
    return __fmaf_rn(e, r, q);
}

// Eq. (1) recovery of the exact offset-applied product S: S / (Qa Qw), each op rounded once.
__device__ __forceinline__ float recover_product(long long S, float Qa, float Qw) {
    return __fdiv_rn(s64_to_f32_rn(S), __fmul_rn(Qa, Qw));
}

// S = acc + zw*rsA + za*csW + K*za*zw: eq. (1)'s sum of (a' + za)(w' + zw) expanded so that the
// inner loop multiplies raw codes only.
__device__ __forceinline__ long long offset_product(int acc, int za, int zw, int rsA, int csW, int K) {
    return (long long)acc + (long long)zw * rsA + (long long)za * csW + (long long)K * za * zw;
}

// Pinned fp32 exponential: Cody-Waite reduction x = n ln2 + r (n = round(x log2 e), ln 2 split
// into a 16-significant-bit head and its remainder), e^r by its degree-7 Taylor polynomial in
// Horner form with fused multiply-adds, times 2^n assembled from exponent bits. x is clamped to
// [-87, 88] so every result is a finite normal number. n is rounded half-to-even by adding
// 1.5 * 2^23 (|x log2 e| <= 127), which leaves n in the low significand bits.
__device__ __forceinline__ float pexp(float x) {
    x = x < -87.0f ? -87.0f : x;
    x = x > 88.0f ? 88.0f : x;
    const float t = __fadd_rn(__fmul_rn(x, 1.44269504088896341f), 12582912.0f);
    const int n = __float_as_int(t) - 0x4B400000;
    const float nf = __fsub_rn(t, 12582912.0f);
    float r = __fmaf_rn(-nf, 0.693145751953125f, x);
    r = __fmaf_rn(-nf, 1.428606820309417232e-06f, r);
    float p = 1.984126984126984127e-04f;
    p = __fmaf_rn(p, r, 1.388888888888888889e-03f);
    p = __fmaf_rn(p, r, 8.333333333333333333e-03f);
    p = __fmaf_rn(p, r, 4.166666666666666667e-02f);
    p = __fmaf_rn(p, r, 1.666666666666666667e-01f);
    p = __fmaf_rn(p, r, 0.5f);
    p = __fmaf_rn(p, r, 1.0f);
    p = __fmaf_rn(p, r, 1.0f);
    return __fmul_rn(p, __int_as_float((n + 127) << 23));
}

// sigma(x) = 1/(E(-x) + 1) and tanh(x) = 1 - 2/(E(2x) + 1), each quotient correctly rounded.
// The quotients are taken from the correctly rounded reciprocal r of d = E + 1 (d >= 1): 1/d is r
// itself, and 2/d is 2 r exactly whenever r is a normal number; where it is not (d > 2^126) the
// quotient is below 2^-125 and 1 - 2/d rounds to 1 from either.
__device__ __forceinline__ float psigmoid(float x) { return __frcp_rn(__fadd_rn(1.0f, pexp(-x))); }

__device__ __forceinline__ float ptanh(float x) {
    return __fsub_rn(1.0f, __fmul_rn(2.0f, __frcp_rn(__fadd_rn(pexp(__fmul_rn(2.0f, x)), 1.0f))));
}

// psigmoid(x) or ptanh(x) without a branch (lanes of one warp may need different ones): the same
// operations in the same order.
__device__ __forceinline__ float gate_activation(float x, bool is_tanh) {
    const float e = pexp(is_tanh ? __fmul_rn(2.0f, x) : -x);
    const float r = __frcp_rn(__fadd_rn(e, 1.0f));
    return is_tanh ? __fsub_rn(1.0f, __fmul_rn(2.0f, r)) : r;
}

// LSTM cell update from the gate activations (no peepholes): c' = f c + i g; returns m = o tanh(c').
__device__ __forceinline__ float lstm_cell_update(float ig, float fg, float gg, float og, float &c) {
    c = __fadd_rn(__fmul_rn(fg, c), __fmul_rn(ig, gg));
    return __fmul_rn(og, ptanh(c));
}

// LSTM cell from the gate pre-activations [i, f, g, o]: sigmoid, sigmoid, tanh, sigmoid, then the update.
__device__ __forceinline__ void lstm_cell(float pi, float pf, float pg, float po, float &c, float &m) {
    float ig = psigmoid(pi), fg = psigmoid(pf), gg = ptanh(pg), og = psigmoid(po);
    m = lstm_cell_update(ig, fg, gg, og, c);
}

// The same functions on two values at once with the paired fp32 instructions of sm_100 and later
// (mul/add/fma .rn.f32x2: per component the same IEEE round-to-nearest operation as __fmul_rn,
// __fadd_rn, __fmaf_rn), so each component equals the scalar function bit for bit while the
// exponential's polynomial takes half the instructions. A paired product whose rounded result
// feeds a paired sum was observed fused into one multiply-add (with the compiler's paired
// intrinsics, and on one lane even through explicit-rounding PTX), so those two steps stay scalar
// wherever the product is inexact; the paired ops are used for fused multiply-adds, sums, and
// products that are exact (powers of two) or feed no sum.
__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }
__device__ __forceinline__ float2 fmul2_rn(float2 a, float2 b) {
    float2 d;
    asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mul.rn.f32x2 rd, ra, rb;\n"
        " mov.b64 {%0, %1}, rd;\n}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 fadd2_rn(float2 a, float2 b) {
    float2 d;
    asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n add.rn.f32x2 rd, ra, rb;\n"
        " mov.b64 {%0, %1}, rd;\n}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 ffma2_rn(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n mov.b64 rc, {%6, %7};\n"
        " fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

__device__ __forceinline__ float2 pexp2(float2 x) {
    x.x = x.x < -87.0f ? -87.0f : x.x;
    x.y = x.y < -87.0f ? -87.0f : x.y;
    x.x = x.x > 88.0f ? 88.0f : x.x;
    x.y = x.y > 88.0f ? 88.0f : x.y;
    // the rounded product x log2(e) and the sum stay scalar: a paired product followed by a paired
    // sum was observed contracted into one multiply-add (one rounding fewer)
    const float2 t = make_float2(__fadd_rn(__fmul_rn(x.x, 1.44269504088896341f), 12582912.0f),
                                 __fadd_rn(__fmul_rn(x.y, 1.44269504088896341f), 12582912.0f));
    const int nx = __float_as_int(t.x) - 0x4B400000, ny = __float_as_int(t.y) - 0x4B400000;
    const float2 nf = fadd2_rn(t, f2(-12582912.0f));
    const float2 mnf = make_float2(-nf.x, -nf.y);
    float2 r = ffma2_rn(mnf, f2(0.693145751953125f), x);
    r = ffma2_rn(mnf, f2(1.428606820309417232e-06f), r);
    float2 p = f2(1.984126984126984127e-04f);
    p = ffma2_rn(p, r, f2(1.388888888888888889e-03f));
    p = ffma2_rn(p, r, f2(8.333333333333333333e-03f));
    p = ffma2_rn(p, r, f2(4.166666666666666667e-02f));
    p = ffma2_rn(p, r, f2(1.666666666666666667e-01f));
    p = ffma2_rn(p, r, f2(0.5f));
    p = ffma2_rn(p, r, f2(1.0f));
    p = ffma2_rn(p, r, f2(1.0f));
    return fmul2_rn(p, make_float2(__int_as_float((nx + 127) << 23), __int_as_float((ny + 127) << 23)));
}

__device__ __forceinline__ float2 psigmoid2(float2 x) {
    const float2 d = fadd2_rn(f2(1.0f), pexp2(make_float2(-x.x, -x.y)));
    return make_float2(__frcp_rn(d.x), __frcp_rn(d.y));
}

__device__ __forceinline__ float2 ptanh2(float2 x) {
    const float2 d = fadd2_rn(pexp2(fmul2_rn(f2(2.0f), x)), f2(1.0f));
    const float2 t = fmul2_rn(f2(2.0f), make_float2(__frcp_rn(d.x), __frcp_rn(d.y)));
    return fadd2_rn(f2(1.0f), make_float2(-t.x, -t.y));
}

// lstm_cell on two cells: pre-activations of gates i, f, g, o (one float2 each), cell state c in/out.
__device__ __forceinline__ float2 lstm_cell2(float2 pi, float2 pf, float2 pg, float2 po, float2 &c) {
    const float2 ig = psigmoid2(pi), fg = psigmoid2(pf), gg = ptanh2(pg), og = psigmoid2(po);
    c = make_float2(__fadd_rn(__fmul_rn(fg.x, c.x), __fmul_rn(ig.x, gg.x)),
                    __fadd_rn(__fmul_rn(fg.y, c.y), __fmul_rn(ig.y, gg.y)));  // scalar: see pexp2
    return fmul2_rn(og, ptanh2(c));
}

// div_by_recip on two numerators with one divisor.
__device__ __forceinline__ float2 div_by_recip2(float2 x, float d, float r) {
    const float2 q = fmul2_rn(x, f2(r));
    const float2 e = ffma2_rn(make_float2(-q.x, -q.y), f2(d), x);
    return ffma2_rn(e, f2(r), q);
}

// Device clock in nanoseconds (%globaltimer).
__device__ __forceinline__ unsigned long long global_timer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait for the phase with the given parity of a shared-memory mbarrier, for at most limit_ns: on
// time-out, record QNN_ERR_TIMEOUT and return false (the caller then skips ahead, so the kernel
// ends and the host reads the status instead of finding the GPU hung). After a first test, each
// further test lets the thread be suspended until the phase completes, for at most kSuspendNs
// (mbarrier.try_wait's suspend-time hint), so a warp that waits long issues a few instructions per
// microsecond instead of spinning against the warps that do the work.
constexpr unsigned kSuspendNs = 1000;
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, unsigned parity, int *status,
                                                  unsigned long long limit_ns) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    if (ok) return true;
    const unsigned long long t0 = global_timer_ns();
    while (true) {
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(bar), "r"(parity), "r"(kSuspendNs)
            : "memory");
        if (ok) return true;
        if (global_timer_ns() - t0 > limit_ns) {
            record_status(status, QNN_ERR_TIMEOUT);
            return false;
        }
    }
}

// Programmatic dependent launch: a kernel launched with the programmatic stream serialization
// attribute may start while the previous kernel of its stream is still running. The wait returns
// once that kernel has completed and its memory operations are visible (at once without such a
// launch); the trigger lets the next kernel of the stream start early.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Warp-wide reductions.
__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
// Float sum by an xor butterfly: every lane ends with the same value (each step adds a symmetric pair).
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

}  // namespace qnn
