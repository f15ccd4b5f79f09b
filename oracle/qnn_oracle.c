/*
 * qnn_oracle.c — plain, slow CPU oracle for 8-bit quantized LSTM inference
 * (Alvarez, Prabhavalkar, Bakhtin, "On the efficient representation and execution of
 * deep acoustic models", INTERSPEECH 2016).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may link or call this file: only the
 * test suite, the smoke check and the CPU-baseline leg of the benchmark use it. It shares no
 * code, header, table or constant generator with the CUDA path.
 *
 * Build: cc -O2 -std=c11 -ffp-contract=off -fno-fast-math -fPIC -shared (see oracle/__init__.py).
 * -ffp-contract=off matters: every fp32 operation below is one IEEE operation, rounded once,
 * in the order written (gcc on aarch64 would otherwise fuse a*b+c).
 *
 * Precision: the paper's numbers are 32-bit floats quantized to 8-bit integers with 32-bit
 * integer accumulation (abstract; Sec. 3.1 "Multiplication of quantized values"). Every float
 * that decides a code is therefore computed in fp32, in the order written here. Integer
 * products are exact (int32 raw accumulator, int64 offset-applied product).
 *
 * Readings where the paper is silent (each one is listed with its reason in the design notes):
 *   R1 nudge: Q is raised one ulp at a time until round(Q*vmax) - round(Q*vmin) >= 255, so
 *      that the range maximum reaches the top code (Sec. 3 "Quantizing": use the whole scale).
 *   R2 clamp: codes are clamped to [0, 255]; the clamp only fires when the fp32 top lands on 256.
 *   R3 degenerate unit: R == 0, or |Q*vmin| or |Q*vmax| >= 2^22, gives Q = 255/max|v| (Q = 1
 *      when every value is 0) and z = round(Q*vmin); every code is then 0 or near it.
 *   R4 LSTM cell: the standard LSTM without peepholes, gate order [i, f, g, o]; the
 *      pre-activation is (R(x-product) + b) + R(h-product); c = f*c + i*g; m = o*tanh(c);
 *      with a projection r = R(Q(m) Wp), no bias, no nonlinearity.
 *   R5 E: a pinned fp32 exponential (Cody-Waite reduction, degree-7 Taylor polynomial by fmaf
 *      Horner, exact power-of-two scale) used for sigmoid, tanh and softmax on both sides.
 *   R6 granularity: weights one unit per gate matrix (Sec. 3.1 last paragraph), or per block of
 *      its rows when the descriptor asks for sub-matrices; activations one unit per row (one frame
 *      of one sequence) inside the LSTM.
 *   R7 output layer: logits = R(Q(r) Wo) + bo then softmax ("quant-all", Sec. 5); the float
 *      variant ("quant") computes the logits in fp64 and rounds them once to fp32.
 *   R11 softmax normalisation: the paper does not fix its precision; the terms E(l - max) are
 *      fp32 (R5), their sum and each quotient fp64, rounded once. (A sequential fp32 sum of 8192
 *      nearly equal terms drifts by a few 1e-5 relative, beyond the 1e-5 bar on the posteriors.)
 *   R9 frame stacking (Sec. 4 frontend): network input t' is the n frames starting at frame
 *      stride*t' (the frame and n-1 frames of right context), concatenated; T' = ceil(T/stride)
 *      inputs; frames past the end of the sequence repeat its last frame.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    float vmin, vmax, Q;
    int32_t z;
} orc_qparams;

enum {
    ORC_OK = 0,
    ORC_ERR_INVALID_ARG = 1,
    ORC_ERR_NONFINITE = 2,
    ORC_ERR_K_TOO_LARGE = 3,
};

enum { ORC_PER_MATRIX = 0, ORC_PER_ROW = 1 };
enum { ORC_OUT_NONE = 0, ORC_OUT_QUANT = 1, ORC_OUT_FLOAT = 2 };

/* Largest K for which the raw int32 accumulator of 8-bit codes cannot overflow:
 * K * 255 * 255 <= 2^31 - 1  <=>  K <= 33025 (Sec. 3.1: 8-bit operands, 32-bit accumulators). */
#define ORC_K_MAX 33025

/* ------------------------------------------------------------------------------------------ */
/* Quantizer, Sec. 3 "Quantizing" and eq. (2)                                                 */
/* ------------------------------------------------------------------------------------------ */

static float next_up_positive(float q) /* next fp32 above a positive finite q */
{
    uint32_t u;
    memcpy(&u, &q, 4);
    u += 1u;
    memcpy(&q, &u, 4);
    return q;
}

/* Scale and offset from a range. Sec. 3: S = 255, R = vmax - vmin, Q = S / R; eq. (2): the offset
 * is round(Q * vmin). Readings R1 (nudge) and R3 (degenerate unit). */
void orc_params_from_range(float vmin, float vmax, orc_qparams *p)
{
    const float S = 255.0f;
    const float LIM = 4194304.0f; /* 2^22 */
    float R = vmax - vmin;
    float Q = (R > 0.0f) ? S / R : 0.0f;
    int degenerate = !(R > 0.0f) || !isfinite(Q) || !(fabsf(Q * vmin) < LIM) || !(fabsf(Q * vmax) < LIM);
    p->vmin = vmin;
    p->vmax = vmax;
    if (degenerate) {
        float amax = fmaxf(fabsf(vmin), fabsf(vmax));
        Q = (amax > 0.0f) ? S / amax : 1.0f;
        p->Q = Q;
        p->z = (int32_t)rintf(Q * vmin);
        return;
    }
    int32_t z = (int32_t)rintf(Q * vmin);
    for (int it = 0; it < 64; ++it) {
        int32_t top = (int32_t)rintf(Q * vmax) - z;
        if (top >= 255) break;
        Q = next_up_positive(Q);
        z = (int32_t)rintf(Q * vmin);
    }
    p->Q = Q;
    p->z = z;
}

/* Exact fp32 min and max of a strided set (Sec. 3: the range to squeeze into S). */
int orc_range(const float *v, int64_t n, int64_t stride, float *vmin, float *vmax)
{
    if (n <= 0) return ORC_ERR_INVALID_ARG;
    float mn = v[0], mx = v[0];
    for (int64_t i = 0; i < n; ++i) {
        float x = v[i * stride];
        if (!isfinite(x)) return ORC_ERR_NONFINITE;
        if (x < mn) mn = x;
        if (x > mx) mx = x;
    }
    *vmin = mn;
    *vmax = mx;
    return ORC_OK;
}

/* Eq. (2): V' = round(Q V) - round(Q Vmin), clamped to [0, S] (reading R2). */
uint8_t orc_code(float v, const orc_qparams *p)
{
    int32_t c = (int32_t)rintf(p->Q * v) - p->z;
    if (c < 0) c = 0;
    if (c > 255) c = 255;
    return (uint8_t)c;
}

/* Eq. (3): V = (V' + round(Q Vmin)) / Q. */
float orc_recover(uint8_t c, const orc_qparams *p)
{
    return (float)((int32_t)c + p->z) / p->Q;
}

/* Quantize a rows x cols matrix (row stride ldx), per matrix or per row. Writes codes (row stride
 * ldc), the parameters (1 or rows of them) and, if sums != NULL, the per-row code sums. */
int orc_quantize(const float *x, int64_t rows, int64_t cols, int64_t ldx, int gran, uint8_t *codes,
                 int64_t ldc, orc_qparams *params, int32_t *sums)
{
    if (rows <= 0 || cols <= 0 || ldx < cols || ldc < cols) return ORC_ERR_INVALID_ARG;
    if (gran == ORC_PER_MATRIX) {
        float mn = 0, mx = 0;
        for (int64_t r = 0; r < rows; ++r) {
            float a, b;
            int st = orc_range(x + r * ldx, cols, 1, &a, &b);
            if (st) return st;
            if (r == 0 || a < mn) mn = a;
            if (r == 0 || b > mx) mx = b;
        }
        orc_params_from_range(mn, mx, &params[0]);
    } else if (gran == ORC_PER_ROW) {
        for (int64_t r = 0; r < rows; ++r) {
            float a, b;
            int st = orc_range(x + r * ldx, cols, 1, &a, &b);
            if (st) return st;
            orc_params_from_range(a, b, &params[r]);
        }
    } else {
        return ORC_ERR_INVALID_ARG;
    }
    for (int64_t r = 0; r < rows; ++r) {
        const orc_qparams *p = (gran == ORC_PER_MATRIX) ? &params[0] : &params[r];
        int32_t s = 0;
        for (int64_t k = 0; k < cols; ++k) {
            uint8_t c = orc_code(x[r * ldx + k], p);
            codes[r * ldc + k] = c;
            s += c;
        }
        if (sums) sums[r] = s;
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Quantized product, eq. (1) with the offsets of eq. (2)                                     */
/* ------------------------------------------------------------------------------------------ */

/* Offset-applied integer product of one activation row and one weight row (eq. 1 numerator):
 * S = sum_k (a'_k + za) (w'_k + zw), where V'' = V' + round(Q Vmin). Exact in int64. */
static int64_t offset_product(const uint8_t *a, int32_t za, const uint8_t *w, int32_t zw, int64_t K)
{
    int64_t s = 0;
    for (int64_t k = 0; k < K; ++k) s += (int64_t)((int32_t)a[k] + za) * (int64_t)((int32_t)w[k] + zw);
    return s;
}

/* Eq. (1) recovery: Vc = S / (Qa * Qb), fp32 multiply then fp32 divide. */
static float recover_product(int64_t S, float Qa, float Qw)
{
    float den = Qa * Qw;
    return (float)S / den;
}

/* Y[m, n] = S[m, n] / (Qa Qw) (+ bias[n]); acc[m, n] = sum_k a'[m, k] w'[n, k] (int32, 8-bit
 * operands into 32-bit accumulators, Sec. 3.1). A has per-matrix (ga = 0) or per-row (ga = 1)
 * parameters; W has n_blocks equal row blocks, each its own unit (Sec. 3.1, one unit per gate
 * matrix). Any of Y, acc, S64 may be NULL. */
int orc_qmatmul(const uint8_t *A, int64_t lda, const orc_qparams *pa, int ga, int64_t M, int64_t K,
                const uint8_t *W, int64_t ldw, const orc_qparams *pw, int64_t n_blocks, int64_t N,
                const float *bias, float *Y, int64_t ldy, int32_t *acc, int64_t *S64)
{
    if (M <= 0 || N <= 0 || K <= 0 || n_blocks <= 0 || N % n_blocks) return ORC_ERR_INVALID_ARG;
    if (K > ORC_K_MAX) return ORC_ERR_K_TOO_LARGE;
    int64_t rows_per_block = N / n_blocks;
    for (int64_t m = 0; m < M; ++m) {
        const orc_qparams *qa = (ga == ORC_PER_ROW) ? &pa[m] : &pa[0];
        for (int64_t n = 0; n < N; ++n) {
            const orc_qparams *qw = &pw[n / rows_per_block];
            const uint8_t *a = A + m * lda, *w = W + n * ldw;
            if (acc) {
                int32_t s = 0;
                for (int64_t k = 0; k < K; ++k) s += (int32_t)a[k] * (int32_t)w[k];
                acc[m * N + n] = s;
            }
            int64_t S = offset_product(a, qa->z, w, qw->z, K);
            if (S64) S64[m * N + n] = S;
            if (Y) {
                float y = recover_product(S, qa->Q, qw->Q);
                if (bias) y = y + bias[n];
                Y[m * ldy + n] = y;
            }
        }
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Pinned fp32 transcendentals (reading R5)                                                   */
/* ------------------------------------------------------------------------------------------ */

/* E(x) ~ exp(x) in fp32. Cody-Waite: x = n ln2 + r with n = round(x log2(e)) and ln 2 split into
 * ln2_hi (ln 2 truncated to 16 significant bits) and ln2_lo = ln 2 - ln2_hi; e^r by the Taylor
 * polynomial sum_{k<=7} r^k / k! in Horner form with fused multiply-adds; times 2^n built from
 * its exponent bits. x is first clamped to [-87, 88] so that the result is a finite normal. */
float orc_exp(float x)
{
    if (x < -87.0f) x = -87.0f;
    if (x > 88.0f) x = 88.0f;
    float t = x * 1.44269504088896341f;
    float nf = rintf(t);
    int32_t n = (int32_t)nf;
    float r = fmaf(-nf, 0.693145751953125f, x);
    r = fmaf(-nf, 1.428606820309417232e-06f, r);
    float p = 1.984126984126984127e-04f;   /* 1/7! */
    p = fmaf(p, r, 1.388888888888888889e-03f); /* 1/6! */
    p = fmaf(p, r, 8.333333333333333333e-03f); /* 1/5! */
    p = fmaf(p, r, 4.166666666666666667e-02f); /* 1/4! */
    p = fmaf(p, r, 1.666666666666666667e-01f); /* 1/3! */
    p = fmaf(p, r, 0.5f);
    p = fmaf(p, r, 1.0f);
    p = fmaf(p, r, 1.0f);
    uint32_t bits = (uint32_t)(n + 127) << 23;
    float scale;
    memcpy(&scale, &bits, 4);
    return p * scale;
}

float orc_sigmoid(float x) { return 1.0f / (1.0f + orc_exp(-x)); }

float orc_tanh(float x) { return 1.0f - 2.0f / (orc_exp(2.0f * x) + 1.0f); }

/* ------------------------------------------------------------------------------------------ */
/* Quantized LSTM / LSTMP stack with an optional softmax output layer                         */
/* ------------------------------------------------------------------------------------------ */

typedef struct {
    int32_t num_layers;  /* L */
    int32_t input_dim;   /* I */
    int32_t hidden;      /* H, cells per layer */
    int32_t proj;        /* P, recurrent projection size; 0 = none */
    int32_t num_classes; /* C, output classes; 0 = no output layer */
    int32_t output_mode; /* ORC_OUT_NONE / ORC_OUT_QUANT / ORC_OUT_FLOAT */
    int32_t weight_blocks; /* Sec. 3.1 granularity: units per weight matrix, as equal blocks of rows
                              (sub-matrices); 0 or 1 = one unit per matrix */
} orc_lstm_desc;

/* Packed fp32 parameter layout, layer by layer (Ik = I for the first layer, else Rr = P or H):
 *   Wx[4][H][Ik], Wh[4][H][Rr], b[4][H], then Wp[P][H] when P > 0;
 * then Wo[C][Rr] and bo[C] when C > 0. Gate order [i, f, g, o]. */
int64_t orc_lstm_param_count(const orc_lstm_desc *d)
{
    int64_t H = d->hidden, P = d->proj, R = P > 0 ? P : H, n = 0;
    for (int l = 0; l < d->num_layers; ++l) {
        int64_t Ik = (l == 0) ? d->input_dim : R;
        n += 4 * H * Ik + 4 * H * R + 4 * H + (P > 0 ? P * H : 0);
    }
    if (d->num_classes > 0) n += (int64_t)d->num_classes * R + d->num_classes;
    return n;
}

/* One quantized weight matrix: rows x cols codes, its rows split into nb equal blocks
 * (sub-matrices), each block one quantization unit with its own parameters (Sec. 3.1). */
typedef struct {
    uint8_t *codes;
    orc_qparams *p; /* [nb] */
    int64_t rows, cols, nb;
} qunit;

static int make_unit(const float *w, int64_t rows, int64_t cols, int64_t nb, qunit *u)
{
    u->rows = rows;
    u->cols = cols;
    u->nb = nb;
    u->codes = (uint8_t *)malloc((size_t)(rows * cols));
    u->p = (orc_qparams *)calloc((size_t)nb, sizeof(orc_qparams));
    if (!u->codes || !u->p || rows % nb) return ORC_ERR_INVALID_ARG;
    const int64_t per = rows / nb;
    for (int64_t b = 0; b < nb; ++b) {
        int st = orc_quantize(w + b * per * cols, per, cols, cols, ORC_PER_MATRIX, u->codes + b * per * cols, cols,
                              &u->p[b], NULL);
        if (st) return st;
    }
    return ORC_OK;
}

static void free_unit(qunit *u)
{
    free(u->codes);
    free(u->p);
}

/* Recovered product of one quantized activation row with row n of a weight matrix, with the
 * parameters of the block (unit) that row belongs to. */
static float unit_dot(const uint8_t *a, const orc_qparams *pa, const qunit *u, int64_t n)
{
    const orc_qparams *pw = &u->p[n / (u->rows / u->nb)];
    int64_t S = offset_product(a, pa->z, u->codes + n * u->cols, pw->z, u->cols);
    return recover_product(S, pa->Q, pw->Q);
}

/* Units per weight matrix (Sec. 3.1 granularity), or 0 when a matrix's rows do not split evenly. */
static int64_t blocks_of(const orc_lstm_desc *d)
{
    const int64_t nb = d->weight_blocks > 1 ? d->weight_blocks : 1;
    if (d->hidden % nb) return 0;
    if (d->proj > 0 && d->proj % nb) return 0;
    if (d->num_classes > 0 && d->output_mode == ORC_OUT_QUANT && d->num_classes % nb) return 0;
    return nb;
}

/* Quantize one activation row (one unit, reading R6). */
static int quantize_row(const float *v, int64_t n, uint8_t *codes, orc_qparams *p)
{
    return orc_quantize(v, 1, n, n, ORC_PER_ROW, codes, n, p, NULL);
}

/* Softmax (R11): y_c = E(l_c - max) / sum_j E(l_j - max) with the pinned E (R5) on fp32
 * differences; the normalising sum and each quotient are taken in fp64 and rounded once. */
static void softmax_row(const float *logits, int64_t C, float *y)
{
    float mx = logits[0];
    for (int64_t c = 1; c < C; ++c)
        if (logits[c] > mx) mx = logits[c];
    double s = 0.0;
    for (int64_t c = 0; c < C; ++c) {
        y[c] = orc_exp(logits[c] - mx);
        s = s + (double)y[c];
    }
    for (int64_t c = 0; c < C; ++c) y[c] = (float)((double)y[c] / s);
}

/*
 * Forward pass of the quantized LSTM stack (Sec. 3.1 and Fig. 1: each layer takes fp32 inputs,
 * quantizes them on the fly, multiplies in integers, recovers to fp32 and applies the bias and
 * the activation in fp32; weights are quantized offline, one unit per gate matrix).
 *
 *   x       [B][T][I] fp32 frames
 *   y       [B][T][C] softmax outputs when C > 0, else [B][T][Rr] top-layer outputs
 *   h_state [L][B][Rr], c_state [L][B][H]: initial state in, final state out (NULL = zeros)
 *   h_all   [L][B][T][Rr], every layer's output at every frame (NULL = not written)
 *   logits  [B][T][C] pre-softmax outputs (NULL = not written)
 */
int orc_lstm_forward(const orc_lstm_desc *d, const float *params, const float *x, int64_t B, int64_t T,
                     float *y, float *h_state, float *c_state, float *h_all, float *logits_out)
{
    const int64_t L = d->num_layers, I = d->input_dim, H = d->hidden, P = d->proj, C = d->num_classes;
    const int64_t R = P > 0 ? P : H;
    if (L <= 0 || I <= 0 || H <= 0 || P < 0 || C < 0 || B < 0 || T < 0) return ORC_ERR_INVALID_ARG;
    if (C > 0 && d->output_mode != ORC_OUT_QUANT && d->output_mode != ORC_OUT_FLOAT) return ORC_ERR_INVALID_ARG;
    if (I > ORC_K_MAX || H > ORC_K_MAX || R > ORC_K_MAX) return ORC_ERR_K_TOO_LARGE;
    const int64_t nb = blocks_of(d);
    if (!nb) return ORC_ERR_INVALID_ARG;

    /* a1: offline weight quantization, one unit per gate matrix (or per block of its rows) */
    qunit *wx = (qunit *)calloc((size_t)(4 * L), sizeof(qunit));
    qunit *wh = (qunit *)calloc((size_t)(4 * L), sizeof(qunit));
    qunit *wp = (qunit *)calloc((size_t)L, sizeof(qunit));
    const float **bias = (const float **)calloc((size_t)L, sizeof(float *));
    qunit wo;
    memset(&wo, 0, sizeof(wo));
    const float *wo_f = NULL, *bo = NULL;
    int st = ORC_OK;
    const float *q = params;
    for (int64_t l = 0; l < L && !st; ++l) {
        int64_t Ik = (l == 0) ? I : R;
        for (int g = 0; g < 4 && !st; ++g) st = make_unit(q + g * H * Ik, H, Ik, nb, &wx[4 * l + g]);
        q += 4 * H * Ik;
        for (int g = 0; g < 4 && !st; ++g) st = make_unit(q + g * H * R, H, R, nb, &wh[4 * l + g]);
        q += 4 * H * R;
        bias[l] = q;
        q += 4 * H;
        if (P > 0) {
            if (!st) st = make_unit(q, P, H, nb, &wp[l]);
            q += P * H;
        }
    }
    if (C > 0 && !st) {
        wo_f = q;
        if (d->output_mode == ORC_OUT_QUANT) st = make_unit(q, C, R, nb, &wo);
        q += C * R;
        bo = q;
    }

    /* the widest row any step quantizes: the network input, the cell outputs m_t or the recurrent
       input r_t (R = P can exceed H) */
    int64_t maxK = I > H ? I : H;
    if (R > maxK) maxK = R;
    float *hprev = (float *)calloc((size_t)(L * R), sizeof(float));
    float *cprev = (float *)calloc((size_t)(L * H), sizeof(float));
    float *layer_in = (float *)calloc((size_t)maxK, sizeof(float));
    float *m = (float *)calloc((size_t)H, sizeof(float));
    float *hnew = (float *)calloc((size_t)R, sizeof(float));
    float *lg = (float *)calloc((size_t)(C > 0 ? C : 1), sizeof(float));
    uint8_t *cx = (uint8_t *)calloc((size_t)maxK, 1);
    uint8_t *ch = (uint8_t *)calloc((size_t)maxK, 1);

    for (int64_t b = 0; b < B && !st; ++b) {
        for (int64_t l = 0; l < L; ++l) {
            for (int64_t k = 0; k < R; ++k) hprev[l * R + k] = h_state ? h_state[(l * B + b) * R + k] : 0.0f;
            for (int64_t k = 0; k < H; ++k) cprev[l * H + k] = c_state ? c_state[(l * B + b) * H + k] : 0.0f;
        }
        for (int64_t t = 0; t < T && !st; ++t) {
            memcpy(layer_in, x + (b * T + t) * I, (size_t)I * sizeof(float));
            int64_t Kin = I;
            for (int64_t l = 0; l < L && !st; ++l) {
                orc_qparams px, ph;
                st = quantize_row(layer_in, Kin, cx, &px); /* inputs quantized on the fly */
                if (!st) st = quantize_row(hprev + l * R, R, ch, &ph);
                if (st) break;
                float *cl = cprev + l * H;
                for (int64_t j = 0; j < H; ++j) {
                    float gate[4];
                    for (int g = 0; g < 4; ++g) {
                        float yx = unit_dot(cx, &px, &wx[4 * l + g], j);
                        float yh = unit_dot(ch, &ph, &wh[4 * l + g], j);
                        gate[g] = (yx + bias[l][g * H + j]) + yh;
                    }
                    float ig = orc_sigmoid(gate[0]);
                    float fg = orc_sigmoid(gate[1]);
                    float gg = orc_tanh(gate[2]);
                    float og = orc_sigmoid(gate[3]);
                    float fc = fg * cl[j];
                    float in = ig * gg;
                    cl[j] = fc + in;
                    m[j] = og * orc_tanh(cl[j]);
                }
                if (P > 0) {
                    orc_qparams pm;
                    st = quantize_row(m, H, cx, &pm);
                    if (st) break;
                    for (int64_t k = 0; k < P; ++k) hnew[k] = unit_dot(cx, &pm, &wp[l], k);
                } else {
                    memcpy(hnew, m, (size_t)H * sizeof(float));
                }
                memcpy(hprev + l * R, hnew, (size_t)R * sizeof(float));
                if (h_all) memcpy(h_all + ((l * B + b) * T + t) * R, hnew, (size_t)R * sizeof(float));
                memcpy(layer_in, hnew, (size_t)R * sizeof(float));
                Kin = R;
            }
            if (st) break;
            float *yrow = y ? y + (b * T + t) * (C > 0 ? C : R) : NULL;
            if (C > 0) {
                if (d->output_mode == ORC_OUT_QUANT) {
                    orc_qparams pr;
                    st = quantize_row(layer_in, R, cx, &pr);
                    if (st) break;
                    for (int64_t c = 0; c < C; ++c) lg[c] = unit_dot(cx, &pr, &wo, c) + bo[c];
                } else {
                    for (int64_t c = 0; c < C; ++c) {
                        double s = 0.0;
                        for (int64_t k = 0; k < R; ++k) s += (double)wo_f[c * R + k] * (double)layer_in[k];
                        lg[c] = (float)(s + (double)bo[c]);
                    }
                }
                if (logits_out) memcpy(logits_out + (b * T + t) * C, lg, (size_t)C * sizeof(float));
                if (yrow) softmax_row(lg, C, yrow);
            } else if (yrow) {
                memcpy(yrow, layer_in, (size_t)R * sizeof(float));
            }
        }
        for (int64_t l = 0; l < L && !st; ++l) {
            if (h_state) memcpy(h_state + (l * B + b) * R, hprev + l * R, (size_t)R * sizeof(float));
            if (c_state) memcpy(c_state + (l * B + b) * H, cprev + l * H, (size_t)H * sizeof(float));
        }
    }

    for (int64_t i = 0; i < 4 * L; ++i) {
        free_unit(&wx[i]);
        free_unit(&wh[i]);
    }
    for (int64_t i = 0; i < L; ++i) free_unit(&wp[i]);
    free_unit(&wo);
    free(wx);
    free(wh);
    free(wp);
    free(bias);
    free(hprev);
    free(cprev);
    free(layer_in);
    free(m);
    free(hnew);
    free(lg);
    free(cx);
    free(ch);
    (void)wo_f;
    return st;
}

/* Weight quantization alone (offline step), for parity of the offline codes: writes every unit's
 * codes at the offsets of the packed parameter layout (bias slots untouched) and the parameters
 * of each unit in order (4 Wx, 4 Wh, Wp per layer, then Wo). */
int orc_lstm_quantize_weights(const orc_lstm_desc *d, const float *params, uint8_t *codes, orc_qparams *qp,
                              int64_t *n_units)
{
    const int64_t L = d->num_layers, I = d->input_dim, H = d->hidden, P = d->proj, C = d->num_classes;
    const int64_t R = P > 0 ? P : H;
    const int64_t nb = blocks_of(d);
    if (!nb) return ORC_ERR_INVALID_ARG;
    const float *q = params;
    int64_t u = 0, off = 0;
    int st = ORC_OK;
    /* one matrix of `rows` rows as nb units of rows/nb rows each, codes at the packed offset */
#define ORC_UNITS(W, ROWS, COLS)                                                                      \
    for (int64_t b_ = 0; b_ < nb && !st; ++b_, ++u)                                                   \
        st = orc_quantize((W) + b_ * ((ROWS) / nb) * (COLS), (ROWS) / nb, (COLS), (COLS), ORC_PER_MATRIX, \
                          codes + off + b_ * ((ROWS) / nb) * (COLS), (COLS), &qp[u], NULL);
    for (int64_t l = 0; l < L && !st; ++l) {
        int64_t Ik = (l == 0) ? I : R;
        for (int g = 0; g < 4 && !st; ++g) {
            ORC_UNITS(q + g * H * Ik, H, Ik)
            off += H * Ik;
        }
        q += 4 * H * Ik;
        for (int g = 0; g < 4 && !st; ++g) {
            ORC_UNITS(q + g * H * R, H, R)
            off += H * R;
        }
        q += 4 * H * R + 4 * H;
        off += 4 * H; /* bias slot: no codes */
        if (P > 0 && !st) {
            ORC_UNITS(q, P, H)
            off += P * H;
            q += P * H;
        }
    }
    if (C > 0 && d->output_mode == ORC_OUT_QUANT && !st) {
        ORC_UNITS(q, C, R)
    }
#undef ORC_UNITS
    if (n_units) *n_units = u;
    return st;
}

/* Sec. 4 frontend: features of n consecutive frames are stacked (the frame and n-1 frames of
 * right context) and only every stride-th stacked frame is presented to the network.
 * x [B][T][I] -> out [B][T'][n*I], T' = ceil(T / stride); out[b][t'][k*I + i] is frame
 * stride*t' + k of sequence b (the last frame where that is past the end, R9). */
int orc_stack_frames(const float *x, int64_t B, int64_t T, int64_t I, int n, int stride, float *out)
{
    if (B < 0 || T < 1 || I < 1 || n < 1 || stride < 1) return ORC_ERR_INVALID_ARG;
    const int64_t Tp = (T + stride - 1) / stride;
    for (int64_t b = 0; b < B; ++b)
        for (int64_t tp = 0; tp < Tp; ++tp)
            for (int k = 0; k < n; ++k) {
                int64_t t = tp * stride + k;
                if (t > T - 1) t = T - 1;
                for (int64_t i = 0; i < I; ++i) out[((b * Tp + tp) * n + k) * I + i] = x[(b * T + t) * I + i];
            }
    return ORC_OK;
}
