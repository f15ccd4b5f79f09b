// tc_gemm.h — host interface of the exact fp16 tcgen05 product (qgemm_tc.cu) for the other
// translation units (not part of the ABI).
//
// Operands are centered codes (c - 128) in fp16, row-major, K padded with zeros to kp (a multiple
// of 64). The product is the exact integer sum of eq. (1); see qgemm_tc.cu.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>

#include "qnn_host.h"

namespace qnn {

// The two operands of one product, as TMA tensor maps: A [M][kp] and W [N][kp]. `bn` is the tile
// width (rows of W per tile: 32, 64, 128 or 256; the LSTM epilogue takes 32, 64 or 128, the row
// epilogue 64 or 128); the maps depend on
// it. With `pdl` set the product is launched as a programmatic dependent launch: its block setup
// may overlap the previous kernel of the stream (it waits for that kernel before reading).
struct TcOperands {
    CUtensorMap a, w;
    int64_t M = 0, N = 0, kp = 0;
    int bn = 256;
    bool pdl = false;
    bool row_epilogue = false;  // linear products: set by tc_operands when kp <= 1024 and bn <= 128
    // LSTM epilogues: a last, partial wave of tiles may run as half-width items (QNN_TC_HALF=0: never)
    bool half_items = true;
    // persistent grid: at most this many blocks (0: one per SM)
    int max_blocks = 0;
};
qnn_status tc_operands(TcOperands *op, const __half *A16, int64_t M, const __half *W16, int64_t N, int64_t kp, int bn);
// Default tile width of a linear product (QNN_TC_BN overrides).
int tc_pick_bn(int64_t M, int64_t N, int64_t kp);
// Of the candidate tile widths (widest first), the widest whose share of busy SMs over the last
// wave of tiles is within 10% of the best candidate's (QNN_TC_BN overrides when it is a candidate).
int tc_choose_bn(int64_t M, int64_t N, const int *cands, int n);

// Recovered product (eq. 1, eq. 3) plus optional bias into Y [M][ldy]; acc_out [M][N] (nullable)
// receives the raw int32 code products. K is the true reduction length (<= QNN_K_MAX).
qnn_status tc_linear(const TcOperands &op, const qnn_qparams *pa, int per_row, const int32_t *rsA, int64_t K,
                     const qnn_qparams *pw, int64_t rows_per_block, const int32_t *csW, const float *bias, float *Y,
                     int64_t ldy, int32_t *acc_out, cudaStream_t st);

// Destination of the fused LSTM epilogue for one step: px row b at px + b*px_ld holds the four
// recovered input products plus bias ([i f g o] x H), c [B][H] the cell state (updated in place),
// the cell outputs m_t go to h + b*h_ld. H must be a multiple of 4 and the pointers 16-byte aligned.
struct TcLstmOut {
    const float *px;
    int64_t px_ld;
    float *c;
    float *h;
    int64_t h_ld;
    int H;
    int ups = 1;  // weight units per gate matrix (Sec. 3.1 sub-matrices); pw4 then has 4 ups entries
    int cpu = 0;  // cells per unit (H / ups, a multiple of 4)
};

// The input side of a step when it is fused into the gate kernel (tc_lstm_gates_x): centered fp16
// codes of x_t (row b at x16 + b * x_pitch, kx columns: K_x true values then zeros, kx a multiple of
// 64 and at most 1024), row b's unit and code sum at pa[b * stride] and rs[b * stride], the Wx gate
// matrices interleaved like Wh ([4 round_up(H, 8)][kx]), their units (4 ups, gate-major), row code
// sums in gate-major order [4][H] and the bias [4H].
struct TcLstmInput {
    const __half *x16 = nullptr;
    int64_t x_pitch = 0, kx = 0;
    int K_x = 0;
    const qnn_qparams *pa = nullptr;
    const int32_t *rs = nullptr;
    int64_t stride = 1;
    const __half *wx16 = nullptr;
    const qnn_qparams *pw4 = nullptr;
    const int32_t *cs = nullptr;
    const float *bias = nullptr;
    // the same column constants as one [12][H] fp32 table, staged per tile by TMA: rows 0-3 the bias
    // of gates i f g o, rows 4-7 the Wx row code sums, rows 8-11 the Wh row code sums (integers below
    // 2^24, exact in fp32); 16-byte aligned, H a multiple of 4
    const void *colc = nullptr;
};

// One recurrent step's gate product and cell update: A = centered codes of h_{t-1} (one unit per
// row: pa, rsA), W = the four Wh gate matrices interleaved in 8-cell groups [i f g o] x 8 rows
// (op.N = 4 * round_up(H, 8)), pw4 the gate units (4 ups, gate-major), cs their row code sums in
// gate-major order [4][H]. K (true) <= 1024.
// As tc_lstm_gates, with the step's input product computed in the same kernel (a second operand
// pair and accumulator) instead of read from out.px: pre = (R(x_t Wx) + b) + R(h_{t-1} Wh), the
// same operations in the same order as the batched product followed by tc_lstm_gates.
qnn_status tc_lstm_gates_x(const TcOperands &op, const qnn_qparams *pa, const int32_t *rsA, int64_t K,
                           const qnn_qparams *pw4, const int32_t *cs, const TcLstmOut &out, const TcLstmInput &in,
                           cudaStream_t st);
qnn_status tc_lstm_gates(const TcOperands &op, const qnn_qparams *pa, const int32_t *rsA, int64_t K,
                         const qnn_qparams *pw4, const int32_t *cs, const TcLstmOut &out, cudaStream_t st);

// Split-K partial sums of the centered integer product: part[s][m][n] = sum over K range s of
// (a - 128)(w - 128), int32, ranges of at most 1024 so that each is exact in one accumulator;
// the slices add up to P = acc - 128 (rsA + csW) + 128^2 K. ldpart >= N (elements).
// K ranges giving at most one wave of work items (each range one exact chunk; at most
// max(max_splits, the chunks K needs) ranges); without fill_sms, the fewest exact chunks.
int tc_partial_splits(const TcOperands &op, int max_splits, bool fill_sms = true);
qnn_status tc_partial(const TcOperands &op, int splits, int32_t *part, int64_t ldpart, cudaStream_t st);

// u8 codes [rows][ldi] -> centered fp16 [rows][ldo], zero past K.
qnn_status launch_center_fp16(const uint8_t *in, int64_t rows, int64_t K, int64_t ldi, __half *out, int64_t ldo,
                              cudaStream_t st);

}  // namespace qnn
