// qnn_host.h — host-side helpers shared by the libqnn translation units (not part of the ABI).
#pragma once

#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cuda_runtime.h>

#include "../../include/qnn.h"

namespace qnn {

#define QNN_CUDA_TRY(expr)                                                                   \
    do {                                                                                     \
        cudaError_t _e = (expr);                                                             \
        if (_e != cudaSuccess) {                                                             \
            if (std::getenv("QNN_DEBUG"))                                                    \
                std::fprintf(stderr, "qnn: %s failed: %s (%s:%d)\n", #expr, cudaGetErrorString(_e), \
                             __FILE__, __LINE__);                                            \
            return _e == cudaErrorMemoryAllocation ? QNN_ERR_NO_MEMORY : QNN_ERR_CUDA;      \
        }                                                                                    \
    } while (0)

// A failure status, reported with its source location on stderr when QNN_DEBUG is set.
inline qnn_status debug_fail(qnn_status s, const char *file, int line) {
    if (std::getenv("QNN_DEBUG")) std::fprintf(stderr, "qnn: status %d at %s:%d\n", (int)s, file, line);
    return s;
}
#define QNN_FAIL(code) ::qnn::debug_fail((code), __FILE__, __LINE__)

#define QNN_TRY(expr)                       \
    do {                                    \
        qnn_status _s = (expr);             \
        if (_s != QNN_OK) return _s;        \
    } while (0)

inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

// True if p is memory the current device can use as a plain device pointer (device or managed
// allocations). Pinned or pageable host memory is rejected by the compute calls.
bool is_device_ptr(const void *p);

// The address under which kernels of the current device reach p when p is pinned (page-locked)
// host memory mapped into the device's address space; null for any other memory. Kernels that
// write a host output through it send each byte over the host link once, with no staging copy.
void *host_mapped_ptr(void *p);

// Library-owned, grow-only device scratch of the current device (one slot per purpose).
enum ScratchSlot { kScratchReduce = 0, kScratchTc = 1, kScratchCount = 2 };
qnn_status scratch(ScratchSlot slot, size_t bytes, void **out);

// The device status word of the current device (allocated and zeroed on first use).
qnn_status status_word(int **out);

// Streaming multiprocessor count of the current device (cached).
int sm_count();

// While kernel timing is enabled (qnn_profile_enable), brackets the launches made during its
// lifetime with CUDA events on `st`, accounted under `name` (a static string).
class ProfScope {
  public:
    ProfScope(const char *name, cudaStream_t st);
    ~ProfScope();
    ProfScope(const ProfScope &) = delete;
    ProfScope &operator=(const ProfScope &) = delete;

  private:
    cudaStream_t st_;
    int idx_;
};

// Launches (host side) used across translation units.
qnn_status launch_quantize_rows(const float *x, int64_t rows, int64_t cols, int64_t ldx, uint8_t *codes,
                                int64_t ldc, qnn_qparams *params, int32_t *sums, cudaStream_t st);
qnn_status launch_quantize_matrix(const float *x, int64_t rows, int64_t cols, int64_t ldx, uint8_t *codes,
                                  int64_t ldc, qnn_qparams *params, int32_t *sums, float *partials,
                                  unsigned *counter, int max_blocks, cudaStream_t st);
qnn_status launch_qgemm(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA, int64_t M,
                        int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw, int64_t rows_per_block,
                        const int32_t *csW, int64_t N, const float *bias, float *Y, int64_t ldy, int32_t *acc_out,
                        cudaStream_t st);
// The two product datapaths behind launch_qgemm: the warp-level integer MMA (any shape) and the
// exact fp16 tcgen05 path (needs fp16 copies of both operands in `scratch`, tc_scratch_bytes).
qnn_status launch_qgemm_imma(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA,
                             int64_t M, int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw,
                             int64_t rows_per_block, const int32_t *csW, int64_t N, const float *bias, float *Y,
                             int64_t ldy, int32_t *acc_out, cudaStream_t st);
qnn_status launch_qgemm_tc(const uint8_t *A, int64_t lda, const qnn_qparams *pa, int ga, const int32_t *rsA, int64_t M,
                           int64_t K, const uint8_t *W, int64_t ldw, const qnn_qparams *pw, int64_t rows_per_block,
                           const int32_t *csW, int64_t N, const float *bias, float *Y, int64_t ldy, int32_t *acc_out,
                           void *scratch, cudaStream_t st);
size_t tc_scratch_bytes(int64_t M, int64_t N, int64_t K);
// Softmax of rows of logits into y. With tm_B > 0 the rows are time-major, frames tm_t0 .. of tm_B
// sequences (row i: frame tm_t0 + i / tm_B of sequence i % tm_B), and each goes to its row of the
// sequence-major y [tm_B][tm_T][C].
qnn_status launch_softmax_rows(const float *logits, int64_t rows, int64_t C, float *y, cudaStream_t st,
                               int64_t tm_B = 0, int64_t tm_T = 0, int64_t tm_t0 = 0);
// Sec. 4 frame stacking (frontend.cu): x [B][T][I] -> out [B][ceil(T/stride)][n I], device memory.
qnn_status launch_stack_frames(const float *x, int64_t B, int64_t T, int64_t I, int n, int stride, float *out,
                               cudaStream_t st);

}  // namespace qnn
