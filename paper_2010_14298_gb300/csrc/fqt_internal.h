// fqt_internal.h -- declarations shared by the translation units of the
// GB300 FQT library (kernel argument blocks and host launchers).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "fqt.h"

namespace fqt {

enum { KIND_PTQ = 0, KIND_PSQ = 1, KIND_BHQ = 2, KIND_SHIFT = 3, KIND_DET = 4 };



// Arguments of the quantizer kernel (see fqt_quant.cu for the mapping).
struct QuantArgs {
  const void *h;
  int64_t N;
  int C, CO;
  int kind, bits, block;
  uint32_t key0, key1;
  uint32_t round_keys[20];  // Philox4x32-10 key schedule of (key0, key1)
  // code set 2: Q_b2 (gradient) or the forward operand (KIND_DET)
  uint8_t *c2;
  uint16_t *f2;  // fp16 carriers of code set 2 (may be null)
  float *inv2, *zero2;
  int32_t *rsum2, *csum2, *lead2;
  // code set 1: Q_b1, 8-bit stochastic PTQ (may be null)
  uint8_t *c1;
  uint16_t *f1;  // fp16 carriers of code set 1 (may be null)
  float *inv1, *zero1;
  int32_t *rsum1, *csum1;
  float *hz, *hr;  // BHQ grad_X offsets of code set 2 (may be null)
  const int32_t *perm, *gstart;  // adaptive BHQ groups (block 0)
  unsigned *slots;               // their work queue (zeroed by the grouping)
  // the shift quantizer (KIND_SHIFT): shifted carriers, shifts, their column
  // sums and the common scale / zero point
  uint16_t *fs;
  int32_t *shift, *scs;
  float *sscale;
  const float2 *part;
  int npart;
  // code pass of the two-pass quantizers: column parts per chunk of rows
  // (> 1: the row sums are accumulated atomically, cleared by the first pass)
  int code_split;
  int *status;
  // launch geometry
  int TW, OPT, RL, RPL, GT, G, nchunk, unit_rows, stage_bytes;
  int64_t n_units;
};

fqt_status quant_geometry(QuantArgs &a, int num_sms, int *nth, int *grid,
                          size_t *smem);
cudaError_t launch_quant(const QuantArgs &a, bool bf16, int nth, int grid,
                         size_t smem, cudaStream_t st);
fqt_status quant2_geometry(QuantArgs &a, bool bf16, int num_sms, int *grid,
                           size_t *smem);
cudaError_t launch_quant2(const QuantArgs &a, bool bf16, int grid, size_t smem,
                          cudaStream_t st);
cudaError_t launch_range(const void *x, bool bf16, int64_t count, float2 *part,
                         int *npart, int32_t *z0, int64_t nz0, int32_t *z1,
                         int64_t nz1, int num_sms, cudaStream_t st);

fqt_status launch_fwd_codes(const void *X, bool bf16, int64_t rows, int cols, int bits,
                            uint16_t *f16, uint8_t *c8, int32_t *col_sum, const float2 *part,
                            int npart, float *inv_out, float *zero_out, int *status,
                            int num_sms, cudaStream_t st, int conv_zero = 0,
                            int32_t *code_zero_out = nullptr);
fqt_status launch_conv_colsum(const uint16_t *f16, int64_t n, int h, int w, int c, int kh,
                              int kw, int pad, int bits, int32_t *col_sum, cudaStream_t st);
bool bhq_pass_supported(int C, int block, bool bf16);
size_t bhq_pass_bytes(int64_t N, int64_t C);
fqt_status launch_bhq_passes(QuantArgs &a, bool bf16, int num_sms, void *scratch,
                             float2 *part, cudaStream_t st);
size_t sample_pass_bytes(int64_t N, int64_t C, int64_t rows_per_sample);
fqt_status launch_sample_passes(QuantArgs &a, bool bf16, int64_t rows_per_sample, int num_sms,
                                void *scratch, float2 *part, cudaStream_t st);
fqt_status launch_shift(QuantArgs &a, bool bf16, int num_sms, cudaStream_t st);
cudaError_t launch_bhq_offsets(const float *zero, const int32_t *rsum,
                               const int32_t *lead, float *hz, float *hr, int64_t N,
                               int C, int bits, int block, cudaStream_t st);

size_t group_workspace_bytes(int64_t N);
// grad_X work lists of the adaptive groups: two counters, the groups of up to
// 32 rows (at most N) and the larger ones (at most N / 33)
inline size_t group_list_bytes(int64_t N) {
  const size_t n = N > 0 ? (size_t)N : 0;
  return 256 + ((n * 4 + 255) & ~(size_t)255) + (n / 32 + 1) * 4;
}
fqt_status launch_bhq_grouping(const void *dH, bool bf16, int64_t N, int C, int32_t *perm,
                               int32_t *gstart, int32_t *gsize, void *scratch,
                               size_t scratch_bytes, unsigned **slot_counter, cudaStream_t st);
fqt_status launch_bhq_groups(QuantArgs &a, bool bf16, int num_sms, cudaStream_t st);

int device_sm_count();

// Records the CUDA error behind an FQT_ECUDA return (per thread) and returns
// FQT_ECUDA, or FQT_OK for cudaSuccess.
fqt_status cuda_fail(cudaError_t e, const char *where);

size_t gemm_workspace_bytes(int64_t N, int64_t C, int64_t D);
size_t debug_workspace_bytes(int64_t M, int64_t N, int64_t K);
fqt_status grad_w_fixed_scratch(const fqt_qtensor *qa, const fqt_qtensor *qx,
                                float *grad_W, cudaStream_t st);
fqt_status fixed_scratch_status(int **out);
fqt_status debug_wait_timeout(void *ws, size_t ws_bytes, uint64_t limit_ns, cudaStream_t st);
size_t conv_grad_x_ws_bytes(int64_t cin);
fqt_status conv_grad_x_nhwc(const fqt_qtensor *q2, const fqt_qtensor *qw, int64_t n, int64_t h,
                            int64_t w, int64_t cin, int k, int pad, float *out, void *ws,
                            size_t ws_bytes, cudaStream_t st);
fqt_status debug_mma_peak(int kind, int64_t iters, double *ops_out, void *ws, size_t ws_bytes,
                          cudaStream_t st);
fqt_status linear_forward(const fqt_qtensor *qx, const fqt_qtensor *qw, float *H, void *ws,
                          size_t ws_bytes, cudaStream_t st);
fqt_status linear_backward(const fqt_qtensor *q_b2, const fqt_qtensor *q_b1,
                           const fqt_qtensor *qx, const fqt_qtensor *qw,
                           float *grad_X, float *grad_W, void *ws,
                           size_t ws_bytes, cudaStream_t st);
fqt_status debug_int_gemm(const uint8_t *A, int a_kmajor, int a_bits,
                          const uint8_t *Bm, int b_kmajor, int b_bits, int64_t M,
                          int64_t N, int64_t K, int64_t *out, void *ws,
                          size_t ws_bytes, cudaStream_t st);
fqt_status debug_int_gemm_u8(const uint8_t *A, int a_bits, const uint8_t *Bm, int b_bits,
                             int64_t M, int64_t N, int64_t K, int64_t *out, void *ws,
                             size_t ws_bytes, cudaStream_t st);

}  // namespace fqt
