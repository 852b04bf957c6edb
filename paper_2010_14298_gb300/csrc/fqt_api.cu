// fqt_api.cu -- the extern "C" entry points of include/fqt.h: argument
// validation, workspace carving, launches, and the device status word.
#include <cuda_runtime.h>
#include <stdio.h>
#include <string.h>

#include "fqt.h"
#include "fqt_common.cuh"
#include "fqt_internal.h"

namespace fqt {

int device_sm_count() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < 64 && cached[dev]) return cached[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  if (dev < 64) cached[dev] = n;
  return n;
}

static thread_local char g_last_error[160] = "none";

fqt_status cuda_fail(cudaError_t e, const char *where) {
  if (e == cudaSuccess) return FQT_OK;
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s", where, cudaGetErrorName(e));
  return FQT_ECUDA;
}

static bool aligned(const void *p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

static fqt_status check_ws(void *ws, size_t bytes, size_t need) {
  if (!ws || !aligned(ws, 256) || bytes < need) return FQT_EWORKSPACE;
  return FQT_OK;
}

// Deterministic PTQ of a forward operand (Q_f / Q_theta).
static fqt_status quantize_forward(const void *X, fqt_dtype dtype, int64_t rows,
                                   int64_t cols, int bits, fqt_qtensor *out,
                                   void *ws, size_t ws_bytes, void *stream) {
  if (rows < 0 || cols <= 0 || cols > (1 << 20) || bits < 2 || bits > 8) return FQT_EINVAL;
  if (!out) return FQT_EINVAL;
  if (rows > 0 && (!X || (!out->codes && !out->codes_f16) || !out->inv_s || !out->zero))
    return FQT_EINVAL;
  if (dtype != FQT_F32 && dtype != FQT_BF16) return FQT_EINVAL;
  if (cols % 8) return FQT_EUNSUPPORTED;
  if (!aligned(X, 16) || !aligned(out->codes, 16) || !aligned(out->codes_f16, 16))
    return FQT_EINVAL;
  fqt_status s = check_ws(ws, ws_bytes, kGemmOffset);
  if (s != FQT_OK) return s;
  out->rows = rows;
  out->cols = cols;
  out->bits = bits;
  out->kind = FQT_PTQ;
  out->block = 0;
  memset(out->conv, 0, sizeof(out->conv));
  if (rows == 0) return FQT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int nsm = device_sm_count();
  char *w = static_cast<char *>(ws);
  float2 *part = reinterpret_cast<float2 *>(w + kRangeOffset);
  int npart = 0;
  cudaError_t e = launch_range(X, dtype == FQT_BF16, rows * cols, part, &npart,
                               out->col_sum, out->col_sum ? cols : 0, nullptr, 0,
                               nsm, st);
  if (e != cudaSuccess) return cuda_fail(e, "range pass");
  if (!out->row_sum && cols / 8 <= 1024)
    return launch_fwd_codes(X, dtype == FQT_BF16, rows, (int)cols, bits, out->codes_f16,
                            out->codes, out->col_sum, part, npart, out->inv_s, out->zero,
                            reinterpret_cast<int *>(w), nsm, st);
  QuantArgs a;
  memset(&a, 0, sizeof(a));
  a.h = X;
  a.N = rows;
  a.C = (int)cols;
  a.kind = KIND_DET;
  a.bits = bits;
  a.block = 0;
  a.c2 = out->codes;
  a.f2 = out->codes_f16;
  a.inv2 = out->inv_s;
  a.zero2 = out->zero;
  a.rsum2 = out->row_sum;
  a.csum2 = out->col_sum;
  a.part = part;
  a.npart = npart;
  a.status = reinterpret_cast<int *>(w);
  int nth, grid;
  size_t smem;
  s = quant_geometry(a, nsm, &nth, &grid, &smem);
  if (s != FQT_OK) return s;
  e = launch_quant(a, dtype == FQT_BF16, nth, grid, smem, st);
  return cuda_fail(e, "quantizer launch");
}

// Q_f of a stride-1 conv input as its implicit im2col matrix (see fqt.h).
static fqt_status quantize_conv(const void *X, fqt_dtype dtype, int64_t n, int64_t h,
                                int64_t wd, int64_t c, int kh, int kw, int pad, int bits,
                                fqt_qtensor *out, void *ws, size_t ws_bytes, void *stream) {
  if (!out || bits < 2 || bits > 8 || n < 0 || h <= 0 || wd <= 0 || c <= 0 || kh <= 0 ||
      kw <= 0 || pad < 0)
    return FQT_EINVAL;
  const int64_t oh = h + 2 * pad - kh + 1, ow = wd + 2 * pad - kw + 1;
  if (oh <= 0 || ow <= 0 || h > (1 << 16) || wd > (1 << 16) || c > (1 << 16)) return FQT_EINVAL;
  if (dtype != FQT_F32 && dtype != FQT_BF16) return FQT_EINVAL;
  if (n > 0 && (!X || !out->codes_f16 || !out->inv_s || !out->zero || !out->col_sum))
    return FQT_EINVAL;
  if (out->row_sum) return FQT_EUNSUPPORTED;  // row sums of the im2col rows: not built
  if (c % 8 || c > 4096) return FQT_EUNSUPPORTED;  // column sums stage c ints in shared memory
  if (!aligned(X, 16) || !aligned(out->codes, 16) || !aligned(out->codes_f16, 16))
    return FQT_EINVAL;
  const int64_t pixels = n * h * wd;
  fqt_status s = check_ws(ws, ws_bytes, kGemmOffset);
  if (s != FQT_OK) return s;
  out->rows = n * oh * ow;
  out->cols = (int64_t)kh * kw * c;
  out->bits = bits;
  out->kind = FQT_PTQ;
  out->block = 0;
  const int32_t geo[7] = {(int32_t)n, (int32_t)h, (int32_t)wd, (int32_t)c, kh, kw, pad};
  memcpy(out->conv, geo, sizeof(geo));
  out->conv[7] = 0;
  if (n == 0) return FQT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int nsm = device_sm_count();
  char *w = static_cast<char *>(ws);
  float2 *part = reinterpret_cast<float2 *>(w + kRangeOffset);
  int npart = 0;
  cudaError_t e = launch_range(X, dtype == FQT_BF16, pixels * c, part, &npart, out->col_sum,
                               (int64_t)kh * kw * c, nullptr, 0, nsm, st);
  if (e != cudaSuccess) return cuda_fail(e, "range pass");
  // code(0.0), the padding's code, follows the column sums (device memory)
  int32_t *zc = out->col_sum + (int64_t)kh * kw * c;
  s = launch_fwd_codes(X, dtype == FQT_BF16, pixels, (int)c, bits, out->codes_f16, out->codes,
                       nullptr, part, npart, out->inv_s, out->zero, reinterpret_cast<int *>(w),
                       nsm, st, pad > 0 ? 1 : 0, zc);
  if (s != FQT_OK) return s;
  return launch_conv_colsum(out->codes_f16, n, (int)h, (int)wd, (int)c, kh, kw, pad, bits,
                            out->col_sum, st);
}

}  // namespace fqt

using namespace fqt;

extern "C" {

fqt_status fqt_quantize_act_conv(const void *X, fqt_dtype dtype, int64_t n, int64_t h,
                                 int64_t w, int64_t c, int kh, int kw, int pad, int bits,
                                 fqt_qtensor *out, void *workspace, size_t ws_bytes,
                                 void *stream) {
  return quantize_conv(X, dtype, n, h, w, c, kh, kw, pad, bits, out, workspace, ws_bytes,
                       stream);
}

size_t fqt_workspace_size(int64_t N, int64_t C, int64_t D) {
  size_t need = gemm_workspace_bytes(N, C, D);
  const size_t grp = group_workspace_bytes(N);         // adaptive BHQ grouping
  const size_t list = group_list_bytes(N);               // its grad_X work lists
  const size_t bhq = bhq_pass_bytes(N, C);                // two-pass BHQ scratch
  const size_t smp = sample_pass_bytes(N, C, 1);          // per-sample PSQ scratch
  if (grp > need) need = grp;
  if (smp > need) need = smp;
  if (bhq > need) need = bhq;
  if (list > need) need = list;
  return kGemmOffset + need;
}

size_t fqt_debug_workspace_size(int64_t M, int64_t N, int64_t K) {
  return debug_workspace_bytes(M, N, K);
}

fqt_status fqt_quantize_act(const void *X, fqt_dtype dtype, int64_t rows,
                            int64_t cols, int bits, fqt_qtensor *out,
                            void *workspace, size_t ws_bytes, void *stream) {
  return quantize_forward(X, dtype, rows, cols, bits, out, workspace, ws_bytes,
                          stream);
}

fqt_status fqt_quantize_weight(const void *W, fqt_dtype dtype, int64_t rows,
                               int64_t cols, int bits, fqt_qtensor *out,
                               void *workspace, size_t ws_bytes, void *stream) {
  return quantize_forward(W, dtype, rows, cols, bits, out, workspace, ws_bytes,
                          stream);
}

fqt_status fqt_quantize_grad_samples(const void *dH, fqt_dtype dtype, int64_t N, int64_t C,
                                     int64_t rows_per_sample, fqt_kind kind, int bits,
                                     uint64_t seed, fqt_qtensor *q_b2, fqt_qtensor *q_b1,
                                     void *workspace, size_t ws_bytes, void *stream) {
  if (N < 0 || C <= 0 || C > (1 << 20) || bits < 2 || bits > 8 || rows_per_sample < 1)
    return FQT_EINVAL;
  if (!q_b2 || (N > 0 && N % rows_per_sample)) return FQT_EINVAL;
  if (kind == FQT_PTQ) {  // one scale for the whole tensor: the per-tensor quantizer
    const fqt_status s = fqt_quantize_grad(dH, dtype, N, C, kind, bits, 0, seed, q_b2, q_b1,
                                           workspace, ws_bytes, stream);
    if (s == FQT_OK) q_b2->rows_per_sample = (int32_t)rows_per_sample;
    return s;
  }
  if (kind != FQT_PSQ) return kind == FQT_BHQ ? FQT_EUNSUPPORTED : FQT_EINVAL;
  if (N > 0 && (!dH || (!q_b2->codes && !q_b2->codes_f16) || !q_b2->inv_s || !q_b2->zero))
    return FQT_EINVAL;
  if (dtype != FQT_F32 && dtype != FQT_BF16) return FQT_EINVAL;
  if (N > 0 && q_b1 && ((!q_b1->codes && !q_b1->codes_f16) || !q_b1->inv_s || !q_b1->zero))
    return FQT_EINVAL;
  if (!(C == 64 || C == 128 || C == 256 || C == 512 || C == 1024 || C == 2048 ||
        C == 4096))
    return FQT_EUNSUPPORTED;
  if (N / rows_per_sample > ((int64_t)1 << 20) || rows_per_sample > (1 << 30))
    return FQT_EUNSUPPORTED;
  if (!aligned(dH, 16) || !aligned(q_b2->codes, 16) || !aligned(q_b2->codes_f16, 16) ||
      (q_b1 && (!aligned(q_b1->codes, 16) || !aligned(q_b1->codes_f16, 16))))
    return FQT_EINVAL;
  fqt_status s =
      check_ws(workspace, ws_bytes, kGemmOffset + sample_pass_bytes(N, C, rows_per_sample));
  if (s != FQT_OK) return s;
  q_b2->rows = N;
  q_b2->cols = C;
  q_b2->bits = bits;
  q_b2->kind = FQT_PSQ;
  q_b2->block = 0;
  q_b2->rows_per_sample = (int32_t)rows_per_sample;
  if (q_b1) {
    q_b1->rows = N;
    q_b1->cols = C;
    q_b1->bits = 8;
    q_b1->kind = FQT_PTQ;
    q_b1->block = 0;
    q_b1->rows_per_sample = 1;
  }
  if (N == 0) return FQT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char *w = static_cast<char *>(workspace);
  QuantArgs a;
  memset(&a, 0, sizeof(a));
  a.h = dH;
  a.N = N;
  a.C = (int)C;
  a.kind = FQT_PSQ;
  a.bits = bits;
  a.block = 1;
  a.key0 = (uint32_t)seed;
  a.key1 = (uint32_t)(seed >> 32);
  for (int r = 0; r < 10; ++r) {  // Philox4x32-10 round keys (Weyl sequence)
    a.round_keys[2 * r] = a.key0 + (uint32_t)r * 0x9E3779B9u;
    a.round_keys[2 * r + 1] = a.key1 + (uint32_t)r * 0xBB67AE85u;
  }
  a.c2 = q_b2->codes;
  a.f2 = q_b2->codes_f16;
  a.inv2 = q_b2->inv_s;
  a.zero2 = q_b2->zero;
  a.rsum2 = q_b2->row_sum;
  a.csum2 = q_b1 ? nullptr : q_b2->col_sum;
  if (q_b1) {
    a.c1 = q_b1->codes;
    a.f1 = q_b1->codes_f16;
    a.inv1 = q_b1->inv_s;
    a.zero1 = q_b1->zero;
    a.rsum1 = q_b1->row_sum;
    a.csum1 = q_b1->col_sum;
  }
  a.status = reinterpret_cast<int *>(w);
  return launch_sample_passes(a, dtype == FQT_BF16, rows_per_sample, device_sm_count(),
                              w + kGemmOffset, reinterpret_cast<float2 *>(w + kRangeOffset), st);
}

fqt_status fqt_quantize_grad(const void *dH, fqt_dtype dtype, int64_t N,
                             int64_t C, fqt_kind kind, int bits, int block,
                             uint64_t seed, fqt_qtensor *q_b2,
                             fqt_qtensor *q_b1, void *workspace,
                             size_t ws_bytes, void *stream) {
  if (N < 0 || C <= 0 || C > (1 << 20) || bits < 2 || bits > 8) return FQT_EINVAL;
  if (!q_b2) return FQT_EINVAL;
  // an empty batch has nothing to read or write (its tensors may be NULL)
  if (N > 0 && (!dH || (!q_b2->codes && !q_b2->codes_f16) || !q_b2->inv_s || !q_b2->zero))
    return FQT_EINVAL;
  if (dtype != FQT_F32 && dtype != FQT_BF16) return FQT_EINVAL;
  if (kind != FQT_PTQ && kind != FQT_PSQ && kind != FQT_BHQ && kind != FQT_SHIFT)
    return FQT_EINVAL;
  if (kind == FQT_SHIFT) {
    if (N > 0 && (!q_b2->shift_f16 || !q_b2->shift || !q_b2->shift_col_sum ||
                  !q_b2->shift_scale))
      return FQT_EINVAL;
    if (C % 8 || (C / 8 != 8 && C / 8 != 16 && C / 8 != 32 && C / 8 != 64 && C / 8 != 128))
      return FQT_EUNSUPPORTED;
    if (!aligned(q_b2->shift_f16, 16)) return FQT_EINVAL;
  }
  // BHQ block 0: the adaptive groups of App. D.5
  const bool adapt = kind == FQT_BHQ && block == 0;
  if (kind == FQT_BHQ) {
    if (block < 0 || block > 128 || (block & (block - 1))) return FQT_EINVAL;
    if (N > 0 && !adapt && !q_b2->lead) return FQT_EINVAL;
    if (N > 0 && adapt && (!q_b2->perm || !q_b2->gstart || !q_b2->gsize)) return FQT_EINVAL;
  } else {
    block = 0;
  }
  if (N > 0 && q_b1 && ((!q_b1->codes && !q_b1->codes_f16) || !q_b1->inv_s || !q_b1->zero))
    return FQT_EINVAL;
  // the grad_X offsets of BHQ (hz, hr) are reflected row sums: both or neither
  const bool want_off = kind == FQT_BHQ && block != 1 && (q_b2->hz || q_b2->hr);
  if (N > 0 && want_off && (!q_b2->hz || !q_b2->hr || !q_b2->row_sum)) return FQT_EINVAL;
  if (C % 8) return FQT_EUNSUPPORTED;
  if (!aligned(dH, 16) || !aligned(q_b2->codes, 16) || !aligned(q_b2->codes_f16, 16) ||
      (q_b1 && (!aligned(q_b1->codes, 16) || !aligned(q_b1->codes_f16, 16))))
    return FQT_EINVAL;
  if (adapt && (C != 64 && C != 128 && C != 256)) return FQT_EUNSUPPORTED;
  if (adapt && N > ((int64_t)1 << 20)) return FQT_EUNSUPPORTED;
  // fixed BHQ blocks of supported shapes: the two-pass quantizer, whose
  // statistics pass also takes the range (no separate range pass)
  const bool two_pass = kind == FQT_BHQ && !adapt &&
                        bhq_pass_supported((int)C, block, dtype == FQT_BF16);
  fqt_status s = check_ws(workspace, ws_bytes,
                          kGemmOffset + (adapt ? group_workspace_bytes(N)
                                         : two_pass ? bhq_pass_bytes(N, C) : 0));
  if (s != FQT_OK) return s;
  q_b2->rows = N;
  q_b2->cols = C;
  q_b2->bits = bits;
  q_b2->kind = kind;
  q_b2->block = block;
  q_b2->rows_per_sample = 1;
  if (q_b1) {
    q_b1->rows = N;
    q_b1->cols = C;
    q_b1->bits = 8;
    q_b1->kind = FQT_PTQ;
    q_b1->block = 0;
    q_b1->rows_per_sample = 1;
  }
  if (N == 0) return FQT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int nsm = device_sm_count();
  char *w = static_cast<char *>(workspace);
  float2 *part = reinterpret_cast<float2 *>(w + kRangeOffset);
  int npart = 0;
  int32_t *csum = q_b1 ? q_b1->col_sum : (adapt ? nullptr : q_b2->col_sum);
  // the column sums the quantizer accumulates into are cleared by the range pass
  int32_t *csum2 = kind == FQT_SHIFT ? q_b2->shift_col_sum : nullptr;
  cudaError_t e = cudaSuccess;
  if (!two_pass) {
    e = launch_range(dH, dtype == FQT_BF16, N * C, part, &npart, csum, csum ? C : 0, csum2,
                     csum2 ? C : 0, nsm, st);
    if (e != cudaSuccess) return cuda_fail(e, "range pass");
  }
  QuantArgs a;
  memset(&a, 0, sizeof(a));
  a.h = dH;
  a.N = N;
  a.C = (int)C;
  a.kind = (int)kind;
  a.bits = bits;
  a.block = block;
  a.key0 = (uint32_t)seed;
  a.key1 = (uint32_t)(seed >> 32);
  for (int r = 0; r < 10; ++r) {  // Philox4x32-10 round keys (Weyl sequence)
    a.round_keys[2 * r] = a.key0 + (uint32_t)r * 0x9E3779B9u;
    a.round_keys[2 * r + 1] = a.key1 + (uint32_t)r * 0xBB67AE85u;
  }
  a.c2 = q_b2->codes;
  a.f2 = q_b2->codes_f16;
  a.inv2 = q_b2->inv_s;
  a.zero2 = q_b2->zero;
  a.rsum2 = q_b2->row_sum;
  a.csum2 = q_b1 ? nullptr : q_b2->col_sum;
  a.lead2 = q_b2->lead;
  if (q_b1) {
    a.c1 = q_b1->codes;
    a.f1 = q_b1->codes_f16;
    a.inv1 = q_b1->inv_s;
    a.zero1 = q_b1->zero;
    a.rsum1 = q_b1->row_sum;
    a.csum1 = q_b1->col_sum;
  }
  a.part = part;
  a.npart = npart;
  a.status = reinterpret_cast<int *>(w);
  int nth, grid;
  size_t smem;
  const bool bf16 = dtype == FQT_BF16;
  if (kind == FQT_SHIFT) {
    QuantArgs as = a;
    as.fs = q_b2->shift_f16;
    as.shift = q_b2->shift;
    as.scs = q_b2->shift_col_sum;
    as.sscale = q_b2->shift_scale;
    as.csum2 = nullptr;
    return launch_shift(as, bf16, nsm, st);
  }
  if (adapt) {
    unsigned *slots = nullptr;
    s = launch_bhq_grouping(dH, bf16, N, (int)C, q_b2->perm, q_b2->gstart, q_b2->gsize,
                            w + kGemmOffset, ws_bytes - kGemmOffset, &slots, st);
    if (s != FQT_OK) return s;
    QuantArgs ag = a;
    ag.slots = slots;
    ag.perm = q_b2->perm;
    ag.gstart = q_b2->gstart;
    if (want_off) {
      ag.hz = q_b2->hz;
      ag.hr = q_b2->hr;
    }
    return launch_bhq_groups(ag, bf16, nsm, st);
  }
  if (two_pass) {
    QuantArgs aw = a;
    if (want_off) {
      aw.hz = q_b2->hz;
      aw.hr = q_b2->hr;
    }
    return launch_bhq_passes(aw, bf16, nsm, w + kGemmOffset, part, st);
  }
  {
    QuantArgs a2 = a;  // staged kernel for rows of up to 1024 columns
    if (quant2_geometry(a2, bf16, nsm, &grid, &smem) == FQT_OK) {
      e = launch_quant2(a2, bf16, grid, smem, st);
      if (e != cudaSuccess) return cuda_fail(e, "staged quantizer launch");
    } else {
      s = quant_geometry(a, nsm, &nth, &grid, &smem);
      if (s != FQT_OK) return s;
      e = launch_quant(a, bf16, nth, grid, smem, st);
      if (e != cudaSuccess) return cuda_fail(e, "quantizer launch");
    }
  }
  if (want_off) {
    e = launch_bhq_offsets(q_b2->zero, q_b2->row_sum, q_b2->lead, q_b2->hz, q_b2->hr, N,
                           (int)C, bits, block, st);
    if (e != cudaSuccess) return cuda_fail(e, "BHQ offsets launch");
  }
  return FQT_OK;
}

fqt_status fqt_linear_forward(const fqt_qtensor *qx, const fqt_qtensor *qw, float *H,
                              void *workspace, size_t ws_bytes, void *stream) {
  return linear_forward(qx, qw, H, workspace, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_linear_backward(const fqt_qtensor *q_b2, const fqt_qtensor *q_b1,
                               const fqt_qtensor *qx, const fqt_qtensor *qw,
                               float *grad_X, float *grad_W, void *workspace,
                               size_t ws_bytes, void *stream) {
  return linear_backward(q_b2, q_b1, qx, qw, grad_X, grad_W, workspace, ws_bytes,
                         reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_grad_w_fixed_scratch(const fqt_qtensor *q_b1, const fqt_qtensor *qx,
                                    float *grad_W, void *stream) {
  return grad_w_fixed_scratch(q_b1, qx, grad_W, reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_debug_int_gemm(const uint8_t *A, int a_kmajor, int a_bits,
                              const uint8_t *Bm, int b_kmajor, int b_bits,
                              int64_t M, int64_t N, int64_t K, int64_t *out,
                              void *workspace, size_t ws_bytes, void *stream) {
  return debug_int_gemm(A, a_kmajor, a_bits, Bm, b_kmajor, b_bits, M, N, K, out,
                        workspace, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_debug_int_gemm_u8(const uint8_t *A, int a_bits, const uint8_t *Bm, int b_bits,
                                 int64_t M, int64_t N, int64_t K, int64_t *out,
                                 void *workspace, size_t ws_bytes, void *stream) {
  return debug_int_gemm_u8(A, a_bits, Bm, b_bits, M, N, K, out, workspace, ws_bytes,
                           reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_sync_status(void *workspace, void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  if (!workspace) return FQT_EWORKSPACE;
  int code = 0;
  e = cudaMemcpy(&code, workspace, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "status read");
  if (code != 0) {
    e = cudaMemset(workspace, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "status clear");
  }
  return static_cast<fqt_status>(code);
}

fqt_status fqt_fixed_scratch_sync_status(void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  int *word = nullptr;
  const fqt_status s = fixed_scratch_status(&word);
  if (s != FQT_OK) return s;
  int code = 0;
  e = cudaMemcpy(&code, word, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "status read");
  if (code != 0) {
    e = cudaMemset(word, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "status clear");
  }
  return static_cast<fqt_status>(code);
}

fqt_status fqt_debug_wait_timeout(void *workspace, size_t ws_bytes, uint64_t limit_ns,
                                  void *stream) {
  return debug_wait_timeout(workspace, ws_bytes, limit_ns,
                            reinterpret_cast<cudaStream_t>(stream));
}

fqt_status fqt_debug_mma_peak(int kind, int64_t iters, double *ops_out, void *workspace,
                              size_t ws_bytes, void *stream) {
  return debug_mma_peak(kind, iters, ops_out, workspace, ws_bytes,
                        reinterpret_cast<cudaStream_t>(stream));
}

size_t fqt_conv_grad_x_workspace_size(int64_t cin) { return conv_grad_x_ws_bytes(cin); }

fqt_status fqt_conv_grad_x_nhwc(const fqt_qtensor *q_b2, const fqt_qtensor *qw, int64_t n,
                                int64_t h, int64_t w, int64_t cin, int k, int pad,
                                float *grad_X, void *workspace, size_t ws_bytes, void *stream) {
  return conv_grad_x_nhwc(q_b2, qw, n, h, w, cin, k, pad, grad_X, workspace, ws_bytes,
                          reinterpret_cast<cudaStream_t>(stream));
}

const char *fqt_last_cuda_error(void) { return g_last_error; }

const char *fqt_status_string(fqt_status status) {
  switch (status) {
    case FQT_OK: return "ok";
    case FQT_EINVAL: return "invalid argument";
    case FQT_EUNSUPPORTED: return "unsupported shape or option";
    case FQT_ECUDA: return "CUDA error";
    case FQT_ENONFINITE: return "non-finite input";
    case FQT_ETIMEOUT: return "device-side wait timed out";
    case FQT_EWORKSPACE: return "workspace missing, misaligned or too small";
  }
  return "unknown status";
}

}  // extern "C"
