/*
 * fqt.h -- C ABI of the GB300 library for the quantized backward pass of one
 * linear (or im2col-lowered conv) layer under fully quantized training (FQT),
 * "A Statistical Framework for Low-bitwidth Training of Deep Neural
 * Networks" (Chen, Gai, Yao, Mahoney, Gonzalez, NeurIPS 2020).
 *
 * Notation (PyTorch layout): dH is N x C (N samples / tokens / im2col rows,
 * C output features), X is N x D, W is C x D (out x in).  The paper's
 * Theta is W^T, so its grad_Theta = X~^T Q(dH) (Eq. 6) is the transpose of
 * grad_W returned here.  b = bits, B = 2^b - 1.
 *
 * Conventions for every entry point:
 *  - All tensor pointers are DEVICE pointers owned by the caller; the library
 *    allocates nothing.  `stream` is a cudaStream_t passed as void* (NULL =
 *    the legacy default stream).  Work is enqueued on `stream` and the call
 *    returns without synchronising.
 *  - Argument errors are returned synchronously and enqueue nothing.
 *    Conditions found on the device (non-finite input, a wait that ran out)
 *    are recorded in the status word at the start of the workspace and are
 *    returned by fqt_sync_status().
 *  - `workspace` is caller-owned device memory of at least
 *    fqt_workspace_size() bytes, 256-byte aligned and zero-filled before its
 *    first use.  Calls that share a workspace must be ordered (same stream
 *    or synchronised); concurrent calls need separate workspaces.
 *  - Outputs depend only on the inputs and the seed, not on the launch
 *    configuration.  Alignment: every pointer 16-byte aligned; quantizer
 *    inputs need cols % 8 == 0; GEMM operands need cols % 16 == 0.
 */
#ifndef FQT_H_
#define FQT_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define FQT_API __attribute__((visibility("default")))
#else
#define FQT_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FQT_OK = 0,
  FQT_EINVAL = 1,          /* bad argument: null pointer, size, bits, layout */
  FQT_EUNSUPPORTED = 2,    /* valid request this build does not implement */
  FQT_ECUDA = 3,           /* a CUDA runtime / driver call failed */
  FQT_ENONFINITE = 4,      /* input held NaN or Inf (device-side) */
  FQT_ETIMEOUT = 5,        /* a bounded device-side wait gave up */
  FQT_EWORKSPACE = 6       /* workspace missing, misaligned or too small */
} fqt_status;

typedef enum { FQT_PTQ = 0, FQT_PSQ = 1, FQT_BHQ = 2, FQT_SHIFT = 3 } fqt_kind;
typedef enum { FQT_F32 = 0, FQT_BF16 = 1 } fqt_dtype;

/*
 * A quantized matrix: the encoding of Eq. 9 (Sec. 4),
 *     value = S^-1 (codes + z' 1^T) = diag(inv_s) Q_blk (codes + z' 1^T),
 * with Q_blk = I for PTQ (Sec. 3.3) and PSQ (Sec. 4.1), and for BHQ
 * (Sec. 4.2) the block-diagonal Householder reflections
 * Q = I - 2 n n^T / ||n||^2, n = 1/sqrt(nb) 1 - e_p, one per block of
 * `block` consecutive rows (nb = rows of that block, p = its lead row), or,
 * with block 0, one per adaptive group of App. D.5 (rows reordered by
 * `perm`, each group's lead row first).
 *
 * The caller allocates every array (device memory) and sets the pointers;
 * the quantize calls fill rows, cols, bits, kind and block and write every
 * non-NULL output.  `codes` (1 byte per entry) and `codes_f16` (2 bytes, the
 * same integers centred and widened) are two encodings of one code matrix;
 * either may be NULL.
 */
typedef struct fqt_qtensor {
  int64_t rows, cols;
  int32_t bits;      /* b in [2, 8] */
  int32_t kind;      /* fqt_kind */
  int32_t block;     /* BHQ rows per block (power of two, <= 128); else 0 */
  int32_t rows_per_sample; /* written by the gradient quantizers: rows of dH
                        that form one sample (Sec. 4.1), 1 for fqt_quantize_grad,
                        R for fqt_quantize_grad_samples; 0 elsewhere */
  uint8_t *codes;    /* rows x cols, row-major, values in [0, 2^b - 1] */
  float *inv_s;      /* PTQ: 1 entry; PSQ, BHQ: rows entries (1/s_i; BHQ rows
                        of a block whose other rows are all zero hold 0) */
  float *zero;       /* same count: z' in the scaled / transformed domain */
  int32_t *row_sum;  /* rows entries: sum_j codes_ij, or NULL (not computed) */
  int32_t *col_sum;  /* cols entries: sum_i codes_ij, or NULL (not computed) */
  int32_t *lead;     /* BHQ: ceil(rows / block) entries, lead row offset p
                        within each block; else unused (may be NULL) */
  uint16_t *codes_f16; /* rows x cols, row-major: the centred code
                        code - 2^(b-1) as an IEEE fp16 bit pattern (exact),
                        the operand format of the tensor-core contractions;
                        NULL = not written.  Required by fqt_linear_backward. */
  float *hz;         /* BHQ: rows entries, (Q_blk d)_i, where the offset
                        2^(b-1) + zero_i = m_i + d_i with m_i = rint of its
                        fp32 sum and |d_i| <= 1/2; NULL = not written; else
                        unused.  With hr, required by fqt_linear_backward for
                        a BHQ q_b2 with block > 1. */
  float *hr;         /* BHQ: rows entries, (Q_blk R)_i with R_i = row_sum_i -
                        cols 2^(b-1) + cols m_i */
  int32_t *perm;     /* BHQ with block 0 (the adaptive groups of App. D.5):
                        rows entries, perm[k] = row of dH held by stored row
                        k; codes, inv_s, zero, row_sum, hz and hr are then in
                        this stored order.  Else unused (may be NULL). */
  int32_t *gstart;   /* BHQ block 0: rows + 1 entries, gstart[i] = first
                        stored row of group i (its lead row), rows for every
                        i >= G (the number of groups) */
  int32_t *gsize;    /* BHQ block 0: rows entries, size of the group of each
                        stored row */
  uint16_t *shift_f16; /* FQT_SHIFT: rows x cols, the codes on the common scale
                        of all rows, a = 2^(4 - shift_i) (code - 2^(b-1)), as
                        exact fp16 (|a| <= 16 (2^(b-1) - 1)): the grad_W
                        operand.  Else unused (may be NULL). */
  int32_t *shift;    /* FQT_SHIFT: rows entries, shift_i in [0, 4] */
  int32_t *shift_col_sum; /* FQT_SHIFT: cols entries, sum_i a_ic */
  float *shift_scale; /* FQT_SHIFT: 2 entries, the common scale 2^-4 / s of a
                        and 0 (its zero point) */
  int32_t conv[8];   /* written by fqt_quantize_act_conv: {n, h, w, c, kh, kw,
                        pad, 0}, the geometry of an implicit im2col operand;
                        all zero for an ordinary matrix (the other quantize
                        calls clear it) */
} fqt_qtensor;

/* Bytes of workspace a layer with dH N x C, X N x D, W C x D needs for any
 * call below (quantizers and backward). */
FQT_API size_t fqt_workspace_size(int64_t N, int64_t C, int64_t D);

/*
 * Deterministic 8-bit (or `bits`-bit) PTQ of a forward operand, the
 * activation quantizer Q_f of Eq. 3 and App. E: z = min X, s = B / R(X),
 * codes = round_half_even(s (X - z)) (Sec. 2.1).  X: rows x cols, row-major,
 * fp32 or bf16.  Fills out->codes, inv_s[0], zero[0] and, when non-NULL,
 * row_sum and col_sum.
 */
FQT_API fqt_status fqt_quantize_act(const void *X, fqt_dtype dtype, int64_t rows,
                            int64_t cols, int bits, fqt_qtensor *out,
                            void *workspace, size_t ws_bytes, void *stream);

/*
 * Q_f of a stride-1 convolution's input without forming its im2col matrix:
 * X is an NHWC tensor n x h x w x c (fp32 or bf16); the quantized operand is
 * the im2col matrix of kh x kw taps with `pad` zeros on every side
 * (rows = n oh ow output pixels, oh = h + 2 pad - kh + 1, ow likewise;
 * cols = kh kw c, tap-major then channel), exactly the codes that
 * fqt_quantize_act gives for that matrix: z = min and s = B / R over X and,
 * when pad > 0, the padding zeros (Sec. 2.1, App. E).  Storage is NHWC:
 * out->codes_f16 (n h w x c) holds code - 2^(b-1) as for any operand;
 * out->codes (optional) the codes; inv_s[0], zero[0];
 * out->col_sum (required, kh kw c + 1 entries) the column sums of the
 * im2col matrix followed by code(0.0); out->conv the geometry.  row_sum must
 * be NULL.  c % 8 == 0, c <= 4096.  The workspace holds the status word and range
 * partials only (fqt_workspace_size(n h w, c, 16) bytes suffice).
 * fqt_linear_backward reads such an operand as qx for grad_W (stride 1,
 * c % 64 == 0, pad <= 17, and ow <= 64 or ow % 32 == 0): rows of up to 64 output
 * pixels go to the split-K tile kernel in blocks of whole output rows,
 * wider rows to the one-range-per-CTA kernel.
 */
FQT_API fqt_status fqt_quantize_act_conv(const void *X, fqt_dtype dtype, int64_t n, int64_t h,
                                         int64_t w, int64_t c, int kh, int kw, int pad,
                                         int bits, fqt_qtensor *out, void *workspace,
                                         size_t ws_bytes, void *stream);

/* The same quantizer for the weight, Q_theta of Eq. 3 (W: C x D). */
FQT_API fqt_status fqt_quantize_weight(const void *W, fqt_dtype dtype, int64_t rows,
                               int64_t cols, int bits, fqt_qtensor *out,
                               void *workspace, size_t ws_bytes, void *stream);

/*
 * Gradient quantizers with unbiased stochastic rounding (Sec. 3.3, 4.1, 4.2,
 * 4.3) and the bifurcation of App. E:
 *   q_b2 <- Q_b2(dH): kind (PTQ, PSQ, BHQ), `bits`, BHQ `block`; feeds grad_X.
 *   q_b1 <- Q_b1(dH): 8-bit stochastic PTQ; feeds grad_W.  May be NULL.
 * SR draws 16-bit uniforms from Philox4x32-10 keyed by `seed`, counter
 * (flat_index / 8, stream, 0), stream 0 for q_b2 and 1 for q_b1.
 * dH: N x C row-major, fp32 or bf16, C % 8 == 0.  BHQ: block a power of
 * two <= 128 and block * C <= 65536; q_b2->hz and q_b2->hr are written when
 * non-NULL (row_sum must then be non-NULL too).
 * BHQ with block 0 takes the adaptive groups of App. D.5, as this library
 * reads it: rows sorted by M_i = ||dH_i||_inf (descending, ties by index);
 * for every group count G the estimate V(G) = sum_i (M_i^(2/3) s_i^(-1/3) +
 * M_(G+1)^(2/3) s_i^(2/3))^3 of App. D.4's bound with the paper's group
 * sizes s_i = (N - G) M_i / sum_(i<=G) M_i; G = argmin V (smallest on ties);
 * integer sizes by cumulative rounding of the s_i, small rows dealt from the
 * smallest up.  It writes q_b2->perm, gstart, gsize (required) and stores
 * the groups one after another, SR uniforms drawn by stored index.  Needs
 * C in {64, 128, 256}, N <= 2^20, and hz, hr, row_sum for the backward.
 * FQT_SHIFT is the per-sample power-of-two shift quantizer that Sec. 4.3
 * proposes for hardware, as this library reads it: one symmetric per-tensor
 * range [-M, M], M = max |dH|, s = (2^(b-1) - 1) / M; row i uses the scale
 * s 2^shift_i, shift_i the largest integer in [0, 4] with
 * 2^shift_i ||dH_i||_inf <= M, around the midpoint code 2^(b-1):
 * code = SR(s 2^shift_i dH_ij + 2^(b-1)); inv_s_i = 2^-shift_i / s,
 * zero_i = -2^(b-1).  It also writes shift, shift_f16, shift_col_sum and
 * shift_scale (required): grad_W then contracts the shifted integer codes
 * (the samples' accumulators shifted before the sum, Sec. 4.3), so q_b1 may
 * be NULL (no bifurcation).  Needs C in {64, 128, 256, 512, 1024}.
 */
FQT_API fqt_status fqt_quantize_grad(const void *dH, fqt_dtype dtype, int64_t N,
                             int64_t C, fqt_kind kind, int bits, int block,
                             uint64_t seed, fqt_qtensor *q_b2,
                             fqt_qtensor *q_b1, void *workspace,
                             size_t ws_bytes, void *stream);

/*
 * Q_b2 with per-image samples (Sec. 4.1: a sample is one input's gradient,
 * here `rows_per_sample` = R consecutive rows of dH, e.g. an image's H W
 * output pixels of a conv layer lowered to im2col, Sec. 2.1) and Q_b1 as in
 * fqt_quantize_grad.  PSQ: the scale and zero point of sample i come from
 * all R C entries of its rows, s_i = B / R(h_i), z_i = min h_i; codes are
 * SR(s_i (h - z_i)) with the uniforms of fqt_quantize_grad (the flat index
 * of dH).  inv_s and zero hold one entry per ROW (the sample's value
 * repeated), row_sum per row, so the result is an ordinary PSQ operand of
 * fqt_linear_backward, and q_b2->rows_per_sample = R.  PTQ is the
 * per-tensor quantizer.  BHQ returns FQT_EUNSUPPORTED (its reflection mixes
 * samples at every pixel, which neither contraction's epilogue forms).
 * Needs N % R == 0, C in {64, 128, 256, 512, 1024, 2048, 4096}, N / R <= 2^20.
 */
FQT_API fqt_status fqt_quantize_grad_samples(const void *dH, fqt_dtype dtype, int64_t N,
                                             int64_t C, int64_t rows_per_sample,
                                             fqt_kind kind, int bits, uint64_t seed,
                                             fqt_qtensor *q_b2, fqt_qtensor *q_b1,
                                             void *workspace, size_t ws_bytes, void *stream);

/*
 * The two low-bit contractions of Eq. 6 with App. E's bifurcation:
 *   grad_X = Q_b2(dH) W~          (N x D, fp32, row-major; may be NULL)
 *   grad_W = Q_b1(dH)^T X~        (C x D, fp32, row-major; may be NULL)
 * The integer products of the codes are exact; dequantization and, for BHQ,
 * the inverse Householder transform of each block are applied in the
 * epilogue.  Reads the operands' codes_f16 and needs q_b2->row_sum (or, for
 * BHQ with block > 1, q_b2->hz and q_b2->hr; for block 0 all three and perm,
 * gstart, gsize, in which case the inverse reflections of groups of two or
 * more rows run as a separate pass over their grad_X rows, and the product
 * must have the fp32-exact form: C 2^(bw + b - 2) < 2^24 and C at most one
 * exact chunk, else FQT_EUNSUPPORTED), qw->col_sum (grad_X) and
 * q_b1->col_sum, qx->col_sum (grad_W).  q_b1 may be
 * NULL when q_b2 is PTQ with col_sum set, or FQT_SHIFT: grad_W then uses
 * q_b2 (for FQT_SHIFT its shift_f16, shift_col_sum and shift_scale).
 * grad_W's two code sets may instead both be given as bytes only (codes set,
 * codes_f16 NULL; not the shift quantizer's, not an implicit im2col X~): the
 * split-K contraction then reads 1 byte per code and widens the codes to fp16
 * on chip, with the same exact integer products (and so the same grad_W, bit
 * for bit).  One set as bytes and the other as carriers is FQT_EINVAL.
 * C % 16 == 0 and D % 16 == 0.
 */
FQT_API fqt_status fqt_linear_backward(const fqt_qtensor *q_b2,
                               const fqt_qtensor *q_b1,
                               const fqt_qtensor *qx, const fqt_qtensor *qw,
                               float *grad_X, float *grad_W, void *workspace,
                               size_t ws_bytes, void *stream);

/*
 * grad_X of a stride-1 k x k convolution directly in NHWC (n x h x w x cin,
 * fp32): col2im of Q_b2(dH) W~ (Eq. 6 for a conv lowered to im2col rows,
 * Sec. 2.1) fused into the contraction, computed as the transposed
 * convolution dX[p] = sum over taps t of Q_b2(dH)[o(p, t)] W~[:, t, :]
 * (o(p, t) the output pixel tap t of input pixel p reads; taps reading
 * outside the image add nothing).  q_b2: the dH rows of the conv's output
 * pixels (n h w x cout, row order (n, y, x)), PTQ (fqt_quantize_grad) or PSQ
 * with one sample per image (fqt_quantize_grad_samples with rows_per_sample
 * = h w): the scale must be the same for all pixels of an image so that it
 * factors out of the sum over taps.  codes_f16, row_sum, inv_s, zero.
 * qw: W~ from fqt_quantize_weight on the im2col weight cout x (k k cin)
 * (columns (ky, kx, c_in)), codes_f16 and col_sum.  Needs k = 3, pad = 1,
 * h, w >= 2, w <= 128, cin % 32 == 0, cout % 64 == 0 and one exact chunk
 * (9 cout <= 2^(26 - b - bw)); else FQT_EUNSUPPORTED.  `workspace`: at least
 * fqt_conv_grad_x_workspace_size(cin) bytes (status word and tables).
 */
FQT_API size_t fqt_conv_grad_x_workspace_size(int64_t cin);
FQT_API fqt_status fqt_conv_grad_x_nhwc(const fqt_qtensor *q_b2, const fqt_qtensor *qw,
                                        int64_t n, int64_t h, int64_t w, int64_t cin, int k,
                                        int pad, float *grad_X, void *workspace,
                                        size_t ws_bytes, void *stream);

/*
 * The quantized forward of the layer (Sec. 2.1, Eq. 3): H = X~ W~^T, the
 * product of the dequantized 8-bit PTQ operands, N x C fp32 row-major.  The
 * integer product of the codes is exact (fp16 carriers on the tensor cores,
 * as for the backward); dequantization is applied in the epilogue.  Needs
 * qx and qw from fqt_quantize_act / fqt_quantize_weight with codes_f16 and
 * row_sum set (rows of X: N x D, rows of W: C x D).  D % 16 == 0 and
 * C % 16 == 0.  `workspace` holds the status word only.
 */
FQT_API fqt_status fqt_linear_forward(const fqt_qtensor *qx, const fqt_qtensor *qw,
                                      float *H, void *workspace, size_t ws_bytes,
                                      void *stream);

/*
 * grad_W = Q_b1(dH)^T X~ exactly as fqt_linear_backward computes it, for
 * callers that cannot allocate device memory when they need the backward --
 * a loop whose memory budget is frozen after warm-up, or a C host with no
 * allocator of its own that must not call cudaMalloc (which may synchronise
 * the device).  It takes no workspace: the split-K partials live in a fixed
 * 8 MiB array inside the library, which every GPU that loads the library
 * keeps until the process exits.  The paper has no counterpart; this is a
 * deployment convenience.
 *  - Limit: C * D * 4 bytes of partials per split must fit 8 MiB with few
 *    enough splits to keep each below 2^31 / 2^(b1 + bx - 2) rows; larger
 *    problems return FQT_EWORKSPACE without launching anything.
 *  - The first call on a device looks up the array's device address (a
 *    runtime call with that device current); make that first call before any
 *    stream capture.
 *  - All calls on a device share the array and it keeps the last call's
 *    contents, so calls that overlap on the GPU (other streams, other host
 *    threads) race and give wrong results: order them.
 *  - Device-side conditions (a bounded wait that ran out) are recorded in
 *    the array's status word and returned by fqt_fixed_scratch_sync_status.
 * Operands as for fqt_linear_backward (codes_f16, col_sum, PTQ), but plain
 * matrices only: an implicit im2col operand (from fqt_quantize_act_conv,
 * conv[0] > 0) returns FQT_EUNSUPPORTED before anything is enqueued.
 */
FQT_API fqt_status fqt_grad_w_fixed_scratch(const fqt_qtensor *q_b1,
                                            const fqt_qtensor *qx, float *grad_W,
                                            void *stream);

/* Synchronises `stream`, returns the first device-side condition recorded by
 * fqt_grad_w_fixed_scratch calls on the current device since the previous
 * call of this function (or FQT_OK) and clears it.  Allocates nothing; like
 * the first fqt_grad_w_fixed_scratch call it looks up the array's address
 * once per device.  Has no counterpart in the paper. */
FQT_API fqt_status fqt_fixed_scratch_sync_status(void *stream);

/* Synchronises `stream`, returns the first device-side condition recorded in
 * `workspace` since the previous call (or FQT_OK) and clears it. */
FQT_API fqt_status fqt_sync_status(void *workspace, void *stream);

/* Exact integer contraction, for bit-exact tests of the GEMM core:
 *   out_ij = sum_k (A_ik - 2^(a_bits-1)) (B_kj - 2^(b_bits-1))   (int64)
 * A is M x K, stored row-major (a_kmajor = 1) or as its K x M transpose;
 * B is K x N, stored as K x N row-major (b_kmajor = 0) or as N x K; both
 * u8 codes.  The stored row pitch must be a multiple of 8 and N % 4 == 0.
 * The workspace must hold fqt_debug_workspace_size(M, N, K) bytes. */
FQT_API size_t fqt_debug_workspace_size(int64_t M, int64_t N, int64_t K);

/* The same exact contraction with both operands given as MN-major byte codes
 * (A stored K x M, B stored K x N, 16-byte aligned, M % 16 == 0, N % 16 == 0),
 * read as bytes and widened to fp16 carriers on chip: the path
 * fqt_linear_backward's grad_W takes when both of its code sets are given as
 * bytes only.  Workspace as for fqt_debug_int_gemm. */
FQT_API fqt_status fqt_debug_int_gemm_u8(const uint8_t *A, int a_bits, const uint8_t *Bm,
                                         int b_bits, int64_t M, int64_t N, int64_t K,
                                         int64_t *out, void *workspace, size_t ws_bytes,
                                         void *stream);

FQT_API fqt_status fqt_debug_int_gemm(const uint8_t *A, int a_kmajor, int a_bits,
                              const uint8_t *Bm, int b_kmajor, int b_bits,
                              int64_t M, int64_t N, int64_t K, int64_t *out,
                              void *workspace, size_t ws_bytes, void *stream);

/* Check of the device-side timeout path: one thread waits on an mbarrier
 * that nothing arrives at, with the bounded wait the contraction kernels
 * use, here bounded by limit_ns (at most 10 s, else FQT_EINVAL) instead of
 * their 2 s.  When it runs out the kernel records FQT_ETIMEOUT and returns.
 * The condition goes to `workspace` (then read by fqt_sync_status; at least
 * 256 bytes, 256-byte aligned) or, with workspace NULL, to the fixed array
 * of fqt_grad_w_fixed_scratch (read by fqt_fixed_scratch_sync_status).
 * No bulk copy or tensor-core operation is in flight during the wait.  Has
 * no counterpart in the paper. */
FQT_API fqt_status fqt_debug_wait_timeout(void *workspace, size_t ws_bytes,
                                          uint64_t limit_ns, void *stream);

/* Dense tensor-core rate kernels, the denominators of the contractions'
 * rooflines: kind 0 tcgen05 kind::f16 (fp16 x fp16 -> fp32, the operand
 * format of this library's contractions), kind 1 tcgen05 kind::f8f6f4 (e4m3
 * x e4m3 -> fp32), kind 2 warp-level mma.sync m16n8k32 u8 x s8 -> s32.
 * (tcgen05 kind::i8 does not assemble for sm_103a.)  Enqueues one launch on
 * `stream` that runs `iters` rounds of back-to-back MMAs on zero operands
 * on every SM and sets *ops_out (host memory) to the multiply-add
 * operations it performs (2 per multiply-add); the caller times the launch.
 * The workspace holds the status word (at least 256 bytes, 256-byte
 * aligned).  Has no counterpart in the paper. */
FQT_API fqt_status fqt_debug_mma_peak(int kind, int64_t iters, double *ops_out,
                                      void *workspace, size_t ws_bytes, void *stream);

/* Static description of a status code. */
FQT_API const char *fqt_status_string(fqt_status status);

/* After a call of this thread returned FQT_ECUDA: the name of the CUDA error
 * behind it and the step that raised it (static storage, per thread);
 * "none" otherwise.  Has no counterpart in the paper. */
FQT_API const char *fqt_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* FQT_H_ */
