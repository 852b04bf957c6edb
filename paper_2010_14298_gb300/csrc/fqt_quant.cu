// fqt_quant.cu -- quantizer kernels of the GB300 FQT library.
//
//  k_range  : per-CTA (min, max) of a tensor and a non-finite flag (the
//             dynamic range R(X) = max X - min X of Sec. 3.3); also clears
//             the column-sum outputs the quantizer accumulates into.
//  k_quant  : one templated kernel for
//             KIND_PTQ  per-tensor stochastic quantizer (Sec. 3.3),
//             KIND_PSQ  per-sample quantizer (Sec. 4.1),
//             KIND_BHQ  block Householder quantizer (Sec. 4.2, App. D.4),
//             KIND_DET  deterministic PTQ of the forward operands (Sec. 2.1),
//             fused with the 8-bit stochastic PTQ Q_b1 of App. E.
//
// Thread mapping.  A row (sample) is handled by a team of TW consecutive
// threads; each thread owns OPT "octs" (8 consecutive columns) of the row,
// octs cl, cl + TW, ...  Rows of a unit are spread over RL row lanes, RPL
// rows per lane.  For BHQ a unit is one block of `block` rows and a CTA runs
// G such groups side by side.  Row reductions use shuffles inside the team
// (TW <= 32) or shared memory (TW > 32); the BHQ column sums go through
// shared memory in a fixed order.  When the row does not fit the registers
// (nchunk > 1, only BHQ with long rows) every pass re-reads its chunk.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <math.h>
#include <algorithm>

#include "fqt_common.cuh"
#include "fqt_internal.h"

namespace fqt {

constexpr int kMaxOct = 4;  // octs a thread keeps in registers per pass

// ---------------------------------------------------------------------------
// Range pass
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_range(const T *__restrict__ x,
                                               int64_t n_oct, float2 *part,
                                               int32_t *z0, int64_t nz0,
                                               int32_t *z1, int64_t nz1) {
  float mn = INFINITY, mx = -INFINITY;
  int bad = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; o + 3 * stride < n_oct; o += 4 * stride) {
    float v[4][8];
#pragma unroll
    for (int u = 0; u < 4; ++u) load_oct(x + (o + u * stride) * 8, v[u]);
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        bad |= !isfinite(v[u][i]);
        mn = fminf(mn, v[u][i]);
        mx = fmaxf(mx, v[u][i]);
      }
  }
  for (; o < n_oct; o += stride) {
    float v[8];
    load_oct(x + o * 8, v);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      bad |= !isfinite(v[i]);
      mn = fminf(mn, v[i]);
      mx = fmaxf(mx, v[i]);
    }
  }
  const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (int64_t i = g; i < nz0; i += stride) z0[i] = 0;
  for (int64_t i = g; i < nz1; i += stride) z1[i] = 0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  __shared__ float smn[8], smx[8];
  __shared__ int sbad[8];
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    smn[w] = mn;
    smx[w] = mx;
    sbad[w] = bad;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < (int)(blockDim.x >> 5); ++i) {
      mn = fminf(mn, smn[i]);
      mx = fmaxf(mx, smx[i]);
      bad |= sbad[i];
    }
    part[blockIdx.x] = bad ? make_float2(NAN, NAN) : make_float2(mn, mx);
  }
}

// ---------------------------------------------------------------------------
// Team reductions (a team = TW consecutive threads owning one row)
// ---------------------------------------------------------------------------
struct OpMinMax {
  __device__ float2 operator()(float2 a, float2 b) const {
    return make_float2(fminf(a.x, b.x), fmaxf(a.y, b.y));
  }
};
struct OpMin {
  __device__ float operator()(float a, float b) const { return fminf(a, b); }
};
struct OpAdd {
  __device__ int operator()(int a, int b) const { return a + b; }
};
struct OpAddF {
  __device__ float operator()(float a, float b) const { return a + b; }
};
struct OpMaxF {
  __device__ float operator()(float a, float b) const { return fmaxf(a, b); }
};

__device__ __forceinline__ float shfl_x(float v, int off) {
  return __shfl_xor_sync(0xffffffffu, v, off);
}
__device__ __forceinline__ int shfl_x(int v, int off) {
  return __shfl_xor_sync(0xffffffffu, v, off);
}
__device__ __forceinline__ float2 shfl_x(float2 v, int off) {
  return make_float2(__shfl_xor_sync(0xffffffffu, v.x, off),
                     __shfl_xor_sync(0xffffffffu, v.y, off));
}

// Reduces v over the TW lanes of each team; every lane of the team receives
// the result.  Must be reached by the whole CTA (barriers when TW > 32);
// `red` holds 32 entries of V.
template <class V, class Op>
__device__ __forceinline__ V team_reduce(V v, int TW, V *red, Op op) {
  if (TW <= 32) {
    for (int off = TW >> 1; off > 0; off >>= 1) v = op(v, shfl_x(v, off));
    return v;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = op(v, shfl_x(v, off));
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[warp] = v;
  __syncthreads();
  const int w0 = (threadIdx.x / TW) * (TW >> 5);
  V acc = red[w0];
  for (int w = 1; w < (TW >> 5); ++w) acc = op(acc, red[w0 + w]);
  __syncthreads();
  return acc;
}

// ---------------------------------------------------------------------------
// The quantizer kernel
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ const T *row_ptr(const void *h, int64_t row, int C) {
  return reinterpret_cast<const T *>(h) + row * (int64_t)C;
}

template <int KIND, typename T, int NTMAX>
__global__ void __launch_bounds__(NTMAX) k_quant(const QuantArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  // with 1024 threads the register file allows no per-thread column sums
  constexpr bool kRegColSums = NTMAX <= 256;
  const int nth = blockDim.x, tid = threadIdx.x;
  const int grp = tid / a.GT, gt = tid - grp * a.GT;
  const int rl = gt / a.TW, cl = gt - rl * a.TW;
  const int TW = a.TW, OPT = a.OPT, RL = a.RL, C = a.C, CO = a.CO;
  const int chunk_octs = TW * OPT;
  const int chunk_cols = chunk_octs * 8;

  // shared memory carve-up (sizes computed by quant_smem_bytes on the host)
  float2 *red2 = reinterpret_cast<float2 *>(smem);    // 32
  float *redf = reinterpret_cast<float *>(red2 + 32);  // 32
  int *redi = reinterpret_cast<int *>(redf + 32);      // 32
  int *csum_s = redi + 32;                             // C
  float *bpar = reinterpret_cast<float *>(csum_s + C);  // G * 8
  float2 *rowst = reinterpret_cast<float2 *>(bpar + 8 * a.G);  // G * block
  float *wcol = reinterpret_cast<float *>(rowst + a.G * a.block);  // G * C
  float *colp = wcol + a.G * C;  // G * RL * chunk_cols

  // ---- global range from the range-pass partials ----
  float gmin = INFINITY, gmax = -INFINITY;
  int bad = 0;
  for (int i = tid; i < a.npart; i += nth) {
    const float2 p = a.part[i];
    bad |= isnan(p.x);
    gmin = fminf(gmin, p.x);
    gmax = fmaxf(gmax, p.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if ((tid & 31) == 0) {
    red2[tid >> 5] = make_float2(gmin, gmax);
    redi[tid >> 5] = bad;
  }
  for (int i = tid; i < C; i += nth) csum_s[i] = 0;
  __syncthreads();
  gmin = red2[0].x;
  gmax = red2[0].y;
  bad = redi[0];
  for (int w = 1; w < (nth >> 5); ++w) {
    gmin = fminf(gmin, red2[w].x);
    gmax = fmaxf(gmax, red2[w].y);
    bad |= redi[w];
  }
  __syncthreads();
  if (bad) {
    if (blockIdx.x == 0 && tid == 0) record_status(a.status, FQT_ENONFINITE);
    return;
  }
  const uint32_t B2 = (1u << a.bits) - 1u;
  const float s_g2 = affine_scale(gmin, gmax, B2);    // PTQ / DET scale
  const float s_g1 = affine_scale(gmin, gmax, 255u);  // Q_b1 scale
  const float s_g1_16 = __fmul_rn(s_g1, 65536.0f);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  if (blockIdx.x == 0 && tid == 0) {
    if (KIND == KIND_PTQ || KIND == KIND_DET) {
      a.inv2[0] = __fdiv_rn(1.0f, s_g2);
      a.zero2[0] = __fmul_rn(s_g2, gmin);
    }
    if (has_b1) {
      a.inv1[0] = __fdiv_rn(1.0f, s_g1);
      a.zero1[0] = __fmul_rn(s_g1, gmin);
    }
  }
  // column sums of the code set that feeds grad_W (Q_b1 when present)
  int32_t *const csum_g = has_b1 ? a.csum1 : a.csum2;
  const bool want_cs = csum_g != nullptr;
  const bool reg_cs = kRegColSums && a.nchunk == 1;
  int cs[kMaxOct][8];
#pragma unroll
  for (int k = 0; k < kMaxOct; ++k)
#pragma unroll
    for (int j = 0; j < 8; ++j) cs[k][j] = 0;

  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];
  float x[kMaxOct][8];

  for (int64_t ub = (int64_t)blockIdx.x * a.G; ub < a.n_units;
       ub += (int64_t)gridDim.x * a.G) {
    const int64_t u = ub + grp;
    const bool uvalid = u < a.n_units;
    const int64_t r0 = u * a.unit_rows;
    const int nrows = uvalid ? (int)min((int64_t)a.unit_rows, a.N - r0) : 0;
    const bool rvalid = rl < nrows;
    const int64_t row = r0 + rl;

    auto oct_of = [&](int ch, int k) { return ch * chunk_octs + cl + TW * k; };
    auto oct_ok = [&](int ch, int k) {
      return k < OPT && rvalid && oct_of(ch, k) < CO;
    };
    auto load_chunk = [&](int ch) {
#pragma unroll
      for (int k = 0; k < kMaxOct; ++k) {
        if (oct_ok(ch, k)) {
          load_oct(row_ptr<T>(a.h, row, C) + oct_of(ch, k) * 8, x[k]);
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) x[k][j] = 0.0f;
        }
      }
    };

    // ---------------- per-row statistics (PSQ, BHQ) ----------------
    float2 st = make_float2(INFINITY, -INFINITY);
    if (KIND == KIND_PSQ || KIND == KIND_BHQ) {
      for (int ch = 0; ch < a.nchunk; ++ch) {
        load_chunk(ch);
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          if (oct_ok(ch, k)) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              st.x = fminf(st.x, x[k][j]);
              st.y = fmaxf(st.y, x[k][j]);
            }
          }
        }
      }
      st = team_reduce(st, TW, red2, OpMinMax());
    }

    // ---------------- BHQ: block scalars, Householder, row minima ----------
    float s_row = 0.0f, c_row = 0.0f;
    if (KIND == KIND_BHQ) {
      if (cl == 0 && rvalid) rowst[grp * a.block + rl] = st;
      __syncthreads();
      if (gt == 0 && uvalid) {
        const float2 *rs = rowst + grp * a.block;
        int p = 0;
        float np = -1.0f;
        for (int k = 0; k < nrows; ++k) {  // lead row: largest ||h_k||_inf
          const float nk = fmaxf(fabsf(rs[k].x), fabsf(rs[k].y));
          if (nk > np) { np = nk; p = k; }
        }
        float lam2 = 0.0f;
        for (int k = 0; k < nrows; ++k)
          if (k != p) lam2 = fmaxf(lam2, fmaxf(fabsf(rs[k].x), fabsf(rs[k].y)));
        lam2 = 2.0f * lam2;
        float s1f = 0.0f, s2f = 0.0f, rho = 0.0f, kap = 0.0f;
        if (np > 0.0f) {
          float lam1 = __fsub_rn(rs[p].y, rs[p].x);
          if (!(lam1 > 0.0f)) lam1 = 2.0f * np;
          const double Nd = (double)nrows;
          double s1, s2 = 0.0;
          if (lam2 > 0.0f) {  // s1, s2 of App. D.4
            const double c1 = cbrt((double)lam1), c2 = cbrt((double)lam2);
            const double den = c1 * c1 * pow(Nd, -1.0 / 3.0) +
                               c2 * c2 * pow(Nd, 2.0 / 3.0);
            s1 = (double)B2 * pow(Nd, 1.0 / 6.0) / (c1 * den);
            s2 = (double)B2 * pow(Nd, 1.0 / 6.0) / (c2 * den);
          } else {  // limit lambda2 -> 0: the other rows are zero
            s1 = (double)B2 * sqrt(Nd) / (double)lam1;
          }
          s1f = (float)s1;
          s2f = lam2 > 0.0f ? (float)s2 : 0.0f;
          if (nrows > 1) {
            const double r = 1.0 / sqrt(Nd);
            rho = (float)r;
            kap = (float)(1.0 / (1.0 - r));
          }
        }
        float *bp = bpar + grp * 8;
        bp[0] = s1f;
        bp[1] = s2f;
        bp[2] = rho;
        bp[3] = kap;
        bp[4] = __int_as_float(p);
        a.lead2[u] = p;
      }
      __syncthreads();
      const float *bp = bpar + grp * 8;
      const int p = __float_as_int(bp[4]);
      const bool lead = rl == p;
      s_row = lead ? bp[0] : bp[1];
      c_row = lead ? bp[2] - 1.0f : bp[2];  // rho - delta_kp
      const float e_row = bp[3] * c_row;    // (rho - delta_kp) / (1 - rho)
      // w_j = sum_k e_k s_k h_kj, so that (Q g)_k = g_k - c_k w (g = s h)
      float *cp = colp + grp * RL * chunk_cols;
      float *wc = wcol + grp * C;
      float tmin = INFINITY;
      for (int ch = 0; ch < a.nchunk; ++ch) {
        if (a.nchunk > 1) load_chunk(ch);
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          if (k < OPT) {
            float *dst = cp + rl * chunk_cols + (cl + TW * k) * 8;
#pragma unroll
            for (int j = 0; j < 8; ++j)
              dst[j] = __fmul_rn(e_row, __fmul_rn(s_row, x[k][j]));
          }
        }
        __syncthreads();
        for (int c = gt; c < chunk_cols; c += a.GT) {
          const int col = ch * chunk_cols + c;
          if (col < C) {
            float acc = 0.0f;
            for (int r = 0; r < RL; ++r) acc += cp[r * chunk_cols + c];
            wc[col] = acc;
          }
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          if (oct_ok(ch, k)) {
            const int col0 = oct_of(ch, k) * 8;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float t = fmaf(-c_row, wc[col0 + j], __fmul_rn(s_row, x[k][j]));
              tmin = fminf(tmin, t);
            }
          }
        }
      }
      st.x = team_reduce(tmin, TW, redf, OpMin());  // z'_k
    }

    // ---------------- scale of this thread's row ----------------
    float s2, z2;
    if (KIND == KIND_PSQ) {
      s2 = affine_scale(st.x, st.y, B2);
      z2 = st.x;
    } else if (KIND == KIND_BHQ) {
      s2 = s_row;
      z2 = st.x;
    } else {
      s2 = s_g2;
      z2 = gmin;
    }

    // ---------------- rounding, packing, sums ----------------
    int rs2 = 0, rs1 = 0;
    for (int ch = 0; ch < a.nchunk; ++ch) {
      if (a.nchunk > 1 || KIND == KIND_PTQ || KIND == KIND_DET) load_chunk(ch);
#pragma unroll
      for (int k = 0; k < kMaxOct; ++k) {
        if (!oct_ok(ch, k)) continue;
        const int o = oct_of(ch, k);
        const uint64_t q = (uint64_t)row * (uint64_t)CO + (uint64_t)o;
        uint32_t c[8];
        if (KIND == KIND_DET) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float v = __fmul_rn(__fsub_rn(x[k][j], z2), s2);
            const int r = __float2int_rn(v);
            c[j] = (uint32_t)min(max(r, 0), (int)B2);
          }
        } else {
          const uint4 w = philox_oct(q, 0u, key);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float v;
            if (KIND == KIND_BHQ) {
              const float t = fmaf(-c_row, wcol[grp * C + o * 8 + j],
                                   __fmul_rn(s_row, x[k][j]));
              v = __fsub_rn(t, z2);
            } else {
              v = __fmul_rn(__fsub_rn(x[k][j], z2), s2);
            }
            c[j] = sr_code(v, u16_of(w, j), B2);
          }
        }
        if (a.c2) store_codes8(a.c2 + row * (int64_t)C + o * 8, c);
        if (a.f2) store_carriers8(a.f2 + row * (int64_t)C + o * 8, c, (B2 + 1u) >> 1);
#pragma unroll
        for (int j = 0; j < 8; ++j) rs2 += (int)c[j];
        const uint32_t *sumc = c;
        uint32_t d[8];
        if (has_b1) {
          const uint4 w = philox_oct(q, 1u, key);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float v = __fmul_rn(__fsub_rn(x[k][j], gmin), s_g1);
            d[j] = sr_code(v, u16_of(w, j), 255u);
            rs1 += (int)d[j];
          }
          if (a.c1) store_codes8(a.c1 + row * (int64_t)C + o * 8, d);
          if (a.f1) store_carriers8(a.f1 + row * (int64_t)C + o * 8, d, 128u);
          sumc = d;
        }
        if (want_cs) {
          if (reg_cs) {
#pragma unroll
            for (int j = 0; j < 8; ++j) cs[k][j] += (int)sumc[j];
          } else {
#pragma unroll
            for (int j = 0; j < 8; ++j)
              if (sumc[j]) atomicAdd(&csum_s[o * 8 + j], (int)sumc[j]);
          }
        }
      }
    }

    // ---------------- row metadata ----------------
    if (a.rsum2) rs2 = team_reduce(rs2, TW, redi, OpAdd());
    if (has_b1 && a.rsum1) rs1 = team_reduce(rs1, TW, redi, OpAdd());
    if (cl == 0 && rvalid) {
      if (a.rsum2) a.rsum2[row] = rs2;
      if (has_b1 && a.rsum1) a.rsum1[row] = rs1;
      if (KIND == KIND_PSQ) {
        a.inv2[row] = __fdiv_rn(1.0f, s2);
        a.zero2[row] = __fmul_rn(s2, z2);
      } else if (KIND == KIND_BHQ) {
        a.inv2[row] = s2 > 0.0f ? __fdiv_rn(1.0f, s2) : 0.0f;
        a.zero2[row] = z2;
      }
    }
    if (KIND == KIND_BHQ) __syncthreads();  // bpar / wcol / colp are reused
  }

  // ---------------- column sums ----------------
  if (want_cs) {
    if (reg_cs) {
#pragma unroll
      for (int k = 0; k < kMaxOct; ++k) {
        const int o = cl + TW * k;
        if (k < OPT && o < CO) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (cs[k][j]) atomicAdd(&csum_s[o * 8 + j], cs[k][j]);
        }
      }
    }
    __syncthreads();
    for (int i = tid; i < C; i += nth)
      if (csum_s[i]) atomicAdd(&csum_g[i], csum_s[i]);
  }
}

// ---------------------------------------------------------------------------
// Staged quantizer (rows of up to 1024 columns).
//
// Units of consecutive rows are copied into shared memory with one
// cp.async.bulk each (double-buffered: the next unit streams in while the
// current one is processed).  Row work uses "row segments": LPR lanes of a
// warp own one row, each lane OPL octs of it, so row reductions are short
// shuffle trees and every shared-memory read of a warp is contiguous.  The
// BHQ column sums of the Householder reflection (w_j = sum_k e_k s_k h_kj)
// run one thread per (block, column) over the staged block.
// ---------------------------------------------------------------------------
constexpr int kQ2Threads = 256;

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src,
                                         uint32_t bytes, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

template <typename T>
__device__ __forceinline__ void load_oct_smem(const unsigned char *row, int o,
                                              int lane, float (&x)[8]);

template <>
__device__ __forceinline__ void load_oct_smem<float>(const unsigned char *row,
                                                     int o, int lane,
                                                     float (&x)[8]) {
  // two 16-byte halves; lanes 4..7 of each quarter warp start with the
  // second half so that a quarter warp touches every bank once
  const int h0 = (lane >> 2) & 1;
  const float4 a = *reinterpret_cast<const float4 *>(row + o * 32 + h0 * 16);
  const float4 b = *reinterpret_cast<const float4 *>(row + o * 32 + (h0 ^ 1) * 16);
  const float4 lo = h0 ? b : a, hi = h0 ? a : b;
  x[0] = lo.x; x[1] = lo.y; x[2] = lo.z; x[3] = lo.w;
  x[4] = hi.x; x[5] = hi.y; x[6] = hi.z; x[7] = hi.w;
}

template <>
__device__ __forceinline__ void load_oct_smem<__nv_bfloat16>(
    const unsigned char *row, int o, int lane, float (&x)[8]) {
  const uint4 v = *reinterpret_cast<const uint4 *>(row + o * 16);
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

template <typename T>
__device__ __forceinline__ float elem_smem(const unsigned char *base, int64_t idx) {
  if (sizeof(T) == 4) return reinterpret_cast<const float *>(base)[idx];
  const uint16_t b = reinterpret_cast<const uint16_t *>(base)[idx];
  return __uint_as_float((uint32_t)b << 16);
}

// Reduction over the LPR lanes of a row segment (LPR a power of two <= 32).
template <class V, class Op>
__device__ __forceinline__ V seg_reduce(V v, int LPR, Op op) {
  for (int off = LPR >> 1; off > 0; off >>= 1) v = op(v, shfl_x(v, off));
  return v;
}

template <int KIND, typename T>
__global__ void __launch_bounds__(kQ2Threads) k_quant2(const QuantArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int C = a.C, CO = a.CO;
  const int LPR = a.TW, OPL = a.OPT, R = a.RL;  // lanes per row, octs per lane, rows per warp step
  const int U = a.unit_rows, nb = a.block > 0 ? a.block : 1;
  const int G = a.G;  // BHQ blocks per unit
  const int seg = lane / LPR, sl = lane - seg * LPR;
  const int row_bytes = C * (int)sizeof(T);
  const size_t stage_bytes = (size_t)a.stage_bytes;

  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + 2 * stage_bytes);
  float2 *red = reinterpret_cast<float2 *>(bar + 2);              // 8
  int *redi = reinterpret_cast<int *>(red + 8);                   // 8
  int *csum_s = redi + 8;                                          // C
  float2 *rowst = reinterpret_cast<float2 *>(csum_s + C);         // U
  float *bpar = reinterpret_cast<float *>(rowst + U);             // G * 8
  float *wcol = bpar + 8 * G;                                      // G * C

  // ---- global range from the range-pass partials ----
  float gmin = INFINITY, gmax = -INFINITY;
  int bad = 0;
  for (int i = tid; i < a.npart; i += kQ2Threads) {
    const float2 p = a.part[i];
    bad |= isnan(p.x);
    gmin = fminf(gmin, p.x);
    gmax = fmaxf(gmax, p.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(gmin, gmax);
    redi[warp] = bad;
  }
  for (int i = tid; i < C; i += kQ2Threads) csum_s[i] = 0;
  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_barrier_init();
  }
  __syncthreads();
  gmin = red[0].x;
  gmax = red[0].y;
  bad = redi[0];
  for (int w = 1; w < kQ2Threads / 32; ++w) {
    gmin = fminf(gmin, red[w].x);
    gmax = fmaxf(gmax, red[w].y);
    bad |= redi[w];
  }
  if (bad) {
    if (blockIdx.x == 0 && tid == 0) record_status(a.status, FQT_ENONFINITE);
    return;
  }
  const uint32_t B2 = (1u << a.bits) - 1u;
  const float s_g2 = affine_scale(gmin, gmax, B2);
  const float s_g1 = affine_scale(gmin, gmax, 255u);
  const float s_g1_16 = __fmul_rn(s_g1, 65536.0f);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  if (blockIdx.x == 0 && tid == 0) {
    if (KIND == KIND_PTQ) {
      a.inv2[0] = __fdiv_rn(1.0f, s_g2);
      a.zero2[0] = __fmul_rn(s_g2, gmin);
    }
    if (has_b1) {
      a.inv1[0] = __fdiv_rn(1.0f, s_g1);
      a.zero1[0] = __fmul_rn(s_g1, gmin);
    }
  }
  int32_t *const csum_g = has_b1 ? a.csum1 : a.csum2;
  const bool want_cs = csum_g != nullptr;
  int cs[kMaxOct][8];
#pragma unroll
  for (int k = 0; k < kMaxOct; ++k)
#pragma unroll
    for (int j = 0; j < 8; ++j) cs[k][j] = 0;
  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];

  auto issue = [&](int64_t u, int b) {
    const int64_t r0 = u * U;
    const int rows = (int)min((int64_t)U, a.N - r0);
    const uint32_t bytes = (uint32_t)rows * (uint32_t)row_bytes;
    fence_proxy_async_smem();
    mbar_expect_tx(&bar[b], bytes);
    bulk_g2s(smem + (size_t)b * stage_bytes, reinterpret_cast<const unsigned char *>(a.h) + r0 * row_bytes,
             bytes, &bar[b]);
  };
  if (tid == 0 && (int64_t)blockIdx.x < a.n_units) issue(blockIdx.x, 0);

  int it = 0;
  for (int64_t u = blockIdx.x; u < a.n_units; u += gridDim.x, ++it) {
    const int b = it & 1;
    if (tid == 0 && u + gridDim.x < a.n_units) issue(u + gridDim.x, b ^ 1);
    const bool ok = mbar_wait(&bar[b], (uint32_t)(it >> 1) & 1u, a.status);
    if (__syncthreads_or(!ok)) break;
    const unsigned char *sh = smem + (size_t)b * stage_bytes;
    const int64_t r0 = u * U;
    const int rows = (int)min((int64_t)U, a.N - r0);
    const int steps = (rows + 8 * R - 1) / (8 * R);

    // ---------------- BHQ: statistics, block scalars, column sums ----------
    if (KIND == KIND_BHQ) {
      for (int st = 0; st < steps; ++st) {
        const int r = (st * 8 + warp) * R + seg;
        const bool rv = r < rows;
        float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          const int o = sl + LPR * k;
          if (k < OPL && rv && o < CO) {
            float x[8];
            load_oct_smem<T>(sh + (size_t)r * row_bytes, o, lane, x);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              mm.x = fminf(mm.x, x[j]);
              mm.y = fmaxf(mm.y, x[j]);
            }
          }
        }
        mm = seg_reduce(mm, LPR, OpMinMax());
        if (rv && sl == 0) rowst[r] = mm;
      }
      __syncthreads();
      if (tid < G) {
        const int k0 = tid * nb;
        const int nrows = min(nb, rows - k0);
        float s1f = 0.0f, s2f = 0.0f, rho = 0.0f, kap = 0.0f;
        int p = 0;
        if (nrows > 0) {
          float np = -1.0f;
          for (int k = 0; k < nrows; ++k) {  // lead row: largest ||h_k||_inf
            const float2 q = rowst[k0 + k];
            const float nk = fmaxf(fabsf(q.x), fabsf(q.y));
            if (nk > np) { np = nk; p = k; }
          }
          float lam2 = 0.0f;
          for (int k = 0; k < nrows; ++k) {
            const float2 q = rowst[k0 + k];
            if (k != p) lam2 = fmaxf(lam2, fmaxf(fabsf(q.x), fabsf(q.y)));
          }
          lam2 = 2.0f * lam2;
          if (np > 0.0f) {
            float lam1 = __fsub_rn(rowst[k0 + p].y, rowst[k0 + p].x);
            if (!(lam1 > 0.0f)) lam1 = 2.0f * np;
            const float Nf = (float)nrows;
            if (lam2 > 0.0f) {  // s1, s2 of App. D.4
              const float c1 = cbrtf(lam1), c2 = cbrtf(lam2);
              const float n3 = cbrtf(Nf), n6 = sqrtf(n3);
              const float den = c1 * c1 / n3 + c2 * c2 * n3 * n3;
              s1f = (float)B2 * n6 / (c1 * den);
              s2f = (float)B2 * n6 / (c2 * den);
            } else {  // lambda2 -> 0: the other rows are zero
              s1f = (float)B2 * sqrtf(Nf) / lam1;
            }
            if (nrows > 1) {
              rho = 1.0f / sqrtf(Nf);
              kap = 1.0f / (1.0f - rho);
            }
          }
          a.lead2[(r0 / nb) + tid] = p;
        }
        float *bp = bpar + tid * 8;
        bp[0] = s1f;
        bp[1] = s2f;
        bp[2] = rho;
        bp[3] = kap;
        bp[4] = __int_as_float(p);
      }
      __syncthreads();
      // w_j of every block and column of the unit, rows in order
      const int gu = (rows + nb - 1) / nb;
      for (int item = tid; item < gu * C; item += kQ2Threads) {
        const int bb = item / C, j = item - bb * C;
        const float *bp = bpar + bb * 8;
        const int p = __float_as_int(bp[4]);
        const float s1f = bp[0], s2f = bp[1], rho = bp[2], kap = bp[3];
        const int nrows = min(nb, rows - bb * nb);
        float acc = 0.0f;
        for (int k = 0; k < nrows; ++k) {
          const float hv = elem_smem<T>(sh, (int64_t)(bb * nb + k) * C + j);
          const bool lead = k == p;
          const float e = kap * (lead ? rho - 1.0f : rho);
          acc = fmaf(e, __fmul_rn(lead ? s1f : s2f, hv), acc);
        }
        wcol[bb * C + j] = acc;
      }
      __syncthreads();
    }

    // ---------------- per row: scale, rounding, packing, sums ----------------
    for (int st = 0; st < steps; ++st) {
      const int r = (st * 8 + warp) * R + seg;
      const bool rv = r < rows;
      const int64_t row = r0 + r;
      float x[kMaxOct][8];
#pragma unroll
      for (int k = 0; k < kMaxOct; ++k) {
        const int o = sl + LPR * k;
        if (k < OPL && rv && o < CO) {
          load_oct_smem<T>(sh + (size_t)r * row_bytes, o, lane, x[k]);
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) x[k][j] = 0.0f;
        }
      }
      float s2 = s_g2, z2 = gmin, c_row = 0.0f;
      const float *wrow = wcol;
      if (KIND == KIND_PSQ) {
        float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          if (k < OPL && rv && sl + LPR * k < CO) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              mm.x = fminf(mm.x, x[k][j]);
              mm.y = fmaxf(mm.y, x[k][j]);
            }
          }
        }
        mm = seg_reduce(mm, LPR, OpMinMax());
        s2 = affine_scale(mm.x, mm.y, B2);
        z2 = mm.x;
      } else if (KIND == KIND_BHQ) {
        const int bb = rv ? r / nb : 0;
        const float *bp = bpar + bb * 8;
        const bool lead = rv && (r - bb * nb) == __float_as_int(bp[4]);
        s2 = lead ? bp[0] : bp[1];
        c_row = lead ? bp[2] - 1.0f : bp[2];
        wrow = wcol + bb * C;
        float tmin = INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxOct; ++k) {
          const int o = sl + LPR * k;
          if (k < OPL && rv && o < CO) {
#pragma unroll
            for (int j = 0; j < 8; ++j)
              tmin = fminf(tmin, fmaf(-c_row, wrow[o * 8 + j], __fmul_rn(s2, x[k][j])));
          }
        }
        z2 = seg_reduce(tmin, LPR, OpMin());
      }
      const float s2_16 = __fmul_rn(s2, 65536.0f);
      int rs2 = 0, rs1 = 0;
#pragma unroll
      for (int k = 0; k < kMaxOct; ++k) {
        const int o = sl + LPR * k;
        if (!(k < OPL && rv && o < CO)) continue;
        const uint64_t q = (uint64_t)row * (uint64_t)CO + (uint64_t)o;
        uint32_t c[8];
        const uint4 w2 = philox_oct(q, 0u, key);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float v;
          if (KIND == KIND_BHQ) {
            const float t = fmaf(-c_row, wrow[o * 8 + j], __fmul_rn(s2, x[k][j]));
            v = __fmul_rn(__fsub_rn(t, z2), 65536.0f);
          } else {
            v = __fmul_rn(__fsub_rn(x[k][j], z2), s2_16);  // = v 2^16 exactly
          }
          c[j] = sr_code16(v, u16_of(w2, j), B2);
          rs2 += (int)c[j];
        }
        if (a.c2) store_codes8(a.c2 + row * (int64_t)C + o * 8, c);
        if (a.f2) store_carriers8(a.f2 + row * (int64_t)C + o * 8, c, (B2 + 1u) >> 1);
        if (has_b1) {
          const uint4 w1 = philox_oct(q, 1u, key);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float v = __fmul_rn(__fsub_rn(x[k][j], gmin), s_g1_16);
            c[j] = sr_code16(v, u16_of(w1, j), 255u);
            rs1 += (int)c[j];
          }
          if (a.c1) store_codes8(a.c1 + row * (int64_t)C + o * 8, c);
          if (a.f1) store_carriers8(a.f1 + row * (int64_t)C + o * 8, c, 128u);
        }
        if (want_cs) {
#pragma unroll
          for (int j = 0; j < 8; ++j) cs[k][j] += (int)c[j];
        }
      }
      if (a.rsum2) rs2 = seg_reduce(rs2, LPR, OpAdd());
      if (has_b1 && a.rsum1) rs1 = seg_reduce(rs1, LPR, OpAdd());
      if (rv && sl == 0) {
        if (a.rsum2) a.rsum2[row] = rs2;
        if (has_b1 && a.rsum1) a.rsum1[row] = rs1;
        if (KIND == KIND_PSQ) {
          a.inv2[row] = __fdiv_rn(1.0f, s2);
          a.zero2[row] = __fmul_rn(s2, z2);
        } else if (KIND == KIND_BHQ) {
          a.inv2[row] = s2 > 0.0f ? __fdiv_rn(1.0f, s2) : 0.0f;
          a.zero2[row] = z2;
        }
      }
    }
    __syncthreads();  // the stage buffer and the BHQ tables are reused
  }

  // ---------------- column sums ----------------
  if (want_cs) {
#pragma unroll
    for (int k = 0; k < kMaxOct; ++k) {
      const int o = sl + LPR * k;
      const bool valid = k < OPL && o < CO;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        // the segments of a warp own the same columns: fold them first
        int v = valid ? cs[k][j] : 0;
        for (int off = LPR; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (valid && seg == 0 && v) atomicAdd(&csum_s[o * 8 + j], v);
      }
    }
    __syncthreads();
    for (int i = tid; i < C; i += kQ2Threads)
      if (csum_s[i]) atomicAdd(&csum_g[i], csum_s[i]);
  }
}

// ---------------------------------------------------------------------------
// BHQ gradient quantizer for fixed blocks (Sec. 4.2, App. D.4) fused with
// Q_b1 (App. E), in two passes over dH.  The statistics pass holds each
// block in registers: a team of TEAM warps per block of nb rows, each warp
// owning a slab of 8 LPR columns (TEAM > 1 only with LPR = 32, slabs of 256
// columns), lane l owning oct l % LPR of the slab in row l / LPR of each of
// the STEPS row groups (nb = (32 / LPR) STEPS); row reductions are shuffles
// inside a warp and one shared-memory exchange at a named barrier of the
// team.  Its per-entry work is light (statistics, column sums, row minima),
// so the unrolled block fits the instruction cache.  The code pass streams
// the rows with rolled loops (rounding, packing, sums need no block-wide
// exchange once z'_k and w_j are known); k_bhq_offsets then reflects the
// grad_X offsets hz, hr of each block.
//
// Stochastic rounding runs on the fp32 pipe: with U = 128 + u 2^-16 (u the
// 16-bit uniform, exact in fp32), floor(v + u 2^-16) = floor(rd(v + U)) - 128
// because rounding down never crosses an integer, and a second round-down
// addition of 2^23 + 0x6400 - 128 leaves 0x4B006400 + code in the bits:
// code = floor(v + u 2^-16) = (floor(v 2^16) + u) >> 16, the rule of sr_code16
// (R1) for v in [0, B].  Byte 0 of those bits is the code and byte 1 is 0x64,
// so one byte permutation packs two fp16 carriers 1024 + code.
// ---------------------------------------------------------------------------
template <int FROM, class V, class Op>
__device__ __forceinline__ V xor_reduce(V v, Op op) {
#pragma unroll
  for (int off = FROM; off < 32; off <<= 1) v = op(v, shfl_x(v, off));
  return v;
}

// Reduction over the LPR lanes of a row (LPR a power of two, compile time).
template <int LPR, class V, class Op>
__device__ __forceinline__ V row_reduce(V v, Op op) {
#pragma unroll
  for (int off = LPR >> 1; off > 0; off >>= 1) v = op(v, shfl_x(v, off));
  return v;
}

constexpr float kSrMagic = 8414080.0f;     // 2^23 + 0x6400 - 128
constexpr uint32_t kSrBits = 0x4B006400u;  // bits of 2^23 + 0x6400

// 128 + u 2^-16 for the low and the high 16-bit uniform of a Philox word
__device__ __forceinline__ float sr_u_lo(uint32_t w) {
  return __uint_as_float(0x43000000u | (w & 0xFFFFu));
}
__device__ __forceinline__ float sr_u_hi(uint32_t w) {
  return __uint_as_float(__byte_perm(w, 0x43000000u, 0x7632));
}
// uniform j (0..7) of an oct: half (j mod 2) of word j / 2
__device__ __forceinline__ float sr_u(const uint4 &w, int j) {
  const uint32_t word = (j >> 1) == 0 ? w.x : (j >> 1) == 1 ? w.y : (j >> 1) == 2 ? w.z : w.w;
  return (j & 1) ? sr_u_hi(word) : sr_u_lo(word);
}

// kSrBits + code, code = SR(v) for v in [0, B] (v already clamped)
__device__ __forceinline__ uint32_t sr_bits(float v, float U) {
  return __float_as_uint(__fadd_rd(__fadd_rd(v, U), kSrMagic));
}

// Eight codes (kSrBits + code) as centred fp16 carriers code - off.
__device__ __forceinline__ void store_carriers_bits(uint16_t *dst, const uint32_t (&b)[8],
                                                    __half2 bias) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t h = __byte_perm(b[2 * i], b[2 * i + 1], 0x5410);
    __half2 v = __hsub2(*reinterpret_cast<const __half2 *>(&h), bias);
    w[i] = *reinterpret_cast<uint32_t *>(&v);
  }
  *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

// Eight codes (kSrBits + code) as bytes.
__device__ __forceinline__ void store_codes_bits(uint8_t *dst, const uint32_t (&b)[8]) {
  uint2 v;
  v.x = __byte_perm(__byte_perm(b[0], b[1], 0x0040), __byte_perm(b[2], b[3], 0x0040), 0x5410);
  v.y = __byte_perm(__byte_perm(b[4], b[5], 0x0040), __byte_perm(b[6], b[7], 0x0040), 0x5410);
  *reinterpret_cast<uint2 *>(dst) = v;
}

// Named barrier of one team of TEAM warps (ids 1..8; 0 is __syncthreads).
template <int TEAM>
__device__ __forceinline__ void team_sync(int team) {
  if constexpr (TEAM > 1)
    asm volatile("bar.sync %0, %1;" ::"r"(1 + team), "n"(32 * TEAM) : "memory");
}

constexpr int kTeamRows = 16;  // rows of a block when TEAM > 1 (LPR = 32, STEPS <= 16)

// Per-block results of the statistics pass, read by the code pass: lead row
// p (as an integer bit pattern), s1, s2 and rho = 1/sqrt(nb) (0 for a block
// of one row or of zeros), followed in the workspace by w_j for every block.
struct BhqBlock {
  float p, s1, s2, rho;
};

// Workspace bytes of the two-pass BHQ quantizer for blocks of at least 4
// rows: the per-block record and the C column sums w of every block.
size_t bhq_pass_bytes(int64_t N, int64_t C) {
  const int64_t nblk = (N + 3) / 4;
  return (size_t)nblk * sizeof(BhqBlock) + (size_t)nblk * (size_t)C * sizeof(float) + 512;
}

// ---------------------------------------------------------------------------
// Statistics pass of BHQ (the first of the two passes over dH): for every
// block its row statistics, lead row, lambda1, lambda2, s1, s2 (App. D.4),
// the reflection's column sums w_j = sum_k e_k s_k h_kj and the row minima
// z'_k of T = Q diag(s) H (Sec. 4.2), plus the per-CTA (min, max) and
// non-finite flag of the whole tensor (the range of Q_b1) and the clearing of
// the column sums the code pass accumulates into.
// ---------------------------------------------------------------------------
template <typename T, int LPR, int STEPS, int TEAM, int H>
__global__ void __launch_bounds__(256, (STEPS >= 8 ? 1 : 2))
    k_bhq_stats(const QuantArgs a, BhqBlock *__restrict__ bst, float *__restrict__ wsum,
                float2 *__restrict__ part) {
  static_assert(TEAM == 1 || (LPR == 32 && STEPS <= kTeamRows), "team layout");
  static_assert(H == 1 || TEAM == 8, "column halves only for a full team");
  // H column parts of SLAB * TEAM columns each: a part is read, reduced and
  // read again (from L2) after the block's scalars are known
  constexpr int RS = 32 / LPR, SLAB = 8 * LPR, C = SLAB * TEAM * H;
  constexpr int TPC = 8 / TEAM;  // teams per CTA
  constexpr int XW = TEAM > 1 ? 8 : 1;
  __shared__ float2 xs_mm[XW][kTeamRows];
  __shared__ float xs_tm[XW][kTeamRows];
  __shared__ float2 red[8];
  __shared__ int redi[8];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int team = warp / TEAM, wi = warp - team * TEAM;
  const int nb = a.block;
  const int sub = lane / LPR, o = lane - sub * LPR;
  auto col_of = [&](int h) { return ((h * TEAM + wi) * LPR + o) * 8; };
  const float fB2 = (float)((1u << a.bits) - 1u);
  // the code pass accumulates column sums (and, split, row sums) into these
  {
    const int64_t g = (int64_t)blockIdx.x * blockDim.x + tid;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = g; i < C; i += stride) {
      if (a.csum1) a.csum1[i] = 0;
      if (a.csum2) a.csum2[i] = 0;
    }
    if (a.code_split > 1)
      for (int64_t i = g; i < a.N; i += stride) {
        if (a.rsum1) a.rsum1[i] = 0;
        if (a.rsum2) a.rsum2[i] = 0;
      }
  }
  float gmn = INFINITY, gmx = -INFINITY, nanacc = 0.0f;
  const int64_t nblocks = (a.N + nb - 1) / nb;
  const int64_t tstride = (int64_t)gridDim.x * TPC;
  for (int64_t blk = (int64_t)blockIdx.x * TPC + team; blk < nblocks; blk += tstride) {
    const int64_t r0 = blk * nb;
    const int nrows = (int)min((int64_t)nb, a.N - r0);
    float x[STEPS][8];
    bool rv[STEPS];
#pragma unroll
    for (int s = 0; s < STEPS; ++s) rv[s] = sub + RS * s < nrows;
    auto load_part = [&](int h) {
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        const int k = sub + RS * s;
        if (rv[s]) {
          load_oct(reinterpret_cast<const T *>(a.h) + (r0 + k) * C + col_of(h), x[s]);
        } else {
#pragma unroll
          for (int j = 0; j < 8; ++j) x[s][j] = 0.0f;
        }
      }
    };
    // ---- row statistics (and a NaN that any non-finite entry leaves) ----
    float rmin[STEPS], rmax[STEPS];
#pragma unroll
    for (int s = 0; s < STEPS; ++s) {
      rmin[s] = INFINITY;
      rmax[s] = -INFINITY;
    }
#pragma unroll 1
    for (int h = 0; h < H; ++h) {
      load_part(h);
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          mm.x = fminf(mm.x, x[s][j]);
          mm.y = fmaxf(mm.y, x[s][j]);
          nanacc = fmaf(x[s][j], 0.0f, nanacc);
        }
        mm = row_reduce<LPR>(mm, OpMinMax());
        rmin[s] = fminf(rmin[s], mm.x);
        rmax[s] = fmaxf(rmax[s], mm.y);
      }
    }
    if constexpr (TEAM > 1) {
      if (lane == 0) {
#pragma unroll
        for (int s = 0; s < STEPS; ++s) xs_mm[warp][s] = make_float2(rmin[s], rmax[s]);
      }
      team_sync<TEAM>(team);
      float2 mine = make_float2(INFINITY, -INFINITY);
      if (lane < STEPS) {
#pragma unroll
        for (int w2 = 0; w2 < TEAM; ++w2) mine = OpMinMax()(mine, xs_mm[team * TEAM + w2][lane]);
      }
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        rmin[s] = __shfl_sync(0xffffffffu, mine.x, s);
        rmax[s] = __shfl_sync(0xffffffffu, mine.y, s);
      }
    }
#pragma unroll
    for (int s = 0; s < STEPS; ++s)
      if (rv[s]) {
        gmn = fminf(gmn, rmin[s]);
        gmx = fmaxf(gmx, rmax[s]);
      }
    // ---- lead row (largest ||h_k||_inf, lowest index on ties), lambda2 ----
    float bestv = -1.0f;
    int bestk = 0x7fffffff;
#pragma unroll
    for (int s = 0; s < STEPS; ++s) {
      const int k = sub + RS * s;
      const float nk = fmaxf(fabsf(rmin[s]), fabsf(rmax[s]));
      if (rv[s] && (nk > bestv || (nk == bestv && k < bestk))) {
        bestv = nk;
        bestk = k;
      }
    }
#pragma unroll
    for (int off = LPR; off < 32; off <<= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bestv, off);
      const int ok = __shfl_xor_sync(0xffffffffu, bestk, off);
      if (ov > bestv || (ov == bestv && ok < bestk)) {
        bestv = ov;
        bestk = ok;
      }
    }
    const int p = bestk < nrows ? bestk : 0;
    const float np = bestv;
    float l2 = 0.0f;
#pragma unroll
    for (int s = 0; s < STEPS; ++s) {
      const int k = sub + RS * s;
      if (rv[s] && k != p) l2 = fmaxf(l2, fmaxf(fabsf(rmin[s]), fabsf(rmax[s])));
    }
    l2 = xor_reduce<LPR>(l2, OpMaxF());
    const float lam2 = 2.0f * l2;
    // range of the lead row, from the lanes that own it
    float pmin = 0.0f, pmax = 0.0f;
#pragma unroll
    for (int s = 0; s < STEPS; ++s)
      if (s == p / RS) {
        pmin = rmin[s];
        pmax = rmax[s];
      }
    pmin = __shfl_sync(0xffffffffu, pmin, (p % RS) * LPR);
    pmax = __shfl_sync(0xffffffffu, pmax, (p % RS) * LPR);
    // ---- block scalars s1, s2 (App. D.4) and the reflection ----
    float s1f = 0.0f, s2f = 0.0f, rho = 0.0f, kap = 0.0f;
    if (np > 0.0f) {
      float lam1 = __fsub_rn(pmax, pmin);
      if (!(lam1 > 0.0f)) lam1 = 2.0f * np;
      const float Nf = (float)nrows;
      if (lam2 > 0.0f) {
        const float c1 = cbrtf(lam1), c2 = cbrtf(lam2);
        const float n3 = cbrtf(Nf), n6 = sqrtf(n3);
        const float den = c1 * c1 / n3 + c2 * c2 * n3 * n3;
        s1f = fB2 * n6 / (c1 * den);
        s2f = fB2 * n6 / (c2 * den);
      } else {
        s1f = fB2 * sqrtf(Nf) / lam1;
      }
      if (nrows > 1) {
        rho = 1.0f / sqrtf(Nf);
        kap = 1.0f / (1.0f - rho);
      }
    }
    float tmin[STEPS];
#pragma unroll
    for (int s = 0; s < STEPS; ++s) tmin[s] = INFINITY;
    // the last part read is still in registers; the others are read again
#pragma unroll 1
    for (int h = H - 1; h >= 0; --h) {
      if (h != H - 1) load_part(h);
      // w_j = sum_k e_k s_k h_kj over the block (lane: its 8 columns)
      float w[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = 0.0f;
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        const bool lead = (sub + RS * s) == p;
        const float esk = __fmul_rn(kap * (lead ? rho - 1.0f : rho), lead ? s1f : s2f);
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = fmaf(esk, x[s][j], w[j]);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = xor_reduce<LPR>(w[j], OpAddF());
      // ---- row minima of T; the code pass recomputes each t_kj with this
      // same sequence of roundings, so z'_k is exactly its row minimum ----
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        const bool lead = (sub + RS * s) == p;
        const float sk = lead ? s1f : s2f;
        const float ck = lead ? rho - 1.0f : rho;
        float tm = INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) tm = fminf(tm, fmaf(-ck, w[j], __fmul_rn(sk, x[s][j])));
        tmin[s] = fminf(tmin[s], row_reduce<LPR>(tm, OpMin()));
      }
      if (sub == 0) {
        float *wd = wsum + blk * (int64_t)C + col_of(h);
        *reinterpret_cast<float4 *>(wd) = make_float4(w[0], w[1], w[2], w[3]);
        *reinterpret_cast<float4 *>(wd + 4) = make_float4(w[4], w[5], w[6], w[7]);
      }
    }
    if constexpr (TEAM > 1) {
      if (lane == 0) {
#pragma unroll
        for (int s = 0; s < STEPS; ++s) xs_tm[warp][s] = tmin[s];
      }
      team_sync<TEAM>(team);
      float mine = INFINITY;
      if (lane < STEPS) {
#pragma unroll
        for (int w2 = 0; w2 < TEAM; ++w2) mine = fminf(mine, xs_tm[team * TEAM + w2][lane]);
      }
#pragma unroll
      for (int s = 0; s < STEPS; ++s) tmin[s] = __shfl_sync(0xffffffffu, mine, s);
    }
    // ---- outputs ----
    if (wi == 0 && o == 0) {
#pragma unroll
      for (int s = 0; s < STEPS; ++s) {
        const int k = sub + RS * s;
        if (!rv[s]) continue;
        const float sk = k == p ? s1f : s2f;
        a.inv2[r0 + k] = sk > 0.0f ? __fdiv_rn(1.0f, sk) : 0.0f;
        a.zero2[r0 + k] = tmin[s];
      }
      if (sub == 0) {
        bst[blk] = BhqBlock{__int_as_float(p), s1f, s2f, rho};
        a.lead2[blk] = p;
      }
    }
  }
  // ---- range partials of the CTA (NaN marks a non-finite input) ----
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmn = fminf(gmn, __shfl_xor_sync(0xffffffffu, gmn, off));
    gmx = fmaxf(gmx, __shfl_xor_sync(0xffffffffu, gmx, off));
    nanacc += __shfl_xor_sync(0xffffffffu, nanacc, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(gmn, gmx);
    redi[warp] = isnan(nanacc) ? 1 : 0;
  }
  __syncthreads();
  if (tid == 0) {
    int bad = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
      gmn = fminf(gmn, red[i].x);
      gmx = fmaxf(gmx, red[i].y);
      bad |= redi[i];
    }
    part[blockIdx.x] = bad ? make_float2(NAN, NAN) : make_float2(gmn, gmx);
  }
}

// ---------------------------------------------------------------------------
// Code pass of BHQ (the second pass over dH), fused with Q_b1 (App. E): per
// entry t = s_k h_kj - c_k w_j (c_k = rho - 1 on the lead row, rho
// elsewhere) as the statistics pass computed it, v = t - z'_k, stochastic
// rounding of v (Q_b2) and of s (h - min H) (Q_b1), fp16 carriers (and
// optional bytes), row sums of Q_b2 and column sums of the grad_W code set.
// A lane owns two octs of a row, o and o + LPR of a slab of 16 LPR columns
// (one coalesced 16 LPR x 4-byte access per oct); a warp takes units of
// kCodeRows rows and 1 / code_split of the row's slabs, walks those slabs one
// after another and, inside a slab, the unit's rows 32 / LPR at a time,
// issuing the loads of its next row before it rounds the current one.  A
// block's w_j and scalars stay in registers while the lane's rows belong to
// it.  Loops stay rolled; a row's parts meet only in its row sums (atomic
// when code_split > 1, so that wide rows of few chunks still fill the GPU).
// ---------------------------------------------------------------------------
constexpr int kCodeRows = 32;

template <typename T>
__device__ __forceinline__ void load_two_octs(const T *row, int c_a, int c_b, float (&x)[16]) {
  float lo[8], hi[8];
  load_oct(row + c_a, lo);
  load_oct(row + c_b, hi);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    x[j] = lo[j];
    x[8 + j] = hi[j];
  }
}

// SAMPLES: the per-sample PSQ of fqt_quantize_grad_samples instead of BHQ:
// v = s_i (h - z_i) with the scalars of sample i = row / rows_per_sample
// (srec: s, z, inv_s, zero per sample), written per row as well.
template <typename T, int LPR, bool SAMPLES = false>
__global__ void __launch_bounds__(256, 2) k_bhq_codes(const QuantArgs a,
                                                   const BhqBlock *__restrict__ bst,
                                                   const float *__restrict__ wsum, int lg_nb,
                                                   const float4 *__restrict__ srec = nullptr,
                                                   int rows_per_sample = 1) {
  constexpr int RS = 32 / LPR, SLAB = 16 * LPR;
  __shared__ float2 red[8];
  __shared__ int redi[8];
  __shared__ int rs_s[8][2][kCodeRows];
  extern __shared__ int csum_s[];  // C column sums of the grad_W code set
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = a.C, CO = C / 8;
  const int sub = lane / LPR, o = lane - sub * LPR;

  // ---- global range (Q_b1 scale) from the statistics-pass partials ----
  float gmin = INFINITY, gmax = -INFINITY;
  int bad = 0;
  for (int i = tid; i < a.npart; i += blockDim.x) {
    const float2 p = a.part[i];
    bad |= isnan(p.x);
    gmin = fminf(gmin, p.x);
    gmax = fmaxf(gmax, p.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(gmin, gmax);
    redi[warp] = bad;
  }
  for (int i = tid; i < C; i += blockDim.x) csum_s[i] = 0;
  __syncthreads();
  gmin = red[0].x;
  gmax = red[0].y;
  bad = redi[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
    gmin = fminf(gmin, red[w].x);
    gmax = fmaxf(gmax, red[w].y);
    bad |= redi[w];
  }
  if (bad) {
    if (blockIdx.x == 0 && tid == 0) record_status(a.status, FQT_ENONFINITE);
    return;
  }
  const uint32_t B2 = (1u << a.bits) - 1u;
  const float fB2 = (float)B2;
  const float s_g1 = affine_scale(gmin, gmax, 255u);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  if (blockIdx.x == 0 && tid == 0 && has_b1) {
    a.inv1[0] = __fdiv_rn(1.0f, s_g1);
    a.zero1[0] = __fmul_rn(s_g1, gmin);
  }
  int32_t *const csum_g = has_b1 ? a.csum1 : a.csum2;
  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];
  const __half2 bias2 = __half2half2(__int2half_rn(1024 + (int)((B2 + 1u) >> 1)));
  const __half2 bias1 = __half2half2(__int2half_rn(1024 + 128));
  const bool want_rs1 = has_b1 && a.rsum1 != nullptr;
  const T *const h = reinterpret_cast<const T *>(a.h);
  const int nbm = (1 << lg_nb) - 1;

  const int64_t nchunks = (a.N + kCodeRows - 1) / kCodeRows;
  // code_split: a power of two dividing C / SLAB
  const int lg_split = a.code_split > 1 ? __ffs(a.code_split) - 1 : 0;
  const int split = 1 << lg_split;
  const int part_cols = C >> lg_split;
  const int64_t nunits = nchunks << lg_split;
  const int64_t wstride = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t u = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp; u < nunits;
       u += wstride) {
    const int64_t ch = u >> lg_split;
    const int cpart = (int)u & (split - 1);
    const int64_t row0 = ch * kCodeRows;
    const int rows = (int)min((int64_t)kCodeRows, a.N - row0);
    rs_s[warp][0][lane] = 0;
    rs_s[warp][1][lane] = 0;
    __syncwarp();
#pragma unroll 1
    for (int c0 = cpart * part_cols; c0 < (cpart + 1) * part_cols; c0 += SLAB) {
      const int ca = c0 + o * 8, cb = ca + 8 * LPR;  // this lane's two octs
      uint32_t cs[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) cs[j] = 0u;
      uint32_t cs_rows = 0;
      int64_t cur_blk = -1;
      float w[16];
      float sk_l = 0.0f, sk_o = 0.0f, ck_l = 0.0f, ck_o = 0.0f;
      int p_lead = -1;
      // the first row's loads; every later row's are issued one row ahead
      float xn[16];
      float zn = 0.0f;
      {
        const int rr = sub;
        if (rr < rows) {
          load_two_octs(h + (row0 + rr) * C, ca, cb, xn);
          if (!SAMPLES) zn = a.zero2[row0 + rr];
        }
      }
#pragma unroll 1
      for (int rb = 0; rb < rows; rb += RS) {  // the same trip count in every lane
        const int rr = rb + sub;
        const bool valid = rr < rows;  // the LPR lanes of a row agree
        float x[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) x[j] = xn[j];
        const float zr = zn;
        if (rr + RS < rows) {
          load_two_octs(h + (row0 + rr + RS) * C, ca, cb, xn);
          if (!SAMPLES) zn = a.zero2[row0 + rr + RS];
        }
        uint32_t acc1 = 0u, acc2 = 0u;
        if (valid) {
          const int64_t row = row0 + rr;
          const int64_t blk = SAMPLES ? row / rows_per_sample : row >> lg_nb;
          if (blk != cur_blk) {  // a new block (sample): its w_j and scalars
            if constexpr (SAMPLES) {
              const float4 sr = srec[blk];  // s, z, inv_s, zero of the sample
              sk_l = sr.x;
              ck_l = sr.y;
              sk_o = sr.z;
              ck_o = sr.w;
            } else {
              const BhqBlock bs = bst[blk];
              p_lead = __float_as_int(bs.p);
              sk_l = bs.s1;
              sk_o = bs.s2;
              ck_l = bs.rho - 1.0f;
              ck_o = bs.rho;
              load_two_octs(wsum + blk * (int64_t)C, ca, cb, w);
            }
            cur_blk = blk;
          }
          if (SAMPLES && o == 0 && c0 == 0) {
            a.inv2[row] = sk_o;
            a.zero2[row] = ck_o;
          }
          const bool lead = (int)(row & nbm) == p_lead;
          const float sk = lead ? sk_l : sk_o;
          const float ck = lead ? ck_l : ck_o;
          const uint64_t qa = (uint64_t)row * (uint64_t)CO + (uint64_t)(ca >> 3);
          const uint64_t qb = qa + (uint64_t)LPR;
          if (has_b1) {
            const uint4 ua = philox_oct(qa, 1u, key), ub = philox_oct(qb, 1u, key);
            uint32_t b[16];
            acc1 = 0u - 16u * kSrBits;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float v = fminf(__fmul_rn(__fsub_rn(x[j], gmin), s_g1), 255.0f);
              b[j] = sr_bits(v, sr_u(j < 8 ? ua : ub, j & 7));
              cs[j] += b[j];
              acc1 += b[j];
            }
            ++cs_rows;
            uint32_t (&b0)[8] = *reinterpret_cast<uint32_t(*)[8]>(&b[0]);
            uint32_t (&b1)[8] = *reinterpret_cast<uint32_t(*)[8]>(&b[8]);
            if (a.c1) {
              store_codes_bits(a.c1 + row * (int64_t)C + ca, b0);
              store_codes_bits(a.c1 + row * (int64_t)C + cb, b1);
            }
            if (a.f1) {
              store_carriers_bits(a.f1 + row * (int64_t)C + ca, b0, bias1);
              store_carriers_bits(a.f1 + row * (int64_t)C + cb, b1, bias1);
            }
          }
          const uint4 ua = philox_oct(qa, 0u, key), ub = philox_oct(qb, 0u, key);
          uint32_t b[16];
          acc2 = 0u - 16u * kSrBits;
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            // BHQ: t - z'; per-sample PSQ: s (h - z) with the sample's s, z (Sec. 4.1)
            const float v = SAMPLES ? __fmul_rn(__fsub_rn(x[j], ck_l), sk_l)
                                    : __fsub_rn(fmaf(-ck, w[j], __fmul_rn(sk, x[j])), zr);
            b[j] = sr_bits(fminf(v, fB2), sr_u(j < 8 ? ua : ub, j & 7));
            acc2 += b[j];
            if (!has_b1) cs[j] += b[j];
          }
          if (!has_b1) ++cs_rows;
          uint32_t (&b0)[8] = *reinterpret_cast<uint32_t(*)[8]>(&b[0]);
          uint32_t (&b1)[8] = *reinterpret_cast<uint32_t(*)[8]>(&b[8]);
          if (a.c2) {
            store_codes_bits(a.c2 + row * (int64_t)C + ca, b0);
            store_codes_bits(a.c2 + row * (int64_t)C + cb, b1);
          }
          if (a.f2) {
            store_carriers_bits(a.f2 + row * (int64_t)C + ca, b0, bias2);
            store_carriers_bits(a.f2 + row * (int64_t)C + cb, b1, bias2);
          }
        }
        if (want_rs1) {
          const int r1 = row_reduce<LPR>((int)acc1, OpAdd());
          if (o == 0 && valid) rs_s[warp][1][rr] += r1;
        }
        const int r2 = row_reduce<LPR>((int)acc2, OpAdd());
        if (o == 0 && valid) rs_s[warp][0][rr] += r2;
      }
      // this slab's column sums: the lanes of one column add theirs
      if (csum_g) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int v = xor_reduce<LPR>((int)(cs[j] - cs_rows * kSrBits), OpAdd());
          if (sub == 0 && v) atomicAdd(&csum_s[(j < 8 ? ca : cb) + (j & 7)], v);
        }
      }
    }
    __syncwarp();
    if (lane < rows) {
      if (split > 1) {
        if (a.rsum2) atomicAdd(&a.rsum2[row0 + lane], rs_s[warp][0][lane]);
        if (want_rs1) atomicAdd(&a.rsum1[row0 + lane], rs_s[warp][1][lane]);
      } else {
        if (a.rsum2) a.rsum2[row0 + lane] = rs_s[warp][0][lane];
        if (want_rs1) a.rsum1[row0 + lane] = rs_s[warp][1][lane];
      }
    }
    __syncwarp();
  }
  if (csum_g) {
    __syncthreads();
    for (int i = tid; i < C; i += blockDim.x)
      if (csum_s[i]) atomicAdd(&csum_g[i], csum_s[i]);
  }
}

// Column parts per chunk of kCodeRows rows in the code pass: slabs of a row
// are split until the (chunk, part) units reach about 64 per SM.
static int code_split_of(int64_t N, int C, int lpr, int num_sms) {
  const int nslab = C / (16 * lpr);
  const int64_t nchunks = (N + kCodeRows - 1) / kCodeRows;
  const int64_t target = (int64_t)num_sms * 64;
  int split = 1;
  while (split < nslab && nchunks * split < target) split *= 2;
  return split;
}

template <typename T, int LPR, int STEPS, int TEAM, int H = 1>
static cudaError_t launch_stats(const QuantArgs &a, BhqBlock *bst, float *wsum, float2 *part,
                                int num_sms, int *grid_out, cudaStream_t st) {
  auto kern = k_bhq_stats<T, LPR, STEPS, TEAM, H>;
  int per_sm = 0;
  const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, 0);
  if (e != cudaSuccess) return e;
  const int64_t nblocks = (a.N + a.block - 1) / a.block;
  constexpr int TPC = 8 / TEAM;
  int64_t grid = (nblocks + TPC - 1) / TPC;
  int64_t cap = (int64_t)num_sms * (per_sm > 0 ? per_sm : 1);
  if (cap > kMaxRangeCtas) cap = kMaxRangeCtas;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  *grid_out = (int)grid;
  kern<<<(int)grid, 256, 0, st>>>(a, bst, wsum, part);
  return cudaGetLastError();
}

template <typename T, int LPR>
static cudaError_t launch_codes(const QuantArgs &a, const BhqBlock *bst, const float *wsum,
                                int num_sms, cudaStream_t st) {
  int lg_nb = 0;
  while ((1 << lg_nb) < a.block) ++lg_nb;
  auto kern = k_bhq_codes<T, LPR>;
  const size_t smem = sizeof(int) * (size_t)a.C;
  int per_sm = 0;
  const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, smem);
  if (e != cudaSuccess) return e;
  const int64_t nunits = (a.N + kCodeRows - 1) / kCodeRows * (a.code_split > 1 ? a.code_split : 1);
  int64_t grid = (nunits + 7) / 8;
  const int64_t cap = (int64_t)num_sms * (per_sm > 0 ? per_sm : 1);
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  kern<<<(int)grid, 256, smem, st>>>(a, bst, wsum, lg_nb, nullptr, 1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Per-sample PSQ (fqt_quantize_grad_samples; Sec. 4.1 with a sample = R
// consecutive rows of dH, an image's output pixels): k_sample_part takes the
// (min, max) of chunks of kSampleChunk rows' worth of entries inside one
// sample; k_sample_finish reduces each sample's chunks to s = B / R(h_i),
// z = min h_i (affine_scale, as the row quantizer), 1 / s and s z, and leaves
// per-CTA (min, max) of the whole tensor (the range of Q_b1).  The code pass
// (k_bhq_codes, SAMPLES) then rounds and packs.
// ---------------------------------------------------------------------------
constexpr int kSampleChunkElems = 16384;

template <typename T>
__global__ void __launch_bounds__(256) k_sample_part(const QuantArgs a, int64_t sample_elems,
                                                     int chunks_per_sample, float2 *cpart) {
  __shared__ float2 red[8];
  __shared__ int redi[8];
  const int64_t ch = blockIdx.x;
  const int64_t smp = ch / chunks_per_sample;
  const int64_t e0 = smp * sample_elems + (ch - smp * chunks_per_sample) * kSampleChunkElems;
  const int64_t e1 = min(smp * sample_elems + sample_elems, e0 + kSampleChunkElems);
  const T *h = reinterpret_cast<const T *>(a.h);
  float mn = INFINITY, mx = -INFINITY, nanacc = 0.0f;
  for (int64_t e = e0 + (int64_t)threadIdx.x * 8; e < e1; e += (int64_t)blockDim.x * 8) {
    float x[8];
    load_oct(h + e, x);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      mn = fminf(mn, x[j]);
      mx = fmaxf(mx, x[j]);
      nanacc = fmaf(x[j], 0.0f, nanacc);
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    nanacc += __shfl_xor_sync(0xffffffffu, nanacc, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(mn, mx);
    redi[warp] = isnan(nanacc) ? 1 : 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int bad = 0;
    for (int i = 0; i < 8; ++i) {
      mn = fminf(mn, red[i].x);
      mx = fmaxf(mx, red[i].y);
      bad |= redi[i];
    }
    cpart[ch] = bad ? make_float2(NAN, NAN) : make_float2(mn, mx);
  }
}

__global__ void __launch_bounds__(256) k_sample_finish(const QuantArgs a, int64_t nsamples,
                                                       int chunks_per_sample,
                                                       const float2 *cpart, float4 *srec,
                                                       float2 *part) {
  __shared__ float2 red[8];
  __shared__ int redi[8];
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint32_t B = (1u << a.bits) - 1u;
  float mn = INFINITY, mx = -INFINITY;
  int bad = 0;
  if (i < nsamples) {
    for (int k = 0; k < chunks_per_sample; ++k) {
      const float2 p = cpart[i * chunks_per_sample + k];
      bad |= isnan(p.x);
      mn = fminf(mn, p.x);
      mx = fmaxf(mx, p.y);
    }
    const float s = affine_scale(mn, mx, B);
    srec[i] = make_float4(s, mn, __fdiv_rn(1.0f, s), __fmul_rn(s, mn));
  }
  // the CTA's (min, max) of the whole tensor, for Q_b1
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, off));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(mn, mx);
    redi[warp] = bad;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < 8; ++w) {
      mn = fminf(mn, red[w].x);
      mx = fmaxf(mx, red[w].y);
      bad |= redi[w];
    }
    mn = fminf(mn, red[0].x);
    mx = fmaxf(mx, red[0].y);
    bad |= redi[0];
    part[blockIdx.x] = bad ? make_float2(NAN, NAN) : make_float2(mn, mx);
  }
  // the code pass accumulates column sums (and, split, row sums) into these
  for (int64_t k = i; k < a.C; k += (int64_t)gridDim.x * blockDim.x) {
    if (a.csum1) a.csum1[k] = 0;
    if (a.csum2) a.csum2[k] = 0;
  }
  if (a.code_split > 1)
    for (int64_t k = i; k < a.N; k += (int64_t)gridDim.x * blockDim.x) {
      if (a.rsum1) a.rsum1[k] = 0;
      if (a.rsum2) a.rsum2[k] = 0;
    }
}

// Workspace bytes of the per-sample quantizer: chunk partials and records.
size_t sample_pass_bytes(int64_t N, int64_t C, int64_t rows_per_sample) {
  if (rows_per_sample < 1) return 0;
  const int64_t ns = N / rows_per_sample;
  const int64_t cps = (rows_per_sample * C + kSampleChunkElems - 1) / kSampleChunkElems;
  return (size_t)(ns * cps) * sizeof(float2) + (size_t)ns * sizeof(float4) + 512;
}

// The per-sample PSQ with Q_b1: rows of C in {64, 128, 256 t} columns
// (t = 1, 2, 4, 8), N a multiple of rows_per_sample, at most 2^20 samples.
fqt_status launch_sample_passes(QuantArgs &a, bool bf16, int64_t rows_per_sample, int num_sms,
                                void *scratch, float2 *part, cudaStream_t st) {
  const int C = a.C;
  if (!(C == 64 || C == 128 || C == 256 || C == 512 || C == 1024 || C == 2048 || C == 4096))
    return FQT_EUNSUPPORTED;
  const int64_t ns = a.N / rows_per_sample;
  if (ns > ((int64_t)1 << 20)) return FQT_EUNSUPPORTED;
  const int64_t se = rows_per_sample * C;
  const int cps = (int)((se + kSampleChunkElems - 1) / kSampleChunkElems);
  float2 *cpart = static_cast<float2 *>(scratch);
  float4 *srec = reinterpret_cast<float4 *>(
      (reinterpret_cast<uintptr_t>(cpart + ns * cps) + 255) & ~(uintptr_t)255);
  const int lpr = C == 64 ? 4 : C == 128 ? 8 : C == 256 ? 16 : 32;
  a.code_split = code_split_of(a.N, C, lpr, num_sms);
  if (bf16)
    k_sample_part<__nv_bfloat16><<<(unsigned)(ns * cps), 256, 0, st>>>(a, se, cps, cpart);
  else
    k_sample_part<float><<<(unsigned)(ns * cps), 256, 0, st>>>(a, se, cps, cpart);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "sample statistics launch");
  const int fin = (int)((ns + 255) / 256);
  k_sample_finish<<<fin, 256, 0, st>>>(a, ns, cps, cpart, srec, part);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "sample scalars launch");
  QuantArgs a2 = a;
  a2.part = part;
  a2.npart = fin;
  const int R = (int)rows_per_sample;
#define FQT_SC(TT, L)                                                                        \
  {                                                                                          \
    auto kern = k_bhq_codes<TT, L, true>;                                                    \
    const size_t smem = sizeof(int) * (size_t)C;                                             \
    int per_sm = 0;                                                                          \
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, smem);             \
    if (e == cudaSuccess) {                                                                  \
      const int64_t nunits = (a.N + kCodeRows - 1) / kCodeRows * a2.code_split;              \
      int64_t grid = (nunits + 7) / 8;                                                       \
      const int64_t cap = (int64_t)num_sms * (per_sm > 0 ? per_sm : 1);                     \
      if (grid > cap) grid = cap;                                                            \
      if (grid < 1) grid = 1;                                                                \
      kern<<<(int)grid, 256, smem, st>>>(a2, nullptr, nullptr, 0, srec, R);                  \
      e = cudaGetLastError();                                                                \
    }                                                                                        \
  }
  if (!bf16) {
    if (lpr == 4) FQT_SC(float, 4) else if (lpr == 8) FQT_SC(float, 8)
    else if (lpr == 16) FQT_SC(float, 16) else FQT_SC(float, 32)
  } else {
    if (lpr == 4) FQT_SC(__nv_bfloat16, 4) else if (lpr == 8) FQT_SC(__nv_bfloat16, 8)
    else if (lpr == 16) FQT_SC(__nv_bfloat16, 16) else FQT_SC(__nv_bfloat16, 32)
  }
#undef FQT_SC
  return cuda_fail(e, "sample code pass launch");
}

// The two-pass BHQ quantizer takes fixed blocks of 4, 8 or 16 rows and rows
// of 64, 128 or 256 t (t = 1, 2, 4, 8, 16) columns; bf16 input with blocks of 16.
bool bhq_pass_supported(int C, int block, bool bf16) {
  if (block != 4 && block != 8 && block != 16) return false;
  if (bf16 && block != 16) return false;
  return C == 64 || C == 128 || C == 256 || C == 512 || C == 1024 || C == 2048 || C == 4096;
}

// Statistics pass, code pass and the grad_X offsets (k_bhq_offsets) of the
// fixed-block BHQ quantizer with Q_b1.  `scratch` (bhq_pass_bytes) holds the
// per-block records and column sums w between the passes; `part` receives
// the statistics pass's range partials, which the code pass reduces.
fqt_status launch_bhq_passes(QuantArgs &a, bool bf16, int num_sms, void *scratch,
                             float2 *part, cudaStream_t st) {
  if (a.kind != KIND_BHQ || !bhq_pass_supported(a.C, a.block, bf16)) return FQT_EUNSUPPORTED;
  const int64_t nblocks = (a.N + a.block - 1) / a.block;
  BhqBlock *bst = static_cast<BhqBlock *>(scratch);
  float *wsum = reinterpret_cast<float *>(
      (reinterpret_cast<uintptr_t>(bst + nblocks) + 255) & ~(uintptr_t)255);
  const int C = a.C, nb = a.block;
  // lanes per row of the code pass: a lane owns 16 columns (two octs) of a
  // slab of 16 LPR
  const int lpr = C == 64 ? 4 : C == 128 ? 8 : C == 256 ? 16 : 32;
  a.code_split = code_split_of(a.N, C, lpr, num_sms);
  int grid1 = 0;
  cudaError_t e = cudaErrorInvalidValue;
#define FQT_ST(TT, L, S, TM) e = launch_stats<TT, L, S, TM>(a, bst, wsum, part, num_sms, &grid1, st);
  // C = 4096: a team of 8 warps over two column halves
#define FQT_ST2(TT, L, S) e = launch_stats<TT, L, S, 8, 2>(a, bst, wsum, part, num_sms, &grid1, st);
  if (!bf16) {
    if (C == 64) {
      if (nb == 4) { FQT_ST(float, 8, 1, 1) } else if (nb == 8) { FQT_ST(float, 8, 2, 1) }
      else { FQT_ST(float, 8, 4, 1) }
    } else if (C == 128) {
      if (nb == 4) { FQT_ST(float, 16, 2, 1) } else if (nb == 8) { FQT_ST(float, 16, 4, 1) }
      else { FQT_ST(float, 16, 8, 1) }
    } else {
      const int team = C / 256;
#define FQT_ST_T(S)                                                                  \
  if (team == 1) { FQT_ST(float, 32, S, 1) } else if (team == 2) { FQT_ST(float, 32, S, 2) } \
  else if (team == 4) { FQT_ST(float, 32, S, 4) } else if (team == 8) { FQT_ST(float, 32, S, 8) } \
  else { FQT_ST2(float, 32, S) }
      if (nb == 4) { FQT_ST_T(4) } else if (nb == 8) { FQT_ST_T(8) } else { FQT_ST_T(16) }
#undef FQT_ST_T
    }
  } else {
    if (C == 64) { FQT_ST(__nv_bfloat16, 8, 4, 1) }
    else if (C == 128) { FQT_ST(__nv_bfloat16, 16, 8, 1) }
    else if (C == 256) { FQT_ST(__nv_bfloat16, 32, 16, 1) }
    else if (C == 512) { FQT_ST(__nv_bfloat16, 32, 16, 2) }
    else if (C == 1024) { FQT_ST(__nv_bfloat16, 32, 16, 4) }
    else if (C == 2048) { FQT_ST(__nv_bfloat16, 32, 16, 8) }
    else { FQT_ST2(__nv_bfloat16, 32, 16) }
  }
#undef FQT_ST
#undef FQT_ST2
  if (e != cudaSuccess) return cuda_fail(e, "BHQ statistics pass launch");
  QuantArgs a2 = a;
  a2.part = part;
  a2.npart = grid1;
  if (!bf16) {
    e = lpr == 4    ? launch_codes<float, 4>(a2, bst, wsum, num_sms, st)
        : lpr == 8  ? launch_codes<float, 8>(a2, bst, wsum, num_sms, st)
        : lpr == 16 ? launch_codes<float, 16>(a2, bst, wsum, num_sms, st)
                    : launch_codes<float, 32>(a2, bst, wsum, num_sms, st);
  } else {
    e = lpr == 4    ? launch_codes<__nv_bfloat16, 4>(a2, bst, wsum, num_sms, st)
        : lpr == 8  ? launch_codes<__nv_bfloat16, 8>(a2, bst, wsum, num_sms, st)
        : lpr == 16 ? launch_codes<__nv_bfloat16, 16>(a2, bst, wsum, num_sms, st)
                    : launch_codes<__nv_bfloat16, 32>(a2, bst, wsum, num_sms, st);
  }
  if (e != cudaSuccess) return cuda_fail(e, "BHQ code pass launch");
  if (a.hz && a.hr) {
    e = launch_bhq_offsets(a.zero2, a.rsum2, a.lead2, a.hz, a.hr, a.N, C, a.bits, a.block, st);
    if (e != cudaSuccess) return cuda_fail(e, "BHQ offsets launch");
  }
  return FQT_OK;
}

// ---------------------------------------------------------------------------
// Per-sample power-of-two shift quantizer (Sec. 4.3; the reading is stated in
// include/fqt.h): one symmetric per-tensor range [-M, M] from the range pass,
// s = (2^(b-1) - 1) / M, and per row the largest shift in [0, 4] with
// 2^shift ||h_i||_inf <= M; code = SR(s 2^shift h + 2^(b-1)).  A row is held
// by LPR lanes, OPL octs (8 columns) each, in registers; a warp step covers
// RS = 32 / LPR rows.  Besides the grad_X encoding (codes, centred fp16
// carriers, row sums, inv_s = 2^-shift / s, zero = -2^(b-1)) it writes the
// grad_W operand: the codes on the common scale 2^-4 / s, a = 2^(4 - shift)
// (code - 2^(b-1)), as exact fp16, and their column sums.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void store_shifted8(uint16_t *dst, const uint32_t (&c)[8],
                                               uint32_t off, float mul) {
  const __half2 bias = __half2half2(__int2half_rn(1024 + (int)off));
  const __half2 m2 = __float2half2_rn(mul);  // a power of two: exact products
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t hb = (0x6400u | c[2 * i]) | ((0x6400u | c[2 * i + 1]) << 16);
    __half2 v = __hmul2(__hsub2(*reinterpret_cast<const __half2 *>(&hb), bias), m2);
    w[i] = *reinterpret_cast<uint32_t *>(&v);
  }
  *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename T, int LPR, int OPL>
__global__ void __launch_bounds__(256) k_shift(const QuantArgs a) {
  __shared__ float2 red[8];
  __shared__ int redi[8];
  extern __shared__ int csum_s[];  // [C] shifted-code column sums, [C] Q_b1 column sums
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int RS = 32 / LPR, C = 8 * LPR * OPL, CO = C / 8;
  const int sub = lane / LPR, o = lane - sub * LPR;

  // ---- global range from the range-pass partials ----
  float gmin = INFINITY, gmax = -INFINITY;
  int bad = 0;
  for (int i = tid; i < a.npart; i += blockDim.x) {
    const float2 p = a.part[i];
    bad |= isnan(p.x);
    gmin = fminf(gmin, p.x);
    gmax = fmaxf(gmax, p.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(gmin, gmax);
    redi[warp] = bad;
  }
  for (int i = tid; i < 2 * C; i += blockDim.x) csum_s[i] = 0;
  __syncthreads();
  gmin = red[0].x;
  gmax = red[0].y;
  bad = redi[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
    gmin = fminf(gmin, red[w].x);
    gmax = fmaxf(gmax, red[w].y);
    bad |= redi[w];
  }
  if (bad) {
    if (blockIdx.x == 0 && tid == 0) record_status(a.status, FQT_ENONFINITE);
    return;
  }
  const uint32_t B = (1u << a.bits) - 1u, z0 = 1u << (a.bits - 1);
  const float M = fmaxf(fabsf(gmin), fabsf(gmax));
  float s = __fdiv_rn((float)(z0 - 1u), M);
  if (!(M > 0.0f) || !isfinite(s)) s = 1.0f;
  const float inv = __fdiv_rn(1.0f, s);
  const float s_g1 = affine_scale(gmin, gmax, 255u);
  const float s_g1_16 = __fmul_rn(s_g1, 65536.0f);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  if (blockIdx.x == 0 && tid == 0) {
    a.sscale[0] = __fmul_rn(inv, 0.0625f);
    a.sscale[1] = 0.0f;
    if (has_b1) {
      a.inv1[0] = __fdiv_rn(1.0f, s_g1);
      a.zero1[0] = __fmul_rn(s_g1, gmin);
    }
  }
  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];
  int csA[OPL][8], cs1[OPL][8];
#pragma unroll
  for (int q = 0; q < OPL; ++q)
#pragma unroll
    for (int j = 0; j < 8; ++j) csA[q][j] = cs1[q][j] = 0;
  const T *h = reinterpret_cast<const T *>(a.h);
  const int64_t step = (int64_t)gridDim.x * (blockDim.x >> 5) * RS;
  for (int64_t r0 = ((int64_t)blockIdx.x * (blockDim.x >> 5) + warp) * RS; r0 < a.N;
       r0 += step) {
    const int64_t row = r0 + sub;
    const bool v = row < a.N;
    float x[OPL][8];
#pragma unroll
    for (int q = 0; q < OPL; ++q) {
      if (v) {
        load_oct(h + row * C + (q * LPR + o) * 8, x[q]);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) x[q][j] = 0.0f;
      }
    }
    float mi = 0.0f;
#pragma unroll
    for (int q = 0; q < OPL; ++q)
#pragma unroll
      for (int j = 0; j < 8; ++j) mi = fmaxf(mi, fabsf(x[q][j]));
    mi = row_reduce<LPR>(mi, OpMaxF());
    // largest shift in [0, 4] with 2^shift ||h_i||_inf <= M (exact products)
    int sh = 0;
#pragma unroll
    for (int k = 1; k <= 4; ++k)
      if (__fmul_rn(mi, (float)(1 << k)) <= M) sh = k;
    const float sr = __fmul_rn(s, (float)(1 << sh));
    const float mul = (float)(1 << (4 - sh));
    int rs2 = 0, rs1 = 0;
#pragma unroll
    for (int q = 0; q < OPL; ++q) {
      if (!v) continue;
      const int oct = q * LPR + o;
      const uint64_t qi = (uint64_t)row * (uint64_t)CO + (uint64_t)oct;
      const uint4 w2 = philox_oct(qi, 0u, key);
      uint32_t c[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float vv = __fadd_rn(__fmul_rn(sr, x[q][j]), (float)z0);
        c[j] = sr_code16(__fmul_rn(vv, 65536.0f), u16_of(w2, j), B);
        rs2 += (int)c[j];
        csA[q][j] += ((int)c[j] - (int)z0) * (1 << (4 - sh));
      }
      if (a.c2) store_codes8(a.c2 + row * (int64_t)C + oct * 8, c);
      if (a.f2) store_carriers8(a.f2 + row * (int64_t)C + oct * 8, c, z0);
      store_shifted8(a.fs + row * (int64_t)C + oct * 8, c, z0, mul);
      if (has_b1) {
        const uint4 w1 = philox_oct(qi, 1u, key);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float vv = __fmul_rn(__fsub_rn(x[q][j], gmin), s_g1_16);
          c[j] = sr_code16(vv, u16_of(w1, j), 255u);
          rs1 += (int)c[j];
          cs1[q][j] += (int)c[j];
        }
        if (a.c1) store_codes8(a.c1 + row * (int64_t)C + oct * 8, c);
        if (a.f1) store_carriers8(a.f1 + row * (int64_t)C + oct * 8, c, 128u);
      }
    }
    rs2 = row_reduce<LPR>(rs2, OpAdd());
    if (has_b1) rs1 = row_reduce<LPR>(rs1, OpAdd());
    if (v && o == 0) {
      if (a.rsum2) a.rsum2[row] = rs2;
      if (has_b1 && a.rsum1) a.rsum1[row] = rs1;
      a.inv2[row] = __fmul_rn(inv, __fdiv_rn(1.0f, (float)(1 << sh)));
      a.zero2[row] = -(float)z0;
      a.shift[row] = sh;
    }
  }
  // ---- column sums: rows of a step, then the CTA, then global ----
#pragma unroll
  for (int q = 0; q < OPL; ++q)
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int va = xor_reduce<LPR>(csA[q][j], OpAdd());
      const int v1 = has_b1 ? xor_reduce<LPR>(cs1[q][j], OpAdd()) : 0;
      if (sub == 0) {
        if (va) atomicAdd(&csum_s[(q * LPR + o) * 8 + j], va);
        if (v1) atomicAdd(&csum_s[C + (q * LPR + o) * 8 + j], v1);
      }
    }
  __syncthreads();
  for (int i = tid; i < C; i += blockDim.x) {
    if (csum_s[i]) atomicAdd(&a.scs[i], csum_s[i]);
    if (has_b1 && a.csum1 && csum_s[C + i]) atomicAdd(&a.csum1[i], csum_s[C + i]);
  }
}

fqt_status launch_shift(QuantArgs &a, bool bf16, int num_sms, cudaStream_t st) {
  if (a.C % 8) return FQT_EUNSUPPORTED;
  const int CO = a.C / 8;
  int lpr, opl;
  switch (CO) {
    case 8: lpr = 8; opl = 1; break;
    case 16: lpr = 16; opl = 1; break;
    case 32: lpr = 32; opl = 1; break;
    case 64: lpr = 32; opl = 2; break;
    case 128: lpr = 32; opl = 4; break;
    default: return FQT_EUNSUPPORTED;
  }
  const int rs = 32 / lpr;
  int64_t grid = (a.N + 8 * rs - 1) / (8 * rs);
  const int64_t cap = (int64_t)num_sms * 4;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  const size_t smem = 2 * sizeof(int) * (size_t)a.C;
#define FQT_SH(L, P)                                                                   \
  if (lpr == L && opl == P) {                                                          \
    if (bf16)                                                                          \
      k_shift<__nv_bfloat16, L, P><<<(int)grid, 256, smem, st>>>(a);                   \
    else                                                                               \
      k_shift<float, L, P><<<(int)grid, 256, smem, st>>>(a);                           \
  }
  FQT_SH(8, 1)
  FQT_SH(16, 1)
  FQT_SH(32, 1)
  FQT_SH(32, 2)
  FQT_SH(32, 4)
#undef FQT_SH
  return cuda_fail(cudaGetLastError(), "shift quantizer launch");
}

// ---------------------------------------------------------------------------
// Codes of a forward operand (deterministic PTQ, Sec. 2.1 and App. E):
// code = round_half_even((x - z) s) clamped to [0, B], z = min X, s = B / R(X).
// A thread owns one column oct (8 columns) in every row it visits, so its
// column sums stay in registers; a CTA covers rpi rows per step.  Row groups
// are visited from the end of the matrix, which the range pass read last
// and left in L2.  Rounding adds 1.5 2^23 (exact round-half-even of values
// below 2^22 by the FADD itself).
// ---------------------------------------------------------------------------
constexpr int kFwdUnroll = 4;
constexpr int kFwdMaxThreads = 1024;

template <typename T>
__global__ void __launch_bounds__(kFwdMaxThreads)
    k_fwd_codes(const T *__restrict__ X, int64_t rows, int cols, int rpi,
                uint16_t *__restrict__ f16, uint8_t *__restrict__ c8,
                int32_t *__restrict__ col_sum, const float2 *__restrict__ part, int npart,
                float *inv_out, float *zero_out, int bits, int *status, int conv_zero,
                int32_t *code_zero_out) {
  extern __shared__ int csum_s[];  // cols
  __shared__ float2 red[kFwdMaxThreads / 32];
  __shared__ int redi[kFwdMaxThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float gmin = INFINITY, gmax = -INFINITY;
  int bad = 0;
  for (int i = tid; i < npart; i += blockDim.x) {
    const float2 p = part[i];
    bad |= isnan(p.x);
    gmin = fminf(gmin, p.x);
    gmax = fmaxf(gmax, p.y);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    gmin = fminf(gmin, __shfl_xor_sync(0xffffffffu, gmin, off));
    gmax = fmaxf(gmax, __shfl_xor_sync(0xffffffffu, gmax, off));
    bad |= __shfl_xor_sync(0xffffffffu, bad, off);
  }
  if (lane == 0) {
    red[warp] = make_float2(gmin, gmax);
    redi[warp] = bad;
  }
  for (int i = tid; i < cols; i += blockDim.x) csum_s[i] = 0;
  __syncthreads();
  gmin = red[0].x;
  gmax = red[0].y;
  bad = redi[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
    gmin = fminf(gmin, red[w].x);
    gmax = fmaxf(gmax, red[w].y);
    bad |= redi[w];
  }
  if (bad) {
    if (blockIdx.x == 0 && tid == 0) record_status(status, FQT_ENONFINITE);
    return;
  }
  const uint32_t B = (1u << bits) - 1u;
  if (conv_zero) {  // the im2col matrix also holds the padding zeros
    gmin = fminf(gmin, 0.0f);
    gmax = fmaxf(gmax, 0.0f);
  }
  const float s = affine_scale(gmin, gmax, B), z = gmin;
  const uint32_t off = (B + 1u) >> 1;  // carriers: code - 2^(b-1)
  if (blockIdx.x == 0 && tid == 0) {
    inv_out[0] = __fdiv_rn(1.0f, s);
    zero_out[0] = __fmul_rn(s, z);
    if (code_zero_out) {  // the code of 0.0 (a conv operand's padding)
      const float v0 = __fmul_rn(__fsub_rn(0.0f, z), s);
      *code_zero_out = (int32_t)min(__float_as_uint(__fadd_rn(v0, 12582912.0f)) - 0x4B400000u, B);
    }
  }
  const int opr = cols / 8;
  const int rl = tid / opr, o = tid - rl * opr;
  const bool lane_on = rl < rpi;
  int cs[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) cs[j] = 0;
  const int64_t groups = (rows + rpi - 1) / rpi;
  for (int64_t i0 = blockIdx.x; i0 < groups; i0 += (int64_t)kFwdUnroll * gridDim.x) {
    float x[kFwdUnroll][8];
    int64_t row[kFwdUnroll];
    bool ok[kFwdUnroll];
#pragma unroll
    for (int u = 0; u < kFwdUnroll; ++u) {
      const int64_t gi = i0 + (int64_t)u * gridDim.x;
      row[u] = (groups - 1 - gi) * rpi + rl;
      ok[u] = lane_on && gi < groups && row[u] < rows;
      if (ok[u]) load_oct(X + row[u] * cols + o * 8, x[u]);
    }
#pragma unroll
    for (int u = 0; u < kFwdUnroll; ++u) {
      if (!ok[u]) continue;
      uint32_t c[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float v = __fmul_rn(__fsub_rn(x[u][j], z), s);
        const uint32_t r = __float_as_uint(__fadd_rn(v, 12582912.0f)) - 0x4B400000u;
        c[j] = min(r, B);  // v >= 0: r is the rounded value
        cs[j] += (int)c[j];
      }
      const int64_t e = row[u] * cols + o * 8;
      if (f16) store_carriers8(f16 + e, c, off);
      if (c8) store_codes8(c8 + e, c);
    }
  }
  if (col_sum) {
    if (lane_on) {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (cs[j]) atomicAdd(&csum_s[o * 8 + j], cs[j]);
    }
    __syncthreads();
    for (int i = tid; i < cols; i += blockDim.x)
      if (csum_s[i]) atomicAdd(&col_sum[i], csum_s[i]);
  }
}

fqt_status launch_fwd_codes(const void *X, bool bf16, int64_t rows, int cols, int bits,
                            uint16_t *f16, uint8_t *c8, int32_t *col_sum, const float2 *part,
                            int npart, float *inv_out, float *zero_out, int *status,
                            int num_sms, cudaStream_t st, int conv_zero,
                            int32_t *code_zero_out) {
  const int opr = cols / 8;
  if (cols % 8 || opr > kFwdMaxThreads) return FQT_EUNSUPPORTED;
  int rpi = 512 / opr;  // about 512 threads: two CTAs per SM
  if (rpi < 1) rpi = 1;
  const int nth = ((rpi * opr + 31) / 32) * 32;
  const int64_t groups = (rows + rpi - 1) / rpi;
  int64_t grid = (int64_t)num_sms * (kFwdMaxThreads * 2 / nth >= 2 ? 2 : 1) * 4;
  const int64_t need = (groups + kFwdUnroll - 1) / kFwdUnroll;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  const size_t smem = (size_t)cols * sizeof(int);
  if (bf16)
    k_fwd_codes<__nv_bfloat16><<<(int)grid, nth, smem, st>>>(
        reinterpret_cast<const __nv_bfloat16 *>(X), rows, cols, rpi, f16, c8, col_sum, part,
        npart, inv_out, zero_out, bits, status, conv_zero, code_zero_out);
  else
    k_fwd_codes<float><<<(int)grid, nth, smem, st>>>(
        reinterpret_cast<const float *>(X), rows, cols, rpi, f16, c8, col_sum, part, npart,
        inv_out, zero_out, bits, status, conv_zero, code_zero_out);
  return cuda_fail(cudaGetLastError(), "forward codes launch");
}

// ---------------------------------------------------------------------------
// Column sums of the implicit im2col matrix of a conv operand (stride 1):
// im2col column (ky, kx, ch) holds, for every output pixel (n, oy, ox), the
// code of input pixel (oy + ky - pad, ox + kx - pad) or the code of 0.0 in
// the padding.  With carriers a = code - 2^(b-1), the sum is the carriers
// over the input rectangle that tap (ky, kx) reads, plus 2^(b-1) for each of
// its n_valid entries and code(0) for each of the rows - n_valid padding
// entries.  One CTA per (tap, image) sums its rectangle (the carriers are in
// L2 after the codes pass) and adds into the column sums, which the range
// pass cleared; code(0) sits after them.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_conv_colsum(const uint16_t *__restrict__ f16, int h,
                                                     int w, int c, int kh, int kw, int pad,
                                                     int oh, int ow, int64_t nimg, int centre,
                                                     int32_t *col_sum) {
  extern __shared__ int acc_s[];  // c
  const int taps = kh * kw;
  const int tap = (int)(blockIdx.x % taps);
  const int64_t img = blockIdx.x / taps;
  const int ky = tap / kw, kx = tap - ky * kw;
  const int y0 = max(0, ky - pad), y1 = min(h, ky - pad + oh);
  const int x0 = max(0, kx - pad), x1 = min(w, kx - pad + ow);
  const int octs = c / 8;
  for (int i = threadIdx.x; i < c; i += blockDim.x) acc_s[i] = 0;
  __syncthreads();
  const int lanes = blockDim.x >= octs ? blockDim.x / octs : 1;
  const int rw = x1 - x0, npix = (y1 > y0 && rw > 0) ? (y1 - y0) * rw : 0;
  for (int oc = threadIdx.x % octs; oc < octs; oc += blockDim.x) {
    const int pl = blockDim.x >= octs ? (int)threadIdx.x / octs : 0;
    if (pl >= lanes) continue;
    int a8[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int p = pl; p < npix; p += lanes) {
      const int y = y0 + p / rw, x = x0 + p % rw;
      const uint4 v = __ldg(reinterpret_cast<const uint4 *>(
          f16 + ((img * h + y) * (int64_t)w + x) * c + oc * 8));
      const uint32_t wds[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const __half2 hh = *reinterpret_cast<const __half2 *>(&wds[q]);
        const float2 f = __half22float2(hh);
        a8[2 * q] += (int)f.x;
        a8[2 * q + 1] += (int)f.y;
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (a8[j]) atomicAdd(&acc_s[oc * 8 + j], a8[j]);
  }
  __syncthreads();
  const int zc = col_sum[(int64_t)taps * c];
  const int64_t rows = nimg * oh * ow, nvalid = nimg * (int64_t)npix;
  const int base = img == 0 ? (int)(nvalid * centre + (rows - nvalid) * (int64_t)zc) : 0;
  for (int i = threadIdx.x; i < c; i += blockDim.x) {
    const int v = acc_s[i] + base;
    if (v) atomicAdd(&col_sum[(int64_t)tap * c + i], v);
  }
}

// The same sums in one pass when the border classes fit shared memory.  Tap
// (ky, kx) reads the input rows [max(0, ky - pad), min(h, ky - pad + oh));
// for stride 1 every tap reads all rows but some of the top and bottom m =
// kh - 1 - pad ones (columns alike, mw = kw - 1 - pad).  So each input pixel
// falls in one of (2m + 1)(2mw + 1) classes: its row is one of the m top
// rows, one of the m bottom rows or inside, its column likewise.  A CTA takes
// a contiguous range of the n h w pixels (across rows and images: the column
// sums run over all images), adds the inside pixels' carriers in registers
// (most of them) and the border pixels' into shared memory by class, and
// then adds each tap's share, the classes whose row and column the tap
// reads, into the column sums.  Reads are 16 bytes per thread, six in
// flight.
constexpr int kConvMaxClasses = 25;
constexpr int kConvUnroll = 6;

__device__ __forceinline__ int conv_class(int y, int m, int h) {
  return y < m ? y : (y >= h - m ? 2 * m - (h - 1 - y) : m);
}

// the one input row (column) of border class r, or -1 for the inside class
__device__ __forceinline__ int conv_class_row(int r, int m, int h) {
  return r < m ? r : (r > m ? h - 1 - (2 * m - r) : -1);
}

__global__ void __launch_bounds__(256, 3) k_conv_colsum1(const uint16_t *__restrict__ f16, int h,
                                                      int w, int c, int kh, int kw, int pad,
                                                      int oh, int ow, int64_t nimg, int centre,
                                                      int64_t px_per_cta, int32_t *col_sum) {
  extern __shared__ int cls_s[];  // classes x c
  const int m = max(0, kh - 1 - pad), mw = max(0, kw - 1 - pad);
  const int cc = 2 * mw + 1, ncls = (2 * m + 1) * cc, inner = m * cc + mw;
  const int64_t npx = nimg * h * (int64_t)w;
  const int64_t p0 = (int64_t)blockIdx.x * px_per_cta;
  const int64_t p1 = min(npx, p0 + px_per_cta);
  for (int i = threadIdx.x; i < ncls * c; i += blockDim.x) cls_s[i] = 0;
  __syncthreads();
  const int octs = c / 8;
  const int lanes = blockDim.x >= octs ? blockDim.x / octs : 1;
  const int pl = blockDim.x >= octs ? (int)threadIdx.x / octs : 0;
  for (int oc = threadIdx.x % octs; oc < octs && pl < lanes; oc += blockDim.x) {
    int acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    uint32_t pk[4] = {0u, 0u, 0u, 0u};  // inside pixels, two lanes v + 512 a word
    int npk = 0;
    auto flush = [&]() {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        acc[2 * q] += (int)(pk[q] & 0xFFFFu) - 512 * npk;
        acc[2 * q + 1] += (int)(pk[q] >> 16) - 512 * npk;
        pk[q] = 0u;
      }
      npk = 0;
    };
    int64_t p = p0 + pl;
    int y = (int)((p / w) % h), x = (int)(p % w);
    while (p < p1) {
      uint4 v[kConvUnroll];
      int py[kConvUnroll], px[kConvUnroll];
#pragma unroll
      for (int u = 0; u < kConvUnroll; ++u) {
        py[u] = y;
        px[u] = x;
        v[u] = make_uint4(0u, 0u, 0u, 0u);
        if (p < p1)
          v[u] = __ldg(reinterpret_cast<const uint4 *>(f16 + p * c + oc * 8));
        else
          py[u] = -1;
        p += lanes;
        x += lanes;
        while (x >= w) {
          x -= w;
          if (++y == h) y = 0;
        }
      }
#pragma unroll
      for (int u = 0; u < kConvUnroll; ++u) {
        if (py[u] < 0) continue;
        const uint32_t t[4] = {carrier_lanes(v[u].x), carrier_lanes(v[u].y),
                               carrier_lanes(v[u].z), carrier_lanes(v[u].w)};
        const int k = conv_class(py[u], m, h) * cc + conv_class(px[u], mw, w);
        if (k == inner) {
#pragma unroll
          for (int q = 0; q < 4; ++q) pk[q] += t[q];
          if (++npk == kLaneAdds) flush();
        } else {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int lo = (int)(t[q] & 0xFFFFu) - 512, hi = (int)(t[q] >> 16) - 512;
            if (lo) atomicAdd(&cls_s[k * c + oc * 8 + 2 * q], lo);
            if (hi) atomicAdd(&cls_s[k * c + oc * 8 + 2 * q + 1], hi);
          }
        }
      }
    }
    flush();
    // lanes of a warp that share a channel oct add up by shuffles first
    const bool shfl_ok = octs <= 32 && (32 % octs) == 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      int v = acc[j];
      if (shfl_ok) {
        for (int off = octs; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if ((int)(threadIdx.x & 31) >= octs) v = 0;
      }
      if (v) atomicAdd(&cls_s[inner * c + oc * 8 + j], v);
    }
  }
  __syncthreads();
  const int taps = kh * kw;
  const int zc = col_sum[(int64_t)taps * c];
  const int64_t rows = nimg * oh * ow;
  for (int i = threadIdx.x; i < taps * c; i += blockDim.x) {
    const int t = i / c, ch = i - t * c, ky = t / kw, kx = t - ky * kw;
    const int y0 = max(0, ky - pad), y1 = min(h, ky - pad + oh);
    const int x0 = max(0, kx - pad), x1 = min(w, kx - pad + ow);
    int v = 0;
    for (int ry = 0; ry < 2 * m + 1; ++ry) {
      const int yr = conv_class_row(ry, m, h);
      if (yr >= 0 && (yr < y0 || yr >= y1)) continue;
      for (int rx = 0; rx < cc; ++rx) {
        const int xr = conv_class_row(rx, mw, w);
        if (xr >= 0 && (xr < x0 || xr >= x1)) continue;
        v += cls_s[(ry * cc + rx) * c + ch];
      }
    }
    if (blockIdx.x == 0) {
      const int ry = y1 - y0, rx = x1 - x0;
      const int64_t nvalid = nimg * (int64_t)(ry > 0 && rx > 0 ? ry * rx : 0);
      v += (int)(nvalid * centre + (rows - nvalid) * (int64_t)zc);
    }
    if (v) atomicAdd(&col_sum[i], v);
  }
}

fqt_status launch_conv_colsum(const uint16_t *f16, int64_t n, int h, int w, int c, int kh,
                              int kw, int pad, int bits, int32_t *col_sum, cudaStream_t st) {
  const int oh = h + 2 * pad - kh + 1, ow = w + 2 * pad - kw + 1;
  if (n <= 0) return FQT_OK;
  const int m = std::max(0, kh - 1 - pad), mw = std::max(0, kw - 1 - pad);
  const int ncls = (2 * m + 1) * (2 * mw + 1);
  if (ncls <= kConvMaxClasses && h > 2 * m && w > 2 * mw &&
      (size_t)ncls * c * sizeof(int) <= 48 * 1024) {
    // about 32 loads of 16 bytes per thread, at most three CTAs per SM (each
    // CTA adds taps x c sums into the column sums once)
    const int64_t npx = n * h * (int64_t)w, octs = c / 8;
    const int64_t want = (npx * octs + 256 * 32 - 1) / (256 * 32);
    const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(want, 3 * device_sm_count()));
    const int64_t per = (npx + grid - 1) / grid;
    k_conv_colsum1<<<(int)((npx + per - 1) / per), 256, sizeof(int) * (size_t)ncls * c, st>>>(
        f16, h, w, c, kh, kw, pad, oh, ow, n, 1 << (bits - 1), per, col_sum);
    return cuda_fail(cudaGetLastError(), "conv column sums launch");
  }
  const int64_t grid = n * kh * kw;
  if (grid > 0x7fffffff) return FQT_EUNSUPPORTED;
  k_conv_colsum<<<(int)grid, 256, sizeof(int) * (size_t)c, st>>>(
      f16, h, w, c, kh, kw, pad, oh, ow, n, 1 << (bits - 1), col_sum);
  return cuda_fail(cudaGetLastError(), "conv column sums launch");
}

// ---------------------------------------------------------------------------
// Offsets of the BHQ grad_X epilogue.  Each row's offset 2^(b-1) + z' is
// split into an integer m (which the epilogue folds into the exact integer
// product) and a fraction d, |d| <= 1/2.  With a the centred codes, w the
// centred codes of W~ and y = 2^(bw-1) + z_w,
//   (a + m + d)(w + y) summed over c = [P + m CWc] + y R + d U,
//   P = a w, CWc_j = sum_c w_cj, R_i = sum_c (a_ic + m_i), U_j = CWc_j + C y
// (Eq. 9).  The reflection of Sec. 4.2 is linear in the rows, so the epilogue
// needs hz = Q_blk d and hr = Q_blk R, reflected here in float-float, one
// thread per row, a block of rows inside one CTA.
// ---------------------------------------------------------------------------
constexpr int kOffThreads = 128;

__global__ void __launch_bounds__(kOffThreads)
    k_bhq_offsets(const float *__restrict__ zero, const int32_t *__restrict__ rsum,
                  const int32_t *__restrict__ lead, float *hz, float *hr, int64_t N,
                  int C, int oa, int nb) {
  __shared__ float2 ds[kOffThreads];
  __shared__ long long Rs[kOffThreads];
  const int t = threadIdx.x;
  const int64_t r0 = (int64_t)blockIdx.x * kOffThreads;
  const int64_t k = r0 + t;
  const bool kv = k < N;
  ff d = {0.0f, 0.0f};
  long long R = 0;
  if (kv) {
    const ff x = two_sum((float)oa, zero[k]);
    const float m = rintf(x.h);  // the epilogue rounds the same fp32 sum
    d = fast_two_sum(__fsub_rn(x.h, m), x.l);
    R = (long long)rsum[k] - (long long)C * oa + (long long)C * (long long)m;
  }
  ds[t] = make_float2(d.h, d.l);
  Rs[t] = R;
  __syncthreads();
  if (!kv) return;
  const int base = (t / nb) * nb;  // nb divides kOffThreads: blocks stay in the CTA
  const int64_t kb = r0 + base;
  const int nact = (int)min((int64_t)nb, N - kb);
  if (nact < 2) {  // a one-row block is not transformed
    hz[k] = ff_round(d);
    hr[k] = ff_round(ff_from_int(R));
    return;
  }
  const int p = lead[kb / nb];
  ff sd = {0.0f, 0.0f};
  long long sR = 0;
  for (int l = 0; l < nact; ++l) {
    sd = ff_add(sd, {ds[base + l].x, ds[base + l].y});
    sR += Rs[base + l];
  }
  const HhConst c = hh_const(nact);
  // (Q v)_k = v_k - kappa (rho sum(v) - v_p) off the lead row; rho sum(v) on it
  const ff rsd = ff_mul(c.rho, sd);
  const ff rsR = ff_mul(c.rho, ff_from_int(sR));
  if (t - base == p) {
    hz[k] = ff_round(rsd);
    hr[k] = ff_round(rsR);
    return;
  }
  const ff wd = ff_add(rsd, ff_neg({ds[base + p].x, ds[base + p].y}));
  const ff wR = ff_add(rsR, ff_neg(ff_from_int(Rs[base + p])));
  hz[k] = ff_round(ff_add(d, ff_neg(ff_mul(c.kap, wd))));
  hr[k] = ff_round(ff_add(ff_from_int(R), ff_neg(ff_mul(c.kap, wR))));
}

cudaError_t launch_bhq_offsets(const float *zero, const int32_t *rsum,
                               const int32_t *lead, float *hz, float *hr, int64_t N,
                               int C, int bits, int block, cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  const int64_t grid = (N + kOffThreads - 1) / kOffThreads;
  k_bhq_offsets<<<(unsigned)grid, kOffThreads, 0, st>>>(zero, rsum, lead, hz, hr, N, C,
                                                        1 << (bits - 1), block);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
static int pow2ceil(int v) {
  int p = 1;
  while (p < v) p <<= 1;
  return p;
}

size_t quant_smem_bytes(const QuantArgs &a) {
  const size_t chunk_cols = (size_t)a.TW * a.OPT * 8;
  size_t b = sizeof(float2) * 32 + sizeof(float) * 32 + sizeof(int) * 32;
  b += sizeof(int) * a.C;
  b += sizeof(float) * 8 * a.G;
  if (a.kind == KIND_BHQ) {
    b += sizeof(float2) * a.G * a.block;
    b += sizeof(float) * a.G * a.C;
    b += sizeof(float) * a.G * a.RL * chunk_cols;
  }
  return b;
}

// Chooses the thread mapping of k_quant for an N x C problem: TW threads per
// row, each holding OPT <= 4 octs per pass; nchunk passes cover long rows.
fqt_status quant_geometry(QuantArgs &a, int num_sms, int *nth_out,
                          int *grid_out, size_t *smem_out) {
  const int C = a.C;
  if (C <= 0 || C % 8) return FQT_EUNSUPPORTED;
  const int CO = C / 8;
  a.CO = CO;
  int opt = CO < kMaxOct ? CO : kMaxOct;
  int TW = pow2ceil((CO + opt - 1) / opt);
  const int rows_per_unit = a.kind == KIND_BHQ ? a.block : 1;
  // a group (one BHQ block, or one row) may use at most 1024 threads
  while ((int64_t)TW * rows_per_unit > 1024 && TW > 1) TW >>= 1;
  if ((int64_t)TW * rows_per_unit > 1024) return FQT_EUNSUPPORTED;
  opt = (CO + TW - 1) / TW;
  if (opt > kMaxOct) opt = kMaxOct;
  const int nchunk = (CO + TW * opt - 1) / (TW * opt);
  if (nchunk > 1 && a.kind != KIND_BHQ) return FQT_EUNSUPPORTED;
  a.TW = TW;
  a.OPT = opt;
  a.RPL = 1;
  a.nchunk = nchunk;
  int nth;
  if (a.kind == KIND_BHQ) {
    a.RL = a.block;
    a.GT = a.RL * TW;
    nth = a.GT < 256 ? 256 : a.GT;
    a.G = nth / a.GT;
    a.unit_rows = a.block;
    a.n_units = (a.N + a.block - 1) / a.block;
  } else {
    nth = TW < 256 ? 256 : TW;
    a.RL = nth / TW;
    a.GT = nth;
    a.G = 1;
    a.unit_rows = a.RL;
    a.n_units = (a.N + a.RL - 1) / a.RL;
  }
  const size_t smem = quant_smem_bytes(a);
  if (smem > 200 * 1024) return FQT_EUNSUPPORTED;
  const int per_sm = nth <= 256 ? 4 : 1;
  const int64_t need = (a.n_units + a.G - 1) / a.G;
  int64_t grid = (int64_t)num_sms * per_sm;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  *nth_out = nth;
  *grid_out = (int)grid;
  *smem_out = smem;
  return FQT_OK;
}

// Geometry of the staged kernel; FQT_EUNSUPPORTED sends the call to k_quant.
fqt_status quant2_geometry(QuantArgs &a, bool bf16, int num_sms, int *grid_out,
                           size_t *smem_out) {
  const int C = a.C;
  if (C <= 0 || C % 8 || a.kind == KIND_DET) return FQT_EUNSUPPORTED;
  const int CO = C / 8;
  if (CO > 32 * kMaxOct) return FQT_EUNSUPPORTED;  // rows longer than 1024
  const int esize = bf16 ? 2 : 4;
  const int LPR = CO >= 32 ? 32 : pow2ceil(CO);
  const int OPL = (CO + LPR - 1) / LPR;
  const size_t row_bytes = (size_t)C * esize;
  size_t stage = 32768;
  int U, G;
  if (a.kind == KIND_BHQ) {
    const size_t blk = (size_t)a.block * row_bytes;
    if (blk > stage) stage = (blk + 127) & ~(size_t)127;
    if (stage > 98304) return FQT_EUNSUPPORTED;
    U = (int)(stage / row_bytes / a.block) * a.block;
    G = U / a.block;
  } else {
    U = (int)(stage / row_bytes);
    G = 1;
  }
  if (U < 1) return FQT_EUNSUPPORTED;
  a.CO = CO;
  a.TW = LPR;
  a.OPT = OPL;
  a.RL = 32 / LPR;
  a.RPL = 1;
  a.GT = kQ2Threads;
  a.G = G;
  a.unit_rows = U;
  a.nchunk = 1;
  a.stage_bytes = (int)stage;
  a.n_units = (a.N + U - 1) / U;
  size_t smem = 2 * stage + 16 + sizeof(float2) * 8 + sizeof(int) * 8 +
                sizeof(int) * (size_t)C + sizeof(float2) * (size_t)U +
                sizeof(float) * 8 * (size_t)G;
  if (a.kind == KIND_BHQ) smem += sizeof(float) * (size_t)G * C;
  if (smem > 220 * 1024) return FQT_EUNSUPPORTED;
  int per_sm = (int)((220 * 1024) / smem);
  if (per_sm > 4) per_sm = 4;
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)num_sms * per_sm;
  if (grid > a.n_units) grid = a.n_units;
  if (grid < 1) grid = 1;
  *grid_out = (int)grid;
  *smem_out = smem;
  return FQT_OK;
}

template <int KIND, typename T>
static cudaError_t launch_quant2_t(const QuantArgs &a, int grid, size_t smem,
                                   cudaStream_t st) {
  auto fn = k_quant2<KIND, T>;
  cudaError_t e = cudaFuncSetAttribute(
      fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  fn<<<grid, kQ2Threads, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_quant2(const QuantArgs &a, bool bf16, int grid, size_t smem,
                          cudaStream_t st) {
  switch (a.kind * 2 + (bf16 ? 1 : 0)) {
    case KIND_PTQ * 2: return launch_quant2_t<KIND_PTQ, float>(a, grid, smem, st);
    case KIND_PTQ * 2 + 1: return launch_quant2_t<KIND_PTQ, __nv_bfloat16>(a, grid, smem, st);
    case KIND_PSQ * 2: return launch_quant2_t<KIND_PSQ, float>(a, grid, smem, st);
    case KIND_PSQ * 2 + 1: return launch_quant2_t<KIND_PSQ, __nv_bfloat16>(a, grid, smem, st);
    case KIND_BHQ * 2: return launch_quant2_t<KIND_BHQ, float>(a, grid, smem, st);
    case KIND_BHQ * 2 + 1: return launch_quant2_t<KIND_BHQ, __nv_bfloat16>(a, grid, smem, st);
  }
  return cudaErrorInvalidValue;
}

template <int KIND, typename T>
static cudaError_t launch_quant_t(const QuantArgs &a, int nth, int grid,
                                  size_t smem, cudaStream_t st) {
  auto fn = nth <= 256 ? k_quant<KIND, T, 256> : k_quant<KIND, T, 1024>;
  cudaError_t e = cudaFuncSetAttribute(
      fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  fn<<<grid, nth, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_quant(const QuantArgs &a, bool bf16, int nth, int grid,
                         size_t smem, cudaStream_t st) {
  switch (a.kind * 2 + (bf16 ? 1 : 0)) {
    case KIND_PTQ * 2: return launch_quant_t<KIND_PTQ, float>(a, nth, grid, smem, st);
    case KIND_PTQ * 2 + 1: return launch_quant_t<KIND_PTQ, __nv_bfloat16>(a, nth, grid, smem, st);
    case KIND_PSQ * 2: return launch_quant_t<KIND_PSQ, float>(a, nth, grid, smem, st);
    case KIND_PSQ * 2 + 1: return launch_quant_t<KIND_PSQ, __nv_bfloat16>(a, nth, grid, smem, st);
    case KIND_BHQ * 2: return launch_quant_t<KIND_BHQ, float>(a, nth, grid, smem, st);
    case KIND_BHQ * 2 + 1: return launch_quant_t<KIND_BHQ, __nv_bfloat16>(a, nth, grid, smem, st);
    case KIND_DET * 2: return launch_quant_t<KIND_DET, float>(a, nth, grid, smem, st);
    case KIND_DET * 2 + 1: return launch_quant_t<KIND_DET, __nv_bfloat16>(a, nth, grid, smem, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_range(const void *x, bool bf16, int64_t count, float2 *part,
                         int *npart, int32_t *z0, int64_t nz0, int32_t *z1,
                         int64_t nz1, int num_sms, cudaStream_t st) {
  const int64_t n_oct = count / 8;
  int64_t grid = (n_oct + 255) / 256;
  const int64_t cap = (int64_t)num_sms * 8;
  if (grid > cap) grid = cap;
  if (grid > kMaxRangeCtas) grid = kMaxRangeCtas;
  if (grid < 1) grid = 1;
  *npart = (int)grid;
  if (bf16)
    k_range<__nv_bfloat16><<<(int)grid, 256, 0, st>>>(
        reinterpret_cast<const __nv_bfloat16 *>(x), n_oct, part, z0, nz0, z1, nz1);
  else
    k_range<float><<<(int)grid, 256, 0, st>>>(
        reinterpret_cast<const float *>(x), n_oct, part, z0, nz0, z1, nz1);
  return cudaGetLastError();
}

}  // namespace fqt
