// fqt_group.cu -- the adaptive groups of the block Householder quantizer
// (App. D.5) and the quantizer over them.
//
// The grouping, as this library reads App. D.5:
//  * M_i = ||h_i||_inf; rows sorted by M descending, ties by row index.
//  * For G = 1 .. N-1 the first G rows are "large", one per group, and the
//    other N - G rows are "small"; group i gets size_i = (N - G) M_i / S_G
//    small rows (S_G = sum of the G large M).  The variance of the grouping
//    is estimated with App. D.4's bound per group,
//        V(G) = sum_i (M_i^(2/3) size_i^(-1/3) + L^(2/3) size_i^(2/3))^3,
//    L = M_(G+1) (no small row is larger).  With L -> 0 this is App. D.5's
//    own sum_i M_i^2 / size_i, which alone would always choose G = 1.
//    Expanding the cube, V(G) = t^3 S1 + 3 t^2 u S4/3 + 3 t u^2 S5/3 + u^3 S2
//    with t = (S1 / (N - G))^(1/3), u = L^(2/3) ((N - G) / S1)^(2/3) and
//    S_p = sum over the G large rows of M^p: prefix sums of the sorted M.
//  * G = argmin V (smallest G on ties; N = 1 gives G = 1).
//  * Integer sizes by cumulative rounding: e_0 = 0, e_G = N - G and
//    e_i = floor((N - G) (C_i / S_G) + 1/2), C_i = sum of the first i sorted
//    M; group i takes e_i - e_(i-1) small rows, dealt from the smallest up.
//  * Stored order: group after group, the lead (large) row first, then its
//    small rows in descending M.  perm[k] = row of dH stored at k; gstart[i]
//    = first stored row of group i (N for i >= G); gsize[k] = size of the
//    group of stored row k.
//
//  k_grp_keys    : M_i as a descending sort key and the first digit
//                  histogram (one CTA per tile of 4096 keys).
//  k_grp_radix   : one stable 8-bit pass of an LSD radix sort; four passes
//                  sort the 32-bit keys, ties keep the row order.
//  k_grp_tsum    : per 1024 sorted rows, the sums of M, M^(4/3), M^(5/3), M^2.
//  k_grp_choose  : prefix sums, V(G) for every G, argmin over G (the last
//                  CTA to finish reduces the per-CTA minima).
//  k_grp_layout  : sizes, perm, gstart, gsize.
//  k_bhq_groups  : BHQ of every group (Sec. 4.2, App. D.4), one warp per
//                  group, fused with the 8-bit PTQ Q_b1 of App. E.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "fqt.h"
#include "fqt_common.cuh"
#include "fqt_internal.h"

namespace fqt {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;  // keys per sort tile
constexpr int kSortTileLog = 12;
constexpr int kCntPitch = kSortThreads + 2;  // uint16 counters per digit row
constexpr size_t kCntBytes = sizeof(uint16_t) * 256 * kCntPitch;
constexpr int kScanTile = 1024;  // sorted rows per CTA of the choice kernels
constexpr int kKeysThreads = 1024;
// the sort's tile offsets are summed per CTA over all tiles: 256 tiles at most
constexpr int64_t kMaxGroupRows = (int64_t)1 << 20;

__device__ __forceinline__ float warp_max_xor(float v, int from_lanes) {
  for (int off = from_lanes >> 1; off > 0; off >>= 1)
    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// Exclusive prefix sum of one int per thread over a 256-thread CTA.
__device__ __forceinline__ int cta_excl_scan256(int v, int *wsum) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  int base = 0;
  for (int w = 0; w < warp; ++w) base += wsum[w];
  __syncthreads();
  return base + x - v;
}

// ---------------------------------------------------------------------------
// Sort keys: key = ~bits(M) orders M >= 0 descending as unsigned integers.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kKeysThreads) k_grp_keys(const T *__restrict__ h, int64_t N,
                                                            int C, int lpr, uint32_t *keys,
                                                            int32_t *vals, int32_t *hist,
                                                            int nt, unsigned *count) {
  __shared__ int cnt[256];
  const int tid = threadIdx.x;
  for (int i = tid; i < 256; i += blockDim.x) cnt[i] = 0;
  // the later passes accumulate into their histograms: clear them here
  const int64_t nclear = (int64_t)3 * nt * 256;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + tid; i < nclear;
       i += (int64_t)gridDim.x * blockDim.x)
    hist[(int64_t)nt * 256 + i] = 0;
  if (blockIdx.x == 0 && tid == 0) *count = 0u;
  __syncthreads();
  const int lane = tid & 31, warp = tid >> 5;
  const int rpw = 32 / lpr, sub = lane / lpr, o = lane - sub * lpr;
  const int octs = C / 8;
  const int64_t r0 = (int64_t)blockIdx.x * kSortTile;
  for (int rr = warp * rpw + sub; rr - sub < kSortTile; rr += (kKeysThreads / 32) * rpw) {
    const int64_t row = r0 + rr;
    float m = 0.0f;
    if (rr < kSortTile && row < N) {
      for (int c8 = o; c8 < octs; c8 += lpr) {
        float x[8];
        load_oct(h + row * C + c8 * 8, x);
#pragma unroll
        for (int j = 0; j < 8; ++j) m = fmaxf(m, fabsf(x[j]));
      }
    }
    m = warp_max_xor(m, lpr);
    if (o == 0 && rr < kSortTile && row < N) {
      const uint32_t key = ~__float_as_uint(m);
      keys[row] = key;
      vals[row] = (int32_t)row;
      atomicAdd(&cnt[key & 255u], 1);
    }
  }
  __syncthreads();
  for (int i = tid; i < 256; i += blockDim.x) hist[(int64_t)blockIdx.x * 256 + i] = cnt[i];
}

// ---------------------------------------------------------------------------
// One stable pass over digit (key >> shift) & 255.  Thread t holds keys
// t*16 .. t*16+15 of its tile (tile order = thread-major), counts its digits
// into column t of a 256 x 256 counter table, and a digit-major scan of the
// table gives every key its rank in the tile.  The tile's global offsets
// come from the histograms of all tiles (digit start + earlier tiles).  The
// next pass's histogram is accumulated from the output positions.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kSortThreads) k_grp_radix(
    const uint32_t *__restrict__ kin, const int32_t *__restrict__ vin, uint32_t *kout,
    int32_t *vout, int64_t N, int nt, int shift, const int32_t *__restrict__ hcur,
    int32_t *hnext) {
  extern __shared__ uint16_t cnt[];
  __shared__ int wsum[kSortThreads / 32];
  __shared__ int gbase[256];
  const int tid = threadIdx.x;
  const int64_t i0 = (int64_t)blockIdx.x * kSortTile + (int64_t)tid * kSortItems;
  uint32_t k[kSortItems];
  int32_t v[kSortItems];
  if (i0 + kSortItems <= N) {
#pragma unroll
    for (int q = 0; q < kSortItems / 4; ++q) {
      const uint4 a = __ldg(reinterpret_cast<const uint4 *>(kin + i0) + q);
      const int4 b = __ldg(reinterpret_cast<const int4 *>(vin + i0) + q);
      k[4 * q] = a.x; k[4 * q + 1] = a.y; k[4 * q + 2] = a.z; k[4 * q + 3] = a.w;
      v[4 * q] = b.x; v[4 * q + 1] = b.y; v[4 * q + 2] = b.z; v[4 * q + 3] = b.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < kSortItems; ++i) {
      k[i] = i0 + i < N ? kin[i0 + i] : 0u;
      v[i] = i0 + i < N ? vin[i0 + i] : 0;
    }
  }
  for (int d = 0; d < 256; ++d) cnt[d * kCntPitch + tid] = 0;
#pragma unroll
  for (int i = 0; i < kSortItems; ++i)
    if (i0 + i < N) ++cnt[((k[i] >> shift) & 255u) * kCntPitch + tid];
  __syncthreads();
  // thread d: the row of digit d
  int tot = 0;
  for (int t = 0; t < kSortThreads; ++t) tot += cnt[tid * kCntPitch + t];
  const int dstart = cta_excl_scan256(tot, wsum);
  int pre = 0, all = 0;
  for (int b = 0; b < nt; ++b) {
    const int hv = __ldg(hcur + (int64_t)b * 256 + tid);
    all += hv;
    if (b < (int)blockIdx.x) pre += hv;
  }
  const int dglob = cta_excl_scan256(all, wsum);
  int run = dstart;
  for (int t = 0; t < kSortThreads; ++t) {
    const int c = cnt[tid * kCntPitch + t];
    cnt[tid * kCntPitch + t] = (uint16_t)run;
    run += c;
  }
  gbase[tid] = dglob + pre - dstart;
  __syncthreads();
#pragma unroll
  for (int i = 0; i < kSortItems; ++i) {
    if (i0 + i >= N) continue;
    const uint32_t d = (k[i] >> shift) & 255u;
    const int r = cnt[d * kCntPitch + tid];
    cnt[d * kCntPitch + tid] = (uint16_t)(r + 1);
    const int64_t pos = (int64_t)gbase[d] + r;
    if (pos < 0 || pos >= N) continue;  // unreachable with consistent histograms
    kout[pos] = k[i];
    vout[pos] = v[i];
    if (hnext) atomicAdd(&hnext[(pos >> kSortTileLog) * 256 + ((k[i] >> (shift + 8)) & 255u)], 1);
  }
}

__device__ __forceinline__ double key_m(uint32_t key) {
  return (double)__uint_as_float(~key);
}

// Sums of M^p (p = 1, 4/3, 5/3, 2) over one thread's 4 sorted rows.
__device__ __forceinline__ void pow_terms(double M, double (&a)[4]) {
  const double c = cbrt(M);
  a[0] = M;
  a[1] = M * c;
  a[2] = M * c * c;
  a[3] = M * M;
}

// Sum over a 256-thread CTA in a fixed order (deterministic).
__device__ __forceinline__ double cta_sum256(double v, double *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double s = 0.0;
  for (int w = 0; w < 8; ++w) s += red[w];
  __syncthreads();
  return s;
}

__global__ void __launch_bounds__(256) k_grp_tsum(const uint32_t *__restrict__ keys, int64_t N,
                                                  double *tsum) {
  __shared__ double red[8];
  const int64_t i0 = (int64_t)blockIdx.x * kScanTile + threadIdx.x * 4;
  double s[4] = {0.0, 0.0, 0.0, 0.0};
  for (int e = 0; e < 4; ++e) {
    if (i0 + e >= N) break;
    double a[4];
    pow_terms(key_m(keys[i0 + e]), a);
    for (int q = 0; q < 4; ++q) s[q] += a[q];
  }
  for (int q = 0; q < 4; ++q) {
    const double t = cta_sum256(s[q], red);
    if (threadIdx.x == 0) tsum[(int64_t)blockIdx.x * 4 + q] = t;
  }
}

// Exclusive prefix over a 256-thread CTA of one double per thread.
__device__ __forceinline__ double cta_excl_scan256d(double v, double *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  double x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const double y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) red[warp] = x;
  __syncthreads();
  double base = 0.0;
  for (int w = 0; w < warp; ++w) base += red[w];
  __syncthreads();
  return base + (x - v);
}

struct Best {
  double v;
  long long g;
};

__device__ __forceinline__ bool better(double v, long long g, double bv, long long bg) {
  return v < bv || (v == bv && g < bg);
}

__global__ void __launch_bounds__(256) k_grp_choose(const uint32_t *__restrict__ keys, int64_t N,
                                                    const double *__restrict__ tsum, double *cincl,
                                                    double2 *best, long long *Gout, double *SGout,
                                                    unsigned *count) {
  __shared__ double red[8];
  __shared__ double bv_s[8];
  __shared__ long long bg_s[8];
  __shared__ int last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x;
  // sums over the earlier tiles
  double base[4];
  for (int q = 0; q < 4; ++q) {
    double p = 0.0;
    for (int bb = tid; bb < b; bb += 256) p += tsum[(int64_t)bb * 4 + q];
    base[q] = cta_sum256(p, red);
  }
  const int64_t i0 = (int64_t)b * kScanTile + tid * 4;
  double loc[4][4];
  double tot[4] = {0.0, 0.0, 0.0, 0.0};
  double Mv[5];
  for (int e = 0; e < 5; ++e) Mv[e] = i0 + e < N ? key_m(keys[i0 + e]) : 0.0;
  for (int e = 0; e < 4; ++e) {
    double a[4] = {0.0, 0.0, 0.0, 0.0};
    if (i0 + e < N) pow_terms(Mv[e], a);
    for (int q = 0; q < 4; ++q) {
      tot[q] += a[q];
      loc[e][q] = tot[q];
    }
  }
  double off[4];
  for (int q = 0; q < 4; ++q) off[q] = cta_excl_scan256d(tot[q], red);
  double bv = INFINITY;
  long long bg = 0x7fffffffffffffffll;
  for (int e = 0; e < 4; ++e) {
    const int64_t i = i0 + e;
    if (i >= N) break;
    double S[4];
    for (int q = 0; q < 4; ++q) S[q] = base[q] + off[q] + loc[e][q];
    cincl[i] = S[0];
    if (i + 1 >= N) break;  // G = N is not a candidate
    const long long G = i + 1;
    const double nG = (double)(N - G), L = Mv[e + 1];
    double V = 0.0;
    if (S[0] > 0.0) {
      const double t3 = S[0] / nG;
      const double t = cbrt(t3);
      const double cl = cbrt(L), r = cbrt(nG / S[0]);
      const double u = cl * cl * r * r;
      V = t3 * S[0] + 3.0 * t * t * u * S[1] + 3.0 * t * u * u * S[2] + u * u * u * S[3];
    }
    if (better(V, G, bv, bg)) {
      bv = V;
      bg = G;
    }
  }
  __threadfence();  // cincl is read by the last CTA
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const double ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const long long og = __shfl_xor_sync(0xffffffffu, bg, o);
    if (better(ov, og, bv, bg)) {
      bv = ov;
      bg = og;
    }
  }
  if (lane == 0) {
    bv_s[warp] = bv;
    bg_s[warp] = bg;
  }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < 8; ++w)
      if (better(bv_s[w], bg_s[w], bv, bg)) {
        bv = bv_s[w];
        bg = bg_s[w];
      }
    best[b] = make_double2(bv, (double)bg);
    __threadfence();
    last = atomicAdd(count, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last || tid != 0) return;
  __threadfence();
  double fv = INFINITY;
  long long fg = 0x7fffffffffffffffll;
  for (int bb = 0; bb < (int)gridDim.x; ++bb) {
    const double2 x = __ldcg(best + bb);
    if (better(x.x, (long long)x.y, fv, fg)) {
      fv = x.x;
      fg = (long long)x.y;
    }
  }
  if (fg < 1 || fg >= N) fg = 1;  // N = 1: one group
  *Gout = fg;
  *SGout = __ldcg(cincl + fg - 1);
  *count = 0u;
}

__device__ __forceinline__ int64_t cum_size(int64_t j, int64_t N, int64_t G, double SG,
                                            const double *cincl) {
  if (j <= 0) return 0;
  if (j >= G) return N - G;
  if (!(SG > 0.0)) return 0;
  const double q = (double)(N - G) * (cincl[j - 1] / SG);
  int64_t e = (int64_t)floor(q + 0.5);
  if (e < 0) e = 0;
  if (e > N - G) e = N - G;
  return e;
}

__global__ void __launch_bounds__(256) k_grp_layout(const int32_t *__restrict__ vals, int64_t N,
                                                    const double *__restrict__ cincl,
                                                    const long long *Gp, const double *SGp,
                                                    int32_t *perm, int32_t *gstart,
                                                    int32_t *gsize) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i > N) return;
  const int64_t G = *Gp;
  if (i >= G) {
    gstart[i] = (int32_t)N;
    return;
  }
  const double SG = *SGp;
  const int64_t e0 = cum_size(i, N, G, SG, cincl);
  int64_t e1 = cum_size(i + 1, N, G, SG, cincl);
  if (e1 < e0) e1 = e0;
  const int64_t k0 = i + e0, ns = e1 - e0;
  gstart[i] = (int32_t)k0;
  perm[k0] = vals[i];
  for (int64_t t = 0; t < ns; ++t) perm[k0 + 1 + t] = vals[N - e1 + t];
  for (int64_t t = 0; t <= ns; ++t) gsize[k0 + t] = (int32_t)(ns + 1);
}

// ---------------------------------------------------------------------------
// Quantizer over the groups: a warp per group, RS = 32 / LPR rows per step
// (LPR lanes per row, 8 columns per lane).  Pass 1 reads the rows for the
// lead row's range, lambda2 and the column sums of the small rows; pass 2
// re-reads them (L2) for the transform, the row minima, SR and packing; the
// grad_X offsets hz, hr are reflected at the end (see k_bhq_warp).
// ---------------------------------------------------------------------------
template <int LPR>
__device__ __forceinline__ float2 row_minmax(float2 v) {
#pragma unroll
  for (int off = LPR >> 1; off > 0; off >>= 1) {
    v.x = fminf(v.x, __shfl_xor_sync(0xffffffffu, v.x, off));
    v.y = fmaxf(v.y, __shfl_xor_sync(0xffffffffu, v.y, off));
  }
  return v;
}
template <int LPR>
__device__ __forceinline__ float row_min(float v) {
#pragma unroll
  for (int off = LPR >> 1; off > 0; off >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}
template <int LPR>
__device__ __forceinline__ int row_add(int v) {
#pragma unroll
  for (int off = LPR >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}
// across the rows of a step (lanes with the same column offset)
template <int LPR>
__device__ __forceinline__ float sub_add(float v) {
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}
template <int LPR>
__device__ __forceinline__ float sub_max(float v) {
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}
template <int LPR>
__device__ __forceinline__ int sub_addi(int v) {
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

template <typename T, int LPR>
__global__ void __launch_bounds__(256, 2) k_bhq_groups(const QuantArgs a) {
  __shared__ float2 red[8];
  __shared__ int redi[8];
  extern __shared__ int csum_s[];  // C column sums of Q_b1
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int CO = LPR, RS = 32 / LPR, C = 8 * LPR;
  const int sub = lane / LPR, o = lane - sub * LPR;
  const int64_t N = a.N;
  const T *h = reinterpret_cast<const T *>(a.h);

  // ---- global range (Q_b1 scale) from the range-pass partials ----
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
  const uint32_t og2 = (B2 + 1u) >> 1;
  const float s_g1 = affine_scale(gmin, gmax, 255u);
  const float s_g1_16 = __fmul_rn(s_g1, 65536.0f);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  if (blockIdx.x == 0 && tid == 0 && has_b1) {
    a.inv1[0] = __fdiv_rn(1.0f, s_g1);
    a.zero1[0] = __fmul_rn(s_g1, gmin);
  }
  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];
  int cs[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) cs[j] = 0;
  bool badp = false;

  const int64_t wstride = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t gi = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp; gi < N; gi += wstride) {
    const int64_t k0 = __ldg(a.gstart + gi);
    if (k0 >= N) break;  // groups past G are empty and gstart does not decrease
    int64_t k1 = __ldg(a.gstart + gi + 1);
    if (k1 > N) k1 = N;
    if (k1 <= k0) continue;
    const int nb = (int)(k1 - k0);

    // ---- pass 1: lead row, lambda2, column sums of the small rows ----
    float xl[8], csm[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) xl[j] = csm[j] = 0.0f;
    float pmin = 0.0f, pmax = 0.0f, l2 = 0.0f;
    for (int r0 = 0; r0 < nb; r0 += RS) {
      const int r = r0 + sub;
      const bool v = r < nb;
      int64_t src = v ? (int64_t)__ldg(a.perm + k0 + r) : 0;
      if (src < 0 || src >= N) {
        badp = true;
        src = 0;
      }
      float x[8];
      if (v) {
        load_oct(h + src * C + o * 8, x);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) x[j] = 0.0f;
      }
      float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        mm.x = fminf(mm.x, x[j]);
        mm.y = fmaxf(mm.y, x[j]);
      }
      mm = row_minmax<LPR>(mm);
      if (v) {
        if (r == 0) {
          pmin = mm.x;
          pmax = mm.y;
#pragma unroll
          for (int j = 0; j < 8; ++j) xl[j] = x[j];
        } else {
          l2 = fmaxf(l2, fmaxf(fabsf(mm.x), fabsf(mm.y)));
#pragma unroll
          for (int j = 0; j < 8; ++j) csm[j] += x[j];
        }
      }
    }
    pmin = __shfl_sync(0xffffffffu, pmin, 0);
    pmax = __shfl_sync(0xffffffffu, pmax, 0);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      xl[j] = __shfl_sync(0xffffffffu, xl[j], o);
      csm[j] = sub_add<LPR>(csm[j]);
    }
    l2 = sub_max<LPR>(l2);
    const float lam2 = 2.0f * l2;
    const float np = fmaxf(fabsf(pmin), fabsf(pmax));
    // ---- group scalars s1, s2 (App. D.4) and the reflection ----
    float s1f = 0.0f, s2f = 0.0f, rho = 0.0f, kap = 0.0f;
    if (np > 0.0f) {
      float lam1 = __fsub_rn(pmax, pmin);
      if (!(lam1 > 0.0f)) lam1 = 2.0f * np;
      const float Nf = (float)nb;
      if (lam2 > 0.0f) {
        const float c1 = cbrtf(lam1), c2 = cbrtf(lam2);
        const float n3 = cbrtf(Nf), n6 = sqrtf(n3);
        const float den = c1 * c1 / n3 + c2 * c2 * n3 * n3;
        s1f = (float)B2 * n6 / (c1 * den);
        s2f = (float)B2 * n6 / (c2 * den);
      } else {
        s1f = (float)B2 * sqrtf(Nf) / lam1;
      }
      if (nb > 1) {
        rho = 1.0f / sqrtf(Nf);
        kap = 1.0f / (1.0f - rho);
      }
    }
    // w_j = sum_k e_k s_k h_kj, e_lead = kap (rho - 1), e_small = kap rho
    const float el = kap * (rho - 1.0f), es = kap * rho;
    float w[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      w[j] = fmaf(es, __fmul_rn(s2f, csm[j]), el * __fmul_rn(s1f, xl[j]));

    // ---- pass 2: transform, row minimum, rounding, packing, sums ----
    ff sd = {0.0f, 0.0f};
    long long sR = 0;
    float dp = 0.0f;
    long long Rp = 0;
    for (int r0 = 0; r0 < nb; r0 += RS) {
      const int r = r0 + sub;
      const bool v = r < nb;
      int64_t src = v ? (int64_t)__ldg(a.perm + k0 + r) : 0;
      if (src < 0 || src >= N) src = 0;
      float x[8];
      if (v) {
        load_oct(h + src * C + o * 8, x);
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) x[j] = 0.0f;
      }
      const bool lead = r == 0;
      const float sk = lead ? s1f : s2f;
      const float ck = lead ? rho - 1.0f : rho;
      float t[8];
      float tmin = INFINITY;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        t[j] = fmaf(-ck, w[j], __fmul_rn(sk, x[j]));
        tmin = fminf(tmin, t[j]);
      }
      const float z2 = row_min<LPR>(tmin);
      const int64_t row = k0 + r;
      uint32_t c[8];
      int rs2 = 0, rs1 = 0;
      if (v) {
        const uint4 w2 = philox_oct((uint64_t)row * (uint64_t)CO + (uint64_t)o, 0u, key);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          c[j] = sr_code16(__fmul_rn(__fsub_rn(t[j], z2), 65536.0f), u16_of(w2, j), B2);
          rs2 += (int)c[j];
        }
        if (a.c2) store_codes8(a.c2 + row * (int64_t)C + o * 8, c);
        if (a.f2) store_carriers8(a.f2 + row * (int64_t)C + o * 8, c, og2);
        if (has_b1) {
          const uint4 w1 = philox_oct((uint64_t)src * (uint64_t)CO + (uint64_t)o, 1u, key);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float vv = __fmul_rn(__fsub_rn(x[j], gmin), s_g1_16);
            c[j] = sr_code16(vv, u16_of(w1, j), 255u);
            rs1 += (int)c[j];
            cs[j] += (int)c[j];
          }
          if (a.c1) store_codes8(a.c1 + src * (int64_t)C + o * 8, c);
          if (a.f1) store_carriers8(a.f1 + src * (int64_t)C + o * 8, c, 128u);
        }
      }
      rs2 = row_add<LPR>(rs2);
      if (has_b1) rs1 = row_add<LPR>(rs1);
      // the row's offset split 2^(b-1) + z' = m + d, R = sum_c (a + m)
      const ff xo = two_sum((float)og2, z2);
      const float m = rintf(xo.h);
      const ff d = fast_two_sum(__fsub_rn(xo.h, m), xo.l);
      const long long R = (long long)rs2 - (long long)C * og2 + (long long)C * __float2ll_rn(m);
      if (v && o == 0) {
        if (a.rsum2) a.rsum2[row] = rs2;
        if (has_b1 && a.rsum1) a.rsum1[src] = rs1;
        a.inv2[row] = sk > 0.0f ? __fdiv_rn(1.0f, sk) : 0.0f;
        a.zero2[row] = z2;
        if (a.hz) {
          a.hz[row] = ff_round(d);
          a.hr[row] = (float)R;
        }
        sd = ff_add(sd, d);
        sR += R;
        if (lead) {
          dp = ff_round(d);
          Rp = R;
        }
      }
    }
    if (a.hz && nb >= 2) {
      // group sums of d (float-float) and R over the lanes that added them
#pragma unroll
      for (int off = LPR; off < 32; off <<= 1) {
        const ff od = {__shfl_xor_sync(0xffffffffu, sd.h, off),
                       __shfl_xor_sync(0xffffffffu, sd.l, off)};
        sd = ff_add(sd, od);
        sR += __shfl_xor_sync(0xffffffffu, sR, off);
      }
      sd.h = __shfl_sync(0xffffffffu, sd.h, 0);
      sd.l = __shfl_sync(0xffffffffu, sd.l, 0);
      sR = __shfl_sync(0xffffffffu, sR, 0);
      dp = __shfl_sync(0xffffffffu, dp, 0);
      Rp = __shfl_sync(0xffffffffu, Rp, 0);
      __syncwarp();  // every row's unreflected d, R is in hz, hr
      const HhConst hcst = hh_const(nb);
      const ff rsd = ff_mul(hcst.rho, sd);
      const ff rsR = ff_mul(hcst.rho, ff_from_int(sR));
      const ff wd = ff_add(rsd, {-dp, 0.0f});
      const ff wR = ff_add(rsR, ff_neg(ff_from_int(Rp)));
      const ff kd = ff_mul(hcst.kap, wd), kR = ff_mul(hcst.kap, wR);
      for (int r = lane; r < nb; r += 32) {
        const int64_t row = k0 + r;
        if (r == 0) {
          a.hz[row] = ff_round(rsd);
          a.hr[row] = ff_round(rsR);
        } else {
          const float dr = a.hz[row], Rr = a.hr[row];
          a.hz[row] = ff_round(ff_add({dr, 0.0f}, ff_neg(kd)));
          a.hr[row] = ff_round(ff_add({Rr, 0.0f}, ff_neg(kR)));
        }
      }
      __syncwarp();
    }
  }
  if (__any_sync(0xffffffffu, badp) && lane == 0) record_status(a.status, FQT_EINVAL);
  // ---- column sums of Q_b1 ----
  if (has_b1 && a.csum1) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int v = sub_addi<LPR>(cs[j]);
      if (sub == 0 && v) atomicAdd(&csum_s[o * 8 + j], v);
    }
    __syncthreads();
    for (int i = tid; i < C; i += blockDim.x)
      if (csum_s[i]) atomicAdd(&a.csum1[i], csum_s[i]);
  }
}

struct GroupScratch {
  uint32_t *k0, *k1;
  int32_t *v0, *v1;
  int32_t *hist;
  double *tsum, *cincl;
  double2 *best;
  long long *G;
  double *SG;
  unsigned *count;
};

size_t carve(char *base, int64_t N, GroupScratch *s) {
  const int64_t nt = (N + kSortTile - 1) / kSortTile;
  const int64_t ntc = (N + kScanTile - 1) / kScanTile;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char *p = base ? base + off : nullptr;
    off += (bytes + 255) & ~(size_t)255;
    return p;
  };
  const size_t nk = (size_t)(nt * kSortTile);
  char *k0 = take(nk * 4), *k1 = take(nk * 4), *v0 = take(nk * 4), *v1 = take(nk * 4);
  char *hist = take((size_t)4 * nt * 256 * 4);
  char *tsum = take((size_t)ntc * 4 * 8);
  char *cincl = take((size_t)N * 8 + 8);
  char *best = take((size_t)ntc * 16);
  char *G = take(8), *SG = take(8), *count = take(8);
  if (s) {
    s->k0 = reinterpret_cast<uint32_t *>(k0);
    s->k1 = reinterpret_cast<uint32_t *>(k1);
    s->v0 = reinterpret_cast<int32_t *>(v0);
    s->v1 = reinterpret_cast<int32_t *>(v1);
    s->hist = reinterpret_cast<int32_t *>(hist);
    s->tsum = reinterpret_cast<double *>(tsum);
    s->cincl = reinterpret_cast<double *>(cincl);
    s->best = reinterpret_cast<double2 *>(best);
    s->G = reinterpret_cast<long long *>(G);
    s->SG = reinterpret_cast<double *>(SG);
    s->count = reinterpret_cast<unsigned *>(count);
  }
  return off;
}

}  // namespace

size_t group_workspace_bytes(int64_t N) { return N > 0 ? carve(nullptr, N, nullptr) : 0; }

fqt_status launch_bhq_grouping(const void *dH, bool bf16, int64_t N, int C, int32_t *perm,
                               int32_t *gstart, int32_t *gsize, void *scratch,
                               size_t scratch_bytes, cudaStream_t st) {
  if (N <= 0) return FQT_OK;
  if (N > kMaxGroupRows) return FQT_EUNSUPPORTED;
  GroupScratch s;
  if (carve(nullptr, N, nullptr) > scratch_bytes) return FQT_EWORKSPACE;
  carve(static_cast<char *>(scratch), N, &s);
  const int nt = (int)((N + kSortTile - 1) / kSortTile);
  const int ntc = (int)((N + kScanTile - 1) / kScanTile);
  int lpr = 1;
  while (lpr < 32 && lpr < C / 8) lpr <<= 1;
  if (bf16)
    k_grp_keys<__nv_bfloat16><<<nt, kKeysThreads, 0, st>>>(
        static_cast<const __nv_bfloat16 *>(dH), N, C, lpr, s.k0, s.v0, s.hist, nt, s.count);
  else
    k_grp_keys<float><<<nt, kKeysThreads, 0, st>>>(static_cast<const float *>(dH), N, C, lpr,
                                                    s.k0, s.v0, s.hist, nt, s.count);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "grouping keys launch");
  e = cudaFuncSetAttribute(k_grp_radix, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kCntBytes);
  if (e != cudaSuccess) return cuda_fail(e, "radix smem attribute");
  uint32_t *kin = s.k0, *kout = s.k1;
  int32_t *vin = s.v0, *vout = s.v1;
  for (int p = 0; p < 4; ++p) {
    int32_t *hc = s.hist + (int64_t)p * nt * 256;
    int32_t *hn = p < 3 ? hc + (int64_t)nt * 256 : nullptr;
    k_grp_radix<<<nt, kSortThreads, kCntBytes, st>>>(kin, vin, kout, vout, N, nt, 8 * p, hc, hn);
    uint32_t *tk = kin;
    kin = kout;
    kout = tk;
    int32_t *tv = vin;
    vin = vout;
    vout = tv;
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "radix sort launch");
  // after four passes the sorted keys are back in k0 / v0
  k_grp_tsum<<<ntc, 256, 0, st>>>(kin, N, s.tsum);
  k_grp_choose<<<ntc, 256, 0, st>>>(kin, N, s.tsum, s.cincl, s.best, s.G, s.SG, s.count);
  k_grp_layout<<<(int)((N + 1 + 255) / 256), 256, 0, st>>>(vin, N, s.cincl, s.G, s.SG, perm,
                                                             gstart, gsize);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "grouping choice launch");
  return FQT_OK;
}

fqt_status launch_bhq_groups(QuantArgs &a, bool bf16, int num_sms, cudaStream_t st) {
  if (a.C % 8) return FQT_EUNSUPPORTED;
  const int CO = a.C / 8;
  if (CO != 8 && CO != 16 && CO != 32) return FQT_EUNSUPPORTED;
  const int grid = num_sms * 2;
  const size_t smem = sizeof(int) * (size_t)a.C;
#define FQT_BG(L)                                                                      \
  if (CO == L) {                                                                       \
    if (bf16)                                                                          \
      k_bhq_groups<__nv_bfloat16, L><<<grid, 256, smem, st>>>(a);                      \
    else                                                                               \
      k_bhq_groups<float, L><<<grid, 256, smem, st>>>(a);                              \
  }
  FQT_BG(8)
  FQT_BG(16)
  FQT_BG(32)
#undef FQT_BG
  return cuda_fail(cudaGetLastError(), "BHQ group quantizer launch");
}

}  // namespace fqt
