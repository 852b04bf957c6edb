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
// keys per sort tile: 1024 (4 per thread) up to 2^17 rows, else 4096
__host__ __device__ constexpr int sort_ipt(int64_t N) { return N <= ((int64_t)1 << 17) ? 4 : 16; }
constexpr int kScanTile = 1024;  // sorted rows per CTA of the choice kernels
constexpr int kKeysThreads = 1024;
// Groups of more than kBigGroup rows are quantized by a CTA each.  Group
// sizes follow the sorted norms (non-increasing up to the rounding), so
// every such group has an index below N / kBigGroup + 1.
constexpr int kBigGroup = 64;
__host__ __device__ inline int64_t big_grid(int64_t N) { return N / kBigGroup + 1; }
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
                                                            int C, int lpr, int tile,
                                                            uint32_t *keys, int32_t *vals,
                                                            int32_t *hist, int nt,
                                                            unsigned *count) {
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
  const int64_t r0 = (int64_t)blockIdx.x * tile;
  for (int rr = warp * rpw + sub; rr - sub < tile; rr += (kKeysThreads / 32) * rpw) {
    const int64_t row = r0 + rr;
    float m = 0.0f;
    if (rr < tile && row < N) {
      for (int c8 = o; c8 < octs; c8 += lpr) {
        float x[8];
        load_oct(h + row * C + c8 * 8, x);
#pragma unroll
        for (int j = 0; j < 8; ++j) m = fmaxf(m, fabsf(x[j]));
      }
    }
    m = warp_max_xor(m, lpr);
    if (o == 0 && rr < tile && row < N) {
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
// One stable pass over digit (key >> shift) & 255 of a tile of 256 * IPT
// keys.  Thread t holds the keys at tile positions i * 256 + t (i < IPT), so
// the tile order is (i, warp, lane).  Per round i every warp ranks its 32
// keys among equal digits with match.any and counts them per digit; a
// digit-major scan of the (round, warp) counts gives each key its place in
// the tile.  The tile's global offsets come from the histograms of all
// tiles (digit start + earlier tiles).  The next pass's histogram is
// accumulated from the output positions.
// ---------------------------------------------------------------------------
template <int IPT>
__global__ void __launch_bounds__(kSortThreads) k_grp_radix(
    const uint32_t *__restrict__ kin, const int32_t *__restrict__ vin, uint32_t *kout,
    int32_t *vout, int64_t N, int nt, int shift, const int32_t *__restrict__ hcur,
    int32_t *hnext) {
  constexpr int T = kSortThreads * IPT;
  constexpr int W = kSortThreads / 32;
  extern __shared__ uint16_t cnt_s[];  // [IPT][W][256] counts, then offsets
  auto cnt = [&](int i, int w, int d) -> uint16_t & { return cnt_s[(i * W + w) * 256 + d]; };
  __shared__ int wsum[W];
  __shared__ int gbase[256];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t t0 = (int64_t)blockIdx.x * T;
  for (int e = tid; e < IPT * W * 256; e += kSortThreads) cnt_s[e] = 0;
  uint32_t k[IPT];
  int32_t v[IPT];
  int rk[IPT];
#pragma unroll
  for (int i = 0; i < IPT; ++i) {
    const int64_t idx = t0 + i * kSortThreads + tid;
    k[i] = idx < N ? __ldg(kin + idx) : 0u;
    v[i] = idx < N ? __ldg(vin + idx) : 0;
  }
  __syncthreads();
  const unsigned lt = (1u << lane) - 1u;
#pragma unroll
  for (int i = 0; i < IPT; ++i) {
    const bool ok = t0 + i * kSortThreads + tid < N;
    const uint32_t d = ok ? (k[i] >> shift) & 255u : 256u + lane;
    const unsigned peers = __match_any_sync(0xffffffffu, d);
    rk[i] = __popc(peers & lt);
    if (ok && (peers & lt) == 0u) cnt(i, warp, d) = (uint16_t)__popc(peers);
  }
  __syncthreads();
  // thread d: running offsets of digit d over (round, warp), its total
  int run = 0;
#pragma unroll
  for (int i = 0; i < IPT; ++i)
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const int c = cnt(i, w, tid);
      cnt(i, w, tid) = (uint16_t)run;
      run += c;
    }
  // digit d over all tiles and over the earlier ones: 16 loads in flight
  int pre = 0, all = 0;
  int b = 0;
  for (; b + 16 <= nt; b += 16) {
    int hv[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) hv[q] = __ldg(hcur + (int64_t)(b + q) * 256 + tid);
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      all += hv[q];
      if (b + q < (int)blockIdx.x) pre += hv[q];
    }
  }
  for (; b < nt; ++b) {
    const int hv = __ldg(hcur + (int64_t)b * 256 + tid);
    all += hv;
    if (b < (int)blockIdx.x) pre += hv;
  }
  const int dglob = cta_excl_scan256(all, wsum);
  gbase[tid] = dglob + pre;
  __syncthreads();
#pragma unroll
  for (int i = 0; i < IPT; ++i) {
    const bool ok = t0 + i * kSortThreads + tid < N;
    const uint32_t d = (k[i] >> shift) & 255u;
    int64_t pos = ok ? (int64_t)gbase[d] + cnt(i, warp, d) + rk[i] : -1;
    if (pos >= N) pos = -1;  // unreachable with consistent histograms
    if (pos >= 0) {
      kout[pos] = k[i];
      vout[pos] = v[i];
    }
    if (hnext) {
      const uint32_t key2 = pos >= 0 ? (uint32_t)((pos / T) * 256 + ((k[i] >> (shift + 8)) & 255u))
                                     : 0xFFFFFFFFu - lane;
      const unsigned peers = __match_any_sync(0xffffffffu, key2);
      if (pos >= 0 && (peers & lt) == 0u) atomicAdd(&hnext[key2], __popc(peers));
    }
  }
}

__device__ __forceinline__ float key_m(uint32_t key) { return __uint_as_float(~key); }

// ---------------------------------------------------------------------------
// The estimate V(G) is evaluated in float-float (about 2^-46 relative, on the
// fp32 pipe; fp64 is a narrow pipe on this part).  Candidate estimates differ
// by far more than that on real data; the decision is as precise as a
// double-precision evaluation with the same summation order would be.
// ---------------------------------------------------------------------------
__device__ __forceinline__ ff ff_sub(ff a, ff b) { return ff_add(a, ff_neg(b)); }

// 1 / x for x > 0: fp32 reciprocal and one correction in float-float.
__device__ __forceinline__ ff ff_rcp(ff x) {
  const float y0 = __frcp_rn(x.h);
  const ff p = ff_mul(x, {y0, 0.0f});
  const float e = __fsub_rn(__fsub_rn(1.0f, p.h), p.l);
  return fast_two_sum(y0, __fmul_rn(y0, e));
}

// x^(1/3) for x >= 0: fp32 cube root and one Newton correction.
__device__ __forceinline__ ff ff_cbrt(ff x) {
  if (!(x.h > 0.0f)) return {0.0f, 0.0f};
  const float c0 = cbrtf(x.h);
  const ff c3 = ff_mul(two_prod(c0, c0), {c0, 0.0f});
  const ff r = ff_sub(x, c3);
  return fast_two_sum(c0, __fdiv_rn(r.h, __fmul_rn(3.0f, __fmul_rn(c0, c0))));
}

// M, M^(4/3), M^(5/3), M^2 of one row.
__device__ __forceinline__ void pow_terms(float M, ff (&a)[4]) {
  const ff c = ff_cbrt({M, 0.0f});
  a[0] = {M, 0.0f};
  a[1] = ff_mul({M, 0.0f}, c);
  a[2] = ff_mul(a[1], c);
  a[3] = two_prod(M, M);
}

__device__ __forceinline__ ff shfl_xor_ff(ff v, int off) {
  return {__shfl_xor_sync(0xffffffffu, v.h, off), __shfl_xor_sync(0xffffffffu, v.l, off)};
}

// Sum over a 256-thread CTA in a fixed order (deterministic).
__device__ __forceinline__ ff cta_sum256(ff v, ff *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = ff_add(v, shfl_xor_ff(v, off));
  if (lane == 0) red[warp] = v;
  __syncthreads();
  ff s = {0.0f, 0.0f};
  for (int w = 0; w < 8; ++w) s = ff_add(s, red[w]);
  __syncthreads();
  return s;
}

__global__ void __launch_bounds__(256) k_grp_tsum(const uint32_t *__restrict__ keys, int64_t N,
                                                  ff *tsum) {
  __shared__ ff red[8];
  const int64_t i0 = (int64_t)blockIdx.x * kScanTile + threadIdx.x * 4;
  ff s[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
  for (int e = 0; e < 4; ++e) {
    if (i0 + e >= N) break;
    ff a[4];
    pow_terms(key_m(keys[i0 + e]), a);
    for (int q = 0; q < 4; ++q) s[q] = ff_add(s[q], a[q]);
  }
  for (int q = 0; q < 4; ++q) {
    const ff t = cta_sum256(s[q], red);
    if (threadIdx.x == 0) tsum[(int64_t)blockIdx.x * 4 + q] = t;
  }
}

// Exclusive prefix over a 256-thread CTA of one float-float per thread.
__device__ __forceinline__ ff cta_excl_scan256ff(ff v, ff *red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  ff x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const ff y = {__shfl_up_sync(0xffffffffu, x.h, off), __shfl_up_sync(0xffffffffu, x.l, off)};
    if (lane >= off) x = ff_add(x, y);
  }
  if (lane == 31) red[warp] = x;
  __syncthreads();
  ff base = {0.0f, 0.0f};
  for (int w = 0; w < warp; ++w) base = ff_add(base, red[w]);
  __syncthreads();
  return ff_add(base, ff_sub(x, v));
}

__device__ __forceinline__ bool better(ff v, long long g, ff bv, long long bg) {
  return v.h < bv.h || (v.h == bv.h && (v.l < bv.l || (v.l == bv.l && g < bg)));
}

struct BestFF {
  float h, l;
  long long g;
};

__global__ void __launch_bounds__(256) k_grp_choose(const uint32_t *__restrict__ keys, int64_t N,
                                                    const ff *__restrict__ tsum, ff *cincl,
                                                    BestFF *best, long long *Gout, ff *SGout,
                                                    unsigned *count) {
  __shared__ ff red[8];
  __shared__ ff bv_s[8];
  __shared__ long long bg_s[8];
  __shared__ int last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int b = blockIdx.x;
  // sums over the earlier tiles
  ff base[4];
  for (int q = 0; q < 4; ++q) {
    ff p = {0.0f, 0.0f};
    for (int bb = tid; bb < b; bb += 256) p = ff_add(p, tsum[(int64_t)bb * 4 + q]);
    base[q] = cta_sum256(p, red);
  }
  const int64_t i0 = (int64_t)b * kScanTile + tid * 4;
  ff loc[4][4];
  ff tot[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
  float Mv[5];
  for (int e = 0; e < 5; ++e) Mv[e] = i0 + e < N ? key_m(keys[i0 + e]) : 0.0f;
  for (int e = 0; e < 4; ++e) {
    ff a[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
    if (i0 + e < N) pow_terms(Mv[e], a);
    for (int q = 0; q < 4; ++q) {
      tot[q] = ff_add(tot[q], a[q]);
      loc[e][q] = tot[q];
    }
  }
  ff off[4];
  for (int q = 0; q < 4; ++q) off[q] = ff_add(base[q], cta_excl_scan256ff(tot[q], red));
  ff bv = {INFINITY, 0.0f};
  long long bg = 0x7fffffffffffffffll;
  for (int e = 0; e < 4; ++e) {
    const int64_t i = i0 + e;
    if (i >= N) break;
    ff S[4];
    for (int q = 0; q < 4; ++q) S[q] = ff_add(off[q], loc[e][q]);
    cincl[i] = S[0];
    if (i + 1 >= N) break;  // G = N is not a candidate
    const long long G = i + 1;
    const float nG = (float)(N - G);  // exact: N <= 2^20
    ff V = {0.0f, 0.0f};
    if (S[0].h > 0.0f) {
      const ff t3 = ff_mul(S[0], ff_rcp({nG, 0.0f}));  // t^3 = S1 / (N - G)
      const ff t = ff_cbrt(t3);
      const ff cl = ff_cbrt({Mv[e + 1], 0.0f});
      const ff r = ff_rcp(t);
      const ff u = ff_mul(ff_mul(cl, cl), ff_mul(r, r));  // L^(2/3) ((N-G)/S1)^(2/3)
      const ff tu = ff_mul(t, u);
      V = ff_mul(t3, S[0]);
      V = ff_add(V, ff_mul(ff_mul({3.0f, 0.0f}, ff_mul(t, tu)), S[1]));
      V = ff_add(V, ff_mul(ff_mul({3.0f, 0.0f}, ff_mul(tu, u)), S[2]));
      V = ff_add(V, ff_mul(ff_mul(ff_mul(u, u), u), S[3]));
    }
    if (better(V, G, bv, bg)) {
      bv = V;
      bg = G;
    }
  }
  __threadfence();  // cincl is read by the last CTA
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const ff ov = shfl_xor_ff(bv, o);
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
    best[b] = BestFF{bv.h, bv.l, bg};
    __threadfence();
    last = atomicAdd(count, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last || tid != 0) return;
  __threadfence();
  ff fv = {INFINITY, 0.0f};
  long long fg = 0x7fffffffffffffffll;
  for (int bb = 0; bb < (int)gridDim.x; ++bb) {
    const volatile BestFF *x = best + bb;
    const ff xv = {x->h, x->l};
    const long long xg = x->g;
    if (better(xv, xg, fv, fg)) {
      fv = xv;
      fg = xg;
    }
  }
  if (fg < 1 || fg >= N) fg = 1;  // N = 1: one group
  *Gout = fg;
  const volatile ff *cg = cincl + fg - 1;
  *SGout = ff{cg->h, cg->l};
  *count = 0u;
}

// e_j of the cumulative rounding, in fp64 (two divisions per group) so that
// exact ties (equal rows) round as in a double-precision evaluation.
__device__ __forceinline__ int64_t cum_size(int64_t j, int64_t N, int64_t G, double SG,
                                            const ff *cincl) {
  if (j <= 0) return 0;
  if (j >= G) return N - G;
  if (!(SG > 0.0)) return 0;
  const ff c = cincl[j - 1];
  const double q = (double)(N - G) * (((double)c.h + (double)c.l) / SG);
  int64_t e = (int64_t)floor(q + 0.5);
  if (e < 0) e = 0;
  if (e > N - G) e = N - G;
  return e;
}

__global__ void __launch_bounds__(256) k_grp_layout(const int32_t *__restrict__ vals, int64_t N,
                                                    const ff *__restrict__ cincl,
                                                    const long long *Gp, const ff *SGp,
                                                    int32_t *perm, int32_t *gstart,
                                                    int32_t *gsize, unsigned *slots) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) *slots = 0u;
  if (i > N) return;
  const int64_t G = *Gp;
  if (i >= G) {
    gstart[i] = (int32_t)N;
    return;
  }
  const double SG = (double)SGp->h + (double)SGp->l;
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
// grad_X offsets hz, hr are reflected at the end (see k_bhq_team).
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
__global__ void __launch_bounds__(256, 3) k_bhq_groups(const QuantArgs a) {
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

  // One row per sub-warp for a slot of RS single-row groups: BHQ of one row
  // is lambda2 = 0, s1 = B / R(h), no reflection (App. D.4 with N = 1).
  auto do_singles = [&](int64_t k0) {
    const int64_t row = k0 + sub;
    int64_t src = __ldg(a.perm + row);
    if (src < 0 || src >= N) {
      badp = true;
      src = 0;
    }
    float x[8];
    load_oct(h + src * C + o * 8, x);
    float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      mm.x = fminf(mm.x, x[j]);
      mm.y = fmaxf(mm.y, x[j]);
    }
    mm = row_minmax<LPR>(mm);
    const float np = fmaxf(fabsf(mm.x), fabsf(mm.y));
    float s1f = 0.0f;
    if (np > 0.0f) {
      float lam1 = __fsub_rn(mm.y, mm.x);
      if (!(lam1 > 0.0f)) lam1 = 2.0f * np;
      s1f = (float)B2 * sqrtf(1.0f) / lam1;
    }
    float t[8];
    float tmin = INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      t[j] = __fmul_rn(s1f, x[j]);
      tmin = fminf(tmin, t[j]);
    }
    const float z2 = row_min<LPR>(tmin);
    uint32_t c[8];
    int rs2 = 0, rs1 = 0;
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
    rs2 = row_add<LPR>(rs2);
    if (has_b1) rs1 = row_add<LPR>(rs1);
    if (o == 0) {
      if (a.rsum2) a.rsum2[row] = rs2;
      if (has_b1 && a.rsum1) a.rsum1[src] = rs1;
      a.inv2[row] = s1f > 0.0f ? __fdiv_rn(1.0f, s1f) : 0.0f;
      a.zero2[row] = z2;
      if (a.hz) {
        const ff xo = two_sum((float)og2, z2);
        const float m = rintf(xo.h);
        const ff d = fast_two_sum(__fsub_rn(xo.h, m), xo.l);
        a.hz[row] = ff_round(d);
        // R = sum_c (a + m); C is a power of two, so C m is exact
        a.hr[row] = ff_round(two_sum((float)(rs2 - C * (int)og2), __fmul_rn((float)C, m)));
      }
    }
  };

  // A warp takes slots of RS consecutive groups from a queue: all single
  // rows -> one step; otherwise the groups one after another, a warp each.
  for (;;) {
    unsigned slot = 0u;
    if (lane == 0) slot = atomicAdd(a.slots, 1u);
    const int64_t g0 = (int64_t)__shfl_sync(0xffffffffu, slot, 0) * RS;
    if (g0 >= N) break;
    const int64_t gk = g0 + (lane < RS ? lane : 0);
    const int64_t ka = gk < N ? __ldg(a.gstart + gk) : N;
    const int64_t kb = gk < N ? __ldg(a.gstart + gk + 1) : N;
    const int64_t s0 = __shfl_sync(0xffffffffu, ka, 0);
    if (s0 >= N) break;  // groups past G are empty and gstart does not decrease
    if (__all_sync(0xffffffffu, lane >= RS || (ka < N && kb == ka + 1))) {
      do_singles(s0);
      continue;
    }
  for (int gs = 0; gs < RS; ++gs) {
    const int64_t gi = g0 + gs;
    if (gi >= N) break;
    const int64_t k0 = __ldg(a.gstart + gi);
    if (k0 >= N) break;
    int64_t k1 = __ldg(a.gstart + gi + 1);
    if (k1 > N) k1 = N;
    if (k1 <= k0) continue;
    const int nb = (int)(k1 - k0);
    // groups of more than kBigGroup rows get a whole CTA (k_bhq_groups_big)
    if (nb > kBigGroup && gi < big_grid(N)) continue;

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
    ff sd = {0.0f, 0.0f}, sR = {0.0f, 0.0f}, Rp = {0.0f, 0.0f};
    float dp = 0.0f;
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
      // R = sum_c (a + m); C is a power of two, so C m is exact
      const ff R = two_sum((float)(rs2 - C * (int)og2), __fmul_rn((float)C, m));
      if (v && o == 0) {
        if (a.rsum2) a.rsum2[row] = rs2;
        if (has_b1 && a.rsum1) a.rsum1[src] = rs1;
        a.inv2[row] = sk > 0.0f ? __fdiv_rn(1.0f, sk) : 0.0f;
        a.zero2[row] = z2;
        if (a.hz) {
          a.hz[row] = ff_round(d);
          a.hr[row] = ff_round(R);
        }
        sd = ff_add(sd, d);
        sR = ff_add(sR, R);
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
        const ff oR = {__shfl_xor_sync(0xffffffffu, sR.h, off),
                       __shfl_xor_sync(0xffffffffu, sR.l, off)};
        sd = ff_add(sd, od);
        sR = ff_add(sR, oR);
      }
      sd.h = __shfl_sync(0xffffffffu, sd.h, 0);
      sd.l = __shfl_sync(0xffffffffu, sd.l, 0);
      sR.h = __shfl_sync(0xffffffffu, sR.h, 0);
      sR.l = __shfl_sync(0xffffffffu, sR.l, 0);
      dp = __shfl_sync(0xffffffffu, dp, 0);
      Rp.h = __shfl_sync(0xffffffffu, Rp.h, 0);
      Rp.l = __shfl_sync(0xffffffffu, Rp.l, 0);
      __syncwarp();  // every row's unreflected d, R is in hz, hr
      const HhConst hcst = hh_const(nb);
      const ff rsd = ff_mul(hcst.rho, sd);
      const ff rsR = ff_mul(hcst.rho, sR);
      const ff wd = ff_add(rsd, {-dp, 0.0f});
      const ff wR = ff_add(rsR, ff_neg(Rp));
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

// ---------------------------------------------------------------------------
// BHQ of one large group per CTA: the eight warps split the group's rows in
// every pass (RS rows per warp step), and the column sums of the small rows,
// lambda2, and the group sums of the offsets d and R go through shared
// memory in a fixed order.  Same arithmetic as k_bhq_groups.
// ---------------------------------------------------------------------------
template <typename T, int LPR>
__global__ void __launch_bounds__(256) k_bhq_groups_big(const QuantArgs a) {
  constexpr int CO = LPR, RS = 32 / LPR, C = 8 * LPR, NW = 8;
  __shared__ float2 red[NW];
  __shared__ int redi[NW];
  __shared__ float col_s[NW][C];   // per-warp column sums, then lead row / w
  __shared__ float lead_s[C];
  __shared__ float misc_s[NW][4];  // l2, pmin, pmax per warp
  __shared__ ff sd_s[NW], sR_s[NW];
  __shared__ float dp_s;
  __shared__ ff Rp_s;
  extern __shared__ int csum_s[];  // C column sums of Q_b1
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int sub = lane / LPR, o = lane - sub * LPR;
  const int64_t N = a.N;
  const int64_t gi = blockIdx.x;
  if (gi >= N) return;
  const int64_t k0 = __ldg(a.gstart + gi);
  if (k0 >= N) return;
  int64_t k1 = __ldg(a.gstart + gi + 1);
  if (k1 > N) k1 = N;
  if (k1 - k0 <= kBigGroup) return;
  const int nb = (int)(k1 - k0);
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
  for (int w = 1; w < NW; ++w) {
    gmin = fminf(gmin, red[w].x);
    gmax = fmaxf(gmax, red[w].y);
    bad |= redi[w];
  }
  if (bad) return;  // k_bhq_groups records the status
  const uint32_t B2 = (1u << a.bits) - 1u;
  const uint32_t og2 = (B2 + 1u) >> 1;
  const float s_g1 = affine_scale(gmin, gmax, 255u);
  const float s_g1_16 = __fmul_rn(s_g1, 65536.0f);
  const bool has_b1 = a.c1 != nullptr || a.f1 != nullptr;
  PhiloxKeys key;
#pragma unroll
  for (int i = 0; i < 20; ++i) key.k[i] = a.round_keys[i];
  bool badp = false;

  // ---- pass 1: lead row, lambda2, column sums of the small rows ----
  float csm[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) csm[j] = 0.0f;
  float l2 = 0.0f;
  for (int r0 = warp * RS; r0 < nb; r0 += NW * RS) {
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
#pragma unroll
        for (int j = 0; j < 8; ++j) lead_s[o * 8 + j] = x[j];
        if (o == 0) {
          misc_s[0][1] = mm.x;
          misc_s[0][2] = mm.y;
        }
      } else {
        l2 = fmaxf(l2, fmaxf(fabsf(mm.x), fabsf(mm.y)));
#pragma unroll
        for (int j = 0; j < 8; ++j) csm[j] += x[j];
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) csm[j] = sub_add<LPR>(csm[j]);
  l2 = sub_max<LPR>(l2);
  if (sub == 0) {
#pragma unroll
    for (int j = 0; j < 8; ++j) col_s[warp][o * 8 + j] = csm[j];
  }
  if (lane == 0) misc_s[warp][0] = l2;
  __syncthreads();
  // reduce over the warps in a fixed order
  l2 = 0.0f;
  for (int w = 0; w < NW; ++w) l2 = fmaxf(l2, misc_s[w][0]);
  const float pmin = misc_s[0][1], pmax = misc_s[0][2];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    float sacc = 0.0f;
    for (int w = 0; w < NW; ++w) sacc += col_s[w][o * 8 + j];
    csm[j] = sacc;
  }
  float xl[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) xl[j] = lead_s[o * 8 + j];
  const float lam2 = 2.0f * l2;
  const float np = fmaxf(fabsf(pmin), fabsf(pmax));
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
    rho = 1.0f / sqrtf(Nf);
    kap = 1.0f / (1.0f - rho);
  }
  const float el = kap * (rho - 1.0f), es = kap * rho;
  float w[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) w[j] = fmaf(es, __fmul_rn(s2f, csm[j]), el * __fmul_rn(s1f, xl[j]));

  // ---- pass 2: transform, row minimum, rounding, packing, sums ----
  ff sd = {0.0f, 0.0f}, sR = {0.0f, 0.0f};
  int cs[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) cs[j] = 0;
  for (int r0 = warp * RS; r0 < nb; r0 += NW * RS) {
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
    const ff xo = two_sum((float)og2, z2);
    const float m = rintf(xo.h);
    const ff d = fast_two_sum(__fsub_rn(xo.h, m), xo.l);
    const ff R = two_sum((float)(rs2 - C * (int)og2), __fmul_rn((float)C, m));
    if (v && o == 0) {
      if (a.rsum2) a.rsum2[row] = rs2;
      if (has_b1 && a.rsum1) a.rsum1[src] = rs1;
      a.inv2[row] = sk > 0.0f ? __fdiv_rn(1.0f, sk) : 0.0f;
      a.zero2[row] = z2;
      if (a.hz) {
        a.hz[row] = ff_round(d);
        a.hr[row] = ff_round(R);
      }
      sd = ff_add(sd, d);
      sR = ff_add(sR, R);
      if (lead) {
        dp_s = ff_round(d);
        Rp_s = R;
      }
    }
  }
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) {
    const ff od = {__shfl_xor_sync(0xffffffffu, sd.h, off), __shfl_xor_sync(0xffffffffu, sd.l, off)};
    const ff oR = {__shfl_xor_sync(0xffffffffu, sR.h, off), __shfl_xor_sync(0xffffffffu, sR.l, off)};
    sd = ff_add(sd, od);
    sR = ff_add(sR, oR);
  }
  if (lane == 0) {
    sd_s[warp] = sd;
    sR_s[warp] = sR;
  }
  // ---- column sums of Q_b1 ----
  if (has_b1 && a.csum1) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int v = sub_addi<LPR>(cs[j]);
      if (sub == 0 && v) atomicAdd(&csum_s[o * 8 + j], v);
    }
  }
  __syncthreads();  // hz, hr of every row are in global memory; sums in shared
  if (a.hz) {
    sd = {0.0f, 0.0f};
    sR = {0.0f, 0.0f};
    for (int w2 = 0; w2 < NW; ++w2) {
      sd = ff_add(sd, sd_s[w2]);
      sR = ff_add(sR, sR_s[w2]);
    }
    const HhConst hcst = hh_const(nb);
    const ff rsd = ff_mul(hcst.rho, sd);
    const ff rsR = ff_mul(hcst.rho, sR);
    const ff wd = ff_add(rsd, {-dp_s, 0.0f});
    const ff wR = ff_add(rsR, ff_neg(Rp_s));
    const ff kd = ff_mul(hcst.kap, wd), kR = ff_mul(hcst.kap, wR);
    for (int r = tid; r < nb; r += blockDim.x) {
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
  }
  if (__any_sync(0xffffffffu, badp) && lane == 0) record_status(a.status, FQT_EINVAL);
  if (has_b1 && a.csum1)
    for (int i = tid; i < C; i += blockDim.x)
      if (csum_s[i]) atomicAdd(&a.csum1[i], csum_s[i]);
}

struct GroupScratch {
  uint32_t *k0, *k1;
  int32_t *v0, *v1;
  int32_t *hist;
  ff *tsum, *cincl;
  BestFF *best;
  long long *G;
  ff *SG;
  unsigned *count;
  unsigned *slots;  // work queue of the group quantizer
};

size_t carve(char *base, int64_t N, GroupScratch *s) {
  const int tile = kSortThreads * sort_ipt(N);
  const int64_t nt = (N + tile - 1) / tile;
  const int64_t ntc = (N + kScanTile - 1) / kScanTile;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char *p = base ? base + off : nullptr;
    off += (bytes + 255) & ~(size_t)255;
    return p;
  };
  const size_t nk = (size_t)(nt * tile);
  char *k0 = take(nk * 4), *k1 = take(nk * 4), *v0 = take(nk * 4), *v1 = take(nk * 4);
  char *hist = take((size_t)4 * nt * 256 * 4);
  char *tsum = take((size_t)ntc * 4 * sizeof(ff));
  char *cincl = take((size_t)N * sizeof(ff) + 8);
  char *best = take((size_t)ntc * sizeof(BestFF));
  char *G = take(8), *SG = take(8), *count = take(8), *slots = take(8);
  if (s) {
    s->k0 = reinterpret_cast<uint32_t *>(k0);
    s->k1 = reinterpret_cast<uint32_t *>(k1);
    s->v0 = reinterpret_cast<int32_t *>(v0);
    s->v1 = reinterpret_cast<int32_t *>(v1);
    s->hist = reinterpret_cast<int32_t *>(hist);
    s->tsum = reinterpret_cast<ff *>(tsum);
    s->cincl = reinterpret_cast<ff *>(cincl);
    s->best = reinterpret_cast<BestFF *>(best);
    s->G = reinterpret_cast<long long *>(G);
    s->SG = reinterpret_cast<ff *>(SG);
    s->count = reinterpret_cast<unsigned *>(count);
    s->slots = reinterpret_cast<unsigned *>(slots);
  }
  return off;
}

}  // namespace

size_t group_workspace_bytes(int64_t N) { return N > 0 ? carve(nullptr, N, nullptr) : 0; }

fqt_status launch_bhq_grouping(const void *dH, bool bf16, int64_t N, int C, int32_t *perm,
                               int32_t *gstart, int32_t *gsize, void *scratch,
                               size_t scratch_bytes, unsigned **slot_counter, cudaStream_t st) {
  if (N <= 0) return FQT_OK;
  if (N > kMaxGroupRows) return FQT_EUNSUPPORTED;
  GroupScratch s;
  if (carve(nullptr, N, nullptr) > scratch_bytes) return FQT_EWORKSPACE;
  carve(static_cast<char *>(scratch), N, &s);
  const int ipt = sort_ipt(N);
  const int tile = kSortThreads * ipt;
  const int nt = (int)((N + tile - 1) / tile);
  const int ntc = (int)((N + kScanTile - 1) / kScanTile);
  int lpr = 1;
  while (lpr < 32 && lpr < C / 8) lpr <<= 1;
  if (bf16)
    k_grp_keys<__nv_bfloat16><<<nt, kKeysThreads, 0, st>>>(
        static_cast<const __nv_bfloat16 *>(dH), N, C, lpr, tile, s.k0, s.v0, s.hist, nt,
        s.count);
  else
    k_grp_keys<float><<<nt, kKeysThreads, 0, st>>>(static_cast<const float *>(dH), N, C, lpr,
                                                    tile, s.k0, s.v0, s.hist, nt, s.count);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "grouping keys launch");
  e = cudaFuncSetAttribute(k_grp_radix<16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)(sizeof(uint16_t) * 16 * (kSortThreads / 32) * 256));
  if (e != cudaSuccess) return cuda_fail(e, "radix smem attribute");
  uint32_t *kin = s.k0, *kout = s.k1;
  int32_t *vin = s.v0, *vout = s.v1;
  for (int p = 0; p < 4; ++p) {
    int32_t *hc = s.hist + (int64_t)p * nt * 256;
    int32_t *hn = p < 3 ? hc + (int64_t)nt * 256 : nullptr;
    const size_t csm = sizeof(uint16_t) * ipt * (kSortThreads / 32) * 256;
    if (ipt == 4)
      k_grp_radix<4><<<nt, kSortThreads, csm, st>>>(kin, vin, kout, vout, N, nt, 8 * p, hc, hn);
    else
      k_grp_radix<16><<<nt, kSortThreads, csm, st>>>(kin, vin, kout, vout, N, nt, 8 * p, hc, hn);
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
                                                             gstart, gsize, s.slots);
  if (slot_counter) *slot_counter = s.slots;
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "grouping choice launch");
  return FQT_OK;
}

fqt_status launch_bhq_groups(QuantArgs &a, bool bf16, int num_sms, cudaStream_t st) {
  if (a.C % 8) return FQT_EUNSUPPORTED;
  const int CO = a.C / 8;
  if (CO != 8 && CO != 16 && CO != 32) return FQT_EUNSUPPORTED;
  const int grid = num_sms * 3;
  const size_t smem = sizeof(int) * (size_t)a.C;
  const int64_t bgrid = big_grid(a.N);
  if (bgrid > 0x7fffffff) return FQT_EUNSUPPORTED;
#define FQT_BG(L)                                                                      \
  if (CO == L) {                                                                       \
    if (bf16) {                                                                        \
      k_bhq_groups<__nv_bfloat16, L><<<grid, 256, smem, st>>>(a);                      \
      k_bhq_groups_big<__nv_bfloat16, L><<<(int)bgrid, 256, smem, st>>>(a);            \
    } else {                                                                           \
      k_bhq_groups<float, L><<<grid, 256, smem, st>>>(a);                              \
      k_bhq_groups_big<float, L><<<(int)bgrid, 256, smem, st>>>(a);                    \
    }                                                                                  \
  }
  FQT_BG(8)
  FQT_BG(16)
  FQT_BG(32)
#undef FQT_BG
  return cuda_fail(cudaGetLastError(), "BHQ group quantizer launch");
}

}  // namespace fqt
