// fqt_common.cuh -- shared device helpers of the GB300 FQT library:
// workspace layout, the Philox4x32-10 generator, stochastic rounding and the
// PTX wrappers (mbarrier, bulk copies, fences) the kernels use.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "fqt.h"

namespace fqt {

// ---------------------------------------------------------------------------
// Workspace layout (caller-owned device memory, zero-filled before first use)
//   [0, 256)               header: int32 status word at offset 0
//   [256, 256 + 32 KiB)    per-CTA (min, max) partials of the range pass
//   [kGemmOffset, ...)     split-K int32 partial tiles of grad_W
// ---------------------------------------------------------------------------
constexpr size_t kHeaderBytes = 256;
constexpr int kMaxRangeCtas = 4096;
constexpr size_t kRangeOffset = kHeaderBytes;
constexpr size_t kRangeBytes = sizeof(float2) * kMaxRangeCtas;
constexpr size_t kGemmOffset = kRangeOffset + kRangeBytes;

// Time limit of every device-side wait (mbarrier polls), in nanoseconds of
// %globaltimer.  A wait that exceeds it records FQT_ETIMEOUT and the kernel
// winds down; no legitimate wait in these kernels lasts a millisecond.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ void record_status(int *status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of the 4x32
// S-box, multipliers 0xD2511F53 / 0xCD9E8D57, Weyl key increments
// 0x9E3779B9 / 0xBB67AE85.
// ---------------------------------------------------------------------------
// The ten round keys (k0 + r W0, k1 + r W1) depend on the seed only: the
// host expands them once and they reach the kernels as launch parameters.
struct PhiloxKeys {
  uint32_t k[20];
};

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, const PhiloxKeys &key) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)0xD2511F53u * c.x;
    const uint64_t p1 = (uint64_t)0xCD9E8D57u * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ key.k[2 * r], (uint32_t)p1,
                   (uint32_t)(p0 >> 32) ^ c.w ^ key.k[2 * r + 1], (uint32_t)p0);
  }
  return c;
}

// Eight 16-bit uniforms for the aligned group of 8 consecutive flat indices
// starting at 8*q of `stream`: uniform i is half (i mod 2) of word i / 2.
__device__ __forceinline__ uint4 philox_oct(uint64_t q, uint32_t stream,
                                            const PhiloxKeys &key) {
  return philox4x32_10(
      make_uint4((uint32_t)q, (uint32_t)(q >> 32), stream, 0u), key);
}

__device__ __forceinline__ uint32_t u16_of(const uint4 &w, int i) {
  const uint32_t word = (i >> 1) == 0 ? w.x : (i >> 1) == 1 ? w.y
                        : (i >> 1) == 2 ? w.z : w.w;
  return (i & 1) ? (word >> 16) : (word & 0xFFFFu);
}

// Stochastic rounding of v >= 0 onto 0..B (Sec. 3.3): the probability
// frac(v) is realised in 16-bit fixed point, code = (floor(v 2^16) + u) >> 16.
// sr_code16 takes v * 2^16 (scaling by 2^16 is exact, so callers may fold it
// into their scale factor).
// floor(v16) is read off the fp32 bits (integer shift of the significand by
// the exponent, no conversion instruction): v16 is capped at 2^24 - 1, which
// leaves every code unchanged (a capped v gives code B either way), so the
// exponent is at most 23 and the right shift 150 - exponent_field >= 0 (a
// funnel shift clamps shifts of 32 and more to 0, covering v16 < 1).
__device__ __forceinline__ uint32_t sr_code16(float v16, uint32_t u16, uint32_t B) {
  v16 = fminf(v16, fminf((float)((B + 1u) << 16), 16777215.0f));
  const uint32_t bits = __float_as_uint(v16);
  const uint32_t sig = (bits & 0x7FFFFFu) | 0x800000u;
  const uint32_t fixed = __funnelshift_rc(sig, 0u, 150u - (bits >> 23));
  const uint32_t code = (fixed + u16) >> 16;
  return min(code, B);
}

__device__ __forceinline__ uint32_t sr_code(float v, uint32_t u16, uint32_t B) {
  return sr_code16(__fmul_rn(v, 65536.0f), u16, B);
}

// Scale B / R of the affine quantizers; R = 0 or an overflowing quotient
// take s = 1 (all codes 0, value = z).
__device__ __forceinline__ float affine_scale(float mn, float mx, uint32_t B) {
  const float R = __fsub_rn(mx, mn);
  if (!(R > 0.0f)) return 1.0f;
  const float s = __fdiv_rn((float)B, R);
  return isfinite(s) ? s : 1.0f;
}

// ---------------------------------------------------------------------------
// Loads of 8 consecutive elements (an "oct") as floats.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void load_oct(const float *p, float (&x)[8]) {
  const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
  const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
  x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}

__device__ __forceinline__ void load_oct(const __nv_bfloat16 *p, float (&x)[8]) {
  const uint4 a = __ldg(reinterpret_cast<const uint4 *>(p));
  const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__device__ __forceinline__ void store_codes8(uint8_t *dst, const uint32_t (&c)[8]) {
  uint2 v;
  v.x = c[0] | (c[1] << 8) | (c[2] << 16) | (c[3] << 24);
  v.y = c[4] | (c[5] << 8) | (c[6] << 16) | (c[7] << 24);
  *reinterpret_cast<uint2 *>(dst) = v;
}

// Eight codes as the fp16 values code - off (exact for |.| <= 2048): the fp16
// bit pattern 0x6400 | c is 1024 + c, and one packed subtraction recentres
// two codes at a time.
__device__ __forceinline__ void store_carriers8(uint16_t *dst, const uint32_t (&c)[8],
                                                uint32_t off) {
  const __half2 bias = __half2half2(__int2half_rn(1024 + (int)off));
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t h = (0x6400u | c[2 * i]) | ((0x6400u | c[2 * i + 1]) << 16);
    __half2 v = __hsub2(*reinterpret_cast<const __half2 *>(&h), bias);
    w[i] = *reinterpret_cast<uint32_t *>(&v);
  }
  *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

// The other way, for sums of carriers: a word of two fp16 carriers v
// (integers, |v| <= 512) as the two 16-bit lanes v + 512.  v + 1536 lies in
// [1024, 2048), where fp16 steps by 1, so the packed addition is exact and
// each half's bits are 0x6400 + v + 512.  kLaneAdds such words add up
// without a carry between the lanes (64 x 1023 < 2^16).
constexpr int kLaneAdds = 64;

__device__ __forceinline__ uint32_t carrier_lanes(uint32_t wd) {
  const __half2 bias = __half2half2(__ushort_as_half((unsigned short)0x6600u));
  const __half2 s = __hadd2(*reinterpret_cast<const __half2 *>(&wd), bias);
  return *reinterpret_cast<const uint32_t *>(&s) - 0x64006400u;
}

// ---------------------------------------------------------------------------
// PTX wrappers: mbarrier, async-proxy fences, bulk / tensor copies.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(count));
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile(
      "mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(
          smem_u32(bar)),
      "r"(bytes)
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait that lets the hardware suspend the thread for up to `ns`
// nanoseconds (it resumes as soon as the phase completes), so a waiting warp
// does not take issue slots from the warps doing work.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity,
                                                    uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait: returns false (and records FQT_ETIMEOUT) if the phase with
// the given parity has not completed within limit_ns nanoseconds.
__device__ __forceinline__ bool mbar_wait_limit(uint64_t *bar, uint32_t parity,
                                                int *status, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (;;) {
    for (int i = 0; i < 8; ++i)
      if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if (global_ns() - t0 > limit_ns) {
      record_status(status, FQT_ETIMEOUT);
      return false;
    }
  }
}

// The kernels' wait: bounded by kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity,
                                          int *status) {
  return mbar_wait_limit(bar, parity, status, kWaitLimitNs);
}

// Sleeps about `ns` nanoseconds (used only on the abort path).
__device__ __forceinline__ void sleep_ns(uint64_t ns) {
  const uint64_t t0 = global_ns();
  while (global_ns() - t0 < ns) __nanosleep(1000);
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Float-float arithmetic (an unevaluated sum h + l of two fp32 values, about
// 48 significant bits) from the error-free transformations of Knuth (two-sum),
// Dekker (fast two-sum) and the fused multiply-add product error.  The
// inverse Householder transform of BHQ subtracts nearly equal quantities;
// carrying them in float-float keeps the result accurate to fp32 rounding of
// the result itself.
// ---------------------------------------------------------------------------
struct ff {
  float h, l;
};

__device__ __forceinline__ ff two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return {s, e};
}

// requires |a| >= |b| (or a == 0)
__device__ __forceinline__ ff fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}

__device__ __forceinline__ ff two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return {p, __fmaf_rn(a, b, -p)};
}

__device__ __forceinline__ ff ff_add(ff x, ff y) {
  const ff s = two_sum(x.h, y.h);
  return fast_two_sum(s.h, __fadd_rn(s.l, __fadd_rn(x.l, y.l)));
}

__device__ __forceinline__ ff ff_neg(ff x) { return {-x.h, -x.l}; }

__device__ __forceinline__ ff ff_mul(ff x, ff y) {
  const ff p = two_prod(x.h, y.h);
  return fast_two_sum(p.h, __fmaf_rn(x.h, y.l, __fmaf_rn(x.l, y.h, p.l)));
}

// An integer (|v| < 2^53) as float-float, exactly for |v| < 2^48.
// Conversions to and from 64-bit integers run on the FP64 pipe, which is
// narrow on this GPU; for |v| < 2^47 the value is split as a 2^24 + b with
// 0 <= b < 2^24 and |a| < 2^23, both exact in fp32 after 32-bit conversions,
// and joined error-free (|a 2^24| >= 2^24 > b when a != 0).
__device__ __forceinline__ ff ff_from_int(long long v) {
  if ((unsigned long long)(v + (1LL << 47)) < (1ULL << 48)) {
    const float a = __int2float_rn((int)(v >> 24));
    const float b = __int2float_rn((int)(v & 0xFFFFFF));
    return fast_two_sum(__fmul_rn(a, 16777216.0f), b);
  }
  const float h = __ll2float_rn(v);
  return {h, __ll2float_rn(v - (long long)h)};
}

__device__ __forceinline__ float ff_round(ff x) { return __fadd_rn(x.h, x.l); }

// An int64 to fp32 rounded to nearest (the value of a 64-bit conversion),
// for |v| < 2^47 without the FP64 pipe: v = a 2^24 + b with a and b exact in
// fp32, and one fused multiply-add rounds a 2^24 + b once.
__device__ __forceinline__ float ll_to_float(long long v) {
  if ((unsigned long long)(v + (1LL << 47)) < (1ULL << 48))
    return __fmaf_rn(__int2float_rn((int)(v >> 24)), 16777216.0f,
                     __int2float_rn((int)(v & 0xFFFFFF)));
  return __ll2float_rn(v);
}

// An int32 as float-float, exactly, with 32-bit conversions only.
__device__ __forceinline__ ff ff_from_i32s(int v) {
  const float h = __int2float_rn(v);
  return {h, __int2float_rn(v - __float2int_rz(h))};
}

// Constants of the block Householder reflection of n >= 2 rows (Sec. 4.2):
// rho = 1/sqrt(n) (the entries of n = rho 1 - e_p besides the lead) and
// kappa = rho / (1 - rho) = 2 rho / ||n||^2, both in float-float.
struct HhConst {
  ff rho, kap;
};

__device__ __forceinline__ HhConst hh_const(int n) {
  const float nf = (float)n;
  const float rh = __fdiv_rn(1.0f, __fsqrt_rn(nf));
  // one Newton step on 1/sqrt(n): rho = rh (1 + r / 2) with r = 1 - n rh^2
  const ff p = two_prod(rh, rh);
  const float r = __fsub_rn(__fmaf_rn(-nf, p.h, 1.0f), __fmul_rn(nf, p.l));
  HhConst c;
  c.rho = fast_two_sum(rh, __fmul_rn(__fmul_rn(0.5f, rh), r));
  // kappa = rho / (1 - rho): quotient and one correction
  const ff om = ff_add({1.0f, 0.0f}, ff_neg(c.rho));
  const float q1 = __fdiv_rn(c.rho.h, om.h);
  const ff rem = ff_add(c.rho, ff_neg(ff_mul({q1, 0.0f}, om)));
  c.kap = fast_two_sum(q1, __fdiv_rn(rem.h, om.h));
  return c;
}

}  // namespace fqt
