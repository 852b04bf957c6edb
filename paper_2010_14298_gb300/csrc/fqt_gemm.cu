// fqt_gemm.cu -- the low-bit contractions of the FQT backward (Eq. 6, App. E)
// on the 5th-generation tensor cores of sm_103a.
//
// sm_103a has no tcgen05.mma kind::i8, so the integer codes ride in fp16:
// every centred code c - 2^(b-1) (|.| <= 128) is an exact fp16 value, their
// products are exact, and the fp32 accumulator in tensor memory stays exact
// while every partial sum is below 2^24 in magnitude.  The reduction is
// therefore cut into exact chunks of K_c = 2^(26 - b_A - b_B) terms; after
// each chunk the epilogue warps drain the accumulator into int32 registers.
//
// Warp roles of the persistent kernel (512 threads, one CTA per SM):
//   warp 0        TMA producer: u8 code tiles (A 128 x 64, B 128 x 64) into
//                 a ring of staging buffers (cp.async.bulk.tensor, mbarrier tx)
//   warp 1        tensor-memory allocator and MMA issuer (one elected lane):
//                 4 x tcgen05.mma.cta_group::1.kind::f16 (M128 N128 K16) per
//                 K-block into one of two TMEM accumulators, tcgen05.commit
//   warps 4..11   epilogue: tcgen05.ld drains, dequantization (and the BHQ
//                 inverse Householder across the rows of each block), TMA
//                 stores of fp32 grad_X tiles or int32 split-K partials
//   warps 12..15  converters: u8 staging -> centred fp16 in the canonical
//                 128-byte-swizzled K-major operand layout (transposing
//                 MN-major sources on the fly)
// Every mbarrier wait is bounded; a wait that runs out records FQT_ETIMEOUT
// and the CTA winds down.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <string.h>

#include "fqt_common.cuh"
#include "fqt_internal.h"

namespace fqt {

constexpr int BM = 128, BN = 128, BK = 64;
constexpr int kS8 = 4;   // u8 staging stages
constexpr int kS16 = 3;  // fp16 operand stages
constexpr int kGemmThreads = 512;
constexpr int kWarpTma = 0, kWarpMma = 1, kWarpEpi0 = 4, kWarpConv0 = 12;
constexpr int kNumEpiWarps = 8, kNumConvWarps = 4;
constexpr uint32_t kTmemCols = 256;  // two 128-column fp32 accumulators

constexpr size_t kOp16Bytes = 16384;                  // one 128 x 64 fp16 tile
constexpr size_t kSt8Bytes = 8192;                    // one 128 x 64 u8 tile
constexpr size_t kOffOp16 = 0;                        // [kS16][2] tiles
constexpr size_t kOffSt8 = kOffOp16 + kS16 * 2 * kOp16Bytes;
constexpr size_t kOffEpi = kOffSt8 + kS8 * 2 * kSt8Bytes;  // [8 warps] 4 KiB
constexpr size_t kOffBhq = kOffEpi + kNumEpiWarps * 4096;  // [2][2][4][32] floats
constexpr size_t kOffBar = kOffBhq + 2 * 2 * 4 * 32 * sizeof(float);
constexpr size_t kNumBars = 2 * kS8 + 2 * kS16 + 6;
constexpr size_t kGemmSmem = kOffBar + kNumBars * 8 + 16 + 1024;  // + align slack

enum { MODE_GRADX = 0, MODE_PARTIAL = 1 };

struct GemmArgs {
  int64_t M, N, K;            // out is M x N, reduction over K
  int a_kmajor, b_kmajor;     // operand storage (see fqt_debug_int_gemm)
  int oa, ob;                 // centring offsets 2^(b-1)
  int kc_blocks;              // K-blocks per exact chunk
  int m_tiles, n_tiles, splits;
  int64_t ks_blocks, kb_total;
  int64_t n_items;
  int mode;
  // grad_X epilogue (MODE_GRADX)
  int kind, block;
  const float *inv_s, *zero;   // Q_b2 metadata (1 or M entries)
  const int32_t *row_sum, *lead;
  const int32_t *col_sum_w;    // W~ column sums over C
  const float *inv_sw, *zero_w;
  int *status;
};

// ---------------------------------------------------------------------------
// PTX wrappers specific to the tensor-core path
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map,
                                            int32_t c0, int32_t c1,
                                            uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int32_t c0,
                                             int32_t c1, const void *src) {
  asm volatile(
      "cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
      ::"l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(src))
      : "memory");
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap *map, int32_t c0,
                                             int32_t c1, int32_t c2,
                                             const void *src) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];"
      ::"l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2),
      "r"(smem_u32(src))
      : "memory");
}

__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_read0() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait0() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

// UMMA shared-memory descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 bytes apart (stride byte offset), version 1 (bit 46).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;              // leading byte offset (unused, 16 B)
  d |= (uint64_t)(1024 >> 4) << 32;    // stride byte offset
  d |= (uint64_t)1 << 46;              // descriptor version
  d |= (uint64_t)2 << 61;              // SWIZZLE_128B
  return d;
}

// Instruction descriptor of kind::f16: A, B fp16 (K-major), D fp32,
// M = 128, N = 128.
constexpr uint32_t kIdesc = (1u << 4) | (0u << 7) | (0u << 10) |
                            ((uint32_t)(BN >> 3) << 17) |
                            ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void umma_f16(uint32_t tmem_d, uint64_t a_desc,
                                         uint64_t b_desc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a_desc), "l"(b_desc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void umma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
        "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]),
        "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t r;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
  return r;
}

// fp16 pair (x0 - off, x1 - off) for two code bytes already placed in byte
// lanes 0 and 2 of `t` (lanes 1 and 3 ignored): 0x64xx is the fp16 1024 + x.
__device__ __forceinline__ uint32_t centred_pair(uint32_t t, uint32_t sel,
                                                 __half2 bias) {
  const uint32_t h = prmt(t, 0x64646464u, sel);
  __half2 v = *reinterpret_cast<const __half2 *>(&h);
  v = __hsub2(v, bias);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Byte offset of the 16-byte chunk `chunk` of row `row` in a 128-byte-swizzled
// K-major tile (rows of 128 bytes, 1024-byte atoms of 8 rows).
__device__ __forceinline__ uint32_t sw128_off(int row, int chunk) {
  return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// Converts one 128 x 64 u8 tile into the fp16 operand tile.
//   kmajor: staging is [128 rows][64 k];  else: staging is [64 k][128 rows].
// k_valid: number of valid k in this K-block (the rest is written as 0).
__device__ __forceinline__ void convert_tile(const uint8_t *st, uint8_t *op,
                                             bool kmajor, int off, int k_valid,
                                             int ct) {
  const __half2 bias = __half2half2(__int2half_rn(1024 + off));
  if (kmajor) {
    // 512 items of 16 k: item -> (row = item / 4, kq = item % 4)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int item = ct + 128 * j;
      const int row = item >> 2, kq = item & 3;
      const uint4 w = *reinterpret_cast<const uint4 *>(st + row * 64 + kq * 16);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
      uint32_t h[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        h[2 * i] = centred_pair(ws[i], 0x4140u, bias);
        h[2 * i + 1] = centred_pair(ws[i], 0x4342u, bias);
      }
      if (kq * 16 + 16 > k_valid) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int k = kq * 16 + 2 * i;
          if (k >= k_valid) h[i] = 0u;
          else if (k + 1 >= k_valid) h[i] &= 0x0000FFFFu;
        }
      }
      *reinterpret_cast<uint4 *>(op + sw128_off(row, 2 * kq)) =
          make_uint4(h[0], h[1], h[2], h[3]);
      *reinterpret_cast<uint4 *>(op + sw128_off(row, 2 * kq + 1)) =
          make_uint4(h[4], h[5], h[6], h[7]);
    }
  } else {
    // 256 items of 8 k x 4 rows: item -> (kq = item / 32, rq = item % 32)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int item = ct + 128 * j;
      const int kq = item >> 5, rq = item & 31;
      uint32_t w[8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        w[i] = *reinterpret_cast<const uint32_t *>(st + (kq * 8 + i) * 128 + rq * 4);
      uint32_t h[4][4];  // [row r][k pair]
#pragma unroll
      for (int pr = 0; pr < 4; ++pr) {
        const uint32_t t01 = prmt(w[2 * pr], w[2 * pr + 1], 0x5140u);  // rows 0,1
        const uint32_t t23 = prmt(w[2 * pr], w[2 * pr + 1], 0x7362u);  // rows 2,3
        h[0][pr] = centred_pair(t01, 0x4140u, bias);
        h[1][pr] = centred_pair(t01, 0x4342u, bias);
        h[2][pr] = centred_pair(t23, 0x4140u, bias);
        h[3][pr] = centred_pair(t23, 0x4342u, bias);
      }
      if (kq * 8 + 8 > k_valid) {
#pragma unroll
        for (int pr = 0; pr < 4; ++pr) {
          const int k = kq * 8 + 2 * pr;
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            if (k >= k_valid) h[r][pr] = 0u;
            else if (k + 1 >= k_valid) h[r][pr] &= 0x0000FFFFu;
          }
        }
      }
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int r = (rr + rq) & 3;  // rotate to spread shared-memory banks
        const int row = rq * 4 + r;
        *reinterpret_cast<uint4 *>(op + sw128_off(row, kq)) =
            make_uint4(h[r][0], h[r][1], h[r][2], h[r][3]);
      }
    }
  }
}

struct Item {
  int64_t m0, n0;
  int split;
  int64_t kb0, kb1;
};

__device__ __forceinline__ Item decode_item(const GemmArgs &g, int64_t it) {
  Item r;
  const int64_t tiles = (int64_t)g.m_tiles * g.n_tiles;
  r.split = (int)(it / tiles);
  const int64_t t = it - (int64_t)r.split * tiles;
  r.m0 = (t / g.n_tiles) * BM;
  r.n0 = (t % g.n_tiles) * BN;
  r.kb0 = (int64_t)r.split * g.ks_blocks;
  r.kb1 = min(g.kb_total, r.kb0 + g.ks_blocks);
  return r;
}

// Segmented sum over aligned groups of `nb` lanes (nb a power of two <= 32).
__device__ __forceinline__ float seg_sum(float v, int nb) {
  for (int off = nb >> 1; off > 0; off >>= 1)
    v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap tmA,
           const __grid_constant__ CUtensorMap tmB,
           const __grid_constant__ CUtensorMap tmOut, const GemmArgs g) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment of the shared-window address (swizzle atoms)
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
  uint64_t *full8 = bars, *empty8 = bars + kS8;
  uint64_t *full16 = bars + 2 * kS8, *empty16 = bars + 2 * kS8 + kS16;
  uint64_t *accf = bars + 2 * kS8 + 2 * kS16, *acce = accf + 2;
  uint64_t *xbar = accf + 4;  // BHQ row-block exchange, one per column half
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + kNumBars);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kS8; ++i) {
      mbar_init(&full8[i], 1);
      mbar_init(&empty8[i], kNumConvWarps);
    }
    for (int i = 0; i < kS16; ++i) {
      mbar_init(&full16[i], kNumConvWarps);
      mbar_init(&empty16[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], kNumEpiWarps);
      mbar_init(&xbar[i], 4);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kWarpMma) {
    asm volatile(
        "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
            smem_u32(tmem_slot)),
        "r"(kTmemCols)
        : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  auto fail = [&]() { *abort_flag = 1; };

  if (warp == kWarpTma) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
        const Item t = decode_item(g, it);
        for (int64_t kb = t.kb0; kb < t.kb1; ++kb) {
          if (!mbar_wait(&empty8[s], ph ^ 1u, g.status)) { fail(); break; }
          mbar_expect_tx(&full8[s], (uint32_t)(2 * kSt8Bytes));
          uint8_t *sa = smem + kOffSt8 + (size_t)(2 * s) * kSt8Bytes;
          uint8_t *sb = sa + kSt8Bytes;
          const int32_t kc = (int32_t)(kb * BK);
          if (g.a_kmajor) tma_load_2d(sa, &tmA, kc, (int32_t)t.m0, &full8[s]);
          else tma_load_2d(sa, &tmA, (int32_t)t.m0, kc, &full8[s]);
          if (g.b_kmajor) tma_load_2d(sb, &tmB, kc, (int32_t)t.n0, &full8[s]);
          else tma_load_2d(sb, &tmB, (int32_t)t.n0, kc, &full8[s]);
          if (++s == kS8) { s = 0; ph ^= 1u; }
        }
      }
      // every issued load lands before the CTA exits: in normal operation the
      // converters have consumed them all; after an abort, give in-flight
      // copies time to complete
      if (*abort_flag) {
        sleep_ns(200000);
      } else {
        for (int i = 0; i < kS8; ++i) {
          if (!mbar_wait(&empty8[s], ph ^ 1u, g.status)) break;
          if (++s == kS8) { s = 0; ph ^= 1u; }
        }
      }
    }
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      int buf = 0;
      uint32_t aph[2] = {0u, 0u};
      for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
        const Item t = decode_item(g, it);
        for (int64_t c0 = t.kb0; c0 < t.kb1 && !*abort_flag; c0 += g.kc_blocks) {
          const int64_t c1 = min(t.kb1, c0 + g.kc_blocks);
          if (!mbar_wait(&acce[buf], aph[buf] ^ 1u, g.status)) { fail(); break; }
          tc_fence_after();
          const uint32_t dt = tmem + (uint32_t)(buf * BN);
          for (int64_t kb = c0; kb < c1; ++kb) {
            if (!mbar_wait(&full16[s], ph, g.status)) { fail(); break; }
            tc_fence_after();
            const uint32_t a_addr = smem_u32(smem + kOffOp16 + (size_t)(2 * s) * kOp16Bytes);
            const uint32_t b_addr = a_addr + (uint32_t)kOp16Bytes;
            const uint64_t da = sw128_desc(a_addr), db = sw128_desc(b_addr);
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)
              umma_f16(dt, da + (uint64_t)(2 * k), db + (uint64_t)(2 * k),
                       (kb > c0 || k > 0) ? 1u : 0u);
            umma_commit(&empty16[s]);
            if (++s == kS16) { s = 0; ph ^= 1u; }
          }
          umma_commit(&accf[buf]);
          aph[buf] ^= 1u;
          buf ^= 1;
        }
      }
    }
  } else if (warp >= kWarpConv0) {
    // ------------------------------------------------------------ converters
    const int ct = threadIdx.x - kWarpConv0 * 32;
    int s8 = 0, s16 = 0;
    uint32_t ph8 = 0, ph16 = 0;
    for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
      const Item t = decode_item(g, it);
      for (int64_t kb = t.kb0; kb < t.kb1; ++kb) {
        bool ok = !*abort_flag && mbar_wait(&full8[s8], ph8, g.status);
        ok = ok && mbar_wait(&empty16[s16], ph16 ^ 1u, g.status);
        if (!__all_sync(0xffffffffu, ok)) { fail(); break; }
        const uint8_t *sa = smem + kOffSt8 + (size_t)(2 * s8) * kSt8Bytes;
        uint8_t *oa = smem + kOffOp16 + (size_t)(2 * s16) * kOp16Bytes;
        const int64_t krem = g.K - kb * BK;
        const int kv = krem >= BK ? BK : (int)krem;
        convert_tile(sa, oa, g.a_kmajor != 0, g.oa, kv, ct);
        convert_tile(sa + kSt8Bytes, oa + kOp16Bytes, g.b_kmajor != 0, g.ob, kv, ct);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&full16[s16]);
          mbar_arrive(&empty8[s8]);
        }
        if (++s8 == kS8) { s8 = 0; ph8 ^= 1u; }
        if (++s16 == kS16) { s16 = 0; ph16 ^= 1u; }
      }
    }
  } else if (warp >= kWarpEpi0) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kWarpEpi0;
    const int q = warp & 3;       // TMEM lane quadrant = rows 32q .. 32q+31
    const int hcol = ew >> 2;     // column half: 64 * hcol .. +63
    uint8_t *stage = smem + kOffEpi + (size_t)ew * 4096;
    float *xch = reinterpret_cast<float *>(smem + kOffBhq);  // [2][2][4][32]
    uint32_t xph = 0;
    int buf = 0;
    uint32_t aph[2] = {0u, 0u};
    bool pending_store = false;
    for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
      const Item t = decode_item(g, it);
      int acc[64];
      bool first = true;
      bool ok = true;
      for (int64_t c0 = t.kb0; c0 < t.kb1; c0 += g.kc_blocks) {
        const bool got = !*abort_flag && mbar_wait(&accf[buf], aph[buf], g.status);
        if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
        tc_fence_after();
        const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN + hcol * 64);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t r[32];
          tmem_ld32(base + (uint32_t)(half * 32), r);
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int v = __float2int_rn(__uint_as_float(r[j]));
            acc[half * 32 + j] = first ? v : acc[half * 32 + j] + v;
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[buf]);
        aph[buf] ^= 1u;
        buf ^= 1;
        first = false;
      }
      if (!ok) { fail(); break; }

      const int64_t row = t.m0 + q * 32 + lane;
      const int64_t col0 = t.n0 + hcol * 64;
      // per-row constants of the grad_X epilogue (Eq. 9 dequantization):
      // V_ij = sum_c (a_ic + z'_i)(w_cj + z'_w) from the exact centred product
      // P_ij and integer row / column sums; with m = round(-z'), d = z' + m,
      // V = I + d_w SA_i + d_i SW_j + C d_i d_w, I = sum (a - m_i)(w - m_w).
      const bool gx = g.mode == MODE_GRADX;
      const bool rv = row < g.M;
      int alpha = 0, rowI = 0, Cn = 0, ob = g.ob, mw = 0, nb = 1;
      float di = 0.0f, rowF = 0.0f, scale = 0.0f, ek = 0.0f, ck = 0.0f;
      if (gx) {
        const int64_t ri = g.kind == FQT_PTQ ? 0 : (rv ? row : 0);
        const float inv_si = rv ? g.inv_s[ri] : 0.0f;
        const float zi = g.zero[ri];
        const int rsum = rv ? g.row_sum[row] : 0;
        const float zw = *g.zero_w;
        Cn = (int)g.K;
        const int mi = __float2int_rn(-zi);
        mw = __float2int_rn(-zw);
        di = zi + (float)mi;
        const float dw = zw + (float)mw;
        alpha = g.oa - mi;
        const int beta = ob - mw;
        rowI = beta * (rsum - Cn * g.oa) + Cn * alpha * beta;
        rowF = dw * (float)(rsum - Cn * mi) + (float)Cn * di * dw;
        scale = (*g.inv_sw) * inv_si;
        if (g.kind == FQT_BHQ) {
          nb = g.block;
          const int64_t b = row / nb;
          const int64_t nb_act = min((int64_t)nb, g.M - b * nb);
          if (rv && nb_act > 1) {  // Q = I - 2 n n^T / |n|^2, n = rho 1 - e_p
            const int p = g.lead[b];
            const float rho = 1.0f / sqrtf((float)nb_act);
            ck = (row - b * nb == p) ? rho - 1.0f : rho;
            ek = ck / (1.0f - rho);
          }
        }
      }
#pragma unroll
      for (int bx = 0; bx < 2; ++bx) {
        float outv[32];
        if (gx) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int64_t col = col0 + bx * 32 + j;
            const int cs = col < g.N ? __ldg(g.col_sum_w + col) : 0;
            const int I = acc[bx * 32 + j] + alpha * (cs - Cn * ob) + rowI;
            outv[j] = (float)I + (rowF + di * (float)(cs - Cn * mw));
          }
          if (g.kind == FQT_BHQ) {
            // inverse Householder of each block: (Q V)_k = V_k - c_k w with
            // w = sum_k e_k V_k over the block's rows (= TMEM lanes)
            if (nb <= 32) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const float w = seg_sum(ek * outv[j], nb);
                outv[j] = fmaf(-ck, w, outv[j]);
              }
            } else {
              // blocks of 64 / 128 rows span 2 / 4 quadrant warps: exchange the
              // per-warp column sums through shared memory, double-buffered,
              // synchronised by an mbarrier of the 4 warps of this column half
              const int qn = nb / 32, q0 = (q / qn) * qn;
              float mv = 0.0f;
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const float ws = seg_sum(ek * outv[j], 32);
                if (lane == j) mv = ws;
              }
              float *area = xch + ((xph & 1u) * 2 + hcol) * 4 * 32;
              area[q * 32 + lane] = mv;
              __syncwarp();
              if (lane == 0) mbar_arrive(&xbar[hcol]);
              const bool got = mbar_wait(&xbar[hcol], xph & 1u, g.status);
              if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
              xph ^= 1u;
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                float w = 0.0f;
                for (int qq = q0; qq < q0 + qn; ++qq) w += area[qq * 32 + j];
                outv[j] = fmaf(-ck, w, outv[j]);
              }
            }
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) outv[j] *= scale;
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) outv[j] = __int_as_float(acc[bx * 32 + j]);
        }
        // stage the 32 x 32 box through shared memory (128-byte swizzle) and
        // hand it to the TMA engine
        if (pending_store) {
          if (lane == 0) bulk_wait_read0();
          __syncwarp();
        }
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const float4 v = make_float4(outv[4 * c], outv[4 * c + 1], outv[4 * c + 2],
                                       outv[4 * c + 3]);
          *reinterpret_cast<float4 *>(stage + sw128_off(lane, c)) = v;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          const int32_t cx = (int32_t)(col0 + bx * 32), cy = (int32_t)(t.m0 + q * 32);
          if (gx) tma_store_2d(&tmOut, cx, cy, stage);
          else tma_store_3d(&tmOut, cx, cy, t.split, stage);
          bulk_commit();
        }
        pending_store = true;
      }
      if (!ok) { fail(); break; }
    }
    if (lane == 0) bulk_wait0();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// Split-K reduction (int64) and the grad_W / raw epilogues
// ---------------------------------------------------------------------------
struct ReduceArgs {
  const int32_t *part;
  int splits;
  int64_t M, N;
  int64_t *out_i64;  // raw sums (debug)
  float *out_f32;    // grad_W
  // grad_W = inv_s1 inv_sx sum_n (a_nc + z'_1)(x_nd + z'_x)
  int64_t Kn;        // rows N of dH / X
  int oa, ob;
  const int32_t *cs_a, *cs_b;  // column sums of Q_b1 codes (M) and X~ codes (N)
  const float *inv_a, *zero_a, *inv_b, *zero_b;
};

__global__ void __launch_bounds__(256) k_reduce(const ReduceArgs r) {
  const int64_t total = r.M * r.N;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += stride) {
    int64_t P = 0;
    for (int s = 0; s < r.splits; ++s) P += r.part[(int64_t)s * total + idx];
    if (r.out_i64) {
      r.out_i64[idx] = P;
      continue;
    }
    const int64_t c = idx / r.N, d = idx - c * r.N;
    const float za = *r.zero_a, zb = *r.zero_b;
    const int64_t ma = __float2int_rn(-za), mb = __float2int_rn(-zb);
    const float da = za + (float)ma, db = zb + (float)mb;
    const int64_t ca = r.cs_a[c], cb = r.cs_b[d];
    // I = sum (a - ma)(b - mb), exact, from the centred product P
    const int64_t I = P + (r.oa - ma) * (cb - r.Kn * r.ob) +
                      (r.ob - mb) * (ca - r.Kn * r.oa) +
                      r.Kn * (r.oa - ma) * (r.ob - mb);
    const float V = (float)I + db * (float)(ca - r.Kn * ma) +
                    da * (float)(cb - r.Kn * mb) + (float)r.Kn * da * db;
    r.out_f32[idx] = (*r.inv_a) * (*r.inv_b) * V;
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t,
                                  void *, const cuuint64_t *, const cuuint64_t *,
                                  const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

static bool make_map_u8(CUtensorMap *m, const void *base, uint64_t inner,
                        uint64_t outer, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims,
            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static bool make_map_out(CUtensorMap *m, void *base, bool is_int, uint64_t cols,
                         uint64_t rows, uint64_t depth) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {cols, rows, depth};
  cuuint64_t strides[2] = {cols * 4, cols * rows * 4};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, is_int ? CU_TENSOR_MAP_DATA_TYPE_INT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
            depth > 1 || is_int ? 3 : 2, base, dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static int exact_chunk_blocks(int a_bits, int b_bits) {
  // centred magnitudes <= 2^(b-1): partial sums stay below 2^24
  const int lg = 26 - a_bits - b_bits;
  int64_t kc = (int64_t)1 << (lg < 0 ? 0 : lg);
  int64_t blocks = kc / BK;
  if (blocks < 1) blocks = 1;
  if (blocks > (1 << 20)) blocks = 1 << 20;
  return (int)blocks;
}

// Split-K plan for an M x N output reduced over K.
struct SplitPlan {
  int m_tiles, n_tiles, splits;
  int64_t ks_blocks, kb_total;
};

static SplitPlan plan_splits(int64_t M, int64_t N, int64_t K, int a_bits,
                             int b_bits, int num_sms, bool allow_split) {
  SplitPlan p;
  p.m_tiles = (int)((M + BM - 1) / BM);
  p.n_tiles = (int)((N + BN - 1) / BN);
  p.kb_total = (K + BK - 1) / BK;
  if (p.kb_total < 1) p.kb_total = 1;
  int splits = 1;
  if (allow_split) {
    const int64_t tiles = (int64_t)p.m_tiles * p.n_tiles;
    splits = (int)((num_sms + tiles - 1) / tiles);
    // int32 partials: a split reduces at most 2^31 / 2^(a+b-2) terms
    const int64_t max_terms = ((int64_t)1 << 31) >> (a_bits + b_bits - 2);
    const int64_t min_splits = (K + max_terms - 1) / max_terms;
    if (splits < min_splits) splits = (int)min_splits;
    if (splits > p.kb_total) splits = (int)p.kb_total;
    if (splits < 1) splits = 1;
  }
  p.ks_blocks = (p.kb_total + splits - 1) / splits;
  p.splits = (int)((p.kb_total + p.ks_blocks - 1) / p.ks_blocks);
  return p;
}

size_t gemm_workspace_bytes(int64_t N, int64_t C, int64_t D) {
  // grad_W: M = C, N = D, K = N (8-bit x 8-bit)
  const SplitPlan p = plan_splits(C, D, N, 8, 8, device_sm_count(), true);
  const size_t bytes = (size_t)p.splits * (size_t)C * (size_t)D * 4;
  return (bytes + 255) & ~(size_t)255;
}

static fqt_status run_gemm(const void *A, int a_kmajor, int a_bits, const void *Bm,
                           int b_kmajor, int b_bits, int64_t M, int64_t N,
                           int64_t K, const SplitPlan &p, GemmArgs &g,
                           void *out, bool out_is_partial, cudaStream_t st) {
  CUtensorMap ta, tb, to;
  bool ok = a_kmajor ? make_map_u8(&ta, A, (uint64_t)K, (uint64_t)M, BK, BM)
                     : make_map_u8(&ta, A, (uint64_t)M, (uint64_t)K, BM, BK);
  ok = ok && (b_kmajor ? make_map_u8(&tb, Bm, (uint64_t)K, (uint64_t)N, BK, BN)
                       : make_map_u8(&tb, Bm, (uint64_t)N, (uint64_t)K, BN, BK));
  ok = ok && make_map_out(&to, out, out_is_partial, (uint64_t)N, (uint64_t)M,
                          out_is_partial ? (uint64_t)p.splits : 1);
  if (!ok) return FQT_ECUDA;
  g.M = M;
  g.N = N;
  g.K = K;
  g.a_kmajor = a_kmajor;
  g.b_kmajor = b_kmajor;
  g.oa = 1 << (a_bits - 1);
  g.ob = 1 << (b_bits - 1);
  g.kc_blocks = exact_chunk_blocks(a_bits, b_bits);
  g.m_tiles = p.m_tiles;
  g.n_tiles = p.n_tiles;
  g.splits = p.splits;
  g.ks_blocks = p.ks_blocks;
  g.kb_total = p.kb_total;
  g.n_items = (int64_t)p.m_tiles * p.n_tiles * p.splits;
  g.mode = out_is_partial ? MODE_PARTIAL : MODE_GRADX;
  static bool attr_set = false;
  if (!attr_set) {
    if (cudaFuncSetAttribute(k_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kGemmSmem) != cudaSuccess)
      return FQT_ECUDA;
    attr_set = true;
  }
  const int nsm = device_sm_count();
  int64_t grid = g.n_items < nsm ? g.n_items : nsm;
  if (grid < 1) grid = 1;
  k_gemm<<<(int)grid, kGemmThreads, kGemmSmem, st>>>(ta, tb, to, g);
  return cudaGetLastError() == cudaSuccess ? FQT_OK : FQT_ECUDA;
}

static void launch_reduce(const ReduceArgs &r, cudaStream_t st) {
  const int64_t total = r.M * r.N;
  int64_t grid = (total + 255) / 256;
  const int64_t cap = (int64_t)device_sm_count() * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  k_reduce<<<(int)grid, 256, 0, st>>>(r);
}

static bool aligned16(const void *p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

fqt_status debug_int_gemm(const uint8_t *A, int a_kmajor, int a_bits,
                          const uint8_t *Bm, int b_kmajor, int b_bits, int64_t M,
                          int64_t N, int64_t K, int64_t *out, void *ws,
                          size_t ws_bytes, cudaStream_t st) {
  if (!A || !Bm || !out || M <= 0 || N <= 0 || K <= 0) return FQT_EINVAL;
  if (a_bits < 2 || a_bits > 8 || b_bits < 2 || b_bits > 8) return FQT_EINVAL;
  if (!aligned16(A) || !aligned16(Bm)) return FQT_EINVAL;
  // TMA: the row pitch of each stored operand must be a multiple of 16 bytes
  if ((a_kmajor ? K : M) % 16 || (b_kmajor ? K : N) % 16 || N % 4) return FQT_EUNSUPPORTED;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return FQT_EUNSUPPORTED;
  const SplitPlan p = plan_splits(M, N, K, a_bits, b_bits, device_sm_count(), true);
  const size_t need = kGemmOffset + (size_t)p.splits * (size_t)M * (size_t)N * 4;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < need)
    return FQT_EWORKSPACE;
  int32_t *part = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kGemmOffset);
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.status = reinterpret_cast<int *>(ws);
  fqt_status s = run_gemm(A, a_kmajor, a_bits, Bm, b_kmajor, b_bits, M, N, K, p,
                          g, part, true, st);
  if (s != FQT_OK) return s;
  ReduceArgs r;
  memset(&r, 0, sizeof(r));
  r.part = part;
  r.splits = p.splits;
  r.M = M;
  r.N = N;
  r.out_i64 = out;
  launch_reduce(r, st);
  return cudaGetLastError() == cudaSuccess ? FQT_OK : FQT_ECUDA;
}

fqt_status linear_backward(const fqt_qtensor *q_b2, const fqt_qtensor *q_b1,
                           const fqt_qtensor *qx, const fqt_qtensor *qw,
                           float *grad_X, float *grad_W, void *ws,
                           size_t ws_bytes, cudaStream_t st) {
  if (!grad_X && !grad_W) return FQT_OK;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u)) return FQT_EWORKSPACE;
  int *status = reinterpret_cast<int *>(ws);
  const int nsm = device_sm_count();
  if (grad_X) {
    if (!q_b2 || !qw || !q_b2->codes || !qw->codes || !q_b2->row_sum || !qw->col_sum ||
        !q_b2->inv_s || !q_b2->zero || !qw->inv_s || !qw->zero)
      return FQT_EINVAL;
    if (q_b2->kind == FQT_BHQ && !q_b2->lead) return FQT_EINVAL;
    const int64_t Nr = q_b2->rows, C = q_b2->cols, D = qw->cols;
    if (qw->rows != C || qw->kind != FQT_PTQ) return FQT_EINVAL;
    if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
    if (C > 8192) return FQT_EUNSUPPORTED;  // int32 epilogue bound
    if (!aligned16(q_b2->codes) || !aligned16(qw->codes) || !aligned16(grad_X))
      return FQT_EINVAL;
    if (Nr > 0) {
      const SplitPlan p = plan_splits(Nr, D, C, q_b2->bits, qw->bits, nsm, false);
      GemmArgs g;
      memset(&g, 0, sizeof(g));
      g.status = status;
      g.kind = q_b2->kind;
      g.block = q_b2->kind == FQT_BHQ ? q_b2->block : 0;
      g.inv_s = q_b2->inv_s;
      g.zero = q_b2->zero;
      g.row_sum = q_b2->row_sum;
      g.lead = q_b2->lead;
      g.col_sum_w = qw->col_sum;
      g.inv_sw = qw->inv_s;
      g.zero_w = qw->zero;
      fqt_status s = run_gemm(q_b2->codes, 1, q_b2->bits, qw->codes, 0, qw->bits, Nr,
                              D, C, p, g, grad_X, false, st);
      if (s != FQT_OK) return s;
    }
  }
  if (grad_W) {
    const fqt_qtensor *qa = q_b1 ? q_b1 : q_b2;
    if (!qa || !qx || !qa->codes || !qx->codes || !qa->col_sum || !qx->col_sum ||
        !qa->inv_s || !qa->zero || !qx->inv_s || !qx->zero)
      return FQT_EINVAL;
    if (qa->kind != FQT_PTQ || qx->kind != FQT_PTQ) return FQT_EINVAL;
    const int64_t Nr = qa->rows, C = qa->cols, D = qx->cols;
    if (qx->rows != Nr) return FQT_EINVAL;
    if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
    if (!aligned16(qa->codes) || !aligned16(qx->codes)) return FQT_EINVAL;
    const SplitPlan p = plan_splits(C, D, Nr, qa->bits, qx->bits, nsm, true);
    const size_t need = kGemmOffset + (size_t)p.splits * (size_t)C * (size_t)D * 4;
    if (ws_bytes < need) return FQT_EWORKSPACE;
    int32_t *part = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kGemmOffset);
    if (Nr > 0) {
      GemmArgs g;
      memset(&g, 0, sizeof(g));
      g.status = status;
      fqt_status s = run_gemm(qa->codes, 0, qa->bits, qx->codes, 0, qx->bits, C, D,
                              Nr, p, g, part, true, st);
      if (s != FQT_OK) return s;
    } else {
      if (cudaMemsetAsync(part, 0, (size_t)C * D * 4, st) != cudaSuccess) return FQT_ECUDA;
    }
    ReduceArgs r;
    memset(&r, 0, sizeof(r));
    r.part = part;
    r.splits = Nr > 0 ? p.splits : 1;
    r.M = C;
    r.N = D;
    r.out_f32 = grad_W;
    r.Kn = Nr;
    r.oa = 1 << (qa->bits - 1);
    r.ob = 1 << (qx->bits - 1);
    r.cs_a = qa->col_sum;
    r.cs_b = qx->col_sum;
    r.inv_a = qa->inv_s;
    r.zero_a = qa->zero;
    r.inv_b = qx->inv_s;
    r.zero_b = qx->zero;
    launch_reduce(r, st);
    if (cudaGetLastError() != cudaSuccess) return FQT_ECUDA;
  }
  return FQT_OK;
}

}  // namespace fqt
