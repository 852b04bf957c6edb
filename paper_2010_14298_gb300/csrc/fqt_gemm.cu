// fqt_gemm.cu -- the low-bit contractions of the FQT backward (Eq. 6, App. E)
// on the 5th-generation tensor cores of sm_103a.
//
// sm_103a has no tcgen05.mma kind::i8, so the integer codes ride in fp16:
// the quantizers emit every code centred, c - 2^(b-1) (|.| <= 128), as an
// exact fp16 value; products are exact and the fp32 accumulator in tensor
// memory stays exact while every partial sum is below 2^24 in magnitude.
// The reduction is therefore cut into exact chunks of K_c = 2^(26 - bA - bB)
// terms; between chunks the epilogue warps fold the accumulator into an
// int32 running sum kept in tensor memory (tcgen05.st).
//
// Warp roles of the persistent kernel (320 threads, one CTA per SM):
//   warp 0        TMA producer: fp16 operand tiles (128 x 64 per operand,
//                 128-byte swizzle) into a ring of shared-memory stages
//                 (cp.async.bulk.tensor, mbarrier transaction counts)
//   warp 1        tensor-memory allocator and MMA issuer (one elected lane):
//                 4 x tcgen05.mma.cta_group::1.kind::f16 (M128 N128 K16) per
//                 stage into one of two TMEM accumulators, tcgen05.commit;
//                 K-major and MN-major operands use the matching descriptors
//   warps 2..9    epilogue: tcgen05.ld, dequantization (and the inverse
//                 Householder of every BHQ block for grad_X), coalesced
//                 16-byte stores of fp32 grad_X or int32 split-K partials
// Every mbarrier wait is bounded; a wait that runs out records FQT_ETIMEOUT
// and the CTA winds down.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <algorithm>
#include <string.h>

#include "fqt_common.cuh"
#include "fqt_internal.h"

namespace fqt {

constexpr int BM = 128, BN = 128, BK = 64;
constexpr int kMaxStages = 8;  // operand stages (A and B fp16 tiles), chosen per launch
constexpr int kWarpTma = 0, kWarpMma = 1, kWarpEpi0 = 2;  // k_gradw's roles
constexpr int kPartialEpiWarps = 8;
// k_gemm: warpgroup 0 holds the TMA producer, the MMA issuer and grad_X's
// per-tile parameter loader (warp 3 idles); the epilogue warps follow in
// sets of four (one per TMEM lane quadrant) that take the tiles in turn.
// The epilogue's arithmetic comes in three forms (FORM):
//   0  int32 integer parts (several exact chunks, or the fp32 form's offset
//      bound below 0);
//   1  the fp32 form for tiles whose row offsets allow it, int32 for the
//      others, in the same epilogue (the fp32 form's offset bound is small);
//   2  the fp32 form only.
// In every form the rare tiles outside it (a row offset m beyond the int32
// form's, or the fp32 form's in FORM 2) are stored raw and finished by the
// CTA after its last tile (gradx_raw_fix).
// FORM 2 has four sets: without the int32 path, warpgroup 0 can hand
// registers to the epilogue warpgroups (setmaxnreg) and 104 per thread
// suffice (96 for blocks of up to 16 rows, whose parameter loader keeps 80); tiles with a long reduction use three of the sets (g.sets), so
// that the tensor cores fill a fourth accumulator while three are drained.
// Otherwise three sets at 128 registers; split-K partials use the first
// eight epilogue warps.
constexpr int kGemmWarpPar = 2, kGemmWarpEpi0 = 4;
template <int MODE, int FORM, int NB = 16>
struct GemmLayout {
  static constexpr int sets = (MODE == 0 && FORM == 2) ? 4 : 3;  // MODE 0: grad_X
  static constexpr int threads = 32 * (kGemmWarpEpi0 + 4 * sets);
  // registers per thread of the launch, and the split (0: no setmaxnreg)
  static constexpr int launch_regs = ((65536 / threads) / 8) * 8;
  static constexpr int regs_ctl = sets == 4 ? (NB <= 16 ? 80 : 64) : 0;
  static constexpr int regs_epi = sets == 4 ? (NB <= 16 ? 96 : 104) : 0;
  static_assert(regs_ctl == 0 || 128 * regs_ctl + 32 * 4 * sets * regs_epi <= threads * launch_regs,
                "register split above the launch's registers");
};
// two 128-column fp32 accumulators and 256 columns of int32 running sums
constexpr uint32_t kTmemCols = 512;

constexpr size_t kTileBytes = 16384;  // one 128 x 64 fp16 operand tile
constexpr size_t kBoxBytes = 4096;   // one 32 x 32 fp32 / int32 output box
// Shared memory, from a 1024-byte-aligned base:
//   [0, kFixedBytes)           per-warp epilogue tables and barriers
//   [kFixedBytes, +S * 32 KiB) S operand stages (A, B)
//   [..., + 8 * R * 4 KiB)     R output boxes per epilogue warp (TMA store ring)
// grad_X parameter stages (one per tile in flight), each:
//   float4 kp[BN]  per row k: inv_sw inv_s_k, .. hz_k, .. y hr_k, m_k
//   int leads[BN]  lead row of each block;  int msum[BN]  sum of m per block
//   int cs[BM]     W~ column sums of the tile's columns;  int flag
constexpr int kParStages = 4;
constexpr size_t kParBytes = 4096;
constexpr size_t kParLeads = 2048, kParMsum = 2560, kParCs = 3072, kParFlag = 3584;
constexpr size_t kOffPar = 0;
constexpr size_t kOffBar = kOffPar + kParStages * kParBytes;
// operand full / empty, accumulator full / empty (4 each), parameter full /
// empty (4 each)
// ... + the MMA drain barrier + the byte-operand rings' barriers (carrier
// stage widened, carrier stage consumed)
constexpr size_t kNumBars = 4 * kMaxStages + 17;
// grad_X in the fp32 form with fixed blocks: one bit per tile of this CTA
// (in its order) for the tiles left raw, finished by the CTA at the end
constexpr size_t kOffRaw = (kOffBar + kNumBars * 8 + 16 + 15) & ~(size_t)15;
constexpr size_t kRawMaskBytes = 4096;
constexpr int64_t kMaxLocalTiles = (int64_t)kRawMaskBytes * 8;
constexpr size_t kFixedBytes = (kOffRaw + kRawMaskBytes + 1023) & ~(size_t)1023;

// Operand stages: `stages` of the A and B fp16 tiles (32 KB), and with byte
// operands (split-K partials) `ustages` of their 8 KB byte tiles as TMA wrote
// them (16 KB), a deeper ring of their own in front of the carrier ring.
__host__ __device__ constexpr size_t gemm_smem_bytes(int stages, int ring, int ustages = 0) {
  return kFixedBytes + (size_t)stages * 2 * kTileBytes + (size_t)ustages * kTileBytes +
         (size_t)kPartialEpiWarps * ring * kBoxBytes + 1024;  // + alignment slack
}

// MODE_GRADX: grad_X^T = W~^T Q_b2(dH)^T, i.e. M = D (output columns of
// grad_X, TMEM lanes), N = rows of dH (TMEM columns), K = C, with the
// dequantizing epilogue.  MODE_PARTIAL: raw int32 split-K partials.
enum { MODE_GRADX = 0, MODE_PARTIAL = 1 };

struct GemmArgs {
  int64_t M, N, K;            // out is M x N, reduction over K
  int a_kmajor, b_kmajor;     // operand storage (see fqt_debug_int_gemm)
  uint32_t mn_lbo, mn_sbo;    // MN-major descriptor strides (bytes)
  int kc_blocks;              // K-blocks per exact chunk
  int m_tiles, n_tiles, splits;
  int64_t ks_blocks, kb_total;
  int64_t n_items;
  int stages, ring;           // operand stages, output boxes per epilogue warp
  int nacc;                   // TMEM accumulators in rotation (2 or 4)
  int m_fast;                 // item order: M tiles fastest (grad_X: the D
                              // tiles of the same output rows together)
  // grad_X epilogue (MODE_GRADX); rows of Q_b2 are the N dimension
  int kind;
  int og, ow;                  // centring offsets 2^(b-1) of Q_b2 and W~ codes
  const float *inv_s, *zero;   // Q_b2 metadata (1 or N entries)
  const int32_t *row_sum, *lead;
  const float *hz, *hr;        // BHQ offsets (block > 1)
  const int32_t *perm, *gsize; // adaptive BHQ groups (NB = 0): output row and
                               // group size of every stored row of Q_b2
  float raw_mmax;              // NB = 0: largest |m| of a row finished here
  float flt_mmax;              // largest |m| of a tile for the fp32 form
  float i32_mmax;              // largest |m| of a tile for the int32 form
  const int32_t *col_sum_w;    // W~ column sums over C
  const float *inv_sw, *zero_w;
  float *out;                  // grad_X (N x M row-major) for MODE_GRADX
  int sets;                    // grad_X epilogue sets in use (3 or 4)
  int bw, b2;                  // code bits of W~ and of Q_b2
  int small_p;                 // every |P| < 2^22 (block sums off the fp32 bits)
  int u8;                      // MODE_PARTIAL: byte operands, widened on chip
  int ustages;                 // ... through a ring of this many byte stages
  // MODE_PARTIAL with an implicit im2col X~ (stride 1): K blocks of 64
  // output-pixel slots = rpb output rows of pw slots (pw >= ow, the slots
  // past ow zero); A (Q_b1) and B (the NHWC codes at each tap's offset) are
  // read as 4-D boxes of (64 channels, pw, rpb, 1)
  int conv, cpw, crpb, cybi, coh, cih, cin, ckw, cpad, cow, ciw;
  int64_t cnimg;
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

__device__ __forceinline__ void tma_load_4d(void *dst, const CUtensorMap *map, int32_t c0,
                                            int32_t c1, int32_t c2, int32_t c3,
                                            uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
      "r"(smem_u32(bar))
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

// Waits until at most n of this thread's bulk store groups still read
// shared memory (n = ring depth - 1 frees the oldest slot).
__device__ __forceinline__ void bulk_wait_read(int n) {
  switch (n) {
    case 0: asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); break;
    case 1: asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); break;
    case 2: asm volatile("cp.async.bulk.wait_group.read 2;" ::: "memory"); break;
    default: asm volatile("cp.async.bulk.wait_group.read 3;" ::: "memory"); break;
  }
}

__device__ __forceinline__ void bulk_wait_all() {
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

// UMMA shared-memory descriptor of an MN-major operand with 128-byte
// swizzle: 64-element (128-byte) MN atoms of 8 K rows (1024 bytes); atoms
// `lbo` bytes apart along MN and `sbo` bytes apart along K.
__device__ __forceinline__ uint64_t sw128_desc_mn(uint32_t saddr, uint32_t lbo,
                                                  uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor of kind::f16: A, B fp16, D fp32, M = 128, N = 128;
// bit 15 / 16 select MN-major A / B.
__host__ __device__ constexpr uint32_t make_idesc(bool a_mn, bool b_mn) {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((a_mn ? 1u : 0u) << 15) |
         ((b_mn ? 1u : 0u) << 16) | ((uint32_t)(BN >> 3) << 17) |
         ((uint32_t)(BM >> 4) << 24);
}

__device__ __forceinline__ void umma_f16(uint32_t tmem_d, uint64_t a_desc,
                                         uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
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

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
      "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
      "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 32 columns of this warp's 32 lanes, without waiting (see tmem_wait_ld).
__device__ __forceinline__ void tmem_ld32_nw(uint32_t taddr, uint32_t (&r)[32]) {
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
}

__device__ __forceinline__ void tmem_ld16_nw(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
        "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld8_nw(uint32_t taddr, uint32_t (&r)[8]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7])
      : "r"(taddr));
}

// W consecutive columns (W = 8, 16 or 32) of this warp's 32 lanes.
template <int W>
__device__ __forceinline__ void tmem_ldw_nw(uint32_t taddr, uint32_t (&r)[W]) {
  if constexpr (W == 32) tmem_ld32_nw(taddr, r);
  else if constexpr (W == 16) tmem_ld16_nw(taddr, r);
  else tmem_ld8_nw(taddr, r);
}

// One column of this warp's 32 lanes, without waiting.
__device__ __forceinline__ uint32_t tmem_ld1_nw(uint32_t taddr) {
  uint32_t v;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(v) : "r"(taddr));
  return v;
}

// Waits for every tcgen05.ld this thread has issued.  The registers of the
// loads are passed through so that no use is scheduled before the wait.
template <int NR>
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&r)[NR]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < NR; ++i) asm volatile("" : "+r"(r[i]));
}

// Byte offset of the 16-byte chunk `chunk` of row `row` in a 128-byte-swizzled
// K-major tile (rows of 128 bytes, 1024-byte atoms of 8 rows).
__device__ __forceinline__ uint32_t sw128_off(int row, int chunk) {
  return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// The 32 rows r0 .. r0 + 31 of this thread's column j of grad_X.  The 32
// lanes of a warp hold 32 consecutive columns, so every store of a row is one
// coalesced 128-byte write; no staging is needed.
struct BoxOut {
  float *p;       // &grad_X[row r0][j]
  int64_t ld;     // row stride (D)
  int rows;       // rows of the box inside the matrix (0 .. 32)
  bool jv;        // column j inside the matrix
  __device__ __forceinline__ void st(int row, float v) const {
    if (jv && row < rows) __stcs(p + row * ld, v);
  }
  // all 32 values of the box (then the lead-row overwrites, same thread)
  __device__ __forceinline__ void st32(const float (&o)[32]) const {
    if (!jv) return;
    if (rows == 32) {
#pragma unroll
      for (int i = 0; i < 32; ++i) __stcs(p + i * ld, o[i]);
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i < rows) __stcs(p + i * ld, o[i]);
    }
  }
};


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
  if (g.m_fast) {  // the M tiles of the same N rows side by side
    r.m0 = (t % g.m_tiles) * BM;
    r.n0 = (t / g.m_tiles) * BN;
  } else {
    r.m0 = (t / g.n_tiles) * BM;
    r.n0 = (t % g.n_tiles) * BN;
  }
  r.kb0 = (int64_t)r.split * g.ks_blocks;
  r.kb1 = min(g.kb_total, r.kb0 + g.ks_blocks);
  return r;
}

// The items of one step of a CTA's schedule: item it, and with pairs the
// CTA's next item it + gridDim.x when it exists.  Returns their count.
__device__ __forceinline__ int group_items(const GemmArgs &g, int64_t it, bool pairs,
                                           Item (&tt)[2]) {
  tt[0] = decode_item(g, it);
  tt[1] = tt[0];
  if (pairs && it + (int64_t)gridDim.x < g.n_items) {
    tt[1] = decode_item(g, it + (int64_t)gridDim.x);
    return 2;
  }
  return 1;
}

__device__ __forceinline__ BoxOut box_out(const GemmArgs &g, const Item &t, int q, int lane,
                                          int r0) {
  BoxOut w;
  const int64_t j = t.m0 + q * 32 + lane, row0 = t.n0 + r0;
  w.jv = j < g.M;
  const int64_t left = g.N - row0;
  w.rows = left >= 32 ? 32 : (int)(left > 0 ? left : 0);
  w.ld = g.M;
  w.p = g.out + (w.rows > 0 && w.jv ? row0 * g.M + j : 0);
  return w;
}

// ---------------------------------------------------------------------------
// grad_X epilogue.  The accumulator holds P^T: TMEM lane = output column j of
// grad_X, TMEM column = row k of dH, so each thread owns one column j and the
// rows of a BHQ block are consecutive registers of one thread.
//
// Dequantization (Eq. 9).  With a the centred codes of Q_b2 (code - 2^(b-1)),
// w those of W~, the row offset 2^(b-1) + z'_k = m_k + d_k (m_k an integer,
// |d_k| <= 1/2) and y = 2^(bw-1) + z_w,
//   V_kj = sum_c (a_kc + m_k + d_k)(w_cj + y) = I_kj + y R_k + d_k U_j,
//   I_kj = P_kj + m_k CWc_j (an exact integer), CWc_j = sum_c w_cj,
//   R_k = sum_c (a_kc + m_k), U_j = CWc_j + C y = col_sum_w_j + C z_w,
// and grad_X = inv_sw diag(inv_s) Q_blk V.  The reflection is linear in the
// rows: Q V = Q I + y (Q R) 1^T + (Q d) U^T, with Q R and Q d per row (hr,
// hz; the identity for PTQ / PSQ).  Per block of nb rows with lead p,
//   (Q I)_k = I_k - beta (k != p),  (Q I)_p = rho S,
//   S = sum_k I_k, beta = kappa (rho S - I_p), rho = 1/sqrt(nb),
//   kappa = rho / (1 - rho).
// S and I_p are exact integers, beta is formed in float-float and split into
// an integer and a remainder, so I_k - beta loses nothing to the cancellation
// of the reflection: every term left in fp32 is small or row-constant.
//
// Two forms of the integer part, chosen per tile from the largest row offset
// |m_k| of its rows:
//   fp32   every |I| (2 + sqrt(nb)) below 2^24 (|I| below 2^24 without
//          reflection): one exact chunk and |m_k| <= flt_mmax;
//   int32  every |I| (2 + sqrt(nb)) below 2^31: |m_k| <= i32_mmax.  Every sum
//          then fits in int32 (wrapping partial sums are harmless) and each
//          result is one rounding of the exact integer.
// A tile outside both keeps its exact products P (as int32 bit patterns
// after several chunks) and the CTA finishes it after its last tile in int64
// and float-float (gradx_raw_fix).  Conversions to and from 64-bit integers
// run on the FP64 pipe, which is narrow on this GPU: the per-element path
// uses none.
// ---------------------------------------------------------------------------
// fp32 integers of magnitude below 2^22 to int32 with one FADD: x + 1.5 2^23
// holds x in its low mantissa bits.
constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23
constexpr uint32_t kMagicBits = 0x4B400000u;

__device__ __forceinline__ uint32_t magic_bits(float x) {
  return __float_as_uint(__fadd_rn(x, kMagic));
}

__device__ __forceinline__ int magic_int(float x) { return (int)(magic_bits(x) - kMagicBits); }

// beta = kappa (rho S - I_p) split as bi + bf (bi an integer, |bi| < 2^31 in
// the int32 form) and the lead value rho S, for a block of nact >= 2 rows.
struct BlockFix {
  float bf, lead;
  int bi;
};

__device__ __forceinline__ BlockFix block_fix(const HhConst &c, long long S, int Ip) {
  const ff rS = ff_mul(c.rho, ff_from_int(S));
  const ff w = ff_add(rS, ff_neg(ff_from_i32s(Ip)));
  const ff beta = ff_mul(c.kap, w);
  BlockFix f;
  const float bi = rintf(beta.h);
  f.bi = __float2int_rn(bi);
  f.bf = __fadd_rn(__fsub_rn(beta.h, bi), beta.l);
  f.lead = ff_round(rS);
  return f;
}

// out = sc (t + hz U) + sc y hr, with kq = (sc, sc hz, sc y hr, m)
__device__ __forceinline__ float dequant(const float4 &kq, float t, float U) {
  return __fmaf_rn(kq.x, t, __fmaf_rn(kq.y, U, kq.z));
}

// The integer parts I = P + m CWc of 32 rows (one box) of this thread's
// column in the int32 form.
struct Ints {
  int v[32];
  __device__ __forceinline__ float f(int i) const { return __int2float_rn(v[i]); }
  __device__ __forceinline__ float minus(int i, const BlockFix &b) const {
    return __fsub_rn(__int2float_rn((int)((uint32_t)v[i] - (uint32_t)b.bi)), b.bf);
  }
};

// The exact products P of one TMEM column group: the chunk's fp32 value plus
// the int32 running sum of the earlier chunks.
__device__ __forceinline__ void load_products(uint32_t acc, uint32_t ints, bool multi, int c0,
                                              int (&P)[32]) {
  uint32_t r[32], s[32];
  tmem_ld32_nw(acc + (uint32_t)c0, r);
  if (multi) tmem_ld32_nw(ints + (uint32_t)c0, s);
  tmem_wait_ld(r);
  if (multi) tmem_wait_ld(s);
#pragma unroll
  for (int i = 0; i < 32; ++i)
    P[i] = (int)((uint32_t)__float2int_rn(__uint_as_float(r[i])) + (multi ? s[i] : 0u));
}

// Loads the products of the 32 rows at TMEM column c0 and forms I
// (|m| <= i32_mmax and |CWc| <= C 2^(bw-1) are below 2^22).
__device__ __forceinline__ void load_ints(uint32_t acc, uint32_t ints, bool multi, int c0,
                                          const float4 *kp, float cwc, Ints &I) {
  load_products(acc, ints, multi, c0, I.v);
  const uint32_t cw = (uint32_t)magic_int(cwc);
#pragma unroll
  for (int i = 0; i < 32; ++i)
    I.v[i] = (int)((uint32_t)I.v[i] + (uint32_t)magic_int(kp[c0 + i].w) * cw);
}

// I of one row (TMEM column col) of this thread's column.
__device__ __forceinline__ int load_int1(uint32_t acc, uint32_t ints, bool multi, int col,
                                         float m, float cwc) {
  uint32_t v[2];
  v[0] = tmem_ld1_nw(acc + (uint32_t)col);
  v[1] = multi ? tmem_ld1_nw(ints + (uint32_t)col) : 0u;
  tmem_wait_ld(v);
  const uint32_t P = (uint32_t)__float2int_rn(__uint_as_float(v[0])) + v[1];
  return (int)(P + (uint32_t)magic_int(m) * (uint32_t)magic_int(cwc));
}

// One box (32 rows r0 .. r0 + 31 of the tile) of blocks of NB <= 32 rows:
// reflection, dequantization, store into the swizzled box.
// lead products loaded per box: one per block of NB <= 32 rows
__host__ __device__ constexpr int leads_per_box(int nb) { return nb > 1 && nb <= 32 ? 32 / nb : 1; }

template <int NB>
__device__ __forceinline__ void box_small(const Ints &I, const int (&Ip)[leads_per_box(NB)],
                                          const HhConst &hc, const float4 *kp,
                                          const int *leads, int r0, int64_t row0,
                                          int64_t N, float U, const BoxOut &w) {
  if (NB == 1) {
#pragma unroll
    for (int i = 0; i < 32; ++i) w.st(i, dequant(kp[r0 + i], I.f(i), U));
    return;
  }
  constexpr int NBB = NB > 1 ? NB : 2;
#pragma unroll
  for (int b = 0; b < 32 / NBB; ++b) {
    const int kb0 = r0 + b * NBB;
    const int64_t left = N - (row0 + b * NBB);
    const int nact = left >= NBB ? NBB : (int)(left > 0 ? left : 0);
    if (nact < 2) {  // a one-row block is not transformed
#pragma unroll
      for (int l = 0; l < NBB; ++l) w.st(b * NBB + l, dequant(kp[kb0 + l], I.f(b * NBB + l), U));
      continue;
    }
    long long S = 0;
#pragma unroll
    for (int l = 0; l < NBB; ++l) S += I.v[b * NBB + l];
    const BlockFix f = block_fix(nact == NBB ? hc : hh_const(nact), S, Ip[b]);
#pragma unroll
    for (int l = 0; l < NBB; ++l) w.st(b * NBB + l, dequant(kp[kb0 + l], I.minus(b * NBB + l, f), U));
    const int p = leads[kb0 / NBB];  // the lead row: a later store of the same thread
    w.st(b * NBB + p, dequant(kp[kb0 + p], f.lead, U));
  }
}

// The final chunk of one tile for this warp in the int32 form: groups of GW
// rows (a box, or one block of NB > 32 rows spanning several boxes).  raw: a
// tile outside both forms, whose row terms are units (m = 0, so I = P): its
// exact products P are stored as int32 bit patterns for gradx_raw_fix.
template <int NB>
__device__ __forceinline__ void gradx_tile(const GemmArgs &g, const Item &t, uint32_t acc,
                                           uint32_t ints, bool multi, const float4 *kp,
                                           const int *leads, const HhConst &hc, float cwc,
                                           float U, uint64_t *acce_set, int q, int lane,
                                           bool raw) {
  constexpr int GW = NB > 32 ? NB : 32;
  constexpr int NPP = leads_per_box(NB);
#pragma unroll 1
  for (int g0 = 0; g0 < BN; g0 += GW) {
    // blocks of more than 32 rows: their sums over all boxes first
    long long S_big = 0;
    int Ip_big = 0, p_big = 0;
    if (NB > 32) {
#pragma unroll 1
      for (int bx = 0; bx < GW / 32; ++bx) {
        Ints I;
        load_ints(acc, ints, multi, g0 + bx * 32, kp, cwc, I);
#pragma unroll
        for (int i = 0; i < 32; ++i) S_big += I.v[i];
      }
      p_big = leads[g0 / (NB > 32 ? NB : 1)];
      Ip_big = load_int1(acc, ints, multi, g0 + p_big, kp[g0 + p_big].w, cwc);
    }
#pragma unroll 1
    for (int bx = 0; bx < GW / 32; ++bx) {
      const int r0 = g0 + bx * 32;
      const BoxOut w = box_out(g, t, q, lane, r0);
      Ints I;
      load_ints(acc, ints, multi, r0, kp, cwc, I);
      int Ip[NPP];
#pragma unroll
      for (int b = 0; b < NPP; ++b) {
        Ip[b] = 0;
        if (NB > 1 && NB <= 32) {
          const int col = r0 + b * (32 / NPP) + leads[(r0 + b * (32 / NPP)) / (32 / NPP)];
          Ip[b] = load_int1(acc, ints, multi, col, kp[col].w, cwc);
        }
      }
      if (r0 + 32 == BN) {  // the accumulator has been read in full
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acce_set);
      }
      if (raw) {
        w.st32(reinterpret_cast<const float (&)[32]>(I.v));
        continue;
      }
      if constexpr (NB <= 32) {
        box_small<NB>(I, Ip, hc, kp, leads, r0, t.n0 + r0, g.N, U, w);
      } else {
        const int64_t left = g.N - (t.n0 + g0);
        const int nact = left >= NB ? NB : (int)(left > 0 ? left : 0);
        if (nact < 2) {
#pragma unroll
          for (int i = 0; i < 32; ++i) w.st(i, dequant(kp[r0 + i], I.f(i), U));
        } else {
          const BlockFix f = block_fix(nact == NB ? hc : hh_const(nact), S_big, Ip_big);
#pragma unroll
          for (int i = 0; i < 32; ++i) w.st(i, dequant(kp[r0 + i], I.minus(i, f), U));
          if (p_big >= bx * 32 && p_big < bx * 32 + 32)
            w.st(p_big - bx * 32, dequant(kp[g0 + p_big], f.lead, U));
        }
      }
    }
  }
}

struct BlockFixF {
  float bi, bf, lead;
};

__device__ __forceinline__ BlockFixF block_fix_f(const HhConst &c, int S, int Ip) {
  const ff rS = ff_mul(c.rho, ff_from_i32s(S));
  const ff w = ff_add(rS, ff_neg(ff_from_i32s(Ip)));
  const ff beta = ff_mul(c.kap, w);
  BlockFixF f;
  f.bi = rintf(beta.h);
  f.bf = __fadd_rn(__fsub_rn(beta.h, f.bi), beta.l);
  f.lead = ff_round(rS);
  return f;
}

// (Q I)_k of a non-lead row in the fp32 form: (P - bi) + m CWc is exact
// (every magnitude below 2^24), then the remainder bf.
__device__ __forceinline__ float reflect_f(float P, const float4 &kq, float cwc,
                                           const BlockFixF &f) {
  return __fsub_rn(__fmaf_rn(kq.w, cwc, __fsub_rn(P, f.bi)), f.bf);
}

// The final chunk of one tile in the fp32 form (one exact chunk, |P| < 2^22,
// |m| <= mmax).  Block sums S = sum P + CWc sum m, I_p = P_p + m_p CWc.
// raw: a tile outside the fp32 form, whose row terms are units (1, 0, 0, 0):
// no block is transformed, so the stores are its exact products P.
template <int NB>
__device__ __forceinline__ void gradx_tile_f(const GemmArgs &g, const Item &t, uint32_t acc,
                                             const float4 *kp, const int *leads,
                                             const int *msum, const HhConst &hc, float cwc,
                                             float U, uint64_t *acce_set, int q, int lane,
                                             bool raw) {
  constexpr int GW = NB > 32 ? NB : 32;
  constexpr int NPP = leads_per_box(NB);
  constexpr int NBD = NB > 1 ? NB : 1;
  const int cwi = (int)cwc;
  if constexpr (NB <= 32) {
    // one block (NB >= 8) or 16 rows (no reflection) per step, loaded from
    // TMEM on its own, so few values are live at a time
    constexpr int CH = NB >= 8 ? NB : (NB <= 1 ? 16 : 8);
    constexpr int BPC = NB > 1 ? CH / NB : 0;  // blocks per chunk
    const int64_t j = t.m0 + q * 32 + lane;
    const bool jv = j < g.M;
#pragma unroll 1
    for (int r0 = 0; r0 < BN; r0 += CH) {
      uint32_t r[CH];
      tmem_ldw_nw<CH>(acc + (uint32_t)r0, r);
      uint32_t pp[BPC > 0 ? BPC : 1];
#pragma unroll
      for (int b = 0; b < BPC; ++b)
        pp[b] = tmem_ld1_nw(acc + (uint32_t)(r0 + b * NBD + leads[(r0 + b * NBD) / NBD]));
      tmem_wait_ld(r);
      if (BPC > 0) tmem_wait_ld(pp);
      if (r0 + CH == BN) {  // the accumulator has been read in full
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acce_set);
      }
      const int64_t row0 = t.n0 + r0;
      const int64_t left = g.N - row0;
      const int rows = left >= CH ? CH : (int)(left > 0 ? left : 0);
      float *po = g.out + (jv && rows > 0 ? row0 * g.M + j : 0);
      if constexpr (NB <= 1) {
#pragma unroll
        for (int i = 0; i < CH; ++i) {
          const float4 kq = kp[r0 + i];
          r[i] = __float_as_uint(dequant(kq, __fmaf_rn(kq.w, cwc, __uint_as_float(r[i])), U));
        }
      }
      int lrow[BPC > 0 ? BPC : 1];
      float lval[BPC > 0 ? BPC : 1];
#pragma unroll
      for (int b = 0; b < (BPC > 0 ? BPC : 1); ++b) {
        lrow[b] = -1;
        lval[b] = 0.0f;
      }
      if constexpr (NB > 1) {
#pragma unroll
        for (int b = 0; b < BPC; ++b) {
          const int kb0 = r0 + b * NBD;
          const int64_t lb = g.N - (t.n0 + kb0);
          const int nact = lb >= NBD ? NBD : (int)(lb > 0 ? lb : 0);
          if (nact < 2 || raw) {  // a one-row block is not transformed
#pragma unroll
            for (int l = 0; l < NBD; ++l) {
              const float4 kq = kp[kb0 + l];
              r[b * NBD + l] = __float_as_uint(
                  dequant(kq, __fmaf_rn(kq.w, cwc, __uint_as_float(r[b * NBD + l])), U));
            }
            continue;
          }
          uint32_t sb = 0u;
#pragma unroll
          for (int l = 0; l < NBD; ++l) sb += magic_bits(__uint_as_float(r[b * NBD + l]));
          const int S = (int)(sb - (uint32_t)NBD * kMagicBits) + cwi * msum[kb0 / NBD];
          const int p = leads[kb0 / NBD];
          const float4 kl = kp[kb0 + p];
          const int Ip = magic_int(__uint_as_float(pp[b])) + (int)kl.w * cwi;
          const BlockFixF f = block_fix_f(nact == NBD ? hc : hh_const(nact), S, Ip);
#pragma unroll
          for (int l = 0; l < NBD; ++l) {
            const float4 kq = kp[kb0 + l];
            r[b * NBD + l] = __float_as_uint(
                dequant(kq, reflect_f(__uint_as_float(r[b * NBD + l]), kq, cwc, f), U));
          }
          lrow[b] = b * NBD + p;
          lval[b] = dequant(kl, f.lead, U);
        }
      }
      if constexpr (NB == 0) {
        // adaptive groups: row r0 + i of the tile is row leads[r0 + i] of grad_X
        if (jv) {
#pragma unroll
          for (int i = 0; i < CH; ++i)
            if (i < rows) __stcs(g.out + (int64_t)leads[r0 + i] * g.M + j, __uint_as_float(r[i]));
        }
      } else if (jv) {
        if (rows == CH) {
#pragma unroll
          for (int i = 0; i < CH; ++i) __stcs(po + (int64_t)i * g.M, __uint_as_float(r[i]));
        } else {
#pragma unroll
          for (int i = 0; i < CH; ++i)
            if (i < rows) __stcs(po + (int64_t)i * g.M, __uint_as_float(r[i]));
        }
        // the lead rows: later stores of the same thread to the same address
#pragma unroll
        for (int b = 0; b < BPC; ++b)
          if (lrow[b] >= 0 && lrow[b] < rows) __stcs(po + (int64_t)lrow[b] * g.M, lval[b]);
      }
    }
  } else {
#pragma unroll 1
  for (int g0 = 0; g0 < BN; g0 += GW) {
    int S_big = 0, Ip_big = 0, p_big = 0;
    if constexpr (NB > 32) {
      uint32_t sb = 0u;
#pragma unroll 1
      for (int bx = 0; bx < GW / 32; ++bx) {
        uint32_t r[32];
        tmem_ld32_nw(acc + (uint32_t)(g0 + bx * 32), r);
        tmem_wait_ld(r);
#pragma unroll
        for (int i = 0; i < 32; ++i) sb += magic_bits(__uint_as_float(r[i]));
      }
      S_big = (int)(sb - (uint32_t)NB * kMagicBits) + cwi * msum[g0 / NBD];
      p_big = leads[g0 / NBD];
      uint32_t v[1];
      v[0] = tmem_ld1_nw(acc + (uint32_t)(g0 + p_big));
      tmem_wait_ld(v);
      Ip_big = magic_int(__uint_as_float(v[0])) + (int)kp[g0 + p_big].w * cwi;
    }
#pragma unroll 1
    for (int bx = 0; bx < GW / 32; ++bx) {
      const int r0 = g0 + bx * 32;
      const BoxOut w = box_out(g, t, q, lane, r0);
      uint32_t r[32];
      tmem_ld32_nw(acc + (uint32_t)r0, r);
      uint32_t pp[NPP];
#pragma unroll
      for (int b = 0; b < NPP; ++b)
        pp[b] = (NB > 1 && NB <= 32)
                    ? tmem_ld1_nw(acc + (uint32_t)(r0 + b * NBD + leads[(r0 + b * NBD) / NBD]))
                    : 0u;
      tmem_wait_ld(r);
      tmem_wait_ld(pp);
      if (r0 + 32 == BN) {  // the accumulator has been read in full
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acce_set);
      }
      // every output of the box is formed in registers before the first
      // store, so the per-row loads from shared memory need not wait for
      // the stores into the (possibly aliasing) box
      // outputs overwrite the products in place (r holds fp32 bit patterns)
      int lead_row = -1;
      float lead_val = 0.0f;
      if constexpr (NB == 1) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float4 kq = kp[r0 + i];
          r[i] = __float_as_uint(dequant(kq, __fmaf_rn(kq.w, cwc, __uint_as_float(r[i])), U));
        }
      } else if constexpr (NB <= 32) {
        float lv[32 / NBD];
        int lp[32 / NBD];
#pragma unroll
        for (int b = 0; b < 32 / NBD; ++b) {
          const int kb0 = r0 + b * NBD;
          const int64_t left = g.N - (t.n0 + kb0);
          const int nact = left >= NBD ? NBD : (int)(left > 0 ? left : 0);
          lp[b] = -1;
          lv[b] = 0.0f;
          if (nact < 2 || raw) {  // a one-row block is not transformed
#pragma unroll
            for (int l = 0; l < NBD; ++l) {
              const float4 kq = kp[kb0 + l];
              r[b * NBD + l] = __float_as_uint(dequant(kq, __fmaf_rn(kq.w, cwc, __uint_as_float(r[b * NBD + l])), U));
            }
            continue;
          }
          uint32_t sb = 0u;
#pragma unroll
          for (int l = 0; l < NBD; ++l) sb += magic_bits(__uint_as_float(r[b * NBD + l]));
          const int S = (int)(sb - (uint32_t)NBD * kMagicBits) + cwi * msum[kb0 / NBD];
          const int p = leads[kb0 / NBD];
          const int Ip = magic_int(__uint_as_float(pp[b])) + (int)kp[kb0 + p].w * cwi;
          const BlockFixF f = block_fix_f(nact == NBD ? hc : hh_const(nact), S, Ip);
#pragma unroll
          for (int l = 0; l < NBD; ++l) {
            const float4 kq = kp[kb0 + l];
            r[b * NBD + l] = __float_as_uint(dequant(kq, reflect_f(__uint_as_float(r[b * NBD + l]), kq, cwc, f), U));
          }
          lp[b] = b * NBD + p;
          lv[b] = dequant(kp[kb0 + p], f.lead, U);
        }
        w.st32(reinterpret_cast<const float (&)[32]>(r));
        // the lead rows: later stores of the same thread
#pragma unroll
        for (int b = 0; b < 32 / NBD; ++b)
          if (lp[b] >= 0) w.st(lp[b], lv[b]);
      } else {
        const int64_t left = g.N - (t.n0 + g0);
        const int nact = left >= NB ? NB : (int)(left > 0 ? left : 0);
        if (nact < 2 || raw) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float4 kq = kp[r0 + i];
            r[i] = __float_as_uint(dequant(kq, __fmaf_rn(kq.w, cwc, __uint_as_float(r[i])), U));
          }
        } else {
          const BlockFixF f = block_fix_f(nact == NB ? hc : hh_const(nact), S_big, Ip_big);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float4 kq = kp[r0 + i];
            r[i] = __float_as_uint(dequant(kq, reflect_f(__uint_as_float(r[i]), kq, cwc, f), U));
          }
          if (p_big >= bx * 32 && p_big < bx * 32 + 32) {
            lead_row = p_big - bx * 32;
            lead_val = dequant(kp[g0 + p_big], f.lead, U);
          }
        }
      }
      if constexpr (NB == 1 || NB > 32) {
        w.st32(reinterpret_cast<const float (&)[32]>(r));
        if (lead_row >= 0) w.st(lead_row, lead_val);
      }
    }
  }
  }
}

// The global inputs of one tile's parameters (lane-owned rows and columns).
struct TileLoads {
  float inv[BN / 32], zero[BN / 32], hz[BN / 32], hr[BN / 32];
  int rs[BN / 32], cs[BM / 32], lead[2];
  int gs[BN / 32], pr[BN / 32];  // NB = 0: group size and output row
};

template <int NB>
__device__ __forceinline__ void tile_loads(const GemmArgs &g, const Item &t, int lane,
                                           TileLoads &L) {
  constexpr int NBD = NB > 1 ? NB : 1;
#pragma unroll
  for (int i = 0; i < BN / 32; ++i) {
    const int64_t k = t.n0 + lane + 32 * i;
    const bool kv = k < g.N;
    const int64_t ri = g.kind == FQT_PTQ ? 0 : (kv ? k : 0);
    L.inv[i] = kv ? __ldg(g.inv_s + ri) : 0.0f;
    L.zero[i] = kv ? __ldg(g.zero + ri) : 0.0f;
    if (NB > 1) {
      L.hz[i] = kv ? __ldg(g.hz + k) : 0.0f;
      L.hr[i] = kv ? __ldg(g.hr + k) : 0.0f;
      L.rs[i] = 0;
    } else {
      L.hz[i] = L.hr[i] = 0.0f;
      L.rs[i] = kv ? __ldg(g.row_sum + k) : 0;
    }
    if (NB == 0) {
      L.gs[i] = kv ? __ldg(g.gsize + k) : 1;
      L.pr[i] = kv ? __ldg(g.perm + k) : 0;
    } else {
      L.gs[i] = 1;
      L.pr[i] = 0;
    }
  }
#pragma unroll
  for (int i = 0; i < BM / 32; ++i) {
    const int64_t j = t.m0 + lane + 32 * i;
    L.cs[i] = j < g.M ? __ldg(g.col_sum_w + j) : 0;
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {  // BN / NB <= 64 blocks per tile
    const int b = lane + 32 * u;
    L.lead[u] = 0;
    if (NB > 1 && b < BN / NBD) {
      const int64_t kb = t.n0 / NBD + b;
      L.lead[u] = kb * NBD < g.N ? __ldg(g.lead + kb) : 0;
    }
  }
}

// Parameter loader of grad_X (one warp): for every tile of this CTA, in
// order, the per-row terms of its rows and the column sums of its columns go
// into a parameter stage ahead of the epilogue warps that use them.  The
// global loads of the next tile are in flight while this tile's are used.
template <int NB, int FORM>
__device__ __forceinline__ void gradx_params(const GemmArgs &g, uint8_t *smem, uint64_t *pfull,
                                             uint64_t *pempty, volatile int *abort_flag,
                                             int lane) {
  uint32_t *raw_mask = reinterpret_cast<uint32_t *>(smem + kOffRaw);
  const float inv_sw = *g.inv_sw, zw = *g.zero_w;
  const ff y = two_sum((float)g.ow, zw);
  const int Cn = (int)g.K;
  TileLoads cur, nxt;
  if ((int64_t)blockIdx.x < g.n_items) tile_loads<NB>(g, decode_item(g, blockIdx.x), lane, cur);
  int64_t local = 0;
  for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x, ++local) {
    if (it + gridDim.x < g.n_items) tile_loads<NB>(g, decode_item(g, it + gridDim.x), lane, nxt);
    const int s = (int)(local % kParStages);
    const uint32_t wrap = (uint32_t)(local / kParStages);
    const bool got = mbar_wait(&pempty[s], (wrap & 1u) ^ 1u, g.status);
    if (!__all_sync(0xffffffffu, got)) { *abort_flag = 1; break; }
    const Item t = decode_item(g, it);
    uint8_t *P = smem + kOffPar + (size_t)s * kParBytes;
    float4 *kp = reinterpret_cast<float4 *>(P);
    int *leads = reinterpret_cast<int *>(P + kParLeads);
    int *msum = reinterpret_cast<int *>(P + kParMsum);
    int *cs = reinterpret_cast<int *>(P + kParCs);
    float mabs = 0.0f;
    float mrow[BN / 32];
#pragma unroll
    for (int i = 0; i < BN / 32; ++i) {
      const int64_t k = t.n0 + lane + 32 * i;
      float sc = 0.0f, A = 0.0f, B = 0.0f, m = 0.0f;
      if (k < g.N) {
        sc = __fmul_rn(inv_sw, cur.inv[i]);
        const ff x = two_sum((float)g.og, cur.zero[i]);
        m = rintf(x.h);
        float hd, hR;
        if (NB > 1) {
          hd = cur.hz[i];
          hR = cur.hr[i];
        } else {
          // R = sum_c (a + m); rounding relative to R itself suffices for a
          // row-constant term
          hd = ff_round(fast_two_sum(__fsub_rn(x.h, m), x.l));
          hR = __fadd_rn((float)(cur.rs[i] - Cn * g.og), __fmul_rn((float)Cn, m));
        }
        A = __fmul_rn(sc, hd);
        B = __fmul_rn(sc, __fmaf_rn(hR, y.h, __fmul_rn(hR, y.l)));
        if (NB == 0 && (cur.gs[i] > 1 || !(fabsf(m) <= g.raw_mmax))) {
          // finished by the group pass: the exact integer product P alone
          sc = 1.0f;
          A = B = m = 0.0f;
        }
      }
      kp[lane + 32 * i] = make_float4(sc, A, B, m);
      mabs = fmaxf(mabs, fabsf(m));
      mrow[i] = m;
    }
    if constexpr (NB == 0) {
#pragma unroll
      for (int i = 0; i < BN / 32; ++i)
        leads[lane + 32 * i] = min(max(cur.pr[i], 0), (int)(g.N - 1));
    }
    if constexpr (NB > 1) {
      // sums of m over each block (the fp32 form's S = sum P + CWc sum m)
      constexpr int SEG = NB > 32 ? 32 : NB;
#pragma unroll
      for (int i = 0; i < BN / 32; ++i) {
        float v = mrow[i];
#pragma unroll
        for (int off = 1; off < SEG; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        mrow[i] = v;
      }
      if constexpr (NB <= 32) {
#pragma unroll
        for (int i = 0; i < BN / 32; ++i)
          if (lane % NB == 0) msum[(32 * i + lane) / NB] = (int)mrow[i];
      } else if (lane == 0) {
#pragma unroll
        for (int b = 0; b < BN / NB; ++b) {
          float v = 0.0f;
#pragma unroll
          for (int i = 0; i < NB / 32; ++i) v += mrow[b * (NB / 32) + i];
          msum[b] = (int)v;
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u)
        if (lane + 32 * u < BN / NB) leads[lane + 32 * u] = cur.lead[u];
    }
#pragma unroll
    for (int i = 0; i < BM / 32; ++i) cs[lane + 32 * i] = cur.cs[i];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
      mabs = fmaxf(mabs, __shfl_xor_sync(0xffffffffu, mabs, off));
    // a tile with a row offset beyond its forms (FORM 2: the fp32 form;
    // otherwise the int32 form, which holds more) keeps the exact products P
    // (unit row terms); its bit sends it to the CTA's final pass
    // (gradx_raw_fix)
    const bool raw = NB != 0 && !(mabs <= (FORM == 2 ? g.flt_mmax : g.i32_mmax));
    if (raw) {
#pragma unroll
      for (int i = 0; i < BN / 32; ++i) kp[lane + 32 * i] = make_float4(1.0f, 0.0f, 0.0f, 0.0f);
      if (lane == 0 && local < kMaxLocalTiles) raw_mask[local >> 5] |= 1u << (local & 31);
    }
    // 1: the fp32 form, 2: the int32 form, 0: raw
    if (lane == 0)
      *reinterpret_cast<int *>(P + kParFlag) =
          NB == 0 || (FORM == 2 && !raw) || (FORM == 1 && mabs <= g.flt_mmax) ? 1
          : raw                                                             ? 0
                                                                            : 2;
    __syncwarp();
    if (lane == 0) mbar_arrive(&pfull[s]);
    cur = nxt;
  }
}

template <int NB, int FORM>
__device__ __forceinline__ void gradx_epilogue(const GemmArgs &g, uint8_t *smem,
                                               uint8_t *ring, uint64_t *accf,
                                               uint64_t *acce, uint64_t *pfull,
                                               uint64_t *pempty, uint32_t tmem,
                                               const CUtensorMap *tmOut,
                                               volatile int *abort_flag, int warp,
                                               int lane) {
  const int ew = warp - kGemmWarpEpi0;
  const int q = warp & 3;     // TMEM lane quadrant: columns j = 32q .. 32q + 31
  const int set = ew >> 2;    // the tiles (every g.sets-th one) this warp serves
  const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
  const float zw = *g.zero_w;
  const int Cn = (int)g.K;
  HhConst hc = {{0.0f, 0.0f}, {0.0f, 0.0f}};
  if (NB > 1) hc = hh_const(NB);
  bool ok = true;
  // this CTA's tiles local = set, set + g.sets, ... (item blockIdx.x + local * grid)
  for (int64_t local = set; set < g.sets; local += g.sets) {
    const int64_t it = (int64_t)blockIdx.x + local * (int64_t)gridDim.x;
    if (it >= g.n_items || *abort_flag) break;
    const Item t = decode_item(g, it);
    const int buf = (int)(local & (g.nacc - 1));
    const uint32_t acc = lane_base + (uint32_t)(buf * BN);
    // int32 running sums (two accumulators only): columns 256 + 128 buf
    const uint32_t ints = lane_base + (uint32_t)(2 * BN + buf * BN);
    const int64_t nchunks = (t.kb1 - t.kb0 + g.kc_blocks - 1) / g.kc_blocks;
    const bool active = t.m0 + q * 32 < g.M;  // warp-uniform
    const int s = (int)(local % kParStages);
    const bool gotp = mbar_wait(&pfull[s], (uint32_t)(local / kParStages) & 1u, g.status);
    if (!__all_sync(0xffffffffu, gotp)) { ok = false; break; }
    const uint8_t *P = smem + kOffPar + (size_t)s * kParBytes;
    const float4 *kp = reinterpret_cast<const float4 *>(P);
    const int *leads = reinterpret_cast<const int *>(P + kParLeads);
    const int *msum = reinterpret_cast<const int *>(P + kParMsum);
    const int cs = reinterpret_cast<const int *>(P + kParCs)[q * 32 + lane];
    const int tform = *reinterpret_cast<const int *>(P + kParFlag);  // 1 fp32, 2 int32, 0 raw
    const float cwc = (float)(cs - Cn * g.ow);
    const float U = __fmaf_rn((float)Cn, zw, (float)cs);
    for (int64_t c = 0; c < nchunks; ++c) {
      // every tile has nchunks chunks: the use count of this accumulator
      // before chunk c of this tile gives the phase
      const uint32_t par = (uint32_t)(((local / g.nacc) * nchunks + c) & 1);
      const bool got = !*abort_flag && mbar_wait(&accf[buf], par, g.status);
      if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
      tc_fence_after();
      const bool last_chunk = c + 1 == nchunks;
      if (!last_chunk && active) {
        // exact chunk boundary: fold the chunk into the int32 running sum
#pragma unroll 1
        for (int grp = 0; grp < BN / 32; ++grp) {
          uint32_t r[32];
          tmem_ld32_nw(acc + (uint32_t)(grp * 32), r);
          tmem_wait_ld(r);
          if (c > 0) {
            uint32_t sr[32];
            tmem_ld32_nw(ints + (uint32_t)(grp * 32), sr);
            tmem_wait_ld(sr);
#pragma unroll
            for (int i = 0; i < 32; ++i)
              r[i] = (uint32_t)(__float2int_rn(__uint_as_float(r[i])) + (int)sr[i]);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = (uint32_t)__float2int_rn(__uint_as_float(r[i]));
          }
          tmem_st32(ints + (uint32_t)(grp * 32), r);
        }
        tmem_wait_st();
      }
      if (!last_chunk || !active) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[buf]);
        continue;
      }
      const bool multi = c > 0;
      if constexpr (NB == 0) {
        gradx_tile_f<0>(g, t, acc, kp, leads, msum, hc, cwc, U, &acce[buf], q, lane, false);
      } else {
        if constexpr (FORM == 2) {
          // a tile outside the fp32 form has unit row terms (kq = (1, 0, 0, 0)):
          // the one-row epilogue stores its exact products P for gradx_raw_fix
          gradx_tile_f<NB>(g, t, acc, kp, leads, msum, hc, cwc, U, &acce[buf], q, lane,
                           tform != 1);
        } else if (FORM == 1 && tform == 1) {
          gradx_tile_f<NB>(g, t, acc, kp, leads, msum, hc, cwc, U, &acce[buf], q, lane, false);
        } else {
          gradx_tile<NB>(g, t, acc, ints, multi, kp, leads, hc, cwc, U, &acce[buf], q, lane,
                         tform == 0);
        }
      }
    }
    // the parameter stage is free again
    __syncwarp();
    if (lane == 0) mbar_arrive(&pempty[s]);
    if (!ok) break;
  }
  if (!ok) *abort_flag = 1;
}

// ---------------------------------------------------------------------------
// Split-K partial epilogue: each warp owns TMEM lanes 32q .. 32q + 31 (rows)
// and 64 columns, stored as two 32 x 32 int32 boxes (3-D tensor map over
// splits x M x N) from a ring of boxes.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void partial_epilogue(const GemmArgs &g, uint8_t *ring,
                                                 uint64_t *accf, uint64_t *acce,
                                                 uint32_t tmem, const CUtensorMap *tmOut,
                                                 volatile int *abort_flag, int warp,
                                                 int lane) {
  const int ew = warp - kGemmWarpEpi0;
  const int q = warp & 3;
  const int hcol = ew >> 2;  // column half: 64 * hcol .. +63
  uint8_t *myring = ring + (size_t)ew * g.ring * kBoxBytes;
  int nbox = 0;
  const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
  const uint32_t int_cols = lane_base + (uint32_t)(2 * BN + hcol * 64);
  int buf = 0;
  uint32_t aph = 0u;  // bit b: phase parity of accumulator b
  bool ok = true;
  for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
    const Item t = decode_item(g, it);
    const int64_t nchunks = (t.kb1 - t.kb0 + g.kc_blocks - 1) / g.kc_blocks;
    for (int64_t c = 0; c < nchunks; ++c) {
      const bool got = !*abort_flag && mbar_wait(&accf[buf], (aph >> buf) & 1u, g.status);
      if (!__all_sync(0xffffffffu, got)) { ok = false; break; }
      tc_fence_after();
      const uint32_t accb = lane_base + (uint32_t)(buf * BN + hcol * 64);
      const bool last = c + 1 == nchunks;
#pragma unroll
      for (int grp = 0; grp < 2; ++grp) {
        uint32_t r[32];
        tmem_ld32_nw(accb + (uint32_t)(grp * 32), r);
        tmem_wait_ld(r);
        if (c > 0) {
          uint32_t s[32];
          tmem_ld32_nw(int_cols + (uint32_t)(grp * 32), s);
          tmem_wait_ld(s);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            r[j] = (uint32_t)(__float2int_rn(__uint_as_float(r[j])) + (int)s[j]);
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) r[j] = (uint32_t)__float2int_rn(__uint_as_float(r[j]));
        }
        if (!last) {
          tmem_st32(int_cols + (uint32_t)(grp * 32), r);
          continue;
        }
        if (grp == 1) {  // this accumulator is no longer read
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acce[buf]);
        }
        uint8_t *tile = myring + (size_t)(nbox % g.ring) * kBoxBytes;
        if (nbox >= g.ring) {
          if (lane == 0) bulk_wait_read(g.ring - 1);
          __syncwarp();
        }
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4)
          *reinterpret_cast<uint4 *>(tile + sw128_off(lane, j4)) =
              make_uint4(r[4 * j4], r[4 * j4 + 1], r[4 * j4 + 2], r[4 * j4 + 3]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_3d(tmOut, (int32_t)(t.n0 + hcol * 64 + grp * 32), (int32_t)(t.m0 + q * 32),
                       t.split, tile);
          bulk_commit();
        }
        ++nbox;
      }
      if (!last) {
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[buf]);
      }
      aph ^= 1u << buf;
      buf ^= 1;
    }
    if (!ok) break;
  }
  if (!ok) *abort_flag = 1;
  if (lane == 0) bulk_wait_all();
  __syncwarp();
}

// ---------------------------------------------------------------------------
// Byte operands of the split-K partials (both MN-major: K rows of 128 codes).
// TMA lands each operand's 128 x 64 byte tile in the stage (128-byte rows,
// 128-byte swizzle); kCvtWarps converter warps widen it into the fp16 carrier
// tile the MMA reads (two 64-wide swizzle atoms, as the fp16 boxes would
// land), code - 2^(b-1) exactly, rows past the end of the reduction as 0
// (a zero byte would widen to -2^(b-1)), then fence the writes for the
// tensor core and release the stage to the MMA issuer.
// ---------------------------------------------------------------------------
constexpr int kCvtWarps = 6;

// Shared-memory offsets of a converter thread's chunks (at most 3 of the
// 512 16-byte chunks of a 128 x 64 byte tile): the byte chunk, and the two
// fp16 chunks it widens into.
struct CvtSlots {
  int n;
  uint32_t src[3], dst0[3], dst1[3];
  int row[3];
};

__device__ __forceinline__ CvtSlots cvt_slots(int t) {
  CvtSlots o;
  o.n = 0;
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const int c = t + i * kCvtWarps * 32;
    const int r = c >> 3, j = c & 7, cc = (j & 3) * 2;
    const uint32_t base = (uint32_t)((j >> 2) * (kTileBytes / 2) + r * 128);
    o.src[i] = (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4));
    o.dst0[i] = base + (uint32_t)((cc ^ (r & 7)) << 4);
    o.dst1[i] = base + (uint32_t)(((cc + 1) ^ (r & 7)) << 4);
    o.row[i] = r;
    if (c < 512) o.n = i + 1;
  }
  return o;
}

// codes 16j .. 16j + 15 of a row: fp16 chunks 2 (j mod 4) and 2 (j mod 4) + 1
// of swizzle atom j / 4; rows from rows_valid on are 0
__device__ __forceinline__ void widen_tile(const uint8_t *src, uint8_t *dst, int rows_valid,
                                           __half2 bias, const CvtSlots &o) {
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    if (i >= o.n) break;
    uint4 lo = make_uint4(0u, 0u, 0u, 0u), hi = lo;
    if (o.row[i] < rows_valid) {
      const uint4 v = *reinterpret_cast<const uint4 *>(src + o.src[i]);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
      uint32_t h[8];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t a = __byte_perm(w[k], 0x6464u, 0x4140);
        const uint32_t b = __byte_perm(w[k], 0x6464u, 0x4342);
        __half2 x = __hsub2(*reinterpret_cast<const __half2 *>(&a), bias);
        __half2 y = __hsub2(*reinterpret_cast<const __half2 *>(&b), bias);
        h[2 * k] = *reinterpret_cast<uint32_t *>(&x);
        h[2 * k + 1] = *reinterpret_cast<uint32_t *>(&y);
      }
      lo = make_uint4(h[0], h[1], h[2], h[3]);
      hi = make_uint4(h[4], h[5], h[6], h[7]);
    }
    *reinterpret_cast<uint4 *>(dst + o.dst0[i]) = lo;
    *reinterpret_cast<uint4 *>(dst + o.dst1[i]) = hi;
  }
}

// Converter warp cw of kCvtWarps: byte stage su (ring of g.ustages) into
// carrier stage sf (ring of g.stages), in the producer's K-block order.
__device__ __noinline__ void partial_convert(const GemmArgs &g, uint8_t *ops, uint8_t *uops,
                                             uint64_t *full, uint64_t *empty, uint64_t *cvt,
                                             uint64_t *fempty, volatile int *abort_flag, int cw,
                                             int lane) {
  const CvtSlots slots = cvt_slots(cw * 32 + lane);
  const __half2 bias_a = __half2half2(__int2half_rn(1024 + (1 << (g.bw - 1))));
  const __half2 bias_b = __half2half2(__int2half_rn(1024 + (1 << (g.b2 - 1))));
  int su = 0, sf = 0;
  uint32_t phu = 0, phf = 0;
  for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
    const Item tt = decode_item(g, it);
    for (int64_t kb = tt.kb0; kb < tt.kb1; ++kb) {
      // the byte tiles have landed, and the MMA is done with the carrier stage
      bool got = mbar_wait(&full[su], phu, g.status);
      got = got && mbar_wait(&fempty[sf], phf ^ 1u, g.status);
      if (!__all_sync(0xffffffffu, got)) { *abort_flag = 1; return; }
      const uint8_t *us = uops + (size_t)su * kTileBytes;
      uint8_t *fs = ops + (size_t)sf * 2 * kTileBytes;
      const int64_t left = g.K - kb * BK;
      const int rows_valid = left >= BK ? BK : (int)(left > 0 ? left : 0);
      widen_tile(us, fs, rows_valid, bias_a, slots);
      widen_tile(us + kTileBytes / 2, fs + kTileBytes, rows_valid, bias_b, slots);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&cvt[sf]);    // the carrier stage is ready for the MMA
        mbar_arrive(&empty[su]);  // the byte stage is free for the next loads
      }
      if (++su == g.ustages) { su = 0; phu ^= 1u; }
      if (++sf == g.stages) { sf = 0; phf ^= 1u; }
    }
  }
}

// The tiles of this CTA left raw by the fp32-form epilogue (defined with the
// group fix-up, whose arithmetic it shares).
template <int NB>
__device__ __noinline__ void gradx_raw_fix(const GemmArgs &g, const uint32_t *raw_mask, int ew,
                                           int nwarps, int lane, bool p_bits);

template <int MODE, int NB, int FORM>
__global__ void __launch_bounds__(GemmLayout<MODE, FORM, NB>::threads, 1)
    k_gemm(const __grid_constant__ CUtensorMap tmA,
           const __grid_constant__ CUtensorMap tmB,
           const __grid_constant__ CUtensorMap tmOut, const GemmArgs g) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte alignment of the shared-window address (swizzle atoms)
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kOffBar);
  const int nstages = g.stages;
  const bool u8ops = MODE == MODE_PARTIAL && g.u8 != 0;
  const int ustages = u8ops ? g.ustages : 0;
  uint8_t *ops = smem + kFixedBytes;                                // carrier stages
  uint8_t *uops = ops + (size_t)nstages * 2 * kTileBytes;          // byte stages
  uint8_t *ring = uops + (size_t)ustages * kTileBytes;             // output boxes
  uint64_t *full = bars, *empty = bars + kMaxStages;
  uint64_t *accf = bars + 2 * kMaxStages, *acce = accf + 4;
  uint64_t *pfull = acce + 4, *pempty = pfull + 4, *drain = pempty + 4;
  // byte operands: carrier stage widened (converters -> MMA), carrier stage
  // consumed (MMA -> converters); full / empty then serve the byte ring
  uint64_t *cvt = bars + 2 * kMaxStages + 17, *fempty = cvt + kMaxStages;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + kNumBars);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  // grad_X: one accumulator per item, served by 4 epilogue warps (one per
  // lane quadrant); partials: accumulators alternate per chunk, 8 warps each
  constexpr bool kPerItem = MODE == MODE_GRADX;
  // grad_X with several exact chunks per tile (two accumulators, each tile on
  // its own): the operand ring carries two tiles at a time, chunk by chunk,
  // so that the fold of one tile's chunk overlaps the other tile's MMAs
  // (FORM 2 runs one exact chunk per tile: never pairs)
  const bool pairs = FORM != 2 && kPerItem && g.nacc == 2;
  const int64_t gstep = (pairs ? 2 : 1) * (int64_t)gridDim.x;
  constexpr uint32_t kEpiArrivals = kPerItem ? 4u : (uint32_t)kPartialEpiWarps;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    const int nring = u8ops ? ustages : nstages;
    for (int i = 0; i < nring; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], u8ops ? kCvtWarps : 1);
    }
    for (int i = 0; u8ops && i < nstages; ++i) {
      mbar_init(&cvt[i], kCvtWarps);
      mbar_init(&fempty[i], 1);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], kEpiArrivals);
      mbar_init(&pfull[i], 1);
      mbar_init(&pempty[i], 4);  // the 4 epilogue warps of the consuming set
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (MODE == MODE_GRADX && NB != 0)
    for (int i = threadIdx.x; i < (int)(kRawMaskBytes / 4); i += blockDim.x)
      reinterpret_cast<uint32_t *>(smem + kOffRaw)[i] = 0u;
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
  using LY = GemmLayout<MODE, FORM, NB>;

  auto fail = [&]() { *abort_flag = 1; };

  // Every warp of a warpgroup executes the same setmaxnreg, and each role's
  // code follows its own warpgroup's setmaxnreg.
  if (warp >= kGemmWarpEpi0) {
    if constexpr (LY::regs_epi > 0)
      asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(LY::regs_epi));
    if (MODE == MODE_GRADX) {
      gradx_epilogue<NB, FORM>(g, smem, ring, accf, acce, pfull, pempty, tmem, &tmOut,
                               abort_flag, warp, lane);
      if constexpr (NB != 0) {
        // every epilogue warp arrives here once; then the tiles left raw
        // (their products stored by this CTA: fp32 values in FORM 2, int32
        // bit patterns otherwise) are finished
        asm volatile("bar.sync 1, %0;" ::"r"(32 * 4 * LY::sets) : "memory");
        if (!*abort_flag)
          gradx_raw_fix<NB>(g, reinterpret_cast<const uint32_t *>(smem + kOffRaw),
                            warp - kGemmWarpEpi0, 4 * LY::sets, lane, FORM != 2);
      }
    }
    else if (warp < kGemmWarpEpi0 + kPartialEpiWarps)
      partial_epilogue(g, ring, accf, acce, tmem, &tmOut, abort_flag, warp, lane);
    else if (u8ops)  // the four warps after the partial epilogue
      partial_convert(g, ops, uops, full, empty, cvt, fempty, abort_flag,
                      2 + warp - (kGemmWarpEpi0 + kPartialEpiWarps), lane);
  } else {
  if constexpr (LY::regs_ctl > 0)
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(LY::regs_ctl));
  if (warp == kWarpTma) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      if (pairs) {
        bool ok = true;
        for (int64_t it = blockIdx.x; ok && it < g.n_items && !*abort_flag; it += gstep) {
          Item tt[2];
          const int nu = group_items(g, it, pairs, tt);
          const int64_t nch = (tt[0].kb1 - tt[0].kb0 + g.kc_blocks - 1) / g.kc_blocks;
          for (int64_t c = 0; ok && c < nch; ++c) {
            for (int u = 0; ok && u < nu; ++u) {
              const Item &t = tt[u];
              const int64_t c0 = t.kb0 + c * g.kc_blocks, c1 = min(t.kb1, c0 + g.kc_blocks);
              for (int64_t kb = c0; kb < c1; ++kb) {
                if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) { fail(); ok = false; break; }
                mbar_expect_tx(&full[s], (uint32_t)(2 * kTileBytes));
                uint8_t *sa = ops + (size_t)(2 * s) * kTileBytes;
                uint8_t *sb = sa + kTileBytes;
                const int32_t kc = (int32_t)(kb * BK);
                // K-major: one 64 x 128 box; MN-major: two 64 (MN) x 64 (K) boxes
                if (g.a_kmajor) {
                  tma_load_2d(sa, &tmA, kc, (int32_t)t.m0, &full[s]);
                } else {
                  tma_load_2d(sa, &tmA, (int32_t)t.m0, kc, &full[s]);
                  tma_load_2d(sa + kTileBytes / 2, &tmA, (int32_t)t.m0 + 64, kc, &full[s]);
                }
                if (g.b_kmajor) {
                  tma_load_2d(sb, &tmB, kc, (int32_t)t.n0, &full[s]);
                } else {
                  tma_load_2d(sb, &tmB, (int32_t)t.n0, kc, &full[s]);
                  tma_load_2d(sb + kTileBytes / 2, &tmB, (int32_t)t.n0 + 64, kc, &full[s]);
                }
                if (++s == nstages) { s = 0; ph ^= 1u; }
              }
            }
          }
        }
      } else {
        for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
          const Item t = decode_item(g, it);
          // implicit im2col: the item's two (tap, channel group) columns of
          // X~ and its first block's (image, row group), then advanced per
          // K block without divisions
          int cimg = 0, cyb = 0, ccg[2] = {0, 0}, ckx[2] = {0, 0}, cky[2] = {0, 0};
          bool cval[2] = {false, false};
          if (MODE == MODE_PARTIAL && g.conv) {
            cimg = (int)(t.kb0 / g.cybi);
            cyb = (int)(t.kb0 - (int64_t)cimg * g.cybi);
            for (int h = 0; h < 2; ++h) {
              const int d = (int)t.n0 + 64 * h;
              const int tap = d / g.cin;
              ccg[h] = d - tap * g.cin;
              cky[h] = tap / g.ckw;
              ckx[h] = tap - cky[h] * g.ckw;
              cval[h] = d < g.N;
            }
          }
          for (int64_t kb = t.kb0; kb < t.kb1; ++kb) {
            if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) { fail(); break; }
            const int32_t kc = (int32_t)(kb * BK);
            if (u8ops) {
              // byte operands (MN-major), into the byte ring: one 128 (MN) x
              // 64 (K) byte box each
              uint8_t *ua = uops + (size_t)s * kTileBytes;
              mbar_expect_tx(&full[s], (uint32_t)kTileBytes);
              tma_load_2d(ua, &tmA, (int32_t)t.m0, kc, &full[s]);
              tma_load_2d(ua + kTileBytes / 2, &tmB, (int32_t)t.n0, kc, &full[s]);
              if (++s == ustages) { s = 0; ph ^= 1u; }
              continue;
            }
            uint8_t *sa = ops + (size_t)(2 * s) * kTileBytes;
            uint8_t *sb = sa + kTileBytes;
            mbar_expect_tx(&full[s], (uint32_t)(2 * kTileBytes));
            if (MODE == MODE_PARTIAL && g.conv) {
              // implicit im2col: K block kb = output rows rpb yb .. of image
              // img, slots 0 .. pw - 1 of each; Q_b1 rows at those pixels,
              // X~ columns n0 .. n0 + 127 = (tap, 64 channels) pairs read at
              // the tap's offset (outside the input: zeros, the padding)
              const int oy0 = cyb * g.crpb;
              tma_load_4d(sa, &tmA, (int32_t)t.m0, 0, oy0, cimg, &full[s]);
              tma_load_4d(sa + kTileBytes / 2, &tmA, (int32_t)t.m0 + 64, 0, oy0, cimg, &full[s]);
              for (int h = 0; h < 2; ++h) {
                if (cval[h])
                  tma_load_4d(sb + h * (kTileBytes / 2), &tmB, ccg[h], ckx[h] - g.cpad,
                              oy0 + cky[h] - g.cpad, cimg, &full[s]);
                else  // past the last tap: a box outside the tensor (zeros)
                  tma_load_4d(sb + h * (kTileBytes / 2), &tmB, 0, 0, g.cih + g.coh + 8, cimg,
                              &full[s]);
              }
              if (++cyb == g.cybi) { cyb = 0; ++cimg; }
              if (++s == nstages) { s = 0; ph ^= 1u; }
              continue;
            }
            // K-major: one 64 x 128 box; MN-major: two 64 (MN) x 64 (K) boxes
            if (g.a_kmajor) {
              tma_load_2d(sa, &tmA, kc, (int32_t)t.m0, &full[s]);
            } else {
              tma_load_2d(sa, &tmA, (int32_t)t.m0, kc, &full[s]);
              tma_load_2d(sa + kTileBytes / 2, &tmA, (int32_t)t.m0 + 64, kc, &full[s]);
            }
            if (g.b_kmajor) {
              tma_load_2d(sb, &tmB, kc, (int32_t)t.n0, &full[s]);
            } else {
              tma_load_2d(sb, &tmB, (int32_t)t.n0, kc, &full[s]);
              tma_load_2d(sb + kTileBytes / 2, &tmB, (int32_t)t.n0 + 64, kc, &full[s]);
            }
            if (++s == nstages) { s = 0; ph ^= 1u; }
          }
        }
      }
      // every issued load lands before the CTA exits: in normal operation
      // the MMAs have consumed them all; after an abort, give in-flight
      // copies time to complete
      if (*abort_flag) {
        sleep_ns(200000);
      } else {
        const int pstages = u8ops ? ustages : nstages;
        for (int i = 0; i < pstages; ++i) {
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) break;
          if (++s == pstages) { s = 0; ph ^= 1u; }
        }
      }
    }
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      int buf = 0;
      uint32_t aph = 0u;  // bit b: phase parity of accumulator b
      const uint32_t idesc = make_idesc(!g.a_kmajor, !g.b_kmajor);
      // start-address step of one K = 16 slice: 32 bytes inside a K-major
      // swizzle row, two 8-row K atoms (2048 bytes) for MN-major
      const uint64_t a_step = g.a_kmajor ? 2u : (2048u >> 4);
      const uint64_t b_step = g.b_kmajor ? 2u : (2048u >> 4);
      if (pairs) {
        int64_t local = 0;
        bool ok = true;
        for (int64_t it = blockIdx.x; ok && it < g.n_items && !*abort_flag; it += gstep) {
          Item tt[2];
          const int nu = group_items(g, it, pairs, tt);
          const int64_t nch = (tt[0].kb1 - tt[0].kb0 + g.kc_blocks - 1) / g.kc_blocks;
          for (int64_t c = 0; ok && c < nch && !*abort_flag; ++c) {
            for (int u = 0; ok && u < nu; ++u) {
              const Item &t = tt[u];
              if (kPerItem) buf = (int)((local + u) & (g.nacc - 1));
              const int64_t c0 = t.kb0 + c * g.kc_blocks, c1 = min(t.kb1, c0 + g.kc_blocks);
              if (!mbar_wait(&acce[buf], ((aph >> buf) & 1u) ^ 1u, g.status)) {
                fail();
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t dt = tmem + (uint32_t)(buf * BN);
              for (int64_t kb = c0; kb < c1; ++kb) {
                if (!mbar_wait(&full[s], ph, g.status)) { fail(); ok = false; break; }
                tc_fence_after();
                const uint32_t a_addr = smem_u32(ops + (size_t)(2 * s) * kTileBytes);
                const uint32_t b_addr = a_addr + (uint32_t)kTileBytes;
                const uint64_t da = g.a_kmajor ? sw128_desc(a_addr)
                                               : sw128_desc_mn(a_addr, g.mn_lbo, g.mn_sbo);
                const uint64_t db = g.b_kmajor ? sw128_desc(b_addr)
                                               : sw128_desc_mn(b_addr, g.mn_lbo, g.mn_sbo);
  #pragma unroll
                for (int k = 0; k < BK / 16; ++k)
                  umma_f16(dt, da + a_step * k, db + b_step * k, idesc,
                           (kb > c0 || k > 0) ? 1u : 0u);
                umma_commit(&empty[s]);
                if (++s == nstages) { s = 0; ph ^= 1u; }
              }
              umma_commit(&accf[buf]);
              aph ^= 1u << buf;
              if (!kPerItem) buf ^= 1;
            }
          }
          local += nu;
        }
      } else {
        int64_t local = 0;
        for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x, ++local) {
          const Item t = decode_item(g, it);
          if (kPerItem) buf = (int)(local & (g.nacc - 1));
          for (int64_t c0 = t.kb0; c0 < t.kb1 && !*abort_flag; c0 += g.kc_blocks) {
            const int64_t c1 = min(t.kb1, c0 + g.kc_blocks);
            if (!mbar_wait(&acce[buf], ((aph >> buf) & 1u) ^ 1u, g.status)) { fail(); break; }
            tc_fence_after();
            const uint32_t dt = tmem + (uint32_t)(buf * BN);
            for (int64_t kb = c0; kb < c1; ++kb) {
              // byte operands: the carrier stage once the converter warps
              // widened it
              if (!mbar_wait(u8ops ? &cvt[s] : &full[s], ph, g.status)) { fail(); break; }
              tc_fence_after();
              const uint32_t a_addr = smem_u32(ops + (size_t)(2 * s) * kTileBytes);
              const uint32_t b_addr = a_addr + (uint32_t)kTileBytes;
              const uint64_t da = g.a_kmajor ? sw128_desc(a_addr)
                                             : sw128_desc_mn(a_addr, g.mn_lbo, g.mn_sbo);
              const uint64_t db = g.b_kmajor ? sw128_desc(b_addr)
                                             : sw128_desc_mn(b_addr, g.mn_lbo, g.mn_sbo);
  #pragma unroll
              for (int k = 0; k < BK / 16; ++k)
                umma_f16(dt, da + a_step * k, db + b_step * k, idesc,
                         (kb > c0 || k > 0) ? 1u : 0u);
              umma_commit(u8ops ? &fempty[s] : &empty[s]);
              if (++s == nstages) { s = 0; ph ^= 1u; }
            }
            umma_commit(&accf[buf]);
            aph ^= 1u << buf;
            if (!kPerItem) buf ^= 1;
          }
        }
      }
      // every MMA this thread issued has completed before TMEM is released
      // (after an abort the epilogue may have stopped waiting for them)
      umma_commit(drain);
      mbar_wait(drain, 0, g.status);
    }
  } else if (warp == kGemmWarpPar) {
    if (MODE == MODE_GRADX) gradx_params<NB, FORM>(g, smem, pfull, pempty, abort_flag, lane);
    else if (u8ops) partial_convert(g, ops, uops, full, empty, cvt, fempty, abort_flag, 0, lane);
  } else if (MODE == MODE_PARTIAL && u8ops && warp == kGemmWarpPar + 1) {
    partial_convert(g, ops, uops, full, empty, cvt, fempty, abort_flag, 1, lane);
  }
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
  // an implicit im2col X~: its padding entered the product as code 2^(bx-1);
  // P += (code(0) - ob) pad_a[c][tap(d)], pad_a = the A carriers summed over
  // the rows whose tap reads padding (C x taps), tap(d) = d / cin
  const int32_t *pad_a, *code_zero;
  int taps, cin;
  const int32_t *cs_a, *cs_b;  // column sums of Q_b1 codes (M) and X~ codes (N)
  const float *inv_a, *zero_a, *inv_b, *zero_b;
  int vec;  // four outputs per thread (N % 4 == 0, 16-byte aligned buffers)
};

// A thread sums four consecutive outputs of one row over all splits (one
// 16-byte load per split, coalesced across the warp, two splits in flight)
// and dequantizes them (r.vec; else one output per thread).
constexpr int kRedThreads = 256;

__global__ void __launch_bounds__(kRedThreads) k_reduce(const ReduceArgs r) {
  const int64_t total = r.M * r.N;
  const bool vec = r.vec != 0;
  const int W = vec ? 4 : 1;
  const int64_t units = vec ? total >> 2 : total;
  // per-tensor terms: z = -m + d with m an integer
  const bool deq = r.out_i64 == nullptr;
  const float za = deq ? *r.zero_a : 0.0f, zb = deq ? *r.zero_b : 0.0f;
  const float sab = deq ? (*r.inv_a) * (*r.inv_b) : 0.0f;
  const int64_t ma = __float2int_rn(-za), mb = __float2int_rn(-zb);
  const float da = za + (float)ma, db = zb + (float)mb;
  const int64_t ob = r.ob;
  const int64_t code_pad = r.pad_a ? (int64_t)*r.code_zero - ob : 0;
  const float kdd = ll_to_float(r.Kn) * da * db;
  // I = sum (a - ma)(b - mb) = P + ka cb + kb ca + k0, exact, from the
  // centred product P (ca, cb the code column sums)
  const int64_t ka = r.oa - ma, kb = ob - mb;
  const int64_t k0 = r.Kn * ka * kb - ka * r.Kn * ob - kb * r.Kn * r.oa;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < units;
       u += (int64_t)gridDim.x * blockDim.x) {
    const int64_t idx = u * W;
    long long P[4] = {0, 0, 0, 0};
    if (vec) {
      const int4 *src = reinterpret_cast<const int4 *>(r.part + idx);
      const int64_t step = total >> 2;
      int sp = 0;
      for (; sp + 1 < r.splits; sp += 2) {
        const int4 x = __ldcs(src + (int64_t)sp * step), y = __ldcs(src + (int64_t)(sp + 1) * step);
        P[0] += (long long)x.x + y.x;
        P[1] += (long long)x.y + y.y;
        P[2] += (long long)x.z + y.z;
        P[3] += (long long)x.w + y.w;
      }
      if (sp < r.splits) {
        const int4 x = __ldcs(src + (int64_t)sp * step);
        P[0] += x.x;
        P[1] += x.y;
        P[2] += x.z;
        P[3] += x.w;
      }
    } else {
      for (int sp = 0; sp < r.splits; ++sp) P[0] += __ldcs(r.part + (int64_t)sp * total + idx);
    }
    if (!deq) {
      for (int i = 0; i < W; ++i) r.out_i64[idx + i] = P[i];
      continue;
    }
    const int64_t c = idx / r.N, d0 = idx - c * r.N;
    const int64_t ca = r.cs_a[c];
    // row term db (ca - Kn ma) of this thread's row
    const float rt = db * ll_to_float(ca - r.Kn * ma);
    const int64_t Ia = kb * ca + k0;
    float o[4];
    for (int i = 0; i < W; ++i) {
      const int64_t d = d0 + i;
      const int64_t cb = r.cs_b[d];
      long long Pi = P[i];
      if (r.pad_a) Pi += code_pad * r.pad_a[c * r.taps + d / r.cin];
      const int64_t I = Pi + ka * cb + Ia;
      o[i] = sab * (ll_to_float(I) + rt + da * ll_to_float(cb - r.Kn * mb) + kdd);
    }
    if (vec)
      *reinterpret_cast<float4 *>(r.out_f32 + idx) = make_float4(o[0], o[1], o[2], o[3]);
    else
      r.out_f32[idx] = o[0];
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

// Tensor map of an fp16 carrier matrix stored row-major as outer x inner,
// box of box_inner x box_outer elements, 128-byte swizzle (the UMMA layout).
static bool make_map_f16(CUtensorMap *m, const void *base, uint64_t inner,
                         uint64_t outer, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(base), dims,
            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D map of NHWC-ordered fp16 carriers (c, w, h, n) with boxes of 64
// channels x bw pixels x bh rows x 1 image, 128-byte swizzle: the image of a
// (bw bh) x 64 MN-major operand tile (one 128-byte row per pixel).
static bool make_map_f16_box4(CUtensorMap *m, const void *base, uint64_t n, uint64_t h,
                              uint64_t w, uint64_t c, uint32_t bw, uint32_t bh) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {c, w, h, n};
  cuuint64_t strides[3] = {c * 2, w * c * 2, h * w * c * 2};
  cuuint32_t box[4] = {64, bw, bh, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(base), dims, strides,
            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of MN-major byte codes stored as outer (K) rows of inner (MN)
// bytes: 128 x 64 boxes (one 128-byte row per K row), 128-byte swizzle.
static bool make_map_u8(CUtensorMap *m, const void *base, uint64_t inner, uint64_t outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner};
  cuuint32_t box[2] = {128, BK};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output tensor map: fp32 M x N (grad_X) or int32 splits x M x N
// (partials), 32 x 32 boxes with 128-byte swizzle.
static bool make_map_out(CUtensorMap *m, void *base, bool is_int, uint64_t cols,
                         uint64_t rows, uint64_t depth) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {cols, rows, depth};
  cuuint64_t strides[2] = {cols * 4, cols * rows * 4};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, is_int ? CU_TENSOR_MAP_DATA_TYPE_INT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
            is_int ? 3 : 2, base, dims, strides, box, es,
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
    // as many splits as keep every (tile, split) item in one wave of CTAs
    const int64_t tiles = (int64_t)p.m_tiles * p.n_tiles;
    splits = (int)(num_sms / tiles);
    if (splits < 1) splits = 1;
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

// The k_gradw plan for grad_W of C x D over K rows, or splits = 0 when the
// shape does not fit it.
struct WPlan {
  int mt, ncb, Cn, stages, splits;
  int64_t ks_blocks, kb_total;
  size_t smem;
};

static WPlan gradw_plan(int64_t K, int64_t C, int64_t D, int b1, int bx, int num_sms);

// An implicit im2col grad_W takes k_gradw (one exact chunk per K range)
// unless its plan would need more than two ranges per SM (wide operands,
// e.g. the shift quantizer's 12-bit shifted codes); plain operands take the
// split-K tile kernel, whose ranges fold several exact chunks.
static bool use_gradw(const WPlan &w, int num_sms) {
  return w.splits > 0 && w.splits <= 2 * num_sms;
}

size_t gemm_workspace_bytes(int64_t N, int64_t C, int64_t D) {
  // grad_W: M = C, N = D, K = N, by either kernel; the operand bits run from
  // 2 (Q_b1) to 12 (shifted 8-bit codes of the shift quantizer)
  const int nsm = device_sm_count();
  int64_t splits = 0;
  for (int b = 2; b <= 12; ++b) {
    const WPlan w = gradw_plan(N, C, D, b, 8, nsm);
    int64_t sp = use_gradw(w, nsm) ? w.splits : plan_splits(C, D, N, b, 8, nsm, true).splits;
    // an implicit im2col operand pads each image's output rows to blocks of
    // 64 slots: at most 2.4 N slots (ow = 9 in blocks of 4 rows of 16)
    const int64_t sc = plan_splits(C, D, (N * 5 + 1) / 2, b, 8, nsm, true).splits;
    if (sc > sp) sp = sc;
    if (sp > splits) splits = sp;
  }
  // + the padding table of an implicit im2col X~ (C x taps, taps <= D)
  const size_t bytes = (size_t)splits * (size_t)C * (size_t)D * 4 + (size_t)C * D * 4;
  return (bytes + 255) & ~(size_t)255;
}

typedef void (*GemmKernel)(CUtensorMap, CUtensorMap, CUtensorMap, GemmArgs);

// The kernel instance of a mode, BHQ block size (1 = no reflection) and
// product representation (fp32-exact or int32).
// The epilogue form (see GemmLayout) of a contraction whose fp32 form holds
// rows with |m| <= mmax, for codes of b bits.  A row whose values straddle 0
// has z' in [-(2^b - 1), 0], so |m| <= 2^(b-1): with mmax at least that, only
// rows of one sign far from 0 leave the form, and form 2 finishes them in a
// final pass; otherwise many tiles can, and form 1 keeps both paths.
// The largest row offset |m| of the int32 form for a reduction over C with
// codes of bw (W~) and b bits and blocks of nb rows: every |I| (2 + sqrt(nb))
// below 2^31 with |I| <= C 2^(bw-1) (2^(b-1) + |m|); -1 when none.
static float int32_form_mmax(int64_t C, int bw, int b, int nb) {
  const double lim = nb <= 1 ? 2147483647.0 : 2147483647.0 / (2.0 + sqrt((double)nb));
  const double m = floor(lim / ((double)C * (double)(1 << (bw - 1)))) - (double)(1 << (b - 1)) - 1.0;
  return m >= 0.0 ? (float)m : -1.0f;
}

static int epilogue_form(bool flt, double mmax, int b) {
  if (!flt) return 0;
  return mmax >= (double)(1 << (b - 1)) ? 2 : 1;
}

static GemmKernel gemm_kernel(int mode, int nb, int form) {
  if (mode == MODE_PARTIAL) return k_gemm<MODE_PARTIAL, 1, 0>;
#define FQT_GX(NBV)                                                          \
  case NBV:                                                                  \
    return form == 2   ? k_gemm<MODE_GRADX, NBV, 2>                           \
           : form == 1 ? k_gemm<MODE_GRADX, NBV, 1>                           \
                       : k_gemm<MODE_GRADX, NBV, 0>;
  switch (nb) {
    case 0:  // adaptive BHQ groups: fp32 form only (raw rows go to the group pass)
      return form == 2 ? k_gemm<MODE_GRADX, 0, 2> : nullptr;
    FQT_GX(1)
    FQT_GX(2)
    FQT_GX(4)
    FQT_GX(8)
    FQT_GX(16)
    FQT_GX(32)
    FQT_GX(64)
    FQT_GX(128)
  }
#undef FQT_GX
  return nullptr;
}

// Launches the contraction of fp16 carrier operands: A is M x K (stored
// M x K if a_kmajor, else K x M), B is the K x N operand (stored N x K if
// b_kmajor, else K x N).  Partials: out is splits x M x N int32.  grad_X:
// out is the N x M fp32 transpose (rows of dH x columns of W~).
static fqt_status run_gemm(const void *A, int a_kmajor, int a_bits, const void *Bm,
                           int b_kmajor, int b_bits, int64_t M, int64_t N, int64_t K,
                           const SplitPlan &p, GemmArgs &g, void *out, int mode, int nb,
                           int form, cudaStream_t st) {
  const bool partial = mode == MODE_PARTIAL;
  // byte operands (g.u8): split-K partials of MN-major operands only
  if (g.u8 && (!partial || a_kmajor || b_kmajor)) return FQT_EUNSUPPORTED;
  CUtensorMap ta, tb;
  bool ok;
  if (g.u8) {
    ok = make_map_u8(&ta, A, (uint64_t)M, (uint64_t)K) &&
         make_map_u8(&tb, Bm, (uint64_t)N, (uint64_t)K);
  } else if (g.conv) {
    // implicit im2col (split-K partials, both MN-major): Q_b1 as (C, ow, oh,
    // n), the NHWC codes as (cin, iw, ih, n)
    if (!partial || a_kmajor || b_kmajor) return FQT_EUNSUPPORTED;
    ok = make_map_f16_box4(&ta, A, (uint64_t)g.cnimg, (uint64_t)g.coh, (uint64_t)g.cow,
                           (uint64_t)M, (uint32_t)g.cpw, (uint32_t)g.crpb) &&
         make_map_f16_box4(&tb, Bm, (uint64_t)g.cnimg, (uint64_t)g.cih, (uint64_t)g.ciw,
                           (uint64_t)g.cin, (uint32_t)g.cpw, (uint32_t)g.crpb);
  } else {
    ok = a_kmajor ? make_map_f16(&ta, A, (uint64_t)K, (uint64_t)M, BK, BM)
                  : make_map_f16(&ta, A, (uint64_t)M, (uint64_t)K, 64, BK);
    ok = ok && (b_kmajor ? make_map_f16(&tb, Bm, (uint64_t)K, (uint64_t)N, BK, BN)
                         : make_map_f16(&tb, Bm, (uint64_t)N, (uint64_t)K, 64, BK));
  }
  CUtensorMap to;
  ok = ok && (partial ? make_map_out(&to, out, true, (uint64_t)N, (uint64_t)M,
                                     (uint64_t)p.splits)
                      : make_map_out(&to, out, false, (uint64_t)M, (uint64_t)N, 1));
  if (!ok) return cuda_fail(cudaErrorInvalidValue, "tensor map encode");
  GemmKernel kern = gemm_kernel(mode, nb, form);
  if (!kern) return FQT_EUNSUPPORTED;
  const bool four = !partial && form == 2;  // GemmLayout: four epilogue sets
  const int threads = four ? GemmLayout<0, 2>::threads : GemmLayout<0, 0>::threads;
  if (four) {
    // the register split needs the launch's registers per thread: with fewer,
    // setmaxnreg.inc would wait for registers that do not exist
    using L16 = GemmLayout<0, 2, 16>;
    using L32 = GemmLayout<0, 2, 32>;
    const int64_t need = nb <= 16 ? 128 * L16::regs_ctl + 32 * 4 * L16::sets * L16::regs_epi
                                  : 128 * L32::regs_ctl + 32 * 4 * L32::sets * L32::regs_epi;
    cudaFuncAttributes fa;
    const cudaError_t e = cudaFuncGetAttributes(&fa, kern);
    if (e != cudaSuccess) return cuda_fail(e, "gemm attributes");
    if ((int64_t)fa.numRegs * L16::threads < need) return FQT_EUNSUPPORTED;
  }
  // the fp32 form: four epilogue sets for tiles bound by their output, three
  // for long reductions; the code bits for the final pass over raw tiles
  g.sets = (four && (K + BK - 1) / BK <= 2) ? 4 : 3;
  g.bw = a_bits;
  g.b2 = b_bits;
  g.small_p = (K << (a_bits + b_bits - 2)) < ((int64_t)1 << 22);
  // HBM-bound output tiles (grad_X): deep store ring; long reductions
  // (split-K partials): deep operand ring
  // byte operands: two carrier stages fed by a ring of six byte stages
  g.stages = partial ? (g.u8 ? 2 : 5) : 2;
  g.ustages = g.u8 ? 6 : 0;
  g.ring = partial ? 1 : 0;  // grad_X stores straight from registers
  // grad_X tiles with a long reduction (K of many blocks: a contraction that
  // is tensor-bound rather than bound by its output) keep more operand
  // stages in flight
  if (!partial && (K + BK - 1) / BK > 2) {
    while (g.stages < kMaxStages && gemm_smem_bytes(g.stages + 1, g.ring) <= 227 * 1024)
      ++g.stages;
  }
  if (!partial) g.out = static_cast<float *>(out);
  // grad_X with one exact chunk per tile: four accumulators in rotation, so
  // the next tile of each epilogue set is ready when it finishes the last;
  // otherwise two, and the other half of tensor memory holds running sums
  g.nacc = (!partial && exact_chunk_blocks(a_bits, b_bits) >= (K + BK - 1) / BK) ? 4 : 2;
  // Several exact chunks per tile (two accumulators): one epilogue set per
  // accumulator, so that each accumulator's chunks are drained by one set in
  // order.  An mbarrier parity wait cannot tell a phase from the one two
  // phases later; with three sets, the set of tile L + 2 could start waiting
  // on accumulator L mod 2 while tile L's chunks still pass through it (the
  // parameter ring holds that set back only until tile L - 4 is done).  With
  // one chunk per tile, tile L's parameters wait for tile L - 4 (the same
  // accumulator of four) to be drained, which is enough.
  if (!partial && g.nacc == 2) g.sets = 2;
  g.m_fast = partial ? 0 : 1;
  g.M = M;
  g.N = N;
  g.K = K;
  g.a_kmajor = a_kmajor;
  g.b_kmajor = b_kmajor;
  g.mn_lbo = (uint32_t)(kTileBytes / 2);  // second 64-wide MN atom column
  g.mn_sbo = 1024;                        // next 8-row K atom
  g.kc_blocks = exact_chunk_blocks(a_bits, b_bits);
  g.m_tiles = p.m_tiles;
  g.n_tiles = p.n_tiles;
  g.splits = p.splits;
  g.ks_blocks = p.ks_blocks;
  g.kb_total = p.kb_total;
  g.n_items = (int64_t)p.m_tiles * p.n_tiles * p.splits;
  const size_t smem = gemm_smem_bytes(g.stages, g.ring, g.ustages);
  const cudaError_t ea =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (ea != cudaSuccess) return cuda_fail(ea, "gemm shared-memory attribute");
  const int nsm = device_sm_count();
  int64_t grid = g.n_items < nsm ? g.n_items : nsm;
  if (grid < 1) grid = 1;
  // the raw-tile bits of a CTA cover kMaxLocalTiles of its tiles
  if (!partial && nb != 0 && (g.n_items + grid - 1) / grid > kMaxLocalTiles)
    return FQT_EUNSUPPORTED;
  kern<<<(int)grid, threads, smem, st>>>(ta, tb, to, g);
  return cuda_fail(cudaGetLastError(), "gemm launch");
}

// u8 codes -> fp16 carriers code - off (debug path only)
__global__ void k_u8_to_f16(const uint8_t *__restrict__ src, uint16_t *dst,
                            int64_t n, int off) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const __half h = __int2half_rn((int)src[i] - off);
    dst[i] = *reinterpret_cast<const uint16_t *>(&h);
  }
}

static void launch_reduce(ReduceArgs r, cudaStream_t st) {
  const int64_t total = r.M * r.N;
  auto a16 = [](const void *q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
  r.vec = (r.N & 3) == 0 && a16(r.part) && (r.out_i64 || a16(r.out_f32));
  const int64_t units = r.vec ? total >> 2 : total;
  int64_t grid = (units + kRedThreads - 1) / kRedThreads;
  const int64_t cap = (int64_t)device_sm_count() * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  k_reduce<<<(int)grid, kRedThreads, 0, st>>>(r);
}

static bool aligned16(const void *p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

static size_t round256(size_t v) { return (v + 255) & ~(size_t)255; }

size_t debug_workspace_bytes(int64_t M, int64_t N, int64_t K) {
  const SplitPlan p = plan_splits(M, N, K, 8, 8, device_sm_count(), true);
  return kGemmOffset + round256((size_t)p.splits * (size_t)M * (size_t)N * 4) +
         round256((size_t)M * (size_t)K * 2) + round256((size_t)N * (size_t)K * 2);
}

fqt_status debug_int_gemm(const uint8_t *A, int a_kmajor, int a_bits,
                          const uint8_t *Bm, int b_kmajor, int b_bits, int64_t M,
                          int64_t N, int64_t K, int64_t *out, void *ws,
                          size_t ws_bytes, cudaStream_t st) {
  if (!A || !Bm || !out || M <= 0 || N <= 0 || K <= 0) return FQT_EINVAL;
  if (a_bits < 2 || a_bits > 8 || b_bits < 2 || b_bits > 8) return FQT_EINVAL;
  // TMA: the row pitch of each stored operand must be a multiple of 16 bytes
  if ((a_kmajor ? K : M) % 8 || (b_kmajor ? K : N) % 8 || N % 4) return FQT_EUNSUPPORTED;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return FQT_EUNSUPPORTED;
  const SplitPlan p = plan_splits(M, N, K, a_bits, b_bits, device_sm_count(), true);
  const size_t part_bytes = round256((size_t)p.splits * (size_t)M * (size_t)N * 4);
  const size_t need = kGemmOffset + part_bytes + round256((size_t)M * K * 2) +
                      round256((size_t)N * K * 2);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < need)
    return FQT_EWORKSPACE;
  char *w = static_cast<char *>(ws);
  int32_t *part = reinterpret_cast<int32_t *>(w + kGemmOffset);
  uint16_t *a16 = reinterpret_cast<uint16_t *>(w + kGemmOffset + part_bytes);
  uint16_t *b16 = reinterpret_cast<uint16_t *>(w + kGemmOffset + part_bytes +
                                               round256((size_t)M * K * 2));
  const int nsm = device_sm_count();
  k_u8_to_f16<<<nsm * 4, 256, 0, st>>>(A, a16, M * K, 1 << (a_bits - 1));
  k_u8_to_f16<<<nsm * 4, 256, 0, st>>>(Bm, b16, N * K, 1 << (b_bits - 1));
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.status = reinterpret_cast<int *>(ws);
  fqt_status s = run_gemm(a16, a_kmajor, a_bits, b16, b_kmajor, b_bits, M, N, K, p,
                          g, part, MODE_PARTIAL, 1, false, st);
  if (s != FQT_OK) return s;
  ReduceArgs r;
  memset(&r, 0, sizeof(r));
  r.part = part;
  r.splits = p.splits;
  r.M = M;
  r.N = N;
  r.out_i64 = out;
  launch_reduce(r, st);
  return cuda_fail(cudaGetLastError(), "split-K reduce launch");
}

// The same contraction with both operands MN-major byte codes (A stored
// K x M, B stored K x N) read as bytes and widened on chip: the path grad_W
// takes with byte operands.
fqt_status debug_int_gemm_u8(const uint8_t *A, int a_bits, const uint8_t *Bm, int b_bits,
                             int64_t M, int64_t N, int64_t K, int64_t *out, void *ws,
                             size_t ws_bytes, cudaStream_t st) {
  if (!A || !Bm || !out || M <= 0 || N <= 0 || K <= 0) return FQT_EINVAL;
  if (a_bits < 2 || a_bits > 8 || b_bits < 2 || b_bits > 8) return FQT_EINVAL;
  // TMA: byte rows of a multiple of 16 bytes, 16-byte aligned bases
  if (M % 16 || N % 16) return FQT_EUNSUPPORTED;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return FQT_EUNSUPPORTED;
  if (!aligned16(A) || !aligned16(Bm)) return FQT_EINVAL;
  const SplitPlan p = plan_splits(M, N, K, a_bits, b_bits, device_sm_count(), true);
  const size_t part_bytes = round256((size_t)p.splits * (size_t)M * (size_t)N * 4);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < kGemmOffset + part_bytes)
    return FQT_EWORKSPACE;
  int32_t *part = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kGemmOffset);
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.status = reinterpret_cast<int *>(ws);
  g.u8 = 1;
  fqt_status s = run_gemm(A, 0, a_bits, Bm, 0, b_bits, M, N, K, p, g, part, MODE_PARTIAL, 1,
                          false, st);
  if (s != FQT_OK) return s;
  ReduceArgs r;
  memset(&r, 0, sizeof(r));
  r.part = part;
  r.splits = p.splits;
  r.M = M;
  r.N = N;
  r.out_i64 = out;
  launch_reduce(r, st);
  return cuda_fail(cudaGetLastError(), "split-K reduce launch");
}

// ---------------------------------------------------------------------------
// grad_W with one CTA per range of K rows and all of C x D (when C <= 256
// and ceil(D / 128) C <= 512 TMEM columns): out^T (D x C) = X~^T Q_b1 over
// the range, as ceil(D / 128) tiles of M = 128 (D) by N = C.  Every k-block
// of 64 rows loads X~'s rows (all D columns) and Q_b1's rows once, both
// contiguous in memory, and issues one MMA group per D tile into its own
// TMEM accumulator.  The range is one exact chunk (<= 2^(26 - b1 - bx)
// terms); the epilogue writes int32 partials [split][C][D] that k_reduce
// sums in int64.
// ---------------------------------------------------------------------------
constexpr int kWThreads = 320;  // TMA, MMA, 8 epilogue warps
constexpr int kWBK = 32;           // rows of K per stage (two K = 16 MMA steps)
constexpr size_t kWBox = 64 * kWBK * 2;  // one 64-wide fp16 box of a stage

struct WArgs {
  int64_t K;          // rows of dH / X
  int C, D, Cn;       // Cn: C rounded up to 16 (MMA N)
  int mt, ncb;        // D tiles of 128, 64-wide boxes of Q_b1
  int splits;
  int64_t ks_blocks, kb_total;
  int stages;
  int32_t *part;      // [splits][C][D]
  int *status;
  // implicit im2col operand (stride 1): X~ is read as 4-D boxes of an NHWC
  // tensor at shifted pixel coordinates; padding comes back as zero carriers
  int conv, ih, iw, oh, ow, cin, kh, kw, pad, taps;
};

__host__ __device__ constexpr uint32_t make_idesc_mn_n(int n) {
  // A and B MN-major, D fp32, M = 128, N = n
  return (1u << 4) | (1u << 15) | (1u << 16) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(BM >> 4) << 24);
}

// The int32 value of an fp32 holding an exact integer of magnitude <= 2^24,
// from its bits (no conversion instruction).
__device__ __forceinline__ int exact_f2i(float x) {
  const uint32_t bits = __float_as_uint(x);
  const uint32_t e = (bits >> 23) & 0xFFu;
  const uint32_t sig = (bits & 0x7FFFFFu) | 0x800000u;
  const uint32_t mag = e >= 150u ? sig << (e - 150u) : __funnelshift_rc(sig, 0u, 150u - e);
  return (bits >> 31) ? -(int)mag : (int)mag;
}

__global__ void __launch_bounds__(kWThreads, 1)
    k_gradw(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmQ,
            const WArgs w) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem);
  uint64_t *full = bars, *empty = bars + kMaxStages, *accf = empty + kMaxStages,
           *acce = accf + 1, *drain = acce + 1;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  uint8_t *ops = smem + 1024;
  const size_t xbytes = (size_t)w.mt * 2 * kWBox;  // per D tile: two 64-wide boxes
  const size_t stage_bytes = xbytes + (size_t)w.ncb * kWBox;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < w.stages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(accf, 1);
    mbar_init(acce, kPartialEpiWarps);
    mbar_init(drain, 1);
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
  const int64_t n_items = w.splits;

  if (warp == kWarpTma) {
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      // implicit im2col: the pixel position advances per K block; the D
      // boxes walk (channel group, tap) without divisions
      for (int64_t it = blockIdx.x; it < n_items && !*abort_flag; it += gridDim.x) {
        const int64_t kb0 = it * w.ks_blocks, kb1 = min(w.kb_total, kb0 + w.ks_blocks);
        int ox0 = 0, oy = 0, nimg = 0;
        if (w.conv) {
          const int64_t p0 = kb0 * kWBK, t = p0 / w.ow;
          ox0 = (int)(p0 - t * w.ow);
          oy = (int)(t % w.oh);
          nimg = (int)(t / w.oh);
        }
        for (int64_t kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[s], ph ^ 1u, w.status)) { *abort_flag = 1; break; }
          mbar_expect_tx(&full[s], (uint32_t)stage_bytes);
          uint8_t *sx = ops + (size_t)s * stage_bytes;
          uint8_t *sq = sx + xbytes;
          const int32_t kc = (int32_t)(kb * kWBK);
          if (w.conv) {
            // 32 output pixels of one output row (ow % 32 == 0); box (64 channels
            // of one tap) x 32 pixels read at the tap's offset
            int cg = 0, kx = 0, ky = 0;
            for (int m = 0; m < 2 * w.mt; ++m) {
              if (ky < w.kh)
                tma_load_4d(sx + (size_t)m * kWBox, &tmX, cg, ox0 + kx - w.pad,
                            oy + ky - w.pad, nimg, &full[s]);
              else  // past the last tap: a box outside the tensor (zeros)
                tma_load_4d(sx + (size_t)m * kWBox, &tmX, 0, 0, w.ih + w.oh + 8, nimg,
                            &full[s]);
              cg += 64;
              if (cg == w.cin) {
                cg = 0;
                if (++kx == w.kw) {
                  kx = 0;
                  ++ky;
                }
              }
            }
            ox0 += kWBK;
            if (ox0 == w.ow) {
              ox0 = 0;
              if (++oy == w.oh) {
                oy = 0;
                ++nimg;
              }
            }
          } else {
            for (int m = 0; m < w.mt; ++m) {
              tma_load_2d(sx + (size_t)m * 2 * kWBox, &tmX, m * 128, kc, &full[s]);
              tma_load_2d(sx + (size_t)m * 2 * kWBox + kWBox, &tmX, m * 128 + 64, kc, &full[s]);
            }
          }
          for (int cb = 0; cb < w.ncb; ++cb)
            tma_load_2d(sq + (size_t)cb * kWBox, &tmQ, cb * 64, kc, &full[s]);
          if (++s == w.stages) { s = 0; ph ^= 1u; }
        }
      }
      if (*abort_flag) {
        sleep_ns(200000);
      } else {
        for (int i = 0; i < w.stages; ++i) {
          if (!mbar_wait(&empty[s], ph ^ 1u, w.status)) break;
          if (++s == w.stages) { s = 0; ph ^= 1u; }
        }
      }
    }
  } else if (warp == kWarpMma) {
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0, eph = 0;
      const uint32_t idesc = make_idesc_mn_n(w.Cn);
      for (int64_t it = blockIdx.x; it < n_items && !*abort_flag; it += gridDim.x) {
        const int64_t kb0 = it * w.ks_blocks, kb1 = min(w.kb_total, kb0 + w.ks_blocks);
        if (!mbar_wait(acce, eph ^ 1u, w.status)) { *abort_flag = 1; break; }
        eph ^= 1u;
        tc_fence_after();
        for (int64_t kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[s], ph, w.status)) { *abort_flag = 1; break; }
          tc_fence_after();
          const uint32_t x_addr = smem_u32(ops + (size_t)s * stage_bytes);
          const uint32_t q_addr = x_addr + (uint32_t)xbytes;
          const uint64_t dq = sw128_desc_mn(q_addr, (uint32_t)kWBox, 1024);
          for (int m = 0; m < w.mt; ++m) {
            const uint64_t dx =
                sw128_desc_mn(x_addr + (uint32_t)(m * 2 * kWBox), (uint32_t)kWBox, 1024);
#pragma unroll
            for (int k = 0; k < kWBK / 16; ++k)
              umma_f16(tmem + (uint32_t)(m * w.Cn), dx + (2048u >> 4) * k, dq + (2048u >> 4) * k,
                       idesc, (kb > kb0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&empty[s]);
          if (++s == w.stages) { s = 0; ph ^= 1u; }
        }
        umma_commit(accf);
      }
      // every MMA this thread issued has completed before TMEM is released
      umma_commit(drain);
      mbar_wait(drain, 0, w.status);
    }
  } else {
    // epilogue: warp (q, h) takes the D tiles m = h, h + 2, ...; a thread owns
    // output column d = 128 m + 32 q + lane of grad_W^T
    const int q = warp & 3, h = (warp - kWarpEpi0) >> 2;
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    uint32_t aph = 0;
    for (int64_t it = blockIdx.x; it < n_items && !*abort_flag; it += gridDim.x) {
      const bool got = mbar_wait(accf, aph, w.status);
      if (!__all_sync(0xffffffffu, got)) { *abort_flag = 1; break; }
      aph ^= 1u;
      tc_fence_after();
      int32_t *pp = w.part + it * (int64_t)w.C * w.D;
      for (int m = h; m < w.mt; m += 2) {
        const int d = m * 128 + q * 32 + lane;
        for (int c0 = 0; c0 < w.Cn; c0 += 32) {
          uint32_t r[32];
          tmem_ld32_nw(lane_base + (uint32_t)(m * w.Cn + c0), r);
          tmem_wait_ld(r);
          if (d < w.D) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (c0 + i < w.C) pp[(int64_t)(c0 + i) * w.D + d] = exact_f2i(__uint_as_float(r[i]));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce);
    }
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

static WPlan gradw_plan(int64_t K, int64_t C, int64_t D, int b1, int bx, int num_sms) {
  WPlan p;
  memset(&p, 0, sizeof(p));
  if (C <= 0 || C > 256 || C % 16 || D <= 0 || D % 8 || K <= 0) return p;
  p.Cn = (int)C;
  p.mt = (int)((D + 127) / 128);
  if ((int64_t)p.mt * p.Cn > (int64_t)kTmemCols) return p;
  p.ncb = (int)((C + 63) / 64);
  const size_t stage = (size_t)p.mt * 2 * kWBox + (size_t)p.ncb * kWBox;
  p.stages = (int)((220 * 1024 - 1024 - 1024) / stage);
  if (p.stages > kMaxStages) p.stages = kMaxStages;
  if (p.stages < 2) {
    p.splits = 0;
    return p;
  }
  p.smem = 1024 + (size_t)p.stages * stage + 1024;
  p.kb_total = (K + kWBK - 1) / kWBK;
  const int64_t kc = exact_chunk_blocks(b1, bx) * (BK / kWBK);  // k-blocks per exact chunk
  int64_t splits = (p.kb_total + kc - 1) / kc;     // every range one exact chunk
  if (splits < num_sms) splits = num_sms;
  if (splits > p.kb_total) splits = p.kb_total;
  p.ks_blocks = (p.kb_total + splits - 1) / splits;
  p.splits = (int)((p.kb_total + p.ks_blocks - 1) / p.ks_blocks);
  return p;
}

// 4-D map of NHWC fp16 carriers (c, w, h, n), boxes of 64 channels x 32
// pixels of one image row, 128-byte swizzle: the same shared-memory image as
// a 64 x 32 box of the im2col matrix.
static bool make_map_f16_nhwc(CUtensorMap *m, const void *base, uint64_t n, uint64_t h,
                              uint64_t w, uint64_t c) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {c, w, h, n};
  cuuint64_t strides[3] = {c * 2, w * c * 2, h * w * c * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)kWBK, 1, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(base), dims, strides,
            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static fqt_status run_gradw(const uint16_t *X16, const uint16_t *Q16, int64_t K, int C, int D,
                            const WPlan &p, int32_t *part, int *status, cudaStream_t st,
                            const int32_t *conv = nullptr) {
  CUtensorMap tx, tq;
  bool ok = conv ? make_map_f16_nhwc(&tx, X16, (uint64_t)conv[0], (uint64_t)conv[1],
                                     (uint64_t)conv[2], (uint64_t)conv[3])
                 : make_map_f16(&tx, X16, (uint64_t)D, (uint64_t)K, 64, kWBK);
  ok = ok && make_map_f16(&tq, Q16, (uint64_t)C, (uint64_t)K, 64, kWBK);
  if (!ok) return cuda_fail(cudaErrorInvalidValue, "tensor map encode");
  WArgs w;
  memset(&w, 0, sizeof(w));
  w.K = K;
  w.C = C;
  w.D = D;
  w.Cn = p.Cn;
  w.mt = p.mt;
  w.ncb = p.ncb;
  w.splits = p.splits;
  w.ks_blocks = p.ks_blocks;
  w.kb_total = p.kb_total;
  w.stages = p.stages;
  w.part = part;
  w.status = status;
  if (conv) {
    w.conv = 1;
    w.ih = conv[1];
    w.iw = conv[2];
    w.cin = conv[3];
    w.kh = conv[4];
    w.kw = conv[5];
    w.pad = conv[6];
    w.oh = conv[1] + 2 * conv[6] - conv[4] + 1;
    w.ow = conv[2] + 2 * conv[6] - conv[5] + 1;
    w.taps = conv[4] * conv[5];
  }
  const cudaError_t ea =
      cudaFuncSetAttribute(k_gradw, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
  if (ea != cudaSuccess) return cuda_fail(ea, "grad_W shared-memory attribute");
  const int nsm = device_sm_count();
  const int grid = p.splits < nsm ? p.splits : nsm;
  k_gradw<<<grid, kWThreads, p.smem, st>>>(tx, tq, w);
  return cuda_fail(cudaGetLastError(), "grad_W launch");
}

// H = X~ W~^T (Sec. 2.1): the grad_X kernel with the roles renamed -- M = C
// (rows of W~, K-major), N = rows of X~, K = D; the row terms of X~ take the
// place of Q_b2's (PTQ: one scale, one zero, the row sums), W~'s row sums the
// place of the column sums over the contraction.
fqt_status linear_forward(const fqt_qtensor *qx, const fqt_qtensor *qw, float *H, void *ws,
                          size_t ws_bytes, cudaStream_t st) {
  if (!qx || !qw || !H) return FQT_EINVAL;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < kHeaderBytes)
    return FQT_EWORKSPACE;
  if (qx->kind != FQT_PTQ || qw->kind != FQT_PTQ) return FQT_EINVAL;
  const int64_t Nr = qx->rows, D = qx->cols, C = qw->rows;
  if (qw->cols != D || Nr < 0) return FQT_EINVAL;
  if (Nr == 0) return FQT_OK;
  if (!qx->codes_f16 || !qw->codes_f16 || !qx->row_sum || !qw->row_sum || !qx->inv_s ||
      !qx->zero || !qw->inv_s || !qw->zero)
    return FQT_EINVAL;
  if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
  if (D > 8192) return FQT_EUNSUPPORTED;
  if (!aligned16(qx->codes_f16) || !aligned16(qw->codes_f16) || !aligned16(H)) return FQT_EINVAL;
  const int nsm = device_sm_count();
  const SplitPlan p = plan_splits(C, Nr, D, qw->bits, qx->bits, nsm, false);
  // no reflection: with P exact (one chunk) the fp32 form holds for all m
  const int64_t kc_terms = (int64_t)exact_chunk_blocks(qw->bits, qx->bits) * BK;
  const double mmax = 1e30;
  const bool flt = D <= kc_terms;
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.status = reinterpret_cast<int *>(ws);
  g.kind = FQT_PTQ;
  g.og = 1 << (qx->bits - 1);
  g.ow = 1 << (qw->bits - 1);
  g.inv_s = qx->inv_s;
  g.zero = qx->zero;
  g.row_sum = qx->row_sum;
  g.col_sum_w = qw->row_sum;
  g.inv_sw = qw->inv_s;
  g.zero_w = qw->zero;
  g.flt_mmax = flt ? (float)mmax : -1.0f;
  g.i32_mmax = int32_form_mmax(D, qw->bits, qx->bits, 1);
  return run_gemm(qw->codes_f16, 1, qw->bits, qx->codes_f16, 1, qx->bits, C, Nr, D, p, g, H,
                  MODE_GRADX, 1, epilogue_form(flt, mmax, qx->bits), st);
}

// ---------------------------------------------------------------------------
// Implicit im2col X~ (stride 1): per tap (ky, kx), the sum over the output
// pixels whose input pixel (oy + ky - pad, ox + kx - pad) lies in the padding
// of the A operand's carriers (C per row), for the padding correction of
// k_reduce.  Only output pixels in the top / bottom pad rows or the left /
// right pad columns can read padding, and whether they do depends only on
// which of those rows and columns they sit in: (2 pad + 1)^2 classes (the
// inside class never).  A CTA (a run of images, a group of channels) adds
// each border pixel's carriers into its class in shared memory (16-byte
// loads, four in flight per thread), then adds each tap's share, the classes
// whose row or column reads padding, into the sums.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int pad_class(int y, int p, int n) {
  return y < p ? y : (y >= n - p ? 2 * p - (n - 1 - y) : p);
}

// the one output row (column) of border class r, or -1 for the inside class
__device__ __forceinline__ int pad_class_row(int r, int p, int n) {
  return r < p ? r : (r > p ? n - 1 - (2 * p - r) : -1);
}

__global__ void __launch_bounds__(256) k_conv_padsum(const uint16_t *__restrict__ A16, int C,
                                                     int ch_group, int64_t nimg, int imgs_per_cta,
                                                     int h, int w, int kw, int pad, int oh,
                                                     int ow, int taps, int32_t *pad_a) {
  extern __shared__ int cls_s[];  // classes x ch_group
  const int cc = 2 * pad + 1, ncls = cc * cc;
  const int64_t img0 = (int64_t)blockIdx.x * imgs_per_cta;
  const int nim = (int)min((int64_t)imgs_per_cta, nimg - img0);
  const int ch0 = (int)blockIdx.y * ch_group, nch = min(ch_group, C - ch0);
  for (int i = threadIdx.x; i < ncls * ch_group; i += blockDim.x) cls_s[i] = 0;
  __syncthreads();
  const int top = min(pad, oh), nbot = oh - max(top, oh - pad), full_rows = top + nbot;
  const int left = min(pad, ow), nright = ow - max(left, ow - pad), side = left + nright;
  const int full_px = full_rows * ow;
  const int npx = full_px + (oh - full_rows) * side;  // the pixel counts of one image fit int
  const int octs = nch / 8, per_img = npx * octs, items = nim * per_img;
  const uint16_t *base = A16 + (img0 * oh) * (int64_t)ow * C + ch0;
  for (int i0 = threadIdx.x; i0 < items; i0 += 4 * blockDim.x) {
    uint4 v[4];
    int k[4], oc[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int it = i0 + u * (int)blockDim.x;
      k[u] = -1;
      oc[u] = 0;
      v[u] = make_uint4(0u, 0u, 0u, 0u);
      if (it < items) {
        const int im = it / per_img, rem = it - im * per_img, t = rem / octs;
        oc[u] = rem - t * octs;
        int oy, ox;
        if (t < full_px) {
          const int r = t / ow;
          oy = r < top ? r : oh - nbot + (r - top);
          ox = t - r * ow;
        } else {
          const int q = t - full_px, r = q / side, cq = q - r * side;
          oy = top + r;
          ox = cq < left ? cq : ow - nright + (cq - left);
        }
        k[u] = pad_class(oy, pad, oh) * cc + pad_class(ox, pad, ow);
        v[u] = __ldg(reinterpret_cast<const uint4 *>(
            base + (((int64_t)im * oh + oy) * ow + ox) * C + oc[u] * 8));
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (k[u] < 0) continue;
      const uint32_t wds[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&wds[q]));
        int *dst = &cls_s[k[u] * ch_group + oc[u] * 8 + 2 * q];
        if ((int)f.x) atomicAdd(dst, (int)f.x);
        if ((int)f.y) atomicAdd(dst + 1, (int)f.y);
      }
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < nch * taps; i += blockDim.x) {
    const int ch = i / taps, tap = i - ch * taps, ky = tap / kw, kx = tap - ky * kw;
    int v = 0;
    for (int ry = 0; ry < cc; ++ry) {
      const int yr = pad_class_row(ry, pad, oh);
      const bool row_out = yr >= 0 && (yr + ky - pad < 0 || yr + ky - pad >= h);
      for (int rx = 0; rx < cc; ++rx) {
        const int xr = pad_class_row(rx, pad, ow);
        const bool col_out = xr >= 0 && (xr + kx - pad < 0 || xr + kx - pad >= w);
        if (row_out || col_out) v += cls_s[(ry * cc + rx) * ch_group + ch];
      }
    }
    if (v) atomicAdd(&pad_a[(int64_t)(ch0 + ch) * taps + tap], v);
  }
}

// Channels per CTA of k_conv_padsum: a multiple of 8 whose class sums fit
// 40 KB of shared memory (0: the padding is too wide, pad > 17).
static int padsum_group(int C, int pad) {
  const int ncls = (2 * pad + 1) * (2 * pad + 1);
  int grp = (40960 / (ncls * 4)) / 8 * 8;
  if (grp < 8) return 0;
  return grp < C ? grp : C;
}

// ---------------------------------------------------------------------------
// Adaptive BHQ groups (App. D.5).  After the contraction, the grad_X rows of
// every group of two or more rows -- and of single rows whose offset m is
// too large for the fp32 form -- hold the exact integer products P.  This
// pass adds the offsets and applies the group's inverse Householder
// reflection, the second of the two sparse-dense products Sec. 4.3 counts,
// with the arithmetic of the fused epilogue: fp32 where every magnitude is
// exact (block sums off the fp32 bits), int64 / float-float otherwise.
// k_grp_list collects the groups that need it; k_grp_fix gives a warp one
// (group, 128 columns) unit, each lane 4 consecutive columns, and
// k_grp_fix_big a CTA to each group of more than 32 rows.
// ---------------------------------------------------------------------------
struct FixArgs {
  float *out;
  int64_t N, D;
  int C, og, ow, bw, b2;
  const float *inv_s, *zero, *hz, *hr;
  const int32_t *row_sum, *perm, *gstart;
  const float *inv_sw, *zero_w;
  const int32_t *col_sum_w;
  float raw_mmax;
  int small_p;  // every |P| < 2^22: the fp32 block sums apply
  float mmax_nb[33];  // groups of nb <= 32 rows: largest |m| of the fp32 form
  int32_t *list, *list_big;
  int *count, *count_big;
  // fixed blocks (gradx_raw_fix): block size, per-tensor Q_b2 metadata
  // (PTQ) and the lead row of every block
  int nbk, per_tensor;
  const int32_t *lead;
  int p_bits;  // the stored products are int32 bit patterns (else fp32 values)
  int *status;
};

// Per-row terms of the epilogue: scale, the offsets (hd, hR) and m.
struct RowTerms {
  float sc, hd, hR, m;
};

__device__ __forceinline__ float zero_of(const FixArgs &f, int64_t k) {
  return f.zero[f.per_tensor ? 0 : k];
}

__device__ __forceinline__ RowTerms row_terms(const FixArgs &f, int64_t k, float inv_sw,
                                              bool reflected) {
  RowTerms t;
  t.sc = __fmul_rn(inv_sw, f.inv_s[f.per_tensor ? 0 : k]);
  const ff x = two_sum((float)f.og, zero_of(f, k));
  t.m = rintf(x.h);
  // BHQ rows (no row sums here) read their offsets from hz, hr even for a
  // one-row block, where they are the unreflected d and R
  if (reflected || !f.row_sum) {
    t.hd = f.hz[k];
    t.hR = f.hr[k];
  } else {
    t.hd = ff_round(fast_two_sum(__fsub_rn(x.h, t.m), x.l));
    t.hR = __fadd_rn((float)(f.row_sum[k] - f.C * f.og), __fmul_rn((float)f.C, t.m));
  }
  return t;
}

__global__ void __launch_bounds__(256) k_grp_list(const FixArgs f) {
  const int64_t gi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  bool need = false;
  if (gi < f.N) {
    const int64_t k0 = f.gstart[gi];
    if (k0 < f.N) {
      const int64_t k1 = f.gstart[gi + 1];
      if (k1 - k0 > 32) {
        // a CTA of its own (k_grp_fix_big)
        const int slot = atomicAdd(f.count_big, 1);
        f.list_big[slot] = (int32_t)gi;
      } else if (k1 - k0 >= 2) {
        need = true;
      } else if (k1 - k0 == 1) {
        const float m = rintf(two_sum((float)f.og, f.zero[k0]).h);
        need = !(fabsf(m) <= f.raw_mmax);
      }
    }
  }
  const unsigned ball = __ballot_sync(0xffffffffu, need);
  if (!ball) return;
  const int lane = threadIdx.x & 31;
  int base = 0;
  if (lane == 0) base = atomicAdd(f.count, __popc(ball));
  base = __shfl_sync(0xffffffffu, base, 0);
  if (need) f.list[base + __popc(ball & ((1u << lane) - 1u))] = (int32_t)gi;
}

// Any group (or a single row left raw): rows visited one by one; the fp32
// form where it is exact, else int64 integer parts and float-float.  The
// lead row is row `lead` of the group (0 for the stored groups); rows are
// perm[k] of grad_X, or k itself without perm.
__device__ __noinline__ void fix_group_general(const FixArgs &f, int64_t k0, int nb, int64_t j,
                                               bool jv, const float (&cwc)[4],
                                               const int (&cwi)[4], const float (&U)[4],
                                               float inv_sw, const ff &y, int lead) {
  const int lane = threadIdx.x & 31;
  const int Cn = f.C;
  const bool refl = nb >= 2;
  // the fp32 form: |P| < 2^22 and |I| (2 + sqrt(nb)) < 2^24 for every row
  bool fast = refl && f.small_p && !f.p_bits;
  auto pint = [&](float v) -> long long {
    return f.p_bits ? (long long)__float_as_int(v) : (long long)__float2int_rn(v);
  };
  if (fast) {
    const double lim = 16777216.0 / (2.0 + sqrt((double)nb));
    const double mmax = floor(lim / ((double)Cn * (double)(1 << (f.bw - 1)))) -
                        (double)(1 << (f.b2 - 1)) - 1.0;
    for (int r = lane; r < nb; r += 32) {
      const float m = rintf(two_sum((float)f.og, zero_of(f, k0 + r)).h);
      if (!((double)fabsf(m) <= mmax)) fast = false;
    }
    fast = __all_sync(0xffffffffu, fast);
  }
  auto prow = [&](int r) -> float * {
    int64_t pr = f.perm ? (int64_t)f.perm[k0 + r] : k0 + r;
    if (pr < 0 || pr >= f.N) pr = 0;
    return f.out + pr * f.D + j;
  };
  if (fast) {
    const HhConst hc = hh_const(nb);
    uint32_t sb[4] = {0u, 0u, 0u, 0u};
    int msum = 0, Ip[4] = {0, 0, 0, 0};
    for (int r = 0; r < nb; ++r) {
      const float m = rintf(two_sum((float)f.og, zero_of(f, k0 + r)).h);
      msum += (int)m;
      if (!jv) continue;
      const float4 P = *reinterpret_cast<const float4 *>(prow(r));
      const float pv[4] = {P.x, P.y, P.z, P.w};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        sb[c] += magic_bits(pv[c]);
        if (r == lead) Ip[c] = magic_int(pv[c]) + (int)m * cwi[c];
      }
    }
    BlockFixF bf[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int S = (int)(sb[c] - (uint32_t)nb * kMagicBits) + cwi[c] * msum;
      bf[c] = block_fix_f(hc, S, Ip[c]);
    }
    for (int r = 0; r < nb; ++r) {
      const RowTerms t = row_terms(f, k0 + r, inv_sw, true);
      const float A = __fmul_rn(t.sc, t.hd);
      const float B = __fmul_rn(t.sc, __fmaf_rn(t.hR, y.h, __fmul_rn(t.hR, y.l)));
      const float4 kq = make_float4(t.sc, A, B, t.m);
      if (!jv) continue;
      float *po = prow(r);
      const float4 P = *reinterpret_cast<const float4 *>(po);
      const float pv[4] = {P.x, P.y, P.z, P.w};
      float o4[4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
        o4[c] = r == lead ? dequant(kq, bf[c].lead, U[c])
                       : dequant(kq, reflect_f(pv[c], kq, cwc[c], bf[c]), U[c]);
      __stcs(reinterpret_cast<float4 *>(po), make_float4(o4[0], o4[1], o4[2], o4[3]));
    }
  } else {
    // int64 integer parts I = P + m CWc, float-float reflection
    long long S[4] = {0, 0, 0, 0}, Ipl[4] = {0, 0, 0, 0};
    for (int r = 0; r < nb && jv; ++r) {
      const long long m = __float2ll_rn(rintf(two_sum((float)f.og, zero_of(f, k0 + r)).h));
      const float4 P = *reinterpret_cast<const float4 *>(prow(r));
      const float pv[4] = {P.x, P.y, P.z, P.w};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const long long I = pint(pv[c]) + m * cwi[c];
        S[c] += I;
        if (r == lead) Ipl[c] = I;
      }
    }
    ff rS[4], beta[4];
    if (refl) {
      const HhConst hc = hh_const(nb);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        rS[c] = ff_mul(hc.rho, ff_from_int(S[c]));
        beta[c] = ff_mul(hc.kap, ff_add(rS[c], ff_neg(ff_from_int(Ipl[c]))));
      }
    }
    for (int r = 0; r < nb && jv; ++r) {
      const RowTerms t = row_terms(f, k0 + r, inv_sw, refl);
      float *po = prow(r);
      const float4 P = *reinterpret_cast<const float4 *>(po);
      const float pv[4] = {P.x, P.y, P.z, P.w};
      const long long m = __float2ll_rn(t.m);
      float o4[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const ff I = ff_from_int(pint(pv[c]) + m * cwi[c]);
        ff v = !refl ? I : (r == lead ? rS[c] : ff_add(I, ff_neg(beta[c])));
        v = ff_add(v, two_prod(t.hd, U[c]));
        v = ff_add(v, ff_mul({t.hR, 0.0f}, y));
        o4[c] = __fmul_rn(t.sc, ff_round(v));
      }
      __stcs(reinterpret_cast<float4 *>(po), make_float4(o4[0], o4[1], o4[2], o4[3]));
    }
  }
}

// Tiles of a fixed-block grad_X (or of the forward) in the fp32 form that the
// contraction left raw (a row offset m beyond the form): after its last
// tile, every epilogue warp of the CTA takes every nwarps-th (tile, block)
// unit of the CTA's raw tiles -- each lane 4 of the tile's 128 columns --
// with the arithmetic of fix_group_general (int64 integer parts and
// float-float where the fp32 form is not exact).  NB = 1: one row per unit.
template <int NB>
__device__ __noinline__ void gradx_raw_fix(const GemmArgs &g, const uint32_t *raw_mask, int ew,
                                           int nwarps, int lane, bool p_bits) {
  constexpr int NBD = NB > 1 ? NB : 1;
  constexpr int BPT = BN / NBD;  // units per tile
  int64_t n_local = (g.n_items - (int64_t)blockIdx.x + gridDim.x - 1) / gridDim.x;
  if (n_local > kMaxLocalTiles) n_local = kMaxLocalTiles;
  const int nwords = (int)((n_local + 31) / 32);
  bool any = false;
  for (int w = 0; w < nwords; ++w) any |= raw_mask[w] != 0u;
  if (!any) return;
  FixArgs f;
  memset(&f, 0, sizeof(f));
  f.out = g.out;
  f.N = g.N;
  f.D = g.M;
  f.C = (int)g.K;
  f.og = g.og;
  f.ow = g.ow;
  f.bw = g.bw;
  f.b2 = g.b2;
  f.inv_s = g.inv_s;
  f.zero = g.zero;
  f.hz = g.hz;
  f.hr = g.hr;
  f.row_sum = NB > 1 ? nullptr : g.row_sum;
  f.inv_sw = g.inv_sw;
  f.zero_w = g.zero_w;
  f.col_sum_w = g.col_sum_w;
  f.small_p = g.small_p;
  f.p_bits = p_bits;
  f.nbk = NB;
  f.per_tensor = g.kind == FQT_PTQ;
  f.lead = g.lead;
  f.status = g.status;
  const float inv_sw = *g.inv_sw, zw = *g.zero_w;
  const ff y = two_sum((float)g.ow, zw);
  const int Cn = (int)g.K;
  int64_t u = 0;
  for (int w = 0; w < nwords; ++w) {
    uint32_t bits = raw_mask[w];
    while (bits) {
      const int l = w * 32 + __ffs(bits) - 1;
      bits &= bits - 1u;
      const Item t = decode_item(g, (int64_t)blockIdx.x + (int64_t)l * gridDim.x);
      for (int b = 0; b < BPT; ++b, ++u) {
        if ((int)(u % nwarps) != ew) continue;
        const int64_t k0 = t.n0 + (int64_t)b * NBD;
        if (k0 >= g.N) continue;
        const int nb = (int)min((int64_t)NBD, g.N - k0);
        const int64_t j = t.m0 + lane * 4;
        const bool jv = j < g.M;
        float cwc[4], U[4];
        int cwi[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int cs = jv ? g.col_sum_w[j + c] : 0;
          cwc[c] = (float)(cs - Cn * g.ow);
          cwi[c] = (int)cwc[c];
          U[c] = __fmaf_rn((float)Cn, zw, (float)cs);
        }
        int lead = NBD > 1 ? g.lead[k0 / NBD] : 0;
        if (lead < 0 || lead >= nb) lead = 0;
        fix_group_general(f, k0, nb, j, jv, cwc, cwi, U, inv_sw, y, lead);
      }
    }
  }
}

// Groups of more than 32 rows: a CTA each, its warps taking every NW-th
// row (kBigBatch rows in flight per warp) with the int64 integer parts and
// float-float reflection of fix_group_general; the block sums S go through
// shared memory in warp order.
constexpr int kBigFixWarps = 16, kBigBatch = 4;

__global__ void __launch_bounds__(kBigFixWarps * 32) k_grp_fix_big(const FixArgs f) {
  constexpr int NW = kBigFixWarps;
  __shared__ long long s_part[NW][128];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nchunk = (int)((f.D + 127) / 128);
  const int nunits = *f.count_big;
  const float inv_sw = *f.inv_sw, zw = *f.zero_w;
  const ff y = two_sum((float)f.ow, zw);
  const int Cn = f.C;
  for (int u = blockIdx.x; u < nunits; u += gridDim.x) {
    const int64_t gi = f.list_big[u];
    if (gi < 0 || gi >= f.N) {
      if (threadIdx.x == 0) record_status(f.status, FQT_EINVAL);
      continue;
    }
    const int64_t k0 = f.gstart[gi];
    int64_t k1 = f.gstart[gi + 1];
    if (k1 > f.N) k1 = f.N;
    if (k0 < 0 || k1 - k0 < 2) continue;
    const int nb = (int)(k1 - k0);
    const HhConst hc = hh_const(nb);
    auto prow = [&](int r) -> int64_t {
      int64_t pr = f.perm[k0 + r];
      return pr < 0 || pr >= f.N ? 0 : pr;
    };
    for (int ch = 0; ch < nchunk; ++ch) {
      const int64_t j = (int64_t)ch * 128 + lane * 4;
      const bool jv = j < f.D;
      int cwi[4];
      float U[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int cs = jv ? f.col_sum_w[j + c] : 0;
        cwi[c] = cs - Cn * f.ow;
        U[c] = __fmaf_rn((float)Cn, zw, (float)cs);
      }
      // ---- pass 1: S = sum_k I_k, I = P + m CWc ----
      long long S[4] = {0, 0, 0, 0};
      for (int r0 = warp; r0 < nb; r0 += NW * kBigBatch) {
        float4 P[kBigBatch];
        long long m[kBigBatch];
#pragma unroll
        for (int b = 0; b < kBigBatch; ++b) {
          const int r = r0 + b * NW;
          const bool v = r < nb && jv;
          m[b] = v ? __float2ll_rn(rintf(two_sum((float)f.og, f.zero[k0 + r]).h)) : 0;
          P[b] = v ? *reinterpret_cast<const float4 *>(f.out + prow(r) * f.D + j)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int b = 0; b < kBigBatch; ++b) {
          S[0] += (long long)__float2int_rn(P[b].x) + m[b] * cwi[0];
          S[1] += (long long)__float2int_rn(P[b].y) + m[b] * cwi[1];
          S[2] += (long long)__float2int_rn(P[b].z) + m[b] * cwi[2];
          S[3] += (long long)__float2int_rn(P[b].w) + m[b] * cwi[3];
        }
      }
#pragma unroll
      for (int c = 0; c < 4; ++c) s_part[warp][lane * 4 + c] = S[c];
      // the lead row's integer parts (row 0 of the group)
      long long Ipl[4] = {0, 0, 0, 0};
      if (jv) {
        const long long m0 = __float2ll_rn(rintf(two_sum((float)f.og, f.zero[k0]).h));
        const float4 P0 = *reinterpret_cast<const float4 *>(f.out + prow(0) * f.D + j);
        Ipl[0] = (long long)__float2int_rn(P0.x) + m0 * cwi[0];
        Ipl[1] = (long long)__float2int_rn(P0.y) + m0 * cwi[1];
        Ipl[2] = (long long)__float2int_rn(P0.z) + m0 * cwi[2];
        Ipl[3] = (long long)__float2int_rn(P0.w) + m0 * cwi[3];
      }
      __syncthreads();
      ff rS[4], beta[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        long long tot = 0;
        for (int w = 0; w < NW; ++w) tot += s_part[w][lane * 4 + c];
        rS[c] = ff_mul(hc.rho, ff_from_int(tot));
        beta[c] = ff_mul(hc.kap, ff_add(rS[c], ff_neg(ff_from_int(Ipl[c]))));
      }
      // every warp has read the lead row and the sums before any row is
      // overwritten, and before the next chunk reuses s_part
      __syncthreads();
      // ---- pass 2: offsets and the inverse reflection ----
      for (int r0 = warp; r0 < nb; r0 += NW * kBigBatch) {
        float4 P[kBigBatch];
        int64_t pr[kBigBatch];
#pragma unroll
        for (int b = 0; b < kBigBatch; ++b) {
          const int r = r0 + b * NW;
          const bool v = r < nb && jv;
          pr[b] = v ? prow(r) : 0;
          P[b] = v ? *reinterpret_cast<const float4 *>(f.out + pr[b] * f.D + j)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int b = 0; b < kBigBatch; ++b) {
          const int r = r0 + b * NW;
          if (r >= nb || !jv) continue;
          const RowTerms t = row_terms(f, k0 + r, inv_sw, true);
          const long long m = __float2ll_rn(t.m);
          const float pv[4] = {P[b].x, P[b].y, P[b].z, P[b].w};
          float o4[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const ff I = ff_from_int((long long)__float2int_rn(pv[c]) + m * cwi[c]);
            ff v = r == 0 ? rS[c] : ff_add(I, ff_neg(beta[c]));
            v = ff_add(v, two_prod(t.hd, U[c]));
            v = ff_add(v, ff_mul({t.hR, 0.0f}, y));
            o4[c] = __fmul_rn(t.sc, ff_round(v));
          }
          __stcs(reinterpret_cast<float4 *>(f.out + pr[b] * f.D + j),
                 make_float4(o4[0], o4[1], o4[2], o4[3]));
        }
      }
    }
  }
}

// Groups of 2 .. 32 rows in the fp32 form: lane r loads the per-row terms
// of row r once; the rows' products are read 8 at a time (independent
// loads) and, for groups of up to 8 rows, kept in registers for the
// second pass.
constexpr int kFixBatch = 8;

__device__ __forceinline__ float4 ld_row4(const FixArgs &f, int pr, int64_t j, bool jv) {
  return jv ? *reinterpret_cast<const float4 *>(f.out + (int64_t)pr * f.D + j)
            : make_float4(0.f, 0.f, 0.f, 0.f);
}

__global__ void __launch_bounds__(256, 4) k_grp_fix(const FixArgs f) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int nchunk = (int)((f.D + 127) / 128);
  const int64_t nunits = (int64_t)*f.count;
  const float inv_sw = *f.inv_sw, zw = *f.zero_w;
  const ff y = two_sum((float)f.ow, zw);
  const int Cn = f.C;
  for (int64_t u = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); u < nunits;
       u += nw) {
    const int64_t gi = f.list[u];
    if (gi < 0 || gi >= f.N) {
      if (lane == 0) record_status(f.status, FQT_EINVAL);
      continue;
    }
    const int64_t k0 = f.gstart[gi];
    int64_t k1 = f.gstart[gi + 1];
    if (k1 > f.N) k1 = f.N;
    if (k0 < 0 || k1 <= k0) continue;
    const int nb = (int)(k1 - k0);
    // ---- per-row terms, lane r for row r (groups of up to 32 rows) ----
    bool fast = nb >= 2 && nb <= 32 && f.small_p;
    float4 kq = make_float4(0.f, 0.f, 0.f, 0.f);
    int pr = 0;
    if (fast) {
      const float mmax = f.mmax_nb[nb];
      bool ok = true;
      if (lane < nb) {
        const RowTerms t = row_terms(f, k0 + lane, inv_sw, true);
        kq = make_float4(t.sc, __fmul_rn(t.sc, t.hd),
                         __fmul_rn(t.sc, __fmaf_rn(t.hR, y.h, __fmul_rn(t.hR, y.l))), t.m);
        ok = fabsf(t.m) <= mmax;
        const int p = f.perm[k0 + lane];
        pr = p < 0 || p >= f.N ? 0 : p;
      }
      fast = __all_sync(0xffffffffu, ok);
    }
    int msum = (int)kq.w;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) msum += __shfl_xor_sync(0xffffffffu, msum, off);
    const float mp = __shfl_sync(0xffffffffu, kq.w, 0);
    const HhConst hc = hh_const(nb >= 2 ? nb : 2);
    for (int ch = 0; ch < nchunk; ++ch) {
      const int64_t j = (int64_t)ch * 128 + lane * 4;
      const bool jv = j < f.D;
      float cwc[4], U[4];
      int cwi[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int cs = jv ? f.col_sum_w[j + c] : 0;
        cwc[c] = (float)(cs - Cn * f.ow);
        cwi[c] = (int)cwc[c];
        U[c] = __fmaf_rn((float)Cn, zw, (float)cs);
      }
      if (!fast) {
        fix_group_general(f, k0, nb, j, jv, cwc, cwi, U, inv_sw, y, 0);
        continue;
      }
      // ---- pass 1: block sums S = sum P + CWc sum m, lead I_p ----
      uint32_t sb[4] = {0u, 0u, 0u, 0u};
      float4 Pb[kFixBatch];
      float4 P0 = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int r0 = 0; r0 < nb; r0 += kFixBatch) {
#pragma unroll
        for (int b = 0; b < kFixBatch; ++b) {
          const int prb = __shfl_sync(0xffffffffu, pr, (r0 + b) & 31);
          Pb[b] = r0 + b < nb ? ld_row4(f, prb, j, jv) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int b = 0; b < kFixBatch; ++b) {
          if (r0 + b >= nb) break;
          sb[0] += magic_bits(Pb[b].x);
          sb[1] += magic_bits(Pb[b].y);
          sb[2] += magic_bits(Pb[b].z);
          sb[3] += magic_bits(Pb[b].w);
        }
        if (r0 == 0) P0 = Pb[0];
      }
      const float p0[4] = {P0.x, P0.y, P0.z, P0.w};
      BlockFixF bf[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int S = (int)(sb[c] - (uint32_t)nb * kMagicBits) + cwi[c] * msum;
        bf[c] = block_fix_f(hc, S, magic_int(p0[c]) + (int)mp * cwi[c]);
      }
      // ---- pass 2: offsets and the inverse reflection ----
      for (int r0 = 0; r0 < nb; r0 += kFixBatch) {
        if (nb > kFixBatch) {
#pragma unroll
          for (int b = 0; b < kFixBatch; ++b) {
            const int prb = __shfl_sync(0xffffffffu, pr, (r0 + b) & 31);
            Pb[b] = r0 + b < nb ? ld_row4(f, prb, j, jv) : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
#pragma unroll
        for (int b = 0; b < kFixBatch; ++b) {
          const int r = r0 + b;
          const int src = r & 31;
          const float4 q = make_float4(__shfl_sync(0xffffffffu, kq.x, src),
                                       __shfl_sync(0xffffffffu, kq.y, src),
                                       __shfl_sync(0xffffffffu, kq.z, src),
                                       __shfl_sync(0xffffffffu, kq.w, src));
          const int prb = __shfl_sync(0xffffffffu, pr, src);
          if (r >= nb || !jv) continue;
          const float pv[4] = {Pb[b].x, Pb[b].y, Pb[b].z, Pb[b].w};
          float o4[4];
#pragma unroll
          for (int c = 0; c < 4; ++c)
            o4[c] = r == 0 ? dequant(q, bf[c].lead, U[c])
                           : dequant(q, reflect_f(pv[c], q, cwc[c], bf[c]), U[c]);
          __stcs(reinterpret_cast<float4 *>(f.out + (int64_t)prb * f.D + j),
                 make_float4(o4[0], o4[1], o4[2], o4[3]));
        }
      }
    }
  }
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
    if (!q_b2 || !qw || !q_b2->codes_f16 || !qw->codes_f16 || !qw->col_sum ||
        !q_b2->inv_s || !q_b2->zero || !qw->inv_s || !qw->zero)
      return FQT_EINVAL;
    // BHQ with block 0: the adaptive groups of App. D.5 (NB = 0 kernels)
    const bool adapt = q_b2->kind == FQT_BHQ && q_b2->block == 0;
    const int nb = adapt ? 0 : (q_b2->kind == FQT_BHQ && q_b2->block > 1 ? q_b2->block : 1);
    if (nb > 1 && (!q_b2->lead || !q_b2->hz || !q_b2->hr)) return FQT_EINVAL;
    if (nb <= 1 && !q_b2->row_sum) return FQT_EINVAL;
    if (adapt && (!q_b2->perm || !q_b2->gstart || !q_b2->gsize || !q_b2->hz || !q_b2->hr))
      return FQT_EINVAL;
    if (nb > 128 || (nb & (nb - 1))) return FQT_EINVAL;
    const int64_t Nr = q_b2->rows, C = q_b2->cols, D = qw->cols;
    if (qw->rows != C || qw->kind != FQT_PTQ) return FQT_EINVAL;
    if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
    if (C > 8192) return FQT_EUNSUPPORTED;  // int32 epilogue bound
    if (!aligned16(q_b2->codes_f16) || !aligned16(qw->codes_f16) || !aligned16(grad_X))
      return FQT_EINVAL;
    if (Nr > 0) {
      // transposed: M = D (columns of W~), N = rows of dH, K = C
      const SplitPlan p = plan_splits(D, Nr, C, qw->bits, q_b2->bits, nsm, false);
      // fp32 form of the integer parts I = P + m CWc: one exact chunk,
      // |P| < 2^22 and |I| (2 + sqrt(nb)) < 2^24 (|I| < 2^24 without
      // reflection) for every row offset |m| <= mmax, with
      // |I| <= C 2^(bw-1) (2^(b-1) + |m|)
      // Without reflection (nb = 1) and with P exact (one chunk), fma(m,
      // CWc, P) is the correctly rounded exact I for every row offset: the
      // value the integer forms round to, so the fp32 form holds for all m.
      const int64_t kc_terms = (int64_t)exact_chunk_blocks(qw->bits, q_b2->bits) * BK;
      const double lim = nb <= 1 ? 16777216.0 : 16777216.0 / (2.0 + sqrt((double)nb));
      const double mmax = nb == 1 ? 1e30
                                  : floor(lim / ((double)C * (double)(1 << (qw->bits - 1)))) -
                                        (double)(1 << (q_b2->bits - 1)) - 1.0;
      const int64_t pmax = C << (qw->bits + q_b2->bits - 2);
      // the block sums of the reflection read |P| < 2^22 off the fp32 bits
      const bool flt = C <= kc_terms && mmax >= 0.0 && (nb <= 1 || pmax < ((int64_t)1 << 22));
      // the adaptive groups need the fp32 form (rows are scattered by perm)
      if (adapt && !flt) return FQT_EUNSUPPORTED;
      const size_t list_bytes = group_list_bytes(Nr);
      if (adapt && ws_bytes < kGemmOffset + list_bytes) return FQT_EWORKSPACE;
      GemmArgs g;
      memset(&g, 0, sizeof(g));
      g.status = status;
      g.kind = q_b2->kind;
      g.og = 1 << (q_b2->bits - 1);
      g.ow = 1 << (qw->bits - 1);
      g.inv_s = q_b2->inv_s;
      g.zero = q_b2->zero;
      g.row_sum = q_b2->row_sum;
      g.lead = q_b2->lead;
      g.hz = q_b2->hz;
      g.hr = q_b2->hr;
      g.flt_mmax = flt ? (float)mmax : -1.0f;
      g.i32_mmax = int32_form_mmax(C, qw->bits, q_b2->bits, nb);
      g.col_sum_w = qw->col_sum;
      g.inv_sw = qw->inv_s;
      g.zero_w = qw->zero;
      g.perm = q_b2->perm;
      g.gsize = q_b2->gsize;
      g.raw_mmax = (float)mmax;
      fqt_status s = run_gemm(qw->codes_f16, 0, qw->bits, q_b2->codes_f16, 1, q_b2->bits,
                              D, Nr, C, p, g, grad_X, MODE_GRADX, nb,
                              adapt ? 2 : epilogue_form(flt, mmax, q_b2->bits), st);
      if (s != FQT_OK) return s;
      if (adapt) {
        FixArgs f;
        memset(&f, 0, sizeof(f));
        f.out = grad_X;
        f.N = Nr;
        f.D = D;
        f.C = (int)C;
        f.og = g.og;
        f.ow = g.ow;
        f.bw = qw->bits;
        f.b2 = q_b2->bits;
        f.inv_s = q_b2->inv_s;
        f.zero = q_b2->zero;
        f.hz = q_b2->hz;
        f.hr = q_b2->hr;
        f.row_sum = q_b2->row_sum;
        f.perm = q_b2->perm;
        f.gstart = q_b2->gstart;
        f.inv_sw = qw->inv_s;
        f.zero_w = qw->zero;
        f.col_sum_w = qw->col_sum;
        f.raw_mmax = (float)mmax;
        f.small_p = pmax < ((int64_t)1 << 22);
        for (int n = 2; n <= 32; ++n) {
          const double l = 16777216.0 / (2.0 + sqrt((double)n));
          f.mmax_nb[n] = (float)(floor(l / ((double)C * (double)(1 << (qw->bits - 1)))) -
                                 (double)(1 << (q_b2->bits - 1)) - 1.0);
        }
        char *lw = static_cast<char *>(ws) + kGemmOffset;
        f.count = reinterpret_cast<int *>(lw);
        f.count_big = reinterpret_cast<int *>(lw + 4);
        f.list = reinterpret_cast<int32_t *>(lw + 256);
        f.list_big = reinterpret_cast<int32_t *>(lw + 256 + (((size_t)Nr * 4 + 255) & ~(size_t)255));
        f.status = status;
        cudaError_t e = cudaMemsetAsync(f.count, 0, 2 * sizeof(int), st);
        if (e != cudaSuccess) return cuda_fail(e, "group list clear");
        k_grp_list<<<(int)((Nr + 255) / 256), 256, 0, st>>>(f);
        k_grp_fix_big<<<nsm * 2, kBigFixWarps * 32, 0, st>>>(f);
        k_grp_fix<<<nsm * 8, 256, 0, st>>>(f);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_fail(e, "group fix-up launch");
      }
    }
  }
  if (grad_W) {
    const fqt_qtensor *qa = q_b1 ? q_b1 : q_b2;
    // the shift quantizer feeds grad_W itself: its codes on the common scale
    const bool shifted = qa && qa->kind == FQT_SHIFT;
    // byte operands: both code sets given as bytes only (no fp16 carriers);
    // the split-K kernel widens them on chip
    const bool bytes = qa && qx && !shifted && !qa->codes_f16 && !qx->codes_f16 && qa->codes &&
                       qx->codes && qx->conv[0] == 0;
    if (!qa || !qx || (!qx->codes_f16 && !bytes) || !qx->col_sum || !qx->inv_s || !qx->zero)
      return FQT_EINVAL;
    if (shifted ? (!qa->shift_f16 || !qa->shift_col_sum || !qa->shift_scale)
                : ((!qa->codes_f16 && !bytes) || !qa->col_sum || !qa->inv_s || !qa->zero))
      return FQT_EINVAL;
    if ((!shifted && qa->kind != FQT_PTQ) || qx->kind != FQT_PTQ) return FQT_EINVAL;
    const void *A16 = bytes ? (const void *)qa->codes
                            : shifted ? (const void *)qa->shift_f16 : (const void *)qa->codes_f16;
    const void *X16 = bytes ? (const void *)qx->codes : (const void *)qx->codes_f16;
    // |shifted code| <= 16 (2^(b-1) - 1) < 2^(b+3): b + 4 bits of centred magnitude
    const int a_bits = shifted ? qa->bits + 4 : qa->bits;
    // an implicit im2col operand (its padding is corrected in the reduction)
    const bool conv = qx->conv[0] > 0;
    const int x_bits = qx->bits;
    const int64_t Nr = qa->rows, C = qa->cols, D = qx->cols;
    if (qx->rows != Nr) return FQT_EINVAL;
    if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
    if (!aligned16(A16) || !aligned16(X16)) return FQT_EINVAL;
    if (conv) {
      const int32_t *g = qx->conv;
      const int64_t oh = (int64_t)g[1] + 2 * g[6] - g[4] + 1, ow = (int64_t)g[2] + 2 * g[6] - g[5] + 1;
      if (oh <= 0 || ow <= 0 || (int64_t)g[0] * oh * ow != Nr || (int64_t)g[4] * g[5] * g[3] != D)
        return FQT_EINVAL;
      // 64-channel boxes; rows of up to 64 pixels (the tile kernel) or of a
      // multiple of 32 (k_gradw)
      if (g[3] % 64 || (ow > 64 && ow % kWBK)) return FQT_EUNSUPPORTED;
      if (padsum_group((int)C, g[6]) == 0) return FQT_EUNSUPPORTED;
    }
    // An implicit im2col operand with output rows of at most 64 pixels takes
    // the split-K tile kernel too: K blocks of 64 slots are rpb = 64 / pw
    // whole output rows of pw (the power of two >= ow) slots, the slots past
    // ow and the rows past oh zero in Q_b1 (out of its bounds), so K runs over
    // n ceil(oh / rpb) 64 slots.
    int cpw = 0, crpb = 0, cybi = 0;
    int64_t Kt = Nr;
    if (conv) {
      const int32_t *g = qx->conv;
      const int ow = g[2] + 2 * g[6] - g[5] + 1, oh = g[1] + 2 * g[6] - g[4] + 1;
      if (ow <= 64 && !bytes) {
        cpw = 8;
        while (cpw < ow) cpw *= 2;
        crpb = 64 / cpw;
        cybi = (oh + crpb - 1) / crpb;
        Kt = (int64_t)g[0] * cybi * 64;
        // the workspace holds the partials of at most 2.5 N slots (tiny
        // images would pad far beyond)
        if (2 * Kt > 5 * Nr) {
          cpw = crpb = cybi = 0;
          Kt = Nr;
        }
      }
    }
    const bool conv_tile = cpw > 0;
    const SplitPlan p = plan_splits(C, D, Kt, a_bits, x_bits, nsm, true);
    const WPlan wp = Nr > 0 ? gradw_plan(Nr, C, D, a_bits, x_bits, nsm) : WPlan{};
    // k_gradw serves the implicit im2col operand with wider output rows (4-D
    // boxes of 32 pixels of one row, ow % 32 == 0); plain matrices take the
    // split-K tile kernel, which measured faster wherever both apply (e.g.
    // 66.7 against 110.8 us on a 200704 x 128 x 512 layer) and widens byte
    // operands
    const bool w_ok = use_gradw(wp, nsm) && conv && !conv_tile;
    if (conv && Nr > 0 && !w_ok && !conv_tile) return FQT_EUNSUPPORTED;
    const int splits = w_ok ? wp.splits : p.splits;
    const size_t pbytes = (size_t)splits * (size_t)C * (size_t)D * 4;
    const int taps = conv ? qx->conv[4] * qx->conv[5] : 0;
    const size_t need = kGemmOffset + pbytes + (conv ? (size_t)C * taps * 4 : 0);
    if (ws_bytes < need) return FQT_EWORKSPACE;
    int32_t *part = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kGemmOffset);
    int32_t *pad_a = reinterpret_cast<int32_t *>(static_cast<char *>(ws) + kGemmOffset + pbytes);
    if (conv && Nr > 0) {
      const int32_t *g = qx->conv;
      const int oh = g[1] + 2 * g[6] - g[4] + 1, ow = g[2] + 2 * g[6] - g[5] + 1;
      cudaError_t e = cudaMemsetAsync(pad_a, 0, (size_t)C * taps * 4, st);
      if (e != cudaSuccess) return cuda_fail(e, "padding sums clear");
      const int grp = padsum_group((int)C, g[6]);
      if (g[6] > 0) {  // without padding no tap reads any
        // about 16 loads per thread: runs of images whose border pixels
        // (bounded by the pad rows and columns) fill a CTA
        const int pd = g[6];
        const int64_t border = (int64_t)std::min(oh, 2 * pd) * ow +
                               (int64_t)std::max(0, oh - 2 * pd) * std::min(ow, 2 * pd);
        const int64_t items = std::max<int64_t>(1, border * (grp / 8));
        const int64_t per = std::max<int64_t>(1, (256 * 16) / items);
        const int ipc = (int)std::min<int64_t>(per, g[0]);
        const dim3 grid((unsigned)((g[0] + ipc - 1) / ipc), (unsigned)((C + grp - 1) / grp));
        const int ncls = (2 * pd + 1) * (2 * pd + 1);
        k_conv_padsum<<<grid, 256, sizeof(int) * (size_t)ncls * grp, st>>>(
            static_cast<const uint16_t *>(A16), (int)C, grp, g[0], ipc, g[1], g[2], g[5], pd, oh,
            ow, taps, pad_a);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_fail(e, "padding sums launch");
      }
    }
    if (Nr > 0 && w_ok) {
      fqt_status s = run_gradw(qx->codes_f16, static_cast<const uint16_t *>(A16), Nr, (int)C,
                               (int)D, wp, part, status, st, conv ? qx->conv : nullptr);
      if (s != FQT_OK) return s;
    } else if (Nr > 0) {
      GemmArgs g;
      memset(&g, 0, sizeof(g));
      g.status = status;
      g.u8 = bytes ? 1 : 0;
      if (conv_tile) {
        const int32_t *cv = qx->conv;
        g.conv = 1;
        g.cpw = cpw;
        g.crpb = crpb;
        g.cybi = cybi;
        g.cnimg = cv[0];
        g.cih = cv[1];
        g.ciw = cv[2];
        g.cin = cv[3];
        g.ckw = cv[5];
        g.cpad = cv[6];
        g.coh = cv[1] + 2 * cv[6] - cv[4] + 1;
        g.cow = cv[2] + 2 * cv[6] - cv[5] + 1;
      }
      fqt_status s = run_gemm(A16, 0, a_bits, X16, 0, qx->bits, C, D, Kt, p, g,
                              part, MODE_PARTIAL, 1, false, st);
      if (s != FQT_OK) return s;
    } else {
      const cudaError_t e = cudaMemsetAsync(part, 0, (size_t)C * D * 4, st);
      if (e != cudaSuccess) return cuda_fail(e, "partial clear");
    }
    ReduceArgs r;
    memset(&r, 0, sizeof(r));
    r.part = part;
    r.splits = Nr > 0 ? splits : 1;
    r.M = C;
    r.N = D;
    r.out_f32 = grad_W;
    r.Kn = Nr;
    // shifted codes are their own carriers (offset 0, zero point 0)
    r.oa = shifted ? 0 : 1 << (qa->bits - 1);
    r.ob = 1 << (qx->bits - 1);
    r.cs_a = shifted ? qa->shift_col_sum : qa->col_sum;
    r.cs_b = qx->col_sum;
    if (conv) {
      r.pad_a = pad_a;
      r.code_zero = qx->col_sum + D;
      r.taps = taps;
      r.cin = qx->conv[3];
    }
    r.inv_a = shifted ? qa->shift_scale : qa->inv_s;
    r.zero_a = shifted ? qa->shift_scale + 1 : qa->zero;
    r.inv_b = qx->inv_s;
    r.zero_b = qx->zero;
    launch_reduce(r, st);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "split-K reduce launch");
  }
  return FQT_OK;
}

// ---------------------------------------------------------------------------
// grad_W without a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they need
// the backward: for example a serving or training loop whose memory budget
// is frozen after warm-up, or a plain C host that has no allocator of its
// own to hand (and must not call cudaMalloc, which can synchronise the
// device and stall other streams).  For them the split-K partials of grad_W
// live in a fixed array inside the library.  Every GPU that loads the
// library holds it until the process exits; all calls on a device share it.
// ---------------------------------------------------------------------------
constexpr size_t kFixedPartialBytes = (size_t)8 << 20;  // 8 MiB of int32 partials
static __device__ __align__(256) unsigned char
    g_fixed_scratch[kHeaderBytes + kFixedPartialBytes];

// Device address of g_fixed_scratch on the current device, looked up once
// per device (the host-side symbol is only a stand-in for it).
static fqt_status fixed_scratch_address(void **out) {
  static void *addr[64] = {nullptr};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "get device");
  if (dev < 0 || dev >= 64) return FQT_EUNSUPPORTED;
  if (!addr[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_fixed_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "fixed scratch address");
    addr[dev] = p;
  }
  *out = addr[dev];
  return FQT_OK;
}

fqt_status grad_w_fixed_scratch(const fqt_qtensor *qa, const fqt_qtensor *qx,
                                float *grad_W, cudaStream_t st) {
  if (!grad_W || !qa || !qx || !qa->codes_f16 || !qx->codes_f16 || !qa->col_sum ||
      !qx->col_sum || !qa->inv_s || !qa->zero || !qx->inv_s || !qx->zero)
    return FQT_EINVAL;
  if (qa->kind != FQT_PTQ || qx->kind != FQT_PTQ) return FQT_EINVAL;
  // an implicit im2col operand stores NHWC codes, not the Nr x D matrix the
  // tile kernel below reads: refuse it before anything is enqueued
  if (qa->conv[0] > 0 || qx->conv[0] > 0) return FQT_EUNSUPPORTED;
  const int64_t Nr = qa->rows, C = qa->cols, D = qx->cols;
  if (qx->rows != Nr || Nr < 0) return FQT_EINVAL;
  if (C % 16 || D % 16) return FQT_EUNSUPPORTED;
  if (!aligned16(qa->codes_f16) || !aligned16(qx->codes_f16)) return FQT_EINVAL;
  // the partials of every split must fit the fixed array
  const size_t per_split = (size_t)C * (size_t)D * 4;
  if (per_split == 0 || per_split > kFixedPartialBytes) return FQT_EWORKSPACE;
  const int max_splits = (int)(kFixedPartialBytes / per_split);
  SplitPlan p = plan_splits(C, D, Nr, qa->bits, qx->bits, device_sm_count(), true);
  if (p.splits > max_splits) {
    // fewer, longer splits; each must stay within the int32 partial bound
    const int64_t max_terms = ((int64_t)1 << 31) >> (qa->bits + qx->bits - 2);
    p.ks_blocks = (p.kb_total + max_splits - 1) / max_splits;
    if (p.ks_blocks * BK > max_terms) return FQT_EWORKSPACE;
    p.splits = (int)((p.kb_total + p.ks_blocks - 1) / p.ks_blocks);
  }
  void *base = nullptr;
  fqt_status s = fixed_scratch_address(&base);
  if (s != FQT_OK) return s;
  // the status word keeps the first condition recorded since the last
  // fqt_fixed_scratch_sync_status (it is zero when the library loads); the
  // partials are fully rewritten by every split, so nothing else needs clearing
  int *status = static_cast<int *>(base);
  int32_t *part = reinterpret_cast<int32_t *>(static_cast<char *>(base) + kHeaderBytes);
  if (Nr == 0) {
    const cudaError_t e = cudaMemsetAsync(grad_W, 0, per_split, st);
    return cuda_fail(e, "grad_W clear");
  }
  GemmArgs g;
  memset(&g, 0, sizeof(g));
  g.status = status;
  s = run_gemm(qa->codes_f16, 0, qa->bits, qx->codes_f16, 0, qx->bits, C, D, Nr, p, g,
               part, MODE_PARTIAL, 1, false, st);
  if (s != FQT_OK) return s;
  ReduceArgs r;
  memset(&r, 0, sizeof(r));
  r.part = part;
  r.splits = p.splits;
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
  return cuda_fail(cudaGetLastError(), "split-K reduce launch");
}

// Status word of the fixed array (its first int): the device-side conditions
// of fqt_grad_w_fixed_scratch calls land there, as they land in a caller's
// workspace for the other calls.
fqt_status fixed_scratch_status(int **out) {
  void *base = nullptr;
  const fqt_status s = fixed_scratch_address(&base);
  if (s == FQT_OK) *out = static_cast<int *>(base);
  return s;
}

// ---------------------------------------------------------------------------
// A wait on an mbarrier that nothing arrives at, bounded by limit_ns: the
// same bounded wait the contraction kernels use, made to run out on purpose
// so that the timeout path (FQT_ETIMEOUT in the status word, the kernel
// returns, the context stays usable) can be checked.  No bulk copy or
// tensor-core operation is in flight.
// ---------------------------------------------------------------------------
__global__ void k_wait_nothing(int *status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait_limit(&bar, 0, status, limit_ns);
}

fqt_status debug_wait_timeout(void *ws, size_t ws_bytes, uint64_t limit_ns,
                              cudaStream_t st) {
  if (limit_ns > 10000000000ull) return FQT_EINVAL;  // at most 10 s
  int *status = nullptr;
  if (ws) {
    if (ws_bytes < kHeaderBytes || ((uintptr_t)ws & 255)) return FQT_EWORKSPACE;
    status = static_cast<int *>(ws);
  } else {
    const fqt_status s = fixed_scratch_status(&status);
    if (s != FQT_OK) return s;
  }
  k_wait_nothing<<<1, 32, 0, st>>>(status, limit_ns);
  return cuda_fail(cudaGetLastError(), "wait test launch");
}

}  // namespace fqt

namespace fqt {

// ---------------------------------------------------------------------------
// Dense tensor-core rates of this GPU, the denominators of the contractions'
// rooflines (kind 0: tcgen05 kind::f16, fp16 x fp16 -> fp32; kind 1: tcgen05
// kind::f8f6f4, e4m3 x e4m3 -> fp32; kind 2: warp-level mma.sync m16n8k32
// u8 x s8 -> s32).  tcgen05 kind::i8 does not assemble for sm_103a.  One CTA
// per SM: one thread issues `iters` rounds of four back-to-back M128 N256
// MMAs (K 16 each for f16, 32 for e4m3, i.e. one 128-byte row of operands)
// into one TMEM accumulator, then waits (bounded) for them to drain.
// Operands are zero: the rates do not depend on the values.
// ---------------------------------------------------------------------------
constexpr int kPeakN = 256;

__device__ __forceinline__ void umma_f8(uint32_t tmem_d, uint64_t a_desc, uint64_t b_desc,
                                        uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__global__ void __launch_bounds__(128, 1) k_peak_umma(int kind, int64_t iters, int *status) {
  extern __shared__ __align__(1024) uint8_t peak_raw[];
  uint8_t *ops = peak_raw + ((1024u - (smem_u32(peak_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tslot;
  const int warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < (int)(kTileBytes + 2 * kTileBytes) / 16; i += blockDim.x)
    reinterpret_cast<uint4 *>(ops)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tslot)),
                 "r"((uint32_t)kPeakN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  if (threadIdx.x == 0) {
    // A: 128 rows x 128 bytes, B: 256 rows x 128 bytes, K-major, 128-byte swizzle
    const uint64_t da = sw128_desc(smem_u32(ops));
    const uint64_t db = sw128_desc(smem_u32(ops + kTileBytes));
    // D fp32; A, B fp16 (kind::f16) or e4m3 (kind::f8f6f4, format 0); K-major
    const uint32_t idesc =
        (1u << 4) | ((uint32_t)(kPeakN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (kind == 0)
          umma_f16(tmem, da + 2 * k, db + 2 * k, idesc, (it | k) ? 1u : 0u);
        else
          umma_f8(tmem, da + 2 * k, db + 2 * k, idesc, (it | k) ? 1u : 0u);
      }
    }
    umma_commit(&bar);
    mbar_wait(&bar, 0, status);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"((uint32_t)kPeakN)
                 : "memory");
  }
}

// mma.sync u8 x s8 -> s32 (m16n8k32): eight independent accumulators per warp
__global__ void __launch_bounds__(256) k_peak_imma(int64_t iters, int *sink) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t a0 = 0x01010101u * (lane & 7), a1 = a0 ^ 0x02020202u, a2 = a0 ^ 0x04040404u,
                 a3 = a0 ^ 0x08080808u, b0 = 0x03030303u, b1 = 0x05050505u;
  int acc[8][4];
#pragma unroll
  for (int c = 0; c < 8; ++c)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[c][i] = 0;
  for (int64_t it = 0; it < iters; ++it) {
#pragma unroll
    for (int c = 0; c < 8; ++c)
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.s32.u8.s8.s32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
          "{%8, %9}, {%0, %1, %2, %3};"
          : "+r"(acc[c][0]), "+r"(acc[c][1]), "+r"(acc[c][2]), "+r"(acc[c][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  }
  int s = 0;
#pragma unroll
  for (int c = 0; c < 8; ++c) s += acc[c][0] + acc[c][1] + acc[c][2] + acc[c][3];
  if (s == 0x7fffffff) *sink = s;  // keeps the accumulators live
}

fqt_status debug_mma_peak(int kind, int64_t iters, double *ops_out, void *ws, size_t ws_bytes,
                          cudaStream_t st) {
  if (kind < 0 || kind > 2 || iters <= 0 || iters > ((int64_t)1 << 32) || !ops_out)
    return FQT_EINVAL;
  if (!ws || ws_bytes < kHeaderBytes || ((uintptr_t)ws & 255)) return FQT_EWORKSPACE;
  int *status = static_cast<int *>(ws);
  const int nsm = device_sm_count();
  if (kind <= 1) {
    const size_t smem = 3 * kTileBytes + 1024;
    cudaError_t e = cudaFuncSetAttribute(k_peak_umma, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "peak attribute");
    k_peak_umma<<<nsm, 128, smem, st>>>(kind, iters, status);
    const double k_per = kind == 0 ? 16.0 : 32.0;
    *ops_out = 2.0 * BM * kPeakN * k_per * 4.0 * (double)iters * nsm;
  } else {
    const int ctas = nsm * 4;
    k_peak_imma<<<ctas, 256, 0, st>>>(iters, status + 1);
    *ops_out = 2.0 * 16 * 8 * 32 * 8.0 * (double)iters * ctas * 8;
  }
  return cuda_fail(cudaGetLastError(), "peak launch");
}

}  // namespace fqt

namespace fqt {

// ---------------------------------------------------------------------------
// grad_X of a stride-1 k x k conv in NHWC, col2im fused (Sec. 2.1: a conv is a
// linear layer on im2col rows; grad_X is summed back over the taps): the
// transposed convolution dX[p, j] = sum over taps t and output channels c of
// Q_b2(dH)[o(p, t), c] W~[c, t, j], o(p, t) the output pixel that tap t of
// input pixel p reads (out of the image: no term).  It needs the scale of
// Q_b2 to be the same for every output pixel of an image -- per tensor (PTQ)
// or per image (fqt_quantize_grad_samples) -- so that it factors out of the
// sum over taps.
//
// Contraction: M = C_in (tiles of 128), N = input pixels (a tile is r whole
// image rows of one image, row j in a slot of `slot` >= W pixels starting on
// a 1024-byte boundary), K = k^2 C_out in blocks of 64 (tap, 64 channels).
// A = W~ read MN-major at column offset tap C_in; B = the dH carriers read by
// one 4-D box (64 channels x W pixels x 1 row x 1 image) per image row at the
// tap's shifted output row and column (TMA fills rows and columns outside the
// image with zero carriers, which add nothing).  Exact integer products in
// fp32 (one exact chunk).
//
// Dequantization.  With a, w the centred codes, the image's offset
// 2^(b-1) + z' = m + d and y = 2^(bw-1) + z_w, for the set T(p) of taps of
// p that read a pixel of the image:
//   V_pj = I_pj + y R_p + d U_T(j),  I_pj = P_pj + m CW_T(j),
//   R_p = sum_{t in T(p)} (row_sum[o(p, t)] - C 2^(b-1) + C m),
//   CW_T(j) = sum_{t in T} sum_c w_ctj,  U_T(j) = CW_T(j) + |T| C y,
// and dX = inv_sw inv_s V.  For k = 3, pad 1 the sets T are the nine border
// classes of p (top / middle / bottom row times left / middle / right
// column); the class tables CW, U are formed once per call.
// ---------------------------------------------------------------------------
constexpr int kCvStages = 4;
constexpr int kCvThreads = 320;  // TMA, MMA, two sets of four epilogue warps
constexpr int kCvClasses = 9;

struct ConvXArgs {
  int n, h, w, cin, cout, k, pad;
  int slot, rows;          // pixel slots per image row in a tile, image rows per tile
  int tiles_per_img, m_tiles;
  int64_t n_items;
  int kb_total, cbs;       // K blocks (taps x channel blocks), channel blocks per tap
  int og, ow;              // 2^(b-1) of Q_b2, of W~
  const float *inv_s, *zero;  // Q_b2: per row (per image constant) or one entry
  int per_tensor;
  const int32_t *row_sum;  // Q_b2 row sums (codes), one per output pixel
  const float *inv_sw, *zero_w;
  const float *cw_cls;     // [9][cin] CW_T(j)
  const float *u_cls;      // [9][cin] U_T(j)
  float *out;              // NHWC n h w cin
  int *status;
};

__device__ __forceinline__ int conv_class(int y, int x, int h, int w) {
  const int cy = y == 0 ? 0 : (y == h - 1 ? 2 : 1);
  const int cx = x == 0 ? 0 : (x == w - 1 ? 2 : 1);
  return cy * 3 + cx;
}

// Class tables: CW_T(j) and U_T(j) for the nine border classes of a 3 x 3
// stride-1 pad-1 conv (T = the taps whose output pixel exists).
__global__ void k_conv_classes(const int32_t *__restrict__ col_sum_w, int cin, int cout,
                               int ow, const float *zero_w, float *cw_cls, float *u_cls) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= cin) return;
  const ff y = two_sum((float)ow, *zero_w);
  for (int cls = 0; cls < kCvClasses; ++cls) {
    const int cy = cls / 3, cx = cls % 3;
    long long cw = 0;
    int taps = 0;
    for (int ky = 0; ky < 3; ++ky)
      for (int kx = 0; kx < 3; ++kx) {
        // top row (cy 0): the tap ky = 2 reads output row -1; bottom: ky = 0
        if ((cy == 0 && ky == 2) || (cy == 2 && ky == 0)) continue;
        if ((cx == 0 && kx == 2) || (cx == 2 && kx == 0)) continue;
        cw += (long long)col_sum_w[(ky * 3 + kx) * cin + j] - (long long)cout * ow;
        ++taps;
      }
    cw_cls[cls * cin + j] = (float)cw;
    // U = CW + |T| C y, rounded once from float-float
    const ff tcy = ff_mul({(float)(taps * cout), 0.0f}, y);
    u_cls[cls * cin + j] = ff_round(ff_add(ff_from_int(cw), tcy));
  }
}

__device__ __forceinline__ void conv_decode(const ConvXArgs &g, int64_t it, int &m0, int &img,
                                            int &y0) {
  const int64_t mt = it % g.m_tiles, pt = it / g.m_tiles;
  m0 = (int)mt * BM;
  img = (int)(pt / g.tiles_per_img);
  y0 = (int)(pt - (int64_t)img * g.tiles_per_img) * g.rows;
}

__global__ void __launch_bounds__(kCvThreads, 1)
    k_gradx_nhwc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const ConvXArgs g) {
  extern __shared__ __align__(1024) uint8_t cv_raw[];
  uint8_t *smem = cv_raw + ((1024u - (smem_u32(cv_raw) & 1023u)) & 1023u);
  uint8_t *ops = smem;  // kCvStages x (A 16 KB, B 16 KB)
  float *pbp = reinterpret_cast<float *>(ops + (size_t)kCvStages * 2 * kTileBytes);  // [2][128]
  int *pcls = reinterpret_cast<int *>(pbp + 2 * 128);                                 // [2][128]
  float *pcw = reinterpret_cast<float *>(pcls + 2 * 128);                  // [2][9][128]
  float *pu = pcw + 2 * kCvClasses * 128;                                  // [2][9][128]
  uint64_t *bars = reinterpret_cast<uint64_t *>(pu + 2 * kCvClasses * 128);
  uint64_t *full = bars, *empty = bars + kCvStages, *accf = empty + kCvStages,
           *acce = accf + 2, *drain = acce + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kCvStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], 4);  // the four warps of the set
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(256u)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t b_bytes = (uint32_t)g.rows * (uint32_t)g.w * 128u;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0;
      for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x) {
        int m0, img, y0;
        conv_decode(g, it, m0, img, y0);
        bool ok = true;
        for (int kb = 0; kb < g.kb_total; ++kb) {
          const int t = kb / g.cbs, cb = kb - t * g.cbs;
          const int ky = t / g.k, kx = t - ky * g.k;
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) { ok = false; break; }
          mbar_expect_tx(&full[s], (uint32_t)kTileBytes + b_bytes);
          uint8_t *sa = ops + (size_t)(2 * s) * kTileBytes;
          uint8_t *sb = sa + kTileBytes;
          // A: W~ columns tap t, c_in m0 .. m0 + 127 (two 64-wide MN atoms), 64 output channels
          tma_load_2d(sa, &tmA, m0 + t * g.cin, cb * 64, &full[s]);
          tma_load_2d(sa + kTileBytes / 2, &tmA, m0 + 64 + t * g.cin, cb * 64, &full[s]);
          // B: per image row of the tile, the carriers of output row y + pad - ky at columns
          // x + pad - kx (x = 0 .. w - 1)
          for (int j = 0; j < g.rows; ++j)
            tma_load_4d(sb + (size_t)j * g.slot * 128, &tmB, cb * 64, g.pad - kx,
                        y0 + j + g.pad - ky, img, &full[s]);
          if (++s == kCvStages) { s = 0; ph ^= 1u; }
        }
        if (!ok) { *abort_flag = 1; break; }
      }
      if (*abort_flag) {
        sleep_ns(200000);  // copies in flight land before the CTA exits
      } else {
        for (int i = 0; i < kCvStages; ++i) {
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) break;
          if (++s == kCvStages) { s = 0; ph ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      int s = 0;
      uint32_t ph = 0, aph = 0;
      const uint32_t idesc = make_idesc(true, false);  // A MN-major, B K-major
      int64_t local = 0;
      for (int64_t it = blockIdx.x; it < g.n_items && !*abort_flag; it += gridDim.x, ++local) {
        const int buf = (int)(local & 1);
        if (!mbar_wait(&acce[buf], ((aph >> buf) & 1u) ^ 1u, g.status)) { *abort_flag = 1; break; }
        tc_fence_after();
        const uint32_t dt = tmem + (uint32_t)(buf * BN);
        bool ok = true;
        for (int kb = 0; kb < g.kb_total; ++kb) {
          if (!mbar_wait(&full[s], ph, g.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a_addr = smem_u32(ops + (size_t)(2 * s) * kTileBytes);
          const uint64_t da = sw128_desc_mn(a_addr, (uint32_t)(kTileBytes / 2), 1024);
          const uint64_t db = sw128_desc(a_addr + (uint32_t)kTileBytes);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            umma_f16(dt, da + (2048u >> 4) * k, db + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
          if (++s == kCvStages) { s = 0; ph ^= 1u; }
        }
        umma_commit(&accf[buf]);
        aph ^= 1u << buf;
        if (!ok) { *abort_flag = 1; break; }
      }
      umma_commit(drain);  // every MMA has completed before TMEM is released
      mbar_wait(drain, 0, g.status);
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    // set s owns accumulator s and the tiles local = s, s + 2, ...; warp q
    // of the set reads TMEM lanes 32 q .. 32 q + 31 (output channels)
    const int ew = warp - 2, set = ew >> 2, q = warp & 3;
    const int st = (ew & 3) * 32 + lane;  // 0 .. 127 within the set
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(set * BN);
    float *bp = pbp + set * 128;
    int *cls_s = pcls + set * 128;
    float *cw_s = pcw + set * kCvClasses * 128;
    float *u_s = pu + set * kCvClasses * 128;
    const float inv_sw = *g.inv_sw, zw = *g.zero_w;
    const ff yy = two_sum((float)g.ow, zw);
    const int C = g.cout;
    bool dead = false;
    int cur_m0 = -1;
    int64_t local = set;
    for (;; local += 2) {
      const int64_t it = (int64_t)blockIdx.x + local * (int64_t)gridDim.x;
      if (it >= g.n_items) break;  // the same trip count in the set's four warps
      dead = dead || *abort_flag;
      int m0, img, y0;
      conv_decode(g, it, m0, img, y0);
      // per-image scalars of Q_b2 (one scale per image or per tensor)
      const int64_t prow = (int64_t)img * g.h * g.w;
      const float inv = g.per_tensor ? g.inv_s[0] : g.inv_s[prow];
      const float z = g.per_tensor ? g.zero[0] : g.zero[prow];
      const float sc = __fmul_rn(inv_sw, inv);
      const ff xo = two_sum((float)g.og, z);
      const float m = rintf(xo.h);
      const float dd = ff_round(fast_two_sum(__fsub_rn(xo.h, m), xo.l));
      const float Ad = __fmul_rn(sc, dd);
      // the pixel terms of this tile: thread st takes pixel slot st
      {
        const int jr = st / g.slot, x = st - jr * g.slot, y = y0 + jr;
        const bool pv = !dead && x < g.w && jr < g.rows && y < g.h;
        float B = 0.0f;
        int cl = -1;
        if (pv) {
          cl = conv_class(y, x, g.h, g.w);
          long long R = 0;
          for (int ky = 0; ky < 3; ++ky)
            for (int kx = 0; kx < 3; ++kx) {
              const int oy = y + g.pad - ky, ox = x + g.pad - kx;
              if (oy < 0 || oy >= g.h || ox < 0 || ox >= g.w) continue;
              R += (long long)__ldg(g.row_sum + prow + (int64_t)oy * g.w + ox) -
                   (long long)C * g.og + (long long)C * (long long)m;
            }
          const ff Rf = ff_from_int(R);
          B = __fmul_rn(sc, ff_round(ff_mul(Rf, yy)));
        }
        bp[st] = B;
        cls_s[st] = cl;
        if (m0 != cur_m0) {  // the class tables of this tile's 128 channels
          const int j = m0 + st;
          for (int c = 0; c < kCvClasses; ++c) {
            cw_s[c * 128 + st] = j < g.cin ? __ldg(g.cw_cls + c * g.cin + j) : 0.0f;
            u_s[c * 128 + st] = j < g.cin ? __ldg(g.u_cls + c * g.cin + j) : 0.0f;
          }
        }
      }
      cur_m0 = m0;
      asm volatile("bar.sync %0, 128;" ::"r"(1 + set) : "memory");
      const int64_t n_tile = local >> 1;  // this set's earlier tiles
      bool got = false;
      if (!dead) got = mbar_wait(&accf[set], (uint32_t)(n_tile & 1), g.status);
      got = __all_sync(0xffffffffu, got);
      if (!got) {
        if (!dead) *abort_flag = 1;
        dead = true;
      }
      if (!dead) {
        tc_fence_after();
        const int jl = q * 32 + lane, j = m0 + jl;
        const bool jv = j < g.cin;
#pragma unroll 1
        for (int b = 0; b < BN / 32; ++b) {
          uint32_t r[32];
          tmem_ld32_nw(lane_base + (uint32_t)(b * 32), r);
          tmem_wait_ld(r);
          if (b == BN / 32 - 1) {  // the accumulator has been read in full
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce[set]);
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int c = b * 32 + i;
            const int cl = cls_s[c];  // warp-uniform
            if (cl < 0 || !jv) continue;
            const float cw = cw_s[cl * 128 + jl], u = u_s[cl * 128 + jl];
            const float I = __fmaf_rn(m, cw, __uint_as_float(r[i]));
            const float v = __fmaf_rn(sc, I, __fmaf_rn(Ad, u, bp[c]));
            const int jr = c / g.slot, x = c - jr * g.slot;
            __stcs(g.out + ((prow + (int64_t)(y0 + jr) * g.w + x) * g.cin + j), v);
          }
        }
      }
      asm volatile("bar.sync %0, 128;" ::"r"(1 + set) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256u)
                 : "memory");
  }
}

static bool make_map_f16_rows(CUtensorMap *m, const void *base, uint64_t n, uint64_t h,
                              uint64_t w, uint64_t c) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {c, w, h, n};
  cuuint64_t strides[3] = {c * 2, w * c * 2, h * w * c * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)w, 1, 1};  // 64 channels of one image row
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(base), dims, strides,
            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t conv_grad_x_ws_bytes(int64_t cin) {
  return kGemmOffset + 2 * (size_t)kCvClasses * (size_t)(cin > 0 ? cin : 0) * sizeof(float) + 256;
}

fqt_status conv_grad_x_nhwc(const fqt_qtensor *q2, const fqt_qtensor *qw, int64_t n, int64_t h,
                            int64_t w, int64_t cin, int k, int pad, float *out, void *ws,
                            size_t ws_bytes, cudaStream_t st) {
  if (!q2 || !qw || !out || n <= 0 || h <= 0 || w <= 0 || cin <= 0) return FQT_EINVAL;
  if (!q2->codes_f16 || !q2->row_sum || !q2->inv_s || !q2->zero || !qw->codes_f16 ||
      !qw->col_sum || !qw->inv_s || !qw->zero)
    return FQT_EINVAL;
  if (k != 3 || pad != 1 || h < 2 || w < 2 || w > 128) return FQT_EUNSUPPORTED;
  const int64_t cout = q2->cols;
  if (q2->rows != n * h * w || qw->rows != cout || qw->cols != 9 * cin) return FQT_EINVAL;
  if (cout % 64 || cin % 32) return FQT_EUNSUPPORTED;
  const bool per_tensor = q2->kind == FQT_PTQ;
  if (!per_tensor && !(q2->kind == FQT_PSQ && q2->rows_per_sample == h * w))
    return FQT_EUNSUPPORTED;  // the scale must be constant over every image's pixels
  if (qw->kind != FQT_PTQ || q2->conv[0] || qw->conv[0]) return FQT_EUNSUPPORTED;
  if (9 * cout > (int64_t)exact_chunk_blocks(q2->bits, qw->bits) * BK) return FQT_EUNSUPPORTED;
  if (!aligned16(q2->codes_f16) || !aligned16(qw->codes_f16) || !aligned16(out))
    return FQT_EINVAL;
  if (!ws || ((uintptr_t)ws & 255) || ws_bytes < conv_grad_x_ws_bytes(cin))
    return FQT_EWORKSPACE;
  char *wb = static_cast<char *>(ws);
  float *cw_cls = reinterpret_cast<float *>(wb + kGemmOffset);
  float *u_cls = cw_cls + kCvClasses * cin;
  k_conv_classes<<<(unsigned)((cin + 127) / 128), 128, 0, st>>>(
      qw->col_sum, (int)cin, (int)cout, 1 << (qw->bits - 1), qw->zero, cw_cls, u_cls);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "class tables launch");
  CUtensorMap ta, tb;
  bool ok = make_map_f16(&ta, qw->codes_f16, (uint64_t)(9 * cin), (uint64_t)cout, 64, BK);
  ok = ok && make_map_f16_rows(&tb, q2->codes_f16, (uint64_t)n, (uint64_t)h, (uint64_t)w,
                               (uint64_t)cout);
  if (!ok) return cuda_fail(cudaErrorInvalidValue, "tensor map encode");
  ConvXArgs g;
  memset(&g, 0, sizeof(g));
  g.n = (int)n;
  g.h = (int)h;
  g.w = (int)w;
  g.cin = (int)cin;
  g.cout = (int)cout;
  g.k = k;
  g.pad = pad;
  g.slot = (int)((w + 7) / 8 * 8);
  g.rows = (int)min((int64_t)(128 / g.slot), h);
  g.tiles_per_img = (int)((h + g.rows - 1) / g.rows);
  g.m_tiles = (int)((cin + BM - 1) / BM);
  g.n_items = n * g.tiles_per_img * (int64_t)g.m_tiles;
  g.cbs = (int)(cout / 64);
  g.kb_total = 9 * g.cbs;
  g.og = 1 << (q2->bits - 1);
  g.ow = 1 << (qw->bits - 1);
  g.inv_s = q2->inv_s;
  g.zero = q2->zero;
  g.per_tensor = per_tensor ? 1 : 0;
  g.row_sum = q2->row_sum;
  g.inv_sw = qw->inv_s;
  g.zero_w = qw->zero;
  g.cw_cls = cw_cls;
  g.u_cls = u_cls;
  g.out = out;
  g.status = reinterpret_cast<int *>(ws);
  const size_t smem = 1024 + (size_t)kCvStages * 2 * kTileBytes +
                      (size_t)(2 * 128 * 2 + 2 * 2 * kCvClasses * 128) * 4 + 16 * 8 + 16;
  e = cudaFuncSetAttribute(k_gradx_nhwc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "conv grad_X shared-memory attribute");
  const int nsm = device_sm_count();
  const int64_t grid = g.n_items < nsm ? g.n_items : nsm;
  k_gradx_nhwc<<<(int)grid, kCvThreads, smem, st>>>(ta, tb, g);
  return cuda_fail(cudaGetLastError(), "conv grad_X launch");
}

}  // namespace fqt
