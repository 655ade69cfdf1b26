// sm_103a masked prefill attention on the 5th-generation tensor cores (Sec. 3.1: the modified
// causal mask over every token of a prompt block).
//
// Work items are (sequence, head, 128-query tile); the queries are the last tokens of each
// sequence's history, the keys the sequence's stored rows of one layer, read straight from the
// ragged cache.  Persistent CTAs (two per SM for d_head 64 and 80, one otherwise) each walk a
// contiguous range of items that the host balances.  Per CTA:
//
//   warps 0..3   softmax, one query row per thread: tcgen05.ld of its S row, the per-key rule on the
//                tiles that need it, an online softmax in the exp2 domain, P (16-bit) back into TMEM,
//                the rare rescale of its O row, and the final O / l
//   warp 4       TMA producer: 2-D tiled copies (cp.async.bulk.tensor, swizzled) of 128-row K and V
//                tiles into a ring of shared-memory stages, the tile's mask columns and key classes
//   warp 5       one thread issues tcgen05.mma: S = Q K^T (plus the mask columns) into TMEM, then
//                O += P V with P read from TMEM; completions are signalled with tcgen05.commit
//   warps 6, 7   idle (they complete the producer's warpgroup, whose registers go to the softmax)
//
// Mask (Sec. 3.1, the same rows a decode at the query would see): stored row i is visible to the
// query at stored row iq exactly when i <= iq <= hid(i), except that a <CL> query sees only itself.
// hid(i) is the stored row of the <CR> that closes a span enclosing row i (its interior stops being
// visible after the <CR>), i itself for a <CL> row under the paper policy, and "never" otherwise;
// the host book computes it per stored row.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "device_common.cuh"
#include "kernels.hpp"

namespace kvc {
namespace {

constexpr int kPfRows = 128;  // queries per tile (MMA M) and keys per tile (QK^T N, PV K)
// Threads: a softmax warpgroup (one thread per query row), then a warpgroup holding the producer
// warp, the MMA warp and two idle warps (so that registers can be moved between the two).
constexpr int kPfThreads = 256;
// Work items reach the MMA and softmax warps through a ring of this many slots, filled by the
// producer warp as it takes them from the launch's counter.
constexpr int kItemRing = 4;

// Shared-memory geometry for head dimension D.  Q, K and V tiles are [128 rows][D] split into
// column subtiles of SW bytes per row, the widest swizzle (128 / 64 / 32 bytes) that divides a row;
// each subtile is the canonical K-major (Q, K) or MN-major (V) layout of that swizzle.
//
// SPLIT (bf16): the rotated query and the softmax weights P each go to the tensor cores as a high and
// a low 16-bit part (x = hi + lo with hi = bf16(x), lo = bf16(x - hi), 16 significant bits together),
// so q.k and P.V keep the precision that f16 operands give in one part.  With bf16's 8-bit
// significand a single part moves q.k and the P weights by up to 2^-9 relative, more than the
// decode tolerance allows; the low parts cost a second pass of each product on the tensor cores.
template <int D, bool SPLIT_ = false>
struct PfCfg {
  static constexpr bool SPLIT = SPLIT_;
  static constexpr int SW = (2 * D) % 128 == 0 ? 128 : (2 * D) % 64 == 0 ? 64 : 32;
  static constexpr int SUB = SW / 2;  // columns per subtile
  static constexpr int NSUB = D / SUB;
  static constexpr uint32_t SUBB = kPfRows * SW;  // bytes of one subtile
  static constexpr uint32_t TILE = kPfRows * D * 2;
  // d_head 64 and 80 run two CTAs per SM (their softmax steps interleave), each with a single S
  // tile in TMEM and two K/V stages; larger heads run one CTA per SM with a double-buffered S tile.
  static constexpr int CPS = (D == 64 || D == 80) ? 2 : 1;  // CTAs per SM
  static constexpr int SBUF = CPS == 2 ? 1 : 2;              // S tiles in TMEM
  static constexpr bool PSEP = D == 64 && !SPLIT;            // P in TMEM columns of its own
  static constexpr bool XQT = CPS == 2 && !PSEP;             // Q's mask column in TMEM, not smem
  // SPLIT: the low part of the rotated query, the A operand of a second Q.K^T pass, lives in TMEM
  // with two CTAs per SM (whose shared memory is full) and in shared memory with one
  static constexpr bool QLO_TMEM = SPLIT && CPS == 2;
  static constexpr bool QLO_SMEM = SPLIT && CPS == 1;
  static constexpr int NST = CPS == 2 ? 2 : D <= 96 ? 3 : 2;  // K/V stages
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t QLO_OFF = TILE;  // QLO_SMEM only
  static constexpr uint32_t KV_OFF = TILE * (QLO_SMEM ? 2 : 1);
  // Mask columns: one 16-column subtile (32-byte swizzle) appended to Q (a constant) and to every K
  // stage (0 or a large negative number per key), so keys hidden from a whole query tile are masked
  // by the Q.K^T product itself.
  static constexpr uint32_t XQ_OFF = KV_OFF + NST * 2 * TILE;
  static constexpr uint32_t XK_OFF = XQ_OFF + (XQT ? 0 : kPfRows * 32);
  // d_head 64 has shared memory to spare for O / l: each softmax warp stages 32 rows x 32 columns
  // (4 KB, 128-byte swizzle) for a TMA tensor store
  static constexpr bool OSTAGE = D == 64;
  static constexpr uint32_t OST_OFF = (XK_OFF + NST * kPfRows * 32 + 1023) / 1024 * 1024;
  static constexpr uint32_t OST_WARP = 32 * 32 * 4;
  static constexpr uint32_t SMEM = (OSTAGE ? OST_OFF + 4 * OST_WARP : XK_OFF + NST * kPfRows * 32) +
                                   1024;  // + slack to align the base to 1024
  // TMEM.  d_head 64 (two CTAs per SM, 256 columns each): S [0,128), P [128,192) (16-bit, two
  // per column), O [192,256) -- S is released as soon as the softmax has read it, so the next
  // Q.K^T overlaps the softmax.  d_head 80 (two CTAs per SM): S [0,128) with P written over its
  // first 64 columns, O [128,208), Q's mask column [208,216) -- the next Q.K^T follows the P.V.
  // One CTA per SM: S0 [0,128), S1 [128,256), P written over the first 64 columns of its own S
  // tile, then O0 and O1 (alternating per item).  SPLIT: P's high part over the first 64 columns of
  // its S tile and its low part over the other 64 (d_head 64 then lays TMEM out as d_head 80 does);
  // with two CTAs per SM the query's low part follows Q's mask column (D / 2 columns).
  static constexpr uint32_t P_COL = PSEP ? kPfRows : 0;  // else P lives in its S tile
  static constexpr uint32_t PLO_COL = kPfRows / 2;       // SPLIT: P's low part, after its high part
  static constexpr int OBUF = SBUF == 1 ? 1 : 2;
  static constexpr uint32_t O_COL = SBUF == 2 ? 2 * kPfRows : PSEP ? kPfRows + kPfRows / 2 : kPfRows;
  static constexpr uint32_t XQ_COL = O_COL + OBUF * D;  // with XQT: 8 columns, 16 elements per row
  static constexpr uint32_t QLO_COL = XQ_COL + (XQT ? 8 : 0);
  static constexpr uint32_t TMEM_END = QLO_COL + (QLO_TMEM ? D / 2 : 0);
  static constexpr uint32_t TMEM_COLS = TMEM_END <= 256 ? 256 : 512;
  static_assert(TMEM_END <= TMEM_COLS && TMEM_COLS * CPS <= 512, "TMEM budget");
  static_assert(D % 16 == 0 && SW * NSUB == 2 * D, "bad tile geometry");
  static_assert(SMEM <= 227 * 1024 && (CPS == 1 || SMEM + 4096 <= 113 * 1024), "shared memory budget");
  // Registers with two CTAs per SM: each thread is launched with REG_LAUNCH, then the producer's
  // warpgroup gives registers up (setmaxnreg.dec to REG_OTHER) and the softmax warpgroup takes them
  // (setmaxnreg.inc to REG_SOFTMAX); the two shares add up to exactly what the CTA was launched with.
  static constexpr int REG_LAUNCH = 65536 / (CPS * kPfThreads);
  static constexpr int REG_OTHER = 40;
  static constexpr int REG_SOFTMAX = (REG_LAUNCH * kPfThreads - REG_OTHER * 128) / 128 / 8 * 8;
  static_assert(CPS == 1 || REG_SOFTMAX * 128 + REG_OTHER * 128 <= REG_LAUNCH * kPfThreads,
                "setmaxnreg shares exceed the launch allocation");
  static_assert(CPS == 1 || (REG_SOFTMAX <= 256 && REG_SOFTMAX % 8 == 0 && REG_OTHER % 8 == 0), "setmaxnreg range");
};

// ---------------------------------------------------------------------------------------------
// tcgen05 / TMA wrappers
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}
// Tensor store from shared memory (bulk group of the issuing thread) and its waits.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(src)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D (TMEM) += A (TMEM, M rows in lanes, two 16-bit elements per column) x B (shared memory).
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t* r = reinterpret_cast<uint32_t*>(v);
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float* v) {
  const uint32_t* r = reinterpret_cast<const uint32_t*>(v);
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st16u(uint32_t taddr, const uint32_t* r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st8u(uint32_t taddr, const uint32_t* r) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]), "r"(r[1]),
               "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}
__device__ __forceinline__ void tmem_st4u(uint32_t taddr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

// Shared-memory matrix descriptor: start address, leading / stride byte offsets, version 1, and
// the swizzle (layout type 2 = 128 B, 4 = 64 B, 6 = 32 B).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo, int sw) {
  const uint64_t layout = sw == 128 ? 2 : sw == 64 ? 4 : 6;
  return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | (1ull << 46) | (layout << 61);
}
// Instruction descriptor of kind::f16 with an fp32 accumulator: A and B of one 16-bit type
// (0 = f16, 1 = bf16), A K-major, B K-major (0) or MN-major (1), N >> 3, M >> 4.
__host__ __device__ constexpr uint32_t mma_idesc(int ab_type, int b_mn_major, int M, int N) {
  return (1u << 4) | ((uint32_t)ab_type << 7) | ((uint32_t)ab_type << 10) | ((uint32_t)b_mn_major << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

template <typename T>
struct Pack16;
template <>
struct Pack16<F16T> {
  static constexpr int kType = 0;
  static __device__ __forceinline__ uint32_t two(float a, float b) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
  }
};
template <>
struct Pack16<BF16T> {
  static constexpr int kType = 1;
  static __device__ __forceinline__ uint32_t two(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
  }
};

// The two bf16 values of a packed pair as exact binary32 values (low half first).
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}
// SPLIT: x = hi + lo with hi, lo bf16 (a pair at a time): *hi = bf16(x) and the low part is the
// bf16 rounding of x - hi, which binary32 holds exactly (x and hi agree in their leading bits).
__device__ __forceinline__ uint32_t bf16_split2(float2 x, uint32_t* hi) {
  *hi = Pack16<BF16T>::two(x.x, x.y);
  const float2 h = bf16x2_to_float2(*hi);
  const float2 d = __ffma2_rn(h, make_float2(-1.f, -1.f), x);
  return Pack16<BF16T>::two(d.x, d.y);
}

template <typename T>
constexpr bool kSplit = false;
template <>
constexpr bool kSplit<BF16T> = true;

// 16-byte global -> shared copy that does not go through registers (src_bytes 0: zero fill).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr) : "memory");
  return v;
}

// Bits [0, n) of a 32-bit word, n clamped to [0, 32].
__device__ __forceinline__ uint32_t low_bits(int n) { return n <= 0 ? 0u : n >= 32 ? 0xFFFFFFFFu : (1u << n) - 1u; }

__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Named barrier over the softmax warpgroups that also ANDs a flag across them.
__device__ __forceinline__ bool bar_and(int id, int n, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 q, %1, 0;\n\tbar.red.and.pred p, %2, %3, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// Bounded wait that also gives up as soon as another role of the CTA has given up.
__device__ __forceinline__ bool pf_wait(uint64_t* bar, uint32_t parity, const PrefillArgs& a,
                                        volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63u) == 0) {
      if (*abort_flag) return false;
      if (global_ns() - t0 > a.wait_limit_ns) {
        *abort_flag = 1;
        atomicOr(a.status, STATUS_TIMEOUT);
        return false;
      }
    }
  }
}

// One work item: query tile [qr0, qr_end) of (sequence s, head h), read from the host's table.
struct PfItem {
  PState ps;
  int s, h, qr0, qr_end, nk;
  int64_t row_base;  // K/V plane row of stored row 0 of (layer, s, h)
};

__device__ __forceinline__ PfItem pf_item(const PrefillArgs& a, int64_t it) {
  const int4* r = reinterpret_cast<const int4*>(a.items + it);
  const int4 x = __ldg(r), y = __ldg(r + 1), z = __ldg(r + 2);
  PfItem w;
  w.ps = PState{x.x, x.y, x.z, x.w};
  w.s = y.x;
  w.h = y.y;
  w.qr0 = y.z;
  w.qr_end = y.w;
  w.nk = z.x;
  w.row_base = (int64_t)a.layer * a.H * a.C + (int64_t)(((uint64_t)(uint32_t)z.z << 32) | (uint32_t)z.y);
  return w;
}

// Key tile of the j-th step of item it: consecutive items run their key tiles in opposite
// directions, so an item starts on the tiles its predecessor (same (sequence, head), most often)
// read last, while they are still in L2.
__device__ __forceinline__ int pf_key_tile(int64_t it, int j, int nk) { return (it & 1) ? nk - 1 - j : j; }

// Persistent: the CTAs take items in the table's order from the launch's counter, one at a time (the
// producer warp takes an item when it starts streaming it and passes it on through the ring); every
// barrier phase counts tiles over all of the CTA's items, so the producer streams the next item's
// K/V while the current one finishes (with two S tiles, the O accumulator also alternates between
// two TMEM buffers per item).
template <typename T, int D>
__global__ void __launch_bounds__(kPfThreads, PfCfg<D>::CPS)
    prefill_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                   const __grid_constant__ CUtensorMap tm_o, const PrefillArgs a) {
  using Cf = PfCfg<D, kSplit<T>>;
  constexpr int SW = Cf::SW, SUB = Cf::SUB, NST = Cf::NST, SBUF = Cf::SBUF;
  extern __shared__ uint8_t pf_smem_raw[];
  __shared__ uint64_t full_bar[NST], empty_bar[NST], s_full[SBUF], s_free;
  __shared__ uint64_t q_full, p_full, pv_done, drain;
  // the CTA's k-th item in slot k % kItemRing (-1: none left); full: the producer has written it,
  // empty: the MMA thread and the four softmax warps have read it
  __shared__ int64_t item_ring[kItemRing];
  __shared__ uint64_t item_full[kItemRing], item_empty[kItemRing];
  // Per stage, the tile's keys against its item's query tile [qr0, qr_end): khid has bit c set when
  // key c's bound holds for every query of the tile (hid >= qr_end - 1).  The keys whose bound falls
  // inside it (qr0 <= hid < qr_end - 1: a span closing among the queries) come in runs of one bound
  // -- a span's interior shares its <CR>, a <CL> hidden from every later query is a run of one --
  // kept as the bound (rhid) and the column range [cb, ce) (rcol = cb | ce << 16), kn runs.
  __shared__ uint4 khid[NST];
  __shared__ int32_t rhid[NST][kPfRows];
  __shared__ uint32_t rcol[NST][kPfRows];
  __shared__ int32_t kn[NST];
  __shared__ int32_t kslow[NST];  // the tile needs the per-key rule (else its mask columns decide)
  __shared__ PfItem next_item;  // the item after the current one, as the softmax warps found it
  __shared__ int32_t qmeta[kPfRows];  // mask bounds of the query rows of the next item
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;

  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(pf_smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_slot)),
                 "r"(Cf::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (threadIdx.x == 32) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(&full_bar[i], 32);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < SBUF; ++i) mbar_init(&s_full[i], 1);
    mbar_init(&s_free, 128);  // one S tile: the softmax has read it
    mbar_init(&q_full, 128);
    mbar_init(&p_full, 128);
    mbar_init(&pv_done, 1);
    mbar_init(&drain, 1);
    for (int i = 0; i < kItemRing; ++i) {
      mbar_init(&item_full[i], 1);
      mbar_init(&item_empty[i], 1 + 4);
    }
    abort_flag = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  // At the two-CTA register cap, registers go from the producer's warpgroup to the softmax: each
  // role starts with its setmaxnreg (every warp of a warpgroup executes the same one).
  auto regs_other = [] {
    if constexpr (Cf::CPS == 2) asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(Cf::REG_OTHER));
  };

  if (warp == 4) {
    regs_other();
    // ---------------- producer ----------------
    int64_t g = 0;  // tiles issued
    bool ok = true;
    for (uint32_t k = 0; ok; ++k) {
      // take the next item and pass it on
      const int slot = (int)(k % kItemRing);
      if (k >= kItemRing && !pf_wait(&item_empty[slot], ((k / kItemRing) - 1) & 1, a, &abort_flag)) {
        ok = false;
        break;
      }
      int64_t it = -1;
      if (lane == 0) {
        const unsigned long long t = atomicAdd(a.item_counter, 1ull);
        it = t < (unsigned long long)a.n_items ? (int64_t)t : -1;
        item_ring[slot] = it;
        mbar_arrive(&item_full[slot]);
      }
      it = __shfl_sync(0xFFFFFFFFu, it, 0);
      if (it < 0) break;
      const PfItem w = pf_item(a, it);
      for (int j = 0; j < w.nk; ++j, ++g) {
        const int kt = pf_key_tile(it, j, w.nk);
        const int st = (int)(g % NST);
        if (g >= NST && !pf_wait(&empty_bar[st], (uint32_t)((g / NST) - 1) & 1, a, &abort_flag)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          mbar_expect_tx(&full_bar[st], 2 * Cf::TILE);
          const int y = (int)(w.row_base + (int64_t)kPfRows * kt);
          const uint32_t kt = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE);
#pragma unroll
          for (int u = 0; u < Cf::NSUB; ++u) {
            tma_load_2d(kt + u * Cf::SUBB, &tm_k, u * SUB, y, &full_bar[st]);
            tma_load_2d(kt + Cf::TILE + u * Cf::SUBB, &tm_v, u * SUB, y, &full_bar[st]);
          }
        }
        // per-key mask bounds of the tile ((hid << 1) | is_cl; rows past the stored ones: invisible)
        // sorted into the classes above; the causal part (i <= iq) is left to each query
        uint32_t ok_w[4];
        bool none[4];
        int hp[4];  // the key's bound when it falls among the queries, else -3
#pragma unroll
        for (int w4 = 0; w4 < 4; ++w4) {
          const int c = lane + 32 * w4;
          const int i = kPfRows * kt + c;
          const int hid = (i < w.ps.len ? a.meta[w.ps.moff + i] : -2) >> 1;
          none[w4] = i >= w.qr_end || hid < w.qr0;  // visible to no query of the tile
          ok_w[w4] = __ballot_sync(0xFFFFFFFFu, hid >= w.qr_end - 1);
          hp[w4] = hid >= w.qr0 && hid < w.qr_end - 1 ? hid : -3;
        }
        // runs: a listed key starts one unless key c - 1 is listed with the same bound, and ends one
        // unless key c + 1 is
        int n_run = 0;
#pragma unroll
        for (int w4 = 0; w4 < 4; ++w4) {
          const int c = lane + 32 * w4;
          int prev = __shfl_up_sync(0xFFFFFFFFu, hp[w4], 1);
          int next = __shfl_down_sync(0xFFFFFFFFu, hp[w4], 1);
          const int prev_w = w4 > 0 ? __shfl_sync(0xFFFFFFFFu, hp[w4 > 0 ? w4 - 1 : 0], 31) : -3;
          const int next_w = w4 < 3 ? __shfl_sync(0xFFFFFFFFu, hp[w4 < 3 ? w4 + 1 : 3], 0) : -3;
          if (lane == 0) prev = prev_w;
          if (lane == 31) next = next_w;
          const bool start = hp[w4] >= 0 && prev != hp[w4];
          const bool end = hp[w4] >= 0 && next != hp[w4];
          const uint32_t sb = __ballot_sync(0xFFFFFFFFu, start);
          const int rid = n_run + __popc(sb & ((2u << lane) - 1u)) - 1;  // runs started at or before c, less one
          if (start) {
            rhid[st][rid] = hp[w4];
            reinterpret_cast<uint16_t*>(&rcol[st][rid])[0] = (uint16_t)c;
          }
          if (end) reinterpret_cast<uint16_t*>(&rcol[st][rid])[1] = (uint16_t)(c + 1);
          n_run += __popc(sb);
        }
        if (lane == 0) {
          khid[st] = make_uint4(ok_w[0], ok_w[1], ok_w[2], ok_w[3]);
          // per-key masking is needed when a key's visibility differs between the tile's queries
          // (runs; keys at or past the first query: the causal rule, and a <CL> query sees only
          // itself), or when the tile holds rows past the stored ones (their K may be anything)
          kn[st] = n_run;
          kslow[st] = n_run > 0 || kPfRows * (kt + 1) > w.ps.len || kPfRows * (kt + 1) > w.qr0;
        }
        // mask columns of the tile, 0 or a large negative number per key: column 0 for keys no query
        // of the tile may see, column 1 for keys before the query tile (a <CL> query sees only itself)
#pragma unroll
        for (int w4 = 0; w4 < 4; ++w4) {
          const int c = lane + 32 * w4;
          const uint32_t neg = (uint32_t)T::r(-32768.f);
          const uint32_t x01 = (none[w4] ? neg : 0u) | (kPfRows * kt + c < w.qr0 ? neg << 16 : 0u);
          const uint32_t row = smem_addr(sm + Cf::XK_OFF + st * kPfRows * 32) + c * 32;
          const uint32_t sw = (c >> 2) & 1;  // 32-byte swizzle: the two 16-byte halves swap every 4 rows
          st_shared_v4(row + 16 * sw, x01, 0u, 0u, 0u);
          st_shared_v4(row + 16 * (sw ^ 1), 0u, 0u, 0u, 0u);
        }
        fence_proxy_async_smem();
        __syncwarp();
        mbar_arrive(&full_bar[st]);
      }
    }
    if (!ok && lane == 0) {
      // let the copies already issued land before the CTA exits
      for (int64_t t = g > NST ? g - NST : 0; t < g; ++t)
        mbar_wait_bounded(&full_bar[t % NST], (uint32_t)(t / NST) & 1, 100000000ull);
    }
  } else if (warp == 5) {
    regs_other();
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idS = mma_idesc(Pack16<T>::kType, 0, kPfRows, kPfRows);
      constexpr uint32_t idO = mma_idesc(Pack16<T>::kType, 1, kPfRows, D);
      const uint32_t q_s = smem_addr(sm + Cf::Q_OFF);
      [[maybe_unused]] const uint32_t qlo_s = smem_addr(sm + Cf::QLO_OFF);
      const uint32_t xq_s = smem_addr(sm + Cf::XQ_OFF), xk_s = smem_addr(sm + Cf::XK_OFF);
      int64_t g = 0;
      bool ok = true;
      for (uint32_t k = 0; ok; ++k) {
        const int slot = (int)(k % kItemRing);
        if (!(ok = pf_wait(&item_full[slot], (k / kItemRing) & 1, a, &abort_flag))) break;
        const int64_t it = item_ring[slot];
        mbar_arrive(&item_empty[slot]);
        if (it < 0) break;
        const int nk = pf_item(a, it).nk;
        ok = pf_wait(&q_full, k & 1, a, &abort_flag);
        if (!ok) break;
        tc_fence_after();
        const uint32_t o_t = tmem + Cf::O_COL + (Cf::OBUF == 2 ? (k & 1) * D : 0);
        // S = Q K^T of tile gj into its S tile.  One S tile: once the softmax has read S of tile
        // gj - 1.  Two: the tile last held P of tile gj - 2, whose P.V was issued before (tcgen05.mma
        // from one thread run in issue order).
        auto issue_qk = [&](int64_t gj) -> bool {
          const int st = (int)(gj % NST), sb = (int)(gj % SBUF);
          if (!pf_wait(&full_bar[st], (uint32_t)(gj / NST) & 1, a, &abort_flag)) return false;
          if (Cf::PSEP && gj >= 1 && !pf_wait(&s_free, (uint32_t)(gj - 1) & 1, a, &abort_flag)) return false;
          tc_fence_after();
          const uint32_t k_s = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk * 16) / SUB * Cf::SUBB + (kk * 16) % SUB * 2;
            tc_mma(tmem + sb * kPfRows, smem_desc(q_s + off, 16, 8 * SW, SW), smem_desc(k_s + off, 16, 8 * SW, SW),
                   idS, kk > 0);
          }
          // SPLIT with RoPE: + Q_lo K^T (without RoPE the query is exact in the cache type)
          if constexpr (Cf::SPLIT) {
            if (a.rot > 0) {
#pragma unroll
              for (int kk = 0; kk < D / 16; ++kk) {
                const uint32_t off = (kk * 16) / SUB * Cf::SUBB + (kk * 16) % SUB * 2;
                if constexpr (Cf::QLO_TMEM)
                  tc_mma_ts(tmem + sb * kPfRows, tmem + Cf::QLO_COL + 8 * kk, smem_desc(k_s + off, 16, 8 * SW, SW),
                            idS, 1);
                else
                  tc_mma(tmem + sb * kPfRows, smem_desc(qlo_s + off, 16, 8 * SW, SW),
                         smem_desc(k_s + off, 16, 8 * SW, SW), idS, 1);
              }
            }
          }
          // + the mask column: 256 x (0 or -32768) per key
          if constexpr (Cf::XQT)
            tc_mma_ts(tmem + sb * kPfRows, tmem + Cf::XQ_COL, smem_desc(xk_s + st * kPfRows * 32, 16, 8 * 32, 32), idS, 1);
          else
            tc_mma(tmem + sb * kPfRows, smem_desc(xq_s, 16, 8 * 32, 32),
                   smem_desc(xk_s + st * kPfRows * 32, 16, 8 * 32, 32), idS, 1);
          tc_commit(&s_full[sb]);
          return true;
        };
        // O += P V of tile gp (8 TMEM columns of P per 16 keys); the first of an item: O = P V
        auto issue_pv = [&](int64_t gp, bool first) -> bool {
          const int st = (int)(gp % NST);
          if (!pf_wait(&p_full, (uint32_t)gp & 1, a, &abort_flag)) return false;
          tc_fence_after();
          const uint32_t v_s = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE + Cf::TILE);
          const uint32_t p_t = tmem + (Cf::PSEP ? Cf::P_COL : (uint32_t)(gp % SBUF) * kPfRows);
#pragma unroll
          for (int kk = 0; kk < kPfRows / 16; ++kk)
            tc_mma_ts(o_t, p_t + 8 * kk, smem_desc(v_s + kk * 16 * SW, Cf::SUBB, 8 * SW, SW), idO, (!first || kk > 0));
          if constexpr (Cf::SPLIT) {  // + P_lo V
#pragma unroll
            for (int kk = 0; kk < kPfRows / 16; ++kk)
              tc_mma_ts(o_t, p_t + Cf::PLO_COL + 8 * kk, smem_desc(v_s + kk * 16 * SW, Cf::SUBB, 8 * SW, SW), idO, 1);
          }
          tc_commit(&pv_done);
          tc_commit(&empty_bar[st]);
          return true;
        };
        // Q K^T of the next tile goes in ahead of P.V of the current one: it runs while the softmax
        // works on the current tile
        for (int j = 0; ok && j <= nk; ++j) {
          if (SBUF == 1 && !Cf::PSEP) {  // P sits in the one S tile: its P.V before the next Q K^T
            if (j >= 1) ok = issue_pv(g + j - 1, j == 1);
            if (ok && j < nk) ok = issue_qk(g + j);
          } else {
            if (j < nk) ok = issue_qk(g + j);
            if (ok && j >= 1) ok = issue_pv(g + j - 1, j == 1);
          }
        }
        g += nk;
      }
      // every MMA issued above has completed once this phase does
      tc_commit(&drain);
      mbar_wait_bounded(&drain, 0, a.wait_limit_ns);
    }
  } else if (warp < 4) {
    if constexpr (Cf::CPS == 2) asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(Cf::REG_SOFTMAX));
    // ---------------- softmax: one thread per query row ----------------
    constexpr int CW = kPfRows;  // S columns of one thread
    constexpr int NSM = 128;     // softmax threads (named barrier 1)
    const int r = warp * 32 + lane;  // tile row == TMEM lane
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    const float c2 = a.c2;
    // The query rows of item w into the K-major Q tile (row r per thread), in two halves: q_issue
    // starts 16-byte asynchronous copies of the raw row into its swizzled slots (no registers, so
    // they can be issued early, while the previous item's last tile is still in the softmax);
    // q_finish waits for them, rotates the row in place for RoPE (pairs (e, e + rot/2), at the
    // query's position, rounded to the cache type), writes the row's mask columns (256 in column 0;
    // 256 in column 1 for a <CL> query, which the keys before the query tile then mask) and
    // releases the tile to the MMA thread.
    auto q_chunk = [&](int c8) -> uint32_t {  // shared address of 8-column chunk c8 of row r
      const int e0 = c8 * 8;
      const int u = e0 / SUB, cw = (e0 % SUB) / 8;
      const int phys = cw ^ ((r * SW >> 7) & (SW / 16 - 1));
      return smem_addr(sm + Cf::Q_OFF) + u * Cf::SUBB + r * SW + phys * 16;
    };
    auto q_issue = [&](const PfItem& w) {
      const int iq = w.qr0 + r;
      const bool valid = iq < w.qr_end;
      const int64_t row = valid ? ((int64_t)(w.ps.qtok + (iq - w.ps.q0)) * a.H + w.h) * D : 0;
#pragma unroll
      for (int c8 = 0; c8 < D / 8; ++c8) cp_async16(q_chunk(c8), a.q + row + 8 * c8, valid ? 16u : 0u);
      cp_async4(smem_addr(&qmeta[r]), a.meta + (valid ? w.ps.moff + iq : 0), valid ? 4u : 0u);
      cp_async_commit();
    };
    // SPLIT: the address of chunk c8 of row r in the query's low-part tile (QLO_SMEM)
    [[maybe_unused]] auto qlo_chunk = [&](int c8) -> uint32_t {
      return q_chunk(c8) - smem_addr(sm + Cf::Q_OFF) + smem_addr(sm + Cf::QLO_OFF);
    };
    [[maybe_unused]] auto qlo_store = [&](int c8, uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
      if constexpr (Cf::QLO_TMEM)
        tmem_st4u(tl + Cf::QLO_COL + 4 * c8, w0, w1, w2, w3);  // warp-collective: every lane stores
      else
        st_shared_v4(qlo_chunk(c8), w0, w1, w2, w3);
    };
    auto q_finish = [&](const PfItem& w) {
      cp_async_wait_all();
      const int half = a.rot / 2;
      const int iq = w.qr0 + r;
      if constexpr (Cf::SPLIT) {
        // every row (rows past the tile's queries hold zeros), so the TMEM stores are warp-wide
        if (half > 0) {
          const int32_t qpos = iq < w.qr_end ? a.pos[a.off[w.s] + iq] : 0;
          const int hc = half / 8;  // chunks per rotated half
#pragma unroll
          for (int c8 = 0; c8 < D / 16; ++c8) {
            if (c8 < hc) {
              const uint32_t a1 = q_chunk(c8), a2 = q_chunk(c8 + hc);
              const uint4 u1 = ld_shared_v4(a1), u2 = ld_shared_v4(a2);
              const uint32_t w1[4] = {u1.x, u1.y, u1.z, u1.w}, w2[4] = {u2.x, u2.y, u2.z, u2.w};
              uint32_t h1[4], h2[4], l1[4], l2[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 x1 = T::f2(w1[e]), x2 = T::f2(w2[e]);
                float sn0, cs0, sn1, cs1;
                rope_sincos(qpos, a.rope_g[8 * c8 + 2 * e], &sn0, &cs0);
                rope_sincos(qpos, a.rope_g[8 * c8 + 2 * e + 1], &sn1, &cs1);
                l1[e] = bf16_split2(make_float2(x1.x * cs0 - x2.x * sn0, x1.y * cs1 - x2.y * sn1), &h1[e]);
                l2[e] = bf16_split2(make_float2(x2.x * cs0 + x1.x * sn0, x2.y * cs1 + x1.y * sn1), &h2[e]);
              }
              st_shared_v4(a1, h1[0], h1[1], h1[2], h1[3]);
              st_shared_v4(a2, h2[0], h2[1], h2[2], h2[3]);
              qlo_store(c8, l1[0], l1[1], l1[2], l1[3]);
              qlo_store(c8 + hc, l2[0], l2[1], l2[2], l2[3]);
            }
          }
          // the dimensions past the rotary ones are exact: their low part is zero
#pragma unroll
          for (int c8 = 0; c8 < D / 8; ++c8)
            if (c8 >= 2 * hc) qlo_store(c8, 0u, 0u, 0u, 0u);
        }
      } else if (half > 0 && iq < w.qr_end) {
        const int32_t qpos = a.pos[a.off[w.s] + iq];
        for (int c8 = 0; c8 < half / 8; ++c8) {
          const uint32_t a1 = q_chunk(c8), a2 = q_chunk(c8 + half / 8);
          const uint4 u1 = ld_shared_v4(a1), u2 = ld_shared_v4(a2);
          const uint32_t w1[4] = {u1.x, u1.y, u1.z, u1.w}, w2[4] = {u2.x, u2.y, u2.z, u2.w};
          uint32_t o1[4], o2[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 x1 = T::f2(w1[e]), x2 = T::f2(w2[e]);
            float sn0, cs0, sn1, cs1;
            rope_sincos(qpos, a.rope_g[8 * c8 + 2 * e], &sn0, &cs0);
            rope_sincos(qpos, a.rope_g[8 * c8 + 2 * e + 1], &sn1, &cs1);
            o1[e] = Pack16<T>::two(x1.x * cs0 - x2.x * sn0, x1.y * cs1 - x2.y * sn1);
            o2[e] = Pack16<T>::two(x2.x * cs0 + x1.x * sn0, x2.y * cs1 + x1.y * sn1);
          }
          st_shared_v4(a1, o1[0], o1[1], o1[2], o1[3]);
          st_shared_v4(a2, o2[0], o2[1], o2[2], o2[3]);
        }
      }
      const uint32_t x01 = (uint32_t)T::r(256.f) | (qmeta[r] & 1 ? (uint32_t)T::r(256.f) << 16 : 0u);
      if constexpr (Cf::XQT) {
        const uint32_t wd[8] = {x01, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
        tmem_st8u(tl + Cf::XQ_COL, wd);
        tmem_wait_st();  // also the query's low part (QLO_TMEM)
        tc_fence_before();
      } else {
        const uint32_t row = smem_addr(sm + Cf::XQ_OFF) + r * 32;
        const uint32_t sw = (r >> 2) & 1;  // 32-byte swizzle: the two 16-byte halves swap every 4 rows
        st_shared_v4(row + 16 * sw, x01, 0u, 0u, 0u);
        st_shared_v4(row + 16 * (sw ^ 1), 0u, 0u, 0u, 0u);
      }
      fence_proxy_async_smem();
      mbar_arrive(&q_full);
    };

    // the CTA's kk-th item from the ring (-1: none left, -2: the wait gave up); each softmax warp
    // reads it once and releases the slot
    auto take = [&](uint32_t kk) -> int64_t {
      const int slot = (int)(kk % kItemRing);
      if (!pf_wait(&item_full[slot], (kk / kItemRing) & 1, a, &abort_flag)) return -2;
      const int64_t v = item_ring[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&item_empty[slot]);
      return v;
    };
    bool ok = true;
    int64_t g = 0;  // tiles consumed
    uint32_t k = 0;  // items done
    int64_t it = take(0);
    PfItem w{};
    if (it >= 0) {
      w = pf_item(a, it);
      q_issue(w);
      q_finish(w);
    }
    while (it >= 0) {
      int64_t it_next = -1;  // the next item, taken at this item's last tile
      const int iq = w.qr0 + r;  // stored row of this query
      const bool valid = iq < w.qr_end;
      const bool cl_q = valid && (qmeta[r] & 1);
      const uint32_t o_t = tl + Cf::O_COL + (Cf::OBUF == 2 ? (k & 1) * D : 0);
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < w.nk; ++j) {
        const int64_t gj = g + j;
        const int sb = (int)(gj % SBUF), st = (int)(gj % NST);
        // the S tile, and (acquired from the producer directly) the stage's mask bounds; the stage's
        // barrier cannot move to its next phase before this thread releases P of this tile
        ok = ok && pf_wait(&s_full[sb], (uint32_t)(gj / SBUF) & 1, a, &abort_flag) &&
             pf_wait(&full_bar[st], (uint32_t)(gj / NST) & 1, a, &abort_flag);
        const bool wok = __all_sync(0xFFFFFFFFu, ok);  // tcgen05.ld / st are warp-collective
        float sv[CW];
        if (wok) {
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < CW; c += 32) tmem_ld32(tl + sb * kPfRows + c, sv + c);
          tmem_wait_ld();
          tc_fence_before();
        } else {
#pragma unroll
          for (int c = 0; c < CW; ++c) sv[c] = 0.f;
        }
        if (Cf::PSEP) mbar_arrive(&s_free);  // the next Q K^T may overwrite S
        // S of the item's last tile is in: every Q K^T of the item is complete, the next item's
        // queries may go into the Q tile (the producer has taken that item by now: it takes the
        // next one as soon as it has issued this item's last tile)
        if (j == w.nk - 1) {
          it_next = take(k + 1);
          if (it_next == -2) ok = false;
          if (it_next >= 0) {
            const PfItem nx = pf_item(a, it_next);
            q_issue(nx);
            if (lane == 0) next_item = nx;  // every warp writes the same item
          }
        }
        const int kb = kPfRows * pf_key_tile(it, j, w.nk);
        if (kslow[st]) {
          // visibility of the tile's keys to this query as four 32-bit words: the causal prefix (key
          // row <= iq) with the tile-wide bound words plus the runs whose bound admits iq.  Other
          // tiles are masked by their mask columns alone.
          const int t = iq - kb;  // last visible column
          const uint4 hw = khid[st];
          uint32_t v0 = hw.x, v1 = hw.y, v2 = hw.z, v3 = hw.w;
          const int nr = kn[st];
          for (int e = 0; e < nr; ++e) {
            if (rhid[st][e] >= iq) {
              const uint32_t cc = rcol[st][e];
              const int cb = (int)(cc & 0xFFFFu), ce = (int)(cc >> 16);
              v0 |= low_bits(ce) & ~low_bits(cb);
              v1 |= low_bits(ce - 32) & ~low_bits(cb - 32);
              v2 |= low_bits(ce - 64) & ~low_bits(cb - 64);
              v3 |= low_bits(ce - 96) & ~low_bits(cb - 96);
            }
          }
          // the causal prefix; a <CL> query sees its own key alone
          const int t1 = t + 1, t0 = cl_q ? t : 0;
          v0 &= low_bits(t1) & ~low_bits(t0);
          v1 &= low_bits(t1 - 32) & ~low_bits(t0 - 32);
          v2 &= low_bits(t1 - 64) & ~low_bits(t0 - 64);
          v3 &= low_bits(t1 - 96) & ~low_bits(t0 - 96);
          const uint32_t vw[4] = {v0, v1, v2, v3};
#pragma unroll
          for (int c = 0; c < CW; ++c) sv[c] = (vw[c >> 5] >> (c & 31)) & 1u ? sv[c] : -INFINITY;
        }
        // row max: a tree (eight partial maxima: columns 0-7, then pairs of 8-column blocks, then the
        // last block when one is left over)
        static_assert(CW % 8 == 0, "slice width");
        constexpr int kPairEnd = 8 + (CW - 8) / 16 * 16;  // columns [8, kPairEnd) go in pairs of blocks
        float mx8[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) mx8[u] = sv[u];
#pragma unroll
        for (int c = 8; c < kPairEnd; c += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u) mx8[u] = max3(mx8[u], sv[c + u], sv[c + 8 + u]);
        if constexpr (kPairEnd < CW) {
#pragma unroll
          for (int u = 0; u < 8; ++u) mx8[u] = fmaxf(mx8[u], sv[kPairEnd + u]);
        }
        const float mx = max3(max3(mx8[0], mx8[1], mx8[2]), max3(mx8[3], mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]));
        if (!__all_sync(0xFFFFFFFFu, ok)) {
          // no exchange between the warps, so no barrier inside the tile loop -- a warp that stops
          // here meets the others at the barrier after the loop (their bounded waits give up at once
          // once any role has given up)
          ok = false;
          break;
        }
        // Reference maximum: moved only when the row maximum grows by more than 2^8 (log2 units), so
        // O is rescaled rarely; P stays below 2^8 and its scale cancels exactly in O / l.
        const float cand = mx * c2;
        const bool move = cand > m + 8.f;
        const float m_new = move ? cand : m;
        const float ref = m_new == -INFINITY ? 0.f : m_new;
        const float alpha = !move ? 1.f : (m == -INFINITY ? 0.f : ex2(m - ref));
        // pv_done phases are consumed one by one, each while it is the only one that can be pending
        // (the next P.V waits for this tile's P): phase gj - 1 during tile j >= 1, before this
        // tile's P is written (P.V of the previous tile has read its P) and before O is rescaled;
        // an item's last phase in its epilogue.
        // (With two S tiles, P goes into its own S tile, so the wait can come last unless O needs
        // the rescale.)
        bool pv_early = j >= 1;
        if constexpr (SBUF == 2) pv_early = j >= 1 && __any_sync(0xFFFFFFFFu, alpha != 1.f);
        if (pv_early) {
          ok = pf_wait(&pv_done, (uint32_t)(gj - 1) & 1, a, &abort_flag) && ok;
          if (__all_sync(0xFFFFFFFFu, ok) && __any_sync(0xFFFFFFFFu, alpha != 1.f)) {
            tc_fence_after();
#pragma unroll
            for (int u = 0; u < D / 16; ++u) {
              float o[16];
              tmem_ld16(o_t + 16 * u, o);
              tmem_wait_ld();
#pragma unroll
              for (int e = 0; e < 16; ++e) o[e] *= alpha;
              tmem_st16(o_t + 16 * u, o);
            }
          }
        }
        // P = 2^(s c2 - ref) as 16-bit pairs (row r in lane r), stored 32 columns at a time as they
        // are made; the row sum
        const uint32_t p_tl = tl + (Cf::PSEP ? Cf::P_COL : sb * kPfRows);
        float2 rs4[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
        const float2 c2v = make_float2(c2, c2), nref = make_float2(-ref, -ref);
        const bool sok = __all_sync(0xFFFFFFFFu, ok);
        if (sok) tc_fence_after();
#pragma unroll
        for (int q = 0; q < CW / 32; ++q) {
          uint32_t pk[16];
          [[maybe_unused]] uint32_t pl[16];
#pragma unroll
          for (int c = 0; c < 32; c += 2) {
            const float2 x = __ffma2_rn(make_float2(sv[32 * q + c], sv[32 * q + c + 1]), c2v, nref);
            const float2 p = make_float2(ex2(x.x), ex2(x.y));
            rs4[(c >> 1) & 3] = __fadd2_rn(rs4[(c >> 1) & 3], p);
            if constexpr (Cf::SPLIT)
              pl[c / 2] = bf16_split2(p, &pk[c / 2]);
            else
              pk[c / 2] = Pack16<T>::two(p.x, p.y);
          }
          if (sok) tmem_st16u(p_tl + 16 * q, pk);
          if constexpr (Cf::SPLIT) {
            if (sok) tmem_st16u(p_tl + Cf::PLO_COL + 16 * q, pl);
          }
        }
        const float rs = ((rs4[0].x + rs4[0].y) + (rs4[1].x + rs4[1].y)) + ((rs4[2].x + rs4[2].y) + (rs4[3].x + rs4[3].y));
        l = l * alpha + rs;
        tmem_wait_st();
        if (kb + kPfRows > w.ps.len && kb + r >= w.ps.len) {
          // a V row past the stored rows (stale or another stream's): zero it so 0 * V stays 0
          const uint32_t v_row = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE + Cf::TILE) + r * SW;
#pragma unroll
          for (int u = 0; u < Cf::NSUB; ++u)
#pragma unroll
            for (int b16 = 0; b16 < SW / 16; ++b16) st_shared_v4(v_row + u * Cf::SUBB + b16 * 16, 0, 0, 0, 0);
          fence_proxy_async_smem();
        }
        if constexpr (SBUF == 2) {
          if (j >= 1 && !pv_early) ok = pf_wait(&pv_done, (uint32_t)(gj - 1) & 1, a, &abort_flag) && ok;
        }
        tc_fence_before();
        mbar_arrive(&p_full);
        m = m_new;
      }
      // a wait that ran out after the tile loop's last barrier: decided by every thread together
      if (!bar_and(1, NSM, ok)) {
        ok = false;
        break;
      }
      g += w.nk;
      // the next item's queries go in as soon as this item's last S tile is read (every Q K^T of
      // this item is complete), so its first tiles overlap this item's epilogue
      const bool has_next = it_next >= 0;
      __syncwarp();
      const PfItem wn = has_next ? next_item : w;
      if (has_next) q_finish(wn);
      // epilogue: O / l
      ok = pf_wait(&pv_done, (uint32_t)(g - 1) & 1, a, &abort_flag);
      if (!bar_and(1, NSM, ok)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv = 1.f / l;
      if (Cf::OSTAGE && w.qr_end - w.qr0 == kPfRows) {
        // a full tile: 32 columns at a time, each warp's 32 rows through its swizzled staging buffer
        // into one TMA tensor store of box (32 columns, head h, 32 tokens)
        const uint32_t stage_buf = smem_addr(sm + Cf::OST_OFF + warp * Cf::OST_WARP);
        const int tok = w.ps.qtok + (w.qr0 - w.ps.q0) + 32 * warp;  // token of the warp's first row
#pragma unroll
        for (int hc = 0; hc < D / 32; ++hc) {
          float o[32];
          tmem_ld16(o_t + 32 * hc, o);
          tmem_ld16(o_t + 32 * hc + 16, o + 16);
          tmem_wait_ld();
          if (lane == 0) bulk_wait_read0();  // the warp's previous store has read the buffer
          __syncwarp();
#pragma unroll
          for (int k = 0; k < 8; ++k)
            st_shared_v4(stage_buf + lane * 128 + ((k ^ (lane & 7)) << 4), __float_as_uint(o[4 * k] * inv),
                         __float_as_uint(o[4 * k + 1] * inv), __float_as_uint(o[4 * k + 2] * inv),
                         __float_as_uint(o[4 * k + 3] * inv));
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_3d(&tm_o, stage_buf, 32 * hc, w.h, tok);
            bulk_commit();
          }
        }
      } else {
        const int64_t out_row = valid ? ((int64_t)(w.ps.qtok + (iq - w.ps.q0)) * a.H + w.h) * D : -1;
        // O / l to global memory.  Each group of four lanes (four consecutive query rows) swaps float4s
        // so that lane i of the group writes the i-th 16 bytes of each of the four rows in turn: a
        // store instruction covers 64 contiguous bytes of eight rows, not 16 bytes of 32 rows.
        const int gi = lane & 3;
        int64_t orow[4];
  #pragma unroll
        for (int q = 0; q < 4; ++q) orow[q] = __shfl_sync(0xFFFFFFFFu, out_row, (lane & ~3) | q);
  #pragma unroll
        for (int u = 0; u < D / 16; ++u) {
          float o[16];
          tmem_ld16(o_t + 16 * u, o);
          tmem_wait_ld();
          float4 f[4];
  #pragma unroll
          for (int e = 0; e < 4; ++e) f[e] = make_float4(o[4 * e] * inv, o[4 * e + 1] * inv, o[4 * e + 2] * inv, o[4 * e + 3] * inv);
          // 4 x 4 transpose of float4s across the group: exchange with lane gi ^ m the float4s whose
          // index differs from gi in bit m, for m = 2 then 1
  #pragma unroll
          for (int m = 2; m >= 1; m >>= 1) {
            const bool hi = (gi & m) != 0;
  #pragma unroll
            for (int j0 = 0; j0 < 4; ++j0) {
              if (j0 & m) continue;
              const int j1 = j0 | m;
              const float4 snd = hi ? f[j0] : f[j1];
              float4 rcv;
              rcv.x = __shfl_xor_sync(0xFFFFFFFFu, snd.x, m);
              rcv.y = __shfl_xor_sync(0xFFFFFFFFu, snd.y, m);
              rcv.z = __shfl_xor_sync(0xFFFFFFFFu, snd.z, m);
              rcv.w = __shfl_xor_sync(0xFFFFFFFFu, snd.w, m);
              if (hi)
                f[j0] = rcv;
              else
                f[j1] = rcv;
            }
          }
  #pragma unroll
          for (int q = 0; q < 4; ++q)
            if (orow[q] >= 0) reinterpret_cast<float4*>(a.out + orow[q] + 16 * u)[gi] = f[q];
        }
      }
      tc_fence_before();
      // every warp has read the next item (above) before any of them can overwrite it at the next
      // item's last tile
      bar_and(1, NSM, true);
      it = it_next;
      w = wn;
      ++k;
    }
    if (Cf::OSTAGE && lane == 0) bulk_wait0();  // this warp's tensor stores are complete
  } else {
    regs_other();  // the two idle warps of the producer's warpgroup
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(Cf::TMEM_COLS) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
cudaError_t g_encode_err = cudaSuccess;

cudaError_t encode_plane(const Geometry& g, void* base, unsigned char* out) {
  const int sw = (2 * g.D) % 128 == 0 ? 128 : (2 * g.D) % 64 == 0 ? 64 : 32;
  cuuint64_t dims[2] = {(cuuint64_t)g.D, (cuuint64_t)((int64_t)g.M * g.H * g.C)};
  cuuint64_t strides[1] = {(cuuint64_t)g.D * 2};
  cuuint32_t box[2] = {(cuuint32_t)(sw / 2), (cuuint32_t)kPfRows};
  cuuint32_t elem[2] = {1, 1};
  const CUtensorMapSwizzle swz =
      sw == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : sw == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B;
  CUtensorMap m;
  const CUresult r = g_encode(&m, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, base, dims, strides, box, elem,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  std::memcpy(out, &m, sizeof m);
  return cudaSuccess;
}

template <typename T, int D>
cudaError_t launch_prefill_t(const PrefillMaps& maps, const PrefillArgs& a, int64_t grid, cudaStream_t stream) {
  using Cf = PfCfg<D, kSplit<T>>;
  static std::mutex mu;
  static bool attr_set[64] = {};  // per device: the shared-memory opt-in and the register check
  int dev = 0;
  {
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!attr_set[dev]) {
    const cudaError_t e = cudaFuncSetAttribute(prefill_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)Cf::SMEM);
    if (e != cudaSuccess) return e;
    if (Cf::CPS == 2) {
      // the setmaxnreg shares assume each thread starts with exactly REG_LAUNCH registers; with
      // fewer the softmax warpgroup's increase could never be granted, so refuse to launch
      cudaFuncAttributes fa;
      const cudaError_t e2 = cudaFuncGetAttributes(&fa, prefill_kernel<T, D>);
      if (e2 != cudaSuccess) return e2;
      if (fa.numRegs != Cf::REG_LAUNCH) return cudaErrorInvalidConfiguration;
    }
    attr_set[dev] = true;
  }
  CUtensorMap mk, mv, mo;
  std::memcpy(&mk, maps.k, sizeof mk);
  std::memcpy(&mv, maps.v, sizeof mv);
  std::memset(&mo, 0, sizeof mo);
  if (Cf::OSTAGE && a.n_qtok >= kPfRows) {
    // out as [token][head][D] fp32, stored in boxes of 32 columns x one head x 32 tokens from the
    // softmax warps' swizzled staging buffers (only full query tiles take this path)
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)a.H, (cuuint64_t)a.n_qtok};
    cuuint64_t strides[2] = {(cuuint64_t)D * 4, (cuuint64_t)a.H * D * 4};
    cuuint32_t box[3] = {32, 1, 32};
    cuuint32_t elem[3] = {1, 1, 1};
    const CUresult r = g_encode(&mo, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, a.out, dims, strides, box, elem,
                                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  }
  prefill_kernel<T, D><<<(unsigned)grid, kPfThreads, Cf::SMEM, stream>>>(mk, mv, mo, a);
  return cudaGetLastError();
}

}  // namespace

static cudaError_t load_encoder() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    g_encode_err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&g_encode),
                                                    12000, cudaEnableDefault, &q);
    if (g_encode_err == cudaSuccess && q != cudaDriverEntryPointSuccess) g_encode_err = cudaErrorNotSupported;
  });
  return g_encode_err;
}

cudaError_t encode_append_maps(const Geometry& g, const Buffers& buf, const int64_t* seq_row0, const int32_t* cap,
                               unsigned char* out) {
  static_assert(sizeof(CUtensorMap) == 128, "tensor map size");
  if (g.H > 256 || g.D > 256) return cudaErrorNotSupported;  // box dimensions hold at most 256 elements
  cudaError_t e = load_encoder();
  if (e != cudaSuccess) return e;
  for (int kv = 0; kv < 2; ++kv) {
    for (int s = 0; s < g.b; ++s) {
      uint16_t* base = (kv ? buf.v : buf.k) + seq_row0[s] * g.D;
      cuuint64_t dims[4] = {(cuuint64_t)g.D, (cuuint64_t)cap[s], (cuuint64_t)g.H, (cuuint64_t)g.M};
      cuuint64_t strides[3] = {(cuuint64_t)g.D * 2, (cuuint64_t)cap[s] * g.D * 2, (cuuint64_t)g.H * g.C * g.D * 2};
      cuuint32_t box[4] = {(cuuint32_t)g.D, 1, (cuuint32_t)g.H, 1};
      cuuint32_t elem[4] = {1, 1, 1, 1};
      CUtensorMap m;
      const CUresult r = g_encode(&m, CU_TENSOR_MAP_DATA_TYPE_UINT16, 4, base, dims, strides, box, elem,
                                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                                  CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
      std::memcpy(out + 128 * ((size_t)kv * g.b + s), &m, sizeof m);
    }
  }
  return cudaSuccess;
}

cudaError_t encode_prefill_maps(const Geometry& g, const Buffers& buf, PrefillMaps* maps) {
  static_assert(sizeof(CUtensorMap) == sizeof(maps->k), "tensor map size");
  cudaError_t e = load_encoder();
  if (e != cudaSuccess) return e;
  e = encode_plane(g, buf.k, maps->k);
  if (e == cudaSuccess) e = encode_plane(g, buf.v, maps->v);
  maps->ready = e == cudaSuccess;
  return e;
}

int prefill_ctas_per_sm(int D) {
  switch (D) {
    case 64: return PfCfg<64>::CPS;
    case 80: return PfCfg<80>::CPS;
    case 96: return PfCfg<96>::CPS;
    case 128: return PfCfg<128>::CPS;
    default: return 1;
  }
}

cudaError_t launch_prefill(const Geometry& g, const PrefillMaps& maps, const PrefillArgs& a, cudaStream_t stream) {
  if (a.n_items <= 0 || a.n_ctas <= 0) return cudaSuccess;
  const int64_t grid = a.n_ctas;  // persistent: at most one CTA per SM
  const bool bf = g.dtype == 1;
  switch (g.D) {
    case 64:
      return bf ? launch_prefill_t<BF16T, 64>(maps, a, grid, stream) : launch_prefill_t<F16T, 64>(maps, a, grid, stream);
    case 80:
      return bf ? launch_prefill_t<BF16T, 80>(maps, a, grid, stream) : launch_prefill_t<F16T, 80>(maps, a, grid, stream);
    case 96:
      return bf ? launch_prefill_t<BF16T, 96>(maps, a, grid, stream) : launch_prefill_t<F16T, 96>(maps, a, grid, stream);
    case 128:
      return bf ? launch_prefill_t<BF16T, 128>(maps, a, grid, stream)
                : launch_prefill_t<F16T, 128>(maps, a, grid, stream);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace kvc
