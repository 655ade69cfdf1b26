// sm_103a masked prefill attention on the 5th-generation tensor cores (Sec. 3.1: the modified
// causal mask over every token of a prompt block).
//
// One CTA per (128-query tile, head, sequence).  The queries are the last tokens of each
// sequence's history; the keys are the sequence's stored rows of one layer, read straight from the
// ragged cache.  Per CTA:
//
//   warp 0       TMA producer: 2-D tiled copies (cp.async.bulk.tensor, swizzled) of 128-row K and V
//                tiles into a ring of shared-memory stages, plus the tile's per-key mask bounds
//   warp 1       one thread issues tcgen05.mma: S = Q K^T into a double-buffered TMEM tile, then
//                O += P V into a TMEM accumulator; completions are signalled with tcgen05.commit
//   warps 2..5   one query row per thread: tcgen05.ld of its S row, the sentinel mask, an online
//                softmax in the exp2 domain, the rescale of its O row in TMEM, P (16-bit) into a
//                swizzled shared-memory tile, and the final O / l
//
// Mask (Sec. 3.1, the same rows a decode at the query would see): stored row i is visible to the
// query at stored row iq exactly when i <= iq <= hid(i), except that a <CL> query sees only itself.
// hid(i) is the stored row of the <CR> that closes a span enclosing row i (its interior stops being
// visible after the <CR>), i itself for a <CL> row under the paper policy, and "never" otherwise;
// the host book computes it per stored row.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "device_common.cuh"
#include "kernels.hpp"

namespace kvc {
namespace {

constexpr int kPfRows = 128;     // queries per tile (MMA M) and keys per tile (QK^T N, PV K)
constexpr int kPfThreads = 192;  // producer warp, MMA warp, 4 softmax warps

// Shared-memory geometry for head dimension D.  Q, K and V tiles are [128 rows][D] split into
// column subtiles of SW bytes per row, the widest swizzle (128 / 64 / 32 bytes) that divides a row;
// each subtile is the canonical K-major (Q, K) or MN-major (V) layout of that swizzle.
template <int D>
struct PfCfg {
  static constexpr int SW = (2 * D) % 128 == 0 ? 128 : (2 * D) % 64 == 0 ? 64 : 32;
  static constexpr int SUB = SW / 2;  // columns per subtile
  static constexpr int NSUB = D / SUB;
  static constexpr uint32_t SUBB = kPfRows * SW;  // bytes of one subtile
  static constexpr uint32_t TILE = kPfRows * D * 2;
  static constexpr int NST = D <= 96 ? 3 : 2;  // K/V stages
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t KV_OFF = TILE;
  static constexpr uint32_t P_OFF = KV_OFF + NST * 2 * TILE;
  static constexpr uint32_t P_BYTES = kPfRows * kPfRows * 2;
  static constexpr uint32_t SMEM = P_OFF + P_BYTES + 1024;  // + slack to align the base to 1024
  static constexpr uint32_t TMEM_COLS = 512;                 // S0 [0,128), S1 [128,256), O [256,256+D)
  static_assert(D % 16 == 0 && SW * NSUB == 2 * D, "bad tile geometry");
  static_assert(SMEM <= 227 * 1024, "shared memory budget");
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

// RoPE (rotate-half) of a query row held in registers: pairs (e, e + HALF) for e < HALF, with the
// rotary half-width a compile-time constant so the row stays in registers.
template <int HALF>
__device__ __forceinline__ void rope_rotate(float* x, int32_t pos, const float2* g) {
#pragma unroll
  for (int e = 0; e < HALF; ++e) {
    float sn, cs;
    rope_sincos(pos, g[e], &sn, &cs);
    const float x1 = x[e], x2 = x[e + HALF];
    x[e] = x1 * cs - x2 * sn;
    x[e + HALF] = x2 * cs + x1 * sn;
  }
}
// rotary_dim / 2 is a multiple of 8 in [8, D/2]
template <int D, int HALF = D / 2>
__device__ __forceinline__ void rope_dispatch(float* x, int half, int32_t pos, const float2* g) {
  if constexpr (HALF >= 8) {
    if (half == HALF)
      rope_rotate<HALF>(x, pos, g);
    else
      rope_dispatch<D, HALF - 8>(x, half, pos, g);
  }
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

template <typename T, int D>
__global__ void __launch_bounds__(kPfThreads, 1)
    prefill_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                   const PrefillArgs a) {
  using Cf = PfCfg<D>;
  constexpr int SW = Cf::SW, SUB = Cf::SUB, NST = Cf::NST;
  extern __shared__ uint8_t pf_smem_raw[];
  __shared__ uint64_t full_bar[NST], empty_bar[NST], s_full[2], s_free[2];
  __shared__ uint64_t q_full, p_full, pv_done, drain;
  // Per stage, the tile's keys against this CTA's query tile [qr0, qr_end): khid has bit c set when
  // key c's bound holds for every query of the tile (hid >= qr_end - 1); klist holds the keys whose
  // bound falls inside it (qr0 <= hid < qr_end - 1: a span closing among the queries), kn of them.
  __shared__ uint4 khid[NST];
  __shared__ int2 klist[NST][kPfRows];
  __shared__ int32_t kn[NST];
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;

  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(pf_smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // work item: blocks of sequence s are [H * Pq[s], H * Pq[s+1]), head-major, longest tile first
  const int64_t bid = blockIdx.x;
  int lo = 0, hi = a.b - 1;  // last s with H * Pq[s] <= bid
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((int64_t)a.H * a.Pq[mid] <= bid)
      lo = mid;
    else
      hi = mid - 1;
  }
  const int s = lo;
  const int nqt = a.Pq[s + 1] - a.Pq[s];
  const int64_t local = bid - (int64_t)a.H * a.Pq[s];
  const int h = (int)(local / nqt);
  const int qt = nqt - 1 - (int)(local % nqt);
  const PState ps = a.ps[s];
  const int qr0 = ps.q0 + kPfRows * qt;                 // first query row of the tile
  const int qr_end = min(qr0 + kPfRows, ps.len);        // one past its last
  const int nk = (qr_end + kPfRows - 1) / kPfRows;      // key tiles [0, nk)
  const int64_t row_base = (int64_t)a.layer * a.H * a.C + a.seq_row0[s] + (int64_t)h * a.cap[s];

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
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 128);
    }
    mbar_init(&q_full, 128);
    mbar_init(&p_full, 128);
    mbar_init(&pv_done, 1);
    mbar_init(&drain, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;

  if (warp == 0) {
    // ---------------- producer ----------------
    int issued = 0;
    bool ok = true;
    for (int j = 0; j < nk; ++j) {
      const int st = j % NST;
      if (j >= NST && !pf_wait(&empty_bar[st], ((j / NST) - 1) & 1, a, &abort_flag)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        mbar_expect_tx(&full_bar[st], 2 * Cf::TILE);
        const int y = (int)(row_base + (int64_t)kPfRows * j);
        const uint32_t kt = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE);
#pragma unroll
        for (int u = 0; u < Cf::NSUB; ++u) {
          tma_load_2d(kt + u * Cf::SUBB, &tm_k, u * SUB, y, &full_bar[st]);
          tma_load_2d(kt + Cf::TILE + u * Cf::SUBB, &tm_v, u * SUB, y, &full_bar[st]);
        }
      }
      ++issued;
      // per-key mask bounds of the tile ((hid << 1) | is_cl; rows past the stored ones: invisible)
      // sorted into the classes above; the causal part (i <= iq) is left to each query
      uint32_t ok_w[4];
      int n_part = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const int c = lane + 32 * w4;
        const int i = kPfRows * j + c;
        const int hid = (i < ps.len ? a.meta[ps.moff + i] : -2) >> 1;
        ok_w[w4] = __ballot_sync(0xFFFFFFFFu, hid >= qr_end - 1);
        const bool part = hid >= qr0 && hid < qr_end - 1;
        const uint32_t pb = __ballot_sync(0xFFFFFFFFu, part);
        if (part) klist[st][n_part + __popc(pb & ((1u << lane) - 1u))] = make_int2(c, hid);
        n_part += __popc(pb);
      }
      if (lane == 0) {
        khid[st] = make_uint4(ok_w[0], ok_w[1], ok_w[2], ok_w[3]);
        kn[st] = n_part;
      }
      __syncwarp();
      mbar_arrive(&full_bar[st]);
    }
    if (!ok && lane == 0) {
      // let the copies already issued land before the CTA exits
      for (int j = max(0, issued - NST); j < issued; ++j) mbar_wait_bounded(&full_bar[j % NST], (j / NST) & 1, 100000000ull);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idS = mma_idesc(Pack16<T>::kType, 0, kPfRows, kPfRows);
      constexpr uint32_t idO = mma_idesc(Pack16<T>::kType, 1, kPfRows, D);
      const uint32_t q_s = smem_addr(sm + Cf::Q_OFF), p_s = smem_addr(sm + Cf::P_OFF);
      bool ok = pf_wait(&q_full, 0, a, &abort_flag);
      tc_fence_after();
      for (int j = 0; ok && j <= nk; ++j) {
        if (j < nk) {
          const int st = j % NST, sb = j & 1;
          ok = pf_wait(&full_bar[st], (j / NST) & 1, a, &abort_flag);
          if (ok && j >= 2) ok = pf_wait(&s_free[sb], ((j - 2) >> 1) & 1, a, &abort_flag);
          if (!ok) break;
          tc_fence_after();
          const uint32_t k_s = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk * 16) / SUB * Cf::SUBB + (kk * 16) % SUB * 2;
            tc_mma(tmem + sb * kPfRows, smem_desc(q_s + off, 16, 8 * SW, SW), smem_desc(k_s + off, 16, 8 * SW, SW),
                   idS, kk > 0);
          }
          tc_commit(&s_full[sb]);
        }
        if (j >= 1) {
          const int jj = j - 1, st = jj % NST;
          ok = pf_wait(&p_full, jj & 1, a, &abort_flag);
          if (!ok) break;
          tc_fence_after();
          const uint32_t v_s = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE + Cf::TILE);
#pragma unroll
          for (int kk = 0; kk < kPfRows / 16; ++kk) {
            tc_mma(tmem + 2 * kPfRows, smem_desc(p_s + (kk >> 2) * (kPfRows * 128) + (kk & 3) * 32, 16, 1024, 128),
                   smem_desc(v_s + kk * 16 * SW, Cf::SUBB, 8 * SW, SW), idO, (jj > 0 || kk > 0));
          }
          tc_commit(&pv_done);
          tc_commit(&empty_bar[st]);
        }
      }
      // every MMA issued above has completed once this phase does
      tc_commit(&drain);
      mbar_wait_bounded(&drain, 0, a.wait_limit_ns);
    }
  } else {
    // ---------------- softmax: one query row per thread ----------------
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // tile row == TMEM lane
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
    const int iq = qr0 + r;  // stored row of this query
    const bool valid = iq < qr_end;
    const int64_t out_row = valid ? ((int64_t)(ps.qtok + (iq - ps.q0)) * a.H + h) * D : 0;
    {
      // the query row, rotated at its position (RoPE), rounded to the cache type, into the K-major tile
      float x[D];
      if (valid) {
        const uint4* src = reinterpret_cast<const uint4*>(a.q + out_row);
#pragma unroll
        for (int c8 = 0; c8 < D / 8; ++c8) {
          const uint4 u = __ldg(src + c8);
          const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = T::f2(w[e]);
            x[c8 * 8 + 2 * e] = f.x;
            x[c8 * 8 + 2 * e + 1] = f.y;
          }
        }
        if (a.rot > 0) rope_dispatch<D>(x, a.rot / 2, a.pos[a.off[s] + iq], a.rope_g);
      } else {
#pragma unroll
        for (int e = 0; e < D; ++e) x[e] = 0.f;
      }
      const uint32_t q_s = smem_addr(sm + Cf::Q_OFF);
#pragma unroll
      for (int c8 = 0; c8 < D / 8; ++c8) {
        const int e0 = c8 * 8;
        const int u = e0 / SUB, cw = (e0 % SUB) / 8;
        const int phys = cw ^ ((r * SW >> 7) & (SW / 16 - 1));
        st_shared_v4(q_s + u * Cf::SUBB + r * SW + phys * 16, Pack16<T>::two(x[e0], x[e0 + 1]),
                     Pack16<T>::two(x[e0 + 2], x[e0 + 3]), Pack16<T>::two(x[e0 + 4], x[e0 + 5]),
                     Pack16<T>::two(x[e0 + 6], x[e0 + 7]));
      }
    }
    fence_proxy_async_smem();
    mbar_arrive(&q_full);
    const bool cl_q = valid && (a.meta[ps.moff + iq] & 1);
    const float c2 = a.c2;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    const uint32_t p_row = smem_addr(sm + Cf::P_OFF) + r * 128;
    for (int j = 0; j < nk; ++j) {
      const int sb = j & 1, st = j % NST;
      // the S tile, and (acquired from the producer directly) the stage's mask bounds; the stage's
      // barrier cannot move to its next phase before this thread releases P of this tile.  Warp-
      // uniform outcome: the tcgen05 loads and stores below are .sync.aligned.
      ok = pf_wait(&s_full[sb], (j >> 1) & 1, a, &abort_flag) &&
           pf_wait(&full_bar[st], (j / NST) & 1, a, &abort_flag);
      if (!__all_sync(0xFFFFFFFFu, ok)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float sv[kPfRows];
#pragma unroll
      for (int c = 0; c < kPfRows; c += 32) tmem_ld32(tl + sb * kPfRows + c, sv + c);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&s_free[sb]);
      const int kb = kPfRows * j;
      // visibility of the tile's keys to this query as four 32-bit words: the causal prefix
      // (key row <= iq) and the tile-wide bound words, plus the listed keys whose bound admits iq; a
      // <CL> query sees only its own row
      const int t = iq - kb;  // last visible column
      uint32_t v0, v1, v2, v3;
      {
        auto prefix = [t](int w) -> uint32_t {
          const int n = t - 32 * w + 1;  // columns of word w at or before t
          return n <= 0 ? 0u : n >= 32 ? 0xFFFFFFFFu : (1u << n) - 1u;
        };
        if (cl_q) {
          auto one = [t](int w) -> uint32_t { return (t >> 5) == w ? 1u << (t & 31) : 0u; };
          v0 = one(0), v1 = one(1), v2 = one(2), v3 = one(3);
        } else {
          const uint4 hw = khid[st];
          v0 = hw.x, v1 = hw.y, v2 = hw.z, v3 = hw.w;
          const int np = kn[st];
          for (int e = 0; e < np; ++e) {
            const int2 ent = klist[st][e];
            if (ent.y >= iq) {
              const uint32_t bit = 1u << (ent.x & 31);
              const int w = ent.x >> 5;
              v0 |= w == 0 ? bit : 0u;
              v1 |= w == 1 ? bit : 0u;
              v2 |= w == 2 ? bit : 0u;
              v3 |= w == 3 ? bit : 0u;
            }
          }
          v0 &= prefix(0), v1 &= prefix(1), v2 &= prefix(2), v3 &= prefix(3);
        }
      }
      if ((v0 & v1 & v2 & v3) != 0xFFFFFFFFu) {
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          sv[e] = (v0 >> e) & 1u ? sv[e] : -INFINITY;
          sv[32 + e] = (v1 >> e) & 1u ? sv[32 + e] : -INFINITY;
          sv[64 + e] = (v2 >> e) & 1u ? sv[64 + e] : -INFINITY;
          sv[96 + e] = (v3 >> e) & 1u ? sv[96 + e] : -INFINITY;
        }
      }
      // row max: a tree over 8 partial maxima keeps the dependency chains short
      float mx8[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mx8[u] = sv[u];
#pragma unroll
      for (int c = 8; c < kPfRows; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], sv[c]);
      const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                             fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      // Reference maximum: moved only when the row maximum grows by more than 2^8 (log2 units), so O
      // is rescaled rarely; P stays below 2^8 and its scale cancels exactly in O / l.
      const float cand = mx * c2;
      const bool move = cand > m + 8.f;
      const float m_new = move ? cand : m;
      const float ref = m_new == -INFINITY ? 0.f : m_new;
      uint32_t pk[kPfRows / 2];
      float rs8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < kPfRows; c += 2) {
        const float p0 = ex2(fmaf(sv[c], c2, -ref));
        const float p1 = ex2(fmaf(sv[c + 1], c2, -ref));
        rs8[(c >> 1) & 7] += p0 + p1;
        pk[c / 2] = Pack16<T>::two(p0, p1);
      }
      const float rs = ((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7]));
      const float alpha = !move ? 1.f : (m == -INFINITY ? 0.f : ex2(m - ref));
      l = l * alpha + rs;
      if (j >= 1) {
        // PV of the previous tile is complete: O may be rescaled and the P tile rewritten
        ok = pf_wait(&pv_done, (j - 1) & 1, a, &abort_flag);
        if (!__all_sync(0xFFFFFFFFu, ok)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xFFFFFFFFu, alpha != 1.f)) {
#pragma unroll
          for (int u = 0; u < D / 16; ++u) {
            float o[16];
            tmem_ld16(tl + 2 * kPfRows + 16 * u, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) o[e] *= alpha;
            tmem_st16(tl + 2 * kPfRows + 16 * u, o);
          }
          tmem_wait_st();
        }
      }
#pragma unroll
      for (int c8 = 0; c8 < kPfRows / 8; ++c8) {
        const int phys = (c8 & 7) ^ (r & 7);
        st_shared_v4(p_row + (c8 >> 3) * (kPfRows * 128) + phys * 16, pk[4 * c8], pk[4 * c8 + 1], pk[4 * c8 + 2],
                     pk[4 * c8 + 3]);
      }
      if (kb + kPfRows > ps.len && kb + r >= ps.len) {
        // a V row past the stored rows (stale or another stream's): zero it so 0 * V stays 0
        const uint32_t v_row = smem_addr(sm + Cf::KV_OFF + st * 2 * Cf::TILE + Cf::TILE) + r * SW;
#pragma unroll
        for (int u = 0; u < Cf::NSUB; ++u)
#pragma unroll
          for (int b16 = 0; b16 < SW / 16; ++b16) st_shared_v4(v_row + u * Cf::SUBB + b16 * 16, 0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(&p_full);
      m = m_new;
    }
    if (ok) ok = pf_wait(&pv_done, (nk - 1) & 1, a, &abort_flag);
    if (__all_sync(0xFFFFFFFFu, ok)) {
      tc_fence_after();
      const float inv = 1.f / l;
#pragma unroll
      for (int u = 0; u < D / 16; ++u) {
        float o[16];
        tmem_ld16(tl + 2 * kPfRows + 16 * u, o);
        tmem_wait_ld();
        if (valid) {
          float4* dst = reinterpret_cast<float4*>(a.out + out_row + 16 * u);
#pragma unroll
          for (int e = 0; e < 4; ++e)
            dst[e] = make_float4(o[4 * e] * inv, o[4 * e + 1] * inv, o[4 * e + 2] * inv, o[4 * e + 3] * inv);
        }
      }
    }
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
  static bool attr_set = false;  // per instantiation; setting it twice is harmless
  if (!attr_set) {
    const cudaError_t e = cudaFuncSetAttribute(prefill_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)PfCfg<D>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  CUtensorMap mk, mv;
  std::memcpy(&mk, maps.k, sizeof mk);
  std::memcpy(&mv, maps.v, sizeof mv);
  prefill_kernel<T, D><<<(unsigned)grid, kPfThreads, PfCfg<D>::SMEM, stream>>>(mk, mv, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t encode_prefill_maps(const Geometry& g, const Buffers& buf, PrefillMaps* maps) {
  static_assert(sizeof(CUtensorMap) == sizeof(maps->k), "tensor map size");
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    g_encode_err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&g_encode),
                                                    12000, cudaEnableDefault, &q);
    if (g_encode_err == cudaSuccess && q != cudaDriverEntryPointSuccess) g_encode_err = cudaErrorNotSupported;
  });
  if (g_encode_err != cudaSuccess) return g_encode_err;
  cudaError_t e = encode_plane(g, buf.k, maps->k);
  if (e == cudaSuccess) e = encode_plane(g, buf.v, maps->v);
  maps->ready = e == cudaSuccess;
  return e;
}

cudaError_t launch_prefill(const Geometry& g, const PrefillMaps& maps, const PrefillArgs& a, int64_t grid,
                           cudaStream_t stream) {
  if (grid <= 0) return cudaSuccess;
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
