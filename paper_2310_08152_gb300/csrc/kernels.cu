// sm_103a kernels of the sentinel-compressed KV decode path.
//
//   append_kernel         new tokens' K/V rows into the ragged cache (+ RoPE on K, + metadata)
//   compact_scan_kernel   keep flags -> warp-ballot/popc + block exclusive scan -> source row of every
//                         destination row, in-place move of the position / history-index metadata
//   compact_move_kernel   in-place, ascending, 16-byte vectorised row moves of every
//                         (layer, K/V, head) stream of the affected sequences
//   decode_kernel         split-K single-query attention over the kept rows: every warp is a worker
//                         that streams its share of the rows through a ring of shared-memory
//                         stages with 1-D TMA bulk copies (cp.async.bulk + mbarrier), does packed
//                         fp32 dot products, warp-shuffle reductions and an online softmax; the
//                         parts of a split (sequence, head) are merged by a log-sum-exp combine done
//                         by the last worker to finish (arrival counter).
//
// No tensor cores: one query per (sequence, head) makes decode a GEMV (1 flop per byte read), far
// below any tensor-core ridge; the kernels are bound by HBM bandwidth.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>
#include <vector>

#include "device_common.cuh"
#include "kernels.hpp"

namespace kvc {
namespace {

constexpr unsigned kFull = 0xFFFFFFFFu;

constexpr int kAppendThreads = 256;
constexpr int64_t kAppendMaxBlocks = 16384;

// ---------------------------------------------------------------------------------------------
// a1: append
// ---------------------------------------------------------------------------------------------
// One (layer, token) unit per block iteration: its plan entry and row addresses are found once, then
// the block's threads split the unit's 16-byte vectors -- every V vector and every unrotated K
// vector of every head (copies), and every pair of rotated K vectors (vec, vec + rot/16) of every
// head -- with 32-bit index arithmetic.  The token's RoPE sines and cosines (rot/2 of them) are
// computed once per unit into shared memory.
template <typename T, int D>
__global__ void __launch_bounds__(kAppendThreads) append_kernel(Geometry g, Static st, Buffers buf,
                                                                const TokPlan* __restrict__ plan, int64_t ntok,
                                                                int64_t n_in, int m0, int n_layers, int write_meta,
                                                                const uint16_t* __restrict__ k_in,
                                                                const uint16_t* __restrict__ v_in) {
  constexpr int VPR = D / 8;
  __shared__ float2 rope_cs[D / 2];  // (cos, sin) of the token's rotated pairs
  const int H = g.H;
  const int hv = g.rot / 16;           // vectors per rotated half
  const int kcopy = VPR - 2 * hv;      // unrotated K vectors per row
  const int per_row = VPR + kcopy;     // copy items per head
  const int n_copy = H * per_row;      // copy items per unit
  const int n_items = n_copy + H * hv; // + rotation items per unit
  const int64_t plane = (int64_t)H * g.C;  // rows per (layer, K/V) plane
  const int64_t n_units = (int64_t)n_layers * ntok;
  for (int64_t u = blockIdx.x; u < n_units; u += gridDim.x) {
    const int l = (int)(u / ntok);
    const TokPlan tp = plan[u - (int64_t)l * ntok];
    const uint16_t* k_src = k_in + ((int64_t)l * n_in + tp.in_tok) * H * D;  // head 0 of the token
    const uint16_t* v_src = v_in + ((int64_t)l * n_in + tp.in_tok) * H * D;
    const int64_t row0 = (int64_t)(m0 + l) * plane + st.seq_row0[tp.s] + tp.row;  // head 0's row
    const int64_t hstride = st.cap[tp.s];                                        // rows between heads
    if (hv > 0) {
      __syncthreads();  // the previous unit's rotations are done with the table
      for (int i = threadIdx.x; i < 8 * hv; i += blockDim.x) {
        float sn, cs;
        rope_sincos(tp.pos, st.rope_g[i], &sn, &cs);
        rope_cs[i] = make_float2(cs, sn);
      }
      __syncthreads();
    }
    // copies: every V vector and every unrotated K vector of every head
    for (int j = threadIdx.x; j < n_copy; j += blockDim.x) {
      const int h = j / per_row, c = j - h * per_row;
      const bool is_v = c < VPR;
      const int vec = is_v ? c : 2 * hv + (c - VPR);
      const uint16_t* src = (is_v ? v_src : k_src) + h * D + vec * 8;
      uint16_t* dst = (is_v ? buf.v : buf.k) + (row0 + h * hstride) * D + vec * 8;
      *reinterpret_cast<uint4*>(dst) = __ldg(reinterpret_cast<const uint4*>(src));
    }
    // rotations: one pair of vectors of one head per item
    for (int j = n_copy + threadIdx.x; j < n_items; j += blockDim.x) {
      const int jr = j - n_copy;
      const int h = jr / hv, vec = jr - h * hv;
      const uint16_t* src = k_src + h * D;
      uint16_t* dst = buf.k + (row0 + h * hstride) * D;
      const uint4 a = __ldg(reinterpret_cast<const uint4*>(src + vec * 8));
      const uint4 b = __ldg(reinterpret_cast<const uint4*>(src + (vec + hv) * 8));
      const uint16_t* xa = reinterpret_cast<const uint16_t*>(&a);
      const uint16_t* xb = reinterpret_cast<const uint16_t*>(&b);
      uint4 ya, yb;
      uint16_t* pa = reinterpret_cast<uint16_t*>(&ya);
      uint16_t* pb = reinterpret_cast<uint16_t*>(&yb);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float2 r = rope_cs[vec * 8 + e];
        const float x1 = T::f1(xa[e]), x2 = T::f1(xb[e]);
        pa[e] = T::r(x1 * r.x - x2 * r.y);
        pb[e] = T::r(x2 * r.x + x1 * r.y);
      }
      *reinterpret_cast<uint4*>(dst + vec * 8) = ya;
      *reinterpret_cast<uint4*>(dst + (vec + hv) * 8) = yb;
    }
    if (write_meta && l == 0 && threadIdx.x == 0) {
      buf.pos[st.off[tp.s] + tp.row] = tp.pos;
      buf.orig[st.off[tp.s] + tp.row] = tp.orig;
    }
  }
}

// a1 through TMA, for calls with at least one (layer, token) unit per SM.  A warp is a worker with
// a ring of kAppStages slots; a slot holds one unit's K and V rows of every head, which lie
// contiguously in the input.  Lane 0 brings a unit in with two bulk copies, kAppLag units ahead,
// and writes it out with two tensor stores over the sequence's 4-D map {d, row, head, layer}: the
// box {d, 1, H, 1} sends each head's row to its own (layer, K/V, head) stream.  With RoPE the warp
// rotates K in shared memory in between.  No registers hold the rows, so several units per warp
// and several warps per SM are in flight.
constexpr int kAppStages = 4;
constexpr int kAppLag = 2;
static_assert(kAppLag >= 1 && kAppLag < kAppStages, "loads run ahead of stores by fewer units than slots");

__host__ __device__ constexpr uint32_t app_slot_bytes(int H, int D) { return ((uint32_t)H * D * 2 + 127u) / 128u * 128u; }
inline size_t app_smem_bytes(int H, int D, int rot) {
  return (size_t)kAppStages * 2 * app_slot_bytes(H, D) + 8 * (size_t)kAppStages + 8 * (size_t)(rot > 1 ? rot / 2 : 1);
}

__device__ __forceinline__ void tma_store_4d(const CUtensorMap* map, const void* src, int x, int y, int z, int w) {
  asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%1, %2, %3, %4}], [%5];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(w), "r"(smem_addr(src))
               : "memory");
}
__device__ __forceinline__ void app_bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// waits until at most N of this thread's bulk groups are still reading shared memory
template <int N>
__device__ __forceinline__ void app_bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void app_bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

template <typename T, int D>
__global__ void __launch_bounds__(32, 1) append_tma_kernel(Geometry g, Static st, Buffers buf,
                                                           const TokPlan* __restrict__ plan, int64_t ntok, int64_t n_in,
                                                           int m0, int n_layers, int write_meta,
                                                           const uint16_t* __restrict__ k_in,
                                                           const uint16_t* __restrict__ v_in,
                                                           const CUtensorMap* __restrict__ maps,
                                                           unsigned long long limit_ns) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int lane = threadIdx.x;
  const int H = g.H;
  const uint32_t ub = (uint32_t)H * D * 2;  // bytes of one unit's K (or V) rows
  const uint32_t slot = app_slot_bytes(H, D);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)kAppStages * 2 * slot);
  float2* cs = reinterpret_cast<float2*>(full + kAppStages);  // (cos, sin) per rotated pair, one unit
  const int hp = g.rot / 2;   // rotated pairs per head
  const int hv = g.rot / 16;  // 16-byte vector pairs per head
  const int64_t n_units = (int64_t)n_layers * ntok;
  const int64_t w = blockIdx.x, NW = gridDim.x;
  const int64_t n_my = w < n_units ? (n_units - 1 - w) / NW + 1 : 0;  // units w, w + NW, ...
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kAppStages; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  __syncwarp();
  int64_t loaded = 0;  // units whose copies lane 0 has issued
  int64_t k = 0;
  for (; k < n_my + kAppLag; ++k) {
    if (k < n_my && lane == 0) {
      const int sl = (int)(k % kAppStages);
      // the slot's previous unit (k - kAppStages) has been read out by its stores: stores of at most
      // kAppStages - 1 - kAppLag newer units may still be reading
      if (k >= kAppStages) app_bulk_wait_read<kAppStages - 1 - kAppLag>();
      fence_proxy_async_smem();  // after the generic accesses (rotation) to the slot's previous unit
      const int64_t u = w + k * NW;
      const int l = (int)(u / ntok);
      const int64_t src = ((int64_t)l * n_in + plan[u - (int64_t)l * ntok].in_tok) * H * D;
      unsigned char* d0 = smem + (size_t)sl * 2 * slot;
      mbar_arrive_expect_tx(&full[sl], 2 * ub);
      bulk_g2s(d0, k_in + src, ub, &full[sl]);
      bulk_g2s(d0 + slot, v_in + src, ub, &full[sl]);
      loaded = k + 1;
    }
    const int64_t j = k - kAppLag;
    if (j < 0 || j >= n_my) continue;
    const int sl = (int)(j % kAppStages);
    const int64_t u = w + j * NW;
    const int l = (int)(u / ntok);
    const TokPlan tp = plan[u - (int64_t)l * ntok];
    if (hv > 0) {
      __syncwarp();  // the previous unit's rotations are done with the table
      for (int i = lane; i < hp; i += 32) {
        float sn, c;
        rope_sincos(tp.pos, st.rope_g[i], &sn, &c);
        cs[i] = make_float2(c, sn);
      }
      __syncwarp();
    }
    if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(&full[sl], (uint32_t)(j / kAppStages) & 1, limit_ns))) {
      if (lane == 0) atomicOr(buf.status, STATUS_TIMEOUT);
      break;
    }
    unsigned char* ks = smem + (size_t)sl * 2 * slot;
    if (hv > 0) {
      for (int it = lane; it < H * hv; it += 32) {
        const int h = it / hv, vec = it - h * hv;
        uint4* qa = reinterpret_cast<uint4*>(ks + ((size_t)h * D + vec * 8) * 2);
        uint4* qb = reinterpret_cast<uint4*>(ks + ((size_t)h * D + (vec + hv) * 8) * 2);
        const uint4 a = *qa, b = *qb;
        const uint16_t* xa = reinterpret_cast<const uint16_t*>(&a);
        const uint16_t* xb = reinterpret_cast<const uint16_t*>(&b);
        uint4 ya, yb;
        uint16_t* pa = reinterpret_cast<uint16_t*>(&ya);
        uint16_t* pb = reinterpret_cast<uint16_t*>(&yb);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float2 r = cs[vec * 8 + e];
          const float x1 = T::f1(xa[e]), x2 = T::f1(xb[e]);
          pa[e] = T::r(x1 * r.x - x2 * r.y);
          pb[e] = T::r(x2 * r.x + x1 * r.y);
        }
        *qa = ya;
        *qb = yb;
      }
      fence_proxy_async_smem();  // the rotated rows, before the tensor store reads them
      __syncwarp();
    }
    if (lane == 0) {
      tma_store_4d(maps + tp.s, ks, 0, tp.row, 0, m0 + l);
      tma_store_4d(maps + g.b + tp.s, ks + slot, 0, tp.row, 0, m0 + l);
      app_bulk_commit();
      if (write_meta && l == 0) {
        buf.pos[st.off[tp.s] + tp.row] = tp.pos;
        buf.orig[st.off[tp.s] + tp.row] = tp.orig;
      }
    }
  }
  if (lane == 0) {
    if (k < n_my + kAppLag) {
      // gave up waiting: let the copies still in flight land (bounded) before the slots go away
      for (int64_t x = (k - kAppLag > 0 ? k - kAppLag : 0); x < loaded; ++x)
        (void)mbar_wait_bounded(&full[x % kAppStages], (uint32_t)(x / kAppStages) & 1, limit_ns);
    }
    app_bulk_wait_all();  // every tensor store has completed
  }
}

// Resident one-warp CTAs of append_tma_kernel per SM for `smem` bytes of dynamic shared memory on
// the current device; the opt-in to that size is made per device as needed.
template <typename T, int D>
cudaError_t append_tma_occupancy(size_t smem, int* occ_out) {
  struct Seen {
    size_t smem;
    int occ;
  };
  static std::mutex mu;
  static size_t opted[64] = {};
  static std::vector<Seen> seen[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  for (const Seen& x : seen[dev])
    if (x.smem == smem) {
      *occ_out = x.occ;
      return cudaSuccess;
    }
  if (smem > opted[dev]) {
    e = cudaFuncSetAttribute(append_tma_kernel<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    opted[dev] = smem;
  }
  int o = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, append_tma_kernel<T, D>, 32, smem);
  if (e != cudaSuccess) return e;
  if (o < 1) o = 1;
  seen[dev].push_back({smem, o});
  *occ_out = o;
  return cudaSuccess;
}

// ---------------------------------------------------------------------------------------------
// a3: keep flags + scan (one CTA per affected sequence)
// ---------------------------------------------------------------------------------------------
constexpr int kScanThreads = 1024;
constexpr int kMaxSmemRanges = 1024;

__device__ __forceinline__ bool in_ranges(int32_t o, const int2* rg, int nr) {
  int a = 0, z = nr;  // first range with lo > o
  while (a < z) {
    const int mid = (a + z) >> 1;
    if (rg[mid].x <= o)
      a = mid + 1;
    else
      z = mid;
  }
  return a > 0 && o < rg[a - 1].y;
}

__global__ void __launch_bounds__(kScanThreads) compact_scan_kernel(Static st, Buffers buf,
                                                                    const AffSeq* __restrict__ aff,
                                                                    const int2* __restrict__ ranges,
                                                                    int32_t* __restrict__ src_map) {
  __shared__ int2 srg[kMaxSmemRanges];
  __shared__ int wsum[32];
  __shared__ int total;
  pdl_launch_dependents();  // the row-move kernel may be scheduled; it waits for this grid's results
  const AffSeq a = aff[blockIdx.x];
  const int64_t off = st.off[a.s];
  int32_t* pos = buf.pos + off;
  int32_t* orig = buf.orig + off;
  int32_t* smap = src_map + off;  // smap[dst] = source row of the row that lands at dst
  const int nr = a.n_ranges;
  const int2* rg = ranges + a.range_off;
  if (nr <= kMaxSmemRanges) {
    for (int i = threadIdx.x; i < nr; i += blockDim.x) srg[i] = rg[i];
    rg = srg;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int base = a.first_row;  // new index of the next kept row
  for (int c0 = a.first_row; c0 < a.len_old; c0 += kScanThreads) {
    const int i = c0 + threadIdx.x;
    const bool valid = i < a.len_old;
    int32_t o = 0, p = 0;
    bool keep = false;
    if (valid) {
      o = orig[i];
      p = pos[i];
      keep = !in_ranges(o, rg, nr);
    }
    const unsigned bal = __ballot_sync(kFull, keep);
    const int pre = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) wsum[warp] = __popc(bal);
    __syncthreads();  // also orders every read of this chunk before the writes below
    if (warp == 0) {
      const int v = wsum[lane];
      int incl = v;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int u = __shfl_up_sync(kFull, incl, d);
        if (lane >= d) incl += u;
      }
      wsum[lane] = incl - v;
      if (lane == 31) total = incl;
    }
    __syncthreads();
    const int dst = base + wsum[warp] + pre;
    if (keep) {  // dst <= i: lands on rows already read (this chunk, after the barrier) or earlier chunks
      smap[dst] = i;
      orig[dst] = o;
      pos[dst] = p;
    }
    base += total;
    __syncthreads();
  }
  if (threadIdx.x == 0 && base != a.len_new) atomicOr(buf.status, STATUS_CHECK);
}

// ---------------------------------------------------------------------------------------------
// a4: row moves.  One CTA owns one (sequence, layer, K/V, head) stream and walks its DESTINATION
// rows upward in chunks of 128, so every chunk moves 128 full rows however sparse the kept rows
// are.  A kept row only moves down (source >= destination): the stores of chunk k land below every
// source of chunk k+1, so chunk k+1's loads are issued before chunk k's stores, and a barrier
// separates each chunk's loads from its own stores.
// ---------------------------------------------------------------------------------------------
constexpr int kMoveThreads = 256;
constexpr int kMoveRows = 128;

template <int D>
__global__ void __launch_bounds__(kMoveThreads) compact_move_kernel(Geometry g, Static st, Buffers buf,
                                                                    const AffSeq* __restrict__ aff,
                                                                    const int32_t* __restrict__ src_map) {
  constexpr int VPR = D / 8;                                  // 16-byte vectors per row
  constexpr int U = kMoveRows * VPR / kMoveThreads;           // vectors per thread per chunk
  static_assert(kMoveRows * VPR % kMoveThreads == 0, "chunk must split evenly");
  pdl_wait();  // the source map and the plan come from the scan kernel
  const int streams = g.M * 2 * g.H;
  const int ai = blockIdx.x / streams;
  const int sidx = blockIdx.x % streams;
  const int h = sidx % g.H;
  const int kv = (sidx / g.H) & 1;
  const int m = sidx / (2 * g.H);
  const AffSeq a = aff[ai];
  uint16_t* plane = kv ? buf.v : buf.k;
  uint4* base = reinterpret_cast<uint4*>(
      plane + ((int64_t)m * g.H * g.C + st.seq_row0[a.s] + (int64_t)h * st.cap[a.s]) * D);
  const int32_t* smap = src_map + st.off[a.s];

  uint4 ra[U], rb[U];
  int da[U], db[U];
  auto load = [&](int d0, uint4* reg, int* dv) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int vi = threadIdx.x + u * kMoveThreads;
      const int row = d0 + vi / VPR;  // destination row
      const int col = vi % VPR;
      int d = -1;
      if (row < a.len_new) {
        const int src = __ldg(smap + row);
        reg[u] = base[(int64_t)src * VPR + col];
        d = row * VPR + col;
      }
      dv[u] = d;
    }
  };
  int d0 = a.first_row;
  if (d0 >= a.len_new) return;
  load(d0, ra, da);
  for (; d0 < a.len_new; d0 += kMoveRows) {
    const bool more = d0 + kMoveRows < a.len_new;
    if (more) load(d0 + kMoveRows, rb, db);
    __syncthreads();
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (da[u] >= 0) base[da[u]] = ra[u];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      ra[u] = rb[u];
      da[u] = more ? db[u] : -1;
    }
  }
}

// ---------------------------------------------------------------------------------------------
// a5 + a6: decode
// ---------------------------------------------------------------------------------------------
// Work split ("stream-K" over rows): the attended rows of every (sequence, head) segment are
// concatenated and cut into NW equal contiguous ranges, one per warp.  A warp is an independent
// flash-decoding worker: it streams its rows through its own ring of shared-memory stages (1-D TMA
// bulk copies issued by its lane 0, completion on an mbarrier), keeps an online softmax, and at
// the end of each piece (its part of one segment) either writes the output row (the whole segment
// was its own) or a partial (m, l, o); the last of a segment's workers to finish combines them.
//
// Lane geometry: LPR lanes share one row, lane t of a row holds NV 16-byte chunks.  Row group g
// (lane / LPR) reads chunk t*NV + (i + A*g + B*t) mod NV at step i: the rotation makes every
// 8-lane shared-memory wavefront hit 8 distinct bank groups; q is staged per lane in the same
// rotated order, and partial outputs are written back to their natural columns through shared
// memory, so the rotation never needs register indexing.
template <int D>
struct Lanes {
  static constexpr int RB = D * 2;                        // row bytes
  static constexpr int CH = D / 8;                        // 16-byte chunks per row
  static constexpr int LPR = (D == 96 || D == 128) ? 4 : 2;
  static constexpr int NV = CH / LPR;                     // chunks per lane
  static constexpr int EPL = NV * 8;                      // elements per lane
  static constexpr int RPI = 32 / LPR;                    // rows per warp step
  static constexpr int A = (D == 64 || D == 128) ? 1 : 0;
  static constexpr int B = (D == 128) ? 1 : 0;
  static_assert(D % 16 == 0 && CH % LPR == 0, "unsupported d_head");
};

// Shapes of the per-warp pipeline (rows per lane per tile x stages).  Whole segments want the
// largest in-flight window at three resident warps per SM, in as few tiles as possible (each tile
// costs a fixed share of a warp's issue): 8x2 (128-row tiles, 64 KB per warp) at d=64, 6x2 (96-row
// tiles, 60 KB) at d=80, 4x3 otherwise; measured on the full-size workloads against 4x3, 4x4 and
// 6x3.  The narrow 2x3 shape fits the most warps when one warp per segment needs them.  Stream-K
// runs a full wave of warps: 2x2 fits the most warps per SM.
template <int D>
struct WideShape {
  static constexpr int KPT = D == 64 ? 8 : D == 80 ? 6 : 4;
  static constexpr int S = (D == 64 || D == 80) ? 2 : 3;
};
#ifndef KVC_DEC_SEG2_KPT
#define KVC_DEC_SEG2_KPT 2
#endif
#ifndef KVC_DEC_SEG2_STAGES
#define KVC_DEC_SEG2_STAGES 3
#endif
#ifndef KVC_DEC_STREAM_KPT
#define KVC_DEC_STREAM_KPT 2
#endif
#ifndef KVC_DEC_STREAM_STAGES
#define KVC_DEC_STREAM_STAGES 2
#endif
template <int D, int KPT_, int S_>
struct DecodeCfg {
  using L = Lanes<D>;
  static constexpr int KPT = KPT_;              // rows per lane per tile
  static constexpr int TR = KPT * L::RPI;       // rows per tile
  static constexpr int TILE = TR * L::RB;       // bytes per K (or V) tile
  static constexpr int S = S_;                  // stages per warp
  static constexpr int WARPS = 1;               // warps per CTA
  static constexpr int THREADS = WARPS * 32;
  static constexpr int WARP_SMEM = (2 * S * TILE + D * 4 + S * 8 + 127) / 128 * 128;
  static constexpr int SMEM = WARPS * WARP_SMEM;
  static_assert(L::RPI * D * 4 <= 2 * TILE, "reduction scratch must fit in one stage");
};

struct DecodeDev {
  const uint16_t* k;  // plane of the launch's first layer
  const uint16_t* v;
  const DState* ds;
  const int64_t* P;
  int64_t R;          // rows of one layer (H * P[b])
  int NW;  // workers (warps)
  int n_layers;       // layers of this launch; layer i's segments follow layer i-1's
  int64_t plane;      // elements between consecutive layers' K (or V) planes
  int64_t q_stride;   // elements between consecutive layers' queries
  int64_t out_stride; // floats between consecutive layers' outputs
  const uint16_t* q;
  float* out;
  float* partials;
  int* counters;
  int* status;
  float qscale;  // scale * log2(e)
  unsigned long long limit_ns;
  int kv_before_wait;  // the K/V rows may be streamed before the preceding grid completes
  // k > 0: worker w owns segments [w k, w k + k) whole; -1: worker w owns the whole segments whose
  // first row lies in its even share of the rows; 0: stream-K split of the rows
  int seg_per_worker;
};

// The tiles of a worker: its flat row range [x, hi) of the concatenation over (layer, sequence,
// head) segments, cut into tiles of at most TR rows that never cross a segment.
struct TileIter {
  int64_t x, hi, Lc, r;
  int s, h, layer;
  __device__ __forceinline__ bool done() const { return x >= hi; }
  // rows of the next tile: at most TR, never past the segment, the range, or a ring's end (wrap)
  __device__ __forceinline__ int n(int TR, int64_t wrap) const {
    int64_t k = Lc - r;
    if (hi - x < k) k = hi - x;
    if (r < wrap && wrap - r < k) k = wrap - r;
    return (int)(k < TR ? k : TR);
  }
  // x < hi guarantees a later segment with rows, in this layer or a later one of the launch
  __device__ __forceinline__ void advance(int n, const int64_t* P, int H, int b) {
    x += n;
    r += n;
    if (r == Lc && x < hi) {
      r = 0;
      if (++h == H) {
        h = 0;
        do {
          if (++s == b) {
            s = 0;
            ++layer;
          }
        } while (P[s + 1] == P[s]);
        Lc = P[s + 1] - P[s];
      }
    }
  }
};

__device__ __forceinline__ int worker_of(int64_t x, int64_t R, int NW) { return (int)(((x + 1) * NW - 1) / R); }

// The sequence holding flat row o of a layer (0 <= o < H P[b]): the largest s < b with H P[s] <= o,
// which is a sequence with rows.  A 32-ary search by the whole warp: each round probes 32 evenly
// spaced candidates with one load per lane and keeps the interval after the last one that holds.
__device__ __forceinline__ int seq_of_row(const int64_t* P, int b, int H, int64_t o, int lane) {
  int a = 0, z = b;  // the answer lies in [a, z)
  while (z - a > 1) {
    const int step = (z - a + 31) / 32;
    const int k = a + lane * step;
    const bool le = k < z && (int64_t)H * P[k] <= o;
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, le);
    const int j = 31 - __clz(bal);  // bal != 0: candidate a always holds
    a = a + j * step;
    z = min(z, a + step);
  }
  return a;
}



__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) { return __fmul2_rn(a, b); }

template <typename T, int D, int KPT, int S>
__global__ void __launch_bounds__(32, 1) decode_kernel(Geometry g, Static st, DecodeDev p) {
  using C = DecodeCfg<D, KPT, S>;
  using L = Lanes<D>;
  extern __shared__ __align__(128) unsigned char smem[];
  // The next layer's decode may be scheduled now: its CTAs become resident only as ours retire.
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wid = blockIdx.x * C::WARPS + warp;
  if (wid >= p.NW) {
    pdl_wait();
    return;
  }
  const int H = g.H;
  const int64_t segs_layer = (int64_t)g.b * H;
  int64_t lo, hi;
  if (p.seg_per_worker > 0) {  // segments [sg0, sg1) = (layer, s, h) triples in order, each whole
    // first flat row of segment sg (sg = n_layers * b * H gives the end of the last layer)
    auto seg_row = [&](int64_t sg) {
      const int64_t l = sg / segs_layer, w = sg - l * segs_layer;
      const int s = (int)(w / H);
      const int64_t a = p.P[s], z = p.P[s + 1];
      return l * p.R + (int64_t)H * a + (w - (int64_t)s * H) * (z - a);
    };
    const int64_t sg0 = (int64_t)wid * p.seg_per_worker;
    const int64_t sg1 = min(sg0 + p.seg_per_worker, (int64_t)p.n_layers * segs_layer);
    lo = seg_row(sg0);
    hi = seg_row(sg1);
  } else if (p.seg_per_worker < 0) {
    // whole segments cut by rows: a segment belongs to the worker whose even share of the flat rows
    // [w Rt / NW, (w + 1) Rt / NW) holds its first row, so no segment is split and every worker's
    // rows are within one segment of the even share
    const int64_t Rt = (int64_t)p.n_layers * p.R;
    auto seg_at_or_after = [&](int64_t x) {  // first row of the first segment starting at or after x
      if (x >= Rt) return Rt;
      const int64_t l = x / p.R, o = x - l * p.R;
      const int s = seq_of_row(p.P, g.b, H, o, lane);
      const int64_t a = p.P[s], Lc = p.P[s + 1] - a;
      const int64_t off = o - (int64_t)H * a;
      const int64_t h = off / Lc;
      const int64_t start = l * p.R + (int64_t)H * a + h * Lc;
      return start == x ? start : start + Lc;
    };
    lo = seg_at_or_after((int64_t)wid * Rt / p.NW);
    hi = seg_at_or_after((int64_t)(wid + 1) * Rt / p.NW);
  } else {
    const int64_t Rt = (int64_t)p.n_layers * p.R;
    lo = (int64_t)wid * Rt / p.NW;
    hi = (int64_t)(wid + 1) * Rt / p.NW;
  }
  if (lo >= hi) {
    pdl_wait();
    return;
  }

  unsigned char* base = smem + warp * C::WARP_SMEM;
  unsigned char* stg = base;  // [S][K tile | V tile]
  float* qs = reinterpret_cast<float*>(base + 2 * C::S * C::TILE);  // [D]
  uint64_t* full = reinterpret_cast<uint64_t*>(qs + D);             // [S]

  // stale rows past a tile's end are multiplied by p = 0: start from zeros, never NaN
  for (int i = lane; i < 2 * C::S * C::TILE / 16; i += 32) reinterpret_cast<uint4*>(base)[i] = make_uint4(0, 0, 0, 0);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < C::S; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  fence_proxy_async_smem();
  __syncwarp();

  // the segment holding row `lo`: its layer, then the sequence with rows that holds the offset
  TileIter ci;  // consumed tiles
  ci.layer = (int)(lo / p.R);
  const int64_t o_layer = lo - (int64_t)ci.layer * p.R;
  ci.s = seq_of_row(p.P, g.b, H, o_layer, lane);
  // everything that depends only on the starting sequence, loaded together
  const int64_t P0 = p.P[ci.s], P1 = p.P[ci.s + 1];
  const DState ds0 = p.ds[ci.s];
  int64_t seg_row0 = st.seq_row0[ci.s];  // issue side: row 0 of (s, h = 0)
  int64_t seg_begin = ds0.begin, seg_wrap = ds0.wrap;
  int seg_cap = st.cap[ci.s];
  ci.Lc = P1 - P0;
  {
    const int64_t o = o_layer - (int64_t)H * P0;
    ci.h = (int)(o / ci.Lc);
    ci.r = o - (int64_t)ci.h * ci.Lc;
  }
  ci.x = lo;
  ci.hi = hi;
  TileIter ii = ci;  // issued tiles (lane 0 uses it)
  int seg_s = ci.s;

  auto issue = [&](int stage) {
    if (ii.s != seg_s) {
      seg_s = ii.s;
      const DState d = p.ds[seg_s];
      seg_row0 = st.seq_row0[seg_s];
      seg_begin = d.begin;
      seg_wrap = d.wrap;
      seg_cap = st.cap[seg_s];
    }
    const int n = ii.n(C::TR, seg_wrap);
    const int64_t slot = ii.r < seg_wrap ? seg_begin + ii.r : ii.r - seg_wrap;
    const int64_t row = seg_row0 + (int64_t)ii.h * seg_cap + slot;
    const uint32_t bytes = (uint32_t)n * L::RB;
    mbar_arrive_expect_tx(&full[stage], 2 * bytes);
    const int64_t e0 = (int64_t)ii.layer * p.plane + row * D;
    bulk_g2s(stg + stage * 2 * C::TILE, p.k + e0, bytes, &full[stage]);
    bulk_g2s(stg + stage * 2 * C::TILE + C::TILE, p.v + e0, bytes, &full[stage]);
    ii.advance(n, p.P, H, g.b);
  };
  int issued = 0;
  // K/V of this layer are not written by the preceding decode: stream them before it completes
  if (p.kv_before_wait && lane == 0) {
    while (issued < C::S && !ii.done()) {
      issue(issued);
      ++issued;
    }
  }
  pdl_wait();  // q, out and the split-K scratch may be shared with the preceding grid
  if (lane == 0) {
    while (issued < C::S && !ii.done()) {
      issue(issued);
      ++issued;
    }
  }

  // raw q of the next piece (and its rotation partner), fetched when the current piece starts
  constexpr int QPL = (D + 31) / 32;
  float qa[QPL], qb[QPL];
  auto fetch_q = [&](int l_, int s_, int h_) {
    const uint16_t* qrow = p.q + (int64_t)l_ * p.q_stride + ((int64_t)s_ * H + h_) * D;
    const int half = g.rot / 2;
#pragma unroll
    for (int j = 0; j < QPL; ++j) {
      const int c = lane + 32 * j;
      qa[j] = 0.f;
      qb[j] = 0.f;
      if (c < D) {
        qa[j] = T::f1(qrow[c]);
        if (c < g.rot) qb[j] = T::f1(qrow[c < half ? c + half : c - half]);
      }
    }
  };
  fetch_q(ci.layer, ci.s, ci.h);
  DState dn = ds0;
  const int grp = lane / L::LPR;
  const int tl = lane % L::LPR;
  const int rot = (L::A * grp + L::B * tl) % L::NV;
  float2 qv[L::EPL / 2], o[L::EPL / 2];
  float m = -INFINITY, l = 0.f;
  int64_t mask_lo = ds0.mask_lo, mask_hi = ds0.mask_hi, begin = ds0.begin, wrap = ds0.wrap;
  int32_t qpos = ds0.qpos;
  int cur_s = ci.s;
  bool dead = false;
  bool piece_start = true, piece_whole = false;
  int t = 0;     // tiles consumed
  int t_ok = 0;  // tiles whose copies were seen complete
  while (!ci.done()) {
    const int s = ci.s, h = ci.h, layer = ci.layer;
    const int64_t r0 = ci.r;
    if (piece_start && s != cur_s) {  // the next sequence's state was prefetched with its q
      cur_s = s;
      mask_lo = dn.mask_lo;
      mask_hi = dn.mask_hi;
      begin = dn.begin;
      wrap = dn.wrap;
      qpos = dn.qpos;
    }
    const int n = ci.n(C::TR, wrap);
    const int stage = t % C::S;
    if (piece_start) {
      // stage q (rotated at the query position for RoPE, pre-scaled by scale*log2 e) in natural order
      const int half = g.rot / 2;
#pragma unroll
      for (int j = 0; j < QPL; ++j) {
        const int c = lane + 32 * j;
        if (c < D) {
          float x = qa[j];
          if (c < g.rot) {
            const bool lo_half = c < half;
            float sn, cs;
            rope_sincos(qpos, st.rope_g[lo_half ? c : c - half], &sn, &cs);
            x = lo_half ? x * cs - qb[j] * sn : x * cs + qb[j] * sn;
          }
          qs[c] = x * p.qscale;
        }
      }
      __syncwarp();
#pragma unroll
      for (int i = 0; i < L::NV; ++i) {
        const int c = tl * L::NV + (i + rot) % L::NV;
        const float4 a = reinterpret_cast<const float4*>(qs + c * 8)[0];
        const float4 b = reinterpret_cast<const float4*>(qs + c * 8)[1];
        qv[i * 4 + 0] = make_float2(a.x, a.y);
        qv[i * 4 + 1] = make_float2(a.z, a.w);
        qv[i * 4 + 2] = make_float2(b.x, b.y);
        qv[i * 4 + 3] = make_float2(b.z, b.w);
      }
#pragma unroll
      for (int e = 0; e < L::EPL / 2; ++e) o[e] = make_float2(0.f, 0.f);
      m = -INFINITY;
      l = 0.f;
      piece_whole = (r0 == 0);
      piece_start = false;
      // the next piece's q and sequence state, fetched a whole piece ahead of their use: with short
      // segments one tile of lead does not cover a global load's latency under full memory traffic
      const int64_t rest = ci.Lc - r0;  // rows of this segment from here on
      if (ci.x + rest < ci.hi) {
        TileIter nx = ci;
        nx.advance(rest, p.P, H, g.b);
        fetch_q(nx.layer, nx.s, nx.h);
        if (nx.s != s) dn = p.ds[nx.s];
      }
    }
    if (!dead) {
      if (mbar_wait_bounded(&full[stage], (t / C::S) & 1, p.limit_ns)) {
        t_ok = t + 1;
      } else {
        dead = true;
        if (lane == 0) atomicOr(p.status, STATUS_TIMEOUT);
      }
    }
    const unsigned char* kt = stg + stage * 2 * C::TILE;
    const unsigned char* vt = kt + C::TILE;
    if (!dead) {
      // tile-local bounds of the hidden rows
      const int64_t row0 = begin + r0;
      int hlo = (int)max((int64_t)0, min((int64_t)C::TR, mask_lo - row0));
      int hhi = (int)max((int64_t)0, min((int64_t)C::TR, mask_hi - row0));
      float z[C::KPT];
#pragma unroll
      for (int k = 0; k < C::KPT; ++k) {
        const int j = k * L::RPI + grp;
        const unsigned char* rowp = kt + j * L::RB;
        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < L::NV; ++i) {
          const int c = tl * L::NV + (i + rot) % L::NV;
          const uint4 u = *reinterpret_cast<const uint4*>(rowp + c * 16);
          acc0 = ffma2(qv[i * 4 + 0], T::f2(u.x), acc0);
          acc1 = ffma2(qv[i * 4 + 1], T::f2(u.y), acc1);
          acc0 = ffma2(qv[i * 4 + 2], T::f2(u.z), acc0);
          acc1 = ffma2(qv[i * 4 + 3], T::f2(u.w), acc1);
        }
        float zz = (acc0.x + acc1.x) + (acc0.y + acc1.y);
#pragma unroll
        for (int off = L::LPR / 2; off >= 1; off >>= 1) zz += __shfl_xor_sync(kFull, zz, off);
        const bool valid = j < n && (j < hlo || j >= hhi);
        z[k] = valid ? zz : -INFINITY;
      }
      float mt = z[0];
#pragma unroll
      for (int k = 1; k < C::KPT; ++k) mt = fmaxf(mt, z[k]);
      const float mn = fmaxf(m, mt);
      const float mu = (mn == -INFINITY) ? 0.f : mn;  // every z so far is -inf: keep p = 0, alpha = 0
      const float alpha = exp2f(m - mu);
      l *= alpha;
      const float2 a2 = make_float2(alpha, alpha);
#pragma unroll
      for (int e = 0; e < L::EPL / 2; ++e) o[e] = fmul2(o[e], a2);
#pragma unroll
      for (int k = 0; k < C::KPT; ++k) {
        const int j = k * L::RPI + grp;
        const float pk = exp2f(z[k] - mu);
        l += pk;
        const float2 p2 = make_float2(pk, pk);
        const unsigned char* rowp = vt + j * L::RB;
#pragma unroll
        for (int i = 0; i < L::NV; ++i) {
          const int c = tl * L::NV + (i + rot) % L::NV;
          const uint4 u = *reinterpret_cast<const uint4*>(rowp + c * 16);
          o[i * 4 + 0] = ffma2(p2, T::f2(u.x), o[i * 4 + 0]);
          o[i * 4 + 1] = ffma2(p2, T::f2(u.y), o[i * 4 + 1]);
          o[i * 4 + 2] = ffma2(p2, T::f2(u.z), o[i * 4 + 2]);
          o[i * 4 + 3] = ffma2(p2, T::f2(u.w), o[i * 4 + 3]);
        }
      }
      m = mn;
    }
    __syncwarp();
    const bool seg_done = (r0 + n == ci.Lc);
    ci.advance(n, p.P, H, g.b);
    ++t;
    bool refilled = false;
    if (seg_done || ci.done()) {
      // ------------------------- piece end: merge the row groups -------------------------
      float M = m;
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, off));
      const float Mu = (M == -INFINITY) ? 0.f : M;
      const float e = exp2f(m - Mu);
      float Ls = l * e;
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) Ls += __shfl_xor_sync(kFull, Ls, off);
      Ls *= 1.0f / (float)L::LPR;  // each row group's l is held by its LPR lanes
      // scratch: the stage just consumed (its next copies are issued below)
      float* red = reinterpret_cast<float*>(stg + stage * 2 * C::TILE);  // [RPI][D]
      const float2 e2 = make_float2(e, e);
#pragma unroll
      for (int i = 0; i < L::NV; ++i) {
        const int c = tl * L::NV + (i + rot) % L::NV;
        float4* dst = reinterpret_cast<float4*>(red + grp * D + c * 8);
        const float2 x0 = fmul2(o[i * 4 + 0], e2), x1 = fmul2(o[i * 4 + 1], e2);
        const float2 x2 = fmul2(o[i * 4 + 2], e2), x3 = fmul2(o[i * 4 + 3], e2);
        dst[0] = make_float4(x0.x, x0.y, x1.x, x1.y);
        dst[1] = make_float4(x2.x, x2.y, x3.x, x3.y);
      }
      __syncwarp();
      const int seg = s * H + h;
      if (!dead) {
        if (piece_whole && seg_done) {
          const float inv = 1.f / Ls;
          float* orow = p.out + (int64_t)layer * p.out_stride + (int64_t)seg * D;
          for (int col = lane; col < D; col += 32) {
            float O = 0.f;
#pragma unroll
            for (int r = 0; r < L::RPI; ++r) O += red[r * D + col];
            orow[col] = O * inv;
          }
        } else if (p.n_layers > 1) {
          // launches over several layers take whole segments only (the host plans no split)
          if (lane == 0) atomicOr(p.status, STATUS_CHECK);
        } else {
          float* pp = p.partials + (int64_t)(wid + seg) * (D + 4);
          for (int col = lane; col < D; col += 32) {
            float O = 0.f;
#pragma unroll
            for (int r = 0; r < L::RPI; ++r) O += red[r * D + col];
            pp[4 + col] = O;
          }
          if (lane == 0) {
            pp[0] = M;
            pp[1] = Ls;
          }
          // the stage is read: refill it before the fence and the arrival, which wait on memory
          __syncwarp();
          if (lane == 0 && !ii.done()) {
            fence_proxy_async_smem();
            issue(stage);
            ++issued;
          }
          refilled = true;
          __threadfence();
          __syncwarp();
          const int64_t Lc = p.P[s + 1] - p.P[s];
          const int64_t A = (int64_t)H * p.P[s] + (int64_t)h * Lc;
          const int w_first = worker_of(A, p.R, p.NW);
          const int w_last = worker_of(A + Lc - 1, p.R, p.NW);
          int last = 0;
          if (lane == 0) last = atomicAdd(&p.counters[seg], 1) == (w_last - w_first);
          last = __shfl_sync(kFull, last, 0);
          if (last) {
            __threadfence();
            // lane k holds part w_first + k (parts of one segment are few; loop for more than 32)
            const int np = w_last - w_first + 1;
            float Mx = -INFINITY;
            for (int k = lane; k < np; k += 32) Mx = fmaxf(Mx, __ldcg(p.partials + (int64_t)(w_first + k + seg) * (D + 4)));
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) Mx = fmaxf(Mx, __shfl_xor_sync(kFull, Mx, off));
            const float Mxu = (Mx == -INFINITY) ? 0.f : Mx;
            float Lx = 0.f;
            for (int k = lane; k < np; k += 32) {
              const float* q = p.partials + (int64_t)(w_first + k + seg) * (D + 4);
              Lx += __ldcg(q + 1) * exp2f(__ldcg(q) - Mxu);
            }
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) Lx += __shfl_xor_sync(kFull, Lx, off);
            const float inv = 1.f / Lx;
            for (int col = lane; col < D; col += 32) {
              float O = 0.f;
              for (int k = 0; k < np; ++k) {
                const float* q = p.partials + (int64_t)(w_first + k + seg) * (D + 4);
                O += __ldcg(q + 4 + col) * exp2f(__ldcg(q) - Mxu);
              }
              p.out[(int64_t)seg * D + col] = O * inv;
            }
            if (lane == 0) p.counters[seg] = 0;
          }
        }
      }
      __syncwarp();
      piece_start = true;
    }
    // refill the stage just consumed
    if (lane == 0 && !dead && !refilled && !ii.done()) {
      fence_proxy_async_smem();
      issue(stage);
      ++issued;
    }
  }
  // never leave with copies in flight into this warp's shared memory (only after a timed-out wait)
  if (lane == 0) {
    for (int u = t_ok; u < issued; ++u) mbar_wait_bounded(&full[u % C::S], (u / C::S) & 1, p.limit_ns);
  }
  __syncwarp();
}

// ---------------------------------------------------------------------------------------------
// dispatch
// ---------------------------------------------------------------------------------------------
// Resident CTAs per SM of one kernel instance, per device (the shared-memory attribute is set on
// each device the first time the instance runs there).
template <typename T, int D, int KPT, int S>
cudaError_t decode_occupancy(int* occ_out) {
  using C = DecodeCfg<D, KPT, S>;
  static std::mutex mu;
  static int occ[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (occ[dev] == 0) {
    e = cudaFuncSetAttribute(decode_kernel<T, D, KPT, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    int o = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, decode_kernel<T, D, KPT, S>, C::THREADS, C::SMEM);
    if (e != cudaSuccess) return e;
    occ[dev] = o < 1 ? 1 : o;
  }
  *occ_out = occ[dev];
  return cudaSuccess;
}

template <typename T, int D, int KPT, int S>
cudaError_t launch_decode_cfg(const Geometry& g, const Static& st, const Buffers& buf, const DecodeArgs& a,
                              int64_t NW, int seg_per_worker, cudaStream_t stream, int* grid) {
  using C = DecodeCfg<D, KPT, S>;
  DecodeDev p;
  const int64_t plane = (int64_t)g.H * g.C * D;
  p.k = buf.k + (int64_t)a.layer * plane;
  p.v = buf.v + (int64_t)a.layer * plane;
  p.ds = a.dstate;
  p.P = a.P;
  p.R = a.R;
  p.NW = (int)NW;
  p.n_layers = a.n_layers < 1 ? 1 : a.n_layers;
  p.plane = plane;
  p.q_stride = a.q_layer_stride;
  p.out_stride = a.out_layer_stride;
  p.q = static_cast<const uint16_t*>(a.q);
  p.out = a.out;
  p.partials = a.partials;
  p.counters = a.counters;
  p.status = buf.status;
  p.qscale = a.scale * 1.4426950408889634f;
  p.limit_ns = a.wait_limit_ns;
  p.kv_before_wait = a.kv_before_wait;
  p.seg_per_worker = seg_per_worker;
  const int64_t ctas = (NW + C::WARPS - 1) / C::WARPS;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)ctas);
  cfg.blockDim = dim3(C::THREADS);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  *grid = (int)ctas;
  return cudaLaunchKernelEx(&cfg, decode_kernel<T, D, KPT, S>, g, st, p);
}

// k whole segments per worker, k as small as one wave of `occ` warps per SM allows; `busiest` is
// the segments on the SM with the most resident workers (workers spread evenly over the SMs).
struct SegSplit {
  int64_t k, workers, busiest;
};
inline SegSplit seg_split(int64_t nseg, int occ, int num_sms) {
  const int64_t slots = (int64_t)(occ > 0 ? occ : 1) * num_sms;
  const int64_t k = (nseg + slots - 1) / slots;
  const int64_t workers = (nseg + k - 1) / k;
  return {k, workers, (workers + num_sms - 1) / num_sms * k};
}

// Segments of the uploaded state are balanced: the longest holds at most 1.3x the mean rows.
inline bool decode_balanced(const DecodeArgs& a) {
  return a.n_segments > 0 && 10 * a.max_segment * a.n_segments <= 13 * a.R;
}

template <typename T, int D>
cudaError_t launch_decode_t(const Geometry& g, const Static& st, const Buffers& buf, const DecodeArgs& a, int num_sms,
                            cudaStream_t stream, int* grid, DecodePlan* plan) {
  constexpr int AK = WideShape<D>::KPT, AS = WideShape<D>::S;
  constexpr int BK = KVC_DEC_SEG2_KPT, BS = KVC_DEC_SEG2_STAGES;
  constexpr int TK = KVC_DEC_STREAM_KPT, TS = KVC_DEC_STREAM_STAGES;
  // Balanced segments (longest within 1.3x of the mean) are never split, so no warp writes split-K
  // partials or waits on a combine: one warp per (layer, sequence, head) segment when a wave of
  // resident warps holds them all (the wide pipeline shape first), else k consecutive whole
  // segments per warp.  Otherwise, over several layers whose segments are short beside a warp's
  // share of the rows, whole segments cut by rows; else the rows are split evenly over a full wave
  // (stream-K), one layer per launch.  Whole segments shorter on average than six wide tiles go to
  // the narrow shape (more warps per SM, less fixed work per tile and per segment): on ragged caches
  // the wide shape wins from a mean of about 1,000 kept rows, the narrow one below about 500.
  const int n_layers = a.n_layers < 1 ? 1 : a.n_layers;
  const int64_t nseg = (int64_t)n_layers * g.b * g.H;
  const bool short_segs = a.n_segments > 0 && a.R < 6 * (int64_t)(AK * Lanes<D>::RPI) * a.n_segments;
  const bool balanced = decode_balanced(a);
  if (balanced || n_layers > 1) {
    cudaError_t e;
    int occ_a = 0, occ_b = 0;
    e = decode_occupancy<T, D, AK, AS>(&occ_a);
    if (e == cudaSuccess) e = decode_occupancy<T, D, BK, BS>(&occ_b);
    if (e != cudaSuccess) return e;
    if (!balanced) {
      // Unbalanced segments over several layers: a wave of warps takes whole segments cut by rows
      // when the longest segment is at most 1/16 of a warp's even share (so no warp holds more than
      // ~6 % above the mean); else the caller launches the layers one by one.
      const int occ = short_segs ? occ_b : occ_a;
      int64_t NW = (int64_t)occ * num_sms;
      if (NW > nseg) NW = nseg;
      if (NW < 1 || 16 * a.max_segment > (int64_t)n_layers * a.R / NW) return cudaErrorNotSupported;
      if (short_segs) {
        *plan = {4, (int)NW, BK * Lanes<D>::RPI, BS};
        return launch_decode_cfg<T, D, BK, BS>(g, st, buf, a, NW, -1, stream, grid);
      }
      *plan = {4, (int)NW, AK * Lanes<D>::RPI, AS};
      return launch_decode_cfg<T, D, AK, AS>(g, st, buf, a, NW, -1, stream, grid);
    }
    if (nseg <= (int64_t)occ_a * num_sms) {
      *plan = {1, (int)nseg, AK * Lanes<D>::RPI, AS};
      return launch_decode_cfg<T, D, AK, AS>(g, st, buf, a, nseg, 1, stream, grid);
    }
    if (nseg <= (int64_t)occ_b * num_sms) {
      *plan = {2, (int)nseg, BK * Lanes<D>::RPI, BS};
      return launch_decode_cfg<T, D, BK, BS>(g, st, buf, a, nseg, 1, stream, grid);
    }
    // several whole segments per warp: the narrow shape for short segments, else the shape and k that
    // put the fewest segments on the busiest SM
    const SegSplit sa = seg_split(nseg, occ_a, num_sms), sb = seg_split(nseg, occ_b, num_sms);
    if (!short_segs && sa.busiest <= sb.busiest) {
      *plan = {3, (int)sa.workers, AK * Lanes<D>::RPI, AS};
      return launch_decode_cfg<T, D, AK, AS>(g, st, buf, a, sa.workers, sa.k, stream, grid);
    }
    *plan = {3, (int)sb.workers, BK * Lanes<D>::RPI, BS};
    return launch_decode_cfg<T, D, BK, BS>(g, st, buf, a, sb.workers, sb.k, stream, grid);
  }
  cudaError_t e;
  int occ = 0;
  e = decode_occupancy<T, D, TK, TS>(&occ);
  if (e != cudaSuccess) return e;
  int64_t NW = (int64_t)occ * num_sms;
  if (a.R < NW) NW = a.R;
  if (NW > kMaxDecodeWorkers) NW = kMaxDecodeWorkers;
  if (NW < 1) NW = 1;
  *plan = {0, (int)NW, TK * Lanes<D>::RPI, TS};
  return launch_decode_cfg<T, D, TK, TS>(g, st, buf, a, NW, 0, stream, grid);
}

template <typename T, int D>
cudaError_t launch_append_t(const Geometry& g, const Static& st, const Buffers& buf, const TokPlan* plan, int64_t ntok,
                            int64_t n_in, int m0, int n_layers, bool write_meta, const void* k_in, const void* v_in,
                            const void* maps, int num_sms, unsigned long long limit_ns, cudaStream_t stream) {
  const int64_t n_units = (int64_t)n_layers * ntok;
  const size_t smem = app_smem_bytes(g.H, D, g.rot);
  if (maps != nullptr && num_sms > 0 && n_units >= num_sms && smem <= 200 * 1024) {
    // TMA ring workers, as many one-warp CTAs as fit (capped by the units)
    int occ = 0;
    const cudaError_t e = append_tma_occupancy<T, D>(smem, &occ);
    if (e != cudaSuccess) return e;
    int64_t grid = (int64_t)occ * num_sms;
    if (grid > n_units) grid = n_units;
    append_tma_kernel<T, D><<<(unsigned)grid, 32, smem, stream>>>(
        g, st, buf, plan, ntok, n_in, m0, n_layers, write_meta ? 1 : 0, static_cast<const uint16_t*>(k_in),
        static_cast<const uint16_t*>(v_in), static_cast<const CUtensorMap*>(maps), limit_ns);
    return cudaGetLastError();
  }
  // one (layer, token) unit per block at a time; enough blocks for every SM several times over
  int64_t blocks = n_units;
  if (blocks > kAppendMaxBlocks) blocks = kAppendMaxBlocks;
  if (blocks < 1) blocks = 1;
  append_kernel<T, D><<<(unsigned)blocks, kAppendThreads, 0, stream>>>(g, st, buf, plan, ntok, n_in, m0, n_layers, write_meta ? 1 : 0,
                                                            static_cast<const uint16_t*>(k_in),
                                                            static_cast<const uint16_t*>(v_in));
  return cudaGetLastError();
}

template <typename F>
cudaError_t by_dhead(int D, F&& f) {
  switch (D) {
    case 64:
      return f(std::integral_constant<int, 64>{});
    case 80:
      return f(std::integral_constant<int, 80>{});
    case 96:
      return f(std::integral_constant<int, 96>{});
    case 128:
      return f(std::integral_constant<int, 128>{});
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace

bool dhead_supported(int D) { return D == 64 || D == 80 || D == 96 || D == 128; }

cudaError_t launch_append(const Geometry& g, const Static& st, const Buffers& buf, const TokPlan* plan, int64_t n_plan,
                          int64_t n_in, int m0, int n_layers, bool write_meta, const void* k_in, const void* v_in,
                          const void* maps, int num_sms, unsigned long long limit_ns, cudaStream_t stream) {
  return by_dhead(g.D, [&](auto dc) {
    constexpr int D = decltype(dc)::value;
    if (g.dtype == 1)
      return launch_append_t<BF16T, D>(g, st, buf, plan, n_plan, n_in, m0, n_layers, write_meta, k_in, v_in, maps,
                                       num_sms, limit_ns, stream);
    return launch_append_t<F16T, D>(g, st, buf, plan, n_plan, n_in, m0, n_layers, write_meta, k_in, v_in, maps,
                                    num_sms, limit_ns, stream);
  });
}

cudaError_t launch_compact(const Geometry& g, const Static& st, const Buffers& buf, const AffSeq* aff, int n_aff,
                           const int32_t* ranges, int32_t* src_map, cudaStream_t stream, int* launched,
                           cudaEvent_t between) {
  *launched = 0;
  if (n_aff <= 0) return cudaSuccess;
  compact_scan_kernel<<<n_aff, kScanThreads, 0, stream>>>(st, buf, aff, reinterpret_cast<const int2*>(ranges),
                                                         src_map);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  *launched = 1;
  if (between != nullptr) {
    e = cudaEventRecord(between, stream);
    if (e != cudaSuccess) return e;
  }
  const int64_t blocks = (int64_t)n_aff * g.M * 2 * g.H;
  e = by_dhead(g.D, [&](auto dc) {
    constexpr int D = decltype(dc)::value;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(kMoveThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, compact_move_kernel<D>, g, st, buf, aff, (const int32_t*)src_map);
  });
  if (e == cudaSuccess) *launched = 2;
  return e;
}

cudaError_t launch_decode(const Geometry& g, const Static& st, const Buffers& buf, const DecodeArgs& a, int num_sms,
                          cudaStream_t stream, int* grid, DecodePlan* plan) {
  *grid = 0;
  *plan = {-1, 0, 0, 0};
  if (a.R <= 0) return cudaSuccess;
  return by_dhead(g.D, [&](auto dc) {
    constexpr int D = decltype(dc)::value;
    if (g.dtype == 1) return launch_decode_t<BF16T, D>(g, st, buf, a, num_sms, stream, grid, plan);
    return launch_decode_t<F16T, D>(g, st, buf, a, num_sms, stream, grid, plan);
  });
}

// ---------------------------------------------------------------------------------------------
// Timeout path check: one warp waits, with the decode's bounded wait, on an mbarrier phase that
// nothing completes; when the limit runs out it records STATUS_TIMEOUT like a decode would.
// ---------------------------------------------------------------------------------------------
namespace {
__global__ void bounded_wait_check_kernel(int* status, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncwarp();
  if (!mbar_wait_bounded(&bar, 0, limit_ns) && threadIdx.x == 0) atomicOr(status, STATUS_TIMEOUT);
  __syncwarp();
}
}  // namespace

cudaError_t launch_bounded_wait_check(int* status, unsigned long long limit_ns, cudaStream_t stream) {
  bounded_wait_check_kernel<<<1, 32, 0, stream>>>(status, limit_ns);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// Split-K scratch without allocation.  Every GPU that loads this library holds the array until the
// process exits; all calls share it (kvc_decode_attention_static_scratch documents the contract).
// In host code `g_decode_static_scratch` names a host-side stand-in: only the address returned by
// cudaGetSymbolAddress may be handed to a kernel.
// ---------------------------------------------------------------------------------------------
__device__ __align__(256) unsigned char g_decode_static_scratch[kStaticDecodeScratchBytes];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_static_scratch_mu;
void* g_static_scratch_addr[kMaxDevices] = {};
}  // namespace

cudaError_t static_decode_scratch(void** ptr) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_static_scratch_mu);
  if (g_static_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_decode_static_scratch);
    if (e != cudaSuccess) return e;
    g_static_scratch_addr[dev] = p;
  }
  *ptr = g_static_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace kvc
