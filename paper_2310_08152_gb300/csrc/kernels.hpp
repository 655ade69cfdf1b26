// Internal interface between the host state (kvc.cpp) and the sm_103a kernels (kernels.cu).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace kvc {

// Per-sequence decode state, uploaded after every change of the span book.
// The decode query of sequence s reads stored rows [begin, len) except [mask_lo, mask_hi).  Row
// begin + r lives in slot begin + r while r < wrap and in slot r - wrap after it (a ring, for the
// local-attention cache; wrap is INT32_MAX otherwise).
struct DState {
  int32_t len, begin, mask_lo, mask_hi, qpos, wrap, pad1, pad2;
};

// One stored token: its sequence, destination row, position, history index, and its index among
// the input tokens of the call (tokens freed as they are written have no plan entry).
struct TokPlan {
  int32_t s, row, pos, orig, in_tok, pad0, pad1, pad2;
};

// One sequence of a compaction; its drop ranges (history indices, [lo, hi)) are
// ranges[range_off .. range_off + n_ranges).
struct AffSeq {
  int32_t s, len_old, len_new, first_row, range_off, n_ranges, pad0, pad1;
};

// Status word bits written by kernels.
enum : int { STATUS_TIMEOUT = 1, STATUS_CHECK = 2 };

struct Geometry {
  int M, H, D, b;
  int64_t C;  // sum of capacities (rows per (layer, K/V, head) plane)
  int dtype;  // 0 f16, 1 bf16
  int rot;    // rotary dims (0 = none)
};

struct Static {
  const int64_t* seq_row0;  // [b] H * off[s]
  const int32_t* cap;       // [b]
  const int64_t* off;       // [b]
  const float2* rope_g;     // [rot/2] theta_i / (2 pi) per position as a double-float (hi, lo)
};

struct Buffers {
  uint16_t* k;   // cache K base
  uint16_t* v;   // cache V base
  int32_t* pos;  // [C]
  int32_t* orig; // [C]
  int* status;
};

// Most decode workers (warps); sizes the split-K partial buffer.
constexpr int kMaxDecodeWorkers = 8192;

bool dhead_supported(int D);

// Writes the n_plan stored tokens of a call whose inputs hold n_in tokens per layer (k_in, v_in
// 16-byte aligned).  maps: the device copy of encode_append_maps' output, or NULL; with it, calls of
// at least num_sms (layer, token) units go through the TMA kernel, whose bounded waits give up
// after limit_ns.
cudaError_t launch_append(const Geometry& g, const Static& st, const Buffers& buf, const TokPlan* plan, int64_t n_plan,
                          int64_t n_in, int m0, int n_layers, bool write_meta, const void* k_in, const void* v_in,
                          const void* maps, int num_sms, unsigned long long limit_ns, cudaStream_t stream);
// Bytes of encode_append_maps' output: a 128-byte TMA descriptor per (K/V, sequence).
inline size_t append_maps_bytes(int b) { return 2 * 128 * (size_t)b; }
// Encodes, per sequence s, 4-D TMA descriptors over the K and then the V planes: dims {D, cap[s],
// H, M} from row seq_row0[s] of layer 0's plane, strides (D, cap[s] D, H C D) elements, box
// {D, 1, H, 1}: one (layer, token)'s rows of every head.  seq_row0 and cap are host arrays; out is
// host memory of append_maps_bytes(b).  cudaErrorNotSupported where a box cannot hold H heads.
cudaError_t encode_append_maps(const Geometry& g, const Buffers& buf, const int64_t* seq_row0, const int32_t* cap,
                               unsigned char* out);

// Scan, then row moves.  between: an event recorded on the stream between the two kernels, or NULL.
cudaError_t launch_compact(const Geometry& g, const Static& st, const Buffers& buf, const AffSeq* aff, int n_aff,
                           const int32_t* ranges, int32_t* src_map, cudaStream_t stream, int* launched,
                           cudaEvent_t between = nullptr);

struct DecodeArgs {
  int layer;             // the first layer of the launch
  int n_layers = 1;      // layers layer .. layer + n_layers - 1 in one launch (whole segments only)
  const DState* dstate;  // [b]
  const int64_t* P;      // [b+1] prefix sums of attended-range lengths (len - begin)
  int64_t R;             // H * P[b]
  const void* q;         // [b][H][D] per layer, layer i at q + i * q_layer_stride elements
  float* out;            // [b][H][D] per layer, layer i at out + i * out_layer_stride floats
  int64_t q_layer_stride = 0;
  int64_t out_layer_stride = 0;
  float scale;
  float* partials;       // [(kMaxDecodeWorkers + b*H) * (D + 4)]
  int* counters;         // [b*H], zero between launches
  unsigned long long wait_limit_ns;
  // 1 when the kernel launched before this one on the stream was a decode (which writes no K/V):
  // K/V tiles are then requested before that kernel has completed (programmatic dependent launch).
  int kv_before_wait;
  // segment statistics of the uploaded state: segments with rows, and the longest one
  int64_t n_segments;
  int64_t max_segment;
};

// How a decode launch split its work: mode 0 = stream-K over all rows, 1 / 2 = one warp per
// (layer, sequence, head) segment with the wide / narrow pipeline, 3 = several consecutive whole
// segments per warp, 4 = consecutive whole segments per warp cut by rows (unbalanced segments over
// several layers); workers = warps; tile rows; stages.
struct DecodePlan {
  int mode, workers, tile_rows, stages;
};

// Returns the grid used through *grid (0 if nothing launched) and the plan through *plan.  A launch
// over several layers (a.n_layers > 1) takes whole segments only: when the longest segment is too
// long beside a warp's share of the rows it launches nothing and returns cudaErrorNotSupported, and
// the caller goes layer by layer.
cudaError_t launch_decode(const Geometry& g, const Static& st, const Buffers& buf, const DecodeArgs& a,
                          int num_sms, cudaStream_t stream, int* grid, DecodePlan* plan);

// ---------------------------------------------------------------------------------------------
// Masked prefill attention (prefill.cu)
// ---------------------------------------------------------------------------------------------
// Per sequence: stored rows [0, len); the queries are stored rows [q0, len), the first of them is
// token qtok of the q / out arrays; the per-row mask bounds start at meta[moff].
struct PState {
  int32_t len, q0, qtok, moff;
};
// One prefill work item (sequence s, head h, query tile [qr0, qr_end)) as the host lays it out,
// in the kernel's order; row0 = seq_row0[s] + h * cap[s], the K/V plane row of stored row 0 in
// layer 0 (the kernel adds layer * H * C).
struct PfItemRec {
  PState ps;
  int32_t s, h, qr0, qr_end;
  int32_t nk, row0_lo, row0_hi, pad;
};
static_assert(sizeof(PfItemRec) == 48, "three 16-byte loads");

struct PrefillArgs {
  int layer, H, rot;
  int64_t C;
  const PfItemRec* items;  // [n_items]: sequences with the most stored rows first, then head, then the query tile with the most keys first
  int64_t n_items;         // (query tile, head) work items
  unsigned long long* item_counter;  // zero at launch: the CTAs take items [0, n_items) in order from it
  int n_ctas;              // persistent grid size
  const int32_t* meta;     // per stored row: (hid << 1) | is_cl
  const uint16_t* q;       // [sum n_q][H][D]
  float* out;              // [sum n_q][H][D]
  int64_t n_qtok;          // sum n_q
  float c2;                // scale * log2(e)
  const int32_t* pos;      // [C] stored-row positions
  const int64_t* off;      // [b]: a sequence's first entry in pos
  const float2* rope_g;    // [rot/2]
  int* status;
  unsigned long long wait_limit_ns;
};

// Encoded 2-D TMA descriptors of the K and V planes ([M*H*C rows][D], swizzled column subtiles).
struct alignas(64) PrefillMaps {
  unsigned char k[128];
  unsigned char v[128];
  bool ready = false;
};

cudaError_t encode_prefill_maps(const Geometry& g, const Buffers& buf, PrefillMaps* maps);
// Most CTAs of the persistent prefill grid (sizes its work-range table).
constexpr int kMaxPrefillCtas = 1024;
// CTAs of the prefill kernel that fit on one SM for head dimension D (sizes the persistent grid).
int prefill_ctas_per_sm(int D);
// A persistent grid of a.n_ctas CTAs walks the a.n_items work items.
cudaError_t launch_prefill(const Geometry& g, const PrefillMaps& maps, const PrefillArgs& a, cudaStream_t stream);

// One warp waits on an mbarrier phase that never completes, with the limit given; the bounded wait
// gives up and sets STATUS_TIMEOUT in *status.  Exercises the kernels' timeout reporting.
cudaError_t launch_bounded_wait_check(int* status, unsigned long long limit_ns, cudaStream_t stream);

// Split-K scratch in a file-scope device array (kernels.cu), for callers that cannot allocate
// device memory.  *ptr gets its device address on the current device; the address is looked up
// with cudaGetSymbolAddress the first time a device asks for it.
constexpr size_t kStaticDecodeScratchBytes = size_t(8) << 20;
cudaError_t static_decode_scratch(void** ptr);

}  // namespace kvc
