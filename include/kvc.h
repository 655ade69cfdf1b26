/*
 * kvc.h -- C ABI of the sentinel-compressed KV cache for GB300 (sm_103a).
 *
 * The method (Ren et al., "Context Compression for Auto-regressive
 * Transformers with Sentinel Tokens", EMNLP 2023) brackets spans of tokens
 * with the sentinels <CL> ... <CR>.  Under its modified causal mask (Sec. 1,
 * Sec. 3.1 and the Fig. 1 caption) a <CL> attends only to itself, other tokens
 * attend to earlier <CR> and normal tokens, and no token after a <CR> attends
 * to the tokens between that span's <CL> and <CR>.  The key-value memory of
 * the enclosed tokens can therefore be freed (Sec. 3.1, "Manipulating
 * Key-Value Memory for Inference-time Compression"), which shrinks the cache
 * of shape (M, 2, b, H, L, d_head) that decoding reads (Sec. 2, "Complexity
 * of Attention Mechanism") and raises throughput (Sec. 4.3).
 *
 * This library implements that decode path:
 *   kvc_append            write new tokens' K/V rows and their positions      (Sec. 2; Sec. 3.1 positions)
 *   kvc_compress_spans    free the rows of closed spans by in-place compaction (Sec. 3.1, freeing the KV)
 *   kvc_decode_attention  one query per (sequence, head) over the kept rows    (Sec. 1 / 3.1 mask; Sec. 4.3)
 *   kvc_prefill_attention every query of a prompt block under the mask, on tensor cores (Sec. 3.1)
 *   kvc_masked_reference_layout   the full history, the mask and the stored rows, for verification
 * plus a host-only span book (kvc_book_*) holding the span bookkeeping that
 * decides what each call does.
 *
 * Conventions
 *   - Every device buffer is allocated by the caller; the library owns host
 *     state only (including a pinned staging ring it allocates on first use)
 *     and never frees caller memory.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  Calls on one cache must be ordered on one stream (or the caller
 *     orders them); they are asynchronous unless stated otherwise.
 *   - Every call returns a kvc_status and never aborts or throws.  Argument and
 *     state errors are detected on the host before anything is launched and
 *     leave the object unchanged.  kvc_last_error() gives a one-line detail.
 *   - Token kinds: KVC_NORMAL, KVC_CL, KVC_CR.  Spans may not overlap or nest
 *     (Sec. 3.1): a <CL> inside an open span and a <CR> without an open span
 *     are KVC_ERR_SPAN.
 *   - Positions are whatever the caller passes; kvc_book_next_positions gives
 *     the paper's tied positions (Sec. 3.1: <CL>/<CR> take the position of the
 *     previous token).  Stored positions are never renumbered by compaction.
 */
#ifndef KVC_H
#define KVC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KVC_OK = 0,
  KVC_ERR_INVALID_ARG = 1,  /* null pointer, out-of-range index, bad size */
  KVC_ERR_UNSUPPORTED = 2,  /* d_head, dtype or rotary_dim this build does not handle */
  KVC_ERR_CAPACITY = 3,     /* a sequence would exceed its capacity */
  KVC_ERR_SPAN = 4,         /* ill-formed or already-freed span, overlap, nesting */
  KVC_ERR_STATE = 5,        /* call order violated (layers pending, spans not yet freed, ...) */
  KVC_ERR_CUDA = 6,         /* a CUDA runtime call or launch failed */
  KVC_ERR_DEVICE_CHECK = 7, /* a kernel's own consistency check failed (see kvc_device_status) */
  KVC_ERR_TIMEOUT = 8,      /* a kernel's bounded wait ran out (see kvc_device_status) */
  KVC_ERR_NO_MEMORY = 9     /* host allocation failed */
} kvc_status;

enum { KVC_NORMAL = 0, KVC_CL = 1, KVC_CR = 2 };
enum { KVC_F16 = 0, KVC_BF16 = 1 };

typedef enum {
  /* The paper's mask: <CL> is visible to no later query, so freeing a span drops <CL> and the
   * enclosed rows and keeps <CR>.  Until then the open span's <CL> row is stored but skipped. */
  KVC_POLICY_PAPER = 0,
  /* Keeps <CL> (drops only the rows strictly between the sentinels) and shows it to later queries. */
  KVC_POLICY_KEEP_CL = 1,
  /* The paper's Local Attention baseline (Sec. 4.1; Sec. 4.2: a FIFO queue of key-value memory at
   * inference): token x_t (1-based) attends within (floor(t * local_ratio), t].  The cache of a
   * sequence is a ring of `capacity` rows that holds the window; no sentinel kinds are accepted. */
  KVC_POLICY_LOCAL = 2
} kvc_policy;

/* A static, NUL-terminated description of status `s` ("ok", "span error", ...; a fixed text for a
 * value outside the enum).  Host only, never fails; the caller does not free it. */
const char* kvc_status_string(kvc_status s);
/* Detail of the last error returned on this thread ("" if none).  Valid until the next call. */
const char* kvc_last_error(void);

/* ======================================================================== */
/* Span book: host-only bookkeeping of b token histories (no CUDA).          */
/* ======================================================================== */

typedef struct kvc_book kvc_book;

/* b sequences; capacity[b] (host) bounds the rows each may store.  For KVC_POLICY_LOCAL use
 * kvc_book_create_local. */
kvc_status kvc_book_create(int b, kvc_policy policy, const int64_t* capacity, kvc_book** out);
/* A book of the Local Attention FIFO cache: each sequence's window must fit its capacity. */
kvc_status kvc_book_create_local(int b, float local_ratio, const int64_t* capacity, kvc_book** out);
void kvc_book_destroy(kvc_book* book);

/* Tied positions (Sec. 3.1) of tokens about to be appended: n_new[b] tokens per sequence with
 * kinds[sum n_new] (sequence-major); pos_out[sum n_new] continues each sequence's history.
 * A normal token takes the number of normal tokens before it; a sentinel takes the position of
 * the token before it (0 for a sequence's first token).  Validates kinds like kvc_book_append
 * (capacity is not checked here). */
kvc_status kvc_book_next_positions(const kvc_book* book, const int32_t* n_new, const uint8_t* kinds,
                                   int32_t* pos_out);

/* Record n_new[b] tokens per sequence (kinds and positions sequence-major, host). */
kvc_status kvc_book_append(kvc_book* book, const int32_t* n_new, const uint8_t* kinds, const int32_t* pos);

/* kvc_book_append that frees, as they are recorded, the spans opened and closed among the new
 * tokens of each sequence (the bookkeeping of kvc_append_free_closed). */
kvc_status kvc_book_append_free_closed(kvc_book* book, const int32_t* n_new, const uint8_t* kinds,
                                       const int32_t* pos);

/* Free closed spans: n_spans entries (seq[i], cl[i], cr[i]) given as history indices of the
 * span's <CL> and <CR>.  Each must be a closed span that is not yet freed, listed once. */
kvc_status kvc_book_compress(kvc_book* book, const int32_t* seq, const int64_t* cl, const int64_t* cr,
                             int n_spans);

/* Closed spans of `seq` that are not yet freed: up to `max` (cl, cr) pairs; *n gets the count. */
kvc_status kvc_book_pending_spans(const kvc_book* book, int seq, int64_t* cl, int64_t* cr, int64_t max,
                                  int64_t* n);

/* Mask bounds of the masked prefill (kvc_prefill_attention) of the last n_q tokens of `seq`: for
 * each stored row i (up to `max`; *n gets the stored-row count) meta[i] = (hid << 1) | is_cl, where
 * row i is visible to the query at stored row iq exactly when i <= iq <= hid, except that a query
 * whose own row has is_cl set (a <CL>, Sec. 3.1) sees only itself.  hid is the stored row of the
 * <CR> that closes a span enclosing row i, i itself for a <CL> row under KVC_POLICY_PAPER, and
 * 0x3FFFFFFF otherwise.  KVC_ERR_STATE if the last n_q tokens are not all stored rows;
 * KVC_ERR_UNSUPPORTED under KVC_POLICY_LOCAL. */
kvc_status kvc_book_prefill_keys(const kvc_book* book, int seq, int64_t n_q, int32_t* meta, int64_t max,
                                 int64_t* n);

/* Stored rows per sequence (len_out[b]) and rows the next decode attends to (attend_out[b]);
 * either may be NULL. */
kvc_status kvc_book_lengths(const kvc_book* book, int64_t* len_out, int64_t* attend_out);

/* The full history of `seq` (kinds, positions, n_full = tokens so far), which history tokens the
 * query at the last token attends to under the mask (visible_full), and the stored rows in order
 * as history indices and positions (n_stored).  Buffers hold `cap` entries each (host). */
kvc_status kvc_book_layout(const kvc_book* book, int seq, int64_t cap, uint8_t* kind_full, int32_t* pos_full,
                           uint8_t* visible_full, int64_t* n_full, int32_t* stored_orig_idx, int32_t* stored_pos,
                           int64_t* n_stored);

/* ======================================================================== */
/* Device cache.                                                            */
/* ======================================================================== */

typedef struct kvc_cache kvc_cache;

typedef struct {
  int M;                        /* layers */
  int H;                        /* heads */
  int d_head;                   /* 16..256, a multiple of 16 (built: 64, 80, 96, 128) */
  int b;                        /* sequences */
  int dtype;                    /* KVC_F16 or KVC_BF16, for K, V and q */
  int rotary_dim;               /* 0 = no RoPE; else even multiple of 16, <= d_head (rotate-half) */
  float rope_base;              /* RoPE base (e.g. 10000) */
  kvc_policy policy;
  const int64_t* seq_capacity;  /* host, b entries: rows each sequence may store */
  /* Caller-owned device buffers, sizes from kvc_required_bytes.  Layout (rows of d_head elements):
   *   K, V: [M][H * C] rows, C = sum(capacity); sequence s, head h, stored row i of layer m at
   *         row m*H*C + H*off[s] + h*capacity[s] + i, off[s] = sum of earlier capacities.
   *   pos, orig: int32 [C]; entry off[s] + i describes stored row i of sequence s (its position
   *         and its history index).  All 256-byte aligned. */
  void* k_base;
  void* v_base;
  int32_t* pos_base;
  int32_t* orig_base;
  void* workspace;              /* device scratch owned by the cache while it lives */
  size_t workspace_bytes;
  float local_ratio;            /* KVC_POLICY_LOCAL only: r in [0, 1); the window is ~(1 - r) of the history */
} kvc_config;

/* Byte sizes of the caller-owned buffers for `cfg` (k_base etc. may be NULL).  Any out pointer may
 * be NULL.  Returns KVC_OK or an argument error. */
kvc_status kvc_required_bytes(const kvc_config* cfg, size_t* k_bytes, size_t* v_bytes, size_t* meta_bytes_each,
                              size_t* workspace_bytes);

/* Host state only; CUDA resources (pinned staging, events) are created by the first call that
 * takes a stream, on the device current at that time. */
kvc_status kvc_create(const kvc_config* cfg, kvc_cache** out);
void kvc_destroy(kvc_cache* cache);

/* The cache's span book (read-only view: positions, pending spans, lengths, layout). */
const kvc_book* kvc_get_book(const kvc_cache* cache);

/* Append tokens (Sec. 2: the cache grows by one row per token, layer, K/V and head).
 *   layer == -1: all layers at once; k, v are device [M][N][H][d_head] with N = sum(n_new).
 *   layer == 0 .. M-1: one layer, k, v are [N][H][d_head]; layer 0 starts a new batch of tokens
 *     (n_new, pos, kinds used); layers 1.. must follow in order and ignore n_new/pos/kinds.
 * k and v are 16-byte aligned (else KVC_ERR_INVALID_ARG).
 * n_new[b], pos[N], kinds[N] are host arrays (sequence-major).  With rotary_dim > 0, K is rotated
 * at its position before it is stored.  A <CL> row is stored and skipped by later queries until
 * its span is freed (paper policy).  Errors: KVC_ERR_CAPACITY, KVC_ERR_SPAN, KVC_ERR_STATE. */
kvc_status kvc_append(kvc_cache* cache, int layer, const void* k, const void* v, const int32_t* n_new,
                      const int32_t* pos, const uint8_t* kinds, void* stream);

/* kvc_append with write-time freeing (Sec. 3.1: the enclosed KV can be released all at once after
 * a prefix, or block by block for long prefixes): spans that both open and close among the new
 * tokens of a sequence are freed as the tokens are written -- their <CL> (paper policy) and
 * enclosed rows are never stored, so no compaction has to move anything for them.  Spans closed
 * here but opened by an earlier call, or still open, are stored as by kvc_append (free the former
 * with kvc_compress_spans).  Capacity counts only stored rows.  Same arguments as kvc_append. */
kvc_status kvc_append_free_closed(kvc_cache* cache, int layer, const void* k, const void* v, const int32_t* n_new,
                                  const int32_t* pos, const uint8_t* kinds, void* stream);

/* Free closed spans (Sec. 3.1): for each listed (seq, cl, cr) -- history indices of a closed,
 * not yet freed span -- drop its rows (<CL> and the enclosed tokens under the paper policy, only
 * the enclosed tokens under KEEP_CL), keep <CR>, and compact the survivors in place in every
 * (layer, K/V, head) stream of that sequence, keeping their order, positions and history indices.
 * Requires every layer of the last appended tokens to be written.  Host arrays.
 * Ordering: a <CR> query sees its own span's interior, so free a span after the <CR> token's
 * decode calls; once freed, a decode of that same query reads only the rows that are left. */
kvc_status kvc_compress_spans(kvc_cache* cache, const int32_t* seq, const int64_t* cl, const int64_t* cr,
                              int n_spans, void* stream);

/* Decode attention of layer `layer` (Sec. 1 / Sec. 3.1 mask, Sec. 4.3 throughput): the query of
 * each sequence is its last appended token; q is device [b][H][d_head] in the cache dtype, rotated
 * at that token's position when rotary_dim > 0; out is device fp32 [b][H][d_head]:
 *   out = sum_j softmax_j(scale * <q, k_j>) v_j  over the stored rows j the query may see.
 * A <CL> query attends to its own row only.  Rows of spans closed before the query must have been
 * freed, except at most one contiguous run of hidden rows per sequence (KVC_ERR_STATE otherwise).
 * Split-K over the kept rows with a log-sum-exp combine; reads only the kept rows. */
kvc_status kvc_decode_attention(kvc_cache* cache, int layer, const void* q, float scale, float* out, void* stream);

/* kvc_decode_attention of layers first .. first + n_layers - 1 in one call (the decode step of a
 * model whose queries for all those layers are ready, as in the paper's throughput setting,
 * Sec. 4.3): layer first + i reads q + i * q_layer_stride elements of the cache dtype and writes
 * out + i * out_layer_stride floats; strides are in elements, each layer's slice laid out as for
 * kvc_decode_attention.  One launch covers every layer's segments, each (layer, sequence, head)
 * segment processed whole by one warp exactly as a per-layer launch with the same tile shape does it,
 * when the segments hold about as many rows as each other (the longest at most 1.3x the mean) or when
 * the longest is short beside a warp's even share of all the layers' rows (at most 1/16 of it; the
 * warps then take runs of whole segments cut by rows).  Otherwise the layers are launched one by one,
 * in order, on `stream`, and on an error the layers before the failing one have been launched. */
kvc_status kvc_decode_attention_layers(kvc_cache* cache, int first, int n_layers, const void* q, int64_t q_layer_stride,
                                       float scale, float* out, int64_t out_layer_stride, void* stream);

/* The same decode as kvc_decode_attention, for callers that cannot allocate device memory at run
 * time (for example code running inside a fixed memory pool, or under an allocator that forbids
 * new device allocations): its split-K scratch -- partial results and arrival counters -- lives in
 * a file-scope __device__ array of libkvc instead of the cache workspace, so the call allocates
 * nothing (no cudaMalloc or cudaFree, no allocating library routine).  The paper has no counterpart;
 * this is an interface convenience.
 *   - Size limit: 8 MiB, enough while 4*((8192 + b*H)*(d_head + 4) rounded up to 256) + 4*b*H fits;
 *     larger caches get KVC_ERR_UNSUPPORTED (use kvc_decode_attention).
 *   - Every GPU that loads the library holds the 8 MiB until the process exits.
 *   - The first call on a device looks up the array's device address (cudaGetSymbolAddress); make
 *     that first call before any stream capture.
 *   - All calls share the one array: calls that overlap on the GPU (different streams, caches or
 *     threads without ordering between them) race and give wrong results.  Each call clears the
 *     counters it relies on before its kernel runs, on `stream`. */
kvc_status kvc_decode_attention_static_scratch(kvc_cache* cache, int layer, const void* q, float scale, float* out,
                                               void* stream);

/* Masked prefill attention of layer `layer` on the tensor cores (Sec. 3.1: the modified causal
 * mask holds for every token of a prompt; Manipulating Key-Value Memory: a long prefix may be run
 * block by block).  For every sequence s with n_q[s] > 0 the queries are its last n_q[s] tokens;
 * each attends, under the mask, to the stored rows of s -- exactly the rows a decode step at that
 * token would see (the per-row rule is kvc_book_prefill_keys').
 *   q:   device [sum n_q][H][d_head] in the cache dtype, sequence-major (sequence s's queries
 *        consecutive, oldest first), NOT rotated: the kernel rotates each query at its token's
 *        stored position when rotary_dim > 0, then rounds it to the cache dtype; 16-byte aligned.
 *   n_q: host [b], 0 <= n_q[s] <= tokens of s.
 *   out: device fp32 [sum n_q][H][d_head] = sum_j softmax_j(scale * <q, k_j>) v_j, 16-byte aligned.
 *   scale: > 0.
 * The queries' own K/V rows must be stored: append a block with kvc_append (every layer up to
 * `layer` written), run the prefill of each layer, then free the spans the block closed with
 * kvc_compress_spans -- the block-by-block loop of Sec. 3.1.  Spans closed earlier may still be
 * stored (their rows are masked), so a whole prompt can also be appended and run in one call.
 * Errors: KVC_ERR_STATE when a query token is not stored (for example freed by
 * kvc_append_free_closed) or its layer is not written; KVC_ERR_UNSUPPORTED under
 * KVC_POLICY_LOCAL or when M * H * sum(capacity) >= 2^31 rows.  Asynchronous. */
kvc_status kvc_prefill_attention(kvc_cache* cache, int layer, const void* q, const int32_t* n_q, float scale,
                                 float* out, void* stream);

/* Verification (synchronous: waits for `stream`): the history of `seq` and the mask for its next
 * query as in kvc_book_layout, with the stored rows read back from the device metadata
 * (stored_orig_idx, stored_pos, n_stored = the device's view).  Buffers of `cap` entries. */
kvc_status kvc_masked_reference_layout(kvc_cache* cache, int seq, int64_t cap, uint8_t* kind_full, int32_t* pos_full,
                                       uint8_t* visible_full, int64_t* n_full, int32_t* stored_orig_idx,
                                       int32_t* stored_pos, int64_t* n_stored, void* stream);

/* Reads and clears the kernels' status word (synchronous on `stream`).  *word gets the raw bits
 * (0 = clean; 1 = a bounded wait ran out; 2 = a consistency check failed).  Returns KVC_OK,
 * KVC_ERR_TIMEOUT or KVC_ERR_DEVICE_CHECK accordingly. */
kvc_status kvc_device_status(kvc_cache* cache, void* stream, int32_t* word);

/* Checks the kernels' failure reporting without a fault: launches one warp that waits, with the
 * same bounded wait the decode kernel uses, on a barrier phase that nothing completes.  After
 * limit_ns (0 < limit_ns <= 2e9) the wait gives up and sets the timeout bit of the status word, so
 * that the next kvc_device_status returns KVC_ERR_TIMEOUT; the context stays usable.  Asynchronous. */
kvc_status kvc_check_bounded_wait(kvc_cache* cache, uint64_t limit_ns, void* stream);

/* Number of kernels this cache has launched so far. */
int64_t kvc_launch_count(const kvc_cache* cache);

/* Measurement of the two compaction kernels (Sec. 3.1, freeing the enclosed KV): with enable != 0,
 * every later kvc_compress_spans that moves rows records CUDA events on its stream before the keep
 * flag scan, between the scan and the row moves, and after the row moves (0 turns this off).  The
 * event between the kernels keeps the row moves from being scheduled before the scan completes, so
 * a timed compaction can take a few microseconds longer than an untimed one.  The events are created
 * on the current device at the first timed call and freed by kvc_destroy. */
kvc_status kvc_set_compaction_timing(kvc_cache* cache, int enable);

/* Durations in milliseconds of the last compaction's scan and row moves (synchronous: waits for
 * its last event).  KVC_ERR_STATE if the last kvc_compress_spans was not timed or moved nothing. */
kvc_status kvc_last_compaction_ms(kvc_cache* cache, float* scan_ms, float* move_ms);

/* How the last decode launch divided its work (host-side record, no synchronisation):
 * plan[0] = mode (0: the kept rows split evenly over a full wave of warps, split (sequence, head)
 * segments merged by a log-sum-exp combine; 1 / 2: one warp per segment with the wide / narrow
 * shared-memory pipeline; 3: several consecutive whole segments per warp, no combine; 4: runs of
 * consecutive whole segments per warp cut by rows, over several layers, no combine; -1: nothing
 * launched yet), plan[1] = warps, plan[2] = rows per tile, plan[3] = pipeline stages per warp. */
kvc_status kvc_last_decode_plan(const kvc_cache* cache, int32_t* plan);

#ifdef __cplusplus
}
#endif

#endif /* KVC_H */
