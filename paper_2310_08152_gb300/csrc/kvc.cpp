// C ABI of the sentinel-compressed KV cache (declared in include/kvc.h): argument checks, the span
// book, staging of per-call plans to the device, and kernel launches.
#include "kvc.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <deque>
#include <new>
#include <string>
#include <vector>

#include "book.hpp"
#include "kernels.hpp"

namespace {

thread_local std::string g_last_error;

kvc_status fail(kvc_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

kvc_status ok() {
  g_last_error.clear();
  return KVC_OK;
}

kvc_status cuda_fail(cudaError_t e, const char* what) {
  return fail(KVC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr double kPi = 3.14159265358979323846;

size_t align_up(size_t n, size_t a) { return (n + a - 1) / a * a; }

// Byte offsets of the workspace regions.
struct WsLayout {
  size_t hdr = 0;        // int status word
  size_t st_row0 = 0;    // int64 [b]
  size_t st_cap = 0;     // int32 [b]
  size_t st_off = 0;     // int64 [b]
  size_t st_rope = 0;    // float2 [max(1, rot/2)]
  size_t amaps = 0;      // TMA descriptors of the append kernel: [K/V][b] x 128 bytes
  size_t dyn = 0;        // [DState b][int64 P b+1][payload]
  size_t dyn_P = 0;      // offset of P inside dyn
  size_t dyn_payload = 0;  // offset of the payload inside dyn
  size_t dyn_bytes = 0;
  size_t src_map = 0;    // int32 [C]: source row of each destination row of a compaction
  size_t counters = 0;   // int32 [b*H]
  size_t partials = 0;   // float [(kMaxDecodeWorkers + b*H) * (D + 4)]
  size_t pre_counter = 0;  // uint64: the prefill launch's next work item
  size_t pre = 0;        // prefill plan: [PfItemRec items][int32 meta C]
  size_t pre_items = 0;  // offsets inside the plan; PfItemRec [pre_max_items]
  int64_t pre_max_items = 0;
  size_t pre_meta = 0;
  size_t pre_bytes = 0;
  size_t total = 0;
};

WsLayout ws_layout(int b, int H, int D, int rot, int64_t C) {
  WsLayout L;
  size_t o = 0;
  auto take = [&](size_t n) {
    size_t r = o;
    o += align_up(n, 256);
    return r;
  };
  L.hdr = take(256);
  L.st_row0 = take(8 * (size_t)b);
  L.st_cap = take(4 * (size_t)b);
  L.st_off = take(8 * (size_t)b);
  L.st_rope = take(8 * (size_t)std::max(1, rot / 2));
  L.amaps = take(kvc::append_maps_bytes(b));
  L.dyn_P = align_up(sizeof(kvc::DState) * (size_t)b, 16);
  L.dyn_payload = align_up(L.dyn_P + 8 * (size_t)(b + 1), 16);
  const size_t tok = sizeof(kvc::TokPlan) * (size_t)C;
  const size_t cmp = sizeof(kvc::AffSeq) * (size_t)b + 8 * (size_t)(C / 2 + 1);
  L.dyn_bytes = L.dyn_payload + std::max(tok, cmp);
  L.dyn = take(L.dyn_bytes);
  L.src_map = take(4 * (size_t)C);
  L.counters = take(4 * (size_t)b * H);
  L.partials = take(4 * (size_t)(kvc::kMaxDecodeWorkers + (int64_t)b * H) * (size_t)(D + 4));
  // work items: H per query tile, and a sequence of capacity cap has at most ceil(cap / 128) query
  // tiles, so at most H * (C / 128 + b) in all
  L.pre_items = 0;
  L.pre_max_items = (int64_t)H * ((C + 127) / 128 + b);
  L.pre_meta = align_up(L.pre_items + sizeof(kvc::PfItemRec) * (size_t)L.pre_max_items, 16);
  L.pre_bytes = L.pre_meta + 4 * (size_t)C;
  L.pre_counter = take(8);
  L.pre = take(L.pre_bytes);
  L.total = o;
  return L;
}

kvc_status check_config(const kvc_config* c, int64_t* C_out) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "config is NULL");
  if (c->M <= 0 || c->H <= 0 || c->b <= 0)
    return fail(KVC_ERR_INVALID_ARG, "M=%d, H=%d, b=%d must be positive", c->M, c->H, c->b);
  if (!kvc::dhead_supported(c->d_head))
    return fail(KVC_ERR_UNSUPPORTED, "d_head=%d is not built (64, 80, 96, 128)", c->d_head);
  if (c->dtype != KVC_F16 && c->dtype != KVC_BF16) return fail(KVC_ERR_UNSUPPORTED, "dtype %d", c->dtype);
  if (c->rotary_dim < 0 || c->rotary_dim > c->d_head || c->rotary_dim % 16 != 0)
    return fail(KVC_ERR_UNSUPPORTED, "rotary_dim=%d must be a multiple of 16 in [0, d_head]", c->rotary_dim);
  if (c->rotary_dim > 0 && !(c->rope_base > 1.0f))
    return fail(KVC_ERR_INVALID_ARG, "rope_base=%g must exceed 1", (double)c->rope_base);
  if (c->policy != KVC_POLICY_PAPER && c->policy != KVC_POLICY_KEEP_CL && c->policy != KVC_POLICY_LOCAL)
    return fail(KVC_ERR_INVALID_ARG, "policy %d", (int)c->policy);
  if (c->policy == KVC_POLICY_LOCAL && !(c->local_ratio >= 0.0f && c->local_ratio < 1.0f))
    return fail(KVC_ERR_INVALID_ARG, "local_ratio=%g must be in [0, 1)", (double)c->local_ratio);
  if (!c->seq_capacity) return fail(KVC_ERR_INVALID_ARG, "seq_capacity is NULL");
  int64_t C = 0;
  for (int s = 0; s < c->b; ++s) {
    if (c->seq_capacity[s] < 1 || c->seq_capacity[s] >= INT32_MAX)
      return fail(KVC_ERR_INVALID_ARG, "seq_capacity[%d]=%lld out of range", s, (long long)c->seq_capacity[s]);
    C += c->seq_capacity[s];
  }
  if ((int64_t)c->H * C >= ((int64_t)1 << 40)) return fail(KVC_ERR_INVALID_ARG, "cache too large");
  if (C >= INT32_MAX) return fail(KVC_ERR_INVALID_ARG, "sum of capacities must stay below 2^31");
  *C_out = C;
  return KVC_OK;
}

// Pinned host staging ring: each upload reserves a slot, fills it, enqueues one H2D copy and
// records an event; a slot is reused only after its copy completed.
class PinnedRing {
 public:
  ~PinnedRing() { release(); }
  cudaError_t init(size_t bytes) {
    cap_ = align_up(bytes, 256);
    return cudaHostAlloc(reinterpret_cast<void**>(&base_), cap_, cudaHostAllocDefault);
  }
  void release() {
    for (auto& p : pending_) cudaEventDestroy(p.ev);
    for (auto e : free_) cudaEventDestroy(e);
    pending_.clear();
    free_.clear();
    if (base_) cudaFreeHost(base_);
    base_ = nullptr;
  }
  // Returns nullptr if n exceeds the ring or a wait failed.
  unsigned char* reserve(size_t n, cudaError_t* err) {
    n = align_up(n, 256);
    *err = cudaSuccess;
    if (n > cap_) return nullptr;
    if (head_ + n > cap_) head_ = 0;
    for (auto it = pending_.begin(); it != pending_.end();) {
      if (it->off < head_ + n && head_ < it->off + it->len) {
        cudaError_t e = cudaEventSynchronize(it->ev);
        if (e != cudaSuccess) {
          *err = e;
          return nullptr;
        }
        free_.push_back(it->ev);
        it = pending_.erase(it);
      } else {
        ++it;
      }
    }
    res_ = n;
    return base_ + head_;
  }
  cudaError_t commit(void* dev_dst, size_t bytes, cudaStream_t stream) {
    cudaError_t e = cudaMemcpyAsync(dev_dst, base_ + head_, bytes, cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return e;
    cudaEvent_t ev;
    if (!free_.empty()) {
      ev = free_.back();
      free_.pop_back();
    } else {
      e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
      if (e != cudaSuccess) return e;
    }
    e = cudaEventRecord(ev, stream);
    if (e != cudaSuccess) return e;
    pending_.push_back({head_, res_, ev});
    head_ += res_;
    return cudaSuccess;
  }

 private:
  struct Pending {
    size_t off, len;
    cudaEvent_t ev;
  };
  unsigned char* base_ = nullptr;
  size_t cap_ = 0, head_ = 0, res_ = 0;
  std::deque<Pending> pending_;
  std::vector<cudaEvent_t> free_;
};

}  // namespace

struct kvc_book {
  kvc::Book book;
  kvc_book(int b, kvc::Policy p, const int64_t* cap, double local_ratio = 0.0) : book(b, p, cap, local_ratio) {}
};

struct kvc_cache {
  kvc_config cfg{};
  std::vector<int64_t> cap, off;
  int64_t C = 0;
  kvc_book bk;
  WsLayout ws;
  // device binding (first call with a stream)
  bool cuda_ready = false;
  int device = -1;
  int num_sms = 0;
  PinnedRing ring;
  // token batch in progress: layers [0, layers_done) written
  int layers_done = 0;
  int64_t batch_ntok = 0;  // stored tokens of the batch (plan entries)
  int64_t batch_nin = 0;   // input tokens of the batch (per layer of k, v)
  // decode readiness of the uploaded state
  bool decode_ok = false;
  std::string decode_err;
  int64_t R = 0;
  int64_t n_segments = 0, max_segment = 0;
  int64_t launches = 0;
  // the last kernel this cache launched was a decode (it writes no K/V rows)
  bool last_was_decode = false;
  kvc::DecodePlan last_plan{-1, 0, 0, 0};
  // book changes (appends, compactions); the prefill plan is rebuilt when it moved on
  uint64_t version = 0;
  uint64_t pre_version = UINT64_MAX;
  std::vector<int32_t> pre_nq;
  int64_t pre_tiles = 0;
  int pre_ctas = 0;
  kvc::PrefillMaps maps;
  bool amaps_ok = false;  // the append kernel's TMA descriptors are in the workspace
  // compaction timing (kvc_set_compaction_timing): events before the scan, between the kernels, after
  bool time_compaction = false;
  bool timed_compaction = false;  // the last compaction recorded them
  cudaEvent_t cev[3] = {nullptr, nullptr, nullptr};

  kvc_cache(const kvc_config& c, int64_t C_)
      : cfg(c), C(C_), bk(c.b, (kvc::Policy)c.policy, c.seq_capacity, (double)c.local_ratio) {
    cap.assign(c.seq_capacity, c.seq_capacity + c.b);
    off.resize(c.b);
    int64_t o = 0;
    for (int s = 0; s < c.b; ++s) {
      off[s] = o;
      o += cap[s];
    }
    ws = ws_layout(c.b, c.H, c.d_head, c.rotary_dim, C);
    layers_done = c.M;
  }

  ~kvc_cache() {
    for (auto& e : cev)
      if (e) cudaEventDestroy(e);
  }

  unsigned char* wsp(size_t o) const { return static_cast<unsigned char*>(cfg.workspace) + o; }

  kvc::Geometry geom() const {
    kvc::Geometry g;
    g.M = cfg.M;
    g.H = cfg.H;
    g.D = cfg.d_head;
    g.b = cfg.b;
    g.C = C;
    g.dtype = cfg.dtype;
    g.rot = cfg.rotary_dim;
    return g;
  }
  kvc::Static stat() const {
    kvc::Static s;
    s.seq_row0 = reinterpret_cast<const int64_t*>(wsp(ws.st_row0));
    s.cap = reinterpret_cast<const int32_t*>(wsp(ws.st_cap));
    s.off = reinterpret_cast<const int64_t*>(wsp(ws.st_off));
    s.rope_g = reinterpret_cast<const float2*>(wsp(ws.st_rope));
    return s;
  }
  kvc::Buffers bufs() const {
    kvc::Buffers b;
    b.k = static_cast<uint16_t*>(cfg.k_base);
    b.v = static_cast<uint16_t*>(cfg.v_base);
    b.pos = cfg.pos_base;
    b.orig = cfg.orig_base;
    b.status = reinterpret_cast<int*>(wsp(ws.hdr));
    return b;
  }

  kvc_status ensure_cuda(cudaStream_t stream) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (cuda_ready) {
      if (dev != device) return fail(KVC_ERR_STATE, "cache is bound to device %d but device %d is current", device, dev);
      return KVC_OK;
    }
    e = cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    e = ring.init(2 * ws.dyn_bytes + ws.pre_bytes + 2 * ws.st_rope + kvc::append_maps_bytes(cfg.b) + 65536);
    if (e != cudaSuccess) return cuda_fail(e, "cudaHostAlloc (staging ring)");
    // static tables
    const int b = cfg.b, half = std::max(1, cfg.rotary_dim / 2);
    const size_t st_bytes = ws.st_rope + 8 * (size_t)half - ws.st_row0;
    unsigned char* h = ring.reserve(st_bytes, &e);
    if (!h) return e != cudaSuccess ? cuda_fail(e, "staging") : fail(KVC_ERR_INVALID_ARG, "static tables exceed ring");
    std::memset(h, 0, st_bytes);
    int64_t* row0 = reinterpret_cast<int64_t*>(h + (ws.st_row0 - ws.st_row0));
    int32_t* capd = reinterpret_cast<int32_t*>(h + (ws.st_cap - ws.st_row0));
    int64_t* offd = reinterpret_cast<int64_t*>(h + (ws.st_off - ws.st_row0));
    float* rope = reinterpret_cast<float*>(h + (ws.st_rope - ws.st_row0));
    for (int s = 0; s < b; ++s) {
      row0[s] = (int64_t)cfg.H * off[s];
      capd[s] = (int32_t)cap[s];
      offd[s] = off[s];
    }
    // theta_i / (2 pi) per unit position, i < rot/2, as a double-float pair
    for (int i = 0; i < cfg.rotary_dim / 2; ++i) {
      const double g = std::pow((double)cfg.rope_base, -2.0 * i / (double)cfg.rotary_dim) / (2.0 * kPi);
      const float hi = (float)g;
      rope[2 * i] = hi;
      rope[2 * i + 1] = (float)(g - (double)hi);
    }
    e = ring.commit(wsp(ws.st_row0), st_bytes, stream);
    if (e != cudaSuccess) return cuda_fail(e, "upload static tables");
    // the append kernel's TMA descriptors (64-byte aligned in the workspace); without them (a box
    // cannot hold H heads) appends take the kernel that copies through registers
    amaps_ok = false;
    if ((reinterpret_cast<uintptr_t>(wsp(ws.amaps)) & 63) == 0) {
      std::vector<int32_t> cap32(cap.begin(), cap.end());
      std::vector<int64_t> row0h(b);
      for (int s = 0; s < b; ++s) row0h[s] = (int64_t)cfg.H * off[s];
      const size_t mb = kvc::append_maps_bytes(b);
      unsigned char* hm = ring.reserve(mb, &e);
      if (!hm) return e != cudaSuccess ? cuda_fail(e, "staging") : fail(KVC_ERR_INVALID_ARG, "descriptors exceed ring");
      if (kvc::encode_append_maps(geom(), bufs(), row0h.data(), cap32.data(), hm) == cudaSuccess) {
        e = ring.commit(wsp(ws.amaps), mb, stream);
        if (e != cudaSuccess) return cuda_fail(e, "upload append descriptors");
        amaps_ok = true;
      }
    }
    e = cudaMemsetAsync(wsp(ws.hdr), 0, 256, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(wsp(ws.counters), 0, 4 * (size_t)cfg.b * cfg.H, stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    device = dev;
    cuda_ready = true;
    return KVC_OK;
  }

  // Fill the decode state + prefix at the head of a dyn image.
  void fill_state(unsigned char* img) {
    ++version;
    kvc::DState* ds = reinterpret_cast<kvc::DState*>(img);
    int64_t* P = reinterpret_cast<int64_t*>(img + ws.dyn_P);
    decode_ok = true;
    decode_err.clear();
    P[0] = 0;
    n_segments = 0;
    max_segment = 0;
    for (int s = 0; s < cfg.b; ++s) {
      kvc::DecodeView v;
      std::string err;
      int64_t Lc = 0;
      std::memset(&ds[s], 0, sizeof(kvc::DState));
      if (bk.book.history(s) == 0) {
        // no token yet: nothing to attend to, the sequence is skipped
      } else if (bk.book.decode_view(s, v, err)) {
        ds[s].len = (int32_t)v.len;
        ds[s].begin = (int32_t)v.begin;
        ds[s].mask_lo = (int32_t)v.mask_lo;
        ds[s].mask_hi = (int32_t)v.mask_hi;
        ds[s].qpos = v.qpos;
        ds[s].wrap = (int32_t)std::min<int64_t>(v.wrap, INT32_MAX);
        Lc = v.len - v.begin;
      } else {
        if (decode_ok) decode_err = err;
        decode_ok = false;
      }
      P[s + 1] = P[s] + Lc;
      if (Lc > 0) {
        n_segments += cfg.H;
        max_segment = std::max(max_segment, Lc);
      }
    }
    R = (int64_t)cfg.H * P[cfg.b];
  }
};

extern "C" {

const char* kvc_status_string(kvc_status s) {
  switch (s) {
    case KVC_OK:
      return "ok";
    case KVC_ERR_INVALID_ARG:
      return "invalid argument";
    case KVC_ERR_UNSUPPORTED:
      return "unsupported";
    case KVC_ERR_CAPACITY:
      return "capacity exceeded";
    case KVC_ERR_SPAN:
      return "span error";
    case KVC_ERR_STATE:
      return "state error";
    case KVC_ERR_CUDA:
      return "CUDA error";
    case KVC_ERR_DEVICE_CHECK:
      return "device check failed";
    case KVC_ERR_TIMEOUT:
      return "device wait timed out";
    case KVC_ERR_NO_MEMORY:
      return "out of host memory";
  }
  return "unknown status";
}

const char* kvc_last_error(void) { return g_last_error.c_str(); }

// ------------------------------------------------------------------------------------------
// book
// ------------------------------------------------------------------------------------------

kvc_status kvc_book_create_local(int b, float local_ratio, const int64_t* capacity, kvc_book** out) {
  if (!out || !capacity || b <= 0) return fail(KVC_ERR_INVALID_ARG, "b must be positive, pointers non-NULL");
  if (!(local_ratio >= 0.0f && local_ratio < 1.0f)) return fail(KVC_ERR_INVALID_ARG, "local_ratio must be in [0, 1)");
  for (int s = 0; s < b; ++s)
    if (capacity[s] < 1) return fail(KVC_ERR_INVALID_ARG, "capacity[%d] < 1", s);
  kvc_book* bk = new (std::nothrow) kvc_book(b, kvc::POLICY_LOCAL, capacity, (double)local_ratio);
  if (!bk) return fail(KVC_ERR_NO_MEMORY, "book");
  *out = bk;
  return ok();
}

kvc_status kvc_book_create(int b, kvc_policy policy, const int64_t* capacity, kvc_book** out) {
  if (!out || !capacity || b <= 0) return fail(KVC_ERR_INVALID_ARG, "b must be positive, pointers non-NULL");
  if (policy != KVC_POLICY_PAPER && policy != KVC_POLICY_KEEP_CL)
    return fail(KVC_ERR_INVALID_ARG, "policy %d (a local-attention book is made by kvc_book_create_local)", (int)policy);
  for (int s = 0; s < b; ++s)
    if (capacity[s] < 1) return fail(KVC_ERR_INVALID_ARG, "capacity[%d] < 1", s);
  kvc_book* bk = new (std::nothrow) kvc_book(b, (kvc::Policy)policy, capacity);
  if (!bk) return fail(KVC_ERR_NO_MEMORY, "book");
  *out = bk;
  return ok();
}

void kvc_book_destroy(kvc_book* book) { delete book; }

static kvc_status book_check_append(const kvc::Book& B, const int32_t* n_new, const uint8_t* kinds) {
  if (!n_new) return fail(KVC_ERR_INVALID_ARG, "n_new is NULL");
  int64_t N = 0;
  for (int s = 0; s < B.b(); ++s) N += n_new[s] > 0 ? n_new[s] : 0;
  if (N > 0 && !kinds) return fail(KVC_ERR_INVALID_ARG, "kinds is NULL");
  std::string err;
  int code = 0;
  if (!B.check_append(n_new, kinds, err, code)) return fail((kvc_status)code, "%s", err.c_str());
  return KVC_OK;
}

kvc_status kvc_book_next_positions(const kvc_book* book, const int32_t* n_new, const uint8_t* kinds,
                                   int32_t* pos_out) {
  if (!book) return fail(KVC_ERR_INVALID_ARG, "book is NULL");
  if (!n_new) return fail(KVC_ERR_INVALID_ARG, "n_new is NULL");
  int64_t N = 0;
  for (int s = 0; s < book->book.b(); ++s) N += n_new[s] > 0 ? n_new[s] : 0;
  if (N > 0 && !kinds) return fail(KVC_ERR_INVALID_ARG, "kinds is NULL");
  std::string err;
  int code = 0;  // positions need well-formed kinds, not capacity
  if (!book->book.check_append(n_new, kinds, err, code, false, false)) return fail((kvc_status)code, "%s", err.c_str());
  if (!pos_out) return fail(KVC_ERR_INVALID_ARG, "pos_out is NULL");
  book->book.next_positions(n_new, kinds, pos_out);
  return ok();
}

kvc_status kvc_book_append(kvc_book* book, const int32_t* n_new, const uint8_t* kinds, const int32_t* pos) {
  if (!book) return fail(KVC_ERR_INVALID_ARG, "book is NULL");
  kvc_status st = book_check_append(book->book, n_new, kinds);
  if (st != KVC_OK) return st;
  if (!pos) return fail(KVC_ERR_INVALID_ARG, "pos is NULL");
  book->book.apply_append(n_new, kinds, pos);
  return ok();
}

kvc_status kvc_book_append_free_closed(kvc_book* book, const int32_t* n_new, const uint8_t* kinds,
                                       const int32_t* pos) {
  if (!book) return fail(KVC_ERR_INVALID_ARG, "book is NULL");
  if (!n_new) return fail(KVC_ERR_INVALID_ARG, "n_new is NULL");
  int64_t N = 0;
  for (int s = 0; s < book->book.b(); ++s) N += n_new[s] > 0 ? n_new[s] : 0;
  if (N > 0 && (!kinds || !pos)) return fail(KVC_ERR_INVALID_ARG, "kinds/pos are NULL");
  std::string err;
  int code = 0;
  if (!book->book.check_append(n_new, kinds, err, code, true)) return fail((kvc_status)code, "%s", err.c_str());
  std::vector<uint8_t> kept;
  book->book.kept_in_block(n_new, kinds, kept);
  book->book.apply_append(n_new, kinds, pos, kept.data());
  return ok();
}

kvc_status kvc_book_compress(kvc_book* book, const int32_t* seq, const int64_t* cl, const int64_t* cr, int n_spans) {
  if (!book) return fail(KVC_ERR_INVALID_ARG, "book is NULL");
  if (n_spans < 0 || (n_spans > 0 && (!seq || !cl || !cr))) return fail(KVC_ERR_INVALID_ARG, "span arrays");
  std::vector<kvc::CompactSeq> plan;
  std::string err;
  if (!book->book.plan_compress(seq, cl, cr, n_spans, plan, err)) return fail(KVC_ERR_SPAN, "%s", err.c_str());
  book->book.apply_compress(plan, seq, cl, n_spans);
  return ok();
}

kvc_status kvc_book_pending_spans(const kvc_book* book, int seq, int64_t* cl, int64_t* cr, int64_t max, int64_t* n) {
  if (!book || !n) return fail(KVC_ERR_INVALID_ARG, "NULL argument");
  if (seq < 0 || seq >= book->book.b()) return fail(KVC_ERR_INVALID_ARG, "seq %d out of range", seq);
  std::vector<std::pair<int64_t, int64_t>> v;
  book->book.pending_spans(seq, v);
  *n = (int64_t)v.size();
  for (int64_t i = 0; i < std::min<int64_t>(max, (int64_t)v.size()); ++i) {
    if (cl) cl[i] = v[i].first;
    if (cr) cr[i] = v[i].second;
  }
  return ok();
}

kvc_status kvc_book_prefill_keys(const kvc_book* book, int seq, int64_t n_q, int32_t* meta, int64_t max,
                                 int64_t* n) {
  if (!book || !n) return fail(KVC_ERR_INVALID_ARG, "book/n is NULL");
  if (seq < 0 || seq >= book->book.b()) return fail(KVC_ERR_INVALID_ARG, "seq %d out of range", seq);
  if (book->book.policy() == kvc::POLICY_LOCAL)
    return fail(KVC_ERR_UNSUPPORTED, "masked prefill is not defined for the local-attention cache");
  std::vector<int32_t> m;
  std::string err;
  if (!book->book.prefill_keys(seq, n_q, m, err)) return fail(KVC_ERR_STATE, "%s", err.c_str());
  *n = (int64_t)m.size();
  if ((int64_t)m.size() > max) return fail(KVC_ERR_INVALID_ARG, "meta holds %lld entries, %lld needed", (long long)max,
                                           (long long)m.size());
  if (!m.empty() && !meta) return fail(KVC_ERR_INVALID_ARG, "meta is NULL");
  std::memcpy(meta, m.data(), 4 * m.size());
  return ok();
}

kvc_status kvc_book_lengths(const kvc_book* book, int64_t* len_out, int64_t* attend_out) {
  if (!book) return fail(KVC_ERR_INVALID_ARG, "book is NULL");
  const kvc::Book& B = book->book;
  for (int s = 0; s < B.b(); ++s) {
    if (len_out) len_out[s] = B.stored(s);
    if (attend_out) {
      kvc::DecodeView v;
      std::string err;
      attend_out[s] = (B.history(s) > 0 && B.decode_view(s, v, err)) ? v.attended() : 0;
    }
  }
  return ok();
}

kvc_status kvc_book_layout(const kvc_book* book, int seq, int64_t cap, uint8_t* kind_full, int32_t* pos_full,
                           uint8_t* visible_full, int64_t* n_full, int32_t* stored_orig_idx, int32_t* stored_pos,
                           int64_t* n_stored) {
  if (!book || !n_full || !n_stored) return fail(KVC_ERR_INVALID_ARG, "NULL argument");
  const kvc::Book& B = book->book;
  if (seq < 0 || seq >= B.b()) return fail(KVC_ERR_INVALID_ARG, "seq %d out of range", seq);
  const int64_t T = B.history(seq);
  *n_full = T;
  std::vector<int32_t> o, p;
  B.stored_rows(seq, o, p);
  *n_stored = (int64_t)o.size();
  if (T > cap || (int64_t)o.size() > cap) return fail(KVC_ERR_CAPACITY, "cap %lld < %lld entries", (long long)cap, (long long)T);
  if (kind_full) std::memcpy(kind_full, B.kinds(seq).data(), (size_t)T);
  if (pos_full) std::memcpy(pos_full, B.positions(seq).data(), 4 * (size_t)T);
  if (visible_full) B.visible(seq, visible_full);
  if (stored_orig_idx) std::memcpy(stored_orig_idx, o.data(), 4 * o.size());
  if (stored_pos) std::memcpy(stored_pos, p.data(), 4 * p.size());
  return ok();
}

// ------------------------------------------------------------------------------------------
// cache
// ------------------------------------------------------------------------------------------

kvc_status kvc_required_bytes(const kvc_config* cfg, size_t* k_bytes, size_t* v_bytes, size_t* meta_bytes_each,
                              size_t* workspace_bytes) {
  int64_t C = 0;
  kvc_status st = check_config(cfg, &C);
  if (st != KVC_OK) return st;
  const size_t kv = (size_t)cfg->M * cfg->H * (size_t)C * cfg->d_head * 2;
  if (k_bytes) *k_bytes = kv;
  if (v_bytes) *v_bytes = kv;
  if (meta_bytes_each) *meta_bytes_each = 4 * (size_t)C;
  if (workspace_bytes) *workspace_bytes = ws_layout(cfg->b, cfg->H, cfg->d_head, cfg->rotary_dim, C).total;
  return ok();
}

kvc_status kvc_create(const kvc_config* cfg, kvc_cache** out) {
  if (!out) return fail(KVC_ERR_INVALID_ARG, "out is NULL");
  int64_t C = 0;
  kvc_status st = check_config(cfg, &C);
  if (st != KVC_OK) return st;
  if (!cfg->k_base || !cfg->v_base || !cfg->pos_base || !cfg->orig_base || !cfg->workspace)
    return fail(KVC_ERR_INVALID_ARG, "device buffers must be non-NULL");
  auto al = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 255u) == 0; };
  if (!al(cfg->k_base) || !al(cfg->v_base) || !al(cfg->pos_base) || !al(cfg->orig_base) || !al(cfg->workspace))
    return fail(KVC_ERR_INVALID_ARG, "device buffers must be 256-byte aligned");
  const size_t need = ws_layout(cfg->b, cfg->H, cfg->d_head, cfg->rotary_dim, C).total;
  if (cfg->workspace_bytes < need)
    return fail(KVC_ERR_INVALID_ARG, "workspace_bytes=%zu < required %zu", cfg->workspace_bytes, need);
  kvc_cache* c = new (std::nothrow) kvc_cache(*cfg, C);
  if (!c) return fail(KVC_ERR_NO_MEMORY, "cache");
  c->cfg.seq_capacity = c->cap.data();
  *out = c;
  return ok();
}

void kvc_destroy(kvc_cache* cache) { delete cache; }

const kvc_book* kvc_get_book(const kvc_cache* cache) { return cache ? &cache->bk : nullptr; }

static kvc_status append_impl(kvc_cache* c, int layer, const void* k, const void* v, const int32_t* n_new,
                              const int32_t* pos, const uint8_t* kinds, void* stream_, bool free_in_block) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  const int M = c->cfg.M;
  if (layer < -1 || layer >= M) return fail(KVC_ERR_INVALID_ARG, "layer %d out of range [-1, %d)", layer, M);
  if (!k || !v) return fail(KVC_ERR_INVALID_ARG, "k/v are NULL");
  if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) & 15)
    return fail(KVC_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
  const bool starts = layer <= 0;
  if (starts) {
    if (c->layers_done != M)
      return fail(KVC_ERR_STATE, "layers %d..%d of the previous tokens are not written yet", c->layers_done, M - 1);
    if (!n_new) return fail(KVC_ERR_INVALID_ARG, "n_new is NULL");
    int64_t N = 0;
    for (int s = 0; s < c->cfg.b; ++s) N += n_new[s] > 0 ? n_new[s] : 0;
    if (N > 0 && !kinds) return fail(KVC_ERR_INVALID_ARG, "kinds is NULL");
    std::string err;
    int code = 0;
    if (!c->bk.book.check_append(n_new, kinds, err, code, free_in_block))
      return fail((kvc_status)code, "%s", err.c_str());
    if (N > 0 && !pos) return fail(KVC_ERR_INVALID_ARG, "pos is NULL");
  } else if (c->layers_done != layer) {
    return fail(KVC_ERR_STATE, "layer %d appended out of order (expected %d)", layer, c->layers_done);
  }
  kvc_status st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  const kvc::Geometry g = c->geom();
  if (starts) {
    int64_t N = 0;
    for (int s = 0; s < c->cfg.b; ++s) N += n_new[s];
    const bool local = c->cfg.policy == KVC_POLICY_LOCAL;
    std::vector<uint8_t> kept;
    if (free_in_block && !local) {
      c->bk.book.kept_in_block(n_new, kinds, kept);
    } else if (local) {  // a ring: only the last `capacity` new tokens of a sequence survive the call
      kept.assign((size_t)N, 1);
      int64_t o = 0;
      for (int s = 0; s < c->cfg.b; ++s) {
        for (int i = 0; i < n_new[s] - c->cap[s]; ++i) kept[o + i] = 0;
        o += n_new[s];
      }
    }
    const bool filtered = !kept.empty();
    int64_t n_plan = 0;
    for (int64_t t = 0; t < N; ++t) n_plan += filtered ? kept[t] : 1;
    // destination rows before the book moves on
    std::vector<int64_t> row0(c->cfg.b), orig0(c->cfg.b);
    for (int s = 0; s < c->cfg.b; ++s) {
      row0[s] = c->bk.book.stored(s);
      orig0[s] = c->bk.book.history(s);
    }
    const size_t bytes = c->ws.dyn_payload + sizeof(kvc::TokPlan) * (size_t)n_plan;
    cudaError_t e;
    unsigned char* img = c->ring.reserve(bytes, &e);
    if (!img) return cuda_fail(e, "staging");
    c->bk.book.apply_append(n_new, kinds, pos, (free_in_block && !local) ? kept.data() : nullptr);
    c->fill_state(img);
    kvc::TokPlan* tp = reinterpret_cast<kvc::TokPlan*>(img + c->ws.dyn_payload);
    int64_t t = 0, w = 0;
    for (int s = 0; s < c->cfg.b; ++s) {
      int64_t row = row0[s];
      for (int i = 0; i < n_new[s]; ++i, ++t) {
        if (filtered && !kept[t]) continue;  // freed as it is written (or overtaken in the ring): never stored
        tp[w].s = s;
        tp[w].row = local ? (int32_t)((orig0[s] + i) % c->cap[s]) : (int32_t)row++;
        tp[w].pos = pos[t];
        tp[w].orig = (int32_t)(orig0[s] + i);
        tp[w].in_tok = (int32_t)t;
        tp[w].pad0 = tp[w].pad1 = tp[w].pad2 = 0;
        ++w;
      }
    }
    e = c->ring.commit(c->wsp(c->ws.dyn), bytes, stream);
    if (e != cudaSuccess) return cuda_fail(e, "upload append plan");
    c->batch_ntok = n_plan;
    c->batch_nin = N;
    c->layers_done = 0;
  }
  const int m0 = layer < 0 ? 0 : layer;
  const int nl = layer < 0 ? M : 1;
  if (c->batch_ntok > 0) {
    const kvc::TokPlan* plan = reinterpret_cast<const kvc::TokPlan*>(c->wsp(c->ws.dyn + c->ws.dyn_payload));
    cudaError_t e = kvc::launch_append(g, c->stat(), c->bufs(), plan, c->batch_ntok, c->batch_nin, m0, nl, m0 == 0, k,
                                       v, c->amaps_ok ? c->wsp(c->ws.amaps) : nullptr, c->num_sms, 2000000000ull,
                                       stream);
    if (e != cudaSuccess) return cuda_fail(e, "append kernel");
    c->launches += 1;
    c->last_was_decode = false;
  }
  c->layers_done = m0 + nl;
  return ok();
}

kvc_status kvc_append(kvc_cache* c, int layer, const void* k, const void* v, const int32_t* n_new, const int32_t* pos,
                      const uint8_t* kinds, void* stream) {
  return append_impl(c, layer, k, v, n_new, pos, kinds, stream, false);
}

kvc_status kvc_append_free_closed(kvc_cache* c, int layer, const void* k, const void* v, const int32_t* n_new,
                                  const int32_t* pos, const uint8_t* kinds, void* stream) {
  return append_impl(c, layer, k, v, n_new, pos, kinds, stream, true);
}

kvc_status kvc_compress_spans(kvc_cache* c, const int32_t* seq, const int64_t* cl, const int64_t* cr, int n_spans,
                              void* stream_) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  if (n_spans < 0 || (n_spans > 0 && (!seq || !cl || !cr))) return fail(KVC_ERR_INVALID_ARG, "span arrays");
  if (c->layers_done != c->cfg.M)
    return fail(KVC_ERR_STATE, "layers %d..%d of the last tokens are not written yet", c->layers_done, c->cfg.M - 1);
  std::vector<kvc::CompactSeq> plan;
  std::string err;
  if (!c->bk.book.plan_compress(seq, cl, cr, n_spans, plan, err)) return fail(KVC_ERR_SPAN, "%s", err.c_str());
  if (n_spans == 0) return ok();
  kvc_status st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  size_t n_ranges = 0;
  int n_aff = 0;
  for (auto& p : plan)
    if (!p.drops.empty()) {
      n_ranges += p.drops.size();
      ++n_aff;
    }
  const size_t aff_bytes = sizeof(kvc::AffSeq) * (size_t)n_aff;
  const size_t bytes = c->ws.dyn_payload + aff_bytes + 8 * n_ranges;
  cudaError_t e;
  unsigned char* img = c->ring.reserve(bytes, &e);
  if (!img) return cuda_fail(e, "staging");
  c->bk.book.apply_compress(plan, seq, cl, n_spans);
  c->fill_state(img);
  kvc::AffSeq* aff = reinterpret_cast<kvc::AffSeq*>(img + c->ws.dyn_payload);
  int32_t* rg = reinterpret_cast<int32_t*>(img + c->ws.dyn_payload + aff_bytes);
  int a = 0;
  int32_t ro = 0;
  for (auto& p : plan) {
    if (p.drops.empty()) continue;
    aff[a].s = p.s;
    aff[a].len_old = (int32_t)p.len_old;
    aff[a].len_new = (int32_t)p.len_new;
    aff[a].first_row = (int32_t)p.first_row;
    aff[a].range_off = ro;
    aff[a].n_ranges = (int32_t)p.drops.size();
    aff[a].pad0 = aff[a].pad1 = 0;
    for (auto& d : p.drops) {
      rg[2 * ro] = (int32_t)d.first;
      rg[2 * ro + 1] = (int32_t)d.second;
      ++ro;
    }
    ++a;
  }
  e = c->ring.commit(c->wsp(c->ws.dyn), bytes, stream);
  if (e != cudaSuccess) return cuda_fail(e, "upload compaction plan");
  int launched = 0;
  const bool timed = c->time_compaction && n_aff > 0;
  c->timed_compaction = false;
  if (timed) {
    for (auto& ev : c->cev)
      if (!ev && (e = cudaEventCreate(&ev)) != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
    if ((e = cudaEventRecord(c->cev[0], stream)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
  }
  e = kvc::launch_compact(c->geom(), c->stat(), c->bufs(),
                          reinterpret_cast<const kvc::AffSeq*>(c->wsp(c->ws.dyn + c->ws.dyn_payload)), n_aff,
                          reinterpret_cast<const int32_t*>(c->wsp(c->ws.dyn + c->ws.dyn_payload + aff_bytes)),
                          reinterpret_cast<int32_t*>(c->wsp(c->ws.src_map)), stream, &launched,
                          timed ? c->cev[1] : nullptr);
  c->launches += launched;
  c->last_was_decode = false;
  if (e != cudaSuccess) return cuda_fail(e, "compaction kernels");
  if (timed) {
    if ((e = cudaEventRecord(c->cev[2], stream)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    c->timed_compaction = true;
  }
  return ok();
}

// Checks shared by the decode entry points, for layers [layer, layer + n_layers).
static kvc_status decode_check(kvc_cache* c, int layer, int n_layers, const void* q, float scale, float* out) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  if (n_layers < 1 || layer < 0 || layer + n_layers > c->cfg.M)
    return fail(KVC_ERR_INVALID_ARG, "layers [%d, %d) out of range [0, %d)", layer, layer + n_layers, c->cfg.M);
  if (!q || !out) return fail(KVC_ERR_INVALID_ARG, "q/out are NULL");
  if (!std::isfinite(scale)) return fail(KVC_ERR_INVALID_ARG, "scale is not finite");
  if (layer + n_layers > c->layers_done)
    return fail(KVC_ERR_STATE, "layer %d of the last tokens is not written yet", std::max(layer, c->layers_done));
  if (!c->cuda_ready) return fail(KVC_ERR_STATE, "nothing appended yet");
  if (!c->decode_ok) return fail(KVC_ERR_STATE, "%s", c->decode_err.c_str());
  if (c->R <= 0) return fail(KVC_ERR_STATE, "no sequence has a token to query");
  return KVC_OK;
}

static kvc::DecodeArgs decode_args(kvc_cache* c, int layer, const void* q, float scale, float* out) {
  kvc::DecodeArgs a;
  a.layer = layer;
  a.dstate = reinterpret_cast<const kvc::DState*>(c->wsp(c->ws.dyn));
  a.P = reinterpret_cast<const int64_t*>(c->wsp(c->ws.dyn + c->ws.dyn_P));
  a.R = c->R;
  a.q = q;
  a.out = out;
  a.scale = scale;
  a.partials = reinterpret_cast<float*>(c->wsp(c->ws.partials));
  a.counters = reinterpret_cast<int*>(c->wsp(c->ws.counters));
  a.wait_limit_ns = 2000000000ull;
  a.kv_before_wait = c->last_was_decode ? 1 : 0;
  a.n_segments = c->n_segments;
  a.max_segment = c->max_segment;
  return a;
}

kvc_status kvc_decode_attention(kvc_cache* c, int layer, const void* q, float scale, float* out, void* stream_) {
  kvc_status st = decode_check(c, layer, 1, q, scale, out);
  if (st != KVC_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  const kvc::DecodeArgs a = decode_args(c, layer, q, scale, out);
  int grid = 0;
  cudaError_t e = kvc::launch_decode(c->geom(), c->stat(), c->bufs(), a, c->num_sms, stream, &grid, &c->last_plan);
  if (e != cudaSuccess) return cuda_fail(e, "decode kernel");
  c->launches += grid > 0 ? 1 : 0;
  c->last_was_decode = true;
  return ok();
}

kvc_status kvc_decode_attention_layers(kvc_cache* c, int first, int n_layers, const void* q, int64_t q_layer_stride,
                                       float scale, float* out, int64_t out_layer_stride, void* stream_) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  if (n_layers < 0 || first < 0 || first + n_layers > c->cfg.M)
    return fail(KVC_ERR_INVALID_ARG, "layers [%d, %d) out of range [0, %d)", first, first + n_layers, c->cfg.M);
  if (n_layers == 0) return ok();
  const int64_t need = (int64_t)c->cfg.b * c->cfg.H * c->cfg.d_head;
  if (n_layers > 1 && (q_layer_stride < need || out_layer_stride < need))
    return fail(KVC_ERR_INVALID_ARG, "layer strides (%lld, %lld) below one layer's %lld elements",
                (long long)q_layer_stride, (long long)out_layer_stride, (long long)need);
  kvc_status st = decode_check(c, first, n_layers, q, scale, out);
  if (st != KVC_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  if (n_layers > 1) {
    // whole segments: every layer's in one launch (no per-launch prologue and drain per layer)
    kvc::DecodeArgs a = decode_args(c, first, q, scale, out);
    a.n_layers = n_layers;
    a.q_layer_stride = q_layer_stride;
    a.out_layer_stride = out_layer_stride;
    int grid = 0;
    kvc::DecodePlan plan{-1, 0, 0, 0};
    cudaError_t e = kvc::launch_decode(c->geom(), c->stat(), c->bufs(), a, c->num_sms, stream, &grid, &plan);
    if (e == cudaSuccess) {
      c->last_plan = plan;
      c->launches += grid > 0 ? 1 : 0;
      c->last_was_decode = true;
      return ok();
    }
    if (e != cudaErrorNotSupported) return cuda_fail(e, "decode kernel (layers)");
  }
  // segments too long to be taken whole (split over a wave of warps per layer): one launch per layer
  const uint16_t* qp = static_cast<const uint16_t*>(q);
  for (int i = 0; i < n_layers; ++i) {
    st = kvc_decode_attention(c, first + i, qp + i * q_layer_stride, scale, out + i * out_layer_stride, stream);
    if (st != KVC_OK) return st;
  }
  return ok();
}

kvc_status kvc_decode_attention_static_scratch(kvc_cache* c, int layer, const void* q, float scale, float* out,
                                               void* stream_) {
  kvc_status st0 = decode_check(c, layer, 1, q, scale, out);
  if (st0 != KVC_OK) return st0;
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  // split-K partials for every possible worker and segment, then one arrival counter per segment
  const size_t segs = (size_t)c->cfg.b * c->cfg.H;
  const size_t part_bytes = align_up(4 * ((size_t)kvc::kMaxDecodeWorkers + segs) * (size_t)(c->cfg.d_head + 4), 256);
  const size_t need = part_bytes + 4 * segs;
  if (need > kvc::kStaticDecodeScratchBytes)
    return fail(KVC_ERR_UNSUPPORTED,
                "b*H=%zu with d_head=%d needs %zu bytes of split-K scratch; the static array holds %zu "
                "(use kvc_decode_attention with the cache workspace)",
                segs, c->cfg.d_head, need, kvc::kStaticDecodeScratchBytes);
  kvc_status st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  void* scratch = nullptr;
  cudaError_t e = kvc::static_decode_scratch(&scratch);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress (static decode scratch)");
  int* counters = reinterpret_cast<int*>(static_cast<unsigned char*>(scratch) + part_bytes);
  // the array keeps the previous call's contents: the arrival counters must start from zero
  e = cudaMemsetAsync(counters, 0, 4 * segs, stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync (static decode scratch)");
  kvc::DecodeArgs a;
  a.layer = layer;
  a.dstate = reinterpret_cast<const kvc::DState*>(c->wsp(c->ws.dyn));
  a.P = reinterpret_cast<const int64_t*>(c->wsp(c->ws.dyn + c->ws.dyn_P));
  a.R = c->R;
  a.q = q;
  a.out = out;
  a.scale = scale;
  a.partials = static_cast<float*>(scratch);
  a.counters = counters;
  a.wait_limit_ns = 2000000000ull;
  a.kv_before_wait = 0;
  a.n_segments = c->n_segments;
  a.max_segment = c->max_segment;
  int grid = 0;
  e = kvc::launch_decode(c->geom(), c->stat(), c->bufs(), a, c->num_sms, stream, &grid, &c->last_plan);
  if (e != cudaSuccess) return cuda_fail(e, "decode kernel (static scratch)");
  c->launches += grid > 0 ? 1 : 0;
  c->last_was_decode = true;
  return ok();
}

kvc_status kvc_prefill_attention(kvc_cache* c, int layer, const void* q, const int32_t* n_q, float scale, float* out,
                                 void* stream_) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  const int b = c->cfg.b, H = c->cfg.H, D = c->cfg.d_head;
  if (layer < 0 || layer >= c->cfg.M) return fail(KVC_ERR_INVALID_ARG, "layer %d out of range", layer);
  if (!q || !out || !n_q) return fail(KVC_ERR_INVALID_ARG, "q/out/n_q are NULL");
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(KVC_ERR_INVALID_ARG, "q and out must be 16-byte aligned");
  if (!(scale > 0.0f) || !std::isfinite(scale)) return fail(KVC_ERR_INVALID_ARG, "scale must be positive and finite");
  if (c->cfg.policy == KVC_POLICY_LOCAL)
    return fail(KVC_ERR_UNSUPPORTED, "masked prefill is not defined for the local-attention cache");
  if ((int64_t)c->cfg.M * H * c->C >= ((int64_t)1 << 31))
    return fail(KVC_ERR_UNSUPPORTED, "M*H*sum(capacity) rows exceed the 2^31 rows a tensor-map coordinate reaches");
  if (layer >= c->layers_done) return fail(KVC_ERR_STATE, "layer %d of the last tokens is not written yet", layer);
  for (int s = 0; s < b; ++s)
    if (n_q[s] < 0 || n_q[s] > c->bk.book.history(s))
      return fail(KVC_ERR_INVALID_ARG, "n_q[%d] = %d outside [0, %lld]", s, n_q[s],
                  (long long)c->bk.book.history(s));
  if (!c->cuda_ready) return fail(KVC_ERR_STATE, "nothing appended yet");
  kvc_status st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  cudaError_t e;
  if (!c->maps.ready) {
    e = kvc::encode_prefill_maps(c->geom(), c->bufs(), &c->maps);
    if (e != cudaSuccess) return cuda_fail(e, "cuTensorMapEncodeTiled (K/V planes)");
  }
  const bool same = c->pre_version == c->version && std::equal(c->pre_nq.begin(), c->pre_nq.end(), n_q) &&
                    (int)c->pre_nq.size() == b;
  if (!same) {
    // per-sequence state, tile prefix and per-row mask bounds
    std::vector<std::vector<int32_t>> metas(b);
    size_t n_meta = 0;
    for (int s = 0; s < b; ++s) {
      std::string err;
      if (!c->bk.book.prefill_keys(s, n_q[s], metas[s], err)) return fail(KVC_ERR_STATE, "%s", err.c_str());
      n_meta += metas[s].size();
    }
    const size_t bytes = c->ws.pre_meta + 4 * n_meta;
    unsigned char* img = c->ring.reserve(bytes, &e);
    if (!img) return e != cudaSuccess ? cuda_fail(e, "staging") : fail(KVC_ERR_INVALID_ARG, "prefill plan exceeds ring");
    std::vector<kvc::PState> ps(b);
    std::vector<int32_t> Pq(b + 1);
    int32_t* meta = reinterpret_cast<int32_t*>(img + c->ws.pre_meta);
    int64_t qtok = 0, moff = 0;
    Pq[0] = 0;
    for (int s = 0; s < b; ++s) {
      const int64_t len = c->bk.book.stored(s);
      ps[s].len = (int32_t)len;
      ps[s].q0 = (int32_t)(len - n_q[s]);
      ps[s].qtok = (int32_t)qtok;
      ps[s].moff = (int32_t)moff;
      std::memcpy(meta + moff, metas[s].data(), 4 * metas[s].size());
      moff += (int64_t)metas[s].size();
      qtok += n_q[s];
      Pq[s + 1] = Pq[s] + (n_q[s] + 127) / 128;
    }
    // Work items (sequence, head, query tile) in the kernel's order: sequence (longest first), head,
    // the tile with the most keys first.
    const int64_t n_items = (int64_t)H * Pq[b];
    if (n_items > c->ws.pre_max_items) return fail(KVC_ERR_INVALID_ARG, "prefill work items exceed the plan");
    // a persistent grid: every SM's CTAs, which take the items in this order from the launch's
    // counter, so the items in flight at any time are neighbours sharing K/V tiles in L2
    const int G = (int)std::min<int64_t>(
        std::min(c->num_sms * kvc::prefill_ctas_per_sm(c->cfg.d_head), kvc::kMaxPrefillCtas), n_items);
    {
      // sequences with the most stored rows first, so the heaviest items are taken early and the
      // last ones taken are short
      std::vector<int> order(b);
      for (int s = 0; s < b; ++s) order[s] = s;
      std::stable_sort(order.begin(), order.end(), [&](int x, int y) { return ps[x].len > ps[y].len; });
      kvc::PfItemRec* items = reinterpret_cast<kvc::PfItemRec*>(img + c->ws.pre_items);
      int64_t item = 0;
      for (int s : order) {
        const int nqt = Pq[s + 1] - Pq[s];
        for (int h = 0; h < H; ++h)
          for (int k = 0; k < nqt; ++k, ++item) {
            kvc::PfItemRec& r = items[item];
            const int qt = nqt - 1 - k;
            r.ps = ps[s];
            r.s = s;
            r.h = h;
            r.qr0 = ps[s].q0 + 128 * qt;
            r.qr_end = std::min(r.qr0 + 128, ps[s].len);
            r.nk = (r.qr_end + 127) / 128;
            const int64_t row0 = (int64_t)H * c->off[s] + (int64_t)h * c->cap[s];  // = seq_row0[s] + h * cap[s]
            r.row0_lo = (int32_t)(uint32_t)(uint64_t)row0;
            r.row0_hi = (int32_t)((uint64_t)row0 >> 32);
            r.pad = 0;
          }
      }
    }
    c->pre_ctas = G;
    e = c->ring.commit(c->wsp(c->ws.pre), bytes, stream);
    if (e != cudaSuccess) return cuda_fail(e, "upload prefill plan");
    c->pre_version = c->version;
    c->pre_nq.assign(n_q, n_q + b);
    c->pre_tiles = Pq[b];
  }
  if (c->pre_tiles == 0) return ok();
  kvc::PrefillArgs a;
  a.layer = layer;
  a.H = H;
  a.rot = c->cfg.rotary_dim;
  a.C = c->C;
  a.items = reinterpret_cast<const kvc::PfItemRec*>(c->wsp(c->ws.pre + c->ws.pre_items));
  a.meta = reinterpret_cast<const int32_t*>(c->wsp(c->ws.pre + c->ws.pre_meta));
  a.q = static_cast<const uint16_t*>(q);
  a.out = out;
  a.n_qtok = 0;
  for (int s = 0; s < b; ++s) a.n_qtok += n_q[s];
  a.c2 = (float)((double)scale * 1.4426950408889634);
  a.pos = c->cfg.pos_base;
  const kvc::Static sta = c->stat();
  a.off = sta.off;
  a.rope_g = sta.rope_g;
  a.status = c->bufs().status;
  a.wait_limit_ns = 2000000000ull;
  (void)D;
  a.n_items = (int64_t)H * c->pre_tiles;
  a.item_counter = reinterpret_cast<unsigned long long*>(c->wsp(c->ws.pre_counter));
  a.n_ctas = c->pre_ctas;
  e = cudaMemsetAsync(a.item_counter, 0, sizeof(unsigned long long), stream);
  if (e != cudaSuccess) return cuda_fail(e, "reset the prefill item counter");
  e = kvc::launch_prefill(c->geom(), c->maps, a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "prefill kernel");
  c->launches += 1;
  c->last_was_decode = false;
  return ok();
}

kvc_status kvc_masked_reference_layout(kvc_cache* c, int seq, int64_t cap, uint8_t* kind_full, int32_t* pos_full,
                                       uint8_t* visible_full, int64_t* n_full, int32_t* stored_orig_idx,
                                       int32_t* stored_pos, int64_t* n_stored, void* stream_) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  int64_t ns = 0;
  kvc_status st = kvc_book_layout(&c->bk, seq, cap, kind_full, pos_full, visible_full, n_full, nullptr, nullptr, &ns);
  if (st != KVC_OK) return st;
  *n_stored = ns;
  if (ns == 0) return ok();
  st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  cudaError_t e = cudaSuccess;
  if (c->cfg.policy == KVC_POLICY_LOCAL) {  // the window, oldest first, out of the ring
    const int64_t cap = c->cap[seq];
    std::vector<int32_t> o((size_t)cap), p((size_t)cap);
    e = cudaMemcpyAsync(o.data(), c->cfg.orig_base + c->off[seq], 4 * (size_t)cap, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(p.data(), c->cfg.pos_base + c->off[seq], 4 * (size_t)cap, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, "read back stored rows");
    const int64_t T = c->bk.book.history(seq);
    const int64_t first = c->bk.book.local_first(T - 1);
    for (int64_t k = 0; k < ns; ++k) {
      const int64_t slot = (first + k) % cap;
      if (stored_orig_idx) stored_orig_idx[k] = o[(size_t)slot];
      if (stored_pos) stored_pos[k] = p[(size_t)slot];
    }
    return ok();
  }
  if (stored_orig_idx)
    e = cudaMemcpyAsync(stored_orig_idx, c->cfg.orig_base + c->off[seq], 4 * (size_t)ns, cudaMemcpyDeviceToHost,
                        stream);
  if (e == cudaSuccess && stored_pos)
    e = cudaMemcpyAsync(stored_pos, c->cfg.pos_base + c->off[seq], 4 * (size_t)ns, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "read back stored rows");
  return ok();
}

kvc_status kvc_device_status(kvc_cache* c, void* stream_, int32_t* word) {
  if (!c || !word) return fail(KVC_ERR_INVALID_ARG, "NULL argument");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  *word = 0;
  if (!c->cuda_ready) return ok();
  int32_t w = 0;
  cudaError_t e = cudaMemcpyAsync(&w, c->wsp(c->ws.hdr), 4, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "read status");
  *word = w;
  if (w == 0) return ok();
  e = cudaMemsetAsync(c->wsp(c->ws.hdr), 0, 4, stream);
  // a timed-out decode may leave split-K arrival counters behind: start them from zero again
  if (e == cudaSuccess && (w & kvc::STATUS_TIMEOUT))
    e = cudaMemsetAsync(c->wsp(c->ws.counters), 0, 4 * (size_t)c->cfg.b * c->cfg.H, stream);
  if (e != cudaSuccess) return cuda_fail(e, "clear status");
  if (w & kvc::STATUS_TIMEOUT) return fail(KVC_ERR_TIMEOUT, "a kernel's bounded wait ran out (status 0x%x)", w);
  return fail(KVC_ERR_DEVICE_CHECK, "a kernel's consistency check failed (status 0x%x)", w);
}

kvc_status kvc_check_bounded_wait(kvc_cache* c, uint64_t limit_ns, void* stream_) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  if (limit_ns == 0 || limit_ns > 2000000000ull)
    return fail(KVC_ERR_INVALID_ARG, "limit_ns=%llu must be in (0, 2e9]", (unsigned long long)limit_ns);
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  kvc_status st = c->ensure_cuda(stream);
  if (st != KVC_OK) return st;
  cudaError_t e = kvc::launch_bounded_wait_check(reinterpret_cast<int*>(c->wsp(c->ws.hdr)), limit_ns, stream);
  if (e != cudaSuccess) return cuda_fail(e, "bounded-wait check kernel");
  c->launches += 1;
  c->last_was_decode = false;
  return ok();
}

int64_t kvc_launch_count(const kvc_cache* c) { return c ? c->launches : 0; }

kvc_status kvc_set_compaction_timing(kvc_cache* c, int enable) {
  if (!c) return fail(KVC_ERR_INVALID_ARG, "cache is NULL");
  c->time_compaction = enable != 0;
  return ok();
}

kvc_status kvc_last_compaction_ms(kvc_cache* c, float* scan_ms, float* move_ms) {
  if (!c || !scan_ms || !move_ms) return fail(KVC_ERR_INVALID_ARG, "cache or outputs are NULL");
  if (!c->timed_compaction) return fail(KVC_ERR_STATE, "the last compaction was not timed");
  cudaError_t e = cudaEventSynchronize(c->cev[2]);
  if (e == cudaSuccess) e = cudaEventElapsedTime(scan_ms, c->cev[0], c->cev[1]);
  if (e == cudaSuccess) e = cudaEventElapsedTime(move_ms, c->cev[1], c->cev[2]);
  if (e != cudaSuccess) return cuda_fail(e, "compaction timing events");
  return ok();
}

kvc_status kvc_last_decode_plan(const kvc_cache* c, int32_t* plan) {
  if (!c || !plan) return fail(KVC_ERR_INVALID_ARG, "NULL argument");
  plan[0] = c->last_plan.mode;
  plan[1] = c->last_plan.workers;
  plan[2] = c->last_plan.tile_rows;
  plan[3] = c->last_plan.stages;
  return ok();
}

}  // extern "C"
