// Host-side span bookkeeping (see book.hpp).
#include "book.hpp"

#include <algorithm>
#include <cmath>
#include <cstdio>

namespace kvc {

Book::Book(int b, Policy policy, const int64_t* capacity, double local_ratio)
    : b_(b), policy_(policy), local_ratio_(local_ratio), seqs_(b) {
  for (int s = 0; s < b; ++s) {
    seqs_[s].cap = capacity[s];
    seqs_[s].freed_before.push_back(0);
  }
}

bool Book::check_append(const int32_t* n_new, const uint8_t* kinds, std::string& err, int& code,
                        bool free_in_block, bool check_capacity) const {
  int64_t off = 0;
  char buf[256];
  for (int s = 0; s < b_; ++s) {
    if (n_new[s] < 0) {
      std::snprintf(buf, sizeof buf, "n_new[%d] = %d is negative", s, n_new[s]);
      err = buf;
      code = 1;
      return false;
    }
  }
  // kinds first (the kept count below relies on well-formed spans), then capacity
  for (int s = 0; s < b_; ++s) {
    const Seq& q = seqs_[s];
    bool open = q.open;
    for (int t = 0; t < n_new[s]; ++t) {
      uint8_t k = kinds[off + t];
      if (k > CR) {
        std::snprintf(buf, sizeof buf, "sequence %d token %d: kind %u is not NORMAL/CL/CR", s, t, k);
        err = buf;
        code = 1;
        return false;
      }
      if (k != NORMAL && policy_ == POLICY_LOCAL) {
        std::snprintf(buf, sizeof buf, "sequence %d token %d: sentinel kinds are not used by the local-attention "
                      "cache", s, t);
        err = buf;
        code = 4;
        return false;
      }
      if (k == CL) {
        if (open) {
          std::snprintf(buf, sizeof buf, "sequence %d token %d: <CL> inside an open span (spans may not nest)", s,
                        t);
          err = buf;
          code = 4;
          return false;
        }
        open = true;
      } else if (k == CR) {
        if (!open) {
          std::snprintf(buf, sizeof buf, "sequence %d token %d: <CR> without an open <CL>", s, t);
          err = buf;
          code = 4;
          return false;
        }
        open = false;
      }
    }
    off += n_new[s];
  }
  if (!check_capacity) return true;
  std::vector<uint8_t> kept;
  if (free_in_block) kept_in_block(n_new, kinds, kept);
  off = 0;
  for (int s = 0; s < b_; ++s) {
    const Seq& q = seqs_[s];
    int64_t stored_new = n_new[s];
    if (free_in_block) {
      stored_new = 0;
      for (int t = 0; t < n_new[s]; ++t) stored_new += kept[off + t];
    }
    if (policy_ == POLICY_LOCAL) {
      const int64_t T = (int64_t)q.kind.size() + n_new[s];
      const int64_t window = T > 0 ? T - local_first(T - 1) : 0;
      if (window > q.cap) {
        std::snprintf(buf, sizeof buf, "sequence %d: the local window of %lld rows exceeds capacity %lld", s,
                      (long long)window, (long long)q.cap);
        err = buf;
        code = 3;
        return false;
      }
    } else if (q.stored + stored_new > q.cap) {
      std::snprintf(buf, sizeof buf, "sequence %d: %lld stored + %lld new rows exceed capacity %lld", s,
                    (long long)q.stored, (long long)stored_new, (long long)q.cap);
      err = buf;
      code = 3;
      return false;
    }
    if (q.kind.size() + (size_t)n_new[s] >= (size_t)INT32_MAX) {
      err = "history index would overflow int32";
      code = 3;
      return false;
    }
    off += n_new[s];
  }
  return true;
}

void Book::kept_in_block(const int32_t* n_new, const uint8_t* kinds, std::vector<uint8_t>& kept) const {
  int64_t total = 0;
  for (int s = 0; s < b_; ++s) total += n_new[s];
  kept.assign((size_t)total, 1);
  int64_t off = 0;
  for (int s = 0; s < b_; ++s) {
    int64_t open_at = -1;  // index (within this call) of a <CL> opened by these tokens
    for (int t = 0; t < n_new[s]; ++t) {
      const uint8_t k = kinds[off + t];
      if (k == CL) {
        open_at = t;
      } else if (k == CR && open_at >= 0) {  // opened and closed here: free <CL> (paper) and the interior
        const int64_t lo = policy_ == POLICY_PAPER ? open_at : open_at + 1;
        for (int64_t u = lo; u < t; ++u) kept[off + u] = 0;
        open_at = -1;
      } else if (k == CR) {
        open_at = -1;  // closes a span opened before this call: stored, freed later by compaction
      }
    }
    off += n_new[s];
  }
}

void Book::next_positions(const int32_t* n_new, const uint8_t* kinds, int32_t* pos_out) const {
  int64_t off = 0;
  for (int s = 0; s < b_; ++s) {
    const Seq& q = seqs_[s];
    int64_t normals = q.normals;
    bool have_prev = !q.pos.empty();
    int32_t prev = have_prev ? q.pos.back() : 0;
    for (int t = 0; t < n_new[s]; ++t) {
      int32_t p;
      if (kinds[off + t] == NORMAL) {
        p = (int32_t)normals;  // the next unused position
        normals += 1;
      } else {
        p = have_prev ? prev : 0;  // tied to the previous token
      }
      pos_out[off + t] = p;
      prev = p;
      have_prev = true;
    }
    off += n_new[s];
  }
}

void Book::apply_append(const int32_t* n_new, const uint8_t* kinds, const int32_t* pos, const uint8_t* kept) {
  int64_t off = 0;
  for (int s = 0; s < b_; ++s) {
    Seq& q = seqs_[s];
    const int64_t T0 = (int64_t)q.kind.size();
    int64_t stored_new = 0;
    bool freed_any = false;
    for (int t = 0; t < n_new[s]; ++t) {
      uint8_t k = kinds[off + t];
      int64_t j = (int64_t)q.kind.size();
      q.kind.push_back(k);
      q.pos.push_back(pos[off + t]);
      stored_new += kept ? kept[off + t] : 1;
      if (k == NORMAL) {
        q.normals += 1;
      } else if (k == CL) {
        Span sp;
        sp.cl = j;
        q.spans.push_back(sp);
        q.open = true;
      } else {
        Span& sp = q.spans.back();
        sp.cr = j;
        q.open = false;
        if (kept && sp.cl >= T0) {  // opened and closed in this call: freed as it was written
          sp.freed = true;
          const int64_t lo = policy_ == POLICY_PAPER ? sp.cl : sp.cl + 1;
          if (lo < sp.cr) q.freed.emplace_back(lo, sp.cr);
          freed_any = true;
        }
      }
    }
    if (freed_any) rebuild_prefix(q);
    if (policy_ == POLICY_LOCAL) {
      const int64_t T = (int64_t)q.kind.size();
      q.stored = T > 0 ? T - local_first(T - 1) : 0;  // the window of the last token
    } else {
      q.stored += stored_new;
    }
    off += n_new[s];
  }
}

int64_t Book::local_first(int64_t t) const {
  // x_{t+1} (1-based) attends within (floor((t+1) r), t+1]: 0-based indices floor((t+1) r) .. t
  return (int64_t)std::floor((double)(t + 1) * local_ratio_);
}

int Book::find_span(const Seq& q, int64_t cl) const {
  auto it = std::lower_bound(q.spans.begin(), q.spans.end(), cl,
                             [](const Span& a, int64_t v) { return a.cl < v; });
  if (it == q.spans.end() || it->cl != cl) return -1;
  return (int)(it - q.spans.begin());
}

int64_t Book::stored_index(int s, int64_t j) const {
  const Seq& q = seqs_[s];
  // freed ranges are sorted and disjoint: count freed rows before j
  auto it = std::upper_bound(q.freed.begin(), q.freed.end(), std::make_pair(j, INT64_MAX));
  size_t k = (size_t)(it - q.freed.begin());  // ranges with lo <= j
  if (k > 0 && j < q.freed[k - 1].second) return -1;
  return j - q.freed_before[k];
}

void Book::rebuild_prefix(Seq& q) {
  std::sort(q.freed.begin(), q.freed.end());
  q.freed_before.assign(q.freed.size() + 1, 0);
  for (size_t k = 0; k < q.freed.size(); ++k)
    q.freed_before[k + 1] = q.freed_before[k] + (q.freed[k].second - q.freed[k].first);
}

bool Book::plan_compress(const int32_t* seq, const int64_t* cl, const int64_t* cr, int n,
                         std::vector<CompactSeq>& plan, std::string& err) const {
  char buf[256];
  std::vector<int> slot(b_, -1);
  std::vector<std::vector<int64_t>> listed(b_);
  plan.clear();
  for (int i = 0; i < n; ++i) {
    int s = seq[i];
    if (s < 0 || s >= b_) {
      std::snprintf(buf, sizeof buf, "span %d: sequence %d out of range", i, s);
      err = buf;
      return false;
    }
    const Seq& q = seqs_[s];
    int k = find_span(q, cl[i]);
    if (k < 0 || q.spans[k].cr < 0 || q.spans[k].cr != cr[i]) {
      std::snprintf(buf, sizeof buf, "span %d: (%lld, %lld) of sequence %d is not a closed <CL>..<CR> span", i,
                    (long long)cl[i], (long long)cr[i], s);
      err = buf;
      return false;
    }
    if (q.spans[k].freed) {
      std::snprintf(buf, sizeof buf, "span %d: (%lld, %lld) of sequence %d is already freed", i, (long long)cl[i],
                    (long long)cr[i], s);
      err = buf;
      return false;
    }
    for (int64_t c : listed[s]) {
      if (c == cl[i]) {
        std::snprintf(buf, sizeof buf, "span %d: (%lld, %lld) of sequence %d is listed twice", i, (long long)cl[i],
                      (long long)cr[i], s);
        err = buf;
        return false;
      }
    }
    listed[s].push_back(cl[i]);
    if (slot[s] < 0) {
      slot[s] = (int)plan.size();
      CompactSeq c;
      c.s = s;
      c.len_old = q.stored;
      plan.push_back(c);
    }
    int64_t lo = policy_ == POLICY_PAPER ? cl[i] : cl[i] + 1;
    if (lo < cr[i]) plan[slot[s]].drops.emplace_back(lo, cr[i]);
  }
  for (CompactSeq& c : plan) {
    std::sort(c.drops.begin(), c.drops.end());
    int64_t dropped = 0;
    c.first_row = c.len_old;
    for (auto& d : c.drops) {
      dropped += d.second - d.first;
      c.first_row = std::min(c.first_row, stored_index(c.s, d.first));
    }
    c.len_new = c.len_old - dropped;
  }
  return true;
}

void Book::apply_compress(const std::vector<CompactSeq>& plan, const int32_t* seq, const int64_t* cl, int n) {
  for (int i = 0; i < n; ++i) {
    Seq& q = seqs_[seq[i]];
    int k = find_span(q, cl[i]);
    q.spans[k].freed = true;
  }
  for (const CompactSeq& c : plan) {
    Seq& q = seqs_[c.s];
    for (auto& d : c.drops) q.freed.push_back(d);
    rebuild_prefix(q);
    q.stored = c.len_new;
  }
}

bool Book::decode_view(int s, DecodeView& v, std::string& err) const {
  const Seq& q = seqs_[s];
  char buf[256];
  if (q.kind.empty()) {
    std::snprintf(buf, sizeof buf, "sequence %d has no token to query", s);
    err = buf;
    return false;
  }
  const int64_t tq = (int64_t)q.kind.size() - 1;
  v.len = q.stored;
  v.qpos = q.pos.back();
  v.mask_lo = v.mask_hi = 0;
  v.wrap = INT64_MAX;
  if (policy_ == POLICY_LOCAL) {  // the window [first, tq] in ring slots
    const int64_t first = local_first(tq);
    v.begin = first % q.cap;
    v.len = v.begin + (tq - first + 1);
    v.wrap = q.cap - v.begin;
    return true;
  }
  if (q.kind[tq] == CL) {  // a <CL> attends only to itself (Sec. 3.1)
    v.begin = q.stored - 1;
    return true;
  }
  v.begin = 0;
  // stored rows hidden from the query: history ranges of spans that are not freed
  std::vector<std::pair<int64_t, int64_t>> hid;
  for (const Span& sp : q.spans) {
    if (sp.freed) continue;
    if (sp.cr >= 0 && sp.cr < tq) {  // closed before the query: interior hidden (and <CL> under the paper policy)
      int64_t lo = policy_ == POLICY_PAPER ? sp.cl : sp.cl + 1;
      if (lo < sp.cr) hid.emplace_back(lo, sp.cr);
    } else if (policy_ == POLICY_PAPER) {  // open, or closed by the query itself: only <CL> hidden
      hid.emplace_back(sp.cl, sp.cl + 1);
    }
  }
  if (hid.empty()) return true;
  std::vector<std::pair<int64_t, int64_t>> rows;
  for (auto& h : hid) {
    int64_t a = stored_index(s, h.first);
    rows.emplace_back(a, a + (h.second - h.first));
  }
  std::sort(rows.begin(), rows.end());
  int64_t lo = rows[0].first, hi = rows[0].second;
  for (size_t k = 1; k < rows.size(); ++k) {
    if (rows[k].first > hi) {
      std::snprintf(buf, sizeof buf,
                    "sequence %d: rows hidden from the query form more than one run; free the closed spans "
                    "(kvc_compress_spans) before decoding",
                    s);
      err = buf;
      return false;
    }
    hi = std::max(hi, rows[k].second);
  }
  v.mask_lo = lo;
  v.mask_hi = hi;
  return true;
}

bool Book::prefill_keys(int s, int64_t n_q, std::vector<int32_t>& meta, std::string& err) const {
  const Seq& q = seqs_[s];
  const int64_t T = (int64_t)q.kind.size();
  char buf[256];
  meta.clear();
  if (policy_ == POLICY_LOCAL) {
    err = "masked prefill is not defined for the local-attention cache";
    return false;
  }
  if (n_q < 0 || n_q > T) {
    std::snprintf(buf, sizeof buf, "sequence %d: n_q = %lld outside [0, %lld]", s, (long long)n_q, (long long)T);
    err = buf;
    return false;
  }
  if (n_q == 0) return true;
  if (q.stored >= kPrefillNever) {
    std::snprintf(buf, sizeof buf, "sequence %d: %lld stored rows exceed the prefill limit", s, (long long)q.stored);
    err = buf;
    return false;
  }
  // the queries are the last n_q tokens and must all be stored rows (the tail of the stored rows)
  if (q.stored < n_q || stored_index(s, T - n_q) != q.stored - n_q) {
    std::snprintf(buf, sizeof buf,
                  "sequence %d: the last %lld tokens are not all stored (append them without freeing and "
                  "compress after the prefill)",
                  s, (long long)n_q);
    err = buf;
    return false;
  }
  meta.assign((size_t)q.stored, kPrefillNever << 1);
  for (int64_t j = 0; j < T; ++j) {
    if (q.kind[j] != CL) continue;
    const int64_t i = stored_index(s, j);
    if (i < 0) continue;
    meta[i] = policy_ == POLICY_PAPER ? (int32_t)((i << 1) | 1) : (int32_t)((kPrefillNever << 1) | 1);
  }
  for (const Span& sp : q.spans) {
    if (sp.freed || sp.cr < 0) continue;
    const int64_t hid = stored_index(s, sp.cr);
    for (int64_t j = sp.cl + 1; j < sp.cr; ++j) {
      const int64_t i = stored_index(s, j);
      if (i >= 0) meta[i] = (int32_t)((hid << 1) | (meta[i] & 1));
    }
  }
  return true;
}

void Book::pending_spans(int s, std::vector<std::pair<int64_t, int64_t>>& out) const {
  out.clear();
  for (const Span& sp : seqs_[s].spans)
    if (!sp.freed && sp.cr >= 0) out.emplace_back(sp.cl, sp.cr);
}

void Book::visible(int s, uint8_t* vis) const {
  const Seq& q = seqs_[s];
  const int64_t T = (int64_t)q.kind.size();
  if (T == 0) return;
  const int64_t tq = T - 1;
  if (policy_ == POLICY_LOCAL) {
    const int64_t first = local_first(tq);
    for (int64_t j = 0; j < T; ++j) vis[j] = (uint8_t)(j >= first);
    return;
  }
  if (q.kind[tq] == CL) {
    for (int64_t j = 0; j < T; ++j) vis[j] = (uint8_t)(j == tq);
    return;
  }
  for (int64_t j = 0; j < T; ++j) vis[j] = (uint8_t)!(policy_ == POLICY_PAPER && q.kind[j] == CL);
  for (const Span& sp : q.spans)
    if (sp.cr >= 0 && sp.cr < tq)
      for (int64_t j = sp.cl + 1; j < sp.cr; ++j) vis[j] = 0;
}

void Book::stored_rows(int s, std::vector<int32_t>& orig, std::vector<int32_t>& pos) const {
  const Seq& q = seqs_[s];
  orig.clear();
  pos.clear();
  if (policy_ == POLICY_LOCAL) {  // the window of the last token, oldest first
    const int64_t T = (int64_t)q.kind.size();
    for (int64_t j = T > 0 ? local_first(T - 1) : 0; j < T; ++j) {
      orig.push_back((int32_t)j);
      pos.push_back(q.pos[j]);
    }
    return;
  }
  for (int64_t j = 0; j < (int64_t)q.kind.size(); ++j) {
    if (stored_index(s, j) >= 0) {
      orig.push_back((int32_t)j);
      pos.push_back(q.pos[j]);
    }
  }
}

}  // namespace kvc
