// Host-side span bookkeeping of b token histories (no CUDA).
//
// Tracks, per sequence, the kinds and positions of every token appended so
// far, the <CL> ... <CR> spans (Sec. 3.1: non-overlapping, paired in order),
// which spans have been freed, and the number of stored rows.  From that it
// derives what each device call needs: destination rows of appended tokens,
// drop ranges of a compaction, and the rows a decode query may not see.
#pragma once

#include <cstdint>
#include <string>
#include <utility>
#include <vector>

namespace kvc {

enum Kind : uint8_t { NORMAL = 0, CL = 1, CR = 2 };
enum Policy : int { POLICY_PAPER = 0, POLICY_KEEP_CL = 1, POLICY_LOCAL = 2 };

struct Span {
  int64_t cl = -1;
  int64_t cr = -1;  // -1 while open
  bool freed = false;
};

// What a decode query of one sequence reads: stored rows [begin, len), except [mask_lo, mask_hi).
// Under the local policy the rows live in a ring: row begin + r is slot begin + r for r < wrap and
// slot r - wrap after it.
struct DecodeView {
  int64_t len = 0;
  int64_t begin = 0;
  int64_t mask_lo = 0;
  int64_t mask_hi = 0;
  int64_t wrap = INT64_MAX;
  int32_t qpos = 0;
  int64_t attended() const { return len - begin - (mask_hi - mask_lo); }
};

// One sequence's part of a compaction: drop ranges in history-index space (sorted, disjoint).
struct CompactSeq {
  int s = 0;
  int64_t len_old = 0;
  int64_t len_new = 0;
  int64_t first_row = 0;  // first stored row that is dropped
  std::vector<std::pair<int64_t, int64_t>> drops;
};

class Book {
 public:
  Book(int b, Policy policy, const int64_t* capacity, double local_ratio = 0.0);

  int b() const { return b_; }
  Policy policy() const { return policy_; }
  int64_t capacity(int s) const { return seqs_[s].cap; }
  int64_t stored(int s) const { return seqs_[s].stored; }
  int64_t history(int s) const { return (int64_t)seqs_[s].kind.size(); }
  double local_ratio() const { return local_ratio_; }
  // Local policy: first history index the query at t sees (the window is [local_first(t), t]).
  int64_t local_first(int64_t t) const;
  // Local policy: new token i of sequence s is written when it is among the last capacity tokens.
  int64_t ring_slot(int s, int64_t j) const { return j % seqs_[s].cap; }

  // Validation only (no state change).  On error returns false and sets `err`.  With
  // free_in_block, the capacity check counts only the rows that will be stored.
  bool check_append(const int32_t* n_new, const uint8_t* kinds, std::string& err, int& code,
                    bool free_in_block = false, bool check_capacity = true) const;
  void next_positions(const int32_t* n_new, const uint8_t* kinds, int32_t* pos_out) const;
  // Which of the new tokens are stored when spans opened and closed among them are freed as they
  // are written (their <CL> under the paper policy, and the enclosed tokens, are never stored).
  void kept_in_block(const int32_t* n_new, const uint8_t* kinds, std::vector<uint8_t>& kept) const;
  // kept == nullptr: every new token is stored.
  void apply_append(const int32_t* n_new, const uint8_t* kinds, const int32_t* pos, const uint8_t* kept = nullptr);

  bool plan_compress(const int32_t* seq, const int64_t* cl, const int64_t* cr, int n, std::vector<CompactSeq>& plan,
                     std::string& err) const;
  void apply_compress(const std::vector<CompactSeq>& plan, const int32_t* seq, const int64_t* cl, int n);

  // The decode query of sequence s (its last token).  False (with `err`) if the rows hidden from it
  // are not one contiguous run of stored rows.
  bool decode_view(int s, DecodeView& v, std::string& err) const;

  // Masked prefill of the last n_q history tokens of sequence s over its stored rows (Sec. 3.1).
  // meta[i] = (hid << 1) | is_cl for stored row i: row i is visible to the query at stored row iq
  // exactly when i <= iq <= hid, except that a <CL> query (is_cl of its own row) sees only itself.
  // hid is the stored row of the <CR> closing a span that encloses row i, i itself for a <CL> row
  // under the paper policy, else kPrefillNever.  False (with `err`) when the policy has no prefill
  // or the queries are not the last n_q stored rows.
  static constexpr int32_t kPrefillNever = 0x3FFFFFFF;
  bool prefill_keys(int s, int64_t n_q, std::vector<int32_t>& meta, std::string& err) const;

  void pending_spans(int s, std::vector<std::pair<int64_t, int64_t>>& out) const;
  // history index -> stored row (or -1 when freed)
  int64_t stored_index(int s, int64_t j) const;
  // visibility of every history token to the query at the last token
  void visible(int s, uint8_t* vis) const;
  void stored_rows(int s, std::vector<int32_t>& orig, std::vector<int32_t>& pos) const;
  const std::vector<uint8_t>& kinds(int s) const { return seqs_[s].kind; }
  const std::vector<int32_t>& positions(int s) const { return seqs_[s].pos; }

 private:
  struct Seq {
    std::vector<uint8_t> kind;
    std::vector<int32_t> pos;
    std::vector<Span> spans;  // ordered by cl
    int64_t normals = 0;
    bool open = false;
    int64_t stored = 0;
    int64_t cap = 0;
    std::vector<std::pair<int64_t, int64_t>> freed;  // sorted freed history ranges
    std::vector<int64_t> freed_before;               // prefix sums of freed lengths
  };
  void rebuild_prefix(Seq& q);
  int find_span(const Seq& q, int64_t cl) const;

  int b_;
  Policy policy_;
  double local_ratio_ = 0.0;
  std::vector<Seq> seqs_;
};

}  // namespace kvc
