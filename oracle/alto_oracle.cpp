// CPU oracle for batched re-aggregation of streamed fragments by nested
// ancestry (Alto, arxiv 2403.04311).
//
// TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
// definition that the CUDA library is checked against.  Only the tests, the
// smoke check and the benchmark's CPU-baseline leg may build or call it; the
// library never does, and the two share no code, header or constant.
//
// It processes fragments one at a time, in arrival order, with ordered maps
// keyed by (level, parent_id):
//
//  * Sec. 4.2 (nested ancestry): every pmap entry pushes one tag (id of the
//    parent element, index of the element in the parent's stream); a group is
//    identified by its level and parent id, and its children are indexed by
//    the tag's child index.  Level D-1 children are the fragments themselves.
//  * Sec. 3.1 (hierarchical datatypes): an output stream is known to be
//    complete only when its end-of-output delimiter has arrived; here that is
//    the last-flag bit on the child that closes the group.  A group is
//    complete when its last child is known, every child 0..last is present,
//    and every child is itself complete.
//  * Sec. 3.2 (pmap) and Sec. 4.1: the outputs of a parallel map are put back
//    into the original stream order -- a CONCAT group emits its subtree's
//    leaf payloads ordered by the child-index path.
//  * Sec. 3.3 (aggregate operator): the completed group is collected into one
//    output object; Sec. 4.3: all elements with the same ancestry tags end up
//    at the same aggregation point (here, the same group).
//  * Reductions over scores (the reranker's top-k of Sec. 3.2's example, the
//    top-K thought selection of Sec. 6.1.2): MAX reports the largest leaf
//    score of the subtree; TOPK lists the k children with the largest score
//    (ties to the smaller child index), under IEEE-754 totalOrder.
//  * Streaming release (optional; Sec. 3.2: the pmap's outputs are put back
//    in order and passed on as a stream, not only once the whole group is
//    in): at the end of each batch, a still-open CONCAT group whose run of
//    complete children 0..r-1 grew past what it released before emits that
//    run as a partial record (ops bit 0x80, n_children = r, completion seq =
//    the latest completion among the run); the group's final record carries
//    only the children not yet released.  Records of a batch are ordered by
//    (completion seq, deeper level first).
//
// Error classes are collected per batch and the batch reports the one with
// the highest priority (EINVAL > EDUP > EINCONSIST > ELAST > ECLOSED); the
// first batch with an error latches it and poisons the handle.  A fragment
// for a group that was already emitted always also repeats a slot, names a
// second child for a slot, or passes the last index, so it is reported as
// one of those; ECLOSED ranks last and only names the cause in this file.
//
// Parity pins: the tests check this oracle against an independent
// non-incremental evaluation of the completion predicate over every arrival
// order and batch cut of small trees, against numpy sorts for the single-level
// and single-batch cases, against hand-worked examples in tests/golden/, and
// against invariants (exactly-once emission, parent after descendants,
// payload conservation).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <map>
#include <set>
#include <utility>
#include <vector>

namespace {

// status codes (same values as the public interface; written out here again)
constexpr int kOk = 0;
constexpr int kEInval = -1;
constexpr int kEDup = -4;
constexpr int kELast = -5;
constexpr int kEInconsist = -6;
constexpr int kEClosed = -7;

int priority(int code) {
  switch (code) {
    case kEInval: return 5;
    case kEDup: return 4;
    case kEInconsist: return 3;
    case kELast: return 2;
    case kEClosed: return 1;
    default: return 0;
  }
}

constexpr int kPayloadNone = 0, kPayloadConcat = 1;
constexpr int kScoreNone = 0, kScoreMax = 1, kScoreTopk = 2;

struct OrcRecord {  // 48 bytes
  uint64_t completion_seq;
  uint64_t payload_off;
  uint64_t payload_len;
  uint64_t topk_off;
  uint32_t parent_id;
  uint32_t n_children;
  uint8_t level;
  uint8_t ops;
  uint16_t topk_n;
  float score;
};
static_assert(sizeof(OrcRecord) == 48, "record layout");

struct OrcPair {  // 8 bytes
  uint32_t child_index;
  float score;
};

struct Leaf {
  std::vector<int32_t> tokens;
  float score = 0.0f;
  uint64_t seq = 0;           // arrival index (its completion seq)
};

struct Group {
  bool has_up = false;
  uint64_t up = 0;            // tag one level up under which this group sits
  bool has_last = false;
  uint32_t last = 0;
  bool any_child = false;
  uint32_t max_child = 0;
  std::map<uint32_t, uint32_t> child_group;  // level < D-1: slot -> child id
  std::map<uint32_t, Leaf> leaves;           // level D-1: slot -> leaf
  uint32_t completed = 0;     // number of complete children
  bool emitted = false;
  uint64_t done_seq = 0;      // completion seq, once emitted
  uint32_t released = 0;      // streaming release: children 0..released-1 already emitted
};

// IEEE-754 totalOrder restricted to non-NaN values: the usual order, with
// -0.0 below +0.0.
bool total_less(float a, float b) {
  if (a < b) return true;
  if (a > b) return false;
  return std::signbit(a) && !std::signbit(b);
}

struct Oracle {
  int depth = 0;
  int payload_op[8] = {};
  int score_op[8] = {};
  int topk_k[8] = {};
  bool needs_score = false;
  // Streaming release (Sec. 3.2: as each item of a pmap finishes, the stream
  // is reconstituted in the original order and sent on in a streaming
  // fashion): at the end of every batch, an open CONCAT group whose in-order
  // prefix of complete children advanced emits that part of its payload as a
  // partial record; its final record then holds only the rest.
  bool stream_release = false;
  int concat_level = -1;
  std::set<uint32_t> touched;  // CONCAT-level groups that got fragments in this batch

  std::map<std::pair<int, uint32_t>, Group> groups;
  uint64_t seq_next = 0;       // global sequence number of the next fragment
  uint64_t batches = 0;        // batches accepted so far
  uint64_t drain_first_batch = 0;
  int status = kOk;            // latched error

  std::vector<OrcRecord> records;
  std::vector<int32_t> payload;
  std::vector<OrcPair> topk;
  // drained copies handed to the caller
  std::vector<OrcRecord> out_records;
  std::vector<int32_t> out_payload;
  std::vector<OrcPair> out_topk;

  Group& group(int level, uint32_t id) { return groups[{level, id}]; }

  // Leaves of the subtree of (level, id), concatenated in child-index path
  // order (Sec. 3.2: the stream is reconstituted in its original order);
  // children from..to-1 of the group itself.
  void concat_range(int level, uint32_t id, uint32_t from, uint32_t to, std::vector<int32_t>& out) {
    Group& g = group(level, id);
    for (uint32_t c = from; c < to; ++c) {
      if (level == depth - 1) {
        const Leaf& lf = g.leaves.at(c);
        out.insert(out.end(), lf.tokens.begin(), lf.tokens.end());
      } else {
        concat(level + 1, g.child_group.at(c), out);
      }
    }
  }
  void concat(int level, uint32_t id, std::vector<int32_t>& out) {
    concat_range(level, id, 0, group(level, id).last + 1, out);
  }

  // Child c of (level, id) is complete (a leaf that arrived, or an emitted
  // group); its completion seq.
  bool child_complete(int level, const Group& g, uint32_t c, uint64_t* seq) {
    if (level == depth - 1) {
      auto it = g.leaves.find(c);
      if (it == g.leaves.end()) return false;
      *seq = it->second.seq;
      return true;
    }
    auto it = g.child_group.find(c);
    if (it == g.child_group.end()) return false;
    auto gi = groups.find({level + 1, it->second});
    if (gi == groups.end() || !gi->second.emitted) return false;
    *seq = gi->second.done_seq;
    return true;
  }

  // Largest leaf score of the subtree of (level, id).
  float subtree_max(int level, uint32_t id) {
    Group& g = group(level, id);
    bool have = false;
    float best = 0.0f;
    for (uint32_t c = 0; c <= g.last; ++c) {
      float s = (level == depth - 1) ? g.leaves.at(c).score
                                     : subtree_max(level + 1, g.child_group.at(c));
      if (!have || total_less(best, s)) best = s;
      have = true;
    }
    return best;
  }

  // Sec. 3.3: collect the completed group into one output record.
  void emit(int level, uint32_t id, uint64_t seq) {
    Group& g = group(level, id);
    g.emitted = true;
    g.done_seq = seq;
    OrcRecord r{};
    r.completion_seq = seq;
    r.parent_id = id;
    r.n_children = g.last + 1;
    r.level = static_cast<uint8_t>(level);
    r.ops = static_cast<uint8_t>(payload_op[level] | (score_op[level] << 2));
    r.payload_off = payload.size();
    if (payload_op[level] == kPayloadConcat) {
      // with streaming release, the children released earlier are not repeated
      const uint32_t from = stream_release ? g.released : 0;
      concat_range(level, id, from, g.last + 1, payload);
    }
    r.payload_len = payload.size() - r.payload_off;
    r.topk_off = topk.size();
    r.topk_n = 0;
    r.score = 0.0f;
    if (score_op[level] != kScoreNone) r.score = subtree_max(level, id);
    if (score_op[level] == kScoreTopk) {
      std::vector<OrcPair> kids;
      for (uint32_t c = 0; c <= g.last; ++c) {
        float s = (level == depth - 1) ? g.leaves.at(c).score
                                       : subtree_max(level + 1, g.child_group.at(c));
        kids.push_back({c, s});
      }
      std::stable_sort(kids.begin(), kids.end(), [](const OrcPair& a, const OrcPair& b) {
        if (total_less(b.score, a.score)) return true;   // larger score first
        if (total_less(a.score, b.score)) return false;
        return a.child_index < b.child_index;             // tie: smaller index
      });
      size_t k = std::min<size_t>(kids.size(), static_cast<size_t>(topk_k[level]));
      for (size_t j = 0; j < k; ++j) topk.push_back(kids[j]);
      r.topk_n = static_cast<uint16_t>(k);
    }
    records.push_back(r);
  }

  bool complete(const Group& g) const {
    return g.has_last && g.completed == g.last + 1;
  }

  // One fragment, Sec. 4.2: register it under each of its D tags (outermost
  // first), then walk back up popping one level at a time while groups close.
  void fragment(const uint64_t* tag, const int32_t* tokens, uint32_t len, float score,
                uint64_t seq, std::set<int>& errors) {
    for (int l = 0; l < depth; ++l) {
      uint32_t pid = static_cast<uint32_t>(tag[l] >> 32);
      uint32_t c = static_cast<uint32_t>(tag[l] & 0x7FFFFFFFu);
      bool last = (tag[l] >> 31) & 1u;
      Group& g = group(l, pid);
      if (g.emitted) errors.insert(kEClosed);
      if (l > 0) {
        if (!g.has_up) {
          g.has_up = true;
          g.up = tag[l - 1];
        } else if (g.up != tag[l - 1]) {
          errors.insert(kEInconsist);
        }
      }
      if (l < depth - 1) {
        uint32_t child = static_cast<uint32_t>(tag[l + 1] >> 32);
        auto it = g.child_group.find(c);
        if (it == g.child_group.end()) g.child_group[c] = child;
        else if (it->second != child) errors.insert(kEInconsist);
      } else {
        if (g.leaves.count(c)) {
          errors.insert(kEDup);
        } else {
          Leaf& lf = g.leaves[c];
          lf.tokens.assign(tokens, tokens + len);
          lf.score = score;
          lf.seq = seq;
        }
      }
      if (!g.any_child || c > g.max_child) g.max_child = c;
      g.any_child = true;
      if (last) {
        if (g.has_last && g.last != c) errors.insert(kELast);
        if (!g.has_last) {
          g.has_last = true;
          g.last = c;
        }
      }
      if (g.has_last && g.max_child > g.last) errors.insert(kELast);
      if (stream_release && l == concat_level) touched.insert(pid);
    }
    if (!errors.empty()) return;
    // the leaf is complete on arrival; pop levels while the group closes
    for (int l = depth - 1; l >= 0; --l) {
      uint32_t pid = static_cast<uint32_t>(tag[l] >> 32);
      Group& g = group(l, pid);
      g.completed += 1;
      if (!complete(g)) break;
      emit(l, pid, seq);
    }
  }

  // End of a batch with streaming release: every touched, still open CONCAT
  // group whose in-order prefix of complete children advanced emits those
  // children as a partial record (flag 0x80 in ops, no score or top-k;
  // n_children = children released so far; completion seq = the largest
  // completion seq among them);
  // the batch's records are then put in (completion seq, deeper first) order.
  void release_prefixes(size_t rec_base, size_t pay_base, size_t tk_base) {
    struct Ev {
      OrcRecord r;
      std::vector<int32_t> pay;
      std::vector<OrcPair> tk;
    };
    std::vector<Ev> ev;
    for (size_t k = rec_base; k < records.size(); ++k) {
      Ev e;
      e.r = records[k];
      e.pay.assign(payload.begin() + records[k].payload_off,
                   payload.begin() + records[k].payload_off + records[k].payload_len);
      e.tk.assign(topk.begin() + records[k].topk_off, topk.begin() + records[k].topk_off + records[k].topk_n);
      ev.push_back(std::move(e));
    }
    const int M = concat_level;
    for (uint32_t pid : touched) {
      Group& g = group(M, pid);
      if (g.emitted) continue;
      uint32_t r1 = g.released;
      uint64_t mx = 0, sq = 0;
      while (child_complete(M, g, r1, &sq)) {
        mx = std::max(mx, sq);
        ++r1;
      }
      if (r1 == g.released) continue;
      Ev e;
      e.r = OrcRecord{};
      e.r.completion_seq = mx;
      e.r.parent_id = pid;
      e.r.n_children = r1;
      e.r.level = static_cast<uint8_t>(M);
      e.r.ops = static_cast<uint8_t>(kPayloadConcat | 0x80);   // payload only, no score
      concat_range(M, pid, g.released, r1, e.pay);
      e.r.payload_len = e.pay.size();
      g.released = r1;
      ev.push_back(std::move(e));
    }
    std::stable_sort(ev.begin(), ev.end(), [](const Ev& a, const Ev& b) {
      if (a.r.completion_seq != b.r.completion_seq) return a.r.completion_seq < b.r.completion_seq;
      return a.r.level > b.r.level;
    });
    records.resize(rec_base);
    payload.resize(pay_base);
    topk.resize(tk_base);
    for (Ev& e : ev) {
      e.r.payload_off = payload.size();
      payload.insert(payload.end(), e.pay.begin(), e.pay.end());
      e.r.topk_off = topk.size();
      topk.insert(topk.end(), e.tk.begin(), e.tk.end());
      records.push_back(e.r);
    }
  }

  int push(int64_t n, const uint64_t* tags, const uint32_t* off, int64_t n_payload,
           const int32_t* pay, const float* score) {
    // argument checks: rejected without latching
    if (n < 0 || n_payload < 0) return kEInval;
    if (n > 0 && (tags == nullptr || off == nullptr)) return kEInval;
    if (n > 0 && needs_score && score == nullptr) return kEInval;
    if (n_payload > 0 && pay == nullptr) return kEInval;
    if (status != kOk) return status;
    std::set<int> errors;
    // batch-level validation
    for (int64_t i = 0; i < n; ++i) {
      if (off[i] > off[i + 1]) errors.insert(kEInval);
    }
    if (n > 0 && static_cast<int64_t>(off[n]) > n_payload) errors.insert(kEInval);
    if (needs_score) {
      for (int64_t i = 0; i < n; ++i)
        if (std::isnan(score[i])) errors.insert(kEInval);
    }
    uint64_t seq_base = seq_next;
    const size_t rec_base = records.size(), pay_base = payload.size(), tk_base = topk.size();
    touched.clear();
    if (errors.empty()) {
      std::vector<uint64_t> tag(depth);
      for (int64_t i = 0; i < n; ++i) {
        for (int l = 0; l < depth; ++l) tag[l] = tags[l * n + i];
        fragment(tag.data(), pay + off[i], off[i + 1] - off[i],
                 needs_score ? score[i] : 0.0f, seq_base + i, errors);
      }
    }
    if (errors.empty() && stream_release) release_prefixes(rec_base, pay_base, tk_base);
    seq_next += n;
    batches += 1;
    if (!errors.empty()) {
      int worst = kOk;
      for (int e : errors)
        if (priority(e) > priority(worst)) worst = e;
      status = worst;
    }
    return status;
  }
};

}  // namespace

extern "C" {

struct orc_drain {
  int64_t n_records;
  const OrcRecord* records;
  int64_t n_payload;
  const int32_t* payload;
  int64_t n_topk;
  const OrcPair* topk;
  uint64_t first_batch;
  uint64_t n_batches;
};

// Returns NULL for an invalid configuration (same rules as the library's).
void* orc_create(int depth, const int* payload_op, const int* score_op, const int* topk_k) {
  if (depth < 1 || depth > 8) return nullptr;
  Oracle* o = new Oracle();
  o->depth = depth;
  int n_concat = 0;
  for (int l = 0; l < depth; ++l) {
    o->payload_op[l] = payload_op[l];
    o->score_op[l] = score_op[l];
    o->topk_k[l] = topk_k[l];
    bool ok = (payload_op[l] == kPayloadNone || payload_op[l] == kPayloadConcat) &&
              (score_op[l] >= kScoreNone && score_op[l] <= kScoreTopk) &&
              (score_op[l] != kScoreTopk || (topk_k[l] >= 1 && topk_k[l] <= 32));
    if (!ok) {
      delete o;
      return nullptr;
    }
    n_concat += payload_op[l] == kPayloadConcat;
    if (score_op[l] != kScoreNone) o->needs_score = true;
  }
  if (n_concat > 1) {
    delete o;
    return nullptr;
  }
  return o;
}

int orc_push(void* h, int64_t n, int depth, const uint64_t* tags, const uint32_t* off,
             int64_t n_payload, const int32_t* payload, const float* score) {
  if (h == nullptr) return kEInval;
  Oracle* o = static_cast<Oracle*>(h);
  if (depth != o->depth) return kEInval;
  return o->push(n, tags, off, n_payload, payload, score);
}

int orc_drain(void* h, orc_drain* out) {
  if (h == nullptr || out == nullptr) return kEInval;
  Oracle* o = static_cast<Oracle*>(h);
  o->out_records.swap(o->records);
  o->out_payload.swap(o->payload);
  o->out_topk.swap(o->topk);
  o->records.clear();
  o->payload.clear();
  o->topk.clear();
  if (o->status != kOk) {
    o->out_records.clear();
    o->out_payload.clear();
    o->out_topk.clear();
  }
  out->n_records = static_cast<int64_t>(o->out_records.size());
  out->records = o->out_records.data();
  out->n_payload = static_cast<int64_t>(o->out_payload.size());
  out->payload = o->out_payload.data();
  out->n_topk = static_cast<int64_t>(o->out_topk.size());
  out->topk = o->out_topk.data();
  out->first_batch = o->drain_first_batch;
  out->n_batches = o->batches - o->drain_first_batch;
  o->drain_first_batch = o->batches;
  return o->status;
}

// Streaming release at the CONCAT level (before the first push).
int orc_set_stream_release(void* h, int on) {
  Oracle* o = static_cast<Oracle*>(h);
  if (o == nullptr || o->batches != 0) return kEInval;
  o->concat_level = -1;
  for (int l = 0; l < o->depth; ++l)
    if (o->payload_op[l] == kPayloadConcat) o->concat_level = l;
  if (on && o->concat_level < 0) return kEInval;
  o->stream_release = on != 0;
  return kOk;
}

// Number of groups that have fragments but have not been emitted.
int64_t orc_open_groups(void* h) {
  Oracle* o = static_cast<Oracle*>(h);
  int64_t n = 0;
  for (auto& kv : o->groups) n += !kv.second.emitted;
  return n;
}

void orc_destroy(void* h) { delete static_cast<Oracle*>(h); }

}  // extern "C"
