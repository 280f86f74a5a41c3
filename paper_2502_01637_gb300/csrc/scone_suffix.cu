// Suffix index of an f-gram list (host side of the table build).
//
// Algorithm 1 selects, at each position, the longest window that is an
// f-gram. Taking the lengths one at a time (2, 3, ...) can stop early only
// if an absent window proves that no longer window is an f-gram. That holds
// when every suffix (of length >= 2) of every listed f-gram can be found in
// the table: the extension bit of a slot says that a longer listed f-gram
// ends with the slot's n-gram, and a suffix that is no f-gram itself gets a
// marker slot (no row, extension bit set). This file computes, from the
// list alone, which f-grams get the bit and which marker n-grams are needed.
//
// The hash set below holds references to token runs inside the caller's
// list (a listed f-gram, or a suffix of one), so nothing is copied until the
// markers are written out.

#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include "scone_host.h"

namespace scone {

namespace {

uint64_t mix64(uint64_t z) {
  // SplitMix64 finalizer (Steele, Lea, Flood 2014)
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

uint64_t run_hash(const int32_t* t, int n) {
  uint64_t h = 0x243F6A8885A308D3ull ^ (uint64_t)n;
  for (int j = 0; j < n; ++j) h = mix64(h ^ (uint64_t)(uint32_t)t[j]);
  return h;
}

// Open addressing over references (first token, length); ids in insertion order.
class RunSet {
 public:
  struct Ref {
    const int32_t* t;
    int32_t n;
  };

  bool reserve(int64_t expected) {
    uint64_t cap = 16;
    while (cap < (uint64_t)expected * 2) cap <<= 1;
    return rehash(cap);
  }

  // The id of the run, or -1.
  int64_t find(const int32_t* t, int n) const {
    uint64_t i = run_hash(t, n) & mask_;
    for (;;) {
      const uint32_t s = slots_[i];
      if (s == 0) return -1;
      const Ref& r = refs_[s - 1];
      if (r.n == n && std::memcmp(r.t, t, (size_t)n * sizeof(int32_t)) == 0) return s - 1;
      i = (i + 1) & mask_;
    }
  }

  // Adds a run known to be absent; returns its id, or -1 when out of memory.
  int64_t add(const int32_t* t, int n) {
    if ((refs_.size() + 1) * 2 > slots_.size() && !rehash(slots_.size() * 2)) return -1;
    try {
      refs_.push_back(Ref{t, n});
    } catch (const std::bad_alloc&) {
      return -1;
    }
    place((uint32_t)refs_.size());
    return (int64_t)refs_.size() - 1;
  }

  const Ref& ref(int64_t id) const { return refs_[id]; }

 private:
  void place(uint32_t id1) {
    const Ref& r = refs_[id1 - 1];
    uint64_t i = run_hash(r.t, r.n) & mask_;
    while (slots_[i] != 0) i = (i + 1) & mask_;
    slots_[i] = id1;
  }
  bool rehash(uint64_t cap) {
    try {
      slots_.assign(cap, 0u);
      refs_.reserve(cap / 2);
    } catch (const std::bad_alloc&) {
      return false;
    }
    mask_ = cap - 1;
    for (uint32_t id1 = 1; id1 <= refs_.size(); ++id1) place(id1);
    return true;
  }

  std::vector<uint32_t> slots_;  // id + 1, 0 = empty
  std::vector<Ref> refs_;
  uint64_t mask_ = 0;
};

}  // namespace

int suffix_index(const int32_t* tok, const uint8_t* len, int64_t n, int K, SuffixIndex* out) {
  out->ext.clear();
  out->marker_tok.clear();
  out->marker_len.clear();
  out->n_markers = 0;
  if (n <= 0) return SCONE_OK;
  // ids beyond the list's are markers: n + markers must stay below 2^32 - 1
  int64_t suffixes = 0;
  for (int64_t r = 0; r < n; ++r) suffixes += len[r] > 2 ? len[r] - 2 : 0;
  if (n + suffixes >= (int64_t)0xFFFFFFFE) return SCONE_ERR_UNSUPPORTED;
  RunSet set;
  std::vector<const int32_t*> marker_at;   // first token of each marker's run
  std::vector<uint8_t> ext;
  try {
    ext.assign((size_t)n, 0);
  } catch (const std::bad_alloc&) {
    return SCONE_ERR_NOMEM;
  }
  if (!set.reserve(n + suffixes / 4 + 16)) return SCONE_ERR_NOMEM;
  for (int64_t r = 0; r < n; ++r) {
    const int32_t* t = tok + r * K;
    if (set.find(t, len[r]) >= 0) return SCONE_ERR_DUPLICATE_FGRAM;
    if (set.add(t, len[r]) < 0) return SCONE_ERR_NOMEM;
  }
  for (int64_t r = 0; r < n; ++r) {
    const int32_t* t = tok + r * K;
    const int nr = len[r];
    for (int m = nr - 1; m >= 2; --m) {
      const int32_t* s = t + (nr - m);       // the last m tokens
      const int64_t id = set.find(s, m);
      // a marker, or an f-gram whose bit is set, was reached from a longer
      // f-gram that went on to the shorter suffixes, which are also these
      if (id >= n || (id >= 0 && ext[(size_t)id])) break;
      if (id >= 0) {
        ext[(size_t)id] = 1;
        continue;
      }
      if (set.add(s, m) < 0) return SCONE_ERR_NOMEM;
      try {
        marker_at.push_back(s);
      } catch (const std::bad_alloc&) {
        return SCONE_ERR_NOMEM;
      }
    }
  }
  const int64_t nm = (int64_t)marker_at.size();
  try {
    out->marker_tok.assign((size_t)(nm * K), -1);
    out->marker_len.resize((size_t)nm);
  } catch (const std::bad_alloc&) {
    return SCONE_ERR_NOMEM;
  }
  for (int64_t i = 0; i < nm; ++i) {
    const RunSet::Ref& ref = set.ref(n + i);
    std::memcpy(&out->marker_tok[(size_t)(i * K)], ref.t, (size_t)ref.n * sizeof(int32_t));
    out->marker_len[(size_t)i] = (uint8_t)ref.n;
  }
  out->ext.swap(ext);
  out->n_markers = nm;
  return SCONE_OK;
}

}  // namespace scone

using namespace scone;

extern "C" int scone_fgram_suffix_index(const int32_t* fgram_tok, const uint8_t* fgram_len,
                                        int64_t n_fgrams, int32_t K, uint8_t* ext,
                                        int32_t* marker_tok, uint8_t* marker_len,
                                        int64_t marker_cap, int64_t* n_markers) {
  if (n_fgrams < 0 || K < 2 || K > 8 || marker_cap < 0 || !n_markers) return SCONE_ERR_INVALID_ARG;
  if (n_fgrams > 0 && (!fgram_tok || !fgram_len)) return SCONE_ERR_INVALID_ARG;
  if (marker_cap > 0 && (!marker_tok || !marker_len)) return SCONE_ERR_INVALID_ARG;
  for (int64_t r = 0; r < n_fgrams; ++r)
    if (fgram_len[r] < 2 || fgram_len[r] > K) return SCONE_ERR_INVALID_ARG;
  SuffixIndex si;
  const int rc = suffix_index(fgram_tok, fgram_len, n_fgrams, K, &si);
  if (rc != SCONE_OK) return rc;
  if (ext && n_fgrams > 0) std::memcpy(ext, si.ext.data(), (size_t)n_fgrams);
  const int64_t copy = si.n_markers < marker_cap ? si.n_markers : marker_cap;
  if (copy > 0) {
    std::memcpy(marker_tok, si.marker_tok.data(), (size_t)(copy * K) * sizeof(int32_t));
    std::memcpy(marker_len, si.marker_len.data(), (size_t)copy);
  }
  *n_markers = si.n_markers;
  return SCONE_OK;
}
