// CPU oracle for f-gram discovery (constructing V_fgram from a corpus).
//
// TEST INFRASTRUCTURE. Only the tests, the smoke check and the benchmark's CPU
// baseline may load this library. The product path never calls it, shares no
// code with it, and has no CPU fallback through it.
//
// What it computes is Algorithm 3 ("Constructing a set of f-grams",
// Appendix A) written out plainly:
//
//   for n = 2..K, for every n-gram w: C_w <- number of times w appears in the
//   token sequences
//   sort all n-grams by C_w, largest first; return the first S
//
// The count is taken over every window of every sequence: a window never
// spans two sequences, and overlapping occurrences count separately. The map
// below is keyed by the exact token tuple; nothing is hashed or packed. It does
// not use the K-1 pruned scans of Sec. 3.2: that method is exact for every
// n-gram with count >= the threshold, so its result must equal this one.
//
// Readings where the paper is silent or leaves a choice:
//   * Threshold. Sec. 3.2 keeps only n-grams that appear at least 5 times.
//     Here that is the parameter min_count >= 1, applied to every length; an
//     n-gram below it is never selected. With min_count = 1 the result is
//     Algorithm 3's own, since an n-gram that never appears has count 0.
//   * Ties. Algorithm 3 breaks ties arbitrarily. Here the order is fixed:
//     count descending, then length ascending, then the position of the first
//     occurrence (start index in the flattened B x L corpus) ascending. Two
//     distinct n-grams of one length never share a first occurrence, so this
//     order is total and the selection unique.
//   * Output order. Algorithm 3 returns a set. The list is returned in length
//     ascending, first occurrence ascending order; a table built from it gives
//     f-gram r the r-th row.
//   * Fewer than S qualify: all of them are returned.
//   * A token outside [0, vocab) is an error (status -2): no list is returned.
//
// Status codes: 0 ok, -1 invalid argument, -2 token out of range.

#include <algorithm>
#include <cstdint>
#include <map>
#include <thread>
#include <unordered_map>
#include <vector>

namespace {

struct Entry {
  int64_t count = 0;
  int64_t first = -1;  // start of the first occurrence in the flattened corpus
};

struct Ranked {
  std::vector<int32_t> gram;
  int64_t count;
  int64_t first;
};

// An n-gram as a fixed-size tuple (tokens past n are zero), for the query map.
struct Gram {
  int32_t t[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int32_t n = 0;
  bool operator==(const Gram& o) const {
    if (n != o.n) return false;
    for (int j = 0; j < n; ++j)
      if (t[j] != o.t[j]) return false;
    return true;
  }
};

struct GramHash {
  size_t operator()(const Gram& g) const {  // FNV-1a over the tokens and the length
    uint64_t h = 1469598103934665603ull;
    for (int j = 0; j < g.n; ++j) h = (h ^ (uint32_t)g.t[j]) * 1099511628211ull;
    return (size_t)((h ^ (uint64_t)g.n) * 1099511628211ull);
  }
};

}  // namespace

extern "C" int oracle_discover(const int32_t* tok, int32_t B, int32_t L, int32_t vocab, int32_t K,
                               int64_t S, int32_t min_count, int32_t* out_tok, uint8_t* out_len,
                               uint32_t* out_count, int64_t out_cap, int64_t* n_out,
                               int64_t* distinct, int64_t* frequent) {
  if (B < 0 || L < 0 || vocab < 1 || K < 2 || K > 8 || S < 0 || min_count < 1 || !n_out ||
      out_cap < 0 || (B > 0 && L > 0 && !tok))
    return -1;
  const int64_t m = (int64_t)B * L;
  for (int64_t i = 0; i < m; ++i)
    if (tok[i] < 0 || tok[i] >= vocab) return -2;

  // C_w for every n-gram that appears, n = 2..K (Algorithm 3, the counting loops).
  std::map<std::vector<int32_t>, Entry> counts;
  for (int64_t b = 0; b < B; ++b) {
    const int32_t* seq = tok + b * L;
    for (int32_t n = 2; n <= K; ++n) {
      for (int64_t p = 0; p + n <= L; ++p) {
        Entry& e = counts[std::vector<int32_t>(seq + p, seq + p + n)];
        if (e.count == 0) e.first = b * L + p;
        e.count += 1;
      }
    }
  }

  if (distinct)
    for (int n = 0; n <= K; ++n) distinct[n] = 0;
  if (frequent)
    for (int n = 0; n <= K; ++n) frequent[n] = 0;
  std::vector<Ranked> all;
  for (const auto& kv : counts) {
    const int n = (int)kv.first.size();
    if (distinct) distinct[n] += 1;
    if (kv.second.count < min_count) continue;
    if (frequent) frequent[n] += 1;
    all.push_back(Ranked{kv.first, kv.second.count, kv.second.first});
  }

  // Sorted by count, largest first; ties by length, then first occurrence.
  std::sort(all.begin(), all.end(), [](const Ranked& a, const Ranked& b) {
    if (a.count != b.count) return a.count > b.count;
    if (a.gram.size() != b.gram.size()) return a.gram.size() < b.gram.size();
    return a.first < b.first;
  });
  if ((int64_t)all.size() > S) all.resize((size_t)S);

  // The selected set, listed by length, then first occurrence.
  std::sort(all.begin(), all.end(), [](const Ranked& a, const Ranked& b) {
    if (a.gram.size() != b.gram.size()) return a.gram.size() < b.gram.size();
    return a.first < b.first;
  });
  *n_out = (int64_t)all.size();
  if ((int64_t)all.size() > out_cap) return -1;
  for (size_t r = 0; r < all.size(); ++r) {
    for (int j = 0; j < K; ++j)
      out_tok[r * K + j] = j < (int)all[r].gram.size() ? all[r].gram[j] : -1;
    out_len[r] = (uint8_t)all[r].gram.size();
    if (out_count) out_count[r] = (uint32_t)all[r].count;
  }
  return 0;
}

// Occurrences of given n-grams in a corpus: every window of length 2..K is
// looked up in a hash map of the queries (exact token tuples). Used at sizes
// where the full count map above would not fit the time of a test; the
// corpus is split over `threads` threads by sequence, each with its own
// tallies, summed at the end. q_tok [nq*K] padded, q_len [nq] in [2, K];
// counts[nq] receives the number of windows equal to each query, first[nq]
// the start of its first occurrence in the flattened corpus (or -1).
extern "C" int oracle_count_ngrams(const int32_t* tok, int32_t B, int32_t L, int32_t K,
                                   const int32_t* q_tok, const uint8_t* q_len, int64_t nq,
                                   int64_t* counts, int64_t* first, int32_t threads) {
  if (B < 0 || L < 0 || K < 2 || K > 8 || nq < 0 || !counts || !first) return -1;
  std::unordered_map<Gram, int64_t, GramHash> index;
  for (int64_t q = 0; q < nq; ++q) {
    if (q_len[q] < 2 || q_len[q] > K) return -1;
    Gram g;
    g.n = q_len[q];
    for (int j = 0; j < g.n; ++j) g.t[j] = q_tok[q * K + j];
    if (!index.emplace(g, q).second) return -1;   // the same query twice
  }
  if (threads < 1) threads = (int32_t)std::max(1u, std::thread::hardware_concurrency());
  std::vector<std::vector<int64_t>> c((size_t)threads, std::vector<int64_t>((size_t)nq, 0));
  std::vector<std::vector<int64_t>> f((size_t)threads, std::vector<int64_t>((size_t)nq, -1));
  auto work = [&](int w) {
    for (int64_t b = w; b < B; b += threads) {
      const int32_t* seq = tok + b * L;
      for (int64_t i = 0; i < L; ++i) {
        Gram g;
        for (int n = 2; n <= K && n <= i + 1; ++n) {
          g.n = n;
          for (int j = 0; j < n; ++j) g.t[j] = seq[i - n + 1 + j];
          const auto it = index.find(g);
          if (it == index.end()) continue;
          const int64_t q = it->second;
          const int64_t start = b * L + i - n + 1;
          if (c[w][q] == 0 || start < f[w][q]) f[w][q] = start;
          c[w][q] += 1;
        }
      }
    }
  };
  std::vector<std::thread> pool;
  for (int w = 0; w < threads; ++w) pool.emplace_back(work, w);
  for (auto& t : pool) t.join();
  for (int64_t q = 0; q < nq; ++q) {
    counts[q] = 0;
    first[q] = -1;
    for (int w = 0; w < threads; ++w) {
      counts[q] += c[w][q];
      if (f[w][q] >= 0 && (first[q] < 0 || f[w][q] < first[q])) first[q] = f[w][q];
    }
  }
  return 0;
}
