// CPU oracle for SCONE's inference-time input embedding.
//
// TEST INFRASTRUCTURE. Only the tests, the smoke check and the benchmark's CPU
// baseline may load this library. The product path never calls it, shares no
// code with it, and has no CPU fallback through it.
//
// What it computes is the inference branch of Algorithm 1 (Sec. 3, "SCONE
// method"), written out plainly:
//
//   for i = 1..m:
//     j <- smallest j' < i with (sigma_j', ..., sigma_i) in V_fgram, else i
//     e_i <- T(sigma_i)                 if j = i
//     e_i <- F(sigma_j, ..., sigma_i)   otherwise
//
// V_fgram is a subset of V_token^[2,K] (Sec. 3), so only j' >= i - K + 1 can
// qualify; the loop below scans exactly those j' in increasing order, which is
// "smallest j'" read literally. Membership is an exact lookup of the token
// tuple in a std::map built from the caller's f-gram list; F's row for an
// f-gram is its index in that list (the paper's "hash dictionary that maps
// f-grams to matrix indices", Sec. 2, "Efficient Indexing"). Each map lookup
// counts as one query; Sec. 4.3 ("Space Usage and Query Latency") bounds the
// queries per token by K - 1 for maximum length K.
//
// Readings where the paper is silent:
//   * n-grams never cross sequence boundaries; a sequence's first position
//     always uses T (j' >= 1 within the sequence in Algorithm 1).
//   * A token outside [0, vocab) has no embedding: its output row is zeros,
//     its row is -1 and its length 0, and the call reports status -2. A
//     window containing such a token is not in V_fgram (every listed f-gram
//     has valid tokens), so it never matches.
//   * Duplicate f-grams in the list are an error (status -3): F would have
//     two rows for one key.
//
// Status codes: 0 ok, -1 invalid argument, -2 token out of range,
// -3 duplicate f-gram.
//
// Precision: the outputs are copies of stored bf16 rows (raw 16-bit words);
// there is no floating-point arithmetic.

#include <cstdint>
#include <cstring>
#include <map>
#include <thread>
#include <vector>

namespace {

struct OracleTable {
  int32_t K = 0;
  int32_t vocab = 0;
  std::map<std::vector<int32_t>, int64_t> fgram_row;
};

// Algorithm 1, one position: returns the f-gram row (or -1) and sets j.
// seq points at the start of the sequence; i is 0-based within it.
int64_t select_position(const OracleTable& t, const int32_t* seq, int64_t i, int64_t* j_out,
                        int64_t* queries) {
  int64_t first = i - (t.K - 1);
  if (first < 0) first = 0;
  for (int64_t jp = first; jp < i; ++jp) {
    const std::vector<int32_t> window(seq + jp, seq + i + 1);
    if (queries) ++*queries;
    const auto it = t.fgram_row.find(window);
    if (it != t.fgram_row.end()) {
      *j_out = jp;
      return it->second;
    }
  }
  *j_out = i;
  return -1;
}

bool valid_token(const OracleTable& t, int32_t x) { return x >= 0 && x < t.vocab; }

}  // namespace

extern "C" {

int oracle_table_create(const int32_t* fgram_tok, const uint8_t* fgram_len, int64_t n_fgrams,
                        int32_t K, int32_t vocab, void** out) {
  if (!out || K < 2 || vocab <= 0 || n_fgrams < 0) return -1;
  if (n_fgrams > 0 && (!fgram_tok || !fgram_len)) return -1;
  OracleTable* t = new OracleTable;
  t->K = K;
  t->vocab = vocab;
  for (int64_t r = 0; r < n_fgrams; ++r) {
    const int n = fgram_len[r];
    if (n < 2 || n > K) {
      delete t;
      return -1;
    }
    std::vector<int32_t> key(fgram_tok + r * K, fgram_tok + r * K + n);
    for (int32_t x : key) {
      if (!valid_token(*t, x)) {
        delete t;
        return -1;
      }
    }
    if (!t->fgram_row.emplace(std::move(key), r).second) {
      delete t;
      return -3;
    }
  }
  *out = t;
  return 0;
}

void oracle_table_destroy(void* t) { delete static_cast<OracleTable*>(t); }

int64_t oracle_table_size(const void* t) {
  return (int64_t) static_cast<const OracleTable*>(t)->fgram_row.size();
}

// Selection for every position of B sequences of length L (tok is [B * L]).
// row[p] = F row or -1; len[p] = i - j + 1 (1 = token fallback, 0 = invalid
// token); queries[p] (nullable) = map lookups made for p.
int oracle_select(const void* tp, const int32_t* tok, int32_t B, int32_t L, int64_t* row,
                  uint8_t* len, int64_t* queries) {
  const OracleTable& t = *static_cast<const OracleTable*>(tp);
  if (B < 0 || L < 0 || (B > 0 && L > 0 && (!tok || !row || !len))) return -1;
  int rc = 0;
  for (int64_t b = 0; b < B; ++b) {
    const int32_t* seq = tok + b * L;
    for (int64_t i = 0; i < L; ++i) {
      const int64_t p = b * L + i;
      int64_t q = 0, j = i;
      if (!valid_token(t, seq[i])) {
        row[p] = -1;
        len[p] = 0;
        rc = -2;
      } else {
        row[p] = select_position(t, seq, i, &j, &q);
        len[p] = (uint8_t)(i - j + 1);
      }
      if (queries) queries[p] = q;
    }
  }
  return rc;
}

// Same selection, only at the flattened positions pos[0..npos-1].
int oracle_select_at(const void* tp, const int32_t* tok, int32_t B, int32_t L, const int64_t* pos,
                     int64_t npos, int64_t* row, uint8_t* len) {
  const OracleTable& t = *static_cast<const OracleTable*>(tp);
  if (B < 0 || L <= 0 || npos < 0) return -1;
  int rc = 0;
  for (int64_t k = 0; k < npos; ++k) {
    const int64_t p = pos[k];
    if (p < 0 || p >= (int64_t)B * L) return -1;
    const int64_t b = p / L, i = p % L;
    const int32_t* seq = tok + b * L;
    int64_t j = i;
    if (!valid_token(t, seq[i])) {
      row[k] = -1;
      len[k] = 0;
      rc = -2;
    } else {
      row[k] = select_position(t, seq, i, &j, nullptr);
      len[k] = (uint8_t)(i - j + 1);
    }
  }
  return rc;
}

// Full Algorithm 1 output: out[p * d ..] = F[row] or T[token] (raw bf16
// words), zeros for an invalid token. F is [n_F * d], T is [vocab * d].
int oracle_embed(const void* tp, const int32_t* tok, int32_t B, int32_t L, const uint16_t* F,
                 int64_t n_F, const uint16_t* T, int32_t d, uint16_t* out, int64_t* row,
                 uint8_t* len) {
  const OracleTable& t = *static_cast<const OracleTable*>(tp);
  if (B < 0 || L < 0 || d <= 0) return -1;
  int rc = 0;
  for (int64_t b = 0; b < B; ++b) {
    const int32_t* seq = tok + b * L;
    for (int64_t i = 0; i < L; ++i) {
      const int64_t p = b * L + i;
      uint16_t* e = out + p * d;
      int64_t j = i, r = -1;
      if (!valid_token(t, seq[i])) {
        std::memset(e, 0, sizeof(uint16_t) * (size_t)d);
        if (row) row[p] = -1;
        if (len) len[p] = 0;
        rc = -2;
        continue;
      }
      r = select_position(t, seq, i, &j, nullptr);
      if (j == i) {
        std::memcpy(e, T + (int64_t)seq[i] * d, sizeof(uint16_t) * (size_t)d);
      } else {
        if (r >= n_F) return -1;
        std::memcpy(e, F + r * d, sizeof(uint16_t) * (size_t)d);
      }
      if (row) row[p] = r;
      if (len) len[p] = (uint8_t)(i - j + 1);
    }
  }
  return rc;
}

// The same definition with the sequences split over `threads` std::threads
// (contiguous ranges; each thread runs oracle_embed on its own range, the table
// is only read). Used to time the baseline on every host core.
int oracle_embed_threads(const void* tp, const int32_t* tok, int32_t B, int32_t L,
                         const uint16_t* F, int64_t n_F, const uint16_t* T, int32_t d,
                         uint16_t* out, int64_t* row, uint8_t* len, int32_t threads) {
  if (B < 0 || L < 0 || d <= 0) return -1;
  if (threads < 1) threads = 1;
  if (threads > B) threads = B > 0 ? B : 1;
  std::vector<int> rcs((size_t)threads, 0);
  std::vector<std::thread> pool;
  for (int32_t k = 0; k < threads; ++k) {
    const int64_t b0 = (int64_t)B * k / threads, b1 = (int64_t)B * (k + 1) / threads;
    pool.emplace_back([=, &rcs] {
      const int64_t p0 = b0 * L;
      rcs[(size_t)k] = oracle_embed(tp, tok + p0, (int32_t)(b1 - b0), L, F, n_F, T, d,
                                    out + p0 * d, row ? row + p0 : nullptr,
                                    len ? len + p0 : nullptr);
    });
  }
  for (std::thread& th : pool) th.join();
  int rc = 0;
  for (int r : rcs) {
    if (r == -1) return -1;
    if (r != 0) rc = r;
  }
  return rc;
}

// Decode: S sequences, each with a known prefix of hist_len[s] tokens (the
// last hist_len[s] entries of hist[s * H .. s * H + H - 1], H = hist_stride),
// then `steps` new tokens per sequence, new_tok[step * S + s]. Each new token
// is embedded by Algorithm 1 applied to prefix ++ new tokens so far.
// Outputs are [steps * S] rows of out/row/len.
int oracle_decode(const void* tp, int32_t S, const int32_t* hist, int32_t hist_stride,
                  const int32_t* hist_len, int32_t steps, const int32_t* new_tok, const uint16_t* F,
                  int64_t n_F, const uint16_t* T, int32_t d, uint16_t* out, int64_t* row,
                  uint8_t* len) {
  const OracleTable& t = *static_cast<const OracleTable*>(tp);
  if (S < 0 || steps < 0 || d <= 0 || hist_stride < 0) return -1;
  int rc = 0;
  for (int64_t s = 0; s < S; ++s) {
    const int32_t h = hist_len[s];
    if (h < 0 || h > hist_stride) return -1;
    std::vector<int32_t> seq(hist + s * hist_stride + (hist_stride - h),
                             hist + s * hist_stride + hist_stride);
    for (int64_t k = 0; k < steps; ++k) {
      seq.push_back(new_tok[k * S + s]);
      const int64_t i = (int64_t)seq.size() - 1;
      const int64_t p = k * S + s;
      uint16_t* e = out + p * d;
      if (!valid_token(t, seq[i])) {
        std::memset(e, 0, sizeof(uint16_t) * (size_t)d);
        if (row) row[p] = -1;
        if (len) len[p] = 0;
        rc = -2;
        continue;
      }
      int64_t j = i;
      const int64_t r = select_position(t, seq.data(), i, &j, nullptr);
      if (j == i) {
        std::memcpy(e, T + (int64_t)seq[i] * d, sizeof(uint16_t) * (size_t)d);
      } else {
        if (r >= n_F) return -1;
        std::memcpy(e, F + r * d, sizeof(uint16_t) * (size_t)d);
      }
      if (row) row[p] = r;
      if (len) len[p] = (uint8_t)(i - j + 1);
    }
  }
  return rc;
}

}  // extern "C"
