// Seeded synthetic inputs for the SCONE embedding path.
//
// This module is shared by the CPU oracle side and the CUDA side. It only
// produces inputs (token streams, f-gram lists, embedding rows); it holds none
// of the method's arithmetic (no suffix matching, no lookup, no gather).
//
// Random numbers: SplitMix64 (Steele, Lea, Flood, "Fast splittable
// pseudorandom number generators", OOPSLA 2014) used as a counter-based
// generator: draw c of stream `seed` is mix64(seed + (c + 1) * golden_gamma).
//
// Token law: Zipf(s) over ranks r = 1..V, P(r) proportional to r^-s, token id
// r - 1, sampled by inverse CDF (u = top 53 bits of a draw, token = first k
// with cdf[k] > u), accelerated with a guide table (Chen & Asau 1974), which
// returns exactly the upper_bound result.
//
// Rows: each bf16 element is an Irwin-Hall(4) approximation of N(0, 0.02):
// the four 16-bit quarters of one draw are summed, centred, scaled by one
// fp32 multiply and rounded to bf16 (round to nearest even). All steps are
// integer or single IEEE operations, so CPU and GPU produce the same bytes.
//
// Build with -ffp-contract=off so the CDF table is the same on every host.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

inline uint64_t draw(uint64_t seed, uint64_t ctr) { return mix64(seed + (ctr + 1) * kGamma); }

inline double unit53(uint64_t x) { return (double)(x >> 11) * 0x1.0p-53; }

// ---------------------------------------------------------------- Zipf law
struct Zipf {
  std::vector<double> cdf;
  std::vector<int32_t> guide;
  Zipf(int32_t vocab, double s) : cdf(vocab), guide((size_t)vocab + 1) {
    double acc = 0.0;
    for (int32_t k = 0; k < vocab; ++k) {
      acc += std::pow((double)(k + 1), -s);
      cdf[k] = acc;
    }
    const double total = acc;
    for (int32_t k = 0; k < vocab; ++k) cdf[k] /= total;
    cdf[vocab - 1] = 1.0;
    // guide[j] = first k with cdf[k] > j / M  (M = vocab buckets)
    const size_t M = (size_t)vocab;
    int32_t k = 0;
    for (size_t j = 0; j <= M; ++j) {
      const double lo = (double)j / (double)M;
      while (k < vocab - 1 && cdf[k] <= lo) ++k;
      guide[j] = k;
    }
  }
  int32_t sample(uint64_t x) const {
    const double u = unit53(x);
    size_t j = (size_t)(u * (double)(guide.size() - 1));
    if (j >= guide.size() - 1) j = guide.size() - 2;
    int32_t k = guide[j];
    const int32_t last = (int32_t)cdf.size() - 1;
    while (k < last && cdf[k] <= u) ++k;
    return k;
  }
};

// ------------------------------------------------------- token stream state
// Base Zipf tokens at counter p, optionally overwritten by phrase injection:
// at each position not already inside a phrase, a phrase starts with
// probability inject_p; it overwrites that position and the following ones.
struct Stream {
  const Zipf& zipf;
  uint64_t seed, inj_seed, pick_seed;
  double inject_p;
  const int32_t* ph_tok;   // [n_ph * ph_stride]
  const int32_t* ph_len;   // [n_ph]
  int32_t n_ph, ph_stride;
  uint64_t pos = 0;
  int32_t cur = -1, off = 0;
  Stream(const Zipf& z, uint64_t seed_, double p, const int32_t* pt, const int32_t* pl, int32_t np,
         int32_t stride)
      : zipf(z), seed(seed_), inj_seed(mix64(seed_ ^ 0x1A2B3C4D5E6F7081ull)),
        pick_seed(mix64(seed_ ^ 0x0F1E2D3C4B5A6978ull)), inject_p(p), ph_tok(pt), ph_len(pl),
        n_ph(np), ph_stride(stride) {}
  int32_t next() {
    const uint64_t p = pos++;
    const int32_t base = zipf.sample(draw(seed, p));
    if (n_ph > 0 && inject_p > 0.0) {
      if (cur < 0 && unit53(draw(inj_seed, p)) < inject_p) {
        cur = (int32_t)(draw(pick_seed, p) % (uint64_t)n_ph);
        off = 0;
      }
      if (cur >= 0) {
        const int32_t t = ph_tok[(size_t)cur * ph_stride + off];
        if (++off >= ph_len[cur]) cur = -1;
        return t;
      }
    }
    return base;
  }
};

// ------------------------------------------- distinct-window set per length
// Open addressing over stream positions; equality compares the windows.
struct WindowSet {
  const std::vector<int32_t>& src;
  int n;
  std::vector<int64_t> slots;
  size_t used = 0;
  WindowSet(const std::vector<int32_t>& s, int n_) : src(s), n(n_), slots(1 << 16, -1) {}
  // Slot of the stored window equal to the window at p, or -1.
  int64_t find(int64_t p) const {
    const size_t mask = slots.size() - 1;
    size_t i = hash_at(p) & mask;
    while (slots[i] >= 0) {
      if (same(slots[i], p)) return (int64_t)i;
      i = (i + 1) & mask;
    }
    return -1;
  }
  uint64_t hash_at(int64_t p) const {
    uint64_t h = 0x51ED270B27FA1C3Dull ^ (uint64_t)n;
    for (int j = 0; j < n; ++j) h = mix64(h ^ (uint64_t)(uint32_t)src[p + j]);
    return h;
  }
  bool same(int64_t a, int64_t b) const {
    return std::memcmp(&src[a], &src[b], sizeof(int32_t) * (size_t)n) == 0;
  }
  void grow() {
    std::vector<int64_t> old(slots.size() * 2, -1);
    old.swap(slots);
    const size_t mask = slots.size() - 1;
    for (int64_t p : old) {
      if (p < 0) continue;
      size_t i = hash_at(p) & mask;
      while (slots[i] >= 0) i = (i + 1) & mask;
      slots[i] = p;
    }
  }
  // Inserts the window starting at p; returns true if it was new.
  bool insert(int64_t p) {
    if ((used + 1) * 2 > slots.size()) grow();
    const size_t mask = slots.size() - 1;
    size_t i = hash_at(p) & mask;
    while (slots[i] >= 0) {
      if (same(slots[i], p)) return false;
      i = (i + 1) & mask;
    }
    slots[i] = p;
    ++used;
    return true;
  }
};

inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  const uint32_t bias = 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)((u + bias) >> 16);
}

inline uint16_t row_element(uint64_t seed, uint64_t ctr) {
  const uint64_t x = draw(seed, ctr);
  const int32_t s = (int32_t)(x & 0xFFFF) + (int32_t)((x >> 16) & 0xFFFF) +
                    (int32_t)((x >> 32) & 0xFFFF) + (int32_t)(x >> 48) - 131070;
  const float v = (float)s * 0x1.1bc77ap-21f;  // 0.02 / sqrt(4 * (2^32 - 1) / 12)
  return f32_to_bf16_rne(v);
}

}  // namespace

extern "C" {

uint64_t synth_mix64(uint64_t z) { return mix64(z); }

uint64_t synth_draw(uint64_t seed, uint64_t ctr) { return draw(seed, ctr); }

// Seed of sub-stream `sub` of stream `stream_id` of workload `workload_id`.
uint64_t synth_stream_seed(uint64_t master, uint32_t workload_id, uint32_t stream_id,
                           uint64_t sub) {
  const uint64_t s = mix64(master ^ (((uint64_t)workload_id << 32) | stream_id));
  return mix64(s ^ mix64(sub + kGamma));
}

// n Zipf(s) tokens over [0, vocab) from stream `seed`, with optional phrase
// injection (phrases: ph_tok[i * ph_stride + j], j < ph_len[i]). Returns 0,
// or -1 on bad arguments.
int synth_zipf_tokens(uint64_t seed, int32_t vocab, double s, int64_t n, double inject_p,
                      const int32_t* ph_tok, const int32_t* ph_len, int32_t n_ph, int32_t ph_stride,
                      int32_t* out) {
  if (vocab <= 0 || n < 0 || (n > 0 && !out) || s <= 0.0) return -1;
  Zipf z(vocab, s);
  Stream st(z, seed, inject_p, ph_tok, ph_len, n_ph, ph_stride);
  for (int64_t i = 0; i < n; ++i) out[i] = st.next();
  return 0;
}

// B query sequences of L tokens: sequence k uses the stream seed
// synth_stream_seed(master, workload_id, stream_id, first_sub + k), exactly
// as synth_zipf_tokens called once per sequence; sequences are split over
// `threads` threads. out is [B * L].
int synth_query_batch(uint64_t master, uint32_t workload_id, uint32_t stream_id,
                      uint64_t first_sub, int64_t B, int64_t L, int32_t vocab, double s,
                      double inject_p, const int32_t* ph_tok, const int32_t* ph_len,
                      int32_t n_ph, int32_t ph_stride, int32_t* out, int32_t threads) {
  if (vocab <= 0 || B < 0 || L < 0 || s <= 0.0 || (B * L > 0 && !out)) return -1;
  if (threads < 1) threads = 1;
  const Zipf z(vocab, s);
  std::vector<std::thread> pool;
  const int64_t per = (B + threads - 1) / threads;
  for (int32_t t = 0; t < threads; ++t) {
    const int64_t a = t * per, b = std::min<int64_t>(B, a + per);
    if (a >= b) break;
    pool.emplace_back([=, &z] {
      for (int64_t k = a; k < b; ++k) {
        const uint64_t base = mix64(master ^ (((uint64_t)workload_id << 32) | stream_id));
        const uint64_t seed = mix64(base ^ mix64(first_sub + (uint64_t)k + kGamma));
        Stream st(z, seed, inject_p, ph_tok, ph_len, n_ph, ph_stride);
        int32_t* o = out + k * L;
        for (int64_t i = 0; i < L; ++i) o[i] = st.next();
      }
    });
  }
  for (auto& th : pool) th.join();
  return 0;
}

// Pool of n_ph phrases with lengths uniform in [min_len, max_len] and Zipf(s)
// tokens; tok_out is [n_ph * max_len] (row-padded with -1).
int synth_phrase_pool(uint64_t seed, int32_t vocab, double s, int32_t n_ph, int32_t min_len,
                      int32_t max_len, int32_t* tok_out, int32_t* len_out) {
  if (vocab <= 0 || n_ph < 0 || min_len < 1 || max_len < min_len) return -1;
  Zipf z(vocab, s);
  const uint64_t len_seed = mix64(seed ^ 0x2545F4914F6CDD1Dull);
  uint64_t ctr = 0;
  for (int32_t i = 0; i < n_ph; ++i) {
    const int32_t span = max_len - min_len + 1;
    const int32_t len = min_len + (int32_t)(draw(len_seed, (uint64_t)i) % (uint64_t)span);
    len_out[i] = len;
    for (int32_t j = 0; j < max_len; ++j)
      tok_out[(size_t)i * max_len + j] = j < len ? z.sample(draw(seed, ctr++)) : -1;
  }
  return 0;
}

// Distinct n-grams taken from a Zipf source stream, in first-seen order.
// Scans positions p = 0, 1, ...; at each p, for n = 2..K whose quota (quota[n])
// is not full, the window src[p .. p+n-1] is appended if it was not seen
// before. The stream is extended until every quota is full or max_stream
// tokens were used. Outputs are fgram_tok[N * K] (row-padded with -1) and
// fgram_len[N], N = sum of quotas. If counts is not NULL, counts[r] receives
// the number of windows equal to f-gram r in the whole stream that was
// generated (stream_used tokens). Returns N, or -1 (bad args), -2 (cap hit).
int64_t synth_fgram_set(uint64_t seed, int32_t vocab, double s, int32_t K, const int64_t* quota,
                        double inject_p, const int32_t* ph_tok, const int32_t* ph_len,
                        int32_t n_ph, int32_t ph_stride, int64_t max_stream, int32_t* fgram_tok,
                        uint8_t* fgram_len, int64_t* stream_used, int64_t* counts) {
  if (vocab <= 0 || K < 2 || K > 16 || !quota || !fgram_tok || !fgram_len) return -1;
  int64_t total = 0;
  for (int n = 2; n <= K; ++n) {
    if (quota[n] < 0) return -1;
    total += quota[n];
  }
  Zipf z(vocab, s);
  Stream st(z, seed, inject_p, ph_tok, ph_len, n_ph, ph_stride);
  std::vector<int32_t> src;
  src.reserve(1 << 22);
  std::vector<WindowSet*> sets(K + 1, nullptr);
  std::vector<int64_t> have(K + 1, 0);
  for (int n = 2; n <= K; ++n) sets[n] = new WindowSet(src, n);
  int64_t filled = 0, p = 0;
  int rc = 0;
  while (filled < total) {
    if ((int64_t)src.size() >= max_stream) { rc = -2; break; }
    const int64_t grow = std::min<int64_t>(1 << 20, max_stream - (int64_t)src.size());
    for (int64_t i = 0; i < grow; ++i) src.push_back(st.next());
    const int64_t limit = (int64_t)src.size() - K;  // windows of every length fit
    for (; p <= limit && filled < total; ++p) {
      for (int n = 2; n <= K; ++n) {
        if (have[n] >= quota[n]) continue;
        if (sets[n]->insert(p)) {
          for (int j = 0; j < K; ++j) fgram_tok[(size_t)filled * K + j] = j < n ? src[p + j] : -1;
          fgram_len[filled] = (uint8_t)n;
          ++have[n];
          ++filled;
        }
      }
    }
  }
  if (stream_used) *stream_used = (int64_t)src.size();
  if (counts && rc == 0) {
    // row of each stored window: the f-grams of length n were appended in
    // increasing first position, so row r of length n pairs with the r-th
    // smallest stored position of that length
    std::vector<std::vector<int64_t>> slot_row(K + 1);
    for (int n = 2; n <= K; ++n) {
      std::vector<int64_t> rows;
      for (int64_t r = 0; r < filled; ++r)
        if (fgram_len[r] == n) rows.push_back(r);
      std::vector<std::pair<int64_t, int64_t>> by_pos;  // (stored position, slot)
      const auto& sl = sets[n]->slots;
      for (size_t i = 0; i < sl.size(); ++i)
        if (sl[i] >= 0) by_pos.emplace_back(sl[i], (int64_t)i);
      std::sort(by_pos.begin(), by_pos.end());
      slot_row[n].assign(sl.size(), -1);
      for (size_t k = 0; k < by_pos.size(); ++k) slot_row[n][by_pos[k].second] = rows[k];
    }
    for (int64_t r = 0; r < filled; ++r) counts[r] = 0;
    // every window of the stream, split over threads; counts are atomic adds
    const int64_t end = (int64_t)src.size();
    const int threads = std::max(1u, std::min(16u, std::thread::hardware_concurrency()));
    std::vector<std::thread> pool;
    const int64_t per = (end + threads - 1) / threads;
    for (int t = 0; t < threads; ++t) {
      const int64_t a = t * per, b = std::min<int64_t>(end, a + per);
      if (a >= b) break;
      pool.emplace_back([&, a, b] {
        for (int n = 2; n <= K; ++n)
          for (int64_t p = a; p < b && p + n <= end; ++p) {
            const int64_t i = sets[n]->find(p);
            if (i >= 0) __atomic_fetch_add(&counts[slot_row[n][i]], 1, __ATOMIC_RELAXED);
          }
      });
    }
    for (auto& th : pool) th.join();
  }
  for (int n = 2; n <= K; ++n) delete sets[n];
  return rc ? rc : filled;
}

// bf16 rows: out[i * d + c] = element(seed, row_ids[i] * d + c).
void synth_rows_cpu(uint64_t seed, int32_t d, const int64_t* row_ids, int64_t n, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) {
    const uint64_t base = (uint64_t)row_ids[i] * (uint64_t)d;
    for (int32_t c = 0; c < d; ++c) out[(size_t)i * d + c] = row_element(seed, base + c);
  }
}

// bf16 rows row0 .. row0 + n - 1 into out[n * d], split over `threads` threads.
void synth_rows_range_cpu(uint64_t seed, int32_t d, int64_t row0, int64_t n, uint16_t* out,
                          int32_t threads) {
  if (threads < 1) threads = 1;
  std::vector<std::thread> pool;
  const int64_t per = (n + threads - 1) / threads;
  for (int32_t t = 0; t < threads; ++t) {
    const int64_t a = t * per, b = std::min<int64_t>(n, a + per);
    if (a >= b) break;
    pool.emplace_back([=] {
      for (int64_t i = a; i < b; ++i) {
        const uint64_t base = (uint64_t)(row0 + i) * (uint64_t)d;
        for (int32_t c = 0; c < d; ++c) out[(size_t)i * d + c] = row_element(seed, base + c);
      }
    });
  }
  for (auto& th : pool) th.join();
}

}  // extern "C"
