// Device-side building blocks of the SCONE embedding path (sm_103a).
//
// The f-gram dictionary (Sec. 2, "a hash dictionary that maps f-grams to
// matrix indices") is a bucketized cuckoo hash table: every key lives in one
// of two buckets chosen by two hashes of the key, and a bucket holds two
// slots (cuckoo hashing: Pagh and Rodler 2001; parallel GPU insertion:
// Alcantara et al. 2009). The build fills a key's first bucket before its
// second and never empties a slot, so a key can sit in its second bucket
// only if its first bucket is full. A lookup therefore reads the first
// bucket and stops there unless that bucket is full without holding the
// key; then it reads the second. Every lookup ends after at most two round
// trips (about 1.3 sectors on average at load factor 0.5), where linear
// probing has a long tail of dependent reads.
//
// Key: an injective packing of the n-gram. Token fields of b bits
// (b = ceil(log2 vocab)) hold the newest token at bit 0, the one before it
// at bit b, and so on, so the key of length n+1 extends the key of length n
// by one field; the length n sits in a 4-bit field at the top of the key.
// n >= 2, so a valid key is never all ones, which marks an empty slot.
//
//   FMT16: key of 96 bits (K*b <= 92), 16-byte slot = {key bits 0..63,
//          key bits 64..95 | row << 32}; 32-byte buckets (one sector).
//   FMT32: key of 224 bits (K*b <= 220), 32-byte slot = {key 0..63,
//          64..127, 128..191, key 192..223 | row << 32}; 64-byte buckets.
//
// The row word of an empty slot is 0xFFFFFFFF (row -1).
//
// Suffix index (tables built with one, TableView::suffix_index = 1): bit 31 of
// a row word is the extension bit, set when the slot's n-gram is the suffix
// of a longer listed f-gram; bits 0..30 hold the row, or kMarkerRow for a
// marker: an n-gram that is no f-gram itself but is such a suffix. Every
// suffix (length >= 2) of every listed f-gram is then present, so a lookup
// can take the lengths 2, 3, ... in turn and stop at the first window that
// is absent or has no extension bit: no longer window can be an f-gram.
// find_in_bucket hides both (a marker reads as absent), so every lookup that
// takes the lengths independently works on either kind of table.

#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "scone.h"

namespace scone {

constexpr int FMT16 = 0;
constexpr int FMT32 = 1;
constexpr int kSlotsPerBucket = 2;
constexpr uint32_t kEmptyRow = 0xFFFFFFFFu;
constexpr uint32_t kExtBit = 0x80000000u;     // row word: a longer f-gram ends with this n-gram
constexpr uint32_t kRowMask = 0x7FFFFFFFu;
constexpr uint32_t kMarkerRow = 0x7FFFFFFEu;  // row bits of a marker (no f-gram row)
constexpr uint32_t kMarkerWord = kExtBit | kMarkerRow;
constexpr uint64_t kHashSeed = 0x6A09E667F3BCC908ull;  // frac(sqrt 2), first 64 bits

template <int FMT>
struct Fmt;
template <>
struct Fmt<FMT16> {
  static constexpr int kWords = 2;        // 64-bit key words (96 bits used)
  static constexpr int kSlotBytes = 16;
  static constexpr int kLenShift = 28;    // length field in bits 92..95 (word 1, bits 28..31)
};
template <>
struct Fmt<FMT32> {
  static constexpr int kWords = 4;        // 224 bits used
  static constexpr int kSlotBytes = 32;
  static constexpr int kLenShift = 28;    // bits 220..223 (word 3, bits 28..31)
};
template <int FMT>
__host__ __device__ constexpr int bucket_bytes() {
  return kSlotsPerBucket * Fmt<FMT>::kSlotBytes;
}

// What a kernel needs to know about a table (passed by value).
struct TableView {
  const uint8_t* slots;      // bucket q at slots + q * bucket_bytes
  uint64_t n_buckets;
  uint64_t hash_seed;        // seed of the two bucket hashes (chosen at build)
  int64_t probe_limit;       // buckets one lookup may read: 1 or 2
  int64_t n_fgrams;
  const uint16_t* F;         // device-accessible address of F (HBM or host-mapped)
  const uint16_t* T;
  int* status;               // sticky first device-detected error
  int* status_mirror;        // device address of a host-mapped copy of it, or NULL
  int32_t K;
  int32_t bits;
  int32_t vocab;
  int32_t d;
  int32_t suffix_index;      // 1: extension bits and markers present (see above)
};

template <int NW>
struct KeyBits {
  uint64_t w[NW];
};

struct Bucket {
  uint64_t a, b, c, e;
};

__device__ __forceinline__ uint64_t fmix64(uint64_t z) {
  // SplitMix64 / MurmurHash3 finalizer (Steele, Lea, Flood 2014)
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Inserts field value v (< 2^b) at bit offset off.
template <int NW>
__device__ __forceinline__ void put_field(KeyBits<NW>& k, int off, uint32_t v, int b) {
#pragma unroll
  for (int q = 0; q < NW; ++q) {
    const int rel = off - 64 * q;
    if (rel >= 0 && rel < 64) {
      k.w[q] |= (uint64_t)v << rel;
    } else if (rel < 0 && rel > -b) {
      k.w[q] |= (uint64_t)v >> (-rel);
    }
  }
}

template <int FMT>
__device__ __forceinline__ void put_len(KeyBits<Fmt<FMT>::kWords>& k, int n) {
  k.w[Fmt<FMT>::kWords - 1] |= (uint64_t)n << Fmt<FMT>::kLenShift;
}

template <int FMT>
__device__ __forceinline__ uint64_t key_hash(const KeyBits<Fmt<FMT>::kWords>& k, uint64_t seed) {
  uint64_t h = seed;
#pragma unroll
  for (int q = Fmt<FMT>::kWords - 1; q >= 0; --q) h = fmix64(k.w[q] ^ h);
  return h;
}

// Lemire's multiply-shift range reduction: maps h uniformly onto [0, n).
__device__ __forceinline__ uint64_t fastrange(uint64_t h, uint64_t n) { return __umul64hi(h, n); }

// The key's two candidate buckets (distinct when n >= 2).
__device__ __forceinline__ void cuckoo_buckets(uint64_t h, uint64_t n, uint64_t* b1,
                                               uint64_t* b2) {
  *b1 = fastrange(h, n);
  uint64_t q = fastrange(fmix64(h + 0x9E3779B97F4A7C15ull), n);
  if (q == *b1) q = (q + 1 == n) ? 0 : q + 1;
  *b2 = q;
}

// One 256-bit read-only load (32 bytes, one sector).
__device__ __forceinline__ Bucket ld_bucket(const uint8_t* p) {
  Bucket r;
  asm("ld.global.nc.v4.u64 {%0, %1, %2, %3}, [%4];"
      : "=l"(r.a), "=l"(r.b), "=l"(r.c), "=l"(r.e)
      : "l"(p));
  return r;
}

// A whole bucket in registers: one 32-byte load (FMT16) or two (FMT32).
template <int FMT>
struct BucketData {
  Bucket part[bucket_bytes<FMT>() / 32];
};

template <int FMT>
__device__ __forceinline__ BucketData<FMT> ld_bucket_data(const TableView& t, uint64_t q) {
  BucketData<FMT> v;
  const uint8_t* p = t.slots + q * bucket_bytes<FMT>();
#pragma unroll
  for (int i = 0; i < bucket_bytes<FMT>() / 32; ++i) v.part[i] = ld_bucket(p + 32 * i);
  return v;
}

// Whether both slots of the bucket are taken.
template <int FMT>
__device__ __forceinline__ bool bucket_full(const BucketData<FMT>& v) {
  if constexpr (FMT == FMT16) {
    return (uint32_t)(v.part[0].b >> 32) != kEmptyRow && (uint32_t)(v.part[0].e >> 32) != kEmptyRow;
  } else {
    return (uint32_t)(v.part[0].e >> 32) != kEmptyRow && (uint32_t)(v.part[1].e >> 32) != kEmptyRow;
  }
}

// The row word of the slot holding the key, or kEmptyRow if the bucket
// does not hold it (an empty slot's key bits are all ones, never a key).
template <int FMT>
__device__ __forceinline__ uint32_t find_word_in_bucket(const BucketData<FMT>& v,
                                                        const KeyBits<Fmt<FMT>::kWords>& k) {
  if constexpr (FMT == FMT16) {
    const Bucket& x = v.part[0];
    if (x.a == k.w[0] && (uint32_t)x.b == (uint32_t)k.w[1]) return (uint32_t)(x.b >> 32);
    if (x.c == k.w[0] && (uint32_t)x.e == (uint32_t)k.w[1]) return (uint32_t)(x.e >> 32);
    return kEmptyRow;
  } else {
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const Bucket& x = v.part[s];
      if (x.a == k.w[0] && x.b == k.w[1] && x.c == k.w[2] && (uint32_t)x.e == (uint32_t)k.w[3])
        return (uint32_t)(x.e >> 32);
    }
    return kEmptyRow;
  }
}

// The f-gram row of a row word, or -1 (absent, or a marker).
__device__ __forceinline__ int32_t row_of_word(uint32_t word) {
  const uint32_t r = word & kRowMask;
  return (word == kEmptyRow || r == kMarkerRow) ? -1 : (int32_t)r;
}

// The key's row if one of the bucket's slots holds it as an f-gram, else -1.
template <int FMT>
__device__ __forceinline__ int32_t find_in_bucket(const BucketData<FMT>& v,
                                                  const KeyBits<Fmt<FMT>::kWords>& k) {
  return row_of_word(find_word_in_bucket<FMT>(v, k));
}

// Looks a key up: the first bucket, then the second only if the first is
// full without the key. With a probe limit of 1 the second bucket is never
// read; a lookup that would need it reports SCONE_ERR_PROBE_LIMIT.
template <int FMT>
__device__ __forceinline__ int32_t cuckoo_lookup(const TableView& t,
                                                 const KeyBits<Fmt<FMT>::kWords>& k, int* err) {
  uint64_t b1, b2;
  cuckoo_buckets(key_hash<FMT>(k, t.hash_seed), t.n_buckets, &b1, &b2);
  const BucketData<FMT> v1 = ld_bucket_data<FMT>(t, b1);
  const int32_t r = find_in_bucket<FMT>(v1, k);
  if (r >= 0 || !bucket_full<FMT>(v1)) return r;
  if (t.probe_limit < 2) {
    *err = SCONE_ERR_PROBE_LIMIT;
    return -1;
  }
  return find_in_bucket<FMT>(ld_bucket_data<FMT>(t, b2), k);
}

// The same result as cuckoo_lookup with both candidate buckets loaded in one
// round trip: for latency-bound callers (a decode step) that can spend a
// second 32-byte sector per lookup to save a dependent read. The second
// bucket is used only where cuckoo_lookup would read it.
template <int FMT>
__device__ __forceinline__ int32_t cuckoo_lookup_eager(const TableView& t,
                                                       const KeyBits<Fmt<FMT>::kWords>& k,
                                                       int* err) {
  uint64_t b1, b2;
  cuckoo_buckets(key_hash<FMT>(k, t.hash_seed), t.n_buckets, &b1, &b2);
  const BucketData<FMT> v1 = ld_bucket_data<FMT>(t, b1);
  const BucketData<FMT> v2 = ld_bucket_data<FMT>(t, b2);
  const int32_t r = find_in_bucket<FMT>(v1, k);
  if (r >= 0 || !bucket_full<FMT>(v1)) return r;
  if (t.probe_limit < 2) {
    *err = SCONE_ERR_PROBE_LIMIT;
    return -1;
  }
  return find_in_bucket<FMT>(v2, k);
}

// Records a device-detected error: the first one wins the table's status
// word, and the thread that wins also writes it to the host-mapped mirror, so
// that scone_status finds "no error" by reading host memory alone.
__device__ __forceinline__ void record_error(const TableView& t, int code) {
  if (*reinterpret_cast<volatile int*>(t.status) == 0 && atomicCAS(t.status, 0, code) == 0 &&
      t.status_mirror)
    *reinterpret_cast<volatile int*>(t.status_mirror) = code;
}

__device__ __forceinline__ bool valid_token(int32_t x, int32_t vocab) {
  return (uint32_t)x < (uint32_t)vocab;
}

// Algorithm 1's selection for one position: the longest n in [2, min(K, i+1)]
// whose window (tok[p-n+1 .. p]) is an f-gram. All candidate lengths are
// hashed in registers and their first buckets loaded together (K-1 loads in
// one round trip); the lengths that still need their second bucket load it
// together in a second round trip; then the longest hit wins. Returns the
// row (or -1) and sets *len (n, 1 for the token fallback, 0 for an error
// position) and *err.
template <int FMT, int KT>
__device__ __forceinline__ KeyBits<Fmt<FMT>::kWords> window_key(const int32_t (&w)[KT], int n,
                                                               int bits) {
  constexpr int NW = Fmt<FMT>::kWords;
  KeyBits<NW> k;
#pragma unroll
  for (int q = 0; q < NW; ++q) k.w[q] = 0;
  k.w[0] = (uint32_t)w[0];
#pragma unroll
  for (int j = 1; j < KT; ++j)
    if (j < n) put_field<NW>(k, j * bits, (uint32_t)w[j], bits);
  put_len<FMT>(k, n);
  return k;
}

template <int FMT, int KT>
__device__ __forceinline__ int32_t match_position(const TableView& t,
                                                  const int32_t* __restrict__ tok, int64_t p,
                                                  int32_t i, int32_t tok_p, int* len, int* err) {
  if (!valid_token(tok_p, t.vocab)) {
    *err = SCONE_ERR_TOKEN_RANGE;
    *len = 0;
    return -1;
  }
  int nmax = t.K < i + 1 ? t.K : i + 1;
  int32_t w[KT];
  w[0] = tok_p;
#pragma unroll
  for (int j = 1; j < KT; ++j) w[j] = (j < nmax) ? __ldg(tok + p - j) : 0;
  // a window is usable only if all its tokens are valid
  int nvalid = 1;
#pragma unroll
  for (int j = 1; j < KT; ++j)
    if (nvalid == j && j < nmax && valid_token(w[j], t.vocab)) nvalid = j + 1;
  nmax = nvalid;

  // round trip 1: the first bucket of every candidate length
  BucketData<FMT> v[KT - 1];
#pragma unroll
  for (int n = 2; n <= KT; ++n) {
    if (n <= nmax) {
      uint64_t b1, b2;
      cuckoo_buckets(key_hash<FMT>(window_key<FMT, KT>(w, n, t.bits), t.hash_seed), t.n_buckets,
                     &b1, &b2);
      v[n - 2] = ld_bucket_data<FMT>(t, b1);
    }
  }
  int32_t r1[KT - 1];
  uint32_t second = 0;   // bit n-2: length n needs its second bucket
#pragma unroll
  for (int n = 2; n <= KT; ++n) {
    r1[n - 2] = -1;
    if (n <= nmax) {
      r1[n - 2] = find_in_bucket<FMT>(v[n - 2], window_key<FMT, KT>(w, n, t.bits));
      if (r1[n - 2] < 0 && bucket_full<FMT>(v[n - 2])) second |= 1u << (n - 2);
    }
  }
  // only lengths longer than the longest first-round hit matter
  int best = 0;
#pragma unroll
  for (int n = 2; n <= KT; ++n)
    if (r1[n - 2] >= 0) best = n;
  second &= ~((1u << (best > 1 ? best - 1 : 0)) - 1u);
  if (second) {
    if (t.probe_limit < 2) {
      *err = SCONE_ERR_PROBE_LIMIT;
      *len = 0;
      return -1;
    }
    // round trip 2: the second buckets still needed
#pragma unroll
    for (int n = 2; n <= KT; ++n) {
      if (second & (1u << (n - 2))) {
        uint64_t b1, b2;
        cuckoo_buckets(key_hash<FMT>(window_key<FMT, KT>(w, n, t.bits), t.hash_seed),
                       t.n_buckets, &b1, &b2);
        v[n - 2] = ld_bucket_data<FMT>(t, b2);
      }
    }
#pragma unroll
    for (int n = 2; n <= KT; ++n)
      if (second & (1u << (n - 2)))
        r1[n - 2] = find_in_bucket<FMT>(v[n - 2], window_key<FMT, KT>(w, n, t.bits));
  }
#pragma unroll
  for (int n = KT; n >= 2; --n) {
    if (n <= nmax && r1[n - 2] >= 0) {
      *len = n;
      return r1[n - 2];
    }
  }
  *len = 1;
  return -1;
}

// The same selection for a window whose tokens come from back(j), the token
// j places before the position, for 1 <= j < nmax (nmax <= K: the longest
// window within the sequence and its known history); tok_p is the
// position's own, valid token. Used where a window can reach past the start
// of the packed tokens (ragged and continued batches). match_position keeps
// its own copy of these steps: written through this function, the dense
// kernels' compiled code differs and measured about 1% slower.
struct Match {
  int32_t row;   // F row, or -1
  int len;       // n, 1 for the token fallback, 0 on error
  int err;       // 0 or a SCONE_ERR_* code
};

template <int FMT, int KT, class Back>
__device__ __forceinline__ Match match_window(const TableView& t, int32_t tok_p, int nmax,
                                              Back back) {
  int32_t w[KT];
  w[0] = tok_p;
#pragma unroll
  for (int j = 1; j < KT; ++j) w[j] = (j < nmax) ? back(j) : 0;
  // a window is usable only if all its tokens are valid
  int nvalid = 1;
#pragma unroll
  for (int j = 1; j < KT; ++j)
    if (nvalid == j && j < nmax && valid_token(w[j], t.vocab)) nvalid = j + 1;
  nmax = nvalid;

  // round trip 1: the first bucket of every candidate length
  BucketData<FMT> v[KT - 1];
#pragma unroll
  for (int n = 2; n <= KT; ++n) {
    if (n <= nmax) {
      uint64_t b1, b2;
      cuckoo_buckets(key_hash<FMT>(window_key<FMT, KT>(w, n, t.bits), t.hash_seed), t.n_buckets,
                     &b1, &b2);
      v[n - 2] = ld_bucket_data<FMT>(t, b1);
    }
  }
  int32_t r1[KT - 1];
  uint32_t second = 0;   // bit n-2: length n needs its second bucket
#pragma unroll
  for (int n = 2; n <= KT; ++n) {
    r1[n - 2] = -1;
    if (n <= nmax) {
      r1[n - 2] = find_in_bucket<FMT>(v[n - 2], window_key<FMT, KT>(w, n, t.bits));
      if (r1[n - 2] < 0 && bucket_full<FMT>(v[n - 2])) second |= 1u << (n - 2);
    }
  }
  // only lengths longer than the longest first-round hit matter
  int best = 0;
#pragma unroll
  for (int n = 2; n <= KT; ++n)
    if (r1[n - 2] >= 0) best = n;
  second &= ~((1u << (best > 1 ? best - 1 : 0)) - 1u);
  if (second) {
    if (t.probe_limit < 2) return Match{-1, 0, SCONE_ERR_PROBE_LIMIT};
    // round trip 2: the second buckets still needed
#pragma unroll
    for (int n = 2; n <= KT; ++n) {
      if (second & (1u << (n - 2))) {
        uint64_t b1, b2;
        cuckoo_buckets(key_hash<FMT>(window_key<FMT, KT>(w, n, t.bits), t.hash_seed),
                       t.n_buckets, &b1, &b2);
        v[n - 2] = ld_bucket_data<FMT>(t, b2);
      }
    }
#pragma unroll
    for (int n = 2; n <= KT; ++n)
      if (second & (1u << (n - 2)))
        r1[n - 2] = find_in_bucket<FMT>(v[n - 2], window_key<FMT, KT>(w, n, t.bits));
  }
#pragma unroll
  for (int n = KT; n >= 2; --n) {
    if (n <= nmax && r1[n - 2] >= 0) return Match{r1[n - 2], n, 0};
  }
  return Match{-1, 1, 0};
}

// ------------------------------------------------------------- row copies
template <typename E>
__device__ __forceinline__ E ld_row(const E* p) {
  return __ldg(p);
}
template <>
__device__ __forceinline__ uint4 ld_row<uint4>(const uint4* p) {
  uint4 v;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p));
  return v;
}

template <typename E>
__device__ __forceinline__ void st_out(E* p, const E& v) {
  __stcs(p, v);
}

template <typename E>
__device__ __forceinline__ E zero_of() {
  return E{};
}
template <>
__device__ __forceinline__ uint4 zero_of<uint4>() {
  return make_uint4(0, 0, 0, 0);
}
template <>
__device__ __forceinline__ uint2 zero_of<uint2>() {
  return make_uint2(0, 0);
}

constexpr int kLoadsInFlight = 16;

// A warp copies nrows rows of epr elements of type E: row r from src[r]
// (NULL writes zeros) to dst + r * epr, rows contiguous in dst. The warp
// walks the nrows * epr elements in order, lane l taking every 32nd one, and
// keeps U loads per lane outstanding before the matching streaming stores.
// (row, column) of a lane's element advance incrementally, so any row width
// works without a division.
template <typename E, int U>
__device__ __forceinline__ void warp_copy_rows(const E* const* src, E* __restrict__ dst,
                                               int nrows, int epr, int lane) {
  const int64_t total = (int64_t)nrows * epr;
  int r = 0, col = lane;
  while (col >= epr) {
    col -= epr;
    ++r;
  }
  for (int64_t base = 0; base < total; base += 32 * U) {
    E v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      v[u] = zero_of<E>();
      if (r < nrows) {
        const E* s = src[r];
        if (s != nullptr) v[u] = ld_row<E>(s + col);
      }
      col += 32;
      while (col >= epr) {
        col -= epr;
        ++r;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t c = base + 32 * u + lane;
      if (c < total) st_out<E>(dst + c, v[u]);
    }
  }
}

// Row copy for a width chosen at run time: 16-byte chunks when W == 16
// (U of them in flight per lane), otherwise the widest of 8, 4 or 2 bytes
// that the row size and all three base addresses allow (width_bytes).
template <int W, int U = kLoadsInFlight>
__device__ __forceinline__ void warp_copy_rows_w(const void* const* src, void* dst, int nrows,
                                                 int row_bytes, int width_bytes, int lane) {
  if constexpr (W == 16) {
    warp_copy_rows<uint4, U>(reinterpret_cast<const uint4* const*>(src),
                             reinterpret_cast<uint4*>(dst), nrows, row_bytes >> 4, lane);
  } else {
    if (width_bytes == 8) {
      warp_copy_rows<uint2, kLoadsInFlight>(reinterpret_cast<const uint2* const*>(src),
                                            reinterpret_cast<uint2*>(dst), nrows, row_bytes >> 3,
                                            lane);
    } else if (width_bytes == 4) {
      warp_copy_rows<unsigned int, kLoadsInFlight>(
          reinterpret_cast<const unsigned int* const*>(src), reinterpret_cast<unsigned int*>(dst),
          nrows, row_bytes >> 2, lane);
    } else {
      warp_copy_rows<unsigned short, kLoadsInFlight>(
          reinterpret_cast<const unsigned short* const*>(src),
          reinterpret_cast<unsigned short*>(dst), nrows, row_bytes >> 1, lane);
    }
  }
}

}  // namespace scone
