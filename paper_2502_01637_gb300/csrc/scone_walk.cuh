// The walk over the lengths (tables with a suffix index) and the pieces the
// kernels that interleave it into a row copy share: asynchronous bucket
// loads into shared memory, the per-position walk state, chunked row copies.
//
// Algorithm 1 (Sec. 3) keeps, at each position, the longest window that is
// an f-gram. With a suffix index (scone_device.cuh) every suffix of length
// >= 2 of a listed f-gram is present with an extension bit, so a lookup can
// take n = 2, 3, ... one bucket at a time and stop at the first window that
// is absent or has no extension bit: nothing longer can be an f-gram, and
// every suffix of the longest f-gram is present with its bit, so the walk
// reaches it. One bucket is in flight per lane (two 16-byte cp.async into
// the lane's shared-memory slot); a round consumes it and issues the next.

#pragma once

#include "scone_host.h"

namespace scone {

// Asynchronous 16-byte global -> shared copies (cp.async, L2 only): the
// bucket loads of the match land in shared memory instead of registers, so
// the match state held across a copy segment is a few words per lane.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}
// One 32-byte bucket (16-byte slots) from the table into shared memory.
__device__ __forceinline__ void bucket_async(Bucket* dst, const TableView& t, uint64_t q) {
  const uint8_t* src = t.slots + q * bucket_bytes<FMT16>();
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  cp_async16(d, src);
  cp_async16(d + 16, src + 16);
}

// The walk over the lengths for one position (tables with a suffix index):
// `state` 1 = window tokens loaded, 2 = a bucket of length n in flight into
// this lane's shared-memory slot; 0 = done. Each round() consumes what the
// previous one issued and issues at most one bucket, so a lane takes at
// most 1 + 2 (K - 1) rounds.
template <int KT>
struct PipeWalk {
  int32_t w[KT];      // window tokens, newest first
  int nmax, n, state;
  bool second;        // the bucket in flight is the key's second one
  uint64_t b2;
  int32_t row;        // longest f-gram found so far, or -1
  int len, err;
  int pre_err;        // an error known before the walk (reported after a bad token)
  Bucket* sb;

  // Position p of a dense [B x L] batch, i = p mod L (its index in the sequence).
  __device__ __forceinline__ void start(const TableView& t, const int32_t* __restrict__ tok,
                                        int64_t p, int32_t i, bool act) {
    const int nm = t.K < i + 1 ? t.K : i + 1;
    start_with(act, act ? __ldg(tok + p) : 0, nm, 0,
               [&](int j) { return __ldg(tok + p - j); });
  }
  // A position whose token is x, whose window may span nm tokens (nm <= K)
  // and whose j-th predecessor is back(j), 1 <= j < nm; a nonzero pre (an
  // error found by the caller) makes it an error position unless its token is
  // invalid, which is reported first.
  template <class Back>
  __device__ __forceinline__ void start_with(bool act, int32_t x, int nm, int pre, Back back) {
    state = act ? 1 : 0;
    row = -1;
    len = 1;
    err = 0;
    pre_err = pre;
    nmax = 0;
    if (!act) return;
    w[0] = x;
    nmax = nm;
#pragma unroll
    for (int j = 1; j < KT; ++j) w[j] = (j < nmax) ? back(j) : 0;
  }
  __device__ __forceinline__ void issue_first(const TableView& t) {
    uint64_t b1;
    cuckoo_buckets(key_hash<FMT16>(window_key<FMT16, KT>(w, n, t.bits), t.hash_seed),
                   t.n_buckets, &b1, &b2);
    bucket_async(sb, t, b1);
    cp_async_commit();
    second = false;
    state = 2;
  }
  __device__ __forceinline__ void round(const TableView& t) {
    if (state == 1) {
      state = 0;
      if (!valid_token(w[0], t.vocab)) {
        err = SCONE_ERR_TOKEN_RANGE;
        len = 0;
        return;
      }
      if (pre_err) {
        err = pre_err;
        len = 0;
        return;
      }
      // a window is usable only if all its tokens are valid
      int nvalid = 1;
#pragma unroll
      for (int j = 1; j < KT; ++j)
        if (nvalid == j && j < nmax && valid_token(w[j], t.vocab)) nvalid = j + 1;
      nmax = nvalid;
      if (nmax < 2) return;
      n = 2;
      issue_first(t);
    } else if (state == 2) {
      cp_async_wait_all();
      BucketData<FMT16> v;
      v.part[0] = *sb;
      const uint32_t word = find_word_in_bucket<FMT16>(v, window_key<FMT16, KT>(w, n, t.bits));
      if (word != kEmptyRow) {
        const int32_t r = row_of_word(word);
        if (r >= 0) {
          row = r;
          len = n;
        }
        if ((word & kExtBit) && n < nmax) {
          ++n;
          issue_first(t);
        } else {
          state = 0;
        }
      } else if (!second && bucket_full<FMT16>(v)) {
        if (t.probe_limit < 2) {
          err = SCONE_ERR_PROBE_LIMIT;
          row = -1;
          len = 0;
          state = 0;
          return;
        }
        bucket_async(sb, t, b2);
        cp_async_commit();
        second = true;
      } else {
        state = 0;
      }
    }
  }
};

// Chunks [c_begin, c_end) of a warp's copy of nrows rows of epr 16-byte
// elements (src[r] to dst + r * epr; NULL writes zeros): chunk c covers the
// elements [32 U c, 32 U (c + 1)) in order, lane l taking every 32nd one.
// (r, col) is the lane's cursor, carried from one call to the next.
template <int U>
__device__ __forceinline__ void copy_chunks(const uint4* const* src, uint4* __restrict__ dst,
                                            int nrows, int epr, int64_t total, int lane,
                                            int c_begin, int c_end, int& r, int& col) {
  for (int c = c_begin; c < c_end; ++c) {
    const int64_t base = (int64_t)c * 32 * U;
    uint4 v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      v[u] = make_uint4(0, 0, 0, 0);
      if (r < nrows) {
        const uint4* s = src[r];
        if (s != nullptr) v[u] = ld_row<uint4>(s + col);
      }
      col += 32;
      while (col >= epr) {
        col -= epr;
        ++r;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t e = base + 32 * u + lane;
      if (e < total) st_out<uint4>(dst + e, v[u]);
    }
  }
}

// The source row of a finished walk (NULL for an error position), with the
// row and length written out (row -1 and length 0 at an error position).
template <int KT>
__device__ __forceinline__ const uint4* walk_finish(const TableView& t, const PipeWalk<KT>& m,
                                                    int64_t p, int32_t* __restrict__ row_out,
                                                    uint8_t* __restrict__ len_out) {
  if (row_out) row_out[p] = m.row;
  if (len_out) len_out[p] = (uint8_t)m.len;
  if (m.err) {
    record_error(t, m.err);
    return nullptr;
  }
  return reinterpret_cast<const uint4*>(m.row >= 0 ? t.F + (int64_t)m.row * t.d
                                                   : t.T + (int64_t)m.w[0] * t.d);
}

// The walk's match state is small (no bucket per length in registers), so
// the kernels that walk run with 8 loads in flight per lane at 3 blocks of
// 256 threads per SM (80 registers, no spills); on stress_k5 (K = 5) that
// measured 124.6 us against 125.6 for 16 loads at 2 blocks, and 12 x 3 or
// 6 x 4 spill and were slower. A warp's first tile is 8 positions: its
// rounds run before any row moves and the slowest of its lanes sets how
// many (123.1 us against 124.6 for a first tile of 32).
constexpr int kWalkLoads = 8;
constexpr int kWalkMinBlocks = 3;
constexpr int kWalkFirst = 8;

}  // namespace scone

namespace scone {

// The walk for one position in one thread, with blocking loads (for kernels
// that hide latency with many threads instead of interleaving a copy, such
// as the match kernel): tokens, then n = 2, 3, ... one bucket (or two) at a
// time. Same result, len and err as match_position; the default probe
// limit is assumed (the callers take the all-length lookups otherwise).
template <int KT>
__device__ __forceinline__ int32_t walk_position(const TableView& t,
                                                 const int32_t* __restrict__ tok, int64_t p,
                                                 int32_t i, int32_t x, int* len, int* err) {
  if (!valid_token(x, t.vocab)) {
    *err = SCONE_ERR_TOKEN_RANGE;
    *len = 0;
    return -1;
  }
  int nmax = t.K < i + 1 ? t.K : i + 1;
  int32_t w[KT];
  w[0] = x;
#pragma unroll
  for (int j = 1; j < KT; ++j) w[j] = (j < nmax) ? __ldg(tok + p - j) : 0;
  // a window is usable only if all its tokens are valid
  int nvalid = 1;
#pragma unroll
  for (int j = 1; j < KT; ++j)
    if (nvalid == j && j < nmax && valid_token(w[j], t.vocab)) nvalid = j + 1;
  nmax = nvalid;
  int32_t row = -1;
  *len = 1;
  for (int n = 2; n <= nmax; ++n) {
    const auto k = window_key<FMT16, KT>(w, n, t.bits);
    uint64_t b1, b2;
    cuckoo_buckets(key_hash<FMT16>(k, t.hash_seed), t.n_buckets, &b1, &b2);
    const BucketData<FMT16> v = ld_bucket_data<FMT16>(t, b1);
    uint32_t word = find_word_in_bucket<FMT16>(v, k);
    if (word == kEmptyRow && bucket_full<FMT16>(v))
      word = find_word_in_bucket<FMT16>(ld_bucket_data<FMT16>(t, b2), k);
    if (word == kEmptyRow) break;
    const int32_t r = row_of_word(word);
    if (r >= 0) {
      row = r;
      *len = n;
    }
    if (!(word & kExtBit)) break;
  }
  return row;
}

}  // namespace scone
